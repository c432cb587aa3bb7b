// NVFP4 block-scale selection kernels: ScaleSweep (Sec. 4.2.2 of the paper),
// AbsMax (Sec. 3.2) and 4/6 (Sec. 2), sharing one register-resident skeleton.
//
// Mapping: one thread owns one 16-element segment (32 or 64 bytes of input) and
// keeps it in registers; a scale block of 16/32/64 elements is 1/2/4
// consecutive lanes of a warp, which combine block max and per-candidate losses
// with xor-shuffles (commutative pairwise sums, so every lane of a block holds
// bit-identical losses and takes the same decision).  The grid-stride loop
// walks whole warps so every shuffle runs with all 32 lanes converged, and the
// next segment's input is loaded before the current one is swept.
//
// ScaleSweep per block: y = fl(x*E), m = max|y|, s_base = fl(m/6),
// I0 = floor_E4M3(s_base); for codes c in [I0+lo, I0+hi] clamped to 1..126:
// L_c = sum_i w_i (y_i - q_i v_c)^2 with q_i = RNE_E2M1(fl(y_i * fl(1/v_c)));
// keep the first (lowest-code) minimum.  The per-candidate work on an element
// pair is mul.f32x2 -> cvt e2m1x2 -> cvt f16x2 (exact decode) -> two mixed
// fma.f32.f16 (exact product q*(-v), one rounding) -> fma.f32x2 accumulate.
//
// Candidate table: entry code+128 holds {fl(1/v_c), f16 bits of -v_c} for codes
// 1..126 and a poison entry {+inf, -inf} elsewhere.  (8-byte entries measured
// faster than 16-byte ones holding the packed {r, r} operand.)  A poison candidate's loss
// is inf or NaN, so it never wins the strict "<" -- this lets the default
// windows run a fixed, fully unrolled loop over [I0+lo, I0+hi] with no clamping
// (those windows always contain a real code).  Custom windows clamp instead.
#pragma once
#include <atomic>

#include "nvfp4_device.cuh"
#include "nvfp4_kernels.h"

namespace nvfp4 {

// Resident CTAs per SM of `kernel` launched with `threads` threads on the
// current device, looked up once per device; the per-device atomics make
// first calls from several host threads safe.
constexpr int kOccDevices = 64;
template <typename K>
inline int occupancy_per_sm(std::atomic<int> (&cache)[kOccDevices], K kernel, int threads) {
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess) dev = -1;
    if (dev >= 0 && dev < kOccDevices) {
        const int c = cache[dev].load(std::memory_order_relaxed);
        if (c > 0) return c;
    }
    int b = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&b, kernel, threads, 0) != cudaSuccess || b < 1) b = 1;
    if (dev >= 0 && dev < kOccDevices) cache[dev].store(b, std::memory_order_relaxed);
    return b;
}

struct Cand {
    float r;        // fl(1/v_c)
    uint32_t nv;    // f16 bits of -v_c in the low half
};
constexpr int kTabOff = 128;
constexpr int kTabN = 384;

__device__ __forceinline__ void build_table(Cand* t) {
    for (int i = threadIdx.x; i < kTabN; i += blockDim.x) {
        const int c = i - kTabOff;
        Cand e;
        if (c >= 1 && c <= 126) {
            const uint16_t h = e4m3_to_f16bits((uint32_t)c);
            e.r = __frcp_rn(f16bits_to_f32(h));
            e.nv = (uint32_t)(h ^ 0x8000u);
        } else {
            e.r = __int_as_float(0x7f800000);
            e.nv = 0xFC00u;
        }
        t[i] = e;
    }
}

struct Raw {
    uint4 a, b, c, d;
};

template <int DT>
__device__ __forceinline__ void load_raw(const void* x, int64_t g, Raw& r) {
    if (DT == 0) {
        const uint4* p = reinterpret_cast<const uint4*>(static_cast<const char*>(x) + g * 32);
        r.a = ld_stream16(p);
        r.b = ld_stream16(p + 1);
    } else {
        const uint4* p = reinterpret_cast<const uint4*>(static_cast<const char*>(x) + g * 64);
        r.a = ld_stream16(p);
        r.b = ld_stream16(p + 1);
        r.c = ld_stream16(p + 2);
        r.d = ld_stream16(p + 3);
    }
}

// NaN-propagating maxima: the block max is NaN if any element is NaN, so a
// block holding a non-finite value is recognised from m alone (zero_block).
__device__ __forceinline__ float max3f(float a, float b, float c) {
    float d;
    asm("max.NaN.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}
__device__ __forceinline__ float max2f(float a, float b) {
    float d;
    asm("max.NaN.f32 %0, %1, %2;" : "=f"(d) : "f"(a), "f"(b));
    return d;
}

// Blocks whose largest normalised magnitude m is NaN, infinite or >= 2^48
// take the zero rule (scale code 0, nibbles carry only the signs), as do
// all-zero blocks.  With S = amax/(6 D) every finite input gives m <= 6 D, so
// only non-finite inputs or a caller-supplied S far below the tensor's own
// reach it; below it every fp32 candidate loss stays finite for weights up to
// 2^24 (16..64 terms of at most 2^24 * (2^48 + 2688)^2).
__device__ __forceinline__ bool zero_block(bool usable, float m) {
    return !usable || !(m > 0.0f && m < 281474976710656.0f);
}

// The segment's 16 inputs as 8 packed pairs y = fl(x*E) (one f32x2 multiply
// per pair) and the block max m = max |y|.
template <int DT>
__device__ __forceinline__ float raw_to_y(const Raw& r, u64 E2, u64 (&y2)[8]) {
    uint32_t u[16];
    if (DT == 0) {
        const uint32_t p[8] = {r.a.x, r.a.y, r.a.z, r.a.w, r.b.x, r.b.y, r.b.z, r.b.w};
#pragma unroll
        for (int j = 0; j < 8; j++) {
            u[2 * j] = p[j] << 16;
            u[2 * j + 1] = p[j] & 0xFFFF0000u;
        }
    } else {
        const uint32_t p[16] = {r.a.x, r.a.y, r.a.z, r.a.w, r.b.x, r.b.y, r.b.z, r.b.w,
                                r.c.x, r.c.y, r.c.z, r.c.w, r.d.x, r.d.y, r.d.z, r.d.w};
#pragma unroll
        for (int j = 0; j < 16; j++) u[j] = p[j];
    }
    float av[16];
#pragma unroll
    for (int j = 0; j < 8; j++) {
        y2[j] = mul2(pack2(__uint_as_float(u[2 * j]), __uint_as_float(u[2 * j + 1])), E2);
        float a, b;
        unpack2(y2[j], a, b);
        av[2 * j] = fabsf(a);
        av[2 * j + 1] = fabsf(b);
    }
    // three-input max tree (a NaN element makes m NaN)
    const float p0 = max3f(av[0], av[1], av[2]), p1 = max3f(av[3], av[4], av[5]), p2 = max3f(av[6], av[7], av[8]);
    const float p3 = max3f(av[9], av[10], av[11]), p4 = max3f(av[12], av[13], av[14]);
    return max3f(max3f(p0, p1, p2), max3f(p3, p4, av[15]), 0.0f);
}

// raw_to_y that also returns the largest |y| of each half of the segment
// (elements 0-7 in ma, 8-15 in mb); m = max(ma, mb) is raw_to_y's value.  Its
// max tree takes one more instruction than raw_to_y's, which the methods that
// have no use for the halves (AbsMax, 4/6) therefore keep.
template <int DT>
__device__ __forceinline__ float raw_to_y_halves(const Raw& r, u64 E2, u64 (&y2)[8], float& ma, float& mb) {
    uint32_t u[16];
    if (DT == 0) {
        const uint32_t p[8] = {r.a.x, r.a.y, r.a.z, r.a.w, r.b.x, r.b.y, r.b.z, r.b.w};
#pragma unroll
        for (int j = 0; j < 8; j++) {
            u[2 * j] = p[j] << 16;
            u[2 * j + 1] = p[j] & 0xFFFF0000u;
        }
    } else {
        const uint32_t p[16] = {r.a.x, r.a.y, r.a.z, r.a.w, r.b.x, r.b.y, r.b.z, r.b.w,
                                r.c.x, r.c.y, r.c.z, r.c.w, r.d.x, r.d.y, r.d.z, r.d.w};
#pragma unroll
        for (int j = 0; j < 16; j++) u[j] = p[j];
    }
    float av[16];
#pragma unroll
    for (int j = 0; j < 8; j++) {
        y2[j] = mul2(pack2(__uint_as_float(u[2 * j]), __uint_as_float(u[2 * j + 1])), E2);
        float a, b;
        unpack2(y2[j], a, b);
        av[2 * j] = fabsf(a);
        av[2 * j + 1] = fabsf(b);
    }
    ma = max3f(max3f(av[0], av[1], av[2]), max3f(av[3], av[4], av[5]), max2f(av[6], av[7]));
    mb = max3f(max3f(av[8], av[9], av[10]), max3f(av[11], av[12], av[13]), max2f(av[14], av[15]));
    return max3f(ma, mb, 0.0f);
}

// Loss of one candidate on this thread's 16 elements.
template <int OBJ>
__device__ __forceinline__ float seg_loss(const u64 (&y2)[8], const u64 (&w2)[8], float r, uint16_t nv) {
    const u64 r2 = pack2(r, r);
    u64 acc = 0ull;
#pragma unroll
    for (int j = 0; j < 8; j++) {
        const u64 e2 = cand_err2(y2[j], r2, nv);
        if (OBJ == 1) {
            acc = fma2(mul2(w2[j], e2), e2, acc);
        } else {
            acc = fma2(e2, e2, acc);
        }
    }
    float a, b;
    unpack2(acc, a, b);
    return __fadd_rn(a, b);
}

template <int SEGS>
__device__ __forceinline__ float group_sum(float v) {
    if (SEGS >= 2) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, 1));
    if (SEGS >= 4) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, 2));
    return v;
}
template <int SEGS>
__device__ __forceinline__ float group_max(float v) {
    if (SEGS >= 2) v = max2f(v, __shfl_xor_sync(0xffffffffu, v, 1));
    if (SEGS >= 4) v = max2f(v, __shfl_xor_sync(0xffffffffu, v, 2));
    return v;
}

// Default-window argmin (FIX windows: [I0-3, I0+7] for MSE with blocks of
// 16, [I0-8, I0+7] otherwise) over the candidate table entries tb[0..FIX_K),
// tb[k] being code I0 + FIX_LO + k.  Returns the offset k of the lowest code
// whose loss is minimal and sets `best` to that loss.
//
// The lowest NB offsets are visited last, in descending order, and a warp
// skips one when, for every lane, a lower bound on the block's loss for that
// candidate already exceeds the lane's best loss so far.  The bound is the sum
// of two terms per lane of the block, those of the largest |y| of each half of
// the lane's segment (ma, mb: distinct elements), computed with the loop's own
// arithmetic: cand_err2 gives their errors e bit for bit and the terms are
// fl(e e) (MSE) or fl(fl(w e) e) (WMSE, w the weight of an element of that
// half whose |y| is its maximum).  The loss accumulates every element's
// product exactly once into a rounded running sum, so with non-negative terms
// (squares; WMSE: only while the lane's weights are non-negative, `wok`, else
// no skip) and monotone rounding it is at least the two products' sum with at
// most four roundings (two in a lane, two in the block's shuffle sum), while
// the bound is computed with at most six upward roundings and then multiplied
// by 1 - 2^-20, which covers both: a skipped candidate's loss is above the
// final best, so it can neither win nor tie.  The losses that are computed are
// the same values in the same order, with ties going to the lowest code (<=
// for the codes below every code already visited), so the result is the full
// sweep's, bit for bit.  On the low offsets the largest elements saturate
// (6 v_c < m), which makes the bound tight.  A CPU simulation on the synthetic
// Qwen2.5-72B-shaped weights (warps of 32 consecutive blocks) gives the skips
// per warp: WMSE 3.4 of 16 candidates with blocks of 16 (NB 4; 2.2 with the
// largest element alone), 3.4 / 3.3 with blocks of 32 / 64 (NB 4); MSE 1.2 of
// 11 with blocks of 16 (NB 2), 5.9 / 5.5 of 16 with blocks of 32 / 64 (NB 6).
// NB measured on the grouped call over the full workloads (ms, in-launch
// scales; every setting gave the same output bytes), WMSE16/WMSE32,64/MSE16/
// MSE32,64 = 4/0/1/5, 5/4/2/6, 6/6/3/7: Qwen shapes WMSE block 16
// 1.369/1.369/1.386, block 32 1.502/1.390/1.390, block 64 1.558/1.433/1.454;
// MSE block 16 0.869/0.863/0.886, block 32 0.991/0.954/0.973, block 64
// 1.034/0.997/1.022; Llama-3-8B layer 0.620/0.623/0.632 (no bound: 1.511 Qwen
// WMSE block 16, 0.684 Llama, 0.892 Qwen MSE block 16).
// GROUPED: the grouped kernel (else the per-tensor one), whose best MSE
// block-16 setting differs (per-tensor sweeps, ms, NB 1 against 2: Gaussian
// 16384 x 8192 0.2125/0.218, Student-t 32768 x 8192 0.4154/0.4219, Laplace
// 8192 x 8192 0.1085/0.1104; per-tensor WMSE with NB 4 against the plain
// sweep: 0.3585/0.3831, 0.704/0.757, 0.1815/0.1947).  Per-tensor blocks of
// 32/64 on the same three tensors, MSE NB 6/5/4/0: 0.266/0.274/0.278/0.303 and
// 0.287/0.279/0.289/0.318 (Gaussian), 0.522/0.542/0.550/0.592 and
// 0.547/0.550/0.572/0.630 (Student-t); WMSE NB 4 against 0: 0.381/0.391 and
// 0.387/0.389 (Gaussian), 0.753/0.776 and 0.764/0.764 (Student-t).
template <int OBJ, int BLOCK, bool GROUPED>
__host__ __device__ constexpr int bound_offsets() {
    return OBJ != 0 ? 4 : (BLOCK == 16 ? (GROUPED ? 2 : 1) : 6);
}

template <int OBJ, int BLOCK, bool GROUPED>
__device__ __forceinline__ int default_window_argmin(const u64 (&y2)[8], const u64 (&w2)[8], float ma, float mb,
                                                     const Cand* tb, float& best, bool wok = true) {
    constexpr int SEGS = BLOCK / 16;
    constexpr int FIX_LO = (OBJ == 0 && BLOCK == 16) ? -3 : -8;
    constexpr int FIX_K = 7 - FIX_LO + 1;
    constexpr int NB = bound_offsets<OBJ, BLOCK, GROUPED>();
    best = __int_as_float(0x7f800000);
    int bk = 0;
#pragma unroll
    for (int k = NB; k < FIX_K; k++) {
        const Cand cd = tb[k];
        const float L = group_sum<SEGS>(seg_loss<OBJ>(y2, w2, cd.r, (uint16_t)cd.nv));
        if (L < best) {
            best = L;
            bk = k;
        }
    }
    if (NB == 0) return bk;
    const u64 m2 = pack2(ma, mb);
    u64 wab = 0ull;
    if (OBJ == 1) {
        // the weight of an element of each half whose |y| is that half's max
        float wa = 0.0f, wb = 0.0f;
#pragma unroll
        for (int j = 0; j < 8; j++) {
            float a, b, w0, w1;
            unpack2(y2[j], a, b);
            unpack2(w2[j], w0, w1);
            float& wh = j < 4 ? wa : wb;
            const float mh = j < 4 ? ma : mb;
            wh = fabsf(a) == mh ? w0 : wh;
            wh = fabsf(b) == mh ? w1 : wh;
        }
        if (!wok) wa = __int_as_float(0x7fc00000);     // negative or NaN weights: no skip
        wab = pack2(wa, wb);
    }
#pragma unroll
    for (int k = NB - 1; k >= 0; k--) {
        const Cand cd = tb[k];
        const u64 e2 = cand_err2(m2, pack2(cd.r, cd.r), (uint16_t)cd.nv);
        const u64 t2 = OBJ == 1 ? mul2(mul2(wab, e2), e2) : mul2(e2, e2);
        float ta, tb2;
        unpack2(t2, ta, tb2);
        const float bound = __fmul_rn(group_sum<SEGS>(__fadd_rn(ta, tb2)), 0.99999904632568359375f);
        if (__all_sync(0xffffffffu, bound > best)) continue;                  // warp-uniform
        const float L = group_sum<SEGS>(seg_loss<OBJ>(y2, w2, cd.r, (uint16_t)cd.nv));
        if (L <= best) {
            best = L;
            bk = k;
        }
    }
    return bk;
}

// Whether all 16 weights of a segment are non-negative (NaN counts as not).
__device__ __forceinline__ bool weights_nonneg(const u64 (&w2)[8]) {
    float lo = __int_as_float(0x7f800000);
#pragma unroll
    for (int j = 0; j < 8; j++) {
        float a, b;
        unpack2(w2[j], a, b);
        asm("min.NaN.f32 %0, %1, %2, %3;" : "=f"(lo) : "f"(lo), "f"(a), "f"(b));
    }
    return lo >= 0.0f;
}

// n / d for 32-bit n by multiply-high and shifts (Granlund-Montgomery).
__device__ __forceinline__ uint32_t fast_div(uint32_t n, const FastDiv& d) {
    const uint32_t t = __umulhi(n, d.mul);
    return (t + ((n - t) >> d.s1)) >> d.s2;
}

#ifndef NVFP4_QMINB
#define NVFP4_QMINB 1
#endif


// Dynamic (per-call) global scale inside the sweep launch: every CTA folds the
// max |x| of its grid-stride share into one partial, all CTAs meet at a grid
// barrier (cooperative launch, so all are resident; the counter is zeroed by
// the host before the launch), then each CTA folds all partials into the same
// S = fl(amax / fl(6 D)).  The barrier wait is bounded by the global timer
// (1 s): on timeout the kernel sets bit 1 of the status word and returns
// without writing outputs.  p.wait_extra raises the arrival target (0 in every
// real call; the wait self-test uses it to make the wait run out).
constexpr unsigned long long kBarrierWaitNs = 1000000000ull;

__device__ __forceinline__ unsigned long long globaltimer_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ unsigned ld_acquire_u32(const unsigned* p) {
    unsigned v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

template <int DT>
__device__ __forceinline__ bool dynamic_scale(const QuantParams& p, float& S_out) {
    __shared__ uint32_t sm[32];
    __shared__ int sb[32];
    __shared__ int s_timeout;
    constexpr int PER = DT == 0 ? 8 : 4;
    const int64_t nvec = (p.nseg * 16) / PER;
    const uint4* xv = static_cast<const uint4*>(p.x);
    float m = 0.0f;
    int bad = 0;
    auto fold = [&](const uint4& u) {
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int j = 0; j < 4; j++) {
            if (DT == 0) {
                const float a = bf16lo(w[j]), b = bf16hi(w[j]);
                bad |= (!isfinite(a)) | (!isfinite(b));
                m = fmaxf(m, fmaxf(fabsf(a), fabsf(b)));
            } else {
                const float a = __uint_as_float(w[j]);
                bad |= !isfinite(a);
                m = fmaxf(m, fabsf(a));
            }
        }
    };
    const int64_t gstride = (int64_t)gridDim.x * blockDim.x;
    int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    for (; i + 7 * gstride < nvec; i += 8 * gstride) {      // eight 16-byte loads in flight per thread
        uint4 u[8];
#pragma unroll
        for (int j = 0; j < 8; j++) u[j] = ld_stream16(xv + i + j * gstride);
#pragma unroll
        for (int j = 0; j < 8; j++) fold(u[j]);
    }
    for (; i < nvec; i += gstride) fold(ld_stream16(xv + i));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
    uint32_t mb = __reduce_max_sync(0xffffffffu, __float_as_uint(m));
    int wb = __reduce_or_sync(0xffffffffu, (unsigned)bad);
    if (lane == 0) {
        sm[warp] = mb;
        sb[warp] = wb;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        uint32_t v = 0;
        int b = 0;
        for (int i = 0; i < nw; i++) {
            v = max(v, sm[i]);
            b |= sb[i];
        }
        p.part_max[blockIdx.x] = __uint_as_float(v);
        p.part_bad[blockIdx.x] = b;
        __threadfence();
        atomicAdd(p.barrier, 1u);
        const unsigned long long t0 = globaltimer_ns();
        int timeout = 0;
        while (ld_acquire_u32(p.barrier) < gridDim.x + p.wait_extra) {
            if (globaltimer_ns() - t0 > kBarrierWaitNs) {
                timeout = 1;
                break;
            }
            __nanosleep(128);
        }
        s_timeout = timeout;
    }
    __syncthreads();
    if (s_timeout) {
        if (threadIdx.x == 0 && p.status_dev) atomicOr(p.status_dev, 2);
        return false;
    }
    uint32_t v = 0;
    int b = 0;
    for (int i = threadIdx.x; i < (int)gridDim.x; i += blockDim.x) {
        v = max(v, __float_as_uint(__ldcg(p.part_max + i)));
        b |= __ldcg(p.part_bad + i);
    }
    v = __reduce_max_sync(0xffffffffu, v);
    b = __reduce_or_sync(0xffffffffu, (unsigned)b);
    __syncthreads();
    if (lane == 0) {
        sm[warp] = v;
        sb[warp] = b;
    }
    __syncthreads();
    uint32_t amaxb = 0;
    int anyb = 0;
    for (int i = 0; i < nw; i++) {
        amaxb = max(amaxb, sm[i]);
        anyb |= sb[i];
    }
    S_out = __fdiv_rn(__uint_as_float(amaxb), __fmul_rn(6.0f, p.fp8_div));
    if (blockIdx.x == 0 && threadIdx.x == 0) {
        p.S_out[0] = S_out;
        if (anyb && p.status_dev) atomicOr(p.status_dev, 1);
    }
    return true;
}

// FIX = 1: default window (fixed length, unrolled, poison-padded table).
// DYN = 1: the global scale is computed in this launch (see dynamic_scale).
// On bf16 input, AbsMax is held to 64 registers (4 CTAs per SM) and 4/6 to 80
// (3 CTAs per SM): both are issue- and latency-bound, not register-bound (AbsMax
// 0.0677 -> 0.0636 ms, 4/6 WMSE 0.120 -> 0.115 ms at 16384 x 8192; the
// fp32-input forms would spill, and the ScaleSweep sweeps run slower, at such bounds).
template <int METHOD, int DT>
constexpr int quantize_min_blocks() {
    return DT != 0 ? NVFP4_QMINB : (METHOD == 1 ? 4 : (METHOD == 2 ? 3 : NVFP4_QMINB));
}

template <int DT, int METHOD, int OBJ, int BLOCK, int FIX, int DYN>
__global__ void __launch_bounds__(256, quantize_min_blocks<METHOD, DT>()) quantize_kernel(QuantParams p) {
    constexpr int SEGS = BLOCK / 16;
    constexpr int FIX_LO = (OBJ == 0 && BLOCK == 16) ? -3 : -8;
    __shared__ Cand tab[kTabN];
    build_table(tab);
    __syncthreads();

    float S;
    if (DYN) {
        if (!dynamic_scale<DT>(p, S)) return;
    } else {
        S = __ldg(p.S);
    }
    float E = __frcp_rn(S);
    const bool usable = (S > 0.0f) && isfinite(S) && isfinite(E);
    if (!usable) E = 1.0f;                          // y = x: only signs (and sum w x^2) are emitted
    const u64 E2 = pack2(E, E);
    const int lane = threadIdx.x & 31;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const int64_t nseg_pad = (p.nseg + 31) & ~(int64_t)31;

    int64_t base = (int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31);
    Raw cur;
    if (base + lane < p.nseg) load_raw<DT>(p.x, base + lane, cur);

    for (; base < nseg_pad; base += stride) {
        const int64_t g = base + lane;
        const bool valid = g < p.nseg;
        Raw nxt;
        if (g + stride < p.nseg) load_raw<DT>(p.x, g + stride, nxt);

        u64 y2[8];
        float m = 0.0f, ma = 0.0f, mb = 0.0f;         // ma, mb: largest |y| of each half (offset bound)
        if (valid) {
            m = METHOD == 0 ? raw_to_y_halves<DT>(cur, E2, y2, ma, mb) : raw_to_y<DT>(cur, E2, y2);
        } else {
#pragma unroll
            for (int j = 0; j < 8; j++) y2[j] = 0ull;
        }
        m = group_max<SEGS>(m);
        cur = nxt;

        const int64_t blk = g / SEGS;               // scale-block index
        int64_t row = 0, kbi = 0;
        if (p.need_rowcol) {
            if (p.narrow) {
                const uint32_t b32 = (uint32_t)blk;
                const uint32_t r32 = fast_div(b32, p.kb_div);
                row = r32;
                kbi = b32 - r32 * (uint32_t)p.kb;
            } else {
                row = blk / p.kb;
                kbi = blk - row * p.kb;
            }
        }


        u64 w2[8];
        if (OBJ == 1) {
            const int64_t col = kbi * BLOCK + (int64_t)(g % SEGS) * 16;
            const float* wp = p.w + row * p.w_row_stride + col;
            if (valid) {
#pragma unroll
                for (int j = 0; j < 4; j++) {
                    const uint4 a = ld_ro16(wp + 4 * j);
                    w2[2 * j] = pack2(__uint_as_float(a.x), __uint_as_float(a.y));
                    w2[2 * j + 1] = pack2(__uint_as_float(a.z), __uint_as_float(a.w));
                }
            } else {
#pragma unroll
                for (int j = 0; j < 8; j++) w2[j] = 0ull;
            }
        }

        const bool zero = zero_block(usable, m);
        float best = __int_as_float(0x7f800000);
        int bestc = 0;
        if (METHOD == 0) {
            const float sbase = __fdiv_rn(m, 6.0f);
            const int I0 = e4m3_floor_code(sbase);
            if (FIX) {
                // the lane's weights are reloaded every segment, so their signs
                // are checked every segment too
                const Cand* tb = tab + (I0 + FIX_LO + kTabOff);
                bestc = I0 + FIX_LO + default_window_argmin<OBJ, BLOCK, false>(y2, w2, ma, mb, tb, best,
                                                                               OBJ == 0 || weights_nonneg(w2));
            } else {
                int lo_off = p.win_lo;
                if ((p.tight & 2) && I0 >= 16 && I0 <= 120) {
                    const int b = I0 & 7;                       // Table 2: ceil(4/5 s) is 2 or 3 codes down
                    lo_off = (b == 0 || b == 7) ? -3 : -2;
                }
                const int clo = min(max(I0 + lo_off, 1), 126);
                int chi = min(max(I0 + p.win_hi, 1), 126);
                if (p.tight & 1) {     // Lemma 4.1: 3.5 v_c > m never beats v_c / 2 = code c - 8 (c >= 16)
                    while (chi > clo && chi >= 16 &&
                           __fmul_rn(3.5f, f16bits_to_f32((uint16_t)(tab[chi + kTabOff].nv ^ 0x8000u))) > m)
                        chi--;
                }
                const int n = zero ? 0 : chi - clo + 1;
                const int nmax = __reduce_max_sync(0xffffffffu, (unsigned)n);
                bestc = clo;
                for (int k = 0; k < nmax; k++) {
                    const int c = min(clo + k, chi);    // repeats of chi never win the strict "<"
                    const Cand cd = tab[c + kTabOff];
                    const float L = group_sum<SEGS>(seg_loss<OBJ>(y2, w2, cd.r, (uint16_t)cd.nv));
                    if (L < best) {
                        best = L;
                        bestc = c;
                    }
                }
            }
        } else {
            const float sbase = __fdiv_rn(m, 6.0f);
            const int c6 = max((int)e4m3_rn_code(sbase), 1);
            bestc = c6;
            if (METHOD == 2) {
                const int c4 = max((int)e4m3_rn_code(__fdiv_rn(m, 4.0f)), 1);
                const Cand d6 = tab[c6 + kTabOff], d4 = tab[c4 + kTabOff];
                const float L6 = group_sum<SEGS>(seg_loss<OBJ>(y2, w2, d6.r, (uint16_t)d6.nv));
                const float L4 = group_sum<SEGS>(seg_loss<OBJ>(y2, w2, d4.r, (uint16_t)d4.nv));
                best = L6;
                if (L4 < L6) {
                    best = L4;
                    bestc = c4;
                }
            } else if (p.block_loss) {
                const Cand d6 = tab[c6 + kTabOff];
                best = group_sum<SEGS>(seg_loss<0>(y2, w2, d6.r, (uint16_t)d6.nv));
            }
        }

        // Emit packed nibbles for this thread's 16 elements.
        uint32_t packed[2];
        if (zero) {
#pragma unroll
            for (int h = 0; h < 2; h++) {
                uint32_t acc = 0;
#pragma unroll
                for (int j = 0; j < 4; j++) {
                    float a, b;
                    unpack2(y2[4 * h + j], a, b);
                    const uint32_t byte = (signbit(a) ? 0x08u : 0u) | (signbit(b) ? 0x80u : 0u);
                    acc |= byte << (8 * j);
                }
                packed[h] = acc;
            }
            bestc = 0;
            best = 0.0f;
            if (p.block_loss) {
                float s = 0.0f;
#pragma unroll
                for (int j = 0; j < 8; j++) {
                    float a, b;
                    unpack2(y2[j], a, b);
                    if (OBJ == 1) {
                        float wa, wb;
                        unpack2(w2[j], wa, wb);
                        s = __fmaf_rn(__fmul_rn(wa, a), a, s);
                        s = __fmaf_rn(__fmul_rn(wb, b), b, s);
                    } else {
                        s = __fmaf_rn(a, a, s);
                        s = __fmaf_rn(b, b, s);
                    }
                }
                best = group_sum<SEGS>(s);
            }
        } else {
            const float r = tab[bestc + kTabOff].r;
            const u64 r2 = pack2(r, r);
#pragma unroll
            for (int h = 0; h < 2; h++) {
                uint32_t b[4];
#pragma unroll
                for (int j = 0; j < 4; j++) {
                    float lo, hi;
                    unpack2(mul2(y2[4 * h + j], r2), lo, hi);
                    b[j] = e2m1x2(lo, hi);
                }
                packed[h] = b[0] | (b[1] << 8) | (b[2] << 16) | (b[3] << 24);
            }
        }

        if (valid) {
            *reinterpret_cast<uint2*>(p.codes + g * 8) = make_uint2(packed[0], packed[1]);
            if ((g % SEGS) == 0) {
                if (p.sf_linear) p.sf_linear[blk] = (uint8_t)bestc;
                if (p.sf_swizzled) p.sf_swizzled[swizzle_offset(row, kbi, p.kpad4)] = (uint8_t)bestc;
                if (p.block_loss) p.block_loss[blk] = best;
            }
        }
    }
}


}  // namespace nvfp4
