// Grouped ScaleSweep (Sec. 4.2.2, default windows) or AbsMax (Sec. 3.2) over a
// list of tensors in one launch, blocks of 16, 32 or 64 elements, with each
// tensor's global scale (Sec. 4.2.1, S = fl(amax / fl(6 D))) optionally
// reduced inside the same launch.
//
// Why: a transformer layer has tensors of very different sizes (k/v are 1/14
// of gate/up/down in Llama-3-8B).  One launch per tensor pays a ramp-down tail
// per launch and, with per-call scales, a separate amax launch per tensor.
// Here the segments of all tensors form one concatenated index space walked
// by one grid-stride loop (a single tail).
//
// Sweep (8 warps per CTA).  A CTA walks 256 consecutive segments per
// iteration; every tensor's segment range is padded to a multiple of 256, so
// the tensor index t is CTA-uniform and the descriptor fields are read as
// uniform kernel-parameter operands.  The per-segment sweep is the one of
// quantize_kernel (FIX = 1): y = fl(x E), I0 from fl(m/6), the 11 (MSE, block
// 16) or 16 candidates of the poison-padded table, lowest-code argmin, nibbles
// and both scale layouts; blocks of 32/64 are 2/4 lanes combined by
// xor-shuffles (a CTA's 256 segments always hold whole blocks).
//
// In-launch global scales, two schedules with bit-identical results.
//
// Two-phase (one cooperative launch).  Phase 1: every
// warp of the grid folds max |x| over its share of every tensor (16 loads in
// flight per lane, on the integer pipe: with the sign bit cleared the unsigned
// order of bf16/fp32 bit patterns is the order of the magnitudes) and
// publishes it with an atomicMax on the bit pattern.  A grid barrier (an
// acquire-release arrival count in the caller's workspace, zeroed by a
// memset before the launch; bounded by the global timer, 1 s, then status bit
// 1) separates it from phase 2, the sweep, which reads S[t] = fl(amax_t /
// fl(6 D)).  The reduction is HBM-bound and the sweep FP32-bound; running them
// one after the other keeps the sweep at 8 warps per CTA and the full
// register budget.  (A ninth, reduction-only warp per CTA that overlapped
// tensor t+1's reduction with tensor t's sweep capped every thread at 96
// registers and interfered with the sweep's loads; on the two 242M-element
// matrices of the Qwen2.5-72B shapes, where only half the data can overlap
// at all, it measured 1.674 ms against 1.409 ms for the sweep alone.)
//
// Pipelined (four launches, launch_group_pipelined).  The reduction runs as a
// separate kernel of 32-register threads, which the SM holds beside the sweep
// CTAs on the registers they leave free: the largest tensor is reduced, then
// swept while the other tensors are reduced beside it, then the others are
// swept.  Only the first reduction is exposed.  On the two Qwen2.5-72B-shaped
// matrices (WMSE, full-window sweep) 1.506-1.512 ms per call against
// 1.568-1.573 ms two-phase and 1.406-1.411 ms with static scales; on the
// Llama-3-8B layer 0.681 against 0.735 (static 0.643).
#include <atomic>

#include "group_kernels.h"
#include "quantize_kernel.cuh"

namespace nvfp4 {

namespace {

constexpr int kSweepThreads = 256;                          // sweep threads per CTA
constexpr int kAmaxInFlight = 16;                           // 16-byte loads in flight per reduction lane
constexpr int kReduceThreads = 128;                         // pipelined schedule: reduction CTA size
constexpr int kReduceInFlight = 4;                          // and its loads in flight per lane (32 registers)
constexpr unsigned long long kGroupWaitNs = 1000000000ull;   // give up a wait for a scale after 1 s
#ifndef NVFP4_GROUP_MINB
#define NVFP4_GROUP_MINB 2
#endif
#ifndef NVFP4_GROUP_MINB_MSE
#define NVFP4_GROUP_MINB_MSE 3
#endif
// Pipelined schedule: sweep CTAs per SM beside which the other tensors'
// reduction runs when those tensors hold more than half the first one's bytes.
// The MSE sweep could hold 3 CTAs per SM, which leaves the reduction one warp
// per scheduler: on the two Qwen2.5-72B-shaped matrices (MSE) that reduction
// then outlasts the sweep it should hide behind (0.964 ms per call against
// 0.890 ms with 2 CTAs); on K, V, Q (the rest is half of Q) 3 CTAs are faster
// (0.751 against 0.765-0.774 ms).
constexpr int kPipeSweepCtas = 2;

__device__ __forceinline__ unsigned long long global_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
__device__ __forceinline__ unsigned atom_add_acq_rel(unsigned* p, unsigned v) {
    unsigned old;
    asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
    return old;
}
__device__ __forceinline__ unsigned ld_relaxed_u32(const unsigned* p) {
    unsigned v;
    asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ uint32_t umax_u16x2(uint32_t a, uint32_t b) {
    uint32_t d;
    asm("max.u16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
    return d;
}

// Running max of |x| as bit patterns: with the sign bit cleared, the unsigned
// order of bf16 / fp32 patterns is the order of the magnitudes, inf above every
// finite value and NaN patterns above inf.  Integer ops keep this off the FMA
// pipe the sweep is bound by.  bf16: two u16 maxima per word.
template <int DT>
__device__ __forceinline__ uint32_t fold_vec(uint32_t m, const uint4& u) {
    if (DT == 0) {
        const uint32_t k = 0x7FFF7FFFu;
        return umax_u16x2(umax_u16x2(m, u.x & k), umax_u16x2(u.y & k, umax_u16x2(u.z & k, u.w & k)));
    }
    const uint32_t k = 0x7FFFFFFFu;
    return max(max(m, u.x & k), max(u.y & k, max(u.z & k, u.w & k)));
}

// max |x| over one reduction warp's share of a tensor with NaN skipped (as
// fmaxf does): the slow path, taken only when the share holds a NaN.
template <int DT>
__device__ __noinline__ float rescan_share(const uint4* xv, int64_t nvec, int64_t first, int64_t step) {
    float m = 0.0f;
    for (int64_t v = first; v < nvec; v += step) {
        const uint4 u = ld_stream16(xv + v);
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int k = 0; k < 4; k++) {
            if (DT == 0) m = fmaxf(m, fmaxf(fabsf(bf16lo(w[k])), fabsf(bf16hi(w[k]))));
            else m = fmaxf(m, fabsf(__uint_as_float(w[k])));
        }
    }
    return m;
}

// Phase 1 of a dynamic-scale launch: every warp of the grid folds max |x| over
// its share of every tensor (vector w*32 + lane + j*W*32 for warp w of W, 16
// loads in flight per lane) and publishes it with an atomicMax on the bit
// pattern; a share holding a NaN is rescanned with the NaN-skipping float
// max, so S matches the two-launch path bit for bit, and sets status bit 0
// for NaN/inf.  Each warp's atomics are fenced before the CTA arrives at the
// grid barrier.
template <int DT, int INFLIGHT, int THREADS = kSweepThreads>
__device__ __forceinline__ void reduce_all(const GroupParams& p) {
    const int lane = threadIdx.x & 31;
    const int64_t W = (int64_t)gridDim.x * (THREADS / 32);
    const int64_t w = (int64_t)blockIdx.x * (THREADS / 32) + (threadIdx.x >> 5);
    const int64_t step = W * 32, first = w * 32 + lane;
    bool any_bad = false;
    for (int a = 0; a < p.count; a++) {
        const uint4* xv = static_cast<const uint4*>(p.t[a].x);
        const int64_t nvec = p.t[a].nvec;
        uint32_t m = 0;
        int64_t v = first;
        for (; v + (INFLIGHT - 1) * step < nvec; v += INFLIGHT * step) {
            uint4 u[INFLIGHT];
#pragma unroll
            for (int i = 0; i < INFLIGHT; i++) u[i] = ld_stream16(xv + v + i * step);
#pragma unroll
            for (int i = 0; i < INFLIGHT; i++) m = fold_vec<DT>(m, u[i]);
        }
        for (; v < nvec; v += step) m = fold_vec<DT>(m, ld_stream16(xv + v));
        uint32_t mbits;
        bool nan, inf;
        if (DT == 0) {
            const uint32_t M = max(m & 0xFFFFu, m >> 16);
            nan = M > 0x7F80u;
            inf = M == 0x7F80u;
            mbits = M << 16;
        } else {
            nan = m > 0x7F800000u;
            inf = m == 0x7F800000u;
            mbits = m;
        }
        if (__any_sync(0xffffffffu, nan)) mbits = __float_as_uint(rescan_share<DT>(xv, nvec, first, step));
        const unsigned mb = __reduce_max_sync(0xffffffffu, mbits);
        any_bad |= __any_sync(0xffffffffu, nan || inf);
        if (lane == 0 && mb) atomicMax(p.amax_bits + a, mb);
    }
    if (lane == 0) {
        if (any_bad && p.status_dev) atomicOr(p.status_dev, 1);
        __threadfence();
    }
}

// Grid barrier between the two phases (cooperative launch: every CTA is
// resident, so the count always completes; the wait is bounded anyway by the
// global timer, 1 s, after which bit 1 of the status word is set and the
// launch returns without writing outputs).  p.wait_extra raises the target:
// 0 in every real call, the wait self-test uses it.
__device__ __forceinline__ bool grid_barrier(const GroupParams& p) {
    __shared__ int s_timeout;
    __syncthreads();
    if (threadIdx.x == 0) {
        atom_add_acq_rel(p.arrived, 1u);
        const unsigned long long t0 = global_ns();
        int timeout = 0;
        while (ld_acquire_u32(p.arrived) < gridDim.x + p.wait_extra) {
            if (global_ns() - t0 > kGroupWaitNs) {
                timeout = 1;
                break;
            }
            __nanosleep(128);
        }
        s_timeout = timeout;
        if (timeout && p.status_dev) atomicOr(p.status_dev, 2);
    }
    __syncthreads();
    return !s_timeout;
}

// Pipelined schedule of in-launch global scales: the reduction of one set of
// tensors as a kernel of its own, with 32 registers per thread so that it fits
// beside the sweep kernel's CTAs on an SM.  Every warp folds its share of
// every tensor of p (as phase 1 of the two-phase launch), then the last CTA to
// arrive (a ticket counter in the caller's workspace, zeroed before the
// launch) writes S[t] = fl(amax_t / fl(6 D)).  Nothing waits on another CTA.
// Launched as a programmatic dependent of a sweep kernel, the grid is
// scheduled once every CTA of that sweep is resident, reads only its own
// tensors, and ends with griddepcontrol.wait, so it completes (and the next
// sweep, which waits for it, starts) only after that sweep has completed.
template <int DT, int THREADS = kReduceThreads, int INFLIGHT = kReduceInFlight>
__global__ void __launch_bounds__(THREADS, 2048 / THREADS)
    group_reduce_kernel(const __grid_constant__ GroupParams p, unsigned* ticket) {
    reduce_all<DT, INFLIGHT, THREADS>(p);
    __syncthreads();                                 // every warp's atomics are fenced
    if (threadIdx.x == 0 && atom_add_acq_rel(ticket, 1u) == gridDim.x - 1) {
        for (int a = 0; a < p.count; a++)            // the last CTA sees every CTA's maxima
            p.S[p.t[a].s_index] =
                __fdiv_rn(__uint_as_float(ld_relaxed_u32(p.amax_bits + a)), __fmul_rn(6.0f, p.fp8_div));
    }
    grid_launch_dependents();
    grid_dependency_wait();
}

// One 16-element segment of the grid-stride loop: ScaleSweep (METHOD 0,
// default window) or AbsMax (METHOD 1) for a block of BLOCK elements, which is
// 1, 2 or 4 consecutive lanes (their maxima and losses combined by
// xor-shuffles, as in quantize_kernel).  WMSE weights of the lane's segment
// are kept in w2 across iterations and reloaded only when they come from
// another address (wkey): with a CTA stride that is a multiple of the
// tensor's segments per row a lane keeps its columns, so per-channel weights
// are loaded once per tensor.
template <int DT, int METHOD, int OBJ, int BLOCK>
__device__ __forceinline__ void sweep_segments(const GroupTensor& d, const Cand* tab, const Raw& cur, int64_t g,
                                               bool valid, u64 E2, bool usable, u64 (&w2)[8], const float*& wkey,
                                               bool& wok) {
    constexpr int SEGS = BLOCK / 16;
    constexpr int FIX_LO = (OBJ == 0 && BLOCK == 16) ? -3 : -8;
    u64 y2[8];
    float m = 0.0f, ma = 0.0f, mb = 0.0f;               // ma, mb: largest |y| of each half (offset bound)
    if (valid) {
        m = METHOD == 0 ? raw_to_y_halves<DT>(cur, E2, y2, ma, mb) : raw_to_y<DT>(cur, E2, y2);
    } else {
#pragma unroll
        for (int j = 0; j < 8; j++) y2[j] = 0ull;
    }
    m = group_max<SEGS>(m);
    const int64_t blk = g / SEGS;                           // scale-block index (g >= 0: a shift)
    auto row_col = [&](int64_t& row, int64_t& kbi) {
        if (d.narrow) {
            const uint32_t b32 = (uint32_t)blk;
            const uint32_t r32 = fast_div(b32, d.kb_div);
            row = r32;
            kbi = b32 - r32 * (uint32_t)d.kb;
        } else {
            row = blk / d.kb;
            kbi = blk - row * d.kb;
        }
    };
    if (METHOD == 0 && OBJ == 1) {
        int64_t row, kbi;
        row_col(row, kbi);
        const float* wp = d.w + row * d.w_row_stride + kbi * BLOCK + (g % SEGS) * 16;
        if (valid && wp != wkey) {
#pragma unroll
            for (int j = 0; j < 4; j++) {
                const uint4 a = ld_ro16(wp + 4 * j);
                w2[2 * j] = pack2(__uint_as_float(a.x), __uint_as_float(a.y));
                w2[2 * j + 1] = pack2(__uint_as_float(a.z), __uint_as_float(a.w));
            }
            wkey = wp;
            wok = weights_nonneg(w2);
        }
    }
    const bool zero = zero_block(usable, m);
    int bestc;
    if (METHOD == 0) {
        float best;
        const int I0 = e4m3_floor_code(__fdiv_rn(m, 6.0f));
        const Cand* tb = tab + (I0 + FIX_LO + kTabOff);
        bestc = I0 + FIX_LO + default_window_argmin<OBJ, BLOCK, true>(y2, w2, ma, mb, tb, best, wok);
    } else {
        bestc = max((int)e4m3_rn_code(__fdiv_rn(m, 6.0f)), 1);
    }
    uint32_t packed[2];
    if (zero) {
#pragma unroll
        for (int h = 0; h < 2; h++) {
            uint32_t acc = 0;
#pragma unroll
            for (int j = 0; j < 4; j++) {
                float a, b;
                unpack2(y2[4 * h + j], a, b);
                acc |= ((signbit(a) ? 0x08u : 0u) | (signbit(b) ? 0x80u : 0u)) << (8 * j);
            }
            packed[h] = acc;
        }
        bestc = 0;
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
        *reinterpret_cast<uint2*>(d.codes + g * 8) = make_uint2(packed[0], packed[1]);
        if ((g % SEGS) == 0) {
            if (d.sf_linear) d.sf_linear[blk] = (uint8_t)bestc;
            if (BLOCK == 16 && d.sf_swizzled) {
                int64_t row, kbi;                               // recomputed here: not live across the sweep
                row_col(row, kbi);
                d.sf_swizzled[swizzle_offset(row, kbi, d.kpad4)] = (uint8_t)bestc;
            }
        }
    }
}

// Index of the tensor whose padded segment range holds `seg`, searching
// forward from `t` (segment indices only grow along the loop).  With a
// CTA-uniform `seg` the result is CTA-uniform, so the descriptor fields read
// with it are uniform operands.
__device__ __forceinline__ int tensor_at(const GroupParams& p, int t, int64_t seg) {
    while (t + 1 < p.count && seg >= p.t[t + 1].seg_begin) t++;
    return t;
}

// DYN = 0: static scales read from p.S.  DYN = 1: the scales are reduced in
// the launch first (phase 1, every warp, HBM-bound), then every CTA meets at
// a grid barrier and sweeps with the same 8 warps (phase 2, FP32-bound).
// AbsMax is HBM-bound in both phases: it is held to 64 registers (4 CTAs per
// SM, 8 loads in flight per lane in phase 1) for more loads in flight.
// DYN = 2: the pipelined schedule's sweep, scales from the reduction grid
// launched before it.
template <int METHOD, int OBJ>
constexpr int group_min_blocks() {
    return METHOD == 1 ? 4 : (OBJ == 0 ? NVFP4_GROUP_MINB_MSE : NVFP4_GROUP_MINB);
}

template <int DT, int METHOD, int OBJ, int BLOCK, int DYN>
__global__ void __launch_bounds__(kSweepThreads, group_min_blocks<METHOD, OBJ>())
    quantize_group_kernel(const __grid_constant__ GroupParams p) {
    constexpr int SW = kSweepThreads;
    static_assert(SW == kGroupCtaSegments, "host padding unit");
    __shared__ Cand tab[kTabN];
    build_table(tab);
    if (DYN == 1) {
        reduce_all<DT, METHOD == 1 ? 8 : kAmaxInFlight>(p);
        if (!grid_barrier(p)) return;
        if (blockIdx.x == 0 && (int)threadIdx.x < p.count)        // publish every tensor's S once
            p.S[p.t[threadIdx.x].s_index] =
                __fdiv_rn(__uint_as_float(ld_relaxed_u32(p.amax_bits + threadIdx.x)), __fmul_rn(6.0f, p.fp8_div));
    } else if (DYN == 2) {
        // pipelined schedule: the scales come from the reduction grid launched
        // before this one; once every CTA is resident the next reduction grid
        // may be scheduled beside it
        grid_dependency_wait();
        grid_launch_dependents();
    }
    __syncthreads();

    const int count = p.count;
    const int tid = threadIdx.x;
    const int64_t stride = (int64_t)gridDim.x * SW;
    const int64_t total = p.total_seg;
    int64_t cbase = (int64_t)blockIdx.x * SW;
    int t = tensor_at(p, 0, cbase);

    u64 w2[8];                                           // an invalid lane's losses ignore w2
#pragma unroll
    for (int j = 0; j < 8; j++) w2[j] = 0ull;
    const float* wkey = nullptr;
    bool wok = true;                                     // the lane's weights are all >= 0
    Raw cur;
    if (cbase < total) {
        const int64_t g = cbase + tid - p.t[t].seg_begin;
        if (g < p.t[t].nseg) load_raw<DT>(p.t[t].x, g, cur);
    }

    while (cbase < total) {
        // entering tensor t: its global scale
        const float S =
            DYN == 1 ? __fdiv_rn(__uint_as_float(ld_relaxed_u32(p.amax_bits + t)), __fmul_rn(6.0f, p.fp8_div))
            : DYN == 2 ? __uint_as_float(ld_relaxed_u32(reinterpret_cast<const unsigned*>(p.S + p.t[t].s_index)))
                       : __ldg(p.S + p.t[t].s_index);
        float E = __frcp_rn(S);
        const bool usable = (S > 0.0f) && isfinite(S) && isfinite(E);
        if (!usable) E = 1.0f;
        const u64 E2 = pack2(E, E);
        const int64_t seg_end = t + 1 < count ? p.t[t + 1].seg_begin : total;

        for (; cbase < seg_end; cbase += stride) {
            const GroupTensor& d = p.t[t];
            const int64_t g = cbase + tid - d.seg_begin;
            const bool valid = g < d.nseg;
            Raw nxt;
            const int64_t nb = cbase + stride;
            if (nb < seg_end) {
                if (g + stride < d.nseg) load_raw<DT>(d.x, g + stride, nxt);
            } else if (nb < total) {
                const int tn = tensor_at(p, t, nb);
                const int64_t gn = nb + tid - p.t[tn].seg_begin;
                if (gn < p.t[tn].nseg) load_raw<DT>(p.t[tn].x, gn, nxt);
            }
            sweep_segments<DT, METHOD, OBJ, BLOCK>(d, tab, cur, g, valid, E2, usable, w2, wkey, wok);
            cur = nxt;
        }
        t = tensor_at(p, t, cbase);
    }
}

}  // namespace

namespace {

// Resident sweep CTAs per SM and the grid of one sweep launch over p: the
// whole segment space, capped at the resident maximum (every wait can then
// complete); for WMSE up to 1/32 fewer CTAs if that makes the CTA stride a
// multiple of more tensors' segments per row (lanes then keep their weights).
template <int DT, int METHOD, int OBJ, int BLOCK, int DYN>
int64_t sweep_grid(const GroupParams& p, int sms, int* per_sm, int max_per_sm = 0) {
    constexpr int SW = kSweepThreads;
    constexpr int SEGS = BLOCK / 16;
    static std::atomic<int> occ_cache[kOccDevices];
    int occ = occupancy_per_sm(occ_cache, quantize_group_kernel<DT, METHOD, OBJ, BLOCK, DYN>, SW);
    if (max_per_sm > 0 && occ > max_per_sm) occ = max_per_sm;
    if (per_sm) *per_sm = occ;
    const int64_t cap = (int64_t)sms * occ;
    int64_t grid = (p.total_seg + SW - 1) / SW;
    if (grid > cap) {
        grid = cap;
        if (METHOD == 0 && OBJ == 1) {
            auto covered = [&](int64_t g) {
                int64_t c = 0;
                for (int i = 0; i < p.count; i++)
                    if (p.t[i].w_row_stride == 0 && p.t[i].kb > 0 && (g * SW) % (p.t[i].kb * SEGS) == 0)
                        c += p.t[i].nseg;
                return c;
            };
            int64_t best = grid, best_c = covered(grid);
            for (int64_t g = grid - 1; g >= grid - grid / 32 && g >= 1; g--) {
                const int64_t c = covered(g);
                if (c > best_c) {
                    best = g;
                    best_c = c;
                }
            }
            grid = best;
        }
    }
    return grid < 1 ? 1 : grid;
}

template <int DT, int METHOD, int OBJ, int BLOCK, int DYN>
cudaError_t launch_group(const GroupParams& p, int sms, cudaStream_t s) {
    const int64_t grid = sweep_grid<DT, METHOD, OBJ, BLOCK, DYN>(p, sms, nullptr);
    if (DYN) {
        cudaError_t e = cudaMemsetAsync(p.amax_bits, 0, kGroupWorkspace, s);
        if (e != cudaSuccess) return e;
        void* args[] = {(void*)&p};
        return cudaLaunchCooperativeKernel((const void*)quantize_group_kernel<DT, METHOD, OBJ, BLOCK, 1>,
                                           dim3((unsigned)grid), dim3(kSweepThreads), args, 0, s);
    }
    quantize_group_kernel<DT, METHOD, OBJ, BLOCK, 0><<<(unsigned)grid, kSweepThreads, 0, s>>>(p);
    return cudaGetLastError();
}

// Launch of `kernel` on `s` as a programmatic dependent of the kernel before
// it on the stream.
template <typename... Args>
cudaError_t launch_dependent(void (*kernel)(Args...), int64_t grid, int threads, cudaStream_t s, Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3((unsigned)threads);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// The tensors p.t[first..last) as a group of their own (segment space from 0,
// global-scale slots of the workspace from amax_slot).
GroupParams subgroup(const GroupParams& p, int first, int last, int amax_slot) {
    GroupParams q = p;
    q.count = last - first;
    int64_t seg = 0;
    for (int k = 0; k < q.count; k++) {
        q.t[k] = p.t[first + k];
        q.t[k].seg_begin = seg;
        seg += (q.t[k].nseg + kGroupCtaSegments - 1) / kGroupCtaSegments * kGroupCtaSegments;
    }
    q.total_seg = seg;
    q.amax_bits = p.amax_bits + amax_slot;
    return q;
}

// Pipelined schedule of in-launch global scales (p.count >= 2).  The last
// tensor of p (the largest: p is in ascending size) goes first:
//   reduce(last)  full GPU, ordinary launch;
//   sweep(last)   waits for it, then lets the next grid be scheduled; at most
//                 kPipeSweepCtas CTAs per SM when the rest is over half its size;
//   reduce(rest)  co-resident with sweep(last) on the registers the sweep
//                 leaves free (32 per thread), completes after it;
//   sweep(rest)   one grouped sweep of the other tensors, waits for reduce(rest).
// The three later grids are programmatic dependent launches, so no CTA waits
// on a flag and each grid waits only for the one launched just before it.
// Only the first tensor's reduction stays exposed: the others overlap a sweep
// bound by the FP32 pipe, not by HBM.
template <int DT, int METHOD, int OBJ, int BLOCK>
cudaError_t launch_group_pipelined(const GroupParams& p, int sms, cudaStream_t s) {
    const GroupParams a = subgroup(p, p.count - 1, p.count, 0);
    const GroupParams b = subgroup(p, 0, p.count - 1, 1);
    unsigned* ticket = p.arrived;
    cudaError_t e = cudaMemsetAsync(p.amax_bits, 0, kGroupWorkspace, s);
    if (e != cudaSuccess) return e;
    // the first reduction has the GPU to itself: 512-thread CTAs, 4 per SM, 8
    // loads in flight per lane (0.2-0.4% faster steps than the 128-thread form)
    group_reduce_kernel<DT, 512, 8><<<(unsigned)sms * 4, 512, 0, s>>>(a, ticket);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    int occ = 1;
    const bool big_rest = b.total_seg > a.total_seg / 2;
    const int64_t grid_a = sweep_grid<DT, METHOD, OBJ, BLOCK, 2>(a, sms, &occ, big_rest ? kPipeSweepCtas : 0);
    e = launch_dependent(quantize_group_kernel<DT, METHOD, OBJ, BLOCK, 2>, grid_a, kSweepThreads, s, a);
    if (e != cudaSuccess) return e;
    // reduction CTAs that fit beside `occ` sweep CTAs per SM: each of its warps
    // takes 32 x 32 registers on one of the four schedulers' 16K-register files
    static std::atomic<int> regs_cache[kOccDevices];
    int dev = -1, regs = 0;
    if (cudaGetDevice(&dev) == cudaSuccess && dev >= 0 && dev < kOccDevices)
        regs = regs_cache[dev].load(std::memory_order_relaxed);
    if (regs <= 0) {
        cudaFuncAttributes fa;
        e = cudaFuncGetAttributes(&fa, quantize_group_kernel<DT, METHOD, OBJ, BLOCK, 2>);
        if (e != cudaSuccess) return e;
        regs = fa.numRegs;
        if (dev >= 0 && dev < kOccDevices) regs_cache[dev].store(regs, std::memory_order_relaxed);
    }
    const int warp_regs = (regs + 7) / 8 * 8 * 32;
    const int sweep_warps_per_sched = (occ * (kSweepThreads / 32) + 3) / 4;
    const int free_per_sched = 16384 - sweep_warps_per_sched * warp_regs;
    int per_sm = free_per_sched / (32 * 32) / (kReduceThreads / 32 / 4);
    per_sm = per_sm < 1 ? 1 : (per_sm > 2048 / kReduceThreads ? 2048 / kReduceThreads : per_sm);

    e = launch_dependent(group_reduce_kernel<DT>, (int64_t)sms * per_sm, kReduceThreads, s, b, ticket + 1);
    if (e != cudaSuccess) return e;
    const int64_t grid_b = sweep_grid<DT, METHOD, OBJ, BLOCK, 2>(b, sms, nullptr);
    return launch_dependent(quantize_group_kernel<DT, METHOD, OBJ, BLOCK, 2>, grid_b, kSweepThreads, s, b);
}

template <int DT, int METHOD, int OBJ, int BLOCK>
cudaError_t launch_schedule(const GroupParams& p, int sms, cudaStream_t s) {
    if (!p.dyn) return launch_group<DT, METHOD, OBJ, BLOCK, 0>(p, sms, s);
    if (p.pipelined && METHOD == 0 && p.count >= 2) return launch_group_pipelined<DT, METHOD, OBJ, BLOCK>(p, sms, s);
    return launch_group<DT, METHOD, OBJ, BLOCK, 1>(p, sms, s);
}

template <int DT, int METHOD, int OBJ>
cudaError_t launch_block(const GroupParams& p, int block, int sms, cudaStream_t s) {
    switch (block) {
        case 16: return launch_schedule<DT, METHOD, OBJ, 16>(p, sms, s);
        case 32: return launch_schedule<DT, METHOD, OBJ, 32>(p, sms, s);
        default: return launch_schedule<DT, METHOD, OBJ, 64>(p, sms, s);
    }
}

template <int DT>
cudaError_t launch_method(const GroupParams& p, int method, int obj, int block, int sms, cudaStream_t s) {
    if (method == 1) return launch_block<DT, 1, 0>(p, block, sms, s);
    return obj == 1 ? launch_block<DT, 0, 1>(p, block, sms, s) : launch_block<DT, 0, 0>(p, block, sms, s);
}

}  // namespace

cudaError_t launch_quantize_group(const GroupParams& p, const int64_t* rows, int dtype, int method, int obj,
                                  int block, int sms, cudaStream_t s) {
    cudaError_t e = cudaSuccess;
    if (p.total_seg > 0 || p.dyn) {
        e = dtype == 0 ? launch_method<0>(p, method, obj, block, sms, s) : launch_method<1>(p, method, obj, block, sms, s);
        if (e != cudaSuccess) return e;
    }
    for (int i = 0; i < p.count; i++) {
        const GroupTensor& T = p.t[i];
        if (!T.sf_swizzled) continue;
        QuantParams q{};
        q.sf_swizzled = T.sf_swizzled;
        q.rows = rows[i];
        q.kb = T.kb;
        q.kpad4 = T.kpad4;
        e = launch_swizzle_pad(q, sms, s);
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

}  // namespace nvfp4
