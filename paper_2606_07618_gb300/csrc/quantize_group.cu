// Grouped ScaleSweep (Sec. 4.2.2, default windows) or AbsMax (Sec. 3.2) over a
// list of tensors in one launch, blocks of 16, 32 or 64 elements, with each
// tensor's global scale (Sec. 4.2.1, S = fl(amax / fl(6 D))) optionally
// reduced inside the same launch.
//
// Why: a transformer layer has tensors of very different sizes (k/v are 1/14
// of gate/up/down in Llama-3-8B).  One launch per tensor pays a ramp-down tail
// per launch, and the HBM-bound amax pass of each tensor either runs before
// its ALU-bound sweep or competes with it from a second stream.  Here the
// segments of all tensors form one concatenated index space walked by one
// grid-stride loop (a single tail), and the amax reductions run beside the
// sweep inside the same launch.
//
// Sweep warps (8 per CTA).  A CTA walks 256 consecutive segments per
// iteration; every tensor's segment range is padded to a multiple of 256, so
// the tensor index t is CTA-uniform and the descriptor fields are read as
// uniform kernel-parameter operands.  The per-segment sweep is the one of
// quantize_kernel (FIX = 1): y = fl(x E), I0 from fl(m/6), the 11 (MSE, block
// 16) or 16 candidates of the poison-padded table, lowest-code argmin, nibbles
// and both scale layouts; blocks of 32/64 are 2/4 lanes combined by
// xor-shuffles (a CTA's 256 segments always hold whole blocks).
//
// Reduction warp (a ninth warp per CTA, dynamic scales only).  The reduction
// warps of the grid split every tensor's 16-byte input vectors round-robin
// (vector aw*32 + lane + j*NA*32 for reduction warp aw of NA) and walk the
// tensors in processing order, 16 loads in flight per lane, folding max |x| on
// the integer pipe.  Finishing a tensor a, a reduction warp folds its maximum
// into amax_bits[a] (atomicMax on the bit pattern of a non-negative float) and
// counts itself in arrived[a] (acquire-release); the last to arrive writes
// S[a].  A sweep warp entering tensor t waits until all NA reduction warps
// have arrived for t.  Reduction warps never wait, and the grid is resident
// (cooperative launch), so every wait ends; each is bounded anyway by the
// global timer (1 s; status bit 1, the warp stops).  p.wait_extra raises the
// arrival target: 0 in every real call, the wait self-test uses it.  Tensors are processed in ascending size, so the first
// reduction, the only one no sweep hides, is the smallest.
#include <atomic>

#include "group_kernels.h"
#include "quantize_kernel.cuh"

namespace nvfp4 {

namespace {

constexpr int kSweepThreads = 256;                          // sweep threads per CTA
constexpr int kAmaxInFlight = 16;                           // 16-byte loads in flight per reduction lane
constexpr unsigned long long kGroupWaitNs = 1000000000ull;   // give up a wait for a scale after 1 s
#ifndef NVFP4_GROUP_MINB
#define NVFP4_GROUP_MINB 2
#endif

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

template <int DT>
__device__ __forceinline__ void publish_max(const GroupParams& p, int a, uint32_t m, const uint4* xv, int64_t nvec,
                                            int64_t first, int64_t step, int lane) {
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
    const bool bad = __any_sync(0xffffffffu, nan || inf);
    if (lane == 0) {
        if (mb) atomicMax(p.amax_bits + a, mb);
        if (bad && p.status_dev) atomicOr(p.status_dev, 1);
        const unsigned old = atom_add_acq_rel(p.arrived + a, 1u);
        if (old == gridDim.x - 1) {
            const float amax = __uint_as_float(ld_relaxed_u32(p.amax_bits + a));
            p.S[p.t[a].s_index] = __fdiv_rn(amax, __fmul_rn(6.0f, p.fp8_div));
        }
    }
}

// One reduction warp (aw = blockIdx.x of NA = gridDim.x): its share of every
// tensor, in processing order, vector aw*32 + lane + j*NA*32 for round j.
template <int DT>
__device__ __forceinline__ void reduce_warp(const GroupParams& p, int lane) {
    const int64_t aw = blockIdx.x, step = (int64_t)gridDim.x * 32, first = aw * 32 + lane;
    for (int a = 0; a < p.count; a++) {
        const uint4* xv = static_cast<const uint4*>(p.t[a].x);
        const int64_t nvec = p.t[a].nvec;
        uint32_t m = 0;
        int64_t v = first;
        for (; v + (kAmaxInFlight - 1) * step < nvec; v += kAmaxInFlight * step) {
            uint4 u[kAmaxInFlight];
#pragma unroll
            for (int i = 0; i < kAmaxInFlight; i++) u[i] = ld_stream16(xv + v + i * step);
#pragma unroll
            for (int i = 0; i < kAmaxInFlight; i++) m = fold_vec<DT>(m, u[i]);
        }
        for (; v < nvec; v += step) m = fold_vec<DT>(m, ld_stream16(xv + v));
        publish_max<DT>(p, a, m, xv, nvec, first, step, lane);
    }
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
                                               bool valid, u64 E2, bool usable, u64 (&w2)[8], const float*& wkey) {
    constexpr int SEGS = BLOCK / 16;
    constexpr int FIX_LO = (OBJ == 0 && BLOCK == 16) ? -3 : -8;
    constexpr int FIX_K = 7 - FIX_LO + 1;
    u64 y2[8];
    float m = 0.0f;
    if (valid) {
        m = raw_to_y<DT>(cur, E2, y2);
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
        }
    }
    const bool zero = zero_block(usable, m);
    int bestc;
    if (METHOD == 0) {
        float best = __int_as_float(0x7f800000);
        const int I0 = e4m3_floor_code(__fdiv_rn(m, 6.0f));
        const Cand* tb = tab + (I0 + FIX_LO + kTabOff);
        int bk = 0;
#pragma unroll
        for (int k = 0; k < FIX_K; k++) {
            const Cand cd = tb[k];
            const float L = group_sum<SEGS>(seg_loss<OBJ>(y2, w2, cd.r, (uint16_t)cd.nv));
            if (L < best) {
                best = L;
                bk = k;
            }
        }
        bestc = I0 + FIX_LO + bk;
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

// DYN = 0: static scales read from p.S, 8 sweep warps per CTA; DYN = 1:
// scales reduced in the launch by a ninth warp per CTA.  (Nine warps cap the
// registers at 96 per thread -- two CTAs put five warps on two schedulers --
// which measured faster than seven sweep warps plus one reduction warp.)
template <int DT, int METHOD, int OBJ, int BLOCK, int DYN>
__global__ void __launch_bounds__(DYN ? kSweepThreads + 32 : kSweepThreads, NVFP4_GROUP_MINB)
    quantize_group_kernel(const __grid_constant__ GroupParams p) {
    constexpr int SW = kSweepThreads;
    static_assert(SW == kGroupCtaSegments, "host padding unit");
    __shared__ Cand tab[kTabN];
    build_table(tab);
    __syncthreads();
    if (DYN && threadIdx.x >= SW) {
        reduce_warp<DT>(p, threadIdx.x & 31);
        return;
    }

    const int count = p.count;
    const int tid = threadIdx.x, lane = tid & 31;
    const int64_t stride = (int64_t)gridDim.x * SW;
    const int64_t total = p.total_seg;
    int64_t cbase = (int64_t)blockIdx.x * SW;
    int t = tensor_at(p, 0, cbase);

    u64 w2[8];                                           // an invalid lane's losses ignore w2
#pragma unroll
    for (int j = 0; j < 8; j++) w2[j] = 0ull;
    const float* wkey = nullptr;
    Raw cur;
    if (cbase < total) {
        const int64_t g = cbase + tid - p.t[t].seg_begin;
        if (g < p.t[t].nseg) load_raw<DT>(p.t[t].x, g, cur);
    }

    while (cbase < total) {
        // entering tensor t: its global scale (dynamic: once every reduction
        // warp has arrived for t)
        float S;
        if (DYN) {
            int timeout = 0;
            if (lane == 0) {
                const unsigned long long t0 = global_ns();
                while (ld_acquire_u32(p.arrived + t) < gridDim.x + p.wait_extra) {
                    if (global_ns() - t0 > kGroupWaitNs) {
                        timeout = 1;
                        break;
                    }
                    __nanosleep(128);
                }
            }
            if (__shfl_sync(0xffffffffu, timeout, 0)) {
                if (lane == 0 && p.status_dev) atomicOr(p.status_dev, 2);
                return;
            }
            S = __fdiv_rn(__uint_as_float(ld_relaxed_u32(p.amax_bits + t)), __fmul_rn(6.0f, p.fp8_div));
        } else {
            S = __ldg(p.S + p.t[t].s_index);
        }
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
            sweep_segments<DT, METHOD, OBJ, BLOCK>(d, tab, cur, g, valid, E2, usable, w2, wkey);
            cur = nxt;
        }
        t = tensor_at(p, t, cbase);
    }
}

}  // namespace

namespace {

template <int DT, int METHOD, int OBJ, int BLOCK, int DYN>
cudaError_t launch_group(const GroupParams& p, int sms, cudaStream_t s) {
    constexpr int SW = kSweepThreads, threads = DYN ? kSweepThreads + 32 : kSweepThreads;
    constexpr int SEGS = BLOCK / 16;
    static std::atomic<int> occ_cache[kOccDevices];
    const int64_t cap = (int64_t)sms *
                        occupancy_per_sm(occ_cache, quantize_group_kernel<DT, METHOD, OBJ, BLOCK, DYN>, threads);
    int64_t grid = (p.total_seg + SW - 1) / SW;
    if (grid > cap) {
        grid = cap;                                              // resident grid: every wait can complete
        if (METHOD == 0 && OBJ == 1) {
            // Up to 1/32 fewer CTAs if that makes the CTA stride a multiple of
            // more tensors' segments per row (lanes then keep their weights).
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
    if (grid < 1) grid = 1;
    if (DYN) {
        cudaError_t e = cudaMemsetAsync(p.amax_bits, 0, kGroupWorkspace, s);
        if (e != cudaSuccess) return e;
        void* args[] = {(void*)&p};
        return cudaLaunchCooperativeKernel((const void*)quantize_group_kernel<DT, METHOD, OBJ, BLOCK, 1>,
                                           dim3((unsigned)grid), dim3(threads), args, 0, s);
    }
    quantize_group_kernel<DT, METHOD, OBJ, BLOCK, 0><<<(unsigned)grid, threads, 0, s>>>(p);
    return cudaGetLastError();
}

template <int DT, int METHOD, int OBJ, int BLOCK>
cudaError_t launch_dyn_or_static(const GroupParams& p, int sms, cudaStream_t s) {
    return p.dyn ? launch_group<DT, METHOD, OBJ, BLOCK, 1>(p, sms, s) : launch_group<DT, METHOD, OBJ, BLOCK, 0>(p, sms, s);
}

template <int DT, int METHOD, int OBJ>
cudaError_t launch_block(const GroupParams& p, int block, int sms, cudaStream_t s) {
    switch (block) {
        case 16: return launch_dyn_or_static<DT, METHOD, OBJ, 16>(p, sms, s);
        case 32: return launch_dyn_or_static<DT, METHOD, OBJ, 32>(p, sms, s);
        default: return launch_dyn_or_static<DT, METHOD, OBJ, 64>(p, sms, s);
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
