// Optimal real-valued block scale (Appendix C of the ScaleSweep paper) and the
// FP8-quantised optimal scale, per block, on the GPU.  Analysis kernels: they
// measure how far AbsMax, 4/6 and ScaleSweep are from the best possible FP32
// block scale (the paper's Figs. 1 and 4), not part of the quantisation path.
//
// In the S-normalised domain (a_i = |fl(x_i * fl(1/S))|, weights w_i) the loss
// L(s) = sum_i w_i (a_i - s g_i(s))^2, g_i(s) = RN_E2M1(a_i / s), is piecewise
// quadratic with breakpoints b = a_i / mu_k (mu_k the 7 midpoints of the E2M1
// grid); on the segment just above a breakpoint every g_i is fixed, the segment's
// quadratic A - 2Bs + Cs^2 is minimised at s* = B/C, and its value there is
// sum_i w_i (a_i - s* g_i)^2.  For any fixed assignment that value is an upper
// bound on L(s*) (per-element rounding can only do better), and for the segment
// holding the global minimum it is the minimum itself, so the minimum over all
// segments' values is min_s L(s) -- no sorting of breakpoints is needed.  The
// assignment above breakpoint (i, k) gives element i the lower neighbour of mu_k
// and every other element the grid point nearest to a_j / b, with quotients at
// or within ~1e-6 (relative) of a midpoint sent to the lower neighbour -- the
// segment just above b also when breakpoints coincide (equal magnitudes); only
// segments narrower than ~1e-6 relative can be skipped, and their neighbours,
// which share their endpoints, are enumerated.
//
// The minimum can be attained at several scales; the smallest is reported.
// FP8-quantised optimum: the better of floor_E4M3(s*) and ceil_E4M3(s*) (ties
// to the floor), each scored with the sweep's arithmetic contract.
#include "nvfp4_device.cuh"
#include "nvfp4_kernels.h"

namespace nvfp4 {

__constant__ float kMid[7] = {0.25f, 0.75f, 1.25f, 1.75f, 2.5f, 3.5f, 5.0f};
__constant__ float kGrid[8] = {0.0f, 0.5f, 1.0f, 1.5f, 2.0f, 3.0f, 4.0f, 6.0f};

// Nearest E2M1 magnitude of t >= 0 (ties to even), as a float.
__device__ __forceinline__ float rn_grid(float t) {
    const uint32_t code = e2m1x2(t, 0.0f) & 0x7u;
    const float g[8] = {0.0f, 0.5f, 1.0f, 1.5f, 2.0f, 3.0f, 4.0f, 6.0f};
    float r = 0.0f;
#pragma unroll
    for (int k = 0; k < 8; k++) r = (code == (uint32_t)k) ? g[k] : r;
    return r;
}

// Loss of E4M3 scale code c under the sweep's contract (t = fl(y*fl(1/v)),
// q = RNE_E2M1(t), e = fl(y - q*v), fp32 accumulation in element order).
template <int BLOCK, int OBJ>
__device__ float contract_loss(const float (&y)[BLOCK], const float (&w)[BLOCK], int c) {
    const uint16_t vh = e4m3_to_f16bits((uint32_t)c);
    const float v = f16bits_to_f32(vh);
    const float r = __frcp_rn(v);
    float L = 0.0f;
#pragma unroll
    for (int i = 0; i < BLOCK; i++) {
        const float t = __fmul_rn(y[i], r);
        const float q = copysignf(rn_grid(fabsf(t)), t);
        const float e = __fmaf_rn(-q, v, y[i]);
        L = __fmaf_rn(OBJ ? __fmul_rn(w[i], e) : e, e, L);
    }
    return L;
}

template <int DT, int OBJ, int BLOCK>
__global__ void __launch_bounds__(128) optimal_scale_kernel(OptParams p) {
    const float S = __ldg(p.S);
    const float E = __frcp_rn(S);
    const bool usable = (S > 0.0f) && isfinite(S) && isfinite(E);
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t blk = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; blk < p.nblocks; blk += stride) {
        const int64_t row = blk / p.kb, kbi = blk - row * p.kb;
        const int64_t off = row * p.cols + kbi * BLOCK;
        float y[BLOCK], a[BLOCK], w[BLOCK];
#pragma unroll
        for (int i = 0; i < BLOCK; i++) {
            const float xv = DT == 0 ? __uint_as_float((uint32_t)(static_cast<const uint16_t*>(p.x)[off + i]) << 16)
                                     : static_cast<const float*>(p.x)[off + i];
            y[i] = usable ? __fmul_rn(xv, E) : 0.0f;
            a[i] = fabsf(y[i]);
            w[i] = OBJ ? __ldg(p.w + row * p.w_row_stride + kbi * BLOCK + i) : 1.0f;
        }
        // s -> infinity: everything rounds to 0
        float best = 0.0f;
#pragma unroll
        for (int i = 0; i < BLOCK; i++) best = __fmaf_rn(w[i] * a[i], a[i], best);
        float best_s = 0.0f;
        // s -> 0+: every non-zero element saturates at 6
        {
            float B = 0.0f, C = 0.0f;
#pragma unroll
            for (int i = 0; i < BLOCK; i++) {
                const float g = a[i] > 0.0f ? 6.0f : 0.0f;
                B = __fmaf_rn(w[i] * a[i], g, B);
                C = __fmaf_rn(w[i] * g, g, C);
            }
            if (C > 0.0f) {
                const float s = __fdiv_rn(B, C);
                float L = 0.0f;
#pragma unroll
                for (int i = 0; i < BLOCK; i++) {
                    const float e = __fmaf_rn(-s, a[i] > 0.0f ? 6.0f : 0.0f, a[i]);
                    L = __fmaf_rn(w[i] * e, e, L);
                }
                if (L < best) {
                    best = L;
                    best_s = s;
                }
            }
        }
        for (int i = 0; i < BLOCK; i++) {
            if (!(a[i] > 0.0f)) continue;
            const float ra = __frcp_rn(a[i]);
            for (int k = 0; k < 7; k++) {
                // ~ 1/b for b = a_i / mu_k, shrunk by 2^-20 so that quotients at
                // (or within ~1e-6 of) a midpoint take the lower neighbour: the
                // assignment just above b even when breakpoints coincide
                // (equal magnitudes are common in bf16 blocks)
                const float r = __fmul_rn(__fmul_rn(kMid[k], ra), 1.0f - 9.5367431640625e-07f);
                float B = 0.0f, C = 0.0f;
                float g[BLOCK];
#pragma unroll
                for (int j = 0; j < BLOCK; j++) {
                    g[j] = (j == i) ? kGrid[k] : rn_grid(__fmul_rn(a[j], r));
                    B = __fmaf_rn(w[j] * a[j], g[j], B);
                    C = __fmaf_rn(w[j] * g[j], g[j], C);
                }
                if (!(C > 0.0f)) continue;
                const float s = __fdiv_rn(B, C);
                float L = 0.0f;
#pragma unroll
                for (int j = 0; j < BLOCK; j++) {
                    const float e = __fmaf_rn(-s, g[j], a[j]);
                    L = __fmaf_rn(w[j] * e, e, L);
                }
                // the optimum can be attained on several segments (e.g. one dominant
                // element that can sit on 6, 4, 3, ... grid points while the rest
                // round to 0): keep the smallest such scale, within fp32 ties
                if (L < best * (1.0f - 1e-6f) || (L <= best * (1.0f + 1e-6f) && s < best_s)) {
                    best = fminf(best, L);
                    best_s = s;
                }
            }
        }
        p.s_opt[blk] = best_s;
        p.loss_opt[blk] = best;
        if (p.fp8_code) {
            int code = 0;
            float Lf = best;
            if (best_s > 0.0f) {
                int fl = e4m3_floor_code(best_s);
                if (fl < 1) fl = 1;
                int ce = fl;
                const float vfl = f16bits_to_f32(e4m3_to_f16bits((uint32_t)fl));
                if (vfl < best_s && fl < 126) ce = fl + 1;
                const float Lfl = contract_loss<BLOCK, OBJ>(y, w, fl);
                const float Lce = ce == fl ? Lfl : contract_loss<BLOCK, OBJ>(y, w, ce);
                code = (Lce < Lfl) ? ce : fl;
                Lf = (Lce < Lfl) ? Lce : Lfl;
            }
            p.fp8_code[blk] = (uint8_t)code;
            if (p.loss_fp8) p.loss_fp8[blk] = Lf;
        }
    }
}

template <int DT, int OBJ>
static cudaError_t opt_block(const OptParams& p, int block, int sms, cudaStream_t s) {
    int64_t grid = (p.nblocks + 127) / 128;
    if (grid > (int64_t)sms * 16) grid = (int64_t)sms * 16;
    if (grid < 1) grid = 1;
    switch (block) {
        case 16: optimal_scale_kernel<DT, OBJ, 16><<<(int)grid, 128, 0, s>>>(p); break;
        case 32: optimal_scale_kernel<DT, OBJ, 32><<<(int)grid, 128, 0, s>>>(p); break;
        default: optimal_scale_kernel<DT, OBJ, 64><<<(int)grid, 128, 0, s>>>(p); break;
    }
    return cudaGetLastError();
}

cudaError_t launch_optimal_scale(const OptParams& p, int dtype, int obj, int block, int sms, cudaStream_t s) {
    if (p.nblocks <= 0) return cudaSuccess;
    if (dtype == 0) return obj ? opt_block<0, 1>(p, block, sms, s) : opt_block<0, 0>(p, block, sms, s);
    return obj ? opt_block<1, 1>(p, block, sms, s) : opt_block<1, 0>(p, block, sms, s);
}

}  // namespace nvfp4
