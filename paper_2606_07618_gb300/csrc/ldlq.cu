// LDLQ (GPTQ's error-feedback pass) with fixed NVFP4 block scales and static
// reordering -- Appendix A.2 of the ScaleSweep paper: GPTQ run as LDLQ (QuIP),
// damping 0.01 x the mean Hessian diagonal, block scales fixed beforehand by
// ScaleSweep, input channels processed in descending order of diag(H).
//
// Prepare (depends on H only):
//   lambda = damp * mean(diag H); perm = channels by (diag desc, index asc);
//   A = J H_pi J + lambda I (J reverses the order), A = L L^T by a blocked
//   right-looking Cholesky (64-wide panels: diagonal block factor and inverse
//   in one CTA, panel solve by the inverse, trailing update by the K<=64 GEMM
//   below on lower tiles only); then, in place,
//   H_pi = (U + I) D (U + I)^T with U_ik = L[n-1-i][n-1-k] / L[n-1-k][n-1-k]
//   (J L J is upper triangular) and D_k = L[n-1-k][n-1-k]^2.
// Quantize (rows independent):
//   T = W_pi (fp32); per 64-column panel, one warp per row walks the columns in
//   order -- What_k = Q(T_k) at the element's fixed scale, e_k = W_k - What_k,
//   T_j += e_k U_kj for the later columns of the panel -- then the trailing
//   columns get T += E_panel U_panel,rest (the GEMM); finally the nibbles are
//   scattered back to the original column order.
// Q follows the sweep's float32 contract: y = fl(t*E), q = RNE_E2M1(fl(y*r_c)),
// What = fl(fl(q*v_c)*S); a zero-scale block or an unusable S gives signed
// zeros; an exactly zero y takes the +0 code.
#include <cuda_bf16.h>

#include "nvfp4_device.cuh"
#include "nvfp4_kernels.h"

namespace nvfp4 {

namespace {

constexpr int kP = kLdlqPanel;        // 64
constexpr int kLd = 132;              // GEMM smem row stride (floats): 128 + 4, 16-byte rows

inline int64_t imin64(int64_t a, int64_t b) { return a < b ? a : b; }

__device__ __forceinline__ float sort_key(float v) { return isnan(v) ? -INFINITY : v; }

// d = diag(H), lambda = damp * mean(d) (double sum); bit 4 if any diagonal entry is not finite.
__global__ void __launch_bounds__(1024) diag_kernel(const float* H, int64_t n, float damp, float* d, float* lam,
                                                    int* status) {
    double s = 0.0;
    int bad = 0;
    for (int64_t i = threadIdx.x; i < n; i += blockDim.x) {
        const float v = H[i * n + i];
        d[i] = v;
        if (isfinite(v)) s += (double)v; else bad = 1;
    }
    __shared__ double ss[32];
    __shared__ int sb[32];
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    bad = __reduce_or_sync(0xffffffffu, (unsigned)bad);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) {
        ss[warp] = s;
        sb[warp] = bad;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        double t = 0.0;
        int b = 0;
        for (int w = 0; w < (int)(blockDim.x >> 5); w++) {
            t += ss[w];
            b |= sb[w];
        }
        lam[0] = (float)((double)damp * t / (double)n);
        if (b && status) atomicOr(status, 4);
    }
}

// perm[rank(i)] = i, rank by (key desc, index asc): a total order, so perm is a
// permutation of 0..n-1 whatever the keys.
__global__ void __launch_bounds__(256) rank_kernel(const float* d, int64_t n, int32_t* perm) {
    __shared__ float sd[1024];
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const float di = i < n ? sort_key(d[i]) : 0.0f;
    int64_t rank = 0;
    for (int64_t base = 0; base < n; base += 1024) {
        __syncthreads();
        for (int t = threadIdx.x; t < 1024; t += blockDim.x) sd[t] = base + t < n ? sort_key(d[base + t]) : 0.0f;
        __syncthreads();
        if (i < n) {
            const int lim = (int)min((int64_t)1024, n - base);
            for (int t = 0; t < lim; t++) {
                const float dj = sd[t];
                rank += (dj > di) || (dj == di && base + t < i);
            }
        }
    }
    if (i < n) perm[rank] = (int32_t)i;
}

// A[a][b] = H[p(a)][p(b)] (+ lambda on the diagonal), p(a) = perm[n-1-a].
__global__ void __launch_bounds__(256) gather_h_kernel(const float* H, int64_t n, const int32_t* perm,
                                                       const float* lam, float* A) {
    const float l = lam[0];
    for (int64_t a = blockIdx.x; a < n; a += gridDim.x) {
        const float* hrow = H + (int64_t)perm[n - 1 - a] * n;
        float* arow = A + a * n;
        for (int64_t b = threadIdx.x; b < n; b += blockDim.x) {
            float v = hrow[perm[n - 1 - b]];
            if (a == b) v = __fadd_rn(v, l);
            arow[b] = v;
        }
    }
}

// Cholesky of the nb x nb diagonal block at k0 (lower, in place) and its inverse
// (lower, 64 x 64 with zeros) into Linv.  A pivot that is not positive and finite
// sets bit 4 of the status word and is replaced by 1 so the values stay finite.
__global__ void __launch_bounds__(256) potrf_kernel(float* A, int64_t n, int64_t k0, int nb, float* Linv,
                                                    int* status) {
    __shared__ float a[kP][kP + 1];
    __shared__ float li[kP][kP + 1];
    __shared__ int s_bad;
    for (int e = threadIdx.x; e < kP * kP; e += blockDim.x) {
        const int i = e / kP, j = e % kP;
        a[i][j] = (i < nb && j < nb) ? A[(k0 + i) * n + k0 + j] : 0.0f;
        li[i][j] = 0.0f;
    }
    if (threadIdx.x == 0) s_bad = 0;
    __syncthreads();
    for (int j = 0; j < nb; j++) {
        if (threadIdx.x == 0) {
            float p = a[j][j];
            if (!(p > 0.0f) || !isfinite(p)) {
                s_bad = 1;
                p = 1.0f;
            }
            a[j][j] = __fsqrt_rn(p);
        }
        __syncthreads();
        const float dj = a[j][j];
        for (int i = j + 1 + threadIdx.x; i < nb; i += blockDim.x) a[i][j] = __fdiv_rn(a[i][j], dj);
        __syncthreads();
        const int m = nb - j - 1;
        for (int e = threadIdx.x; e < m * m; e += blockDim.x) {
            const int i = j + 1 + e / m, l = j + 1 + e % m;
            if (l <= i) a[i][l] = __fmaf_rn(-a[i][j], a[l][j], a[i][l]);
        }
        __syncthreads();
    }
    if (threadIdx.x < nb) {                       // column c of L^-1 by forward substitution
        const int c = threadIdx.x;
        li[c][c] = __fdiv_rn(1.0f, a[c][c]);
        for (int i = c + 1; i < nb; i++) {
            float s = 0.0f;
            for (int l = c; l < i; l++) s = __fmaf_rn(a[i][l], li[l][c], s);
            li[i][c] = __fdiv_rn(-s, a[i][i]);
        }
    }
    __syncthreads();
    for (int e = threadIdx.x; e < kP * kP; e += blockDim.x) {
        const int i = e / kP, j = e % kP;
        if (i < nb && j <= i) A[(k0 + i) * n + k0 + j] = a[i][j];
        Linv[e] = li[i][j];
    }
    if (threadIdx.x == 0 && s_bad && status) atomicOr(status, 4);
}

// Panel below the diagonal block: rows i >= k0+nb, X = A_panel * Linv^T (one warp per row).
__global__ void __launch_bounds__(256) trsm_kernel(float* A, int64_t n, int64_t k0, int nb, const float* Linv) {
    __shared__ float li[kP][kP + 1];
    __shared__ float row[8][kP];
    for (int e = threadIdx.x; e < kP * kP; e += blockDim.x) li[e / kP][e % kP] = Linv[e];
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int64_t i = k0 + nb + (int64_t)blockIdx.x * 8 + warp; i < n; i += (int64_t)gridDim.x * 8) {
        float* ai = A + i * n + k0;
        row[warp][lane] = lane < nb ? ai[lane] : 0.0f;
        row[warp][lane + 32] = lane + 32 < nb ? ai[lane + 32] : 0.0f;
        __syncwarp();
        float x0 = 0.0f, x1 = 0.0f;
        for (int l = 0; l < nb; l++) {
            const float al = row[warp][l];
            x0 = __fmaf_rn(al, li[lane][l], x0);
            x1 = __fmaf_rn(al, li[lane + 32][l], x1);
        }
        __syncwarp();
        if (lane < nb) ai[lane] = x0;
        if (lane + 32 < nb) ai[lane + 32] = x1;
    }
}

// C[M, N] += alpha * A[M, K] * op(B), K <= 64.  op(B) = B [K, N] row-major, or
// (BT) B^T with B stored [N, K] row-major.  128 x 128 tiles, 256 threads, 8 x 8
// outputs per thread from K-major shared tiles.  LOWER skips tiles that lie
// entirely above the diagonal (n0 > m0 + 127).
template <bool BT, bool LOWER>
__global__ void __launch_bounds__(256) gemm_k64_kernel(float* C, int64_t ldc, const float* A, int64_t lda,
                                                       const float* B, int64_t ldb, int64_t M, int64_t N, int K,
                                                       float alpha) {
    extern __shared__ __align__(16) float smem[];
    float* As = smem;                 // [64][kLd]: As[k][m]
    float* Bs = smem + kP * kLd;      // [64][kLd]: Bs[k][n]
    const int64_t m0 = (int64_t)blockIdx.y * 128, n0 = (int64_t)blockIdx.x * 128;
    if (LOWER && n0 > m0 + 127) return;
    for (int e = threadIdx.x; e < 128 * kP; e += 256) {
        const int mm = e / kP, k = e % kP;
        As[k * kLd + mm] = (k < K && m0 + mm < M) ? A[(m0 + mm) * lda + k] : 0.0f;
    }
    if (BT) {
        for (int e = threadIdx.x; e < 128 * kP; e += 256) {
            const int nn = e / kP, k = e % kP;
            Bs[k * kLd + nn] = (k < K && n0 + nn < N) ? B[(n0 + nn) * ldb + k] : 0.0f;
        }
    } else {
        for (int e = threadIdx.x; e < 128 * kP; e += 256) {
            const int k = e / 128, nn = e % 128;
            Bs[k * kLd + nn] = (k < K && n0 + nn < N) ? B[k * ldb + n0 + nn] : 0.0f;
        }
    }
    __syncthreads();
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    float acc[8][8];
#pragma unroll
    for (int i = 0; i < 8; i++)
#pragma unroll
        for (int j = 0; j < 8; j++) acc[i][j] = 0.0f;
#pragma unroll 4
    for (int k = 0; k < K; k++) {
        const float4 a0 = *reinterpret_cast<const float4*>(As + k * kLd + ty * 4);
        const float4 a1 = *reinterpret_cast<const float4*>(As + k * kLd + 64 + ty * 4);
        const float4 b0 = *reinterpret_cast<const float4*>(Bs + k * kLd + tx * 4);
        const float4 b1 = *reinterpret_cast<const float4*>(Bs + k * kLd + 64 + tx * 4);
        const float av[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
        const float bv[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
        for (int i = 0; i < 8; i++)
#pragma unroll
            for (int j = 0; j < 8; j++) acc[i][j] = __fmaf_rn(av[i], bv[j], acc[i][j]);
    }
#pragma unroll
    for (int i = 0; i < 8; i++) {
        const int64_t r = m0 + (i < 4 ? ty * 4 + i : 64 + ty * 4 + i - 4);
        if (r >= M) continue;
        float* crow = C + r * ldc;
#pragma unroll
        for (int j = 0; j < 8; j++) {
            const int64_t c = n0 + (j < 4 ? tx * 4 + j : 64 + tx * 4 + j - 4);
            if (c < N) crow[c] = __fmaf_rn(alpha, acc[i][j], crow[c]);
        }
    }
}

template <bool BT, bool LOWER>
cudaError_t launch_gemm(float* C, int64_t ldc, const float* A, int64_t lda, const float* B, int64_t ldb, int64_t M,
                        int64_t N, int K, float alpha, cudaStream_t s) {
    if (M <= 0 || N <= 0 || K <= 0) return cudaSuccess;
    constexpr int kSmem = 2 * kP * kLd * (int)sizeof(float);
    static bool attr_set[64] = {false};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64 || !attr_set[dev]) {
        e = cudaFuncSetAttribute(gemm_k64_kernel<BT, LOWER>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem);
        if (e != cudaSuccess) return e;
        if (dev >= 0 && dev < 64) attr_set[dev] = true;
    }
    const dim3 grid((unsigned)((N + 127) / 128), (unsigned)((M + 127) / 128));
    gemm_k64_kernel<BT, LOWER><<<grid, 256, kSmem, s>>>(C, ldc, A, lda, B, ldb, M, N, K, alpha);
    return cudaGetLastError();
}

__global__ void diag_d_kernel(const float* A, int64_t n, float* D) {
    const int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (k < n) {
        const float l = A[(n - 1 - k) * n + (n - 1 - k)];
        D[k] = __fmul_rn(l, l);
    }
}

// In place: U[n-1-a][n-1-b] = L[a][b] / L[b][b] for a > b; L[a][b] = 0.  Every
// thread reads its own lower entry and a diagonal entry and writes its own lower
// entry and one upper entry that nothing reads, so the threads do not race.
__global__ void __launch_bounds__(256) flip_kernel(float* A, int64_t n) {
    for (int64_t a = blockIdx.x; a < n; a += gridDim.x) {
        for (int64_t b = threadIdx.x; b < a; b += blockDim.x) {
            const float v = __fdiv_rn(A[a * n + b], A[b * n + b]);
            A[(n - 1 - a) * n + (n - 1 - b)] = v;
            A[a * n + b] = 0.0f;
        }
    }
}

__global__ void zero_diag_kernel(float* A, int64_t n) {
    const int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (k < n) A[k * n + k] = 0.0f;
}

// ---------------------------------------------------------------- quantize

__device__ __forceinline__ int32_t checked_index(int32_t p, int64_t n, int* status) {
    if ((uint32_t)p >= (uint64_t)n) {
        if (status) atomicOr(status, 8);
        return 0;
    }
    return p;
}

__global__ void __launch_bounds__(256) invperm_kernel(const int32_t* perm, int64_t n, int32_t* inv, int* status) {
    const int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (k < n) inv[checked_index(perm[k], n, status)] = (int32_t)k;
}

template <int DT>
__device__ __forceinline__ float load_w(const void* W, int64_t idx) {
    if (DT == 0) return __uint_as_float((uint32_t)(static_cast<const uint16_t*>(W)[idx]) << 16);
    return static_cast<const float*>(W)[idx];
}

// T[r][k] = W[r][perm[k]]
template <int DT>
__global__ void __launch_bounds__(256) gather_w_kernel(const void* W, int64_t rows, int64_t n, const int32_t* perm,
                                                       float* T, int* status) {
    for (int64_t r = blockIdx.x; r < rows; r += gridDim.x)
        for (int64_t k = threadIdx.x; k < n; k += blockDim.x)
            T[r * n + k] = load_w<DT>(W, r * n + checked_index(perm[k], n, status));
}

template <int DT>
__global__ void __launch_bounds__(256) panel_kernel(LdlqParams p, int64_t k0, int P) {
    __shared__ float up[kP][kP + 1];                 // up[s][j] = U[k0+s][k0+j] for s < j < P
    for (int e = threadIdx.x; e < kP * kP; e += blockDim.x) {
        const int s = e / kP, j = e % kP;
        up[s][j] = (s < j && j < P) ? p.U[(k0 + s) * p.n + k0 + j] : 0.0f;
    }
    __syncthreads();
    const float S = __ldg(p.S);
    const float Einv = __frcp_rn(S);
    const bool usable = (S > 0.0f) && isfinite(S) && isfinite(Einv);
    const float E = usable ? Einv : 1.0f;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int64_t r = (int64_t)blockIdx.x * 8 + warp; r < p.rows; r += (int64_t)gridDim.x * 8) {
        float t[2], w[2], v[2], rc[2];
        int code[2];
#pragma unroll
        for (int h = 0; h < 2; h++) {
            const int j = lane + 32 * h;
            t[h] = w[h] = v[h] = rc[h] = 0.0f;
            code[h] = 0;
            if (j < P) {
                const int64_t c = checked_index(p.perm[k0 + j], p.n, p.status);
                t[h] = p.T[r * p.n + k0 + j];
                w[h] = load_w<DT>(p.W, r * p.n + c);
                code[h] = p.sf[r * p.kb + c / p.block];
                if (code[h] > 126) code[h] = 0;              // 0x7F (NaN) and above: treated as a zero scale
                v[h] = f16bits_to_f32(e4m3_to_f16bits((uint32_t)code[h]));
                rc[h] = code[h] ? __frcp_rn(v[h]) : 0.0f;
            }
        }
        for (int s = 0; s < P; s++) {
            const int owner = s & 31;
            const bool hi = s >= 32;
            float e = 0.0f;
            if (lane == owner) {
                const float ts = hi ? t[1] : t[0], ws = hi ? w[1] : w[0];
                const float vs = hi ? v[1] : v[0], rs = hi ? rc[1] : rc[0];
                const int cs = hi ? code[1] : code[0];
                const float y = usable ? __fmul_rn(ts, E) : ts;
                uint32_t nib;
                float val;
                if (y == 0.0f) {
                    nib = 0;
                    val = 0.0f;
                } else if (!usable || cs == 0) {
                    nib = signbit(y) ? 8u : 0u;
                    val = signbit(y) ? -0.0f : 0.0f;
                } else {
                    const float tq = __fmul_rn(y, rs);
                    nib = e2m1x2(tq, 0.0f) & 0xFu;
                    uint32_t h2;
                    asm("{\n\t.reg .b8 b;\n\tcvt.u8.u32 b, %1;\n\tcvt.rn.f16x2.e2m1x2 %0, b;\n\t}"
                        : "=r"(h2) : "r"(nib));
                    const float q = f16bits_to_f32((uint16_t)(h2 & 0xFFFFu));
                    val = __fmul_rn(__fmul_rn(q, vs), S);
                }
                e = __fsub_rn(ws, val);
                p.qb[r * p.n + k0 + s] = (uint8_t)nib;
                p.Ep[r * kP + s] = e;
            }
            e = __shfl_sync(0xffffffffu, e, owner);
            t[0] = __fmaf_rn(e, up[s][lane], t[0]);
            t[1] = __fmaf_rn(e, up[s][lane + 32], t[1]);
        }
    }
}

// codes[r][c/2]: nibble of original column c from qb[r][inv[c]]
__global__ void __launch_bounds__(256) pack_kernel(const uint8_t* qb, const int32_t* inv, int64_t rows, int64_t n,
                                                   uint8_t* codes, int* status) {
    const int64_t half = n / 2;
    for (int64_t r = blockIdx.x; r < rows; r += gridDim.x)
        for (int64_t c2 = threadIdx.x; c2 < half; c2 += blockDim.x) {
            const uint8_t lo = qb[r * n + checked_index(inv[2 * c2], n, status)];
            const uint8_t hi = qb[r * n + checked_index(inv[2 * c2 + 1], n, status)];
            codes[r * half + c2] = (uint8_t)((lo & 0xF) | ((hi & 0xF) << 4));
        }
}

}  // namespace

size_t ldlq_prepare_workspace(int64_t n) {
    return (size_t)((n * 4 + 255) / 256 * 256) + 256 + (size_t)kP * kP * 4;
}

cudaError_t launch_ldlq_prepare(const float* H, int64_t n, float damp, int32_t* perm, float* U, float* D,
                                int* status, void* ws, int sms, cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    char* w = static_cast<char*>(ws);
    float* d = reinterpret_cast<float*>(w);
    float* lam = reinterpret_cast<float*>(w + (n * 4 + 255) / 256 * 256);
    float* Linv = lam + 64;
    diag_kernel<<<1, 1024, 0, s>>>(H, n, damp, d, lam, status);
    rank_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(d, n, perm);
    const unsigned rg = (unsigned)imin64(n, (int64_t)sms * 8);
    gather_h_kernel<<<rg, 256, 0, s>>>(H, n, perm, lam, U);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    for (int64_t k0 = 0; k0 < n; k0 += kP) {
        const int nb = (int)imin64(kP, n - k0);
        potrf_kernel<<<1, 256, 0, s>>>(U, n, k0, nb, Linv, status);
        const int64_t rest = n - k0 - nb;
        if (rest > 0) {
            const unsigned tg = (unsigned)imin64((rest + 7) / 8, (int64_t)sms * 8);
            trsm_kernel<<<tg, 256, 0, s>>>(U, n, k0, nb, Linv);
            float* P = U + (k0 + nb) * n + k0;
            e = launch_gemm<true, true>(U + (k0 + nb) * n + k0 + nb, n, P, n, P, n, rest, rest, nb, -1.0f, s);
            if (e != cudaSuccess) return e;
        }
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    diag_d_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(U, n, D);
    flip_kernel<<<rg, 256, 0, s>>>(U, n);
    zero_diag_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(U, n);
    return cudaGetLastError();
}

size_t ldlq_quantize_workspace(int64_t rows, int64_t n) {
    auto up = [](int64_t b) { return (b + 255) / 256 * 256; };
    return (size_t)(up(rows * n * 4) + up(rows * n) + up(rows * kP * 4) + up(n * 4));
}

cudaError_t launch_ldlq_quantize(LdlqParams p, int dtype, uint8_t* codes, void* ws, int sms, cudaStream_t s) {
    if (p.rows <= 0 || p.n <= 0) return cudaSuccess;
    auto up = [](int64_t b) { return (b + 255) / 256 * 256; };
    char* w = static_cast<char*>(ws);
    p.T = reinterpret_cast<float*>(w);
    p.qb = reinterpret_cast<uint8_t*>(w + up(p.rows * p.n * 4));
    p.Ep = reinterpret_cast<float*>(w + up(p.rows * p.n * 4) + up(p.rows * p.n));
    int32_t* inv = reinterpret_cast<int32_t*>(w + up(p.rows * p.n * 4) + up(p.rows * p.n) + up(p.rows * kP * 4));
    cudaError_t e = cudaMemsetAsync(inv, 0, (size_t)p.n * 4, s);
    if (e != cudaSuccess) return e;
    invperm_kernel<<<(unsigned)((p.n + 255) / 256), 256, 0, s>>>(p.perm, p.n, inv, p.status);
    const unsigned rg = (unsigned)imin64(p.rows, (int64_t)sms * 8);
    if (dtype == 0)
        gather_w_kernel<0><<<rg, 256, 0, s>>>(p.W, p.rows, p.n, p.perm, p.T, p.status);
    else
        gather_w_kernel<1><<<rg, 256, 0, s>>>(p.W, p.rows, p.n, p.perm, p.T, p.status);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const unsigned pg = (unsigned)imin64((p.rows + 7) / 8, (int64_t)sms * 4);
    for (int64_t k0 = 0; k0 < p.n; k0 += kP) {
        const int P = (int)imin64(kP, p.n - k0);
        if (dtype == 0)
            panel_kernel<0><<<pg, 256, 0, s>>>(p, k0, P);
        else
            panel_kernel<1><<<pg, 256, 0, s>>>(p, k0, P);
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
        const int64_t rest = p.n - k0 - P;
        if (rest > 0) {
            e = launch_gemm<false, false>(p.T + k0 + P, p.n, p.Ep, kP, p.U + k0 * p.n + k0 + P, p.n, p.rows, rest, P,
                                          1.0f, s);
            if (e != cudaSuccess) return e;
        }
    }
    pack_kernel<<<rg, 256, 0, s>>>(p.qb, inv, p.rows, p.n, codes, p.status);
    return cudaGetLastError();
}

}  // namespace nvfp4
