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
#include <atomic>
#include <mutex>

#include <cuda_bf16.h>

#include "nvfp4_device.cuh"
#include "ldlq_kernels.h"
#include "nvfp4_kernels.h"
#include "tc_gemm.cuh"

namespace nvfp4 {

namespace {

constexpr int kP = 64;                // Cholesky panel width
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
// (lower, 64 x 64) into Linv.  The block is padded to 64 with an identity; each
// of the 256 threads keeps a 4 x 4 tile in registers.  The pivots stay
// unscaled, A = M diag(p) M^T with M unit lower triangular: at column j the
// threads holding column j publish it to shared memory (double-buffered, one
// barrier per column) and every tile subtracts a_ij a_lj / p_j (rows i > j,
// columns l > j; the upper parts of the tiles take the same updates unread).  Then
// L = M diag(sqrt p) and L^-1 = diag(1/sqrt p) M^-1, with M^-1 by forward
// elimination in the same scheme (column k of M and row k of M^-1 published per
// step).  A pivot that is not positive and finite sets bit 4 of the status word
// and is replaced by 1 so the values stay finite.
__global__ void __launch_bounds__(256) potrf_kernel(float* A, int64_t n, int64_t k0, int nb, float* Linv,
                                                    int* status) {
    __shared__ __align__(16) float colv[2][kP];
    __shared__ __align__(16) float rowv[2][kP];
    __shared__ float piv[kP];
    const int r0 = (threadIdx.x >> 4) * 4, c0 = (threadIdx.x & 15) * 4;
    float t[4][4];
    float x[4][4];                                   // X = M^-1 (unit lower), built alongside
#pragma unroll
    for (int di = 0; di < 4; di++)
#pragma unroll
        for (int dl = 0; dl < 4; dl++) {
            const int i = r0 + di, l = c0 + dl;
            float v = (i < nb && l < nb && l <= i) ? A[(k0 + i) * n + k0 + l] : 0.0f;
            if (i >= nb && i == l) v = 1.0f;
            t[di][dl] = v;
            x[di][dl] = i == l ? 1.0f : 0.0f;
        }
    // Step j: column j of the reduced matrix gives the pivot and the multipliers
    // m_ij = a_ij / p_j (= M's column j); the trailing update and the inverse's
    // row operation X_i -= m_ij X_j (row j of X is final at step j) share one
    // barrier.  Per entry the inverse sees its updates in the order k = 0, 1, ...
    int bad = 0;
    // columns in groups of four, so that a tile's column j - c0 (and row j - r0)
    // is a compile-time index: the owners publish without selects
    for (int jb = 0; jb < kP; jb += 4) {
#pragma unroll
        for (int q = 0; q < 4; q++) {
            const int j = jb + q, b = q & 1;
            if (c0 == jb)
#pragma unroll
                for (int di = 0; di < 4; di++) colv[b][r0 + di] = t[di][q];
            if (r0 == jb)                            // row j of X
#pragma unroll
                for (int dc = 0; dc < 4; dc++) rowv[b][c0 + dc] = x[q][dc];
            __syncthreads();
            float p = colv[b][j];
            if (!(p > 0.0f) || !isfinite(p)) {
                bad = 1;
                p = 1.0f;
            }
            if (threadIdx.x == 0) piv[j] = p;
            const float ip = __frcp_rn(p);
            const float4 ci = *reinterpret_cast<const float4*>(&colv[b][r0]);
            const float4 cl = *reinterpret_cast<const float4*>(&colv[b][c0]);
            const float4 xj = *reinterpret_cast<const float4*>(&rowv[b][c0]);
            const float civ[4] = {ci.x, ci.y, ci.z, ci.w}, clv[4] = {cl.x, cl.y, cl.z, cl.w};
            const float xjv[4] = {xj.x, xj.y, xj.z, xj.w};
            // rows i <= j and columns l <= j take a zero multiplier instead of a
            // predicate: the skipped terms are exact zeros (the tiles' upper parts
            // are never read back and stay finite; row j of M^-1 is zero beyond
            // column j), so all 32 updates run unconditionally
            float am[4], cm[4];
#pragma unroll
            for (int d = 0; d < 4; d++) {
                am[d] = r0 + d > j ? __fmul_rn(civ[d], ip) : 0.0f;
                cm[d] = c0 + d > j ? clv[d] : 0.0f;
            }
#pragma unroll
            for (int di = 0; di < 4; di++)
#pragma unroll
                for (int dl = 0; dl < 4; dl++) {
                    t[di][dl] = __fmaf_rn(-am[di], cm[dl], t[di][dl]);
                    x[di][dl] = __fmaf_rn(-am[di], xjv[dl], x[di][dl]);
                }
        }
    }
    __syncthreads();
    // M (strictly lower part) in the tiles: m_il = a_il / p_l
#pragma unroll
    for (int di = 0; di < 4; di++)
#pragma unroll
        for (int dl = 0; dl < 4; dl++)
            if (c0 + dl < r0 + di) t[di][dl] = __fmul_rn(t[di][dl], __frcp_rn(piv[c0 + dl]));
#pragma unroll
    for (int di = 0; di < 4; di++)
#pragma unroll
        for (int dl = 0; dl < 4; dl++) {
            const int i = r0 + di, l = c0 + dl;
            const float sl = __fsqrt_rn(piv[l]);
            if (i < nb && l <= i) A[(k0 + i) * n + k0 + l] = i == l ? sl : __fmul_rn(t[di][dl], sl);
            Linv[i * kP + l] = l <= i ? __fmul_rn(x[di][dl], __frsqrt_rn(piv[i])) : 0.0f;
        }
    if (threadIdx.x == 0 && bad && status) atomicOr(status, 4);
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

// C[M, N] += alpha * op(A) * op(B).  op(A) = A [M, K] row-major, or (AT) A^T
// with A stored [K, M] row-major; op(B) = B [K, N] row-major, or (BT) B^T with
// B stored [N, K] row-major.  128 x 128 tiles, 256 threads, 8 x 8 outputs per
// thread, K in stages of 32 through two shared buffers filled by cp.async
// (global to shared without registers) while the other stage is multiplied.
// LOWER skips tiles entirely above the diagonal (n0 > m0 + 127).  VEC: C rows
// and the column base are 16-byte aligned, so the epilogue moves float4s.
constexpr int kBK = 32;

__device__ __forceinline__ void cp_async4(float* dst, const float* src, bool valid) {
    const uint32_t d = (uint32_t)__cvta_generic_to_shared(dst);
    const int n = valid ? 4 : 0;                    // 0: zero-fill, nothing is read
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(d), "l"(src), "r"(n) : "memory");
}

template <bool AT, bool BT, bool LOWER, bool VEC>
__global__ void __launch_bounds__(256, 2) gemm_kernel(float* C, int64_t ldc, const float* A, int64_t lda,
                                                      const float* B, int64_t ldb, int64_t M, int64_t N, int K,
                                                      float alpha) {
    extern __shared__ __align__(16) float smem[];
    float* As = smem;                         // [2][kBK][kLd]: As[b][k][m]
    float* Bs = smem + 2 * kBK * kLd;         // [2][kBK][kLd]: Bs[b][k][n]
    const int64_t m0 = (int64_t)blockIdx.y * 128, n0 = (int64_t)blockIdx.x * 128;
    if (LOWER && n0 > m0 + 127) return;
    const int tid = threadIdx.x;
    // element e = tid + 256*i of a 128 x 32 (A) or 32 x 128 (B) stage tile
    auto issue = [&](int k0, int b) {
        float* as = As + b * kBK * kLd;
        float* bs = Bs + b * kBK * kLd;
#pragma unroll
        for (int i = 0; i < 16; i++) {
            const int e = tid + 256 * i;
            if (AT) {
                const int k = e / 128, mm = e % 128;
                const bool ok = k0 + k < K && m0 + mm < M;
                cp_async4(as + k * kLd + mm, ok ? A + (int64_t)(k0 + k) * lda + m0 + mm : A, ok);
            } else {
                const int mm = e / kBK, k = e % kBK;
                const bool ok = k0 + k < K && m0 + mm < M;
                cp_async4(as + k * kLd + mm, ok ? A + (m0 + mm) * lda + k0 + k : A, ok);
            }
            if (BT) {
                const int nn = e / kBK, k = e % kBK;
                const bool ok = k0 + k < K && n0 + nn < N;
                cp_async4(bs + k * kLd + nn, ok ? B + (n0 + nn) * ldb + k0 + k : B, ok);
            } else {
                const int k = e / 128, nn = e % 128;
                const bool ok = k0 + k < K && n0 + nn < N;
                cp_async4(bs + k * kLd + nn, ok ? B + (int64_t)(k0 + k) * ldb + n0 + nn : B, ok);
            }
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    };
    const int tx = tid & 15, ty = tid >> 4;
    // 8 x 8 outputs per thread as 8 x 4 packed pairs: one fma.rn.f32x2 per pair
    // (per lane the same IEEE fma as the scalar form, at twice the operands per
    // register read).
    u64 acc[8][4];
#pragma unroll
    for (int i = 0; i < 8; i++)
#pragma unroll
        for (int j = 0; j < 4; j++) acc[i][j] = 0ull;
    const int nst = (K + kBK - 1) / kBK;
    issue(0, 0);
    for (int st = 0; st < nst; st++) {
        const int b = st & 1;
        if (st + 1 < nst) {
            issue((st + 1) * kBK, b ^ 1);
            asm volatile("cp.async.wait_group 1;" ::: "memory");
        } else {
            asm volatile("cp.async.wait_group 0;" ::: "memory");
        }
        __syncthreads();
        const float* as = As + b * kBK * kLd;
        const float* bs = Bs + b * kBK * kLd;
#pragma unroll 8
        for (int k = 0; k < kBK; k++) {
            const float4 a0 = *reinterpret_cast<const float4*>(as + k * kLd + ty * 4);
            const float4 a1 = *reinterpret_cast<const float4*>(as + k * kLd + 64 + ty * 4);
            const float4 b0 = *reinterpret_cast<const float4*>(bs + k * kLd + tx * 4);
            const float4 b1 = *reinterpret_cast<const float4*>(bs + k * kLd + 64 + tx * 4);
            const float av[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
            const u64 bp[4] = {pack2(b0.x, b0.y), pack2(b0.z, b0.w), pack2(b1.x, b1.y), pack2(b1.z, b1.w)};
#pragma unroll
            for (int i = 0; i < 8; i++) {
                const u64 ap = pack2(av[i], av[i]);
#pragma unroll
                for (int j = 0; j < 4; j++) acc[i][j] = fma2(ap, bp[j], acc[i][j]);
            }
        }
        __syncthreads();                           // buffer b is refilled by the next issue
    }
#pragma unroll
    for (int i = 0; i < 8; i++) {
        const int64_t r = m0 + (i < 4 ? ty * 4 + i : 64 + ty * 4 + i - 4);
        if (r >= M) continue;
        float* crow = C + r * ldc;
#pragma unroll
        for (int h = 0; h < 2; h++) {
            const int64_t c = n0 + h * 64 + tx * 4;
            float o[4];
            unpack2(acc[i][2 * h], o[0], o[1]);
            unpack2(acc[i][2 * h + 1], o[2], o[3]);
            if (VEC && c + 3 < N) {
                float4 v = *reinterpret_cast<float4*>(crow + c);
                v.x = __fmaf_rn(alpha, o[0], v.x);
                v.y = __fmaf_rn(alpha, o[1], v.y);
                v.z = __fmaf_rn(alpha, o[2], v.z);
                v.w = __fmaf_rn(alpha, o[3], v.w);
                *reinterpret_cast<float4*>(crow + c) = v;
            } else {
#pragma unroll
                for (int j = 0; j < 4; j++)
                    if (c + j < N) crow[c + j] = __fmaf_rn(alpha, o[j], crow[c + j]);
            }
        }
    }
}

template <bool AT, bool BT, bool LOWER, bool VEC>
cudaError_t launch_gemm_t(float* C, int64_t ldc, const float* A, int64_t lda, const float* B, int64_t ldb, int64_t M,
                          int64_t N, int K, float alpha, cudaStream_t s) {
    constexpr int kSmem = 4 * kBK * kLd * (int)sizeof(float);
    static std::atomic<bool> attr_set[64];        // per device: the shared-memory opt-in is done
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64 || !attr_set[dev].load(std::memory_order_acquire)) {
        e = cudaFuncSetAttribute(gemm_kernel<AT, BT, LOWER, VEC>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem);
        if (e != cudaSuccess) return e;
        if (dev >= 0 && dev < 64) attr_set[dev].store(true, std::memory_order_release);
    }
    const dim3 grid((unsigned)((N + 127) / 128), (unsigned)((M + 127) / 128));
    gemm_kernel<AT, BT, LOWER, VEC><<<grid, 256, kSmem, s>>>(C, ldc, A, lda, B, ldb, M, N, K, alpha);
    return cudaGetLastError();
}

template <bool AT, bool BT, bool LOWER>
cudaError_t launch_gemm(float* C, int64_t ldc, const float* A, int64_t lda, const float* B, int64_t ldb, int64_t M,
                        int64_t N, int K, float alpha, cudaStream_t s) {
    if (M <= 0 || N <= 0 || K <= 0) return cudaSuccess;
    const bool vec = (ldc % 4 == 0) && ((reinterpret_cast<uintptr_t>(C) & 15) == 0);
    return vec ? launch_gemm_t<AT, BT, LOWER, true>(C, ldc, A, lda, B, ldb, M, N, K, alpha, s)
               : launch_gemm_t<AT, BT, LOWER, false>(C, ldc, A, lda, B, ldb, M, N, K, alpha, s);
}

// C += alpha op(A) op(B) for the LDLQ updates: on the tensor cores (tcgen05,
// 3xTF32, tc_gemm.cuh) wherever its TMA alignment rules hold (16-byte aligned
// bases and row strides), else with the SIMT fp32 GEMM above.  AT: A stored
// [K][M]; BT: B stored [N][K] (the tensor-core GEMM's B_MN is !BT).
template <bool AT, bool BT, bool LOWER>
cudaError_t update_gemm(float* C, int64_t ldc, const float* A, int64_t lda, const float* B, int64_t ldb, int64_t M,
                        int64_t N, int K, float alpha, int* status, cudaStream_t s) {
    const cudaError_t e = tc::launch_gemm<AT, !BT, LOWER>(C, ldc, A, lda, B, ldb, M, N, K, alpha, status, s);
    if (e != cudaErrorNotSupported) return e;
    return launch_gemm<AT, BT, LOWER>(C, ldc, A, lda, B, ldb, M, N, K, alpha, s);
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

// T[r][k] = Wp[r][k] = W[r][perm[k]] (fp32) and sfp[r][k] = sf[r][perm[k] / block].
template <int DT>
__global__ void __launch_bounds__(256) gather_w_kernel(LdlqParams p) {
    for (int64_t r = blockIdx.x; r < p.rows; r += gridDim.x)
        for (int64_t k = threadIdx.x; k < p.n; k += blockDim.x) {
            const int64_t c = checked_index(p.perm[k], p.n, p.status);
            const float v = load_w<DT>(p.W, r * p.n + c);
            p.T[r * p.n + k] = v;
            p.Wp[r * p.n + k] = v;
            uint8_t code = p.sf[r * p.kb + c / p.block];
            p.sfp[r * p.n + k] = code > 126 ? 0 : code;      // 0x7F (NaN) and above: a zero scale
        }
}

// One LDLQ panel of P <= 64 columns (P % 16 == 0).  TPR threads per row
// (adjacent lanes), thread k of a row owning columns (64/TPR)k .. (64/TPR)(k+1)-1
// in registers: at column s the owner quantizes it at its fixed scale, writes
// the error to EpT[s][r], and the error reaches the row's other threads by
// shuffle; each thread then updates its targets through up[s][c] = U[k0+s][k0+c]
// (zero for c <= s and past the panel).  Splitting the 64-wide update shortens
// the sequential chain per column.  The CTA's rows of original weights and the
// reciprocal and value of each element's scale code are staged in shared memory
// first, so the owner's step depends on its target alone.  The walk is
// latency-bound (one dependent quantize -> shuffle -> update chain per column), so
// weights with few rows take 16 threads per row (twice the warps in flight) and
// tall ones 8 (fewer shuffles and owner steps per warp).
constexpr int kPanelThreads = 128;
constexpr int64_t kPanelWideRows = 8192;            // below this many rows: 16 threads per row
template <int TPR>
__host__ __device__ constexpr int panel_rows() {
    return kPanelThreads / TPR;
}
template <int TPR>
__host__ __device__ constexpr int panel_smem() {
    return (kP * kP + 128 + 2 * panel_rows<TPR>() * (kP + 1)) * 4 + panel_rows<TPR>() * (kP + 4) * 2;
}

template <int DT, int TPR>
__global__ void __launch_bounds__(kPanelThreads) panel_kernel(LdlqParams p, int64_t k0, int P, float* EpT) {
    constexpr int kPanelTpr = TPR;                    // threads per row
    constexpr int kPanelTargets = kP / TPR;           // targets per thread
    constexpr int kPanelRows = panel_rows<TPR>();
    static_assert(kPanelTargets % 4 == 0 && 16 % kPanelTargets == 0, "a thread's targets are whole float4s in a block");
    extern __shared__ __align__(16) float dsm[];
    float (*up)[kP] = reinterpret_cast<float (*)[kP]>(dsm);                    // [kP][kP]
    float* rtab = dsm + kP * kP;                                               // [128]
    float (*wsm)[kP + 1] = reinterpret_cast<float (*)[kP + 1]>(rtab + 128);    // [kPanelRows][kP + 1] weights
    float (*rsm)[kP + 1] = wsm + kPanelRows;                                   // fl(1/v) of the element's code, or 0
    uint16_t (*vsm)[kP + 4] = reinterpret_cast<uint16_t (*)[kP + 4]>(rsm + kPanelRows);   // f16 bits of v
    for (int e = threadIdx.x; e < kP * kP; e += blockDim.x) {
        const int s = e / kP, c = e % kP;
        up[s][c] = (s < c && c < P) ? p.U[(k0 + s) * p.n + k0 + c] : 0.0f;
    }
    for (int c = threadIdx.x; c < 128; c += blockDim.x)
        rtab[c] = (c >= 1 && c <= 126) ? __frcp_rn(f16bits_to_f32(e4m3_to_f16bits((uint32_t)c))) : 0.0f;
    __syncthreads();                                  // rtab before the row blocks read it
    const float S = __ldg(p.S);
    const float Einv = __frcp_rn(S);
    const bool usable = (S > 0.0f) && isfinite(S) && isfinite(Einv);
    const float E = usable ? Einv : 1.0f;
    const float Sq = usable ? S : 0.0f;               // an unusable S reconstructs zeros (q is a signed zero then)
    const int lane = threadIdx.x & 31;
    const int kq = threadIdx.x % kPanelTpr;           // this thread's share of the columns
    const int rr = threadIdx.x / kPanelTpr;           // row within the CTA's block
    for (int64_t rb = (int64_t)blockIdx.x * kPanelRows; rb < p.rows; rb += (int64_t)gridDim.x * kPanelRows) {
        __syncthreads();                              // rtab written / previous row block done with the row arrays
        {
            float4 wv[kPanelRows * kP / 4 / kPanelThreads];
            uint32_t cv[kPanelRows * kP / 4 / kPanelThreads];
#pragma unroll
            for (int u = 0; u < kPanelRows * kP / 4 / kPanelThreads; u++) {
                const int e = threadIdx.x + kPanelThreads * u, row = e / (kP / 4), j = 4 * (e % (kP / 4));
                const bool ok = rb + row < p.rows && j < P;
                wv[u] = ok ? *reinterpret_cast<const float4*>(p.Wp + (rb + row) * p.n + k0 + j) : make_float4(0, 0, 0, 0);
                cv[u] = ok ? *reinterpret_cast<const uint32_t*>(p.sfp + (rb + row) * p.n + k0 + j) : 0u;
            }
#pragma unroll
            for (int u = 0; u < kPanelRows * kP / 4 / kPanelThreads; u++) {
                const int e = threadIdx.x + kPanelThreads * u, row = e / (kP / 4), j = 4 * (e % (kP / 4));
                const float wq[4] = {wv[u].x, wv[u].y, wv[u].z, wv[u].w};
#pragma unroll
                for (int q = 0; q < 4; q++) {
                    const uint32_t cs = (cv[u] >> (8 * q)) & 0xFFu;
                    wsm[row][j + q] = wq[q];
                    // an unusable S or a zero code: r = 0 turns every target into a signed zero
                    rsm[row][j + q] = usable ? rtab[cs & 127u] : 0.0f;
                    vsm[row][j + q] = e4m3_to_f16bits(cs);
                }
            }
        }
        __syncthreads();
        const int64_t r = rb + rr;
        const bool active = r < p.rows;               // a row's threads share r
        const int c0 = kPanelTargets * kq;
        float t[kPanelTargets];
#pragma unroll
        for (int g = 0; g < kPanelTargets / 4; g++) {
            const float4 v = (active && c0 + 4 * g < P) ? *reinterpret_cast<const float4*>(p.T + r * p.n + k0 + c0 + 4 * g)
                                                        : make_float4(0, 0, 0, 0);
            t[4 * g] = v.x;
            t[4 * g + 1] = v.y;
            t[4 * g + 2] = v.z;
            t[4 * g + 3] = v.w;
        }
        uint32_t packed[kPanelTargets / 4] = {};
#pragma unroll 1
        for (int kb = 0; kb < P / kPanelTargets; kb++) {   // the share whose columns are walked now
            const bool own = kq == kb && active;
            const int src = (lane & ~(kPanelTpr - 1)) | kb;
#pragma unroll
            for (int j = 0; j < kPanelTargets; j++) {
                const int s = kPanelTargets * kb + j;
                // the column's operands do not depend on the targets: loaded ahead of the chain
                const float rs = rsm[rr][s], ws = wsm[rr][s];
                const uint16_t vh = vsm[rr][s];
                float e = 0.0f;
                if (own) {
                    // What = fl(fl(q v) S) with q = RNE_E2M1(fl(y r)), y = fl(t E); q v is
                    // exact, formed by one mixed fma with a +0 addend (a zero q gives +0)
                    const float y = __fmul_rn(t[j], E);
                    uint32_t nib = e2m1x2(__fmul_rn(y, rs), 0.0f) & 0xFu;
                    float qv;
                    asm("{\n\t.reg .b8 b;\n\t.reg .b32 h2;\n\t.reg .b16 ql, qh;\n\t"
                        "cvt.u8.u32 b, %1;\n\tcvt.rn.f16x2.e2m1x2 h2, b;\n\tmov.b32 {ql, qh}, h2;\n\t"
                        "fma.rn.f32.f16 %0, ql, %2, %3;\n\t}"
                        : "=f"(qv) : "r"(nib), "h"(vh), "f"(0.0f));
                    if (y == 0.0f) nib = 0;                // an exactly zero target takes the +0 code
                    e = __fsub_rn(ws, __fmul_rn(qv, Sq));
                    packed[j / 4] |= nib << (8 * (j % 4));
                    EpT[(int64_t)s * p.rows + r] = e;
                }
                e = __shfl_sync(0xffffffffu, e, src);
                const float* us = &up[s][c0];
#pragma unroll
                for (int g = 0; g < kPanelTargets / 4; g++) {
                    const float4 u = *reinterpret_cast<const float4*>(us + 4 * g);
                    t[4 * g + 0] = __fmaf_rn(e, u.x, t[4 * g + 0]);
                    t[4 * g + 1] = __fmaf_rn(e, u.y, t[4 * g + 1]);
                    t[4 * g + 2] = __fmaf_rn(e, u.z, t[4 * g + 2]);
                    t[4 * g + 3] = __fmaf_rn(e, u.w, t[4 * g + 3]);
                }
            }
        }
        if (active && c0 < P) {
            uint8_t* q = p.qb + r * p.n + k0 + c0;    // one byte per column: kPanelTargets bytes
            if constexpr (kPanelTargets == 16)
                *reinterpret_cast<uint4*>(q) = make_uint4(packed[0], packed[1], packed[2], packed[3]);
            else if constexpr (kPanelTargets == 8)
                *reinterpret_cast<uint2*>(q) = make_uint2(packed[0], packed[1]);
            else
                *reinterpret_cast<uint32_t*>(q) = packed[0];
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

// Stream and events of the factorization's look-ahead, one set per device,
// created on the first prepare call on that device and kept for the process.
// The critical chain (diagonal factor, panel solve, next block column) runs on
// `crit`, created with the device's highest priority so its CTAs are placed
// before the pending tiles of the bulk update on the caller's stream.  The
// mutex serialises enqueueing, so the record/wait pairs of two concurrent calls
// cannot interleave.
struct LookAhead {
    cudaStream_t crit = nullptr;
    cudaEvent_t fork = nullptr, panel_done = nullptr, rest_done = nullptr, crit_done = nullptr;
};

cudaError_t lookahead_for_current_device(LookAhead** out, std::unique_lock<std::mutex>* lock) {
    static std::mutex mu;
    static LookAhead state[64];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    *lock = std::unique_lock<std::mutex>(mu);
    LookAhead& la = state[dev];
    if (!la.crit) {
        int least = 0, greatest = 0;
        if ((e = cudaDeviceGetStreamPriorityRange(&least, &greatest)) != cudaSuccess) return e;
        if ((e = cudaStreamCreateWithPriority(&la.crit, cudaStreamNonBlocking, greatest)) != cudaSuccess) return e;
        cudaEvent_t* evs[4] = {&la.fork, &la.panel_done, &la.rest_done, &la.crit_done};
        for (cudaEvent_t* ev : evs)
            if ((e = cudaEventCreateWithFlags(ev, cudaEventDisableTiming)) != cudaSuccess) return e;
    }
    *out = &la;
    return cudaSuccess;
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
    // Look-ahead: the trailing update of panel k is split into the next panel's
    // block column (on the high-priority stream, with the next diagonal factor
    // and panel solve) and the rest (on `s`, overlapping them).  The two
    // updates of one block column from different panels are ordered by events.
    LookAhead* la = nullptr;
    std::unique_lock<std::mutex> lock;
    e = lookahead_for_current_device(&la, &lock);
    if (e != cudaSuccess) return e;
    cudaStream_t c = la->crit;
    if ((e = cudaEventRecord(la->fork, s)) != cudaSuccess) return e;
    if ((e = cudaStreamWaitEvent(c, la->fork, 0)) != cudaSuccess) return e;
    bool have_rest = false;              // rest_done recorded by this call (waits stay inside a capture)
    for (int64_t k0 = 0; k0 < n; k0 += kP) {
        const int nb = (int)imin64(kP, n - k0);
        potrf_kernel<<<1, 256, 0, c>>>(U, n, k0, nb, Linv, status);
        const int64_t rest = n - k0 - nb;
        if (rest > 0) {
            const unsigned tg = (unsigned)imin64((rest + 7) / 8, (int64_t)sms * 8);
            trsm_kernel<<<tg, 256, 0, c>>>(U, n, k0, nb, Linv);
            float* P = U + (k0 + nb) * n + k0;         // the solved panel, rows k0+nb..n-1
            const int64_t nb2 = imin64(kP, rest);      // width of the next panel
            float* C = U + (k0 + nb) * n + k0 + nb;
            if ((e = cudaEventRecord(la->panel_done, c)) != cudaSuccess) return e;
            // the next block column also took the previous panel's rest update
            if (have_rest && (e = cudaStreamWaitEvent(c, la->rest_done, 0)) != cudaSuccess) return e;
            e = update_gemm<false, true, true>(C, n, P, n, P, n, rest, nb2, nb, -1.0f, status, c);
            if (e != cudaSuccess) return e;
            if (rest > nb2) {
                if ((e = cudaStreamWaitEvent(s, la->panel_done, 0)) != cudaSuccess) return e;
                e = update_gemm<false, true, true>(C + nb2 * n + nb2, n, P + nb2 * n, n, P + nb2 * n, n, rest - nb2,
                                                   rest - nb2, nb, -1.0f, status, s);
                if (e != cudaSuccess) return e;
                if ((e = cudaEventRecord(la->rest_done, s)) != cudaSuccess) return e;
                have_rest = true;
            }
        }
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    if ((e = cudaEventRecord(la->crit_done, c)) != cudaSuccess) return e;          // join
    if ((e = cudaStreamWaitEvent(s, la->crit_done, 0)) != cudaSuccess) return e;
    lock.unlock();
    diag_d_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(U, n, D);
    flip_kernel<<<rg, 256, 0, s>>>(U, n);
    zero_diag_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(U, n);
    return cudaGetLastError();
}

// Workspace: T and Wp [rows, n] f32, qb and sfp [rows, n] bytes, two EpT
// [kLdlqPanel, rows] f32 (alternating between super-panels), inv [n].
size_t ldlq_quantize_workspace(int64_t rows, int64_t n) {
    auto up = [](int64_t b) { return (b + 255) / 256 * 256; };
    return (size_t)(2 * up(rows * n * 4) + 2 * up(rows * n) + 2 * up((int64_t)kLdlqPanel * rows * 4) + up(n * 4));
}

// Columns in super-panels of kLdlqPanel (256): each 64-column panel is walked by
// panel_kernel and its errors update the rest of the super-panel at once (K = 64);
// after the super-panel, GEMMs with K = 256 update every later column, so the
// targets are read and written once per 256 columns.  Look-ahead: that update
// is split into the next super-panel's columns, which run with its panel walks
// on the high-priority stream, and the rest, which runs on `s` concurrently
// with them; the super-panels' errors alternate between two EpT buffers.
cudaError_t launch_ldlq_quantize(LdlqParams p, int dtype, uint8_t* codes, void* ws, int sms, cudaStream_t s) {
    if (p.rows <= 0 || p.n <= 0) return cudaSuccess;
    auto up = [](int64_t b) { return (b + 255) / 256 * 256; };
    char* w = static_cast<char*>(ws);
    const int64_t mat4 = up(p.rows * p.n * 4), mat1 = up(p.rows * p.n);
    p.T = reinterpret_cast<float*>(w);
    p.Wp = reinterpret_cast<float*>(w + mat4);
    p.qb = reinterpret_cast<uint8_t*>(w + 2 * mat4);
    p.sfp = reinterpret_cast<uint8_t*>(w + 2 * mat4 + mat1);
    const int64_t ep = up((int64_t)kLdlqPanel * p.rows * 4);
    float* EpTs[2] = {reinterpret_cast<float*>(w + 2 * mat4 + 2 * mat1),
                      reinterpret_cast<float*>(w + 2 * mat4 + 2 * mat1 + ep)};
    int32_t* inv = reinterpret_cast<int32_t*>(w + 2 * mat4 + 2 * mat1 + 2 * ep);
    cudaError_t e = cudaMemsetAsync(inv, 0, (size_t)p.n * 4, s);
    if (e != cudaSuccess) return e;
    invperm_kernel<<<(unsigned)((p.n + 255) / 256), 256, 0, s>>>(p.perm, p.n, inv, p.status);
    const unsigned rg = (unsigned)imin64(p.rows, (int64_t)sms * 8);
    if (dtype == 0)
        gather_w_kernel<0><<<rg, 256, 0, s>>>(p);
    else
        gather_w_kernel<1><<<rg, 256, 0, s>>>(p);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    static std::atomic<bool> attr_set[64];        // per device: the shared-memory opt-in is done
    int dev = 0;
    e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64 || !attr_set[dev].load(std::memory_order_acquire)) {
        e = cudaFuncSetAttribute(panel_kernel<0, 8>, cudaFuncAttributeMaxDynamicSharedMemorySize, panel_smem<8>());
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(panel_kernel<1, 8>, cudaFuncAttributeMaxDynamicSharedMemorySize, panel_smem<8>());
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(panel_kernel<0, 16>, cudaFuncAttributeMaxDynamicSharedMemorySize, panel_smem<16>());
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(panel_kernel<1, 16>, cudaFuncAttributeMaxDynamicSharedMemorySize, panel_smem<16>());
        if (e != cudaSuccess) return e;
        if (dev >= 0 && dev < 64) attr_set[dev].store(true, std::memory_order_release);
    }
    const bool wide = p.rows < kPanelWideRows;
    const int prow = wide ? panel_rows<16>() : panel_rows<8>();
    const unsigned pg = (unsigned)imin64((p.rows + prow - 1) / prow, (int64_t)sms * 16);
    LookAhead* la = nullptr;
    std::unique_lock<std::mutex> lock;
    e = lookahead_for_current_device(&la, &lock);
    if (e != cudaSuccess) return e;
    cudaStream_t c = la->crit;
    if ((e = cudaEventRecord(la->fork, s)) != cudaSuccess) return e;
    if ((e = cudaStreamWaitEvent(c, la->fork, 0)) != cudaSuccess) return e;
    bool have_rest = false;              // rest_done recorded by this call (waits stay inside a capture)
    int sp = 0;
    for (int64_t s0 = 0; s0 < p.n; s0 += kLdlqPanel, sp++) {
        const int64_t span = imin64(kLdlqPanel, p.n - s0);
        float* EpT = EpTs[sp & 1];
        for (int64_t k0 = s0; k0 < s0 + span; k0 += kP) {
            const int P = (int)imin64(kP, s0 + span - k0);
            float* Ek = EpT + (k0 - s0) * p.rows;
            if (wide) {
                if (dtype == 0) panel_kernel<0, 16><<<pg, kPanelThreads, panel_smem<16>(), c>>>(p, k0, P, Ek);
                else panel_kernel<1, 16><<<pg, kPanelThreads, panel_smem<16>(), c>>>(p, k0, P, Ek);
            } else {
                if (dtype == 0) panel_kernel<0, 8><<<pg, kPanelThreads, panel_smem<8>(), c>>>(p, k0, P, Ek);
                else panel_kernel<1, 8><<<pg, kPanelThreads, panel_smem<8>(), c>>>(p, k0, P, Ek);
            }
            e = cudaGetLastError();
            if (e != cudaSuccess) return e;
            const int64_t rest_in = s0 + span - (k0 + P);
            if (rest_in > 0) {
                e = update_gemm<true, false, false>(p.T + k0 + P, p.n, Ek, p.rows, p.U + k0 * p.n + k0 + P, p.n,
                                                    p.rows, rest_in, P, 1.0f, p.status, c);
                if (e != cudaSuccess) return e;
            }
        }
        const int64_t rest = p.n - (s0 + span);
        if (rest > 0) {
            const int64_t next = imin64(kLdlqPanel, rest);
            if ((e = cudaEventRecord(la->panel_done, c)) != cudaSuccess) return e;
            // the next super-panel's columns also took the previous rest update, and
            // that update read the EpT buffer the next super-panel overwrites
            if (have_rest && (e = cudaStreamWaitEvent(c, la->rest_done, 0)) != cudaSuccess) return e;
            e = update_gemm<true, false, false>(p.T + s0 + span, p.n, EpT, p.rows, p.U + s0 * p.n + s0 + span, p.n,
                                                p.rows, next, (int)span, 1.0f, p.status, c);
            if (e != cudaSuccess) return e;
            if (rest > next) {
                if ((e = cudaStreamWaitEvent(s, la->panel_done, 0)) != cudaSuccess) return e;
                e = update_gemm<true, false, false>(p.T + s0 + span + next, p.n, EpT, p.rows,
                                                    p.U + s0 * p.n + s0 + span + next, p.n, p.rows, rest - next,
                                                    (int)span, 1.0f, p.status, s);
                if (e != cudaSuccess) return e;
                if ((e = cudaEventRecord(la->rest_done, s)) != cudaSuccess) return e;
                have_rest = true;
            }
        }
    }
    if ((e = cudaEventRecord(la->crit_done, c)) != cudaSuccess) return e;          // join
    if ((e = cudaStreamWaitEvent(s, la->crit_done, 0)) != cudaSuccess) return e;
    lock.unlock();
    pack_kernel<<<rg, 256, 0, s>>>(p.qb, inv, p.rows, p.n, codes, p.status);
    return cudaGetLastError();
}

}  // namespace nvfp4
