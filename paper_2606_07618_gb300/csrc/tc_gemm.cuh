// fp32 GEMM on the 5th-generation tensor cores (tcgen05) for the LDLQ error
// feedback (Appendix A.2, GPTQ paragraph): C[M, N] += alpha * A[M, K] B[K, N]
// with fp32 operands, fp32 accumulation, three TF32 products per term
// ("3xTF32"):
//
//   a = a_hi + a_lo with a_hi = a with its low 13 mantissa bits cleared (a TF32
//   value) and a_lo = a - a_hi (exact in fp32); the tensor core reads TF32, so
//   a_lo contributes its top 11 bits.  a*b ~ a_hi*b_hi + a_hi*b_lo + a_lo*b_hi,
//   dropping a_lo*b_lo (~2^-22 relative): products to ~2^-21 relative, against
//   2^-24 for one fp32 FMA.
//
// One CTA of 256 threads computes a 128 x 128 tile of C:
//   * operand stages of K = 32 fp32 (128 bytes, one swizzle row) are loaded
//     by TMA (cp.async.bulk.tensor) into a three-stage ring of
//     128-byte-swizzled shared memory, two stages ahead, completion signalled
//     on an mbarrier;
//   * all threads split each staged value into hi and lo tiles in the K-major
//     128-byte-swizzled layout the MMA reads (double buffered);
//   * one thread issues 4 k-steps x 3 tcgen05.mma.kind::tf32 (M = 128, N = 128,
//     K = 8) accumulating into a 128-column fp32 accumulator in tensor memory,
//     and tcgen05.commit signals the stage's completion on a second mbarrier
//     (the buffer is reloaded only after that);
//   * the C tile arrives by TMA during the last stage (into ring slots no
//     stage needs any more); the epilogue reads the accumulator with
//     tcgen05.ld (warps w and w + 4 read TMEM lanes 32(w%4).. = rows, 64
//     columns each), forms
//     C = fma(alpha, acc, C) in shared memory and TMA stores the tile.
// Operands may be K-major (K contiguous) or MN-major (M or N contiguous); the
// shared-memory descriptors and the instruction descriptor say which.
//
// The MMA reads both operands K-major.  An operand stored MN-major (M or N
// contiguous) is loaded by TMA as four 32 x 32 boxes and transposed by the
// split into the K-major layout; a K-major one is split in place order.
//
// Every mbarrier wait is bounded by the global timer (1 s).  On a timeout the
// CTA sets bit 4 (16) of the status word, stops issuing, waits (bounded again)
// for the copies and MMAs it has in flight, frees its tensor memory and
// returns without writing C.
#pragma once
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

namespace nvfp4 {
namespace tc {

constexpr int kTileM = 128;
constexpr int kTileN = 128;
constexpr int kStageK = 32;                               // fp32 per swizzle row (128 bytes)
constexpr int kThreads = 256;                             // 8 warps split; warps w, w + 4 share TMEM lanes 32(w % 4)..
constexpr int kOpBytes = kTileM * kStageK * 4;            // one operand tile: 16 KB
constexpr int kRawStages = 3;                             // TMA landing ring: raw A, raw B
constexpr int kRawBytes = 2 * kOpBytes;
constexpr int kSplitBufs = 2;                             // MMA operands: A hi, A lo, B hi, B lo
constexpr int kSplitBytes = 4 * kOpBytes;
constexpr int kSmemBytes = kRawStages * kRawBytes + kSplitBufs * kSplitBytes + 1024 + 64;  // + align + barriers
constexpr int kTmemCols = kTileN;                         // fp32 accumulator columns
constexpr unsigned long long kWaitNs = 1000000000ull;
constexpr int kStatusTimeout = 16;

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ unsigned long long now_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// ---- mbarriers
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}
// Wait for the phase with the given parity to complete; false after ~1 s.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
    if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long t0 = now_ns();
    while (!mbar_try_wait(bar, parity))
        if (now_ns() - t0 > kWaitNs) return false;
    return true;
}

// ---- TMA: a 2-D box of the tensor map into shared memory, completion on bar
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int c0, int c1, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
        ::"r"(dst), "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, int c0, int c1, uint32_t src) {
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.tile.bulk_group [%0, {%1, %2}], [%3];"
                 ::"l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(src)
                 : "memory");
}
__device__ __forceinline__ void tma_store_commit_and_wait() {
    asm volatile("cp.async.bulk.commit_group;" ::: "memory");
    asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}

// ---- tcgen05
__device__ __forceinline__ void tmem_alloc(uint32_t holder, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(holder), "r"(ncols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// Generic-proxy writes to shared memory become visible to the async proxy
// (the tensor core reading its operands).
__device__ __forceinline__ void fence_proxy_async() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void mma_tf32(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                         uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n\t}"
        ::"r"(d_tmem), "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
__device__ __forceinline__ void mma_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
                 : "memory");
}
// 32 consecutive fp32 accumulator columns of this thread's TMEM lane.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
        "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr)
        : "memory");
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 32; i++) v[i] = __uint_as_float(r[i]);
}

// Shared-memory matrix descriptor of a 128-byte-swizzled operand tile:
// start address >> 4 (bits 0-13), leading-dimension byte offset >> 4 (16-29),
// stride-dimension byte offset >> 4 (32-45), descriptor version 1 (46-47),
// base offset 0 (tiles are 1024-byte aligned), swizzle mode 2 = 128 bytes
// (61-63).  K-major: rows of 128 bytes, SBO = 1024 between 8-row groups.
// MN-major: 128-byte chunks along M (or N), LBO between those chunks, SBO =
// 1024 between 8-row groups along K.
__device__ __forceinline__ uint64_t smem_desc(uint32_t addr, uint32_t lbo, uint32_t sbo) {
    uint64_t d = (uint64_t)((addr >> 4) & 0x3FFFu);
    d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
    d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
}

// Instruction descriptor of tcgen05.mma.kind::tf32 with both operands
// K-major: D fp32 (bits 4-5 = 1), A and B TF32 (bits 7-9, 10-12 = 2), N >> 3
// (bits 17-22), M >> 4 (bits 24-28).
__host__ __device__ constexpr uint32_t idesc_tf32() {
    return (1u << 4) | (2u << 7) | (2u << 10) | ((uint32_t)(kTileN >> 3) << 17) | ((uint32_t)(kTileM >> 4) << 24);
}

}  // namespace tc
}  // namespace nvfp4

namespace nvfp4 {
namespace tc {

__device__ __forceinline__ void split4(const float4& x, float4& h, float4& l) {
    h.x = __uint_as_float(__float_as_uint(x.x) & 0xFFFFE000u);
    h.y = __uint_as_float(__float_as_uint(x.y) & 0xFFFFE000u);
    h.z = __uint_as_float(__float_as_uint(x.z) & 0xFFFFE000u);
    h.w = __uint_as_float(__float_as_uint(x.w) & 0xFFFFE000u);
    l.x = __fsub_rn(x.x, h.x);
    l.y = __fsub_rn(x.y, h.y);
    l.z = __fsub_rn(x.z, h.z);
    l.w = __fsub_rn(x.w, h.w);
}

// Byte offset of element (r, k) -- row r of 128 (M or N), column k of 32 --
// in a K-major 128-byte-swizzled tile: 128-byte rows, the 16-byte chunk index
// XOR-ed with the row index modulo 8 (the layout TMA writes and the MMA reads).
__device__ __forceinline__ uint32_t kmajor_off(int r, int k) {
    return (uint32_t)(r * 128 + ((((k >> 2) ^ r) & 7) << 4) + ((k & 3) << 2));
}
// Byte offset of element (r, k) in an MN-major tile as four TMA boxes of 32
// rows (k) of 128 bytes (32 consecutive r), 4 KB each, 128-byte swizzled.
__device__ __forceinline__ uint32_t mnmajor_off(int r, int k) {
    return (uint32_t)((r >> 5) * 4096 + k * 128 + (((((r & 31) >> 2) ^ k) & 7) << 4) + ((r & 3) << 2));
}

// Split one operand tile (128 rows x 32 k) from the raw landing buffer into
// the K-major hi and lo tiles.  K-major raw: same positions, linear float4s.
// MN-major raw: each of the 256 threads takes one 4 x 4 block (rows 4*bm..,
// k 4*bk..), reads four float4 along r, transposes in registers and writes
// four float4 along k.  bm = lane and bk = (lane % 8 + warp) % 8 cover the 256
// blocks once; within a quarter warp the read chunk (bm ^ k) % 8 and the
// written chunk (bk ^ r) % 8 are then both permutations of 0..7, so neither
// side has bank conflicts.
template <bool MN>
__device__ __forceinline__ void split_tile(const uint8_t* raw, uint8_t* hi, uint8_t* lo, int tid) {
    if (!MN) {
        const float4* x = reinterpret_cast<const float4*>(raw);
        float4* h = reinterpret_cast<float4*>(hi);
        float4* l = reinterpret_cast<float4*>(lo);
#pragma unroll 4
        for (int i = tid; i < kOpBytes / 16; i += kThreads) {
            float4 a, b;
            split4(x[i], a, b);
            h[i] = a;
            l[i] = b;
        }
    } else {
        static_assert(kThreads == 256, "one 4 x 4 block per thread");
        {
            const int bm = tid & 31, bk = ((tid & 7) + (tid >> 5)) & 7;
            float v[4][4];                                   // v[kk][i]: k = 4bk + kk, r = 4bm + i
#pragma unroll
            for (int kk = 0; kk < 4; kk++) {
                const float4 q = *reinterpret_cast<const float4*>(raw + mnmajor_off(4 * bm, 4 * bk + kk));
                v[kk][0] = q.x;
                v[kk][1] = q.y;
                v[kk][2] = q.z;
                v[kk][3] = q.w;
            }
#pragma unroll
            for (int i = 0; i < 4; i++) {
                const float4 x = make_float4(v[0][i], v[1][i], v[2][i], v[3][i]);
                float4 a, b;
                split4(x, a, b);
                const uint32_t o = kmajor_off(4 * bm + i, 4 * bk);
                *reinterpret_cast<float4*>(hi + o) = a;
                *reinterpret_cast<float4*>(lo + o) = b;
            }
        }
    }
}

// C[M, N] (row-major, ldc) += alpha * op(A) op(B) with op(A) [M, K], op(B) [K, N].
// A_MN: A is stored [K][M] (row k at A + k*lda), else [M][K]; B_MN: B is stored
// [K][N], else [N][K].  The tensor maps describe A and B with a box of 32 fp32
// along the contiguous dimension (128 bytes, 128-byte swizzle) by 32 (MN-major)
// or 128 (K-major) along the other.  LOWER skips tiles entirely above the
// diagonal.
//
// Stage s: TMA fills raw[s % 3] (issued two stages ahead, once the split of
// stage s - 3 has read it); the split of s fills buf[s % 2] once the MMAs of
// stage s - 2 have read it (their commit barrier); the MMAs of s run while
// stage s + 1 is split.
template <bool A_MN, bool B_MN, bool LOWER>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                const __grid_constant__ CUtensorMap tmC, int64_t M, int64_t N, int K, float alpha, int* status) {
    extern __shared__ uint8_t smem_raw[];
    __shared__ int s_abort, s_committed, s_arrived, s_issued;
    __shared__ uint32_t s_tmem;
    const int64_t m0 = (int64_t)blockIdx.y * kTileM, n0 = (int64_t)blockIdx.x * kTileN;
    if (LOWER && n0 > m0 + kTileM - 1) return;
    const int nst = (K + kStageK - 1) / kStageK;
    if (nst <= 0) return;
    uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* raw0 = base;
    uint8_t* buf0 = base + kRawStages * kRawBytes;
    uint64_t* bars = reinterpret_cast<uint64_t*>(buf0 + kSplitBufs * kSplitBytes);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const uint32_t full0 = smem_u32(bars), done0 = smem_u32(bars + kRawStages);
    const uint32_t cbar = smem_u32(bars + kRawStages + kSplitBufs);

    if (warp == 0) tmem_alloc(smem_u32(&s_tmem), kTmemCols);
    if (tid == 0) {
        for (int b = 0; b < kRawStages; b++) mbar_init(full0 + 8 * b, 1);
        for (int b = 0; b < kSplitBufs; b++) mbar_init(done0 + 8 * b, 1);
        mbar_init(cbar, 1);
        s_abort = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = s_tmem;

    auto issue = [&](int s) {                                    // thread 0: stage s's operand loads
        const int r = s % kRawStages, k0 = s * kStageK;
        const uint32_t bar = full0 + 8 * r, st = smem_u32(raw0 + r * kRawBytes);
        mbar_expect_tx(bar, kRawBytes);
        if (A_MN) {
#pragma unroll
            for (int j = 0; j < kTileM / 32; j++) tma_load_2d(st + j * 4096, &tmA, (int)(m0 + 32 * j), k0, bar);
        } else {
            tma_load_2d(st, &tmA, k0, (int)m0, bar);
        }
        if (B_MN) {
#pragma unroll
            for (int j = 0; j < kTileN / 32; j++)
                tma_load_2d(st + kOpBytes + j * 4096, &tmB, (int)(n0 + 32 * j), k0, bar);
        } else {
            tma_load_2d(st + kOpBytes, &tmB, k0, (int)n0, bar);
        }
    };
    constexpr uint32_t idesc = idesc_tf32();
    // box j (16 KB) of the C tile: boxes 0-1 and 2-3 in the raw slots of
    // stages nst and nst + 1, free from the last stage on
    auto c_box = [&](int j) {
        return raw0 + ((nst + (j >> 1)) % kRawStages) * kRawBytes + (j & 1) * kOpBytes;
    };
    int issued = 0, arrived = 0, committed = 0, c_issued = 0;   // thread 0's view
    if (tid == 0) {
        for (int s = 0; s < 2 && s < nst; s++) issue(s);
        issued = nst < 2 ? nst : 2;
    }
    for (int s = 0; s < nst; s++) {
        const int r = s % kRawStages, b = s & 1;
        // raw[(s + 2) % 3] was last read by the split of stage s - 1 (done:
        // every thread passed the barrier at the end of that iteration)
        if (tid == 0 && s + 2 < nst) {
            issue(s + 2);
            issued = s + 3;
        }
        if (tid == 0 && s == nst - 1) {
            // the C tile (four 32-column boxes) into the raw slots no stage
            // uses any more, overlapping the last split and MMAs
            mbar_expect_tx(cbar, kTileM * kTileN * 4);
#pragma unroll
            for (int j = 0; j < kTileN / 32; j++)
                tma_load_2d(smem_u32(c_box(j)), &tmC, (int)(n0 + 32 * j), (int)m0, cbar);
            c_issued = 1;
        }
        bool ok = mbar_wait(full0 + 8 * r, (s / kRawStages) & 1);
        if (ok && tid == 0) arrived = s + 1;
        // buf[b] was read by the MMAs of stage s - 2
        if (ok && s >= 2) ok = mbar_wait(done0 + 8 * b, ((s - 2) >> 1) & 1);
        if (ok) {
            const uint8_t* raw = raw0 + r * kRawBytes;
            uint8_t* buf = buf0 + b * kSplitBytes;
            split_tile<A_MN>(raw, buf, buf + kOpBytes, tid);
            split_tile<B_MN>(raw + kOpBytes, buf + 2 * kOpBytes, buf + 3 * kOpBytes, tid);
        } else {
            atomicOr(&s_abort, 1);
        }
        fence_proxy_async();
        __syncthreads();
        if (s_abort) break;                                      // uniform: read after the barrier
        if (tid == 0) {
            tc_fence_after();
            const uint32_t st = smem_u32(buf0 + b * kSplitBytes);
#pragma unroll
            for (int kk = 0; kk < kStageK / 8; kk++) {           // the k-step's 32 bytes of each 128-byte row
                const uint64_t ahi = smem_desc(st + kk * 32, 16, 1024);
                const uint64_t alo = smem_desc(st + kOpBytes + kk * 32, 16, 1024);
                const uint64_t bhi = smem_desc(st + 2 * kOpBytes + kk * 32, 16, 1024);
                const uint64_t blo = smem_desc(st + 3 * kOpBytes + kk * 32, 16, 1024);
                mma_tf32(tmem, ahi, bhi, idesc, (s | kk) != 0);
                mma_tf32(tmem, ahi, blo, idesc, 1);
                mma_tf32(tmem, alo, bhi, idesc, 1);
            }
            mma_commit(done0 + 8 * b);
            committed = s + 1;
        }
    }
    if (tid == 0) {
        s_committed = committed;
        s_arrived = arrived;
        s_issued = issued + c_issued * 1000;
    }
    __syncthreads();
    const int cm = s_committed;
    const bool c_loaded = s_issued >= 1000;
    // the last commit completes after every MMA this CTA issued
    if (cm > 0 && !mbar_wait(done0 + 8 * ((cm - 1) & 1), ((cm - 1) >> 1) & 1)) atomicOr(&s_abort, 1);
    if (c_loaded && !mbar_wait(cbar, 0)) atomicOr(&s_abort, 1);
    if (tid == 0)                                                // copies still in flight: bounded wait
        for (int s = s_arrived; s < s_issued % 1000; s++)
            (void)mbar_wait(full0 + 8 * (s % kRawStages), (s / kRawStages) & 1);
    tc_fence_after();
    __syncthreads();
    if (!s_abort && c_loaded) {
        // C += alpha * acc in shared memory (thread = row; the box rows are
        // 128-byte swizzled, so the eight lanes of a quarter warp touch eight
        // distinct 16-byte chunks), then TMA stores the tile (out-of-range
        // rows and columns are not written)
        const int q = warp & 3, r = 32 * q + lane;               // TMEM lane quarter q = rows 32q..32q+31
#pragma unroll 1
        for (int j = 2 * (warp >> 2); j < 2 * (warp >> 2) + 2; j++) {   // warps 0-3: boxes 0-1, 4-7: 2-3
            float v[32];
            tmem_ld32(tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(32 * j), v);   // .sync.aligned
            uint8_t* box = c_box(j) + r * 128;
#pragma unroll
            for (int g = 0; g < 8; g++) {
                float4* q = reinterpret_cast<float4*>(box + (((g ^ r) & 7) << 4));
                float4 o = *q;
                o.x = __fmaf_rn(alpha, v[4 * g], o.x);
                o.y = __fmaf_rn(alpha, v[4 * g + 1], o.y);
                o.z = __fmaf_rn(alpha, v[4 * g + 2], o.z);
                o.w = __fmaf_rn(alpha, v[4 * g + 3], o.w);
                *q = o;
            }
        }
        fence_proxy_async();
        __syncthreads();
        if (tid == 0) {
#pragma unroll
            for (int j = 0; j < kTileN / 32; j++) tma_store_2d(&tmC, (int)(n0 + 32 * j), (int)m0, smem_u32(c_box(j)));
            tma_store_commit_and_wait();
        }
    } else if (s_abort && tid == 0 && status) {
        atomicOr(status, kStatusTimeout);
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, kTmemCols);
}

}  // namespace tc
}  // namespace nvfp4

#include <atomic>

namespace nvfp4 {
namespace tc {

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

// cuTensorMapEncodeTiled from the driver, looked up once through the runtime
// (no link against libcuda); nullptr if the driver does not provide it.
inline EncodeTiledFn encode_fn() {
    static std::atomic<void*> fn{nullptr};
    static std::atomic<int> looked{0};
    if (!looked.load(std::memory_order_acquire)) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) !=
                cudaSuccess ||
            q != cudaDriverEntryPointSuccess)
            p = nullptr;
        fn.store(p, std::memory_order_release);
        looked.store(1, std::memory_order_release);
    }
    return reinterpret_cast<EncodeTiledFn>(fn.load(std::memory_order_acquire));
}

// A row-major fp32 matrix of `outer` rows of `inner` elements (row stride ld
// elements) as a TMA tensor map with a box of 32 x box_outer and 128-byte
// swizzle; out-of-range elements of a box read as zero.
inline bool make_map(CUtensorMap* m, const float* ptr, int64_t inner, int64_t outer, int64_t ld, uint32_t box_outer) {
    const EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    const cuuint64_t dims[2] = {(cuuint64_t)inner, (cuuint64_t)outer};
    const cuuint64_t strides[1] = {(cuuint64_t)ld * 4};
    const cuuint32_t box[2] = {32, box_outer};
    const cuuint32_t estr[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float*>(ptr), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Whether launch_gemm below can take these operands: 16-byte aligned bases
// and row strides, sizes within the tensor map's limits.
inline bool gemm_eligible(const float* A, int64_t lda, const float* B, int64_t ldb, int64_t M, int64_t N, int K) {
    auto al = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; };
    return al(A) && al(B) && lda % 4 == 0 && ldb % 4 == 0 && M > 0 && N > 0 && K > 0 && M < (1ll << 31) &&
           N < (1ll << 31) && lda < (1ll << 35) && ldb < (1ll << 35) && encode_fn() != nullptr;
}
inline bool c_eligible(const float* C, int64_t ldc) {
    return (reinterpret_cast<uintptr_t>(C) & 15) == 0 && ldc % 4 == 0 && ldc < (1ll << 35);
}

// C[M, N] += alpha * op(A) op(B) on the tensor cores (3xTF32).  A_MN: A stored
// [K][M], else [M][K]; B_MN: B stored [K][N], else [N][K].  Returns
// cudaErrorNotSupported (nothing launched) when gemm_eligible is false.
template <bool A_MN, bool B_MN, bool LOWER>
cudaError_t launch_gemm(float* C, int64_t ldc, const float* A, int64_t lda, const float* B, int64_t ldb, int64_t M,
                        int64_t N, int K, float alpha, int* status, cudaStream_t s) {
    if (M <= 0 || N <= 0 || K <= 0) return cudaSuccess;
    if (!gemm_eligible(A, lda, B, ldb, M, N, K) || !c_eligible(C, ldc)) return cudaErrorNotSupported;
    CUtensorMap ta, tb, tcm;
    const bool ok = (A_MN ? make_map(&ta, A, M, K, lda, 32) : make_map(&ta, A, K, M, lda, kTileM)) &&
                    (B_MN ? make_map(&tb, B, N, K, ldb, 32) : make_map(&tb, B, K, N, ldb, kTileN)) &&
                    make_map(&tcm, C, N, M, ldc, kTileM);
    if (!ok) return cudaErrorNotSupported;
    static std::atomic<bool> attr_set[64];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64 || !attr_set[dev].load(std::memory_order_acquire)) {
        e = cudaFuncSetAttribute(gemm_kernel<A_MN, B_MN, LOWER>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 kSmemBytes);
        if (e != cudaSuccess) return e;
        if (dev >= 0 && dev < 64) attr_set[dev].store(true, std::memory_order_release);
    }
    const dim3 grid((unsigned)((N + kTileN - 1) / kTileN), (unsigned)((M + kTileM - 1) / kTileM));
    gemm_kernel<A_MN, B_MN, LOWER><<<grid, kThreads, kSmemBytes, s>>>(ta, tb, tcm, M, N, K, alpha, status);
    return cudaGetLastError();
}

}  // namespace tc
}  // namespace nvfp4
