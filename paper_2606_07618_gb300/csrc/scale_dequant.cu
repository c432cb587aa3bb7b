// Global scale S = amax / (6 D) (Sec. 3.2 with D = 448; Sec. 4.2.1 with D = 256)
// and NVFP4 dequantisation x_hat = q * s * S (Sec. 3.2).
//
// amax is a two-launch reduction: a persistent grid of streaming 16-byte loads
// writes one partial maximum (and a NaN/inf flag) per CTA into the caller's
// workspace, then a single CTA folds the partials and writes S on the device.
// No atomics and no zero-initialised state, so back-to-back calls on one
// workspace need nothing in between.  Max is exact, so the order is free.
// The folding CTA is a programmatic dependent launch: it is scheduled while
// the partial grid drains and waits (griddepcontrol.wait) for that grid's
// writes, which takes its launch latency off the critical path.
#include <cuda_bf16.h>

#include "nvfp4_device.cuh"
#include "nvfp4_kernels.h"

namespace nvfp4 {

__device__ __forceinline__ void amax_acc(float v, float& m, int& bad) {
    if (!isfinite(v)) bad = 1;
    m = fmaxf(m, fabsf(v));                  // fmaxf drops NaN, keeps inf
}

template <int DT>
__global__ void __launch_bounds__(512) amax_partial_kernel(const void* x, int64_t n, float* part_max,
                                                           int* part_bad) {
    constexpr int PER = DT == 0 ? 8 : 4;      // elements per 16-byte vector
    const int64_t nvec = n / PER;
    float m = 0.0f;
    int bad = 0;
    const uint4* xv = static_cast<const uint4*>(x);
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    auto fold = [&](const uint4& u) {
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int j = 0; j < 4; j++) {
            if (DT == 0) {
                amax_acc(bf16lo(w[j]), m, bad);
                amax_acc(bf16hi(w[j]), m, bad);
            } else {
                amax_acc(__uint_as_float(w[j]), m, bad);
            }
        }
    };
    int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    // two independent 16-byte loads in flight per thread; with 2048 threads
    // per SM that keeps ~10 MB in flight across the GPU
    for (; i + stride < nvec; i += 2 * stride) {
        const uint4 u0 = ld_stream16(xv + i), u1 = ld_stream16(xv + i + stride);
        fold(u0);
        fold(u1);
    }
    if (i < nvec) fold(ld_stream16(xv + i));
    // tail elements (n not a multiple of the vector width)
    if (blockIdx.x == 0 && threadIdx.x < (int)(n - nvec * PER)) {
        const int64_t i = nvec * PER + threadIdx.x;
        float v = DT == 0 ? __uint_as_float((uint32_t)(static_cast<const uint16_t*>(x)[i]) << 16)
                          : static_cast<const float*>(x)[i];
        amax_acc(v, m, bad);
    }
    // every load of this CTA has returned: let the folding kernel be scheduled
    grid_launch_dependents();
    // non-negative floats order like their bit patterns
    uint32_t mb = __reduce_max_sync(0xffffffffu, __float_as_uint(m));
    int anybad = __reduce_or_sync(0xffffffffu, (unsigned)bad);
    __shared__ uint32_t sm[16];
    __shared__ int sb[16];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) {
        sm[warp] = mb;
        sb[warp] = anybad;
    }
    __syncthreads();
    if (warp == 0) {
        uint32_t v = lane < (int)(blockDim.x >> 5) ? sm[lane] : 0u;
        int b = lane < (int)(blockDim.x >> 5) ? sb[lane] : 0;
        v = __reduce_max_sync(0xffffffffu, v);
        b = __reduce_or_sync(0xffffffffu, (unsigned)b);
        if (lane == 0) {
            part_max[blockIdx.x] = __uint_as_float(v);
            part_bad[blockIdx.x] = b;
        }
    }
}

__global__ void __launch_bounds__(256) amax_final_kernel(const float* part_max, const int* part_bad, int nparts,
                                                         float fp8_div, float* S_out, int* status_dev) {
    // launched as a programmatic dependent of amax_partial_kernel: wait until
    // that grid has finished and its partials are visible (a no-op otherwise)
    grid_dependency_wait();
    uint32_t v = 0u;
    int b = 0;
    for (int i = threadIdx.x; i < nparts; i += blockDim.x) {
        v = max(v, __float_as_uint(part_max[i]));
        b |= part_bad[i];
    }
    v = __reduce_max_sync(0xffffffffu, v);
    b = __reduce_or_sync(0xffffffffu, (unsigned)b);
    __shared__ uint32_t sm[8];
    __shared__ int sb[8];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) {
        sm[warp] = v;
        sb[warp] = b;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        uint32_t m = 0;
        int bad = 0;
        for (int i = 0; i < (int)(blockDim.x >> 5); i++) {
            m = max(m, sm[i]);
            bad |= sb[i];
        }
        const float amax = __uint_as_float(m);
        S_out[0] = __fdiv_rn(amax, __fmul_rn(6.0f, fp8_div));
        if (status_dev && bad) atomicOr(status_dev, 1);
    }
}

// The folding CTA, allowed to start before amax_partial_kernel has drained.
static cudaError_t launch_final(const float* part_max, const int* part_bad, int nparts, float fp8_div,
                                float* S_out, int* status_dev, cudaStream_t s) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(1);
    cfg.blockDim = dim3(256);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, amax_final_kernel, part_max, part_bad, nparts, fp8_div, S_out, status_dev);
}

static cudaError_t launch_partial(const void* x, int dtype, int64_t n, float* part_max, int* part_bad, int grid,
                                  int threads, cudaStream_t s) {
    if (dtype == 0)
        amax_partial_kernel<0><<<grid, threads, 0, s>>>(x, n, part_max, part_bad);
    else
        amax_partial_kernel<1><<<grid, threads, 0, s>>>(x, n, part_max, part_bad);
    return cudaGetLastError();
}

cudaError_t launch_global_scale(const void* x, int dtype, int64_t n, float fp8_div, float* S_out,
                                int* status_dev, void* ws, int sms, cudaStream_t s) {
    float* part_max = static_cast<float*>(ws);
    int* part_bad = reinterpret_cast<int*>(part_max + kAmaxParts);
    // 512-thread CTAs, 4 per SM, two loads in flight each: measured fastest of
    // 128/256/512 threads x 1/2/4/8 loads and of 32-byte loads on GB300
    constexpr int kThreads = 512;
    const int per = dtype == 0 ? 8 : 4;
    const int64_t nvec = n / per;
    int64_t grid = (nvec + kThreads * 2 - 1) / (kThreads * 2);
    if (grid > (int64_t)sms * 4) grid = (int64_t)sms * 4;
    if (grid > kAmaxParts) grid = kAmaxParts;
    if (grid < 1) grid = 1;
    cudaError_t e = launch_partial(x, dtype, n, part_max, part_bad, (int)grid, kThreads, s);
    if (e != cudaSuccess) return e;
    return launch_final(part_max, part_bad, (int)grid, fp8_div, S_out, status_dev, s);
}

cudaError_t launch_global_scale_parts(const void* x, int dtype, int64_t n, float fp8_div, float* S_out,
                                      int* status_dev, float* part_max, int* part_bad, int grid, cudaStream_t s) {
    cudaError_t e = launch_partial(x, dtype, n, part_max, part_bad, grid, 256, s);
    if (e != cudaSuccess) return e;
    return launch_final(part_max, part_bad, grid, fp8_div, S_out, status_dev, s);
}

// ---------------------------------------------------------------------------
// Dequantisation: a chunk is 8 bf16 or 4 fp32 outputs (one 16-byte store), and
// lane l of a warp takes chunks l, l+32, ..., l+224 of the warp's 256-chunk
// tile, so every store instruction writes 512 contiguous bytes and every code
// load reads 128 (bf16) or 64 (fp32) contiguous bytes.  All 8 code words and
// scale bytes of a tile are loaded before its first store: the reads are
// small beside the writes, and that keeps enough of them in flight.
// q and s are decoded by the native converts into f16, q*s is exact in f16 (at
// most 7 significant bits, within range), then one fp32 multiply by S rounds once.
constexpr int kDequantUnroll = 8;      // chunks per lane per tile: of 2, 4, 8, 16 and a one-chunk
                                       // prefetch loop, 8 was fastest

// Scale index of element e0.  Swizzled layout: block e0 >> bshift (block =
// 2^bshift), its row and scale column from one multiply-high division by kb
// (kbd) when the block count fits 32 bits (two Qwen2.5-72B-shaped matrices: 0.293 ->
// 0.214 ms against two integer divisions).  Linear layout: e0 / block as
// written measured faster than the shift (0.210 against 0.226 ms on the Qwen
// shapes): the slower index spaces the scale-byte loads behind the code loads.
template <int OUT_BF16>
__global__ void __launch_bounds__(256) dequant_kernel(DequantParams p, FastDiv kbd, int bshift) {
    constexpr int EPT = OUT_BF16 ? 8 : 4;          // elements per thread
    const float S = __ldg(p.S);
    const int64_t nchunk = p.nseg * (16 / EPT);
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    auto scale_offset = [&](int64_t e0) -> int64_t {
        if (!p.swizzled) return e0 / p.block;
        const int64_t blk = e0 >> bshift;           // element index -> scale block
        int64_t row, kbi;
        if (p.narrow) {
            const uint32_t b32 = (uint32_t)blk, k32 = (uint32_t)p.kb;
            const uint32_t t = __umulhi(b32, kbd.mul), r32 = (t + ((b32 - t) >> kbd.s1)) >> kbd.s2;
            row = r32;
            kbi = b32 - r32 * k32;
        } else {
            row = blk / p.kb;
            kbi = blk - row * p.kb;
        }
        return swizzle_offset(row, kbi, p.kpad4);
    };
    auto load_codes = [&](int64_t c) -> uint32_t {
        return EPT == 8 ? __ldg(reinterpret_cast<const uint32_t*>(p.codes) + c)
                        : (uint32_t)__ldg(reinterpret_cast<const uint16_t*>(p.codes) + c);
    };
    int64_t c0 = ((int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31)) * kDequantUnroll + (threadIdx.x & 31);
    for (; c0 < nchunk; c0 += stride * kDequantUnroll) {
        uint32_t cwv[kDequantUnroll];
        uint8_t scv[kDequantUnroll];
#pragma unroll
        for (int u = 0; u < kDequantUnroll; u++) {
            const int64_t c = c0 + 32 * u;
            if (c < nchunk) {
                cwv[u] = load_codes(c);
                scv[u] = __ldg(p.sf + scale_offset(c * EPT));
            }
        }
#pragma unroll
        for (int u = 0; u < kDequantUnroll; u++) {
            const int64_t c = c0 + 32 * u;
            if (c >= nchunk) break;
            const uint32_t cw = cwv[u];
            const uint32_t vv = (uint32_t)e4m3_to_f16bits(scv[u]) * 0x10001u;
            float out[EPT];
#pragma unroll
            for (int j = 0; j < EPT / 2; j++) {
                uint32_t q2, prod;
                const uint16_t byte = (uint16_t)((cw >> (8 * j)) & 0xFFu);
                asm("{\n\t.reg .b8 b;\n\tcvt.u8.u16 b, %1;\n\tcvt.rn.f16x2.e2m1x2 %0, b;\n\t}" : "=r"(q2) : "h"(byte));
                asm("mul.rn.f16x2 %0, %1, %2;" : "=r"(prod) : "r"(q2), "r"(vv));
                out[2 * j] = __fmul_rn(f16bits_to_f32((uint16_t)(prod & 0xFFFF)), S);
                out[2 * j + 1] = __fmul_rn(f16bits_to_f32((uint16_t)(prod >> 16)), S);
            }
            if (OUT_BF16) {
                uint32_t o[4];
#pragma unroll
                for (int j = 0; j < 4; j++) {
                    const __nv_bfloat16 a = __float2bfloat16_rn(out[2 * j]), b = __float2bfloat16_rn(out[2 * j + 1]);
                    o[j] = (uint32_t)__bfloat16_as_ushort(a) | ((uint32_t)__bfloat16_as_ushort(b) << 16);
                }
                reinterpret_cast<uint4*>(p.out)[c] = make_uint4(o[0], o[1], o[2], o[3]);
            } else {
                reinterpret_cast<float4*>(p.out)[c] = make_float4(out[0], out[1], out[2], out[3]);
            }
        }
    }
}

cudaError_t launch_dequantize(const DequantParams& p, int out_dtype, int sms, cudaStream_t s) {
    if (p.nseg <= 0) return cudaSuccess;
    const int64_t nchunk = p.nseg * (out_dtype == 0 ? 2 : 4);
    // one tile per warp, up to 4 CTAs of 256 threads per SM (faster than 8)
    int64_t grid = (nchunk + 256 * kDequantUnroll - 1) / (256 * kDequantUnroll);
    if (grid > (int64_t)sms * 4) grid = (int64_t)sms * 4;
    const FastDiv kbd = (p.swizzled && p.narrow && p.kb > 0) ? make_fast_div((uint32_t)p.kb) : FastDiv{1, 0, 0};
    int bshift = 0;
    while ((1 << bshift) < p.block) bshift++;
    if (out_dtype == 0)
        dequant_kernel<1><<<(int)grid, 256, 0, s>>>(p, kbd, bshift);
    else
        dequant_kernel<0><<<(int)grid, 256, 0, s>>>(p, kbd, bshift);
    return cudaGetLastError();
}

}  // namespace nvfp4
