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
// 1..126 and a poison entry {+inf, -inf} elsewhere.  A poison candidate's loss
// is inf or NaN, so it never wins the strict "<" -- this lets the default
// windows run a fixed, fully unrolled loop over [I0+lo, I0+hi] with no clamping
// (those windows always contain a real code).  Custom windows clamp instead.
#include "nvfp4_device.cuh"
#include "nvfp4_kernels.h"

namespace nvfp4 {

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

template <int DT>
__device__ __forceinline__ void raw_to_float(const Raw& r, float (&xv)[16]) {
    if (DT == 0) {
        const uint32_t u[8] = {r.a.x, r.a.y, r.a.z, r.a.w, r.b.x, r.b.y, r.b.z, r.b.w};
#pragma unroll
        for (int j = 0; j < 8; j++) {
            xv[2 * j] = bf16lo(u[j]);
            xv[2 * j + 1] = bf16hi(u[j]);
        }
    } else {
        const uint32_t u[16] = {r.a.x, r.a.y, r.a.z, r.a.w, r.b.x, r.b.y, r.b.z, r.b.w,
                                r.c.x, r.c.y, r.c.z, r.c.w, r.d.x, r.d.y, r.d.z, r.d.w};
#pragma unroll
        for (int j = 0; j < 16; j++) xv[j] = __uint_as_float(u[j]);
    }
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
    if (SEGS >= 2) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 1));
    if (SEGS >= 4) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 2));
    return v;
}

// n / d for 32-bit n by multiply-high and shifts (Granlund-Montgomery).
__device__ __forceinline__ uint32_t fast_div(uint32_t n, const FastDiv& d) {
    const uint32_t t = __umulhi(n, d.mul);
    return (t + ((n - t) >> d.s1)) >> d.s2;
}

#ifndef NVFP4_QMINB
#define NVFP4_QMINB 1
#endif
#ifndef NVFP4_CAND_UNROLL
#define NVFP4_CAND_UNROLL 16
#endif
constexpr int kCandUnroll = NVFP4_CAND_UNROLL;

// FIX = 1: default window (fixed length, unrolled, poison-padded table).
template <int DT, int METHOD, int OBJ, int BLOCK, int FIX>
__global__ void __launch_bounds__(256, NVFP4_QMINB) quantize_kernel(QuantParams p) {
    constexpr int SEGS = BLOCK / 16;
    constexpr int FIX_LO = (OBJ == 0 && BLOCK == 16) ? -3 : -8;
    constexpr int FIX_K = 7 - FIX_LO + 1;
    __shared__ Cand tab[kTabN];
    build_table(tab);
    __syncthreads();

    const float S = __ldg(p.S);
    const float E = __frcp_rn(S);
    const bool usable = (S > 0.0f) && isfinite(S) && isfinite(E);
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

        float xv[16];
        if (valid) {
            raw_to_float<DT>(cur, xv);
        } else {
#pragma unroll
            for (int i = 0; i < 16; i++) xv[i] = 0.0f;
        }
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

        u64 y2[8];
        float m = 0.0f;
#pragma unroll
        for (int j = 0; j < 8; j++) {
            const float a = usable ? __fmul_rn(xv[2 * j], E) : xv[2 * j];
            const float b = usable ? __fmul_rn(xv[2 * j + 1], E) : xv[2 * j + 1];
            m = fmaxf(m, fmaxf(fabsf(a), fabsf(b)));
            y2[j] = pack2(a, b);
        }
        m = group_max<SEGS>(m);

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

        const bool zero = !usable || !(m > 0.0f);
        float best = __int_as_float(0x7f800000);
        int bestc = 0;
        if (METHOD == 0) {
            const float sbase = __fdiv_rn(m, 6.0f);
            const int I0 = e4m3_floor_code(sbase);
            if (FIX) {
                const Cand* tb = tab + (I0 + FIX_LO + kTabOff);
                int bk = 0;
#pragma unroll kCandUnroll
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
                const int clo = min(max(I0 + p.win_lo, 1), 126);
                const int chi = min(max(I0 + p.win_hi, 1), 126);
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
                uint32_t acc = 0;
#pragma unroll
                for (int j = 0; j < 4; j++) {
                    float a, b;
                    unpack2(mul2(y2[4 * h + j], r2), a, b);
                    acc |= e2m1x2(a, b) << (8 * j);
                }
                packed[h] = acc;
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

// Zero the padding bytes of the swizzled layout (rows past `rows`, scale
// columns past `kb`); only launched when the shape is not 128x4-aligned.
__global__ void swizzle_pad_kernel(uint8_t* sf, int64_t rows, int64_t kb, int64_t kpad4, int64_t rows_pad) {
    const int64_t total = rows_pad * kpad4 * 4;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = i / (kpad4 * 4), k = i - r * (kpad4 * 4);
        if (r >= rows || k >= kb) sf[swizzle_offset(r, k, kpad4)] = 0;
    }
}

template <int DT, int METHOD, int OBJ, int BLOCK, int FIX>
static cudaError_t launch_one(const QuantParams& p, int sms, cudaStream_t s) {
    static int occ = 0;
    if (!occ) {
        int b = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&b, quantize_kernel<DT, METHOD, OBJ, BLOCK, FIX>, 256, 0) !=
                cudaSuccess || b < 1)
            b = 1;
        occ = b;
    }
    const int64_t threads_needed = (p.nseg + 31) & ~(int64_t)31;
    int64_t grid = (threads_needed + 255) / 256;
    const int64_t cap = (int64_t)sms * occ;
    if (grid > cap) grid = cap;
    quantize_kernel<DT, METHOD, OBJ, BLOCK, FIX><<<(int)grid, 256, 0, s>>>(p);
    return cudaGetLastError();
}

template <int DT, int METHOD, int OBJ, int BLOCK>
static cudaError_t dispatch_fix(const QuantParams& p, bool fix, int sms, cudaStream_t s) {
    if (METHOD == 0 && !fix) return launch_one<DT, METHOD, OBJ, BLOCK, 0>(p, sms, s);
    return launch_one<DT, METHOD, OBJ, BLOCK, 1>(p, sms, s);
}

template <int DT, int METHOD, int OBJ>
static cudaError_t dispatch_block(const QuantParams& p, bool fix, int block, int sms, cudaStream_t s) {
    switch (block) {
        case 16: return dispatch_fix<DT, METHOD, OBJ, 16>(p, fix, sms, s);
        case 32: return dispatch_fix<DT, METHOD, OBJ, 32>(p, fix, sms, s);
        default: return dispatch_fix<DT, METHOD, OBJ, 64>(p, fix, sms, s);
    }
}

template <int DT, int METHOD>
static cudaError_t dispatch_obj(const QuantParams& p, int obj, bool fix, int block, int sms, cudaStream_t s) {
    if (obj == 1) return dispatch_block<DT, METHOD, 1>(p, fix, block, sms, s);
    return dispatch_block<DT, METHOD, 0>(p, fix, block, sms, s);
}

FastDiv make_fast_div(uint32_t d) {
    FastDiv f;
    uint32_t l = 0;
    while (l < 32 && (1ull << l) < d) l++;
    f.mul = (uint32_t)(((1ull << 32) * ((1ull << l) - d)) / d + 1);
    f.s1 = l < 1 ? l : 1;
    f.s2 = l > 0 ? l - 1 : 0;
    return f;
}

cudaError_t launch_quantize(const QuantParams& p_in, int dtype, int method, int obj, int block, int sms,
                            cudaStream_t s) {
    QuantParams p = p_in;
    const int def_lo = (obj == 0 && block == 16) ? -3 : -8;
    const bool fix = (method != 0) || (p.win_lo == def_lo && p.win_hi == 7);
    p.need_rowcol = (p.sf_swizzled != nullptr) || (obj == 1);
    if (p.narrow) p.kb_div = make_fast_div((uint32_t)p.kb);
    if (p.nseg > 0) {
        cudaError_t e;
        if (dtype == 0) {
            if (method == 0) e = dispatch_obj<0, 0>(p, obj, fix, block, sms, s);
            else if (method == 1) e = dispatch_block<0, 1, 0>(p, fix, block, sms, s);
            else e = dispatch_obj<0, 2>(p, obj, fix, block, sms, s);
        } else {
            if (method == 0) e = dispatch_obj<1, 0>(p, obj, fix, block, sms, s);
            else if (method == 1) e = dispatch_block<1, 1, 0>(p, fix, block, sms, s);
            else e = dispatch_obj<1, 2>(p, obj, fix, block, sms, s);
        }
        if (e != cudaSuccess) return e;
    }
    if (p.sf_swizzled && (p.rows % 128 != 0 || p.kb % 4 != 0) && p.rows > 0 && p.kb > 0) {
        const int64_t rows_pad = (p.rows + 127) / 128 * 128;
        const int64_t total = rows_pad * p.kpad4 * 4;
        int64_t grid = (total + 255) / 256;
        if (grid > (int64_t)sms * 8) grid = (int64_t)sms * 8;
        swizzle_pad_kernel<<<(int)grid, 256, 0, s>>>(p.sf_swizzled, p.rows, p.kb, p.kpad4, rows_pad);
        return cudaGetLastError();
    }
    return cudaSuccess;
}

}  // namespace nvfp4
