// Device helpers for the NVFP4 ScaleSweep kernels (sm_103a).
//
// Number formats (Sec. 3.2, Appendix A of the ScaleSweep paper): FP4 E2M1
// elements {0, 0.5, 1, 1.5, 2, 3, 4, 6} with a sign bit, FP8 E4M3 block scales
// (bias 7, codes 1..126 positive finite, 0x7F NaN), FP32 global scale.
// Rounding is done by the native converts, which round to nearest-even and
// saturate: cvt.rn.satfinite.e2m1x2.f32 (element codes) and
// cvt.rn.satfinite.e4m3x2.f32 (AbsMax scale).  Every float op whose rounding the
// arithmetic contract fixes is written with an explicit _rn intrinsic or PTX
// instruction so that nvcc cannot contract it into an FMA.
#pragma once
#include <cstdint>
#include <cuda_runtime.h>

namespace nvfp4 {

typedef unsigned long long u64;

__device__ __forceinline__ u64 pack2(float lo, float hi) {
    u64 r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}
__device__ __forceinline__ void unpack2(u64 v, float& lo, float& hi) {
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ u64 mul2(u64 a, u64 b) {
    u64 d;
    asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}
__device__ __forceinline__ u64 fma2(u64 a, u64 b, u64 c) {
    u64 d;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
    return d;
}

// Two fp32 -> one byte of two E2M1 codes (RNE, saturating at 6): `hi` goes to
// the upper nibble, `lo` to the lower nibble.
__device__ __forceinline__ uint32_t e2m1x2(float lo, float hi) {
    uint32_t r;
    asm("{\n\t.reg .b8 q;\n\t"
        "cvt.rn.satfinite.e2m1x2.f32 q, %1, %2;\n\t"
        "cvt.u32.u8 %0, q;\n\t}"
        : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}

// One candidate step on an element pair: t = fl(y*r) (packed), q = RNE_E2M1(t),
// e = fl(y - q*v) computed as fma(q, -v, y) with q and -v as exact f16
// operands, returned packed {e_lo, e_hi}.  nv = f16 bit pattern of -v_c.
__device__ __forceinline__ u64 cand_err2(u64 y2, u64 r2, uint16_t nv) {
    u64 e2;
    asm("{\n\t"
        ".reg .b64 t2;\n\t"
        ".reg .b32 tl, th, yl, yh, h2, el, eh;\n\t"
        ".reg .b16 ql, qh;\n\t"
        ".reg .b8 q;\n\t"
        "mul.rn.f32x2 t2, %1, %2;\n\t"
        "mov.b64 {tl, th}, t2;\n\t"
        "cvt.rn.satfinite.e2m1x2.f32 q, th, tl;\n\t"
        "cvt.rn.f16x2.e2m1x2 h2, q;\n\t"
        "mov.b32 {ql, qh}, h2;\n\t"
        "mov.b64 {yl, yh}, %1;\n\t"
        "fma.rn.f32.f16 el, ql, %3, yl;\n\t"
        "fma.rn.f32.f16 eh, qh, %3, yh;\n\t"
        "mov.b64 %0, {el, eh};\n\t"
        "}"
        : "=l"(e2) : "l"(y2), "l"(r2), "h"(nv));
    return e2;
}

// E4M3 code -> f16 bit pattern of its value (exact), via the native decode.
__device__ __forceinline__ uint16_t e4m3_to_f16bits(uint32_t code) {
    uint32_t h2;
    uint16_t c16 = (uint16_t)(code & 0xFF);
    asm("cvt.rn.f16x2.e4m3x2 %0, %1;" : "=r"(h2) : "h"(c16));
    return (uint16_t)(h2 & 0xFFFF);
}

__device__ __forceinline__ float f16bits_to_f32(uint16_t h) {
    float f;
    asm("cvt.f32.f16 %0, %1;" : "=f"(f) : "h"(h));
    return f;
}

// RN_E4M3 (ties to even, saturating at 448) of a non-negative fp32, as a code.
__device__ __forceinline__ uint32_t e4m3_rn_code(float s) {
    uint16_t d;
    asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(d) : "f"(0.0f), "f"(s));
    return (uint32_t)(d & 0xFF);
}

// floor_E4M3 of a non-negative fp32 as a code: the largest code in 0..126 with
// value <= s (Sec. 3.1 notation, s_base^FP8 of Sec. 4.2.2).  Normal E4M3 values
// truncate the fp32 mantissa to 3 bits; subnormal ones are floor(s * 2^9).
__device__ __forceinline__ int e4m3_floor_code(float s) {
    if (s >= 448.0f) return 126;
    if (!(s >= 0.001953125f)) return 0;           // below 2^-9 (or NaN)
    uint32_t b = __float_as_uint(s);
    int e = (int)(b >> 23) - 127;
    if (e >= -6) return ((e + 7) << 3) | (int)((b >> 20) & 7u);
    return (int)__fmul_rn(s, 512.0f);                // 1..7, exact scaling then truncation
}

// Byte offset of scale (row r, scale column k) in the 128x4-atom swizzled
// layout read by block-scaled MMA (kpad4 = ceil(kblocks/4)).
__device__ __forceinline__ int64_t swizzle_offset(int64_t r, int64_t k, int64_t kpad4) {
    return ((r >> 7) * kpad4 + (k >> 2)) * 512 + (r & 31) * 16 + ((r >> 5) & 3) * 4 + (k & 3);
}

// Streaming 16-byte load that bypasses L1 allocation (each byte is read once).
__device__ __forceinline__ uint4 ld_stream16(const void* p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
    return v;
}
__device__ __forceinline__ uint4 ld_ro16(const void* p) {
    uint4 v;
    asm volatile("ld.global.nc.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
    return v;
}

// Programmatic dependent launch: the running grid lets a kernel launched after
// it with cudaLaunchAttributeProgrammaticStreamSerialization be scheduled once
// every CTA of this grid has executed launch_dependents (or exited); that
// kernel's griddepcontrol.wait returns once this grid has completed and its
// writes are visible (and at once when it was launched the ordinary way).
__device__ __forceinline__ void grid_launch_dependents() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void grid_dependency_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

__device__ __forceinline__ float bf16lo(uint32_t u) { return __uint_as_float(u << 16); }
__device__ __forceinline__ float bf16hi(uint32_t u) { return __uint_as_float(u & 0xFFFF0000u); }

}  // namespace nvfp4
