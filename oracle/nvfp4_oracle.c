/*
 * NVFP4 / ScaleSweep CPU oracle -- TEST INFRASTRUCTURE ONLY.
 *
 * This file is the plain, slow, obviously-correct reference that the CUDA
 * library is checked against.  Only tests/, __graft_entry__.smoke() and the
 * cpu_baseline / reference legs of bench.py may load it.  It shares no code,
 * header, table or constant with the CUDA path (paper_2606_07618_gb300/csrc).
 *
 * Everything follows "ScaleSweep: Accurate NVFP4 Post-Training Quantization of
 * LLMs via Block Scale Initialization":
 *   - number formats: Sec. 3.2 (E2M1 grid) and Appendix A (EeMm values v(c,a,b),
 *     bias 2^(e-1)-1, bit pattern I(v) = c*2^(e+m) + a*2^m + b);
 *   - NVFP4 triple (q, s, S) and reconstruction q*s*S: Sec. 3.2;
 *   - AbsMax initialisation: Sec. 3.2 (S = amax/(448*6), s_k = RN_FP8(.), q = RN_FP4(.));
 *   - weighted loss L(s;x,w) = sum w_i (x_i - RN_FP4(s)(x_i))^2: Sec. 3.1;
 *   - global scale S = amax/(256*6): Sec. 4.2.1;
 *   - normalisation by S, base scale s_base = max|x|/6, s_base^FP8 = floor_FP8(s_base),
 *     sweep windows [-3,7] (MSE) and [-8,7] (WMSE) in bit-pattern space: Sec. 4.2.2;
 *   - 4/6: also try the scale mapping the block max to 4, keep the lower error:
 *     Sec. 2 (FP4 quantization paragraph);
 *   - optimal real-valued block scale by enumerating quadratic segments: Appendix C.
 *
 * Arithmetic contract (readings where the paper fixes no arithmetic):
 *   E  = fl32(1/S);  y_i = fl32(x_i * E)                       (normalise by S)
 *   m  = max|y_i|;   s_base = fl32(m / 6);  I0 = floor_E4M3(s_base) as a code
 *   per candidate code c: v_c = E4M3 value (exact), r_c = fl32(1/v_c),
 *                         t_i = fl32(y_i * r_c),  q_i = RNE_E2M1(t_i) (|t|>6 -> 6),
 *                         L_c = sum_i w_i (y_i - q_i*v_c)^2   in float64
 *   argmin over the window, exact ties -> lowest code.
 *   Zero rule: a block with m == 0, a block holding a NaN, or whose m is
 *   infinite or >= 2^48, and every block when S or fl32(1/S) is unusable, gets
 *   scale code 0 and nibbles carrying only the sign of y (the paper defines no
 *   output for these; the bound keeps fp32 losses finite on the GPU side).
 * The code decisions (q_i, I0, AbsMax rounding) are taken in float32, the
 * precision the GPU kernels decide in; losses are accumulated in float64.
 * Float ops here must not be contracted into FMAs: build with -ffp-contract=off.
 *
 * Parity pins (tests/test_oracle_*.py): format tables, RNE/floor/RN by brute
 * force and against torch's float8_e4m3fn, Lemma-4.2/4.3 tables and the convex
 * certificates recomputed, bounded = exhaustive sweep, ScaleSweep <= AbsMax and
 * <= 4/6, Appendix-C optimum <= every FP8 result, closed-form blocks.
 * The 128x4 swizzled scale layout (oracle_swizzle_scales) is not defined by the
 * paper; it follows NVIDIA's block-scaling layout and is pinned on the GPU
 * against cuBLASLt's NVFP4 block-scaled GEMM (tests/test_gpu_swizzle_pin.py).
 */
#include <math.h>
#include <stdint.h>
#include <stddef.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* ------------------------------------------------------------------------- */
/* Appendix A: EeMm value of a code (sign c, exponent field a, mantissa b).   */
/* ------------------------------------------------------------------------- */
static double eemm_value(int e, int m, int code)
{
    int M = 1 << m;
    int c = (code >> (e + m)) & 1;
    int a = (code >> m) & ((1 << e) - 1);
    int b = code & (M - 1);
    int bias = (1 << (e - 1)) - 1;
    double v;
    if (a != 0)
        v = ldexp(1.0 + (double)b / (double)M, a - bias);
    else
        v = ldexp((double)b / (double)M, 1 - bias);
    return c ? -v : v;
}

double oracle_e2m1_value(int code) { return eemm_value(2, 1, code & 0xF); }

/* E4M3 as used for NVFP4 block scales: code 0x7F (and 0xFF) is NaN, so the
 * positive finite values are codes 0..126 (126 non-zero candidates, Sec. 4.2.2). */
double oracle_e4m3_value(int code)
{
    code &= 0xFF;
    if ((code & 0x7F) == 0x7F) return NAN;
    return eemm_value(4, 3, code);
}

/* Bit-pattern integer I(v) of a positive E4M3 value is its code (Appendix A). */

/* RNE to the E2M1 grid: nearest grid point, ties to the even code (mantissa
 * bit 0), magnitudes above 6 saturate to 6, sign taken from signbit(t). */
int oracle_e2m1_rne(float t)
{
    int sign = signbit(t) ? 8 : 0;
    double a = fabs((double)t);
    if (a >= 6.0) return sign | 7;   /* satfinite; also avoids float64 distance ties for huge |t| */
    int best = 0;
    double bd = INFINITY;
    for (int k = 0; k < 8; k++) {
        double d = fabs(a - oracle_e2m1_value(k));
        if (d < bd || (d == bd && (k % 2) == 0)) {
            best = k;
            bd = d;
        }
    }
    return sign | best;
}

/* floor_FP8: largest code in 0..126 whose value does not exceed s (Sec. 3.1
 * notation); s >= 448 gives 126, s < 2^-9 gives 0. */
int oracle_e4m3_floor(float s)
{
    int best = 0;
    for (int c = 1; c <= 126; c++)
        if (oracle_e4m3_value(c) <= (double)s) best = c;
    return best;
}

/* RN_FP8 with ties to the even code, saturating to 448 (code 126). */
int oracle_e4m3_rn(float s)
{
    double a = (double)s;
    if (a >= 448.0) return 126;      /* satfinite */
    int best = 0;
    double bd = INFINITY;
    for (int c = 0; c <= 126; c++) {
        double d = fabs(a - oracle_e4m3_value(c));
        if (d < bd || (d == bd && (c % 2) == 0)) {
            best = c;
            bd = d;
        }
    }
    return best;
}

/* ------------------------------------------------------------------------- */
/* Global scale (Sec. 3.2 with D = 448, Sec. 4.2.1 with D = 256).            */
/* S = fl32(amax / fl32(6*D)).  *nonfinite = 1 if any input is NaN or inf.   */
/* ------------------------------------------------------------------------- */
int oracle_global_scale(const float* x, int64_t n, float D, float* S_out, int* nonfinite)
{
    float amax = 0.0f;
    int bad = 0;
    for (int64_t i = 0; i < n; i++) {
        float v = x[i];
        if (isnan(v) || isinf(v)) { bad = 1; if (isnan(v)) continue; }
        float a = fabsf(v);
        if (a > amax) amax = a;
    }
    float sixD = 6.0f * D;
    *S_out = amax / sixD;
    if (nonfinite) *nonfinite = bad;
    return 0;
}

/* ------------------------------------------------------------------------- */
/* Block quantisation.                                                        */
/* ------------------------------------------------------------------------- */
enum { ORACLE_SCALESWEEP = 0, ORACLE_ABSMAX = 1, ORACLE_FOUR_SIX = 2 };
enum { ORACLE_MSE = 0, ORACLE_WMSE = 1 };

/* Loss of one candidate code c on one block (Sec. 3.1, weighted loss in the
 * S-normalised domain of Sec. 4.2.2).  Also writes the E2M1 codes if asked. */
static double block_loss(const float* y, const float* w, int n, int c, uint8_t* qcodes)
{
    double v = oracle_e4m3_value(c);
    float vf = (float)v;          /* exact: every E4M3 value is an fp32 value */
    float r = 1.0f / vf;          /* fl32(1/v_c) */
    double L = 0.0;
    for (int i = 0; i < n; i++) {
        float t = y[i] * r;       /* fl32(y_i * r_c) */
        int qc = oracle_e2m1_rne(t);
        double q = oracle_e2m1_value(qc);
        double e = (double)y[i] - q * v;
        double wi = w ? (double)w[i] : 1.0;
        L += wi * e * e;
        if (qcodes) qcodes[i] = (uint8_t)qc;
    }
    return L;
}

static int clampi(int v, int lo, int hi) { return v < lo ? lo : (v > hi ? hi : v); }

/*
 * Quantise a [rows, cols] fp32 tensor (bf16 inputs are converted exactly
 * beforehand) into NVFP4 with blocks of `block` consecutive elements of a row.
 *
 *   method: 0 ScaleSweep, 1 AbsMax, 2 four-over-six.
 *   objective: 0 MSE (w ignored), 1 WMSE with w[row*w_row_stride + col].
 *   win_lo/win_hi: bit-pattern offsets around I0 (ScaleSweep only).
 *   codes: [rows, cols/2] bytes, element 2j in the low nibble, 2j+1 in the high.
 *   sf:    [rows, cols/block] E4M3 codes.
 *   best/second: optional [nblocks] float64 losses of the chosen and of the best
 *                other candidate (second = +inf if the window has one code).
 *   cand: optional [nblocks][cand_stride] float64 loss per window candidate,
 *         slot k for code c_lo + k, NaN past the window end; cand_lo gets c_lo.
 * Returns 0, or -1 on bad arguments.
 */
int oracle_quantize(int method, const float* x, int64_t rows, int64_t cols, int block,
                    float S, int objective, const float* w, int64_t w_row_stride,
                    int win_lo, int win_hi,
                    uint8_t* codes, uint8_t* sf, double* best, double* second,
                    double* cand, int cand_stride, int32_t* cand_lo, int nthreads)
{
    if (block <= 0 || block > 64 || cols % block != 0 || cols % 2 != 0) return -1;
    if (win_lo > win_hi) return -1;
    if (objective == ORACLE_WMSE && !w) return -1;
    int64_t kb = cols / block;
    int64_t nblocks = rows * kb;
    float E = 1.0f / S;
    int usable = (S > 0.0f) && isfinite(S) && isfinite(E);
#ifdef _OPENMP
    if (nthreads <= 0) nthreads = omp_get_max_threads();
#pragma omp parallel for schedule(dynamic, 256) num_threads(nthreads)
#endif
    for (int64_t blk = 0; blk < nblocks; blk++) {
        int64_t row = blk / kb, kbi = blk % kb;
        const float* xb = x + row * cols + kbi * block;
        const float* wb = (objective == ORACLE_WMSE) ? (w + row * w_row_stride + kbi * block) : NULL;
        float y[64];
        uint8_t q[64], qbest[64];
        float m = 0.0f;
        int has_nan = 0;
        for (int i = 0; i < block; i++) {
            y[i] = usable ? xb[i] * E : xb[i];
            float a = fabsf(y[i]);
            if (isnan(a)) has_nan = 1;
            else if (a > m) m = a;
        }
        int chosen = 0;
        double Lbest = INFINITY, Lsecond = INFINITY;
        int clo = 0, chi = -1;
        for (int i = 0; i < block; i++) qbest[i] = signbit(y[i]) ? 8 : 0;
        if (!usable || m == 0.0f || has_nan || !(m < 0x1p48f)) {
            /* Zero rule (zero, non-finite or out-of-range block, or unusable S):
             * scale 0, nibbles keep only the sign. */
            chosen = 0;
            Lbest = 0.0;
            if (objective == ORACLE_WMSE) {
                Lbest = 0.0;
                for (int i = 0; i < block; i++) Lbest += (double)wb[i] * (double)y[i] * (double)y[i];
            } else {
                for (int i = 0; i < block; i++) Lbest += (double)y[i] * (double)y[i];
            }
        } else {
            float sbase = m / 6.0f;                 /* fl32(m/6) */
            if (method == ORACLE_SCALESWEEP) {
                int I0 = oracle_e4m3_floor(sbase);
                clo = clampi(I0 + win_lo, 1, 126);
                chi = clampi(I0 + win_hi, 1, 126);
                for (int c = clo; c <= chi; c++) {
                    double L = block_loss(y, wb, block, c, q);
                    if (cand && c - clo < cand_stride) cand[blk * cand_stride + (c - clo)] = L;
                    if (L < Lbest) {
                        Lsecond = Lbest;
                        Lbest = L;
                        chosen = c;
                        memcpy(qbest, q, (size_t)block);
                    } else if (L < Lsecond) {
                        Lsecond = L;
                    }
                }
            } else {
                int c6 = oracle_e4m3_rn(sbase);
                if (c6 < 1) c6 = 1;
                chosen = c6;
                Lbest = block_loss(y, wb, block, c6, qbest);
                if (method == ORACLE_FOUR_SIX) {
                    float s4 = m / 4.0f;            /* fl32(m/4) */
                    int c4 = oracle_e4m3_rn(s4);
                    if (c4 < 1) c4 = 1;
                    double L4 = block_loss(y, wb, block, c4, q);
                    if (L4 < Lbest) {
                        Lsecond = Lbest;
                        Lbest = L4;
                        chosen = c4;
                        memcpy(qbest, q, (size_t)block);
                    } else {
                        Lsecond = L4;
                    }
                }
            }
        }
        if (cand) {
            for (int k = (chi >= clo ? chi - clo + 1 : 0); k < cand_stride; k++)
                cand[blk * cand_stride + k] = NAN;
            if (cand_lo) cand_lo[blk] = clo;
        }
        sf[row * kb + kbi] = (uint8_t)chosen;
        uint8_t* cb = codes + row * (cols / 2) + kbi * (block / 2);
        for (int j = 0; j < block / 2; j++)
            cb[j] = (uint8_t)((qbest[2 * j] & 0xF) | ((qbest[2 * j + 1] & 0xF) << 4));
        if (best) best[blk] = Lbest;
        if (second) second[blk] = Lsecond;
    }
    return 0;
}

/* Loss of a given scale code on every block, and optionally the packed
 * nibbles it yields (used to score and check a GPU pick on a near-tie). */
int oracle_block_losses_at(const float* x, int64_t rows, int64_t cols, int block, float S,
                           int objective, const float* w, int64_t w_row_stride,
                           const uint8_t* sf_codes, double* out, uint8_t* codes_out, int nthreads)
{
    if (block <= 0 || block > 64 || cols % block != 0) return -1;
    int64_t kb = cols / block, nblocks = rows * kb;
    float E = 1.0f / S;
    int usable = (S > 0.0f) && isfinite(S) && isfinite(E);
#ifdef _OPENMP
    if (nthreads <= 0) nthreads = omp_get_max_threads();
#pragma omp parallel for schedule(dynamic, 256) num_threads(nthreads)
#endif
    for (int64_t blk = 0; blk < nblocks; blk++) {
        int64_t row = blk / kb, kbi = blk % kb;
        const float* xb = x + row * cols + kbi * block;
        const float* wb = (objective == ORACLE_WMSE) ? (w + row * w_row_stride + kbi * block) : NULL;
        float y[64];
        uint8_t q[64];
        for (int i = 0; i < block; i++) y[i] = usable ? xb[i] * E : xb[i];
        int c = sf_codes[blk] & 0x7F;
        if (c == 0 || c == 127) {
            double L = 0.0;
            for (int i = 0; i < block; i++) {
                L += (wb ? (double)wb[i] : 1.0) * (double)y[i] * (double)y[i];
                q[i] = signbit(y[i]) ? 8 : 0;
            }
            out[blk] = L;
        } else {
            out[blk] = block_loss(y, wb, block, c, q);
        }
        if (codes_out) {
            uint8_t* cb = codes_out + row * (cols / 2) + kbi * (block / 2);
            for (int j = 0; j < block / 2; j++)
                cb[j] = (uint8_t)((q[2 * j] & 0xF) | ((q[2 * j + 1] & 0xF) << 4));
        }
    }
    return 0;
}

/* ------------------------------------------------------------------------- */
/* Scale layouts.                                                             */
/* ------------------------------------------------------------------------- */
/* Byte offset of scale (row r, scale column k) in the 128x4-atom swizzled
 * layout: 512-byte atoms of 128 rows x 4 scale columns, atoms ordered
 * row-block major with scale-column blocks fastest; inside an atom
 * offset = (r%32)*16 + ((r/32)%4)*4 + (k%4). */
int64_t oracle_swizzle_offset(int64_t r, int64_t k, int64_t kblocks)
{
    int64_t kpad4 = (kblocks + 3) / 4;
    int64_t atom = (r / 128) * kpad4 + (k / 4);
    return atom * 512 + (r % 32) * 16 + ((r / 32) % 4) * 4 + (k % 4);
}

int64_t oracle_swizzle_bytes(int64_t rows, int64_t kblocks)
{
    return ((rows + 127) / 128) * 128 * ((kblocks + 3) / 4) * 4;
}

int oracle_swizzle_scales(const uint8_t* sf_linear, int64_t rows, int64_t kblocks, uint8_t* out)
{
    memset(out, 0, (size_t)oracle_swizzle_bytes(rows, kblocks));
    for (int64_t r = 0; r < rows; r++)
        for (int64_t k = 0; k < kblocks; k++)
            out[oracle_swizzle_offset(r, k, kblocks)] = sf_linear[r * kblocks + k];
    return 0;
}

/* ------------------------------------------------------------------------- */
/* Dequantisation x_hat = fl32(fl32(q*v)*S) (Sec. 3.2 reconstruction).        */
/* layout 1 = linear scales, 2 = swizzled.  out_bf16 != 0 writes bf16 (RNE of */
/* the fp32 value) into out16, else fp32 into out32.                          */
/* ------------------------------------------------------------------------- */
static uint16_t f32_to_bf16_rne(float f)
{
    uint32_t u;
    memcpy(&u, &f, 4);
    if ((u & 0x7F800000u) == 0x7F800000u && (u & 0x007FFFFFu)) return (uint16_t)((u >> 16) | 0x40);
    uint32_t lsb = (u >> 16) & 1u;
    u += 0x7FFFu + lsb;
    return (uint16_t)(u >> 16);
}

int oracle_dequantize(const uint8_t* codes, const uint8_t* sf, int layout, float S,
                      int64_t rows, int64_t cols, int block, float* out32, uint16_t* out16)
{
    if (block <= 0 || cols % block != 0 || cols % 2 != 0) return -1;
    int64_t kb = cols / block;
#ifdef _OPENMP
#pragma omp parallel for schedule(static)
#endif
    for (int64_t r = 0; r < rows; r++) {
        for (int64_t j = 0; j < cols; j++) {
            int64_t k = j / block;
            int64_t so = (layout == 2) ? oracle_swizzle_offset(r, k, kb) : r * kb + k;
            int sc = sf[so];
            uint8_t byte = codes[r * (cols / 2) + j / 2];
            int qc = (j & 1) ? (byte >> 4) : (byte & 0xF);
            double q = oracle_e2m1_value(qc);
            double v = oracle_e4m3_value(sc);
            float qv = (float)(q * v);      /* exact */
            float xh = qv * S;              /* fl32(q*v*S) */
            if (out16) out16[r * cols + j] = f32_to_bf16_rne(xh);
            else out32[r * cols + j] = xh;
        }
    }
    return 0;
}

/* ------------------------------------------------------------------------- */
/* Appendix C: optimal real block scale.  L(s) = sum w_i (|y_i| - s*g_i(s))^2 */
/* with g_i(s) = RN_E2M1(|y_i|/s) (exact nearest).  Between consecutive       */
/* breakpoints |y_i|/mu_k (mu = midpoints of the E2M1 grid) every g_i is       */
/* constant and L is the quadratic A - 2Bs + Cs^2; each segment's minimum is  */
/* taken at B/C clamped to the segment.  Float64 throughout.                  */
/* ------------------------------------------------------------------------- */
static double exact_rn_mag(double t)
{
    /* nearest E2M1 magnitude, ties to even code, saturating */
    if (t >= 6.0) return 6.0;
    int best = 0;
    double bd = INFINITY;
    for (int k = 0; k < 8; k++) {
        double d = fabs(t - oracle_e2m1_value(k));
        if (d < bd || (d == bd && (k % 2) == 0)) { best = k; bd = d; }
    }
    return oracle_e2m1_value(best);
}

static int cmp_double(const void* a, const void* b)
{
    double x = *(const double*)a, y = *(const double*)b;
    return (x > y) - (x < y);
}

#include <stdlib.h>
int oracle_opt_scale(const float* y, const float* w, int n, double* s_opt, double* L_opt)
{
    static const double mid[7] = {0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0};
    double* bp = (double*)malloc(sizeof(double) * (size_t)(7 * n + 2));
    int nb = 0;
    double A = 0.0, amax = 0.0;
    for (int i = 0; i < n; i++) {
        double a = fabs((double)y[i]), wi = w ? (double)w[i] : 1.0;
        A += wi * a * a;
        if (a > amax) amax = a;
        if (a > 0)
            for (int k = 0; k < 7; k++) bp[nb++] = a / mid[k];
    }
    double bestL = A, bests = (amax > 0) ? amax / 0.25 * 2.0 : 1.0; /* all-zero reconstruction */
    if (amax > 0) {
        qsort(bp, (size_t)nb, sizeof(double), cmp_double);
        /* segments (0, bp0], (bp0, bp1], ..., (bp_last, inf) */
        double lo = 0.0;
        for (int j = 0; j <= nb; j++) {
            double hi = (j < nb) ? bp[j] : INFINITY;
            if (hi > lo) {
                double probe = (j < nb) ? (isfinite(hi) ? 0.5 * (lo + hi) : 2 * lo) : 2 * lo + 1.0;
                if (lo == 0.0 && j < nb) probe = 0.5 * hi;
                double B = 0.0, C = 0.0;
                for (int i = 0; i < n; i++) {
                    double a = fabs((double)y[i]), wi = w ? (double)w[i] : 1.0;
                    double g = exact_rn_mag(a / probe);
                    B += wi * a * g;
                    C += wi * g * g;
                }
                double s;
                if (C > 0) {
                    s = B / C;
                    if (s < lo) s = lo;
                    if (s > hi) s = hi;
                } else {
                    s = probe;
                }
                if (s > 0 && isfinite(s)) {
                    double L = 0.0;
                    for (int i = 0; i < n; i++) {
                        double a = fabs((double)y[i]), wi = w ? (double)w[i] : 1.0;
                        double e = a - s * exact_rn_mag(a / s);
                        L += wi * e * e;
                    }
                    if (L < bestL) { bestL = L; bests = s; }
                }
            }
            lo = hi;
        }
    }
    free(bp);
    *s_opt = bests;
    *L_opt = bestL;
    return 0;
}

/* Appendix C, FP8-quantised optimum: the better of floor_FP8(s*) and ceil_FP8(s*)
 * (s* in the S-normalised domain), scored with the same contract as the sweep. */
int oracle_fp8_opt_code(const float* y, const float* w, int n, double s_opt, int* code, double* L)
{
    int fl = 0, ce = 126;
    for (int c = 1; c <= 126; c++) if (oracle_e4m3_value(c) <= s_opt) fl = c;
    for (int c = 126; c >= 1; c--) if (oracle_e4m3_value(c) >= s_opt) ce = c;
    if (fl < 1) fl = 1;
    double Lf = block_loss(y, w, n, fl, NULL), Lc = block_loss(y, w, n, ce, NULL);
    if (Lc < Lf) { *code = ce; *L = Lc; } else { *code = fl; *L = Lf; }
    return 0;
}
