/*
 * nvfp4ss.h -- C ABI of libnvfp4ss.so: NVFP4 quantisation with ScaleSweep block
 * scales on NVIDIA GB300 (sm_103a).
 *
 * Method: "ScaleSweep: Accurate NVFP4 Post-Training Quantization of LLMs via
 * Block Scale Initialization".  A tensor x is represented as (q, s, S): FP4 E2M1
 * elements q, one FP8 E4M3 scale s per block of consecutive elements and one
 * FP32 global scale S, with x_hat_i = q_i * s_{i/block} * S (Sec. 3.2).
 *
 * Conventions shared by every entry point
 *   - Tensors are row-major [rows, cols]; blocks run along cols (the input
 *     channel of a [out, in] linear weight), so cols % block == 0.
 *   - All tensor pointers are device-accessible pointers (cudaMalloc, torch
 *     CUDA tensors, managed or registered host memory).  The caller allocates
 *     and owns every buffer; the library never allocates, frees or synchronises.
 *   - Every call is asynchronous on `stream` (a cudaStream_t; NULL = legacy
 *     default stream).  S is read from device memory by the kernels, so a
 *     per-call global scale needs no host round trip.
 *   - Argument, shape and alignment errors are detected on the host before any
 *     launch and returned as a status; nothing is launched then.  A failed
 *     launch returns NVFP4_ERR_CUDA.  Data errors (NaN/inf input) are reported
 *     through the device status word of nvfp4_global_scale.
 *   - Packed FP4 layout: codes[rows, cols/2] bytes, element 2j in the low
 *     nibble and element 2j+1 in the high nibble; a nibble is sign (bit 3) and
 *     the 3-bit E2M1 magnitude code (0, 0.5, 1, 1.5, 2, 3, 4, 6).
 *   - Scale layouts: linear sf[rows, cols/block] E4M3 codes; swizzled (block 16
 *     only) is the 128x4-atom layout read by tcgen05 block-scaled MMA:
 *     ceil(rows/128)*128 x ceil(cols/64)*4 bytes, atom (row/128, col4/4) at
 *     ((row/128)*ceil(kb/4) + k/4)*512, inside it (row%32)*16 + ((row/32)%4)*4 + k%4;
 *     padding bytes are written as 0.
 *
 * Arithmetic contract (where the paper fixes no arithmetic; decisions in fp32):
 *   E = fl(1/S), y = fl(x*E); m = max|y| per block; s_base = fl(m/6);
 *   I0 = code of floor_E4M3(s_base); candidate c: t = fl(y*fl(1/v_c)),
 *   q = RNE_E2M1(t) saturating at 6; loss L_c = sum w (y - q v_c)^2;
 *   argmin over the window with exact ties going to the lowest code.
 *   Zero rule: a block with m == 0, a block whose m (NaN counted) is NaN,
 *   infinite or at least 2^48, and every block when S is not a positive finite
 *   float with finite 1/S, gets scale code 0 and nibbles carrying only the sign
 *   of y, for every method.  With S from nvfp4_global_scale a finite input gives
 *   m <= 6*fp8_div, so only NaN/inf inputs (or a caller's S more than 2^36 below
 *   amax/(6 D)) reach the 2^48 bound; below it every fp32 loss the kernels
 *   accumulate stays finite for WMSE weights that are finite, >= 0 and <= 2^24.
 */
#ifndef NVFP4SS_H
#define NVFP4SS_H

#include <limits.h>
#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    NVFP4_OK = 0,
    NVFP4_ERR_INVALID_ARG = 1,   /* null/overlapping pointer, bad enum, bad shape or window */
    NVFP4_ERR_UNSUPPORTED = 2,   /* block not in {16,32,64}; swizzled scales with block != 16 */
    NVFP4_ERR_ALIGNMENT = 3,     /* a pointer misses its required alignment */
    NVFP4_ERR_RANGE = 4,         /* a size overflows int64 or the device limits */
    NVFP4_ERR_CUDA = 5           /* a CUDA runtime call or launch failed */
} nvfp4_status;

typedef enum { NVFP4_IN_BF16 = 0, NVFP4_IN_F32 = 1 } nvfp4_dtype;
typedef enum { NVFP4_OBJ_MSE = 0, NVFP4_OBJ_WMSE = 1 } nvfp4_objective;
typedef enum { NVFP4_SF_LINEAR = 1, NVFP4_SF_SWIZZLED = 2 } nvfp4_sf_layout;

/* Pass as win_lo and win_hi to use the paper's window (Sec. 4.2.2). */
#define NVFP4_WINDOW_DEFAULT INT_MIN
/* Pass as win_lo and win_hi for the paper's window tightened per block without
 * changing the result (the exact-window refinement of Sec. 4.2.2): the upper end
 * drops every code c >= 16 with 3.5 v_c > max|y| (Lemma 4.1: such an s never
 * beats s/2, which is code c - 8 and stays in the window; 3.5 v_c is exact in
 * fp32; below code 16 half a scale need not be a code), and for MSE with block
 * 16 the lower end is the
 * per-mantissa bound of Table 2 (I0 - 2, or I0 - 3 for mantissas 000 and 111;
 * applied for I0 in 16..120, where the ceiling stays normal and Lemma 4.3's
 * 11/7 s <= 448 holds).  A warp runs as many candidates as its widest block. */
#define NVFP4_WINDOW_TIGHT (INT_MIN + 1)

/* Human-readable name of a status code (static storage). */
const char* nvfp4_status_string(nvfp4_status st);

/*
 * Bytes of device workspace nvfp4_global_scale needs for n elements.
 */
size_t nvfp4_global_scale_workspace(int64_t n);

/*
 * Global scale S = fl32(amax / fl32(6*fp8_div)), amax = max_i |x_i| (Sec. 3.2
 * with fp8_div = 448, AbsMax; Sec. 4.2.1 with fp8_div = 256, ScaleSweep).
 *   x          [n] elements of type dt, 16-byte aligned.
 *   S_out      device float written with S.
 *   status_dev optional device int; bit 0 is OR-ed in if x holds NaN or inf
 *              (NaNs are ignored by the max, an inf makes S = inf).
 *   workspace  device scratch of nvfp4_global_scale_workspace(n) bytes,
 *              16-byte aligned; its contents need no initialisation.
 * n == 0 writes S = 0.  Two kernel launches on `stream`, the second a
 * programmatic dependent launch of the first (scheduled while the first drains,
 * ordered after its writes); both can be captured in a CUDA graph.
 */
nvfp4_status nvfp4_global_scale(const void* x, nvfp4_dtype dt, int64_t n, float fp8_div, float* S_out,
                                int* status_dev, void* workspace, size_t ws_bytes, void* stream);

/*
 * nvfp4_global_scale without a workspace argument; the paper has no
 * counterpart (it is a packaging variant of the reduction above).
 * For callers that cannot call cudaMalloc: code that runs under a device-memory
 * plan fixed at start-up (e.g. a serving engine that reserves all GPU memory
 * up front and forbids allocation on the request path) or a host embedding
 * this library without an allocator of its own, and so cannot provide the
 * workspace nvfp4_global_scale needs.  The scratch is a 128 KiB static device
 * array that every GPU which loads the library holds until the process exits;
 * no allocation or free is made by any call.
 *   Same S, status word and alignment rules as nvfp4_global_scale.
 *   n may be at most 2^29 bf16 or 2^28 fp32 elements; a larger n returns
 *   NVFP4_ERR_RANGE and launches nothing.
 *   The first call on each device looks up the scratch's device address
 *   (cudaGetSymbolAddress) once, with that device current; make that first call
 *   before any stream capture.
 *   All calls share the one scratch array: calls whose kernels may overlap on
 *   the GPU (e.g. on unordered streams) race and must be ordered by the caller.
 */
nvfp4_status nvfp4_global_scale_noalloc(const void* x, nvfp4_dtype dt, int64_t n, float fp8_div, float* S_out,
                                        int* status_dev, void* stream);

/*
 * ScaleSweep quantisation (Sec. 4.2.2): per block, sweep the E4M3 scale codes
 * in [I0 + win_lo, I0 + win_hi] (clamped to 1..126), score each with the MSE
 * (Sec. 4.1, Eq. for L^MSE) or WMSE (Sec. 4.1, diagonal-Gram importance)
 * objective, keep the argmin (exact ties -> lowest code) and emit its codes.
 *   x             [rows, cols] of type dt, 16-byte aligned.
 *   block         16, 32 or 64 elements per scale.
 *   S             device float (global scale, e.g. from nvfp4_global_scale).
 *   obj, w        NVFP4_OBJ_WMSE reads per-element weights w[row*w_row_stride + col]
 *                 (float, >= 0, 16-byte aligned; w_row_stride = 0 broadcasts one
 *                 [cols] vector, e.g. per-input-channel importance ||X[:,i]||^2);
 *                 w is ignored for MSE and may be NULL.
 *   win_lo/hi     bit-pattern offsets, -126 <= win_lo <= win_hi <= 126, or both
 *                 NVFP4_WINDOW_DEFAULT: [-3, 7] for MSE with block 16 (Lemma 4.3),
 *                 [-8, 7] otherwise (WMSE: empirical s_base/2; blocks of 32/64:
 *                 the paper gives no window).  (-126, 126) is the exhaustive sweep.
 *                 Both NVFP4_WINDOW_TIGHT: the default window tightened per block.
 *   codes         [rows, cols/2] packed nibbles, 8-byte aligned.
 *   sf_linear     optional [rows, cols/block] scale codes.
 *   sf_swizzled   optional 128x4-atom scale layout (block 16 only).
 *                 At least one of sf_linear / sf_swizzled must be given.
 *   block_loss    optional [rows*cols/block] float: the chosen candidate's loss in
 *                 the S-normalised domain (multiply by S^2 for the x domain).
 * Outputs must not overlap x, w or each other.
 */
nvfp4_status scalesweep_quantize(const void* x, nvfp4_dtype dt, int64_t rows, int64_t cols, int block,
                                 const float* S, nvfp4_objective obj, const float* w, int64_t w_row_stride,
                                 int win_lo, int win_hi, uint8_t* codes, uint8_t* sf_linear,
                                 uint8_t* sf_swizzled, float* block_loss, void* stream);

/*
 * Bytes of device workspace the *_quantize_dynamic entry points need.
 */
size_t nvfp4_dynamic_workspace(void);

/*
 * ScaleSweep quantisation with a per-call (dynamic) global scale computed in
 * the same launch: S = fl32(amax / fl32(6*fp8_div)) (Sec. 4.2.1) over the whole
 * tensor, then the sweep of scalesweep_quantize with that S.  This fuses the
 * reduction into the sweep for dynamic activation quantisation (the paper's
 * kernels leave fusion as future work, Sec. 5.2).  One cooperative launch (all
 * CTAs resident) with a grid barrier in between, preceded by a 4-byte
 * cudaMemsetAsync of the barrier counter in the workspace.
 *   S_out       device float written with S (also returned implicitly by the codes).
 *   status_dev  optional device int: bit 0 OR-ed in for NaN/inf input, bit 1 if the
 *               grid barrier timed out (about a second; the outputs are then not
 *               written -- a resident grid makes this unreachable in practice).
 *   workspace   nvfp4_dynamic_workspace() bytes, 16-byte aligned, no initialisation.
 * Other arguments as scalesweep_quantize.  rows*cols == 0 launches nothing.
 * Concurrent calls must use distinct workspaces.
 */
nvfp4_status scalesweep_quantize_dynamic(const void* x, nvfp4_dtype dt, int64_t rows, int64_t cols, int block,
                                         float fp8_div, nvfp4_objective obj, const float* w, int64_t w_row_stride,
                                         int win_lo, int win_hi, float* S_out, int* status_dev, void* workspace,
                                         size_t ws_bytes, uint8_t* codes, uint8_t* sf_linear, uint8_t* sf_swizzled,
                                         float* block_loss, void* stream);

/*
 * One tensor of a grouped call (scalesweep_quantize_group).  Fields as the
 * arguments of scalesweep_quantize with block = 16:
 *   x             [rows, cols] of the call's dtype, 16-byte aligned, cols % 16 == 0.
 *   w             WMSE importance (w[row*w_row_stride + col], 16-byte aligned;
 *                 w_row_stride 0 broadcasts one [cols] vector); NULL for MSE.
 *   codes         [rows, cols/2], 8-byte aligned.
 *   sf_linear     optional [rows, cols/16]; sf_swizzled optional 128x4-atom
 *                 layout; at least one of the two.
 */
typedef struct {
    const void* x;
    int64_t rows, cols;
    const float* w;
    int64_t w_row_stride;
    uint8_t* codes;
    uint8_t* sf_linear;
    uint8_t* sf_swizzled;
} nvfp4_group_tensor;

#define NVFP4_GROUP_MAX 16

/*
 * Bytes of device workspace scalesweep_quantize_group needs.
 */
size_t scalesweep_quantize_group_workspace(void);

/*
 * ScaleSweep quantisation of `count` tensors (1..NVFP4_GROUP_MAX, e.g. all
 * linear weights of one transformer layer) in one call: for every tensor the
 * result of scalesweep_quantize with the same block and the default window
 * ([-3, 7] MSE with block 16, [-8, 7] otherwise, Sec. 4.2.2), bit for bit.  The
 * segments of all tensors are walked by one grid (with static scales, one
 * launch), so the call has a single launch tail instead of one per tensor.
 *   tensors     host array of `count` descriptors, read during the call only.
 *   dt, obj     input type and objective, shared by all tensors.
 *   block       16, 32 or 64, shared by all tensors (every cols % block == 0);
 *               sf_swizzled only with block 16.
 *   fp8_div     0: static global scales, S[i] is read for tensor i.
 *               > 0: per-call (dynamic) global scales, S[i] = fl32(amax_i /
 *               fl32(6*fp8_div)) over tensor i (Sec. 4.2.1) is computed on the
 *               device during the call and written, by the schedule
 *               NVFP4_GROUP_SCHEDULE_AUTO picks (see
 *               scalesweep_quantize_group_scheduled); either is preceded by a
 *               cudaMemsetAsync of the workspace counters.
 *   S           device float[count].
 *   status_dev  optional device int: bit 0 OR-ed in for NaN/inf input (dynamic
 *               only), bit 1 if the two-phase schedule's grid barrier timed out
 *               (about a second; no outputs are written then -- a resident grid
 *               makes this unreachable in practice).
 *   workspace   scalesweep_quantize_group_workspace() bytes, 16-byte aligned, no
 *               initialisation (dynamic only; may be NULL for static scales).
 * Outputs must not overlap any input, S, status_dev, the workspace or each
 * other.  Concurrent calls must use distinct workspaces.
 */
nvfp4_status scalesweep_quantize_group(const nvfp4_group_tensor* tensors, int count, nvfp4_dtype dt, int block,
                                       nvfp4_objective obj, float fp8_div, float* S, int* status_dev,
                                       void* workspace, size_t ws_bytes, void* stream);

/*
 * How a grouped call with dynamic global scales (fp8_div > 0) orders the
 * reduction of every tensor's amax and the sweep.  Results are identical, bit
 * for bit, under every schedule; only the launches and their overlap differ.
 *   NVFP4_GROUP_SCHEDULE_AUTO       pipelined for a ScaleSweep over at least
 *                                   two tensors and 2^25 elements, else two-phase.
 *   NVFP4_GROUP_SCHEDULE_TWO_PHASE  one cooperative launch: every warp reduces
 *                                   its share of every tensor, a grid barrier
 *                                   (bounded, status bit 1), then the sweep.
 *   NVFP4_GROUP_SCHEDULE_PIPELINED  four launches, the last three programmatic
 *                                   dependent launches: the largest tensor's
 *                                   reduction, its sweep, the other tensors'
 *                                   reduction running beside that sweep on the
 *                                   registers it leaves free, then one grouped
 *                                   sweep of the other tensors.  The HBM-bound
 *                                   reductions hide behind the FP32-bound sweep,
 *                                   except the first.  No device wait is involved.
 *                                   With one tensor, or for AbsMax, two-phase.
 */
typedef enum {
    NVFP4_GROUP_SCHEDULE_AUTO = 0,
    NVFP4_GROUP_SCHEDULE_TWO_PHASE = 1,
    NVFP4_GROUP_SCHEDULE_PIPELINED = 2
} nvfp4_group_schedule;

/*
 * scalesweep_quantize_group with an explicit schedule for dynamic global
 * scales (ignored when fp8_div == 0).  Arguments, outputs and errors as
 * scalesweep_quantize_group; an unknown schedule is NVFP4_ERR_INVALID_ARG.
 */
nvfp4_status scalesweep_quantize_group_scheduled(const nvfp4_group_tensor* tensors, int count, nvfp4_dtype dt,
                                                 int block, nvfp4_objective obj, float fp8_div, float* S,
                                                 int* status_dev, void* workspace, size_t ws_bytes,
                                                 nvfp4_group_schedule schedule, void* stream);

/*
 * AbsMax quantisation (Sec. 3.2, as absmax_quantize) of `count` tensors in one
 * launch, with static or in-launch global scales exactly as
 * scalesweep_quantize_group (same descriptors, arguments, workspace and
 * status word; the descriptors' w and w_row_stride are not read).  The
 * baseline the grouped sweep's overhead is measured against, launch shape for
 * launch shape.
 */
nvfp4_status absmax_quantize_group(const nvfp4_group_tensor* tensors, int count, nvfp4_dtype dt, int block,
                                   float fp8_div, float* S, int* status_dev, void* workspace, size_t ws_bytes,
                                   void* stream);

/*
 * Self-test of the bounded device waits (failure detection; the paper has no
 * counterpart).  Runs scalesweep_quantize_dynamic (which = 0: bf16 x, block
 * 16, MSE, default window) or scalesweep_quantize_group with a dynamic scale
 * (which = 1: x as its one tensor, MSE) with the wait's arrival target raised
 * past what the launch can reach, so every device wait gives up after its
 * limit (about a second): bit 1 is OR-ed into *status_dev (required here), the
 * waiting warps return without writing codes or scales, and the CUDA context
 * stays usable.  Arguments and buffers as in those calls; workspace of
 * max(nvfp4_dynamic_workspace(), scalesweep_quantize_group_workspace()) bytes.
 */
nvfp4_status nvfp4_selftest_wait_timeout(int which, const void* x, int64_t rows, int64_t cols, float* S,
                                         int* status_dev, void* workspace, size_t ws_bytes, uint8_t* codes,
                                         uint8_t* sf_linear, void* stream);

/*
 * AbsMax quantisation with the global scale computed in the same launch, as
 * scalesweep_quantize_dynamic (baseline for the fused dynamic path).
 */
nvfp4_status absmax_quantize_dynamic(const void* x, nvfp4_dtype dt, int64_t rows, int64_t cols, int block,
                                     float fp8_div, float* S_out, int* status_dev, void* workspace, size_t ws_bytes,
                                     uint8_t* codes, uint8_t* sf_linear, uint8_t* sf_swizzled, float* block_loss,
                                     void* stream);

/*
 * AbsMax quantisation (Sec. 3.2): s = max(1, RN_E4M3(s_base)) as a code (a block
 * whose RN scale would be 0 gets the smallest positive scale), q = RNE_E2M1.
 * Arguments as scalesweep_quantize; block_loss is the MSE loss of the chosen
 * scale.  This is the baseline the overhead of the sweep is measured against.
 */
nvfp4_status absmax_quantize(const void* x, nvfp4_dtype dt, int64_t rows, int64_t cols, int block,
                             const float* S, uint8_t* codes, uint8_t* sf_linear, uint8_t* sf_swizzled,
                             float* block_loss, void* stream);

/*
 * 4/6 quantisation (Sec. 2, FP4 quantization): besides the AbsMax scale c6, try
 * c4 = max(1, RN_E4M3(fl(m/4))) (block max mapped to 4) and keep c4 only if its
 * loss under `obj` is strictly lower.  Arguments as scalesweep_quantize.
 */
nvfp4_status four_over_six_quantize(const void* x, nvfp4_dtype dt, int64_t rows, int64_t cols, int block,
                                    const float* S, nvfp4_objective obj, const float* w, int64_t w_row_stride,
                                    uint8_t* codes, uint8_t* sf_linear, uint8_t* sf_swizzled,
                                    float* block_loss, void* stream);

/*
 * Optimal real-valued block scale (Appendix C) and the FP8-quantised optimal
 * scale (Appendix C, second paragraph), per block, in the S-normalised domain
 * (y = fl(x * fl(1/S))): s_opt minimises sum w_i (y_i - s RN_E2M1(y_i/s))^2
 * over real s > 0 by enumerating the quadratic segments between the
 * breakpoints |y_i| / mu (mu the E2M1 midpoints); loss_opt is that minimum
 * (fp32).  fp8_code (optional) is the better of floor_E4M3(s_opt) and
 * ceil_E4M3(s_opt) under the sweep's arithmetic contract (ties to the floor),
 * loss_fp8 (optional, needs fp8_code) its loss.  An analysis entry point: it
 * measures the gap of any FP8 scale choice to the best FP32 scale.
 *   x, S, obj, w, w_row_stride as scalesweep_quantize (4-byte alignment);
 *   s_opt, loss_opt, loss_fp8: [rows*cols/block] float; fp8_code [rows*cols/block].
 */
nvfp4_status nvfp4_optimal_scale(const void* x, nvfp4_dtype dt, int64_t rows, int64_t cols, int block,
                                 const float* S, nvfp4_objective obj, const float* w, int64_t w_row_stride,
                                 float* s_opt, float* loss_opt, uint8_t* fp8_code, float* loss_fp8, void* stream);

/*
 * Dequantisation x_hat = fl32(fl32(q * s) * S) (Sec. 3.2 reconstruction; the
 * simulated quantisation of Sec. 5.1), written as fp32 or as the RNE bf16 of
 * that fp32 value.
 *   codes  [rows, cols/2] packed nibbles (8-byte aligned); sf in `layout`
 *   (NVFP4_SF_SWIZZLED requires block 16); out [rows, cols] of out_dt,
 *   16-byte aligned.
 */
nvfp4_status nvfp4_dequantize(const uint8_t* codes, const uint8_t* sf, nvfp4_sf_layout layout, const float* S,
                              int64_t rows, int64_t cols, int block, void* out, nvfp4_dtype out_dt,
                              void* stream);

/*
 * LDLQ / GPTQ with ScaleSweep block scales (Appendix A.2, "GPTQ" paragraph):
 * GPTQ's error-feedback pass in QuIP's LDLQ form, damping damp * mean(diag H)
 * (the paper uses damp = 0.01), and static reordering -- the block scales are
 * fixed beforehand (e.g. by scalesweep_quantize with WMSE weights diag(H)) and
 * the input channels are processed in descending order of diag(H).
 *
 * nvfp4_ldlq_prepare factors the Hessian once per weight matrix:
 *   H       [n, n] float, the input Gram matrix X^T X (any positive scaling),
 *           symmetric; every entry H[perm[i], perm[j]] is read.  4-byte aligned.
 *   perm    [n] int32 out: perm[k] = original column processed k-th (diagonal
 *           descending, ties by ascending index, NaN last).
 *   U       [n, n] float out (4-byte aligned, must not overlap H): the strictly
 *           upper factor of H_pi + lambda I = (U + I) diag(D) (U + I)^T in
 *           processing order (zeros on and below the diagonal).  Also used as
 *           the factorization's scratch.
 *   D       [n] float out.
 *   status_dev  optional int on the device: |= 4 if the damped Hessian is not
 *           positive definite or has a non-finite diagonal (a failing pivot is
 *           replaced by 1 so the outputs stay finite, but they are not a
 *           factorization then).
 *           |= 16 if a tensor-core update's bounded wait ran out (about a
 *           second; that update is then not applied).
 *   workspace   device bytes, at least nvfp4_ldlq_prepare_workspace(n).
 * Cost: n^3/3 fp32 multiply-adds (blocked Cholesky, 64-wide panels).  The
 * trailing updates run on the tensor cores as three TF32 products per term
 * (products to ~2^-21 relative, accumulated in fp32) when n % 4 == 0 and H,
 * U are 16-byte aligned, else on the FP32 pipe.
 * The factorization's critical chain runs on a high-priority stream the library
 * creates on the first call on a device and keeps (with four events) for the
 * process; it is forked from and joined back into `stream`, so the call stays
 * ordered on `stream` and can be captured in a CUDA graph -- make the first
 * call on each device outside a capture.  Concurrent calls on one device are
 * serialised while they enqueue.
 */
size_t nvfp4_ldlq_prepare_workspace(int64_t n);
nvfp4_status nvfp4_ldlq_prepare(const float* H, int64_t n, float damp, int32_t* perm, float* U, float* D,
                                int* status_dev, void* workspace, size_t ws_bytes, void* stream);

/*
 * ldlq_quantize: W [rows, cols] (bf16 or f32, original column order) to packed
 * NVFP4 codes [rows, cols/2] (original order) with the fixed scales sf_linear
 * [rows, cols/block] (E4M3 codes, linear layout) and global scale S (device).
 * Column k of the processing order gets T_k = W_k + sum_{i<k} (W_i - What_i)
 * U_ik, What_k = Q(T_k), with Q the sweep's fp32 rounding at the fixed scale:
 * y = fl(T*E), q = RNE_E2M1(fl(y*fl(1/v))), What = fl(fl(q*v)*S); a zero scale
 * code or an unusable S quantizes to signed zeros, an exactly zero y to +0.
 *   The error-feedback updates run on the tensor cores (three TF32 products
 *   per term, as in nvfp4_ldlq_prepare; status bit 16 as there) when rows and
 *   cols are multiples of 4 and the buffers 16-byte aligned, else on the FP32
 *   pipe.
 *   perm, U from nvfp4_ldlq_prepare (cols = n); status_dev optional: |= 8 if
 *   perm holds an index outside [0, cols) (the entry is then read as 0).
 *   workspace   device bytes, at least nvfp4_ldlq_workspace(rows, cols):
 *           rows*cols*10 + rows*2048 + cols*4 plus alignment.
 * Cost: rows*cols^2/2 fp32 multiply-adds; rows are independent.  The column
 * walk uses the high-priority stream described under nvfp4_ldlq_prepare (same
 * first-call and concurrency rules).
 */
size_t nvfp4_ldlq_workspace(int64_t rows, int64_t cols);
nvfp4_status ldlq_quantize(const void* W, nvfp4_dtype dt, int64_t rows, int64_t cols, int block, const float* S,
                           const uint8_t* sf_linear, const int32_t* perm, const float* U, uint8_t* codes,
                           int* status_dev, void* workspace, size_t ws_bytes, void* stream);

/*
 * Row partition of one [rows, cols] tensor over `world` shards (ranks, GPUs)
 * for the multi-GPU path: given S every block is independent (Sec. 4.2.1), so
 * shard `rank` quantises rows [row_begin, row_end) alone, with the global
 * scale S = fl32(max_k amax_k / fl32(6 D)) taken as the maximum of the shards'
 * own nvfp4_global_scale results (one max-allreduce of a float: fl32(a/c) is
 * monotone in a, so the maximum of the shards' S is the whole tensor's S, bit
 * for bit; OR-reduce the status words too).  Shard boundaries fall on
 * multiples of 128 rows, so no 128x4 swizzled-scale atom straddles two shards
 * and each shard's outputs are contiguous byte ranges of the whole tensor's:
 * calling scalesweep_quantize (or any quantisation call) on the shard's rows
 * with these offsets added to the whole tensor's output pointers writes
 * exactly the bytes the single call would.  Row blocks of 128 are split as
 * evenly as possible; a shard may be empty (row_begin == row_end) when world
 * exceeds the row blocks.  Host-only: no CUDA call, no device access.
 *   block        16, 32 or 64; the swizzled offsets are -1 unless block == 16.
 *   out          receives the shard's rows and offsets (elements for x, bytes
 *                for the outputs).
 * Returns NVFP4_ERR_INVALID_ARG for a null `out`, world < 1 or rank outside
 * [0, world), and the shape errors of scalesweep_quantize.  The paper has no
 * counterpart: it states the independence the partition relies on.
 */
typedef struct {
    int64_t row_begin, row_end;     /* the shard's rows */
    int64_t x_offset;               /* elements: row_begin * cols */
    int64_t codes_offset;           /* bytes: row_begin * cols / 2 */
    int64_t sf_linear_offset;       /* bytes: row_begin * cols / block */
    int64_t sf_swizzled_offset;     /* bytes: (row_begin / 128) * ceil(cols/64) * 512, or -1 */
    int64_t sf_swizzled_bytes;      /* the shard's swizzled extent, or -1 */
} nvfp4_row_shard;

nvfp4_status nvfp4_row_shard_layout(int64_t rows, int64_t cols, int block, int world, int rank,
                                    nvfp4_row_shard* out);

#ifdef __cplusplus
}
#endif

#endif /* NVFP4SS_H */
