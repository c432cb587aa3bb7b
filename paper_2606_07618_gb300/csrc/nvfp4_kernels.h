// Internal interface between the C-ABI host layer (api.cu) and the kernel
// translation units.  Not part of the public ABI.
#pragma once
#include <cstdint>
#include <cuda_runtime.h>

namespace nvfp4 {

struct FastDiv {            // n / d = (t + ((n - t) >> s1)) >> s2, t = umulhi(n, mul)
    uint32_t mul, s1, s2;
};
FastDiv make_fast_div(uint32_t d);

struct QuantParams {
    const void* x;
    const float* S;
    const float* w;
    int64_t w_row_stride;
    int64_t rows, cols, kb, kpad4;
    int64_t nseg;            // rows * cols / 16
    int narrow;              // rows * kb < 2^32
    int need_rowcol;         // swizzled scales or weights need (row, block column)
    FastDiv kb_div;          // divides a 32-bit block index by kb
    int win_lo, win_hi;
    int tight;               // per-block window: bit 0 Lemma 4.1 upper cut, bit 1 Table 2 lower (MSE, block 16)
    uint8_t* codes;
    uint8_t* sf_linear;
    uint8_t* sf_swizzled;
    float* block_loss;
    // dynamic (per-call) global scale, computed inside the sweep launch
    float fp8_div;
    float* S_out;
    int* status_dev;
    float* part_max;
    int* part_bad;
    unsigned* barrier;
    unsigned wait_extra;     // added to the barrier's arrival target; 0 except in the wait self-test
};

// dtype 0 bf16 / 1 f32; method 0 ScaleSweep / 1 AbsMax / 2 four-over-six;
// obj 0 MSE / 1 WMSE; block 16/32/64; sms = multiprocessor count.
cudaError_t launch_quantize(const QuantParams& p, int dtype, int method, int obj, int block, int sms,
                            cudaStream_t s);
// Same with the global scale computed in the launch (method 0 or 1; p.S unused,
// p.S_out/part_max/part_bad/barrier in the caller's workspace).
cudaError_t launch_quantize_dynamic(const QuantParams& p, int dtype, int method, int obj, int block, int sms,
                                    cudaStream_t s);
// Zero the pads of a swizzled scale buffer when rows % 128 or kb % 4 != 0.
cudaError_t launch_swizzle_pad(const QuantParams& p, int sms, cudaStream_t s);
// Fill the derived fields of p (window mode, row/column need, fast divider).
void prepare_quant_params(QuantParams& p, int method, int obj, int block, bool* fix);

// Global-scale reduction: partial maxima into ws, then S and the status word.
cudaError_t launch_global_scale(const void* x, int dtype, int64_t n, float fp8_div, float* S_out,
                                int* status_dev, void* ws, int sms, cudaStream_t s);
constexpr int kAmaxParts = 1024;   // partial slots in the workspace
// Dynamic-scale workspace: partial maxima, partial flags, barrier counter.
constexpr size_t kDynWorkspace = (size_t)kAmaxParts * 8 + 256;

// Same two kernels with caller-chosen partial slots and grid (grid <= slots).
cudaError_t launch_global_scale_parts(const void* x, int dtype, int64_t n, float fp8_div, float* S_out,
                                      int* status_dev, float* part_max, int* part_bad, int grid, cudaStream_t s);

struct OptParams {
    const void* x;
    const float* S;
    const float* w;
    int64_t w_row_stride;
    int64_t rows, cols, kb, nblocks;
    float* s_opt;
    float* loss_opt;
    uint8_t* fp8_code;
    float* loss_fp8;
};
cudaError_t launch_optimal_scale(const OptParams& p, int dtype, int obj, int block, int sms, cudaStream_t s);

struct DequantParams {
    const uint8_t* codes;
    const uint8_t* sf;
    const float* S;
    int64_t rows, cols, kb, kpad4, nseg;
    int narrow;
    int swizzled;
    int block;
    void* out;
};
cudaError_t launch_dequantize(const DequantParams& p, int out_dtype, int sms, cudaStream_t s);

}  // namespace nvfp4
