// Internal interface of the grouped ScaleSweep launch (quantize_group.cu):
// one launch quantises a list of tensors, e.g. every linear weight of a
// transformer layer, optionally computing each tensor's global scale inside
// the same launch.  Not part of the public ABI.
#pragma once
#include <cstdint>
#include <cuda_runtime.h>

#include "nvfp4_kernels.h"

namespace nvfp4 {

constexpr int kGroupMax = 16;

struct GroupTensor {
    const void* x;
    const float* w;            // WMSE importance (nullptr for MSE)
    int64_t w_row_stride;
    uint8_t* codes;
    uint8_t* sf_linear;
    uint8_t* sf_swizzled;
    int64_t kb, kpad4;
    int64_t nseg;              // 16-element segments
    int64_t seg_begin;         // first index in the concatenated segment space (multiple of 32)
    int64_t nvec;              // 16-byte input vectors (global-scale reduction)
    FastDiv kb_div;
    int narrow;
    int s_index;               // slot of this tensor's global scale in GroupParams::S
};

struct GroupParams {
    GroupTensor t[kGroupMax];  // in processing order
    int count;
    int dyn;                   // 1: S computed in the launch, 0: S read
    int pipelined;             // dyn only: 1 pipelined schedule, 0 two-phase cooperative launch
    int64_t total_seg;         // end of the concatenated segment space
    float fp8_div;
    float* S;                  // [count] by s_index
    int* status_dev;
    unsigned* amax_bits;       // [count] workspace, zeroed before the launch
    unsigned* arrived;         // [count] workspace, zeroed before the launch
    unsigned wait_extra;       // added to the arrival target; 0 except in the wait self-test
};

constexpr size_t kGroupWorkspace = 256;   // amax_bits + arrived for kGroupMax tensors

// Groups of at least this many elements (and two tensors) take the pipelined
// schedule when the caller leaves the choice to the library.
constexpr int64_t kPipelineMinElements = int64_t(1) << 25;

// Segments a CTA sweeps per iteration; each tensor's segment range in the
// concatenated index space is padded to a multiple of it, so a CTA never
// straddles two tensors.
constexpr int kGroupCtaSegments = 256;

// dtype 0 bf16 / 1 f32; method 0 ScaleSweep / 1 AbsMax; obj 0 MSE / 1 WMSE
// (ScaleSweep only); block 16/32/64.  Zeroes the workspace counters (dyn),
// launches the grouped kernel (cooperative when dyn; with p.pipelined, a
// ScaleSweep and at least two tensors, the four launches of the pipelined
// schedule instead) and the swizzle pad kernels for shapes that need them.
cudaError_t launch_quantize_group(const GroupParams& p, const int64_t* rows, int dtype, int method, int obj,
                                  int block, int sms, cudaStream_t s);

}  // namespace nvfp4
