// Internal interface of the LDLQ (GPTQ) kernels in ldlq.cu, used by the C-ABI
// host layer (api.cu).  Not part of the public ABI.
#pragma once
#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

namespace nvfp4 {

// LDLQ (GPTQ) with fixed block scales, static reordering (ldlq.cu).
constexpr int kLdlqPanel = 256;       // columns per trailing update of the error feedback
struct LdlqParams {
    const void* W;            // [rows, n] bf16 or f32, original column order
    int64_t rows, n;
    const int32_t* perm;      // [n] processing order
    const float* U;           // [n, n] strictly upper, processing order
    const uint8_t* sf;        // [rows, kb] fixed E4M3 codes
    int64_t kb;
    int block;
    const float* S;
    int* status;
    float* T;                 // workspace: targets [rows, n], processing order
    float* Wp;                // workspace: W in processing order, f32
    uint8_t* qb;              // workspace: nibbles [rows, n], processing order
    uint8_t* sfp;             // workspace: each element's scale code, processing order
};
size_t ldlq_prepare_workspace(int64_t n);
cudaError_t launch_ldlq_prepare(const float* H, int64_t n, float damp, int32_t* perm, float* U, float* D,
                                int* status, void* ws, int sms, cudaStream_t s);
size_t ldlq_quantize_workspace(int64_t rows, int64_t n);
cudaError_t launch_ldlq_quantize(LdlqParams p, int dtype, uint8_t* codes, void* ws, int sms, cudaStream_t s);

}  // namespace nvfp4
