// nvfp4_global_scale_noalloc: the global-scale reduction for callers that
// cannot allocate device memory, so cannot hand nvfp4_global_scale the
// workspace it needs.  Its scratch (the per-CTA partial maxima and NaN/inf
// flags) lives in a file-scope static device array instead.
//
// Scratch: 16384 partial slots (128 KiB).  Each launch uses one slot per CTA
// and one CTA per 256 threads x 16 vectors of 16 bytes, so one call covers at
// most 2^29 bf16 or 2^28 fp32 elements; larger inputs are refused with
// NVFP4_ERR_RANGE before anything is launched.  Every slot a call reads is
// first written by that call, so nothing needs clearing between calls.
//
// Host code cannot use the array's name as a device address (it is a
// host-side stand-in), so the address is looked up once per device with
// cudaGetSymbolAddress, with that device current, the first time the entry
// point runs on it.
#include <cstdint>
#include <mutex>

#include <cuda_runtime.h>

#include "nvfp4_kernels.h"
#include "nvfp4ss.h"

namespace {

constexpr int kNoallocSlots = 16384;
constexpr int kVecsPerThread = 16;
constexpr int kThreads = 256;

struct NoallocScratch {
    float part_max[kNoallocSlots];
    int part_bad[kNoallocSlots];
};

// One copy on every GPU that loads the library, held until the process exits.
static __device__ __align__(256) NoallocScratch g_noalloc_scratch;

constexpr int kMaxDevices = 64;
std::mutex g_setup_mutex;
NoallocScratch* g_scratch_addr[kMaxDevices] = {nullptr};

// Device address of the scratch on the current device (looked up on first use).
cudaError_t scratch_for_current_device(NoallocScratch** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    if (!g_scratch_addr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) return e;
        g_scratch_addr[dev] = static_cast<NoallocScratch*>(p);
    }
    *out = g_scratch_addr[dev];
    return cudaSuccess;
}

bool is_aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

}  // namespace

extern "C" nvfp4_status nvfp4_global_scale_noalloc(const void* x, nvfp4_dtype dt, int64_t n, float fp8_div,
                                                   float* S_out, int* status_dev, void* stream) {
    if (dt != NVFP4_IN_BF16 && dt != NVFP4_IN_F32) return NVFP4_ERR_INVALID_ARG;
    if (n < 0 || !(fp8_div > 0.0f) || fp8_div > 1e30f) return NVFP4_ERR_INVALID_ARG;
    if (!S_out || (n > 0 && !x)) return NVFP4_ERR_INVALID_ARG;
    const int per = dt == NVFP4_IN_BF16 ? 8 : 4;
    const int64_t max_n = (int64_t)kNoallocSlots * kThreads * kVecsPerThread * per;
    if (n > max_n) return NVFP4_ERR_RANGE;
    if ((x && !is_aligned(x, 16)) || !is_aligned(S_out, 4) || (status_dev && !is_aligned(status_dev, 4)))
        return NVFP4_ERR_ALIGNMENT;
    NoallocScratch* scratch = nullptr;
    if (scratch_for_current_device(&scratch) != cudaSuccess) return NVFP4_ERR_CUDA;
    const int64_t nvec = n / per;
    const int64_t per_cta = (int64_t)kThreads * kVecsPerThread;
    int64_t grid = (nvec + per_cta - 1) / per_cta;
    if (grid < 1) grid = 1;
    cudaError_t e = nvfp4::launch_global_scale_parts(x, dt == NVFP4_IN_BF16 ? 0 : 1, n, fp8_div, S_out, status_dev,
                                                     scratch->part_max, scratch->part_bad, (int)grid,
                                                     static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? NVFP4_OK : NVFP4_ERR_CUDA;
}
