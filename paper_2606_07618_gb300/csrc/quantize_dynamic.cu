// Sweep launches that compute the per-call global scale themselves (one
// cooperative launch instead of amax reduction + final + sweep): the fused
// dynamic-activation path.  The grid barrier counter lives in the caller's
// workspace and is zeroed with an asynchronous memset right before the launch.
#include "quantize_kernel.cuh"

namespace nvfp4 {

template <int DT, int METHOD, int OBJ, int BLOCK, int FIX>
static cudaError_t launch_dyn(const QuantParams& p_in, int sms, cudaStream_t s) {
    static std::atomic<int> occ_cache[kOccDevices];
    const int occ = occupancy_per_sm(occ_cache, quantize_kernel<DT, METHOD, OBJ, BLOCK, FIX, 1>, 256);
    QuantParams p = p_in;
    int64_t grid = (p.nseg + 255) / 256;
    if (grid > (int64_t)sms * occ) grid = (int64_t)sms * occ;   // every CTA resident: the barrier can complete
    if (grid > kAmaxParts) grid = kAmaxParts;
    if (grid < 1) grid = 1;
    cudaError_t e = cudaMemsetAsync(p.barrier, 0, sizeof(unsigned), s);
    if (e != cudaSuccess) return e;
    void* args[] = {(void*)&p};
    return cudaLaunchCooperativeKernel((const void*)quantize_kernel<DT, METHOD, OBJ, BLOCK, FIX, 1>, dim3((unsigned)grid),
                                       dim3(256), args, 0, s);
}

template <int DT, int METHOD, int OBJ>
static cudaError_t dyn_block(const QuantParams& p, bool fix, int block, int sms, cudaStream_t s) {
    if (METHOD == 0 && !fix) {
        switch (block) {
            case 16: return launch_dyn<DT, METHOD, OBJ, 16, 0>(p, sms, s);
            case 32: return launch_dyn<DT, METHOD, OBJ, 32, 0>(p, sms, s);
            default: return launch_dyn<DT, METHOD, OBJ, 64, 0>(p, sms, s);
        }
    }
    switch (block) {
        case 16: return launch_dyn<DT, METHOD, OBJ, 16, 1>(p, sms, s);
        case 32: return launch_dyn<DT, METHOD, OBJ, 32, 1>(p, sms, s);
        default: return launch_dyn<DT, METHOD, OBJ, 64, 1>(p, sms, s);
    }
}

cudaError_t launch_quantize_dynamic(const QuantParams& p_in, int dtype, int method, int obj, int block, int sms,
                                    cudaStream_t s) {
    QuantParams p = p_in;
    bool fix;
    prepare_quant_params(p, method, obj, block, &fix);
    cudaError_t e;
    if (dtype == 0) {
        if (method == 1) e = dyn_block<0, 1, 0>(p, fix, block, sms, s);
        else if (obj == 1) e = dyn_block<0, 0, 1>(p, fix, block, sms, s);
        else e = dyn_block<0, 0, 0>(p, fix, block, sms, s);
    } else {
        if (method == 1) e = dyn_block<1, 1, 0>(p, fix, block, sms, s);
        else if (obj == 1) e = dyn_block<1, 0, 1>(p, fix, block, sms, s);
        else e = dyn_block<1, 0, 0>(p, fix, block, sms, s);
    }
    if (e != cudaSuccess) return e;
    return launch_swizzle_pad(p, sms, s);
}

}  // namespace nvfp4
