// Static-scale launches of the sweep kernel (S read from device memory) and
// the host-side dispatch shared with the dynamic-scale launches.
#include "quantize_kernel.cuh"

namespace nvfp4 {

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
    static std::atomic<int> occ_cache[kOccDevices];
    const int occ = occupancy_per_sm(occ_cache, quantize_kernel<DT, METHOD, OBJ, BLOCK, FIX, 0>, 256);
    const int64_t threads_needed = (p.nseg + 31) & ~(int64_t)31;
    int64_t grid = (threads_needed + 255) / 256;
    const int64_t cap = (int64_t)sms * occ;
    if (grid > cap) grid = cap;
    quantize_kernel<DT, METHOD, OBJ, BLOCK, FIX, 0><<<(int)grid, 256, 0, s>>>(p);
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

void prepare_quant_params(QuantParams& p, int method, int obj, int block, bool* fix) {
    const int def_lo = (obj == 0 && block == 16) ? -3 : -8;
    *fix = (method != 0) || (p.win_lo == def_lo && p.win_hi == 7 && !p.tight);
    p.need_rowcol = (p.sf_swizzled != nullptr) || (obj == 1);
    if (p.narrow) p.kb_div = make_fast_div((uint32_t)p.kb);
}

cudaError_t launch_swizzle_pad(const QuantParams& p, int sms, cudaStream_t s) {
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

cudaError_t launch_quantize(const QuantParams& p_in, int dtype, int method, int obj, int block, int sms,
                            cudaStream_t s) {
    QuantParams p = p_in;
    bool fix;
    prepare_quant_params(p, method, obj, block, &fix);
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
    return launch_swizzle_pad(p, sms, s);
}

}  // namespace nvfp4
