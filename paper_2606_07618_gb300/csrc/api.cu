// Host side of the C ABI declared in include/nvfp4ss.h: argument, alignment and
// overlap checks (all before any launch), then dispatch to the kernels.  The
// library never allocates, frees or synchronises; every call is asynchronous on
// the caller's stream.
#include <atomic>
#include <climits>
#include <cmath>
#include <cstdint>
#include <cstring>

#include <cuda_runtime.h>

#include "group_kernels.h"
#include "ldlq_kernels.h"
#include "nvfp4_kernels.h"
#include "nvfp4ss.h"

using namespace nvfp4;

namespace {

int sm_count() {
    static std::atomic<int> cache[64];           // zero-initialised; 0 = not looked up yet
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 0;
    if (dev < 64) {
        const int c = cache[dev].load(std::memory_order_relaxed);
        if (c > 0) return c;
    }
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    if (dev < 64) cache[dev].store(n, std::memory_order_relaxed);
    return n;
}

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

bool mul_ok(int64_t a, int64_t b, int64_t* out) {
    if (a < 0 || b < 0) return false;
    if (a != 0 && b > INT64_MAX / a) return false;
    *out = a * b;
    return true;
}

// [p, p+n) and [q, q+m) overlap?
bool overlap(const void* p, int64_t n, const void* q, int64_t m) {
    if (!p || !q || n <= 0 || m <= 0) return false;
    uintptr_t a = reinterpret_cast<uintptr_t>(p), b = reinterpret_cast<uintptr_t>(q);
    return a < b + (uintptr_t)m && b < a + (uintptr_t)n;
}

// The kernels dereference these pointers on the device: reject memory the GPU
// cannot address (plain pageable host memory or garbage) before launching.
bool device_accessible(const void* p) {
    if (!p) return true;
    cudaPointerAttributes at;
    cudaError_t e = cudaPointerGetAttributes(&at, p);
    if (e != cudaSuccess) {
        (void)cudaGetLastError();
        return false;
    }
    return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged ||
           (at.type == cudaMemoryTypeHost && at.devicePointer != nullptr);
}

struct Shape {
    int64_t n, kb, kpad4, nblocks, nseg, sw_bytes;
    int narrow;
};

nvfp4_status check_shape(int64_t rows, int64_t cols, int block, Shape* sh) {
    if (rows < 0 || cols < 0) return NVFP4_ERR_INVALID_ARG;
    if (block != 16 && block != 32 && block != 64) return NVFP4_ERR_UNSUPPORTED;
    if (cols % block != 0) return NVFP4_ERR_INVALID_ARG;
    if (!mul_ok(rows, cols, &sh->n)) return NVFP4_ERR_RANGE;
    sh->kb = cols / block;
    sh->kpad4 = (sh->kb + 3) / 4;
    sh->nblocks = rows * sh->kb;
    sh->nseg = sh->n / 16;
    int64_t rows_pad = (rows + 127) / 128 * 128, t;
    if (!mul_ok(rows_pad, sh->kpad4 * 4, &t)) return NVFP4_ERR_RANGE;
    sh->sw_bytes = t;
    sh->narrow = (sh->nblocks < ((int64_t)1 << 32)) && (sh->kb < ((int64_t)1 << 32));
    return NVFP4_OK;
}

// Extra arguments of the dynamic-scale variants (global scale computed in the launch).
struct DynArgs {
    float fp8_div;
    float* S_out;
    int* status_dev;
    void* workspace;
    size_t ws_bytes;
    unsigned wait_extra;     // 0 except in nvfp4_selftest_wait_timeout
};

nvfp4_status quantize_common(int method, const void* x, nvfp4_dtype dt, int64_t rows, int64_t cols, int block,
                             const float* S, nvfp4_objective obj, const float* w, int64_t w_row_stride,
                             int win_lo, int win_hi, uint8_t* codes, uint8_t* sf_linear, uint8_t* sf_swizzled,
                             float* block_loss, void* stream, const DynArgs* dyn = nullptr) {
    if (dt != NVFP4_IN_BF16 && dt != NVFP4_IN_F32) return NVFP4_ERR_INVALID_ARG;
    if (obj != NVFP4_OBJ_MSE && obj != NVFP4_OBJ_WMSE) return NVFP4_ERR_INVALID_ARG;
    Shape sh;
    nvfp4_status st = check_shape(rows, cols, block, &sh);
    if (st != NVFP4_OK) return st;
    if (sf_swizzled && block != 16) return NVFP4_ERR_UNSUPPORTED;
    int tight = 0;
    if (method == 0) {
        if (win_lo == NVFP4_WINDOW_TIGHT && win_hi == NVFP4_WINDOW_TIGHT) {
            tight = 1 | ((obj == NVFP4_OBJ_MSE && block == 16) ? 2 : 0);
            win_lo = win_hi = NVFP4_WINDOW_DEFAULT;
        }
        if (win_lo == NVFP4_WINDOW_DEFAULT && win_hi == NVFP4_WINDOW_DEFAULT) {
            win_lo = (obj == NVFP4_OBJ_MSE && block == 16) ? -3 : -8;   // Lemma 4.3 / Sec. 4.2.2
            win_hi = 7;                                                 // Lemma 4.2, alpha = 12/7
        } else if (win_lo < -126 || win_hi > 126 || win_lo > win_hi) {
            return NVFP4_ERR_INVALID_ARG;
        }
    }
    if (dyn) {
        if (!(dyn->fp8_div > 0.0f) || dyn->fp8_div > 1e30f) return NVFP4_ERR_INVALID_ARG;
        if (!dyn->S_out || !dyn->workspace || dyn->ws_bytes < kDynWorkspace) return NVFP4_ERR_INVALID_ARG;
        if (!aligned(dyn->workspace, 16) || !aligned(dyn->S_out, 4) || (dyn->status_dev && !aligned(dyn->status_dev, 4)))
            return NVFP4_ERR_ALIGNMENT;
        S = dyn->S_out;
    }
    if (sh.n == 0) return NVFP4_OK;
    if (!x || !S || !codes || (!sf_linear && !sf_swizzled)) return NVFP4_ERR_INVALID_ARG;
    if (obj == NVFP4_OBJ_WMSE) {
        if (!w) return NVFP4_ERR_INVALID_ARG;
        if (w_row_stride != 0 && w_row_stride < cols) return NVFP4_ERR_INVALID_ARG;
        if (w_row_stride < 0 || w_row_stride % 4 != 0) return NVFP4_ERR_ALIGNMENT;
        if (!aligned(w, 16)) return NVFP4_ERR_ALIGNMENT;
    }
    if (!aligned(x, 16) || !aligned(codes, 8) || !aligned(S, 4) || (block_loss && !aligned(block_loss, 4)))
        return NVFP4_ERR_ALIGNMENT;
    const int64_t xbytes = sh.n * (dt == NVFP4_IN_BF16 ? 2 : 4);
    int64_t wbytes = 0;
    if (obj == NVFP4_OBJ_WMSE) {
        if (w_row_stride == 0) {
            wbytes = cols * 4;
        } else if (!mul_ok(rows - 1, w_row_stride, &wbytes) || wbytes > INT64_MAX / 4 - cols) {
            return NVFP4_ERR_RANGE;
        } else {
            wbytes = (wbytes + cols) * 4;
        }
    }
    const int64_t cbytes = sh.n / 2, lbytes = sh.nblocks, sbytes = sh.sw_bytes, fbytes = sh.nblocks * 4;
    const void* outs[7] = {codes, sf_linear, sf_swizzled, block_loss, dyn ? dyn->workspace : nullptr,
                           dyn ? (const void*)dyn->status_dev : nullptr, dyn ? (const void*)dyn->S_out : nullptr};
    const int64_t olen[7] = {cbytes, lbytes, sbytes, fbytes, dyn ? (int64_t)dyn->ws_bytes : 0, 4, 4};
    for (int i = 0; i < 7; i++) {
        if (!outs[i]) continue;
        if (overlap(outs[i], olen[i], x, xbytes)) return NVFP4_ERR_INVALID_ARG;
        if (!dyn && overlap(outs[i], olen[i], S, 4)) return NVFP4_ERR_INVALID_ARG;
        if (obj == NVFP4_OBJ_WMSE && overlap(outs[i], olen[i], w, wbytes)) return NVFP4_ERR_INVALID_ARG;
        for (int j = i + 1; j < 7; j++)
            if (overlap(outs[i], olen[i], outs[j], olen[j])) return NVFP4_ERR_INVALID_ARG;
    }
    if (!device_accessible(x) || !device_accessible(S) || !device_accessible(codes) ||
        !device_accessible(sf_linear) || !device_accessible(sf_swizzled) || !device_accessible(block_loss) ||
        (obj == NVFP4_OBJ_WMSE && !device_accessible(w)) ||
        (dyn && (!device_accessible(dyn->workspace) || !device_accessible(dyn->status_dev))))
        return NVFP4_ERR_INVALID_ARG;
    const int sms = sm_count();
    if (sms <= 0) return NVFP4_ERR_CUDA;

    QuantParams p;
    p.x = x;
    p.S = S;
    p.w = (obj == NVFP4_OBJ_WMSE) ? w : nullptr;
    p.w_row_stride = w_row_stride;
    p.rows = rows;
    p.cols = cols;
    p.kb = sh.kb;
    p.kpad4 = sh.kpad4;
    p.nseg = sh.nseg;
    p.narrow = sh.narrow;
    p.win_lo = win_lo;
    p.win_hi = win_hi;
    p.tight = tight;
    p.codes = codes;
    p.sf_linear = sf_linear;
    p.sf_swizzled = sf_swizzled;
    p.block_loss = block_loss;
    p.fp8_div = 0.0f;
    p.S_out = nullptr;
    p.status_dev = nullptr;
    p.part_max = nullptr;
    p.part_bad = nullptr;
    p.barrier = nullptr;
    p.wait_extra = 0;
    const int dti = dt == NVFP4_IN_BF16 ? 0 : 1, obji = obj == NVFP4_OBJ_WMSE ? 1 : 0;
    cudaError_t e;
    if (dyn) {
        p.fp8_div = dyn->fp8_div;
        p.S_out = dyn->S_out;
        p.status_dev = dyn->status_dev;
        p.part_max = static_cast<float*>(dyn->workspace);
        p.part_bad = reinterpret_cast<int*>(p.part_max + kAmaxParts);
        p.barrier = reinterpret_cast<unsigned*>(p.part_bad + kAmaxParts);
        p.wait_extra = dyn->wait_extra;
        e = launch_quantize_dynamic(p, dti, method, obji, block, sms, static_cast<cudaStream_t>(stream));
    } else {
        e = launch_quantize(p, dti, method, obji, block, sms, static_cast<cudaStream_t>(stream));
    }
    return e == cudaSuccess ? NVFP4_OK : NVFP4_ERR_CUDA;
}

}  // namespace

extern "C" {

const char* nvfp4_status_string(nvfp4_status st) {
    switch (st) {
        case NVFP4_OK: return "ok";
        case NVFP4_ERR_INVALID_ARG: return "invalid argument";
        case NVFP4_ERR_UNSUPPORTED: return "unsupported configuration";
        case NVFP4_ERR_ALIGNMENT: return "misaligned pointer";
        case NVFP4_ERR_RANGE: return "size out of range";
        case NVFP4_ERR_CUDA: return "CUDA error";
    }
    return "unknown status";
}

size_t nvfp4_global_scale_workspace(int64_t n) {
    (void)n;
    return (size_t)kAmaxParts * (sizeof(float) + sizeof(int));
}

nvfp4_status nvfp4_global_scale(const void* x, nvfp4_dtype dt, int64_t n, float fp8_div, float* S_out,
                                int* status_dev, void* workspace, size_t ws_bytes, void* stream) {
    if (dt != NVFP4_IN_BF16 && dt != NVFP4_IN_F32) return NVFP4_ERR_INVALID_ARG;
    if (n < 0 || !(fp8_div > 0.0f) || fp8_div > 1e30f) return NVFP4_ERR_INVALID_ARG;
    if (!S_out || !workspace || (n > 0 && !x)) return NVFP4_ERR_INVALID_ARG;
    if (ws_bytes < nvfp4_global_scale_workspace(n)) return NVFP4_ERR_INVALID_ARG;
    if (n > INT64_MAX / 4) return NVFP4_ERR_RANGE;
    if ((x && !aligned(x, 16)) || !aligned(workspace, 16) || !aligned(S_out, 4) ||
        (status_dev && !aligned(status_dev, 4)))
        return NVFP4_ERR_ALIGNMENT;
    const int64_t xbytes = n * (dt == NVFP4_IN_BF16 ? 2 : 4);
    if (overlap(S_out, 4, x, xbytes) || overlap(workspace, (int64_t)ws_bytes, x, xbytes) ||
        overlap(S_out, 4, workspace, (int64_t)ws_bytes) || overlap(status_dev, 4, S_out, 4) ||
        overlap(status_dev, 4, workspace, (int64_t)ws_bytes) || overlap(status_dev, 4, x, xbytes))
        return NVFP4_ERR_INVALID_ARG;
    if (!device_accessible(x) || !device_accessible(S_out) || !device_accessible(workspace) ||
        !device_accessible(status_dev))
        return NVFP4_ERR_INVALID_ARG;
    const int sms = sm_count();
    if (sms <= 0) return NVFP4_ERR_CUDA;
    cudaError_t e = launch_global_scale(x, dt == NVFP4_IN_BF16 ? 0 : 1, n, fp8_div, S_out, status_dev, workspace, sms,
                                        static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? NVFP4_OK : NVFP4_ERR_CUDA;
}

nvfp4_status scalesweep_quantize(const void* x, nvfp4_dtype dt, int64_t rows, int64_t cols, int block,
                                 const float* S, nvfp4_objective obj, const float* w, int64_t w_row_stride,
                                 int win_lo, int win_hi, uint8_t* codes, uint8_t* sf_linear,
                                 uint8_t* sf_swizzled, float* block_loss, void* stream) {
    return quantize_common(0, x, dt, rows, cols, block, S, obj, w, w_row_stride, win_lo, win_hi, codes, sf_linear,
                           sf_swizzled, block_loss, stream);
}

size_t nvfp4_dynamic_workspace(void) { return kDynWorkspace; }

nvfp4_status scalesweep_quantize_dynamic(const void* x, nvfp4_dtype dt, int64_t rows, int64_t cols, int block,
                                         float fp8_div, nvfp4_objective obj, const float* w, int64_t w_row_stride,
                                         int win_lo, int win_hi, float* S_out, int* status_dev, void* workspace,
                                         size_t ws_bytes, uint8_t* codes, uint8_t* sf_linear, uint8_t* sf_swizzled,
                                         float* block_loss, void* stream) {
    const DynArgs d{fp8_div, S_out, status_dev, workspace, ws_bytes, 0};
    return quantize_common(0, x, dt, rows, cols, block, nullptr, obj, w, w_row_stride, win_lo, win_hi, codes,
                           sf_linear, sf_swizzled, block_loss, stream, &d);
}

static_assert(kGroupMax == NVFP4_GROUP_MAX, "group descriptor count");

size_t scalesweep_quantize_group_workspace(void) { return kGroupWorkspace; }

namespace {
// method 0 ScaleSweep (objective obj), 1 AbsMax (obj ignored: MSE, no weights read).
nvfp4_status group_common(int method, const nvfp4_group_tensor* tensors, int count, nvfp4_dtype dt, int block,
                          nvfp4_objective obj, float fp8_div, float* S, int* status_dev, void* workspace,
                          size_t ws_bytes, void* stream, unsigned wait_extra,
                          nvfp4_group_schedule schedule = NVFP4_GROUP_SCHEDULE_AUTO) {
    if (dt != NVFP4_IN_BF16 && dt != NVFP4_IN_F32) return NVFP4_ERR_INVALID_ARG;
    if (schedule != NVFP4_GROUP_SCHEDULE_AUTO && schedule != NVFP4_GROUP_SCHEDULE_TWO_PHASE &&
        schedule != NVFP4_GROUP_SCHEDULE_PIPELINED)
        return NVFP4_ERR_INVALID_ARG;
    if (method == 1) obj = NVFP4_OBJ_MSE;
    if (obj != NVFP4_OBJ_MSE && obj != NVFP4_OBJ_WMSE) return NVFP4_ERR_INVALID_ARG;
    if (!tensors || count < 1 || count > NVFP4_GROUP_MAX || !S) return NVFP4_ERR_INVALID_ARG;
    if (block != 16 && block != 32 && block != 64) return NVFP4_ERR_UNSUPPORTED;
    const bool dyn = fp8_div != 0.0f;
    if (dyn && (!(fp8_div > 0.0f) || fp8_div > 1e30f)) return NVFP4_ERR_INVALID_ARG;
    if (dyn && (!workspace || ws_bytes < kGroupWorkspace)) return NVFP4_ERR_INVALID_ARG;
    if (!aligned(S, 4) || (status_dev && !aligned(status_dev, 4)) || (workspace && !aligned(workspace, 16)))
        return NVFP4_ERR_ALIGNMENT;
    const int64_t esize = dt == NVFP4_IN_BF16 ? 2 : 4;

    // Buffers the launch writes and reads, for the overlap checks.
    constexpr int kMaxW = 3 * NVFP4_GROUP_MAX + 3, kMaxR = 2 * NVFP4_GROUP_MAX + 1;
    const void* wp[kMaxW];
    int64_t wl[kMaxW];
    const void* rp[kMaxR];
    int64_t rl[kMaxR];
    int nw = 0, nr = 0;
    auto add_w = [&](const void* q, int64_t n) { if (q && n > 0) { wp[nw] = q; wl[nw++] = n; } };
    auto add_r = [&](const void* q, int64_t n) { if (q && n > 0) { rp[nr] = q; rl[nr++] = n; } };
    if (dyn) add_w(S, 4 * (int64_t)count);
    else add_r(S, 4 * (int64_t)count);
    add_w(status_dev, 4);
    if (dyn) add_w(workspace, (int64_t)ws_bytes);

    Shape sh[NVFP4_GROUP_MAX];
    for (int i = 0; i < count; i++) {
        const nvfp4_group_tensor& t = tensors[i];
        nvfp4_status st = check_shape(t.rows, t.cols, block, &sh[i]);
        if (st != NVFP4_OK) return st;
        if (t.sf_swizzled && block != 16) return NVFP4_ERR_UNSUPPORTED;
        if (sh[i].n == 0) continue;
        if (!t.x || !t.codes || (!t.sf_linear && !t.sf_swizzled)) return NVFP4_ERR_INVALID_ARG;
        if (!aligned(t.x, 16) || !aligned(t.codes, 8)) return NVFP4_ERR_ALIGNMENT;
        if (sh[i].n > INT64_MAX / 4) return NVFP4_ERR_RANGE;
        int64_t wbytes = 0;
        if (obj == NVFP4_OBJ_WMSE) {
            if (!t.w || (t.w_row_stride != 0 && t.w_row_stride < t.cols)) return NVFP4_ERR_INVALID_ARG;
            if (t.w_row_stride < 0 || t.w_row_stride % 4 != 0 || !aligned(t.w, 16)) return NVFP4_ERR_ALIGNMENT;
            if (t.w_row_stride == 0) {
                wbytes = t.cols * 4;
            } else if (!mul_ok(t.rows - 1, t.w_row_stride, &wbytes) || wbytes > INT64_MAX / 4 - t.cols) {
                return NVFP4_ERR_RANGE;
            } else {
                wbytes = (wbytes + t.cols) * 4;
            }
        }
        add_r(t.x, sh[i].n * esize);
        if (obj == NVFP4_OBJ_WMSE) add_r(t.w, wbytes);
        add_w(t.codes, sh[i].n / 2);
        add_w(t.sf_linear, sh[i].nblocks);
        add_w(t.sf_swizzled, sh[i].sw_bytes);
    }
    for (int a = 0; a < nw; a++) {
        for (int b = a + 1; b < nw; b++)
            if (overlap(wp[a], wl[a], wp[b], wl[b])) return NVFP4_ERR_INVALID_ARG;
        for (int b = 0; b < nr; b++)
            if (overlap(wp[a], wl[a], rp[b], rl[b])) return NVFP4_ERR_INVALID_ARG;
    }
    for (int a = 0; a < nw; a++)
        if (!device_accessible(wp[a])) return NVFP4_ERR_INVALID_ARG;
    for (int b = 0; b < nr; b++)
        if (!device_accessible(rp[b])) return NVFP4_ERR_INVALID_ARG;
    if (!device_accessible(S)) return NVFP4_ERR_INVALID_ARG;
    const int sms = sm_count();
    if (sms <= 0) return NVFP4_ERR_CUDA;

    // Processing order: ascending size (stable), so the reduction that cannot
    // overlap a sweep (the first tensor's) is the smallest.
    int order[NVFP4_GROUP_MAX];
    for (int i = 0; i < count; i++) order[i] = i;
    for (int i = 1; i < count; i++)
        for (int k = i; k > 0 && sh[order[k]].n < sh[order[k - 1]].n; k--) {
            const int tmp = order[k];
            order[k] = order[k - 1];
            order[k - 1] = tmp;
        }
    GroupParams p;
    std::memset(&p, 0, sizeof(p));
    int64_t rows[NVFP4_GROUP_MAX];
    int64_t seg = 0;
    for (int k = 0; k < count; k++) {
        const int i = order[k];
        const nvfp4_group_tensor& t = tensors[i];
        GroupTensor& g = p.t[k];
        g.x = t.x;
        g.w = obj == NVFP4_OBJ_WMSE ? t.w : nullptr;
        g.w_row_stride = t.w_row_stride;
        g.codes = t.codes;
        g.sf_linear = t.sf_linear;
        g.sf_swizzled = t.sf_swizzled;
        g.kb = sh[i].kb;
        g.kpad4 = sh[i].kpad4;
        g.nseg = sh[i].nseg;
        g.seg_begin = seg;
        g.nvec = sh[i].n * esize / 16;
        g.narrow = sh[i].narrow;
        if (g.narrow && g.kb > 0) g.kb_div = make_fast_div((uint32_t)g.kb);
        g.s_index = i;
        rows[k] = t.rows;
        const int64_t unit = kGroupCtaSegments;          // a CTA's segments never straddle two tensors
        if (g.nseg > INT64_MAX - seg - unit) return NVFP4_ERR_RANGE;
        seg += (g.nseg + unit - 1) / unit * unit;
    }
    p.count = count;
    p.dyn = dyn ? 1 : 0;
    int64_t elements = 0;
    for (int i = 0; i < count; i++) elements += sh[i].n < kPipelineMinElements ? sh[i].n : kPipelineMinElements;
    p.pipelined = schedule == NVFP4_GROUP_SCHEDULE_PIPELINED ||
                  (schedule == NVFP4_GROUP_SCHEDULE_AUTO && count >= 2 && elements >= kPipelineMinElements);
    p.total_seg = seg;
    p.fp8_div = fp8_div;
    p.S = S;
    p.status_dev = status_dev;
    p.amax_bits = dyn ? static_cast<unsigned*>(workspace) : nullptr;
    p.arrived = dyn ? static_cast<unsigned*>(workspace) + kGroupMax : nullptr;
    p.wait_extra = wait_extra;
    const cudaError_t e = launch_quantize_group(p, rows, dt == NVFP4_IN_BF16 ? 0 : 1, method,
                                                obj == NVFP4_OBJ_WMSE ? 1 : 0, block, sms,
                                                static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? NVFP4_OK : NVFP4_ERR_CUDA;
}
}  // namespace

nvfp4_status scalesweep_quantize_group(const nvfp4_group_tensor* tensors, int count, nvfp4_dtype dt, int block,
                                       nvfp4_objective obj, float fp8_div, float* S, int* status_dev,
                                       void* workspace, size_t ws_bytes, void* stream) {
    return group_common(0, tensors, count, dt, block, obj, fp8_div, S, status_dev, workspace, ws_bytes, stream, 0);
}

nvfp4_status scalesweep_quantize_group_scheduled(const nvfp4_group_tensor* tensors, int count, nvfp4_dtype dt,
                                                 int block, nvfp4_objective obj, float fp8_div, float* S,
                                                 int* status_dev, void* workspace, size_t ws_bytes,
                                                 nvfp4_group_schedule schedule, void* stream) {
    return group_common(0, tensors, count, dt, block, obj, fp8_div, S, status_dev, workspace, ws_bytes, stream, 0,
                        schedule);
}

nvfp4_status absmax_quantize_group(const nvfp4_group_tensor* tensors, int count, nvfp4_dtype dt, int block,
                                   float fp8_div, float* S, int* status_dev, void* workspace, size_t ws_bytes,
                                   void* stream) {
    return group_common(1, tensors, count, dt, block, NVFP4_OBJ_MSE, fp8_div, S, status_dev, workspace, ws_bytes,
                        stream, 0);
}

nvfp4_status nvfp4_selftest_wait_timeout(int which, const void* x, int64_t rows, int64_t cols, float* S,
                                         int* status_dev, void* workspace, size_t ws_bytes, uint8_t* codes,
                                         uint8_t* sf_linear, void* stream) {
    if ((which != 0 && which != 1) || !status_dev || rows <= 0 || cols <= 0) return NVFP4_ERR_INVALID_ARG;
    if (which == 0) {
        const DynArgs d{256.0f, S, status_dev, workspace, ws_bytes, 1};
        return quantize_common(0, x, NVFP4_IN_BF16, rows, cols, 16, nullptr, NVFP4_OBJ_MSE, nullptr, 0,
                               NVFP4_WINDOW_DEFAULT, NVFP4_WINDOW_DEFAULT, codes, sf_linear, nullptr, nullptr, stream,
                               &d);
    }
    const nvfp4_group_tensor t{x, rows, cols, nullptr, 0, codes, sf_linear, nullptr};
    return group_common(0, &t, 1, NVFP4_IN_BF16, 16, NVFP4_OBJ_MSE, 256.0f, S, status_dev, workspace, ws_bytes,
                        stream, 1, NVFP4_GROUP_SCHEDULE_TWO_PHASE);
}

nvfp4_status absmax_quantize_dynamic(const void* x, nvfp4_dtype dt, int64_t rows, int64_t cols, int block,
                                     float fp8_div, float* S_out, int* status_dev, void* workspace, size_t ws_bytes,
                                     uint8_t* codes, uint8_t* sf_linear, uint8_t* sf_swizzled, float* block_loss,
                                     void* stream) {
    const DynArgs d{fp8_div, S_out, status_dev, workspace, ws_bytes, 0};
    return quantize_common(1, x, dt, rows, cols, block, nullptr, NVFP4_OBJ_MSE, nullptr, 0, 0, 0, codes, sf_linear,
                           sf_swizzled, block_loss, stream, &d);
}

nvfp4_status absmax_quantize(const void* x, nvfp4_dtype dt, int64_t rows, int64_t cols, int block,
                             const float* S, uint8_t* codes, uint8_t* sf_linear, uint8_t* sf_swizzled,
                             float* block_loss, void* stream) {
    return quantize_common(1, x, dt, rows, cols, block, S, NVFP4_OBJ_MSE, nullptr, 0, 0, 0, codes, sf_linear,
                           sf_swizzled, block_loss, stream);
}

nvfp4_status four_over_six_quantize(const void* x, nvfp4_dtype dt, int64_t rows, int64_t cols, int block,
                                    const float* S, nvfp4_objective obj, const float* w, int64_t w_row_stride,
                                    uint8_t* codes, uint8_t* sf_linear, uint8_t* sf_swizzled,
                                    float* block_loss, void* stream) {
    return quantize_common(2, x, dt, rows, cols, block, S, obj, w, w_row_stride, 0, 0, codes, sf_linear, sf_swizzled,
                           block_loss, stream);
}

nvfp4_status nvfp4_optimal_scale(const void* x, nvfp4_dtype dt, int64_t rows, int64_t cols, int block,
                                 const float* S, nvfp4_objective obj, const float* w, int64_t w_row_stride,
                                 float* s_opt, float* loss_opt, uint8_t* fp8_code, float* loss_fp8, void* stream) {
    if (dt != NVFP4_IN_BF16 && dt != NVFP4_IN_F32) return NVFP4_ERR_INVALID_ARG;
    if (obj != NVFP4_OBJ_MSE && obj != NVFP4_OBJ_WMSE) return NVFP4_ERR_INVALID_ARG;
    Shape sh;
    nvfp4_status st = check_shape(rows, cols, block, &sh);
    if (st != NVFP4_OK) return st;
    if (sh.n == 0) return NVFP4_OK;
    if (!x || !S || !s_opt || !loss_opt || (loss_fp8 && !fp8_code)) return NVFP4_ERR_INVALID_ARG;
    if (obj == NVFP4_OBJ_WMSE && (!w || (w_row_stride != 0 && w_row_stride < cols) || w_row_stride < 0))
        return NVFP4_ERR_INVALID_ARG;
    if (!aligned(x, 4) || !aligned(S, 4) || !aligned(s_opt, 4) || !aligned(loss_opt, 4) ||
        (loss_fp8 && !aligned(loss_fp8, 4)) || (w && !aligned(w, 4)))
        return NVFP4_ERR_ALIGNMENT;
    const int64_t xbytes = sh.n * (dt == NVFP4_IN_BF16 ? 2 : 4);
    const void* outs[4] = {s_opt, loss_opt, fp8_code, loss_fp8};
    const int64_t olen[4] = {sh.nblocks * 4, sh.nblocks * 4, sh.nblocks, sh.nblocks * 4};
    for (int i = 0; i < 4; i++) {
        if (!outs[i]) continue;
        if (overlap(outs[i], olen[i], x, xbytes) || overlap(outs[i], olen[i], S, 4)) return NVFP4_ERR_INVALID_ARG;
        for (int j = i + 1; j < 4; j++)
            if (overlap(outs[i], olen[i], outs[j], olen[j])) return NVFP4_ERR_INVALID_ARG;
    }
    if (!device_accessible(x) || !device_accessible(S) || !device_accessible(s_opt) || !device_accessible(loss_opt) ||
        !device_accessible(fp8_code) || !device_accessible(loss_fp8) ||
        (obj == NVFP4_OBJ_WMSE && !device_accessible(w)))
        return NVFP4_ERR_INVALID_ARG;
    const int sms = sm_count();
    if (sms <= 0) return NVFP4_ERR_CUDA;
    OptParams p;
    p.x = x;
    p.S = S;
    p.w = obj == NVFP4_OBJ_WMSE ? w : nullptr;
    p.w_row_stride = w_row_stride;
    p.rows = rows;
    p.cols = cols;
    p.kb = sh.kb;
    p.nblocks = sh.nblocks;
    p.s_opt = s_opt;
    p.loss_opt = loss_opt;
    p.fp8_code = fp8_code;
    p.loss_fp8 = loss_fp8;
    cudaError_t e = launch_optimal_scale(p, dt == NVFP4_IN_BF16 ? 0 : 1, obj == NVFP4_OBJ_WMSE ? 1 : 0, block, sms,
                                         static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? NVFP4_OK : NVFP4_ERR_CUDA;
}

nvfp4_status nvfp4_dequantize(const uint8_t* codes, const uint8_t* sf, nvfp4_sf_layout layout, const float* S,
                              int64_t rows, int64_t cols, int block, void* out, nvfp4_dtype out_dt,
                              void* stream) {
    if (layout != NVFP4_SF_LINEAR && layout != NVFP4_SF_SWIZZLED) return NVFP4_ERR_INVALID_ARG;
    if (out_dt != NVFP4_IN_BF16 && out_dt != NVFP4_IN_F32) return NVFP4_ERR_INVALID_ARG;
    Shape sh;
    nvfp4_status st = check_shape(rows, cols, block, &sh);
    if (st != NVFP4_OK) return st;
    if (layout == NVFP4_SF_SWIZZLED && block != 16) return NVFP4_ERR_UNSUPPORTED;
    if (sh.n == 0) return NVFP4_OK;
    if (!codes || !sf || !S || !out) return NVFP4_ERR_INVALID_ARG;
    if (!aligned(codes, 8) || !aligned(out, 16) || !aligned(S, 4)) return NVFP4_ERR_ALIGNMENT;
    const int64_t obytes = sh.n * (out_dt == NVFP4_IN_BF16 ? 2 : 4);
    const int64_t sfbytes = layout == NVFP4_SF_SWIZZLED ? sh.sw_bytes : sh.nblocks;
    if (overlap(out, obytes, codes, sh.n / 2) || overlap(out, obytes, sf, sfbytes) || overlap(out, obytes, S, 4))
        return NVFP4_ERR_INVALID_ARG;
    if (!device_accessible(codes) || !device_accessible(sf) || !device_accessible(S) || !device_accessible(out))
        return NVFP4_ERR_INVALID_ARG;
    const int sms = sm_count();
    if (sms <= 0) return NVFP4_ERR_CUDA;
    DequantParams p;
    p.codes = codes;
    p.sf = sf;
    p.S = S;
    p.rows = rows;
    p.cols = cols;
    p.kb = sh.kb;
    p.kpad4 = sh.kpad4;
    p.nseg = sh.nseg;
    p.narrow = sh.narrow;
    p.swizzled = layout == NVFP4_SF_SWIZZLED;
    p.block = block;
    p.out = out;
    cudaError_t e = launch_dequantize(p, out_dt == NVFP4_IN_BF16 ? 0 : 1, sms, static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? NVFP4_OK : NVFP4_ERR_CUDA;
}

size_t nvfp4_ldlq_prepare_workspace(int64_t n) { return n > 0 ? ldlq_prepare_workspace(n) : 0; }

nvfp4_status nvfp4_ldlq_prepare(const float* H, int64_t n, float damp, int32_t* perm, float* U, float* D,
                                int* status_dev, void* workspace, size_t ws_bytes, void* stream) {
    if (n < 0 || !(damp >= 0.0f) || !isfinite(damp)) return NVFP4_ERR_INVALID_ARG;
    if (n == 0) return NVFP4_OK;
    if (n > (int64_t)1 << 20) return NVFP4_ERR_RANGE;
    if (!H || !perm || !U || !D || !workspace) return NVFP4_ERR_INVALID_ARG;
    if (ws_bytes < ldlq_prepare_workspace(n)) return NVFP4_ERR_INVALID_ARG;
    if (!aligned(H, 4) || !aligned(perm, 4) || !aligned(U, 4) || !aligned(D, 4) || !aligned(workspace, 256) ||
        (status_dev && !aligned(status_dev, 4)))
        return NVFP4_ERR_ALIGNMENT;
    const int64_t mat = n * n * 4;
    const void* bufs[6] = {H, perm, U, D, workspace, status_dev};
    const int64_t lens[6] = {mat, n * 4, mat, n * 4, (int64_t)ldlq_prepare_workspace(n), 4};
    for (int i = 0; i < 6; i++)
        for (int j = i + 1; j < 6; j++)
            if (overlap(bufs[i], lens[i], bufs[j], lens[j])) return NVFP4_ERR_INVALID_ARG;
    for (int i = 0; i < 6; i++)
        if (!device_accessible(bufs[i])) return NVFP4_ERR_INVALID_ARG;
    const int sms = sm_count();
    if (sms <= 0) return NVFP4_ERR_CUDA;
    cudaError_t e = launch_ldlq_prepare(H, n, damp, perm, U, D, status_dev, workspace, sms,
                                        static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? NVFP4_OK : NVFP4_ERR_CUDA;
}

size_t nvfp4_ldlq_workspace(int64_t rows, int64_t cols) {
    int64_t rc;
    if (rows <= 0 || cols <= 0 || !mul_ok(rows, cols, &rc) || rc > INT64_MAX / 8) return 0;
    return ldlq_quantize_workspace(rows, cols);
}

nvfp4_status ldlq_quantize(const void* W, nvfp4_dtype dt, int64_t rows, int64_t cols, int block, const float* S,
                           const uint8_t* sf_linear, const int32_t* perm, const float* U, uint8_t* codes,
                           int* status_dev, void* workspace, size_t ws_bytes, void* stream) {
    if (dt != NVFP4_IN_BF16 && dt != NVFP4_IN_F32) return NVFP4_ERR_INVALID_ARG;
    Shape sh;
    nvfp4_status st = check_shape(rows, cols, block, &sh);
    if (st != NVFP4_OK) return st;
    if (sh.n == 0) return NVFP4_OK;
    if (cols > (int64_t)1 << 20 || rows > (int64_t)1 << 23) return NVFP4_ERR_RANGE;
    if (!W || !S || !sf_linear || !perm || !U || !codes || !workspace) return NVFP4_ERR_INVALID_ARG;
    if (ws_bytes < ldlq_quantize_workspace(rows, cols)) return NVFP4_ERR_INVALID_ARG;
    if (!aligned(W, dt == NVFP4_IN_BF16 ? 2 : 4) || !aligned(S, 4) || !aligned(perm, 4) || !aligned(U, 4) ||
        !aligned(workspace, 256) || (status_dev && !aligned(status_dev, 4)))
        return NVFP4_ERR_ALIGNMENT;
    const int64_t wbytes = sh.n * (dt == NVFP4_IN_BF16 ? 2 : 4);
    const void* ins[6] = {W, S, sf_linear, perm, U, status_dev};
    const int64_t ilen[6] = {wbytes, 4, sh.nblocks, cols * 4, cols * cols * 4, 4};
    const int64_t wsb = (int64_t)ldlq_quantize_workspace(rows, cols);
    for (int i = 0; i < 6; i++)
        if (overlap(codes, sh.n / 2, ins[i], ilen[i]) || overlap(workspace, wsb, ins[i], ilen[i]))
            return NVFP4_ERR_INVALID_ARG;
    if (overlap(codes, sh.n / 2, workspace, wsb)) return NVFP4_ERR_INVALID_ARG;
    for (int i = 0; i < 6; i++)
        if (!device_accessible(ins[i])) return NVFP4_ERR_INVALID_ARG;
    if (!device_accessible(codes) || !device_accessible(workspace)) return NVFP4_ERR_INVALID_ARG;
    const int sms = sm_count();
    if (sms <= 0) return NVFP4_ERR_CUDA;
    LdlqParams p;
    p.W = W;
    p.rows = rows;
    p.n = cols;
    p.perm = perm;
    p.U = U;
    p.sf = sf_linear;
    p.kb = sh.kb;
    p.block = block;
    p.S = S;
    p.status = status_dev;
    p.T = nullptr;
    p.Wp = nullptr;
    p.qb = nullptr;
    p.sfp = nullptr;
    cudaError_t e = launch_ldlq_quantize(p, dt == NVFP4_IN_BF16 ? 0 : 1, codes, workspace, sms,
                                         static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? NVFP4_OK : NVFP4_ERR_CUDA;
}

nvfp4_status nvfp4_row_shard_layout(int64_t rows, int64_t cols, int block, int world, int rank,
                                    nvfp4_row_shard* out) {
    if (!out || world < 1 || rank < 0 || rank >= world) return NVFP4_ERR_INVALID_ARG;
    Shape sh;
    const nvfp4_status st = check_shape(rows, cols, block, &sh);
    if (st != NVFP4_OK) return st;
    const int64_t rb = (rows + 127) / 128;                       // row blocks of 128
    if (rb > INT64_MAX / world) return NVFP4_ERR_RANGE;
    const int64_t b0 = rb * rank / world, b1 = rb * (rank + 1) / world;
    const int64_t r0 = b0 * 128 < rows ? b0 * 128 : rows, r1 = b1 * 128 < rows ? b1 * 128 : rows;
    out->row_begin = r0;
    out->row_end = r1;
    out->x_offset = r0 * cols;
    out->codes_offset = r0 * cols / 2;
    out->sf_linear_offset = r0 * sh.kb;
    if (block == 16) {
        out->sf_swizzled_offset = b0 * sh.kpad4 * 512;
        out->sf_swizzled_bytes = (b1 - b0) * sh.kpad4 * 512;
    } else {
        out->sf_swizzled_offset = -1;
        out->sf_swizzled_bytes = -1;
    }
    return NVFP4_OK;
}

}  // extern "C"
