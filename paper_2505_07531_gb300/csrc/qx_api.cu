// C ABI of the qx library: argument validation, dispatch, device status.
// The declarations, with the meaning, layout, ownership and error behaviour of
// every argument, are in include/qx.h.
#include <algorithm>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <vector>

#include "qx.h"
#include "qx_kernels.cuh"

#define QX_API extern "C" __attribute__((visibility("default")))

namespace {

constexpr int kMaxDevices = 64;

// One status word per device, in the library's own device memory (a file-scope
// __device__ symbol; nothing is allocated).  Its device address is fetched
// once per device with that device current.
__device__ uint32_t g_status_word;

struct DeviceInfo {
    uint32_t *status = nullptr;
    int num_sms = 0;
    bool ready = false;
};

DeviceInfo g_dev[kMaxDevices];
std::mutex g_mu;

// The name of the CUDA error behind this thread's last QX_ERR_CUDA.
thread_local const char *t_last_error = "no error";

qx_status from_cuda(cudaError_t e) {
    if (e == cudaSuccess) return QX_OK;
    t_last_error = cudaGetErrorName(e);
    return QX_ERR_CUDA;
}

qx_status device_info(DeviceInfo **out) {
    int dev = 0;
    qx_status s = from_cuda(cudaGetDevice(&dev));
    if (s != QX_OK) return s;
    if (dev < 0 || dev >= kMaxDevices) return QX_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_mu);
    DeviceInfo &d = g_dev[dev];
    if (!d.ready) {
        void *p = nullptr;
        if ((s = from_cuda(cudaGetSymbolAddress(&p, g_status_word))) != QX_OK) return s;
        int sms = 0;
        if ((s = from_cuda(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev))) != QX_OK) return s;
        d.status = static_cast<uint32_t *>(p);
        d.num_sms = sms;
        d.ready = true;
    }
    *out = &d;
    return QX_OK;
}

uint64_t wait_limit_ns() {
    // bounded waits inside the tensor-core kernel; QX_WAIT_LIMIT_MS overrides
    const char *s = std::getenv("QX_WAIT_LIMIT_MS");
    uint64_t ms = 2000;
    if (s != nullptr) {
        const long long v = std::atoll(s);
        if (v > 0 && v < 600000) ms = (uint64_t)v;
    }
    return ms * 1000000ull;
}

bool aligned(const void *p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

// rows (tokens) of one qx_quantize_act / qx_dequant_act call
constexpr int64_t kMaxActRows = (int64_t)1 << 24;

int ilog2(int v) {
    int r = 0;
    while ((1 << r) < v) ++r;
    return r;
}

qx_status check_recipe(const qx_recipe *r) {
    if (r == nullptr) return QX_ERR_INVALID_ARG;
    if (r->kind != QX_UNIFORM && r->kind != QX_LUT) return QX_ERR_INVALID_ARG;
    if (r->bits != 3 && r->bits != 4) return QX_ERR_UNSUPPORTED;
    if (r->kind == QX_LUT && r->bits != 3) return QX_ERR_UNSUPPORTED;
    const int g = r->group_size;
    if (g != 32 && g != 64 && g != 128 && g != 256) return QX_ERR_UNSUPPORTED;
    if (r->kind == QX_LUT && (r->lloyd_iters < 0 || r->lloyd_iters > 1000)) return QX_ERR_INVALID_ARG;
    return QX_OK;
}

qx_status check_shape(int64_t n, int64_t k, const qx_recipe *r) {
    if (n < 1 || k < 1) return QX_ERR_INVALID_ARG;
    if (k % 128 != 0 || k % r->group_size != 0) return QX_ERR_UNSUPPORTED;
    // grid and index limits of the kernels
    if (n > (int64_t)1 << 22 || k > (int64_t)1 << 20) return QX_ERR_UNSUPPORTED;
    return QX_OK;
}

qx_status check_packed(const qx_packed *p) {
    if (p == nullptr) return QX_ERR_INVALID_ARG;
    qx_status s = check_recipe(&p->recipe);
    if (s != QX_OK) return s;
    s = check_shape(p->n, p->k, &p->recipe);
    if (s != QX_OK) return s;
    if (p->codes == nullptr) return QX_ERR_INVALID_ARG;
    if (!aligned(p->codes, 16)) return QX_ERR_ALIGNMENT;
    if (p->recipe.kind == QX_UNIFORM) {
        if (p->scales == nullptr || p->zeros == nullptr) return QX_ERR_INVALID_ARG;
        if (!aligned(p->scales, 2)) return QX_ERR_ALIGNMENT;
    } else {
        if (p->luts == nullptr) return QX_ERR_INVALID_ARG;
        if (!aligned(p->luts, 16)) return QX_ERR_ALIGNMENT;
    }
    return QX_OK;
}

}  // namespace

QX_API int32_t qx_version(void) { return 100; }

QX_API const char *qx_last_error_string(void) { return t_last_error; }

QX_API const char *qx_status_string(qx_status s) {
    switch (s) {
        case QX_OK: return "ok";
        case QX_ERR_INVALID_ARG: return "invalid argument";
        case QX_ERR_UNSUPPORTED: return "unsupported recipe, shape or batch";
        case QX_ERR_ALIGNMENT: return "pointer alignment";
        case QX_ERR_CUDA: return "CUDA error";
        case QX_ERR_TIMEOUT: return "device wait timed out";
        case QX_ERR_NONFINITE: return "non-finite weight";
    }
    return "unknown status";
}

QX_API qx_status qx_packed_size(int64_t n, int64_t k, const qx_recipe *recipe, qx_sizes *out) {
    if (out == nullptr) return QX_ERR_INVALID_ARG;
    qx_status s = check_recipe(recipe);
    if (s != QX_OK) return s;
    s = check_shape(n, k, recipe);
    if (s != QX_OK) return s;
    const int64_t G = k / recipe->group_size;
    out->codes = (uint64_t)(n * k * recipe->bits / 8);
    if (recipe->kind == QX_UNIFORM) {
        out->scales = (uint64_t)(n * G * 2);
        out->zeros = (uint64_t)(n * ((G + 1) / 2));
        out->luts = 0;
    } else {
        out->scales = 0;
        out->zeros = 0;
        out->luts = (uint64_t)(n * G * (1 << recipe->bits) * 2);
    }
    return QX_OK;
}

QX_API qx_status qx_quantize(const void *W, int64_t n, int64_t k, const qx_recipe *recipe, const qx_packed *out,
                             void *stream) {
    if (W == nullptr || out == nullptr || recipe == nullptr) return QX_ERR_INVALID_ARG;
    qx_status s = check_packed(out);
    if (s != QX_OK) return s;
    if (out->n != n || out->k != k || out->recipe.bits != recipe->bits ||
        out->recipe.group_size != recipe->group_size || out->recipe.kind != recipe->kind)
        return QX_ERR_INVALID_ARG;
    if (!aligned(W, 16)) return QX_ERR_ALIGNMENT;
    DeviceInfo *d = nullptr;
    if ((s = device_info(&d)) != QX_OK) return s;
    qx::QuantArgs a{};
    a.W = static_cast<const __half *>(W);
    a.n = n;
    a.k = k;
    a.bits = recipe->bits;
    a.g = recipe->group_size;
    a.kind = recipe->kind;
    a.lloyd_iters = recipe->lloyd_iters;
    a.G = (int)(k / a.g);
    a.zbytes = (a.G + 1) / 2;
    a.codes = static_cast<uint8_t *>(out->codes);
    a.scales = static_cast<__half *>(out->scales);
    a.zeros = static_cast<uint8_t *>(out->zeros);
    a.luts = static_cast<__half *>(out->luts);
    a.status = d->status;
    return from_cuda(qx::launch_quantize(a, d->num_sms, static_cast<cudaStream_t>(stream)));
}

QX_API qx_status qx_dequant(const qx_packed *p, void *W_out, void *stream) {
    qx_status s = check_packed(p);
    if (s != QX_OK) return s;
    if (W_out == nullptr) return QX_ERR_INVALID_ARG;
    if (!aligned(W_out, 16)) return QX_ERR_ALIGNMENT;
    DeviceInfo *d = nullptr;
    if ((s = device_info(&d)) != QX_OK) return s;
    qx::DequantArgs a{};
    a.codes = static_cast<const uint8_t *>(p->codes);
    a.scales = static_cast<const __half *>(p->scales);
    a.zeros = static_cast<const uint8_t *>(p->zeros);
    a.luts = static_cast<const __half *>(p->luts);
    a.n = p->n;
    a.k = p->k;
    a.bits = p->recipe.bits;
    a.g = p->recipe.group_size;
    a.kind = p->recipe.kind;
    a.G = (int)(p->k / a.g);
    a.zbytes = (a.G + 1) / 2;
    a.W = static_cast<__half *>(W_out);
    return from_cuda(qx::launch_dequant(a, d->num_sms, static_cast<cudaStream_t>(stream)));
}

namespace {

// Decode plans (CTA slices, shared-memory split, TMA descriptors) depend only
// on the device, the recipe, the shapes, the buffer addresses and the batch
// slice.  A model decodes the same matrices into the same buffers every step,
// so the last plans are kept and reused: planning and descriptor encoding
// would otherwise cost host time on every launch.
struct PlanEntry {
    bool used = false;
    int dev = -1;
    qx::GemvMulti plan;
};
constexpr int kPlanCache = 32;
PlanEntry g_plans[kPlanCache];
int g_plan_next = 0;
std::mutex g_plan_mu;

bool same_inputs(const qx::GemvMulti &p, const qx::GemvMulti &a) {
    if (p.count != a.count || p.bits != a.bits || p.kind != a.kind || p.batch != a.batch || p.y_f32 != a.y_f32 ||
        p.status != a.status || p.wait_limit_ns != a.wait_limit_ns || p.nphase != a.nphase ||
        p.phase_ctr != a.phase_ctr || p.split_part != a.split_part || p.split_flag != a.split_flag)
        return false;
    for (int i = 0; i <= a.nphase; ++i)
        if (p.phase_first[i] != a.phase_first[i]) return false;
    for (int i = 0; i < a.count; ++i) {
        const qx::GemvMat &u = p.mat[i], &v = a.mat[i];
        if (u.codes != v.codes || u.scales != v.scales || u.zeros != v.zeros || u.luts != v.luts || u.x != v.x ||
            u.y != v.y || u.n != v.n || u.k != v.k || u.G != v.G || u.log2g != v.log2g)
            return false;
    }
    return true;
}

// plan_gemv through the cache; `a` holds the inputs on entry, the plan on return.
bool plan_cached(qx::GemvMulti &a, const DeviceInfo *d) {
    int dev = -1;
    cudaGetDevice(&dev);
    {
        std::lock_guard<std::mutex> lock(g_plan_mu);
        for (int i = 0; i < kPlanCache; ++i) {
            if (g_plans[i].used && g_plans[i].dev == dev && same_inputs(g_plans[i].plan, a)) {
                a = g_plans[i].plan;
                return true;
            }
        }
    }
    if (!qx::plan_gemv(a, d->num_sms)) return false;
    std::lock_guard<std::mutex> lock(g_plan_mu);
    PlanEntry &e = g_plans[g_plan_next];
    g_plan_next = (g_plan_next + 1) % kPlanCache;
    e.used = true;
    e.dev = dev;
    e.plan = a;
    return true;
}

// One decode launch over `count` matrices for activation rows b0 .. b0+nb-1.
// Should a plan not fit (a tensor map the driver refuses, or shared memory),
// the group is split per matrix, then the rows are halved.
// The per-matrix launch fields of packed matrix p with activation rows b0..
void fill_mat(qx::GemvMat &M, const qx_packed &p, const void *x, void *y, int b0, int esz) {
    M.codes = static_cast<const uint8_t *>(p.codes);
    M.scales = static_cast<const __half *>(p.scales);
    M.zeros = static_cast<const uint8_t *>(p.zeros);
    M.luts = static_cast<const __half *>(p.luts);
    M.x = static_cast<const __half *>(x) + (int64_t)b0 * p.k;
    M.y = static_cast<uint8_t *>(y) + (int64_t)b0 * p.n * esz;
    M.n = p.n;
    M.k = p.k;
    M.G = (int)(p.k / p.recipe.group_size);
    M.zbytes = (M.G + 1) / 2;
    M.log2g = ilog2(p.recipe.group_size);
}

qx_status gemv_chunk(const qx_packed *mats, int count, const void *const *x, int b0, int nb, void *const *y,
                     int y_dtype, int flags, cudaStream_t st, DeviceInfo *d) {
    const int esz = y_dtype == QX_F32 ? 4 : 2;
    qx::GemvMulti a{};
    a.count = count;
    a.nphase = 1;
    a.phase_first[0] = 0;
    a.phase_first[1] = count;
    a.bits = mats[0].recipe.bits;
    a.kind = mats[0].recipe.kind;
    a.batch = nb;
    a.y_f32 = y_dtype == QX_F32;
    a.status = d->status;
    a.wait_limit_ns = wait_limit_ns();
    for (int i = 0; i < count; ++i) fill_mat(a.mat[i], mats[i], x[i], y[i], b0, esz);
    if (plan_cached(a, d))
        return from_cuda(qx::launch_gemv_multi(a, st, (flags & QX_GEMV_PDL) != 0));
    if (count > 1) {
        for (int i = 0; i < count; ++i) {
            qx_status s = gemv_chunk(&mats[i], 1, &x[i], b0, nb, &y[i], y_dtype, flags, st, d);
            if (s != QX_OK) return s;
        }
        return QX_OK;
    }
    if (nb > 1) {
        const int h = nb / 2;
        qx_status s = gemv_chunk(mats, 1, x, b0, h, y, y_dtype, flags, st, d);
        return s != QX_OK ? s : gemv_chunk(mats, 1, x, b0 + h, nb - h, y, y_dtype, flags, st, d);
    }
    return QX_ERR_UNSUPPORTED;
}

// One launch covers the whole batch (1..16 rows of x): the kernel reads x from
// global memory, so the weights are streamed once whatever the batch.
qx_status run_gemv(const qx_packed *mats, int count, const void *const *x, int batch, void *const *y,
                   int y_dtype, int flags, cudaStream_t st, DeviceInfo *d) {
    return gemv_chunk(mats, count, x, 0, batch, y, y_dtype, flags, st, d);
}

qx_status check_gemv_args(const qx_packed *p, const void *x, int32_t batch, const void *y, int32_t y_dtype) {
    qx_status s = check_packed(p);
    if (s != QX_OK) return s;
    if (x == nullptr || y == nullptr) return QX_ERR_INVALID_ARG;
    if (y_dtype != QX_F16 && y_dtype != QX_F32) return QX_ERR_INVALID_ARG;
    if (batch < 1) return QX_ERR_INVALID_ARG;
    if (batch > 16) return QX_ERR_UNSUPPORTED;
    if (p->k > 32768) return QX_ERR_UNSUPPORTED;  // x and a row must fit shared memory
    if (!aligned(x, 16)) return QX_ERR_ALIGNMENT;
    if (!aligned(y, y_dtype == QX_F32 ? 4 : 2)) return QX_ERR_ALIGNMENT;
    return QX_OK;
}

}  // namespace

QX_API qx_status qx_gemv(const qx_packed *p, const void *x, int32_t batch, void *y, int32_t y_dtype,
                         void *stream) {
    qx_status s = check_gemv_args(p, x, batch, y, y_dtype);
    if (s != QX_OK) return s;
    DeviceInfo *d = nullptr;
    if ((s = device_info(&d)) != QX_OK) return s;
    return run_gemv(p, 1, &x, batch, &y, y_dtype, 0, static_cast<cudaStream_t>(stream), d);
}

namespace {

qx_status check_gemv_multi(const qx_packed *mats, int32_t count, const void *const *x, int32_t batch,
                           void *const *y, int32_t y_dtype, int32_t flags) {
    if (mats == nullptr || x == nullptr || y == nullptr || count < 1) return QX_ERR_INVALID_ARG;
    if (count > qx::kMaxGemvMats) return QX_ERR_UNSUPPORTED;
    if ((flags & ~QX_GEMV_PDL) != 0) return QX_ERR_INVALID_ARG;
    for (int i = 0; i < count; ++i) {
        qx_status s = check_gemv_args(&mats[i], x[i], batch, y[i], y_dtype);
        if (s != QX_OK) return s;
        if (mats[i].recipe.bits != mats[0].recipe.bits || mats[i].recipe.kind != mats[0].recipe.kind)
            return QX_ERR_INVALID_ARG;
    }
    return QX_OK;
}

}  // namespace

QX_API qx_status qx_gemv_multi(const qx_packed *mats, int32_t count, const void *const *x, int32_t batch,
                               void *const *y, int32_t y_dtype, int32_t flags, void *stream) {
    qx_status s = check_gemv_multi(mats, count, x, batch, y, y_dtype, flags);
    if (s != QX_OK) return s;
    DeviceInfo *d = nullptr;
    if ((s = device_info(&d)) != QX_OK) return s;
    return run_gemv(mats, count, x, batch, y, y_dtype, flags, static_cast<cudaStream_t>(stream), d);
}

namespace {

qx_status check_chain(const qx_gemv_group *groups, int32_t ngroups, int32_t batch, int32_t y_dtype, int32_t flags) {
    if (groups == nullptr || ngroups < 1 || ngroups > 64) return QX_ERR_INVALID_ARG;
    for (int i = 0; i < ngroups; ++i) {
        const qx_gemv_group &g = groups[i];
        const qx_status s = check_gemv_multi(g.mats, g.count, g.x, batch, g.y, y_dtype, flags);
        if (s != QX_OK) return s;
    }
    return QX_OK;
}

qx_status run_chain(const qx_gemv_group *groups, int32_t ngroups, int32_t batch, int32_t y_dtype, int32_t flags,
                    cudaStream_t st, DeviceInfo *d) {
    for (int i = 0; i < ngroups; ++i) {
        const qx_gemv_group &g = groups[i];
        const qx_status s = run_gemv(g.mats, g.count, g.x, batch, g.y, y_dtype, flags, st, d);
        if (s != QX_OK) return s;
    }
    return QX_OK;
}

qx_status check_copies(const qx_copy *c, int32_t n) {
    if (n < 0 || n > 16 || (n > 0 && c == nullptr)) return QX_ERR_INVALID_ARG;
    for (int i = 0; i < n; ++i)
        if (c[i].dst == nullptr || c[i].src == nullptr) return QX_ERR_INVALID_ARG;
    return QX_OK;
}

}  // namespace

QX_API qx_status qx_gemv_chain(const qx_gemv_group *groups, int32_t ngroups, int32_t batch, int32_t y_dtype,
                               int32_t flags, void *stream) {
    qx_status s = check_chain(groups, ngroups, batch, y_dtype, flags);
    if (s != QX_OK) return s;
    DeviceInfo *d = nullptr;
    if ((s = device_info(&d)) != QX_OK) return s;
    return run_chain(groups, ngroups, batch, y_dtype, flags, static_cast<cudaStream_t>(stream), d);
}

namespace {

qx_status run_chain_fused(const qx_gemv_group *groups, int32_t ngroups, int32_t batch, int32_t y_dtype,
                          int32_t flags, void *ws, cudaStream_t st, DeviceInfo *d);

// The copies and launches of one decode step, issued on `st` (ws non-null: the
// groups as one fused launch).
// The copies of one direction as one copy kernel (qx_copy.cu) when every
// host buffer is pinned and mapped, every device buffer is device memory and
// they are small (a decode step's x and y): a copy engine's start-up costs
// more than such copies take.  False leaves them to cudaMemcpyAsync.
bool kernel_copies(const qx_copy *c, int32_t n, bool h2d, qx::CopyList &l) {
    if (n < 1 || n > qx::kMaxCopies) return false;
    int64_t total = 0;
    l.n = n;
    for (int i = 0; i < n; ++i) {
        const void *host = h2d ? c[i].src : c[i].dst;
        const void *dev = h2d ? c[i].dst : c[i].src;
        cudaPointerAttributes ah, ad;
        if (cudaPointerGetAttributes(&ah, host) != cudaSuccess || cudaPointerGetAttributes(&ad, dev) != cudaSuccess) {
            cudaGetLastError();
            return false;
        }
        if (ah.type != cudaMemoryTypeHost || ah.devicePointer == nullptr || ad.type != cudaMemoryTypeDevice)
            return false;
        total += (int64_t)c[i].bytes;
        uint8_t *hd = static_cast<uint8_t *>(ah.devicePointer);  // the host buffer's device address
        uint8_t *dd = static_cast<uint8_t *>(const_cast<void *>(dev));
        l.src[i] = h2d ? hd : dd;
        l.dst[i] = h2d ? dd : hd;
        l.bytes[i] = (int64_t)c[i].bytes;
    }
    return total <= ((int64_t)4 << 20);
}

qx_status issue_step(const qx_copy *in, int32_t nin, const qx_gemv_group *groups, int32_t ngroups, int32_t batch,
                     int32_t y_dtype, int32_t flags, void *ws, const qx_copy *out, int32_t nout, cudaStream_t st,
                     DeviceInfo *d) {
    qx_status s = QX_OK;
    qx::CopyList cl{};
    // in: stream-ordered after whatever may still read the device buffers
    if (kernel_copies(in, nin, true, cl)) {
        if ((s = from_cuda(qx::launch_copies(cl, d->num_sms, false, st))) != QX_OK) return s;
    } else {
        for (int i = 0; i < nin; ++i)
            if ((s = from_cuda(cudaMemcpyAsync(in[i].dst, in[i].src, in[i].bytes, cudaMemcpyHostToDevice, st))) !=
                QX_OK)
                return s;
    }
    s = ws != nullptr ? run_chain_fused(groups, ngroups, batch, y_dtype, flags, ws, st, d)
                      : run_chain(groups, ngroups, batch, y_dtype, flags, st, d);
    if (s != QX_OK) return s;
    // out: under PDL the copy kernel starts early and waits in the kernel for
    // the matmuls to finish
    if (kernel_copies(out, nout, false, cl)) {
        if ((s = from_cuda(qx::launch_copies(cl, d->num_sms, true, st))) != QX_OK) return s;
    } else {
        for (int i = 0; i < nout; ++i)
            if ((s = from_cuda(cudaMemcpyAsync(out[i].dst, out[i].src, out[i].bytes, cudaMemcpyDeviceToHost, st))) !=
                QX_OK)
                return s;
    }
    return QX_OK;
}

// A model repeats the same decode step (same buffers, same shapes) every
// token.  Its copies and launches are captured once as a CUDA graph and the
// graph is replayed: one launch instead of a launch per group and a copy per
// buffer, with the groups' programmatic dependencies kept as graph edges.
// The graphs are kept by everything the step depends on, like the plans.
struct StepGraph {
    bool used = false;
    int dev = -1;
    std::vector<uint8_t> key;
    cudaGraphExec_t exec = nullptr;
};
constexpr int kStepGraphs = 16;
StepGraph g_steps[kStepGraphs];
int g_step_next = 0;
std::mutex g_step_mu;
cudaStream_t g_capture[kMaxDevices] = {};

void key_put(std::vector<uint8_t> &k, const void *p, size_t n) {
    const uint8_t *b = static_cast<const uint8_t *>(p);
    k.insert(k.end(), b, b + n);
}

std::vector<uint8_t> step_key(const qx_copy *in, int32_t nin, const qx_gemv_group *groups, int32_t ngroups,
                              int32_t batch, int32_t y_dtype, int32_t flags, const void *ws, const qx_copy *out,
                              int32_t nout) {
    std::vector<uint8_t> k;
    const int32_t sc[6] = {nin, ngroups, batch, y_dtype, flags, nout};
    key_put(k, sc, sizeof(sc));
    key_put(k, &ws, sizeof(ws));
    for (int i = 0; i < nin; ++i) key_put(k, &in[i], sizeof(qx_copy));
    for (int i = 0; i < nout; ++i) key_put(k, &out[i], sizeof(qx_copy));
    for (int gi = 0; gi < ngroups; ++gi) {
        const qx_gemv_group &g = groups[gi];
        key_put(k, &g.count, sizeof(g.count));
        for (int i = 0; i < g.count; ++i) {
            key_put(k, &g.mats[i], sizeof(qx_packed));
            key_put(k, &g.x[i], sizeof(void *));
            key_put(k, &g.y[i], sizeof(void *));
        }
    }
    return k;
}

// Host memory the graph's copy nodes may take: pinned (page-locked) memory.
bool copyable(const qx_copy *c, int32_t n, bool host_src) {
    for (int i = 0; i < n; ++i) {
        cudaPointerAttributes at;
        if (cudaPointerGetAttributes(&at, host_src ? c[i].src : c[i].dst) != cudaSuccess) {
            cudaGetLastError();
            return false;
        }
        if (at.type != cudaMemoryTypeHost) return false;
    }
    return true;
}

qx_status run_step(const qx_copy *in, int32_t nin, const qx_gemv_group *groups, int32_t ngroups, int32_t batch,
                   int32_t y_dtype, int32_t flags, void *ws, const qx_copy *out, int32_t nout, int32_t sync,
                   cudaStream_t st, DeviceInfo *d) {
    int dev = -1;
    qx_status s = from_cuda(cudaGetDevice(&dev));
    if (s != QX_OK) return s;
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    bool direct = cudaStreamIsCapturing(st, &cs) != cudaSuccess || cs != cudaStreamCaptureStatusNone ||
                  dev < 0 || dev >= kMaxDevices;
    cudaGetLastError();
    cudaGraphExec_t exec = nullptr;
    if (!direct) {
        const std::vector<uint8_t> key = step_key(in, nin, groups, ngroups, batch, y_dtype, flags, ws, out, nout);
        std::lock_guard<std::mutex> lock(g_step_mu);
        for (int i = 0; i < kStepGraphs && exec == nullptr; ++i)
            if (g_steps[i].used && g_steps[i].dev == dev && g_steps[i].key == key) exec = g_steps[i].exec;
        if (exec == nullptr && copyable(in, nin, true) && copyable(out, nout, false)) {
            // capture on a stream of the library's own, then keep the instantiated graph
            if (g_capture[dev] == nullptr &&
                cudaStreamCreateWithFlags(&g_capture[dev], cudaStreamNonBlocking) != cudaSuccess) {
                cudaGetLastError();
                g_capture[dev] = nullptr;
            }
            cudaGraph_t graph = nullptr;
            if (g_capture[dev] != nullptr &&
                cudaStreamBeginCapture(g_capture[dev], cudaStreamCaptureModeThreadLocal) == cudaSuccess) {
                const qx_status si =
                    issue_step(in, nin, groups, ngroups, batch, y_dtype, flags, ws, out, nout, g_capture[dev], d);
                const cudaError_t ee = cudaStreamEndCapture(g_capture[dev], &graph);
                if (si == QX_OK && ee == cudaSuccess && graph != nullptr &&
                    cudaGraphInstantiate(&exec, graph, 0) != cudaSuccess)
                    exec = nullptr;
                if (graph != nullptr) cudaGraphDestroy(graph);
                if (si != QX_OK || ee != cudaSuccess) exec = nullptr;
            }
            cudaGetLastError();
            if (exec != nullptr) {
                StepGraph &e = g_steps[g_step_next];
                g_step_next = (g_step_next + 1) % kStepGraphs;
                if (e.used && e.exec != nullptr) {
                    cudaDeviceSynchronize();  // the evicted graph may still run
                    cudaGraphExecDestroy(e.exec);
                }
                e.used = true;
                e.dev = dev;
                e.key = key;
                e.exec = exec;
            }
        }
    }
    if (exec != nullptr) {
        if ((s = from_cuda(cudaGraphLaunch(exec, st))) != QX_OK) return s;
    } else if ((s = issue_step(in, nin, groups, ngroups, batch, y_dtype, flags, ws, out, nout, st, d)) != QX_OK) {
        return s;
    }
    return sync ? from_cuda(cudaStreamSynchronize(st)) : QX_OK;
}

}  // namespace

QX_API qx_status qx_decode_step(const qx_copy *in, int32_t nin, const qx_gemv_group *groups, int32_t ngroups,
                                int32_t batch, int32_t y_dtype, int32_t flags, const qx_copy *out, int32_t nout,
                                int32_t sync, void *stream) {
    qx_status s = check_copies(in, nin);
    if (s == QX_OK) s = check_copies(out, nout);
    if (s == QX_OK) s = check_chain(groups, ngroups, batch, y_dtype, flags);
    if (s != QX_OK) return s;
    DeviceInfo *d = nullptr;
    if ((s = device_info(&d)) != QX_OK) return s;
    return run_step(in, nin, groups, ngroups, batch, y_dtype, flags, nullptr, out, nout, sync,
                    static_cast<cudaStream_t>(stream), d);
}

namespace {

// Workspace of the fused calls: phase counters (one per group of a launch),
// then the flags (one per CTA) and the fp32 partial sums (16 rows of x by 32
// rows per CTA) of row blocks split between two CTAs.
constexpr size_t kFusedFlagOffset = 256;
constexpr size_t kFusedPartOffset = 2048;
constexpr size_t kFusedWorkspaceBytes = kFusedPartOffset + (size_t)qx::kMaxGemvCtas * 16 * 32 * sizeof(float);
static_assert(kFusedFlagOffset + qx::kMaxGemvCtas * sizeof(uint32_t) <= kFusedPartOffset, "workspace layout");

// The groups of a decode step in one persistent launch (qx::GemvMulti with one
// phase per group), its CTAs balanced stage by stage with the workspace.
// *launched is false, with nothing launched, when they cannot share one: more
// groups or matrices than a launch holds, different bits or kinds, or a plan
// that does not fit.
qx_status run_fused(const qx_gemv_group *groups, int ngroups, int batch, int y_dtype, int flags, void *ws,
                    cudaStream_t st, DeviceInfo *d, bool *launched) {
    *launched = false;
    if (ngroups > qx::kMaxGemvPhases) return QX_OK;
    const int esz = y_dtype == QX_F32 ? 4 : 2;
    qx::GemvMulti a{};
    a.bits = groups[0].mats[0].recipe.bits;
    a.kind = groups[0].mats[0].recipe.kind;
    a.batch = batch;
    a.y_f32 = y_dtype == QX_F32;
    a.status = d->status;
    a.wait_limit_ns = wait_limit_ns();
    a.nphase = ngroups;
    a.phase_ctr = static_cast<uint32_t *>(ws);
    a.split_flag = reinterpret_cast<uint32_t *>(static_cast<uint8_t *>(ws) + kFusedFlagOffset);
    a.split_part = reinterpret_cast<float *>(static_cast<uint8_t *>(ws) + kFusedPartOffset);
    int count = 0;
    for (int gi = 0; gi < ngroups; ++gi) {
        const qx_gemv_group &g = groups[gi];
        a.phase_first[gi] = count;
        for (int i = 0; i < g.count; ++i) {
            if (count == qx::kMaxGemvTotal) return QX_OK;
            if (g.mats[i].recipe.bits != a.bits || g.mats[i].recipe.kind != a.kind) return QX_OK;
            fill_mat(a.mat[count++], g.mats[i], g.x[i], g.y[i], 0, esz);
        }
    }
    a.count = count;
    a.phase_first[ngroups] = count;
    if (!plan_cached(a, d)) return QX_OK;
    const cudaError_t e = qx::launch_gemv_multi(a, st, (flags & QX_GEMV_PDL) != 0);
    if (e == cudaErrorCooperativeLaunchTooLarge) {  // not all CTAs resident at once: run them apart
        cudaGetLastError();
        return QX_OK;
    }
    *launched = true;
    return from_cuda(e);
}

qx_status check_fused_ws(const void *ws, size_t bytes) {
    if (ws == nullptr || bytes < kFusedWorkspaceBytes) return QX_ERR_INVALID_ARG;
    if (!aligned(ws, 256)) return QX_ERR_ALIGNMENT;
    return QX_OK;
}

// All groups in one launch (unless QX_GEMV_SEPARATE), else group by group, each
// launch balanced with the workspace; a group no balanced launch can take
// runs as qx_gemv_multi runs it.
qx_status run_chain_fused(const qx_gemv_group *groups, int32_t ngroups, int32_t batch, int32_t y_dtype,
                          int32_t flags, void *ws, cudaStream_t st, DeviceInfo *d) {
    const int lflags = flags & QX_GEMV_PDL;
    if (ngroups > 1 && !(flags & QX_GEMV_SEPARATE)) {
        bool launched = false;
        const qx_status s = run_fused(groups, ngroups, batch, y_dtype, lflags, ws, st, d, &launched);
        if (s != QX_OK || launched) return s;
    }
    for (int i = 0; i < ngroups; ++i) {
        bool launched = false;
        qx_status s = run_fused(groups + i, 1, batch, y_dtype, lflags, ws, st, d, &launched);
        if (s == QX_OK && !launched) s = run_chain(groups + i, 1, batch, y_dtype, lflags, st, d);
        if (s != QX_OK) return s;
    }
    return QX_OK;
}

}  // namespace

QX_API qx_status qx_gemv_fused_workspace(size_t *bytes) {
    if (bytes == nullptr) return QX_ERR_INVALID_ARG;
    *bytes = kFusedWorkspaceBytes;
    return QX_OK;
}

QX_API qx_status qx_gemv_fused(const qx_gemv_group *groups, int32_t ngroups, int32_t batch, int32_t y_dtype,
                               int32_t flags, void *workspace, size_t workspace_bytes, void *stream) {
    qx_status s = check_chain(groups, ngroups, batch, y_dtype, flags & ~QX_GEMV_SEPARATE);
    if (s == QX_OK) s = check_fused_ws(workspace, workspace_bytes);
    if (s != QX_OK) return s;
    DeviceInfo *d = nullptr;
    if ((s = device_info(&d)) != QX_OK) return s;
    return run_chain_fused(groups, ngroups, batch, y_dtype, flags, workspace, static_cast<cudaStream_t>(stream), d);
}

QX_API qx_status qx_decode_step_fused(const qx_copy *in, int32_t nin, const qx_gemv_group *groups, int32_t ngroups,
                                      int32_t batch, int32_t y_dtype, int32_t flags, void *workspace,
                                      size_t workspace_bytes, const qx_copy *out, int32_t nout, int32_t sync,
                                      void *stream) {
    qx_status s = check_copies(in, nin);
    if (s == QX_OK) s = check_copies(out, nout);
    if (s == QX_OK) s = check_chain(groups, ngroups, batch, y_dtype, flags & ~QX_GEMV_SEPARATE);
    if (s == QX_OK) s = check_fused_ws(workspace, workspace_bytes);
    if (s != QX_OK) return s;
    DeviceInfo *d = nullptr;
    if ((s = device_info(&d)) != QX_OK) return s;
    return run_step(in, nin, groups, ngroups, batch, y_dtype, flags, workspace, out, nout, sync,
                    static_cast<cudaStream_t>(stream), d);
}

namespace {

qx_status check_gemm_args(const qx_packed *p, const void *X, int64_t m, const void *Y) {
    qx_status s = check_packed(p);
    if (s != QX_OK) return s;
    if (X == nullptr || Y == nullptr || m < 1) return QX_ERR_INVALID_ARG;
    if (m > ((int64_t)1 << 31) - 1) return QX_ERR_UNSUPPORTED;
    if (!aligned(X, 16)) return QX_ERR_ALIGNMENT;
    if (!aligned(Y, 2)) return QX_ERR_ALIGNMENT;
    return QX_OK;
}

qx::GemmArgs gemm_args(const qx_packed *p, const void *X, int64_t m, void *Y, const DeviceInfo *d) {
    qx::GemmArgs a{};
    a.codes = static_cast<const uint8_t *>(p->codes);
    a.scales = static_cast<const __half *>(p->scales);
    a.zeros = static_cast<const uint8_t *>(p->zeros);
    a.luts = static_cast<const __half *>(p->luts);
    a.n = p->n;
    a.k = p->k;
    a.m = m;
    a.bits = p->recipe.bits;
    a.kind = p->recipe.kind;
    a.log2g = ilog2(p->recipe.group_size);
    a.G = (int)(p->k / p->recipe.group_size);
    a.zbytes = (a.G + 1) / 2;
    a.X = static_cast<const __half *>(X);
    a.Y = static_cast<__half *>(Y);
    a.status = d->status;
    a.wait_limit_ns = wait_limit_ns();
    return a;
}

}  // namespace

QX_API qx_status qx_gemm(const qx_packed *p, const void *X, int64_t m, void *Y, void *stream) {
    qx_status s = check_gemm_args(p, X, m, Y);
    if (s != QX_OK) return s;
    DeviceInfo *d = nullptr;
    if ((s = device_info(&d)) != QX_OK) return s;
    qx::GemmArgs a = gemm_args(p, X, m, Y, d);
    const qx::GemmPlan plan = qx::plan_gemm(p->n, p->k, m, d->num_sms, false);
    a.bn = plan.bn;
    a.splits = 1;
    return from_cuda(qx::launch_gemm(a, d->num_sms, static_cast<cudaStream_t>(stream)));
}

QX_API qx_status qx_gemm_splitk_workspace(int64_t n, int64_t k, int64_t m, const qx_recipe *recipe,
                                          size_t *bytes) {
    if (bytes == nullptr || recipe == nullptr || m < 1) return QX_ERR_INVALID_ARG;
    qx_status s = check_recipe(recipe);
    if (s != QX_OK) return s;
    if ((s = check_shape(n, k, recipe)) != QX_OK) return s;
    if (m > ((int64_t)1 << 31) - 1) return QX_ERR_UNSUPPORTED;
    DeviceInfo *d = nullptr;
    if ((s = device_info(&d)) != QX_OK) return s;
    *bytes = qx::plan_gemm(n, k, m, d->num_sms, true).ws_bytes;
    return QX_OK;
}

QX_API qx_status qx_gemm_splitk_plan(int64_t n, int64_t k, int64_t m, int32_t num_sms, int32_t *token_tile,
                                     int32_t *splits, size_t *bytes) {
    if (token_tile == nullptr || splits == nullptr || bytes == nullptr) return QX_ERR_INVALID_ARG;
    if (n < 1 || k < 1 || m < 1 || num_sms < 1) return QX_ERR_INVALID_ARG;
    if (k % 128 != 0 || n > (int64_t)1 << 22 || k > (int64_t)1 << 20 || m > ((int64_t)1 << 31) - 1)
        return QX_ERR_UNSUPPORTED;
    const qx::GemmPlan plan = qx::plan_gemm(n, k, m, num_sms, true);
    *token_tile = plan.bn;
    *splits = plan.splits;
    *bytes = plan.ws_bytes;
    return QX_OK;
}

QX_API qx_status qx_gemm_splitk(const qx_packed *p, const void *X, int64_t m, void *Y, void *workspace,
                                size_t workspace_bytes, int32_t flags, void *stream) {
    qx_status s = check_gemm_args(p, X, m, Y);
    if (s != QX_OK) return s;
    if ((flags & ~QX_GEMM_PDL) != 0) return QX_ERR_INVALID_ARG;
    DeviceInfo *d = nullptr;
    if ((s = device_info(&d)) != QX_OK) return s;
    const qx::GemmPlan plan = qx::plan_gemm(p->n, p->k, m, d->num_sms, true);
    qx::GemmArgs a = gemm_args(p, X, m, Y, d);
    a.bn = plan.bn;
    a.splits = plan.splits;
    a.pdl = (flags & QX_GEMM_PDL) ? 1 : 0;
    if (plan.splits > 1) {
        if (workspace == nullptr || workspace_bytes < plan.ws_bytes) return QX_ERR_INVALID_ARG;
        if (!aligned(workspace, 256)) return QX_ERR_ALIGNMENT;
        a.ws_cnt = static_cast<uint32_t *>(workspace);
        a.ws_part = reinterpret_cast<float *>(static_cast<uint8_t *>(workspace) + qx::kSplitCounterBytes);
    }
    return from_cuda(qx::launch_gemm(a, d->num_sms, static_cast<cudaStream_t>(stream)));
}

QX_API qx_status qx_gemm_splitk_noalloc(const qx_packed *p, const void *X, int64_t m, void *Y, void *stream) {
    qx_status s = check_gemm_args(p, X, m, Y);
    if (s != QX_OK) return s;
    DeviceInfo *d = nullptr;
    if ((s = device_info(&d)) != QX_OK) return s;
    const qx::GemmPlan plan = qx::plan_gemm(p->n, p->k, m, d->num_sms, true);
    if (plan.ws_bytes > qx::kNoAllocScratchBytes) return QX_ERR_UNSUPPORTED;
    qx::GemmArgs a = gemm_args(p, X, m, Y, d);
    a.bn = plan.bn;
    a.splits = plan.splits;
    if (plan.splits > 1) {
        void *ws = nullptr;
        cudaError_t e = qx::noalloc_scratch(&ws);
        if (e != cudaSuccess) return from_cuda(e);
        // re-arm this call's counters on the stream (they are zero unless an
        // earlier call gave up on a wait); a memset, not an allocation
        e = cudaMemsetAsync(ws, 0, (size_t)plan.tiles * 4 * sizeof(uint32_t), static_cast<cudaStream_t>(stream));
        if (e != cudaSuccess) return from_cuda(e);
        a.ws_cnt = static_cast<uint32_t *>(ws);
        a.ws_part = reinterpret_cast<float *>(static_cast<uint8_t *>(ws) + qx::kSplitCounterBytes);
    }
    return from_cuda(qx::launch_gemm(a, d->num_sms, static_cast<cudaStream_t>(stream)));
}

QX_API qx_status qx_quantize_act(const void *x, int32_t batch, int64_t k, void *q, void *scales, void *stream) {
    if (x == nullptr || q == nullptr || scales == nullptr) return QX_ERR_INVALID_ARG;
    if (batch < 1 || k < 1) return QX_ERR_INVALID_ARG;
    if (batch > kMaxActRows || k % 16 != 0 || k > ((int64_t)1 << 20)) return QX_ERR_UNSUPPORTED;
    if (!aligned(x, 2) || !aligned(q, 16) || !aligned(scales, 4)) return QX_ERR_ALIGNMENT;
    DeviceInfo *d = nullptr;
    qx_status s = device_info(&d);
    if (s != QX_OK) return s;
    return from_cuda(qx::launch_quantize_act(static_cast<const __half *>(x), batch, k, static_cast<int8_t *>(q),
                                             static_cast<float *>(scales), static_cast<cudaStream_t>(stream)));
}

QX_API qx_status qx_dequant_act(const void *q, const void *scales, int64_t m, int64_t k, void *x_hat, void *stream) {
    if (q == nullptr || scales == nullptr || x_hat == nullptr) return QX_ERR_INVALID_ARG;
    if (m < 1 || k < 1) return QX_ERR_INVALID_ARG;
    if (m > kMaxActRows || k % 16 != 0 || k > ((int64_t)1 << 20)) return QX_ERR_UNSUPPORTED;
    if (!aligned(q, 16) || !aligned(scales, 4) || !aligned(x_hat, 16)) return QX_ERR_ALIGNMENT;
    DeviceInfo *d = nullptr;
    const qx_status s = device_info(&d);
    if (s != QX_OK) return s;
    return from_cuda(qx::launch_dequant_act(static_cast<const int8_t *>(q), static_cast<const float *>(scales), m, k,
                                            static_cast<__half *>(x_hat), d->num_sms,
                                            static_cast<cudaStream_t>(stream)));
}

QX_API qx_status qx_gemv_a8(const qx_packed *p, const void *q, const void *scales, int32_t batch, void *y,
                            int32_t y_dtype, void *stream) {
    qx_status s = check_packed(p);
    if (s != QX_OK) return s;
    if (q == nullptr || scales == nullptr || y == nullptr) return QX_ERR_INVALID_ARG;
    if (batch < 1 || batch > 16 || (y_dtype != QX_F16 && y_dtype != QX_F32)) return QX_ERR_INVALID_ARG;
    if (p->recipe.kind != QX_UNIFORM) return QX_ERR_UNSUPPORTED;
    if (!aligned(q, 16) || !aligned(scales, 4) || !aligned(y, 4)) return QX_ERR_ALIGNMENT;
    DeviceInfo *d = nullptr;
    if ((s = device_info(&d)) != QX_OK) return s;
    qx::GemvA8Args a{};
    a.codes = static_cast<const uint8_t *>(p->codes);
    a.scales = static_cast<const __half *>(p->scales);
    a.zeros = static_cast<const uint8_t *>(p->zeros);
    a.n = p->n;
    a.k = p->k;
    a.bits = p->recipe.bits;
    a.log2g = ilog2(p->recipe.group_size);
    a.G = (int)(p->k / p->recipe.group_size);
    a.zbytes = (a.G + 1) / 2;
    a.q = static_cast<const int8_t *>(q);
    a.act_scales = static_cast<const float *>(scales);
    a.batch = batch;
    a.y = y;
    a.y_f32 = y_dtype == QX_F32;
    return from_cuda(qx::launch_gemv_a8(a, static_cast<cudaStream_t>(stream)));
}

namespace {

// Workspace of qx_select_recipe: the largest candidate's packed buffers, the
// dequantized matrix, the error partials, one 16-byte result per candidate
// and, when a Q4X candidate is present, the Q4X learner's workspace.
struct SelectLayout {
    size_t packed, what, partials, results, q4x, total;
};

size_t round256(size_t x) { return (x + 255) / 256 * 256; }

// Byte sizes of one candidate's four buffers: {codes, scales, zeros, luts}
// for the per-group kinds, {codes, scales, books, codebooks} for Q4X.
qx_status candidate_sizes(int64_t n, int64_t k, const qx_recipe *r, uint64_t out[4]) {
    if (r == nullptr) return QX_ERR_INVALID_ARG;
    if (r->kind == QX_Q4X) {
        if (r->lloyd_iters < 0 || r->lloyd_iters > 1000) return QX_ERR_INVALID_ARG;
        if (r->bits != 4 || r->group_size != qx::kQ4xGroup) return QX_ERR_UNSUPPORTED;
        qx_q4x_sizes sz{};
        const qx_status s = qx_q4x_size(n, k, &sz);
        if (s != QX_OK) return s;
        out[0] = sz.codes, out[1] = sz.scales, out[2] = sz.books, out[3] = sz.codebooks;
        return QX_OK;
    }
    qx_sizes sz{};
    const qx_status s = qx_packed_size(n, k, r, &sz);
    if (s != QX_OK) return s;
    out[0] = sz.codes, out[1] = sz.scales, out[2] = sz.zeros, out[3] = sz.luts;
    return QX_OK;
}

qx_status select_layout(int64_t n, int64_t k, const qx_recipe *cands, int32_t count, int num_sms, SelectLayout *L) {
    if (cands == nullptr || count < 1 || count > 16) return QX_ERR_INVALID_ARG;
    size_t packed = 0;
    bool q4x = false;
    for (int i = 0; i < count; ++i) {
        uint64_t sz[4] = {};
        qx_status s = candidate_sizes(n, k, &cands[i], sz);
        if (s != QX_OK) return s;
        packed = std::max(packed, round256(sz[0]) + round256(sz[1]) + round256(sz[2]) + round256(sz[3]));
        q4x = q4x || cands[i].kind == QX_Q4X;
    }
    L->packed = packed;
    L->what = round256((size_t)n * k * 2);
    L->partials = round256((size_t)qx::sq_error_blocks(num_sms) * 16);
    L->results = round256((size_t)count * 16);
    L->q4x = q4x ? round256(qx::q4x_workspace_bytes(n, k)) : 0;
    L->total = L->packed + L->what + L->partials + L->results + L->q4x;
    return QX_OK;
}

}  // namespace

QX_API qx_status qx_select_workspace(int64_t n, int64_t k, const qx_recipe *candidates, int32_t count,
                                     size_t *bytes) {
    if (bytes == nullptr) return QX_ERR_INVALID_ARG;
    DeviceInfo *d = nullptr;
    SelectLayout L{};
    qx_status s = select_layout(n, k, candidates, count, 1, &L);  // validates first
    if (s != QX_OK) return s;
    if ((s = device_info(&d)) != QX_OK) return s;
    if ((s = select_layout(n, k, candidates, count, d->num_sms, &L)) != QX_OK) return s;
    *bytes = L.total;
    return QX_OK;
}

QX_API qx_status qx_select_recipe(const void *W, int64_t n, int64_t k, const qx_recipe *candidates, int32_t count,
                                  double max_bpw, void *workspace, size_t workspace_bytes, int32_t *chosen,
                                  uint64_t *sq_error, double *bpw, void *stream) {
    if (W == nullptr || chosen == nullptr || sq_error == nullptr || bpw == nullptr) return QX_ERR_INVALID_ARG;
    SelectLayout L{};
    qx_status s = select_layout(n, k, candidates, count, 1, &L);
    if (s != QX_OK) return s;
    if (!aligned(W, 16)) return QX_ERR_ALIGNMENT;
    DeviceInfo *d = nullptr;
    if ((s = device_info(&d)) != QX_OK) return s;
    if ((s = select_layout(n, k, candidates, count, d->num_sms, &L)) != QX_OK) return s;
    if (workspace == nullptr || workspace_bytes < L.total) return QX_ERR_INVALID_ARG;
    if (!aligned(workspace, 256)) return QX_ERR_ALIGNMENT;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    void *what = ws + L.packed;
    auto *partials = reinterpret_cast<unsigned long long *>(ws + L.packed + L.what);
    auto *results = reinterpret_cast<unsigned long long *>(ws + L.packed + L.what + L.partials);
    uint8_t *q4x_ws = ws + L.packed + L.what + L.partials + L.results;
    bool eligible[16] = {};
    for (int i = 0; i < count; ++i) {
        uint64_t sz[4] = {};
        candidate_sizes(n, k, &candidates[i], sz);
        bpw[i] = 8.0 * (double)(sz[0] + sz[1] + sz[2] + sz[3]) / ((double)n * (double)k);
        eligible[i] = !(max_bpw > 0.0) || bpw[i] <= max_bpw;
        if (!eligible[i]) continue;
        // quantize into the workspace, dequantize, take the exact error
        void *buf[4] = {};
        uint8_t *at = ws;
        for (int j = 0; j < 4; ++j) {
            buf[j] = sz[j] ? at : nullptr;
            at += round256(sz[j]);
        }
        if (candidates[i].kind == QX_Q4X) {
            const qx_q4x p{n, k, buf[0], buf[1], buf[2], buf[3]};
            if ((s = qx_q4x_quantize(W, candidates[i].lloyd_iters, &p, q4x_ws, L.q4x, stream)) != QX_OK) return s;
            if ((s = qx_q4x_dequant(&p, what, stream)) != QX_OK) return s;
        } else {
            qx_packed p{};
            p.n = n;
            p.k = k;
            p.recipe = candidates[i];
            p.codes = buf[0];
            p.scales = buf[1];
            p.zeros = buf[2];
            p.luts = buf[3];
            if ((s = qx_quantize(W, n, k, &candidates[i], &p, stream)) != QX_OK) return s;
            if ((s = qx_dequant(&p, what, stream)) != QX_OK) return s;
        }
        if ((s = from_cuda(qx::launch_sq_error(static_cast<const __half *>(W), static_cast<const __half *>(what),
                                               n * k, partials, results + 2 * i, d->num_sms, st))) != QX_OK)
            return s;
    }
    unsigned long long host[32] = {};
    if ((s = from_cuda(cudaMemcpyAsync(host, results, (size_t)count * 16, cudaMemcpyDeviceToHost, st))) != QX_OK)
        return s;
    if ((s = from_cuda(cudaStreamSynchronize(st))) != QX_OK) return s;
    uint32_t status = 0;
    if ((s = from_cuda(cudaMemcpy(&status, d->status, sizeof(status), cudaMemcpyDeviceToHost))) != QX_OK) return s;
    if (status & qx::kStatusNonfinite) return QX_ERR_NONFINITE;
    // the smallest error, ties to fewer bits per weight, then to the earlier candidate
    *chosen = -1;
    unsigned __int128 best = 0;
    for (int i = 0; i < count; ++i) {
        if (!eligible[i]) {
            sq_error[2 * i] = sq_error[2 * i + 1] = ~0ull;
            continue;
        }
        sq_error[2 * i] = host[2 * i];
        sq_error[2 * i + 1] = host[2 * i + 1];
        const unsigned __int128 e = ((unsigned __int128)host[2 * i + 1] << 64) | host[2 * i];
        if (*chosen < 0 || e < best || (e == best && bpw[i] < bpw[*chosen])) {
            *chosen = i;
            best = e;
        }
    }
    return QX_OK;
}

namespace {

qx_status check_q4x_shape(int64_t n, int64_t k) {
    if (n < 1 || k < 1) return QX_ERR_INVALID_ARG;
    if (k % qx::kQ4xGroup != 0) return QX_ERR_UNSUPPORTED;
    // value-histogram counts are 32-bit, group indices below 2^32
    if (n > ((int64_t)1 << 31) / k) return QX_ERR_UNSUPPORTED;
    return QX_OK;
}

qx_status check_q4x(const qx_q4x *p) {
    if (p == nullptr) return QX_ERR_INVALID_ARG;
    const qx_status s = check_q4x_shape(p->n, p->k);
    if (s != QX_OK) return s;
    if (p->codes == nullptr || p->scales == nullptr || p->books == nullptr || p->codebooks == nullptr)
        return QX_ERR_INVALID_ARG;
    if (!aligned(p->codes, 16) || !aligned(p->scales, 2) || !aligned(p->codebooks, 2)) return QX_ERR_ALIGNMENT;
    return QX_OK;
}

qx::Q4xMat q4x_mat(const qx_q4x *p) {
    qx::Q4xMat m{};
    m.codes = static_cast<const uint8_t *>(p->codes);
    m.scales = static_cast<const __half *>(p->scales);
    m.books = static_cast<const uint8_t *>(p->books);
    m.codebooks = static_cast<const __half *>(p->codebooks);
    m.n = p->n;
    m.k = p->k;
    m.G = (int)(p->k / qx::kQ4xGroup);
    m.bbytes = (m.G + 3) / 4;
    return m;
}

}  // namespace

QX_API qx_status qx_q4x_size(int64_t n, int64_t k, qx_q4x_sizes *out) {
    if (out == nullptr) return QX_ERR_INVALID_ARG;
    const qx_status s = check_q4x_shape(n, k);
    if (s != QX_OK) return s;
    const int64_t G = k / qx::kQ4xGroup;
    out->codes = (uint64_t)(n * k / 2);
    out->scales = (uint64_t)(n * G * 2);
    out->books = (uint64_t)(n * ((G + 3) / 4));
    out->codebooks = 4 * 16 * 2;
    return QX_OK;
}

QX_API qx_status qx_q4x_workspace(int64_t n, int64_t k, size_t *bytes) {
    if (bytes == nullptr) return QX_ERR_INVALID_ARG;
    const qx_status s = check_q4x_shape(n, k);
    if (s != QX_OK) return s;
    *bytes = qx::q4x_workspace_bytes(n, k);
    return QX_OK;
}

QX_API qx_status qx_q4x_quantize(const void *W, int32_t iters, const qx_q4x *out, void *workspace,
                                 size_t workspace_bytes, void *stream) {
    if (W == nullptr) return QX_ERR_INVALID_ARG;
    qx_status s = check_q4x(out);
    if (s != QX_OK) return s;
    if (iters < 0 || iters > 1000) return QX_ERR_INVALID_ARG;
    if (workspace == nullptr || workspace_bytes < qx::q4x_workspace_bytes(out->n, out->k)) return QX_ERR_INVALID_ARG;
    if (!aligned(W, 16) || !aligned(workspace, 256)) return QX_ERR_ALIGNMENT;
    DeviceInfo *d = nullptr;
    if ((s = device_info(&d)) != QX_OK) return s;
    qx::Q4xQuantArgs a{};
    a.W = static_cast<const __half *>(W);
    a.n = out->n;
    a.k = out->k;
    a.G = (int)(out->k / qx::kQ4xGroup);
    a.bbytes = (a.G + 3) / 4;
    a.iters = iters;
    a.codes = static_cast<uint8_t *>(out->codes);
    a.scales = static_cast<__half *>(out->scales);
    a.books = static_cast<uint8_t *>(out->books);
    a.codebooks = static_cast<__half *>(out->codebooks);
    a.ws = workspace;
    a.status = d->status;
    return from_cuda(qx::launch_q4x_quantize(a, d->num_sms, static_cast<cudaStream_t>(stream)));
}

QX_API qx_status qx_q4x_dequant(const qx_q4x *p, void *W_out, void *stream) {
    qx_status s = check_q4x(p);
    if (s != QX_OK) return s;
    if (W_out == nullptr) return QX_ERR_INVALID_ARG;
    if (!aligned(W_out, 16)) return QX_ERR_ALIGNMENT;
    DeviceInfo *d = nullptr;
    if ((s = device_info(&d)) != QX_OK) return s;
    return from_cuda(qx::launch_q4x_dequant(q4x_mat(p), static_cast<__half *>(W_out), d->num_sms,
                                            static_cast<cudaStream_t>(stream)));
}

namespace {

// Q4X decode on the register-dequant kernel (csrc/qx_gemv.cu, kind 2: the
// books in `zeros`, the codebooks in `luts`), which works in 128-weight
// superblocks.  A matrix's results do not depend on the launch it is in.
bool q4x_ring_fits(const qx::Q4xMat &m) { return m.k % 128 == 0 && m.k <= 32768; }

// *launched stays false, with nothing launched, when the plan does not fit.
qx_status run_q4x_ring(const qx::Q4xGemvMulti &q, cudaStream_t st, DeviceInfo *d, bool *launched) {
    *launched = false;
    qx::GemvMulti a{};
    a.bits = 4;
    a.kind = 2;
    a.batch = q.batch;
    a.y_f32 = q.y_f32;
    a.status = d->status;
    a.wait_limit_ns = wait_limit_ns();
    a.nphase = 1;
    a.count = q.count;
    a.phase_first[0] = 0;
    a.phase_first[1] = q.count;
    for (int i = 0; i < q.count; ++i) {
        const qx::Q4xMat &m = q.mat[i];
        if (!q4x_ring_fits(m)) return QX_OK;
        qx::GemvMat &M = a.mat[i];
        M.codes = m.codes;
        M.scales = m.scales;
        M.zeros = m.books;
        M.luts = m.codebooks;
        M.x = q.x[i];
        M.y = q.y[i];
        M.n = m.n;
        M.k = m.k;
        M.G = m.G;
        M.zbytes = m.bbytes;
        M.log2g = 6;
    }
    if (!plan_cached(a, d)) return QX_OK;
    *launched = true;
    return from_cuda(qx::launch_gemv_multi(a, st, false));
}

}  // namespace

QX_API qx_status qx_q4x_gemv_multi(const qx_q4x *mats, int32_t count, const void *const *x, int32_t batch,
                                   void *const *y, int32_t y_dtype, void *stream) {
    if (mats == nullptr || x == nullptr || y == nullptr) return QX_ERR_INVALID_ARG;
    if (count < 1 || count > qx::kMaxQ4xMats) return QX_ERR_INVALID_ARG;
    if (y_dtype != QX_F16 && y_dtype != QX_F32) return QX_ERR_INVALID_ARG;
    if (batch < 1) return QX_ERR_INVALID_ARG;
    if (batch > 16) return QX_ERR_UNSUPPORTED;
    qx::Q4xGemvMulti a{};
    a.count = count;
    a.batch = batch;
    a.y_f32 = y_dtype == QX_F32;
    a.row_off[0] = 0;
    for (int i = 0; i < count; ++i) {
        qx_status s = check_q4x(&mats[i]);
        if (s != QX_OK) return s;
        if (x[i] == nullptr || y[i] == nullptr) return QX_ERR_INVALID_ARG;
        if (!aligned(x[i], 16) || !aligned(y[i], 4)) return QX_ERR_ALIGNMENT;
        a.mat[i] = q4x_mat(&mats[i]);
        a.x[i] = static_cast<const __half *>(x[i]);
        a.y[i] = y[i];
        a.row_off[i + 1] = a.row_off[i] + mats[i].n;
    }
    DeviceInfo *d = nullptr;
    qx_status s = device_info(&d);
    if (s != QX_OK) return s;
    // the matrices the register-dequant kernel takes in one launch, the rest
    // (k not a multiple of 128) in one launch of the row-per-warp kernel
    const cudaStream_t st = static_cast<cudaStream_t>(stream);
    qx::Q4xGemvMulti part[2]{};
    for (int j = 0; j < 2; ++j) {
        part[j].batch = batch;
        part[j].y_f32 = a.y_f32;
    }
    for (int i = 0; i < count; ++i) {
        qx::Q4xGemvMulti &p = part[q4x_ring_fits(a.mat[i]) ? 0 : 1];
        p.mat[p.count] = a.mat[i];
        p.x[p.count] = a.x[i];
        p.y[p.count] = a.y[i];
        p.row_off[p.count + 1] = p.row_off[p.count] + a.mat[i].n;
        ++p.count;
    }
    if (part[0].count > 0) {
        bool launched = false;
        s = run_q4x_ring(part[0], st, d, &launched);
        if (s != QX_OK) return s;
        if (!launched) s = from_cuda(qx::launch_q4x_gemv(part[0], d->num_sms, st));
        if (s != QX_OK) return s;
    }
    if (part[1].count > 0) s = from_cuda(qx::launch_q4x_gemv(part[1], d->num_sms, st));
    return s;
}

QX_API qx_status qx_q4x_gemv(const qx_q4x *p, const void *x, int32_t batch, void *y, int32_t y_dtype, void *stream) {
    if (p == nullptr) return QX_ERR_INVALID_ARG;
    return qx_q4x_gemv_multi(p, 1, &x, batch, &y, y_dtype, stream);
}

namespace {

qx_status check_q4x_gemm(const qx_q4x *p, const void *X, int64_t m, const void *Y) {
    qx_status s = check_q4x(p);
    if (s != QX_OK) return s;
    if (p->k % 128 != 0) return QX_ERR_UNSUPPORTED;  // the matmul works in 128-weight superblocks
    if (p->n > (int64_t)1 << 22 || p->k > (int64_t)1 << 20) return QX_ERR_UNSUPPORTED;
    if (X == nullptr || Y == nullptr || m < 1) return QX_ERR_INVALID_ARG;
    if (m > ((int64_t)1 << 31) - 1) return QX_ERR_UNSUPPORTED;
    if (!aligned(X, 16)) return QX_ERR_ALIGNMENT;
    if (!aligned(Y, 2)) return QX_ERR_ALIGNMENT;
    return QX_OK;
}

// The tensor-core matmul's arguments for Q4X weights: kind 2, the book bytes
// in `zeros`, the codebooks in `luts`.
qx::GemmArgs q4x_gemm_args(const qx_q4x *p, const void *X, int64_t m, void *Y, const DeviceInfo *d) {
    const qx::Q4xMat q = q4x_mat(p);
    qx::GemmArgs a{};
    a.codes = q.codes;
    a.scales = q.scales;
    a.zeros = q.books;
    a.luts = q.codebooks;
    a.n = p->n;
    a.k = p->k;
    a.m = m;
    a.bits = 4;
    a.kind = 2;
    a.log2g = 6;
    a.G = q.G;
    a.zbytes = q.bbytes;
    a.X = static_cast<const __half *>(X);
    a.Y = static_cast<__half *>(Y);
    a.status = d->status;
    a.wait_limit_ns = wait_limit_ns();
    return a;
}

}  // namespace

QX_API qx_status qx_q4x_gemm(const qx_q4x *p, const void *X, int64_t m, void *Y, void *stream) {
    qx_status s = check_q4x_gemm(p, X, m, Y);
    if (s != QX_OK) return s;
    DeviceInfo *d = nullptr;
    if ((s = device_info(&d)) != QX_OK) return s;
    qx::GemmArgs a = q4x_gemm_args(p, X, m, Y, d);
    const qx::GemmPlan plan = qx::plan_gemm(p->n, p->k, m, d->num_sms, false);
    a.bn = plan.bn;
    a.splits = 1;
    return from_cuda(qx::launch_gemm(a, d->num_sms, static_cast<cudaStream_t>(stream)));
}

QX_API qx_status qx_q4x_gemm_splitk_workspace(int64_t n, int64_t k, int64_t m, size_t *bytes) {
    if (bytes == nullptr || n < 1 || k < 1 || m < 1) return QX_ERR_INVALID_ARG;
    if (k % 128 != 0 || n > (int64_t)1 << 22 || k > (int64_t)1 << 20) return QX_ERR_UNSUPPORTED;
    DeviceInfo *d = nullptr;
    const qx_status s = device_info(&d);
    if (s != QX_OK) return s;
    *bytes = qx::plan_gemm(n, k, m, d->num_sms, true).ws_bytes;
    return QX_OK;
}

QX_API qx_status qx_q4x_gemm_splitk(const qx_q4x *p, const void *X, int64_t m, void *Y, void *workspace,
                                    size_t workspace_bytes, int32_t flags, void *stream) {
    qx_status s = check_q4x_gemm(p, X, m, Y);
    if (s != QX_OK) return s;
    if ((flags & ~QX_GEMM_PDL) != 0) return QX_ERR_INVALID_ARG;
    DeviceInfo *d = nullptr;
    if ((s = device_info(&d)) != QX_OK) return s;
    const qx::GemmPlan plan = qx::plan_gemm(p->n, p->k, m, d->num_sms, true);
    qx::GemmArgs a = q4x_gemm_args(p, X, m, Y, d);
    a.bn = plan.bn;
    a.splits = plan.splits;
    a.pdl = (flags & QX_GEMM_PDL) ? 1 : 0;
    if (plan.splits > 1) {
        if (workspace == nullptr || workspace_bytes < plan.ws_bytes) return QX_ERR_INVALID_ARG;
        if (!aligned(workspace, 256)) return QX_ERR_ALIGNMENT;
        a.ws_cnt = static_cast<uint32_t *>(workspace);
        a.ws_part = reinterpret_cast<float *>(static_cast<uint8_t *>(workspace) + qx::kSplitCounterBytes);
    }
    return from_cuda(qx::launch_gemm(a, d->num_sms, static_cast<cudaStream_t>(stream)));
}

QX_API qx_status qx_selftest_wait_timeout(int32_t limit_us, void *stream) {
    if (limit_us < 1 || limit_us > 1000000) return QX_ERR_INVALID_ARG;
    DeviceInfo *d = nullptr;
    const qx_status s = device_info(&d);
    if (s != QX_OK) return s;
    return from_cuda(qx::launch_wait_selftest((uint64_t)limit_us * 1000ull, d->status,
                                              static_cast<cudaStream_t>(stream)));
}

QX_API qx_status qx_get_device_status(void *stream) {
    DeviceInfo *d = nullptr;
    qx_status s = device_info(&d);
    if (s != QX_OK) return s;
    if ((s = from_cuda(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)))) != QX_OK) return s;
    uint32_t v = 0;
    if ((s = from_cuda(cudaMemcpy(&v, d->status, sizeof(v), cudaMemcpyDeviceToHost))) != QX_OK) return s;
    const uint32_t zero = 0;
    if ((s = from_cuda(cudaMemcpy(d->status, &zero, sizeof(zero), cudaMemcpyHostToDevice))) != QX_OK) return s;
    if (v & qx::kStatusNonfinite) return QX_ERR_NONFINITE;
    if (v & qx::kStatusTimeout) return QX_ERR_TIMEOUT;
    return QX_OK;
}
