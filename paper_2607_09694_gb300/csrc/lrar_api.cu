// lrar_api.cu -- the exported C ABI of liblrar.so (declared in include/lrar.h):
// argument checks, error reporting, and dispatch to the kernel launchers.
// Nothing here allocates device memory or synchronises the host.
#include <math.h>
#include <stdarg.h>
#include <stdio.h>

#include <mutex>
#include <unordered_map>

#include "lrar.h"
#include "lrar_testing.h"
#include "lrar_device.cuh"
#include "lrar_launch.h"

#define LRAR_API extern "C" __attribute__((visibility("default")))

namespace {

thread_local char g_last_error[512] = "";

int fail(int code, const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_last_error, sizeof g_last_error, fmt, ap);
    va_end(ap);
    return code;
}

int cuda_fail(cudaError_t e, const char *where) {
    return fail(LRAR_ERR_CUDA, "%s: %s (%s)", where, cudaGetErrorString(e), cudaGetErrorName(e));
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }
bool aligned4(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 3) == 0; }
bool dtype_ok(int t) { return t == LRAR_F32 || t == LRAR_BF16; }
int esize(int t) { return t == LRAR_BF16 ? 2 : 4; }

// Scalar checks shared by forward and backward.
int check_shape(int variant, int in_dtype, int n_src, int64_t T, int d, int r, float eps) {
    if (variant < LRAR_FULL || variant > LRAR_PROJECTED) return fail(LRAR_ERR_INVALID_ARG, "unknown variant %d", variant);
    if (!dtype_ok(in_dtype)) return fail(LRAR_ERR_INVALID_ARG, "unknown input dtype %d", in_dtype);
    if (n_src < 1) return fail(LRAR_ERR_INVALID_ARG, "n_src must be >= 1 (got %d)", n_src);
    if (n_src > LRAR_MAX_SOURCES)
        return fail(LRAR_ERR_UNSUPPORTED, "n_src %d exceeds LRAR_MAX_SOURCES (%d)", n_src, LRAR_MAX_SOURCES);
    if (T < 0) return fail(LRAR_ERR_INVALID_ARG, "T must be >= 0");
    if (d < 1 || r < 1 || r > d) return fail(LRAR_ERR_INVALID_ARG, "need 1 <= r <= d (got d=%d r=%d)", d, r);
    if (variant == LRAR_FULL && r != d)
        return fail(LRAR_ERR_INVALID_ARG, "full AttnRes keys need r == d (got d=%d r=%d)", d, r);
    if (!(eps > 0.f) || !isfinite(eps)) return fail(LRAR_ERR_INVALID_ARG, "eps must be finite and > 0");
    if ((d * esize(in_dtype)) % 16) return fail(LRAR_ERR_ALIGNMENT, "d * element size must be a multiple of 16 bytes");
    if (d > lrar::max_width(in_dtype))
        return fail(LRAR_ERR_UNSUPPORTED, "d=%d exceeds the kernel width limit %d", d, lrar::max_width(in_dtype));
    return LRAR_OK;
}

struct OccKey {
    const void *k;
    int dev, threads;
    size_t smem;
    bool operator==(const OccKey &o) const {
        return k == o.k && dev == o.dev && threads == o.threads && smem == o.smem;
    }
};
struct OccHash {
    size_t operator()(const OccKey &o) const {
        return std::hash<const void *>()(o.k) ^ (std::hash<size_t>()(o.smem) * 31) ^ (size_t)o.dev * 131 ^
               (size_t)o.threads;
    }
};
std::mutex g_occ_mu;
std::unordered_map<OccKey, int, OccHash> g_occ;  // (kernel, device, block, smem) -> resident CTAs per SM x SMs

}  // namespace

namespace lrar {

int record_error(int code, const char *message) { return fail(code, "%s", message); }

int max_width(int in_dtype) { return 32 * 8 * VecE<float>::value * (in_dtype == LRAR_BF16 ? 2 : 1); }

int persistent_grid(const void *kernel, int threads, size_t smem, int64_t work_ctas, int cap) {
    int dev = 0;
    cudaGetDevice(&dev);
    OccKey key{kernel, dev, threads, smem};
    int slots = 0;
    {
        std::lock_guard<std::mutex> lk(g_occ_mu);
        auto it = g_occ.find(key);
        if (it != g_occ.end()) slots = it->second;
    }
    if (slots == 0) {
        int sms = 0, occ = 0;
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, kernel, threads, smem);
        slots = (sms > 0 ? sms : 1) * (occ > 0 ? occ : 1);
        std::lock_guard<std::mutex> lk(g_occ_mu);
        g_occ[key] = slots;
    }
    int64_t g = slots;
    if (g > work_ctas) g = work_ctas;
    if (g > cap) g = cap;
    if (g < 1) g = 1;
    return (int)g;
}

}  // namespace lrar

LRAR_API int lrar_version(void) { return LRAR_VERSION; }

LRAR_API const char *lrar_last_error(void) { return g_last_error; }

LRAR_API const char *lrar_strerror(int code) {
    switch (code) {
        case LRAR_OK: return "success";
        case LRAR_ERR_INVALID_ARG: return "invalid argument";
        case LRAR_ERR_ALIGNMENT: return "misaligned pointer or row size";
        case LRAR_ERR_UNSUPPORTED: return "unsupported size";
        case LRAR_ERR_CUDA: return "CUDA error";
        case LRAR_ERR_WORKSPACE: return "workspace missing or too small";
        default: return "unknown status code";
    }
}

namespace {

// Source tables of a stacked [n, T, width] buffer: entry i = base + i * T * width.
void stack_table(const void *base, int n, int64_t T, int width, int esz, const void **tab) {
    for (int i = 0; i < n; ++i)
        tab[i] = base ? static_cast<const char *>(base) + (size_t)i * (size_t)T * (size_t)width * (size_t)esz
                      : nullptr;
}

// Every entry of a caller's source table present and 16-byte aligned.
int check_table(const void *const *tab, int n, const char *what) {
    if (!tab) return fail(LRAR_ERR_INVALID_ARG, "%s table is required", what);
    for (int i = 0; i < n; ++i) {
        if (!tab[i]) return fail(LRAR_ERR_INVALID_ARG, "%s[%d] is NULL", what, i);
        if (!aligned16(tab[i])) return fail(LRAR_ERR_ALIGNMENT, "%s[%d] must be 16-byte aligned", what, i);
    }
    return LRAR_OK;
}

int forward_impl(int variant, int in_dtype, int out_dtype, const void *const *values, const void *const *keys,
                 const float *query, int n_src, int64_t T, int d, int r, float eps, void *h, float *lse,
                 void *stream) {
    if (!h) return fail(LRAR_ERR_INVALID_ARG, "h is required");
    if (!query && n_src > 1) return fail(LRAR_ERR_INVALID_ARG, "query is required when n_src > 1");
    if (!aligned16(h) || (query && !aligned4(query)) || (lse && !aligned4(lse)))
        return fail(LRAR_ERR_ALIGNMENT, "tensors must be 16-byte aligned (query and lse 4-byte)");
    lrar::FwdArgs a;
    a.variant = variant;
    a.in_dtype = in_dtype;
    a.out_dtype = out_dtype;
    a.values = values;
    a.keys = variant == LRAR_PROJECTED ? keys : nullptr;
    a.query = query;
    a.n = n_src;
    a.T = T;
    a.d = d;
    a.r = r;
    a.eps = eps;
    a.h = h;
    a.lse = lse;
    cudaError_t e = lrar::launch_forward(a, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "lrar_forward");
    return LRAR_OK;
}

// Scalar checks of the backward (every form of it).
int backward_scalars(int variant, int in_dtype, int grad_dtype, int n_src, int64_t T, int d, int r, float eps,
                     int h_dtype, float *dq, int accumulate) {
    int rc = check_shape(variant, in_dtype, n_src, T, d, r, eps);
    if (rc) return rc;
    if (!dtype_ok(grad_dtype)) return fail(LRAR_ERR_INVALID_ARG, "unknown gradient dtype %d", grad_dtype);
    if (accumulate != 0 && accumulate != 1) return fail(LRAR_ERR_INVALID_ARG, "accumulate must be 0 or 1");
    if (variant == LRAR_FULL && !dtype_ok(h_dtype)) return fail(LRAR_ERR_INVALID_ARG, "unknown h dtype %d", h_dtype);
    if (!dq) return fail(LRAR_ERR_INVALID_ARG, "dq is required");
    return LRAR_OK;
}

// Checks of the backward that do not depend on how the sources are passed;
// returns 1 (with *early set to the status) when nothing is left to launch.
int backward_common(int variant, int in_dtype, int grad_dtype, int n_src, int64_t T, int d, int r, float eps,
                    int h_dtype, float *dq, int accumulate, void *stream, bool *done) {
    *done = false;
    int rc = backward_scalars(variant, in_dtype, grad_dtype, n_src, T, d, r, eps, h_dtype, dq, accumulate);
    if (rc) return rc;
    if (T == 0) {  // dq is a sum over no tokens
        *done = true;
        if (!accumulate) {
            const int rq = variant == LRAR_FULL ? d : r;
            cudaError_t e = cudaMemsetAsync(dq, 0, sizeof(float) * (size_t)rq, static_cast<cudaStream_t>(stream));
            if (e != cudaSuccess) return cuda_fail(e, "lrar_backward");
        }
    }
    return LRAR_OK;
}

// Pointer checks of the backward's per-call tensors (dh, h, lse, query, dq).
int backward_tensors(int variant, const float *query, int n_src, const void *dh, const void *h, const float *lse,
                     const float *dq, const int *status) {
    if (!dh) return fail(LRAR_ERR_INVALID_ARG, "dh is required");
    if (variant == LRAR_FULL && (!h || !lse))
        return fail(LRAR_ERR_INVALID_ARG, "full AttnRes backward needs the forward's h and lse");
    if (!query && n_src > 1) return fail(LRAR_ERR_INVALID_ARG, "query is required when n_src > 1");
    if (!aligned16(dh) || !aligned4(dq) || (variant == LRAR_FULL && !aligned16(h)) || (lse && !aligned4(lse)) ||
        (query && !aligned4(query)) || (status && !aligned4(status)))
        return fail(LRAR_ERR_ALIGNMENT, "tensors must be 16-byte aligned (query, lse, dq and status 4-byte)");
    return LRAR_OK;
}

// Pointer checks of the stacked backward's source and gradient buffers.
int backward_stacks(int variant, const void *values, const void *keys, const void *dvalues, const void *dkeys) {
    if (!values || !dvalues) return fail(LRAR_ERR_INVALID_ARG, "values, dh and dvalues are required");
    if (variant == LRAR_PROJECTED && (!keys || !dkeys))
        return fail(LRAR_ERR_INVALID_ARG, "projected keys and dkeys are required");
    if (!aligned16(values) || !aligned16(dvalues) ||
        (variant == LRAR_PROJECTED && (!aligned16(keys) || !aligned16(dkeys))))
        return fail(LRAR_ERR_ALIGNMENT, "tensors must be 16-byte aligned (query, lse and dq 4-byte)");
    return LRAR_OK;
}

int backward_impl(int variant, int in_dtype, int grad_dtype, const void *const *values, const void *const *keys,
                  const float *query, int n_src, int64_t T, int d, int r, float eps, const void *dh, const void *h,
                  int h_dtype, const float *lse, void *const *dvalues, void *const *dkeys, float *dq,
                  int accumulate, void *workspace, size_t workspace_bytes, int *status, void *stream) {
    int rc = backward_tensors(variant, query, n_src, dh, h, lse, dq, status);
    if (rc) return rc;
    if (!workspace || workspace_bytes < lrar_backward_workspace_size(variant, n_src, T, d, r))
        return fail(LRAR_ERR_WORKSPACE, "workspace needs %zu bytes (got %zu)",
                    lrar_backward_workspace_size(variant, n_src, T, d, r), workspace ? workspace_bytes : (size_t)0);
    if (!aligned16(workspace)) return fail(LRAR_ERR_ALIGNMENT, "workspace must be 16-byte aligned");
    lrar::BwdArgs a;
    a.variant = variant;
    a.in_dtype = in_dtype;
    a.grad_dtype = grad_dtype;
    a.h_dtype = h_dtype;
    a.values = values;
    a.keys = variant == LRAR_PROJECTED ? keys : nullptr;
    a.query = query;
    a.n = n_src;
    a.T = T;
    a.d = d;
    a.r = r;
    a.eps = eps;
    a.dh = dh;
    a.h = variant == LRAR_FULL ? h : nullptr;
    a.lse = variant == LRAR_PROJECTED ? nullptr : lse;  // SLICED: one pass over the values when given
    a.dvalues = dvalues;
    a.dkeys = variant == LRAR_PROJECTED ? dkeys : nullptr;
    a.dq = dq;
    a.accumulate = accumulate;
    a.partials = static_cast<float *>(workspace);
    a.status = status;
    cudaError_t e = lrar::launch_backward(a, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "lrar_backward");
    return LRAR_OK;
}

}  // namespace

LRAR_API int lrar_forward(int variant, int in_dtype, int out_dtype, const void *values, const void *keys,
                          const float *query, int n_src, int64_t T, int d, int r, float eps, void *h, float *lse,
                          void *stream) {
    int rc = check_shape(variant, in_dtype, n_src, T, d, r, eps);
    if (rc) return rc;
    if (!dtype_ok(out_dtype)) return fail(LRAR_ERR_INVALID_ARG, "unknown output dtype %d", out_dtype);
    if (T == 0) return LRAR_OK;
    if (!values || !h) return fail(LRAR_ERR_INVALID_ARG, "values and h are required");
    if (variant == LRAR_PROJECTED && !keys) return fail(LRAR_ERR_INVALID_ARG, "projected keys are required");
    if (!aligned16(values) || (variant == LRAR_PROJECTED && !aligned16(keys)))
        return fail(LRAR_ERR_ALIGNMENT, "tensors must be 16-byte aligned (query and lse 4-byte)");
    const void *vt[LRAR_MAX_SOURCES], *kt[LRAR_MAX_SOURCES];
    stack_table(values, n_src, T, d, esize(in_dtype), vt);
    stack_table(variant == LRAR_PROJECTED ? keys : nullptr, n_src, T, r, esize(in_dtype), kt);
    return forward_impl(variant, in_dtype, out_dtype, vt, kt, query, n_src, T, d, r, eps, h, lse, stream);
}

LRAR_API int lrar_forward_ptrs(int variant, int in_dtype, int out_dtype, const void *const *values,
                               const void *const *keys, const float *query, int n_src, int64_t T, int d, int r,
                               float eps, void *h, float *lse, void *stream) {
    int rc = check_shape(variant, in_dtype, n_src, T, d, r, eps);
    if (rc) return rc;
    if (!dtype_ok(out_dtype)) return fail(LRAR_ERR_INVALID_ARG, "unknown output dtype %d", out_dtype);
    if (T == 0) return LRAR_OK;
    if ((rc = check_table(values, n_src, "values"))) return rc;
    if (variant == LRAR_PROJECTED && (rc = check_table(keys, n_src, "keys"))) return rc;
    return forward_impl(variant, in_dtype, out_dtype, values, keys, query, n_src, T, d, r, eps, h, lse, stream);
}

LRAR_API size_t lrar_backward_workspace_size(int variant, int n_src, int64_t T, int d, int r) {
    (void)n_src;
    (void)T;
    const int rq = variant == LRAR_FULL ? d : r;
    if (rq < 1) return 0;
    return sizeof(float) * (size_t)lrar::kMaxPartials * (size_t)rq;
}

LRAR_API int lrar_backward(int variant, int in_dtype, int grad_dtype, const void *values, const void *keys,
                           const float *query, int n_src, int64_t T, int d, int r, float eps, const void *dh,
                           const void *h, int h_dtype, const float *lse, void *dvalues, void *dkeys, float *dq,
                           int accumulate, void *workspace, size_t workspace_bytes, int *status, void *stream) {
    bool done;
    int rc = backward_common(variant, in_dtype, grad_dtype, n_src, T, d, r, eps, h_dtype, dq, accumulate, stream,
                             &done);
    if (rc || done) return rc;
    if ((rc = backward_stacks(variant, values, keys, dvalues, dkeys))) return rc;
    const int esz = esize(in_dtype), gsz = esize(grad_dtype);
    const void *vt[LRAR_MAX_SOURCES], *kt[LRAR_MAX_SOURCES], *dvt[LRAR_MAX_SOURCES], *dkt[LRAR_MAX_SOURCES];
    const bool pl = variant == LRAR_PROJECTED;
    stack_table(values, n_src, T, d, esz, vt);
    stack_table(pl ? keys : nullptr, n_src, T, r, esz, kt);
    stack_table(dvalues, n_src, T, d, gsz, dvt);
    stack_table(pl ? dkeys : nullptr, n_src, T, r, gsz, dkt);
    return backward_impl(variant, in_dtype, grad_dtype, vt, kt, query, n_src, T, d, r, eps, dh, h, h_dtype, lse,
                         const_cast<void *const *>(dvt), const_cast<void *const *>(dkt), dq, accumulate, workspace,
                         workspace_bytes, status, stream);
}

namespace lrar {

int check_backward(int variant, int in_dtype, int grad_dtype, const void *values, const void *keys,
                   const float *query, int n_src, int64_t T, int d, int r, float eps, const void *dh, const void *h,
                   int h_dtype, const float *lse, const void *dvalues, const void *dkeys, const float *dq,
                   int accumulate, const int *status) {
    int rc = backward_scalars(variant, in_dtype, grad_dtype, n_src, T, d, r, eps, h_dtype, const_cast<float *>(dq),
                              accumulate);
    if (rc || T == 0) return rc;
    if ((rc = backward_stacks(variant, values, keys, dvalues, dkeys))) return rc;
    return backward_tensors(variant, query, n_src, dh, h, lse, dq, status);
}

}  // namespace lrar

LRAR_API int lrar_backward_ptrs(int variant, int in_dtype, int grad_dtype, const void *const *values,
                                const void *const *keys, const float *query, int n_src, int64_t T, int d, int r,
                                float eps, const void *dh, const void *h, int h_dtype, const float *lse,
                                void *const *dvalues, void *const *dkeys, float *dq, int accumulate, void *workspace,
                                size_t workspace_bytes, int *status, void *stream) {
    bool done;
    int rc = backward_common(variant, in_dtype, grad_dtype, n_src, T, d, r, eps, h_dtype, dq, accumulate, stream,
                             &done);
    if (rc || done) return rc;
    if ((rc = check_table(values, n_src, "values"))) return rc;
    if ((rc = check_table(const_cast<const void *const *>(dvalues), n_src, "dvalues"))) return rc;
    if (variant == LRAR_PROJECTED) {
        if ((rc = check_table(keys, n_src, "keys"))) return rc;
        if ((rc = check_table(const_cast<const void *const *>(dkeys), n_src, "dkeys"))) return rc;
    }
    return backward_impl(variant, in_dtype, grad_dtype, values, keys, query, n_src, T, d, r, eps, dh, h, h_dtype, lse,
                         dvalues, dkeys, dq, accumulate, workspace, workspace_bytes, status, stream);
}

LRAR_API size_t lrar_diagnostics_workspace_size(int n_src) {
    return n_src < 1 ? 0 : sizeof(float) * (size_t)lrar::kMaxPartials * (size_t)n_src;
}

LRAR_API int lrar_diagnostics(int variant, int in_dtype, const void *values, const void *keys, const float *query,
                              int n_src, int64_t T, int d, int r, float eps, float *neff, float *mean_alpha,
                              void *workspace, size_t workspace_bytes, void *stream) {
    int rc = check_shape(variant, in_dtype, n_src, T, d, r, eps);
    if (rc) return rc;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (T == 0) {  // no tokens: the mean over them is defined here as 0
        if (mean_alpha) {
            cudaError_t e = cudaMemsetAsync(mean_alpha, 0, sizeof(float) * (size_t)n_src, s);
            if (e != cudaSuccess) return cuda_fail(e, "lrar_diagnostics");
        }
        return LRAR_OK;
    }
    if (!values) return fail(LRAR_ERR_INVALID_ARG, "values are required");
    if (variant == LRAR_PROJECTED && !keys) return fail(LRAR_ERR_INVALID_ARG, "projected keys are required");
    if (!query && n_src > 1) return fail(LRAR_ERR_INVALID_ARG, "query is required when n_src > 1");
    if (!aligned16(values) || (variant == LRAR_PROJECTED && !aligned16(keys)) || (query && !aligned4(query)) ||
        (neff && !aligned4(neff)) || (mean_alpha && !aligned4(mean_alpha)))
        return fail(LRAR_ERR_ALIGNMENT, "tensors must be 16-byte aligned (query, neff and mean_alpha 4-byte)");
    if (mean_alpha && (!workspace || workspace_bytes < lrar_diagnostics_workspace_size(n_src)))
        return fail(LRAR_ERR_WORKSPACE, "mean_alpha needs a workspace of %zu bytes",
                    lrar_diagnostics_workspace_size(n_src));
    if (mean_alpha && !aligned16(workspace)) return fail(LRAR_ERR_ALIGNMENT, "workspace must be 16-byte aligned");
    if (!neff && !mean_alpha) return LRAR_OK;
    const void *vt[LRAR_MAX_SOURCES], *kt[LRAR_MAX_SOURCES];
    stack_table(values, n_src, T, d, esize(in_dtype), vt);
    stack_table(variant == LRAR_PROJECTED ? keys : nullptr, n_src, T, r, esize(in_dtype), kt);
    lrar::FwdArgs a;
    a.variant = variant;
    a.in_dtype = in_dtype;
    a.out_dtype = in_dtype;
    a.values = vt;
    a.keys = variant == LRAR_PROJECTED ? kt : nullptr;
    a.query = query;
    a.n = n_src;
    a.T = T;
    a.d = d;
    a.r = r;
    a.eps = eps;
    a.h = nullptr;
    a.lse = nullptr;
    cudaError_t e = lrar::launch_diagnostics(a, neff, mean_alpha, static_cast<float *>(workspace), s);
    if (e != cudaSuccess) return cuda_fail(e, "lrar_diagnostics");
    return LRAR_OK;
}

namespace {

// values / keys: stacked buffers (tables == false) or host arrays of n_completed pointers (tables == true).
int block_phase1_impl(int variant, int in_dtype, int pre_dtype, const void *values, const void *keys, bool tables,
                      const float *queries, int n_completed, int n_sites, int64_t T, int d, int r, float eps,
                      void *h_pre, float *lse_pre, int *status, long long wait_cycles, bool stall, void *stream) {
    if (variant == LRAR_FULL)
        return fail(LRAR_ERR_UNSUPPORTED, "the two-phase block path serves low-rank keys (sliced, projected)");
    int rc = check_shape(variant, in_dtype, n_completed, T, d, r, eps);
    if (rc) return rc;
    if (!dtype_ok(pre_dtype)) return fail(LRAR_ERR_INVALID_ARG, "unknown phase-1 output dtype %d", pre_dtype);
    if (n_sites < 1 || n_sites > LRAR_MAX_BLOCK_SITES)
        return fail(LRAR_ERR_INVALID_ARG, "n_sites must be in 1..%d (got %d)", LRAR_MAX_BLOCK_SITES, n_sites);
    if (status && !aligned4(status)) return fail(LRAR_ERR_ALIGNMENT, "status must be 4-byte aligned");
    if (T == 0) return LRAR_OK;
    if (!values || !queries || !h_pre || !lse_pre)
        return fail(LRAR_ERR_INVALID_ARG, "values, queries, h_pre and lse_pre are required");
    if (variant == LRAR_PROJECTED && !keys) return fail(LRAR_ERR_INVALID_ARG, "projected keys are required");
    const void *vt[LRAR_MAX_SOURCES], *kt[LRAR_MAX_SOURCES];
    const void *const *vtab = vt, *const *ktab = kt;
    if (tables) {
        vtab = static_cast<const void *const *>(values);
        ktab = static_cast<const void *const *>(keys);
        int rc2 = check_table(vtab, n_completed, "values");
        if (rc2) return rc2;
        if (variant == LRAR_PROJECTED && (rc2 = check_table(ktab, n_completed, "keys"))) return rc2;
    } else {
        if (!aligned16(values) || (variant == LRAR_PROJECTED && !aligned16(keys)))
            return fail(LRAR_ERR_ALIGNMENT, "tensors must be 16-byte aligned (queries and lse_pre 4-byte)");
        stack_table(values, n_completed, T, d, esize(in_dtype), vt);
        stack_table(variant == LRAR_PROJECTED ? keys : nullptr, n_completed, T, r, esize(in_dtype), kt);
    }
    if (!aligned16(h_pre) || !aligned4(queries) || !aligned4(lse_pre))
        return fail(LRAR_ERR_ALIGNMENT, "tensors must be 16-byte aligned (queries and lse_pre 4-byte)");
    lrar::BlockPh1Args a;
    a.variant = variant;
    a.in_dtype = in_dtype;
    a.pre_dtype = pre_dtype;
    a.values = vtab;
    a.keys = variant == LRAR_PROJECTED ? ktab : nullptr;
    a.queries = queries;
    a.n = n_completed;
    a.c = n_sites;
    a.T = T;
    a.d = d;
    a.r = r;
    a.eps = eps;
    a.h_pre = h_pre;
    a.lse_pre = lse_pre;
    a.status = status;
    a.wait_cycles = wait_cycles;
    a.stall = stall;
    if (stall && !lrar::block_phase1_stages_keys(a))
        return fail(LRAR_ERR_UNSUPPORTED, "this shape reads keys from global memory: no waits to stall");
    cudaError_t e = lrar::launch_block_phase1(a, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "lrar_block_phase1");
    return LRAR_OK;
}

}  // namespace

LRAR_API int lrar_block_phase1(int variant, int in_dtype, int pre_dtype, const void *values, const void *keys,
                               const float *queries, int n_completed, int n_sites, int64_t T, int d, int r, float eps,
                               void *h_pre, float *lse_pre, int *status, void *stream) {
    return block_phase1_impl(variant, in_dtype, pre_dtype, values, keys, false, queries, n_completed, n_sites, T, d,
                             r, eps, h_pre, lse_pre, status, lrar::kWaitCycles, false, stream);
}

LRAR_API int lrar_block_phase1_ptrs(int variant, int in_dtype, int pre_dtype, const void *const *values,
                                    const void *const *keys, const float *queries, int n_completed, int n_sites,
                                    int64_t T, int d, int r, float eps, void *h_pre, float *lse_pre, int *status,
                                    void *stream) {
    return block_phase1_impl(variant, in_dtype, pre_dtype, values, keys, true, queries, n_completed, n_sites, T, d,
                             r, eps, h_pre, lse_pre, status, lrar::kWaitCycles, false, stream);
}

LRAR_API int lrar_test_block_phase1_stalled(int variant, int in_dtype, int pre_dtype, const void *values,
                                            const void *keys, const float *queries, int n_completed, int n_sites,
                                            int64_t T, int d, int r, float eps, void *h_pre, float *lse_pre,
                                            int *status, long long wait_cycles, void *stream) {
    if (!status) return fail(LRAR_ERR_INVALID_ARG, "the stalled phase 1 reports through status: it is required");
    if (wait_cycles < 1 || wait_cycles > (1LL << 32))
        return fail(LRAR_ERR_INVALID_ARG, "wait_cycles must be in 1 .. 2^32");
    return block_phase1_impl(variant, in_dtype, pre_dtype, values, keys, false, queries, n_completed, n_sites, T, d,
                             r, eps, h_pre, lse_pre, status, wait_cycles, true, stream);
}

namespace {

int block_phase2_impl(int variant, int in_dtype, int pre_dtype, int out_dtype, const void *h_pre,
                      const float *lse_pre, const void *prev, const void *partial, const void *prev_key,
                      const void *partial_key, const float *query, int64_t T, int d, int r, float eps, void *h,
                      float *lse, void *stream, const char *name);

}  // namespace

LRAR_API int lrar_block_phase2(int variant, int in_dtype, int pre_dtype, int out_dtype, const void *h_pre,
                               const float *lse_pre, const void *partial, const void *partial_key,
                               const float *query, int64_t T, int d, int r, float eps, void *h, float *lse,
                               void *stream) {
    return block_phase2_impl(variant, in_dtype, pre_dtype, out_dtype, h_pre, lse_pre, nullptr, partial, nullptr,
                             partial_key, query, T, d, r, eps, h, lse, stream, "lrar_block_phase2");
}

LRAR_API int lrar_block_phase2_assemble(int variant, int in_dtype, int pre_dtype, int out_dtype, const void *h_pre,
                                        const float *lse_pre, const void *prev_partial, void *member,
                                        const void *prev_partial_key, void *member_key, const float *query,
                                        int64_t T, int d, int r, float eps, void *h, float *lse, void *stream) {
    if (variant == LRAR_FULL)
        return fail(LRAR_ERR_UNSUPPORTED, "the two-phase block path serves low-rank keys (sliced, projected)");
    if (T > 0 && !prev_partial) return fail(LRAR_ERR_INVALID_ARG, "prev_partial is required");
    if (T > 0 && variant == LRAR_PROJECTED && !prev_partial_key)
        return fail(LRAR_ERR_INVALID_ARG, "the previous partial summary's projected key is required");
    if (prev_partial && !aligned16(prev_partial))
        return fail(LRAR_ERR_ALIGNMENT, "tensors must be 16-byte aligned (lse, query and keys 4-byte)");
    if (variant == LRAR_PROJECTED && prev_partial_key && !aligned4(prev_partial_key))
        return fail(LRAR_ERR_ALIGNMENT, "tensors must be 16-byte aligned (lse, query and keys 4-byte)");
    return block_phase2_impl(variant, in_dtype, pre_dtype, out_dtype, h_pre, lse_pre, prev_partial, member,
                             variant == LRAR_PROJECTED ? prev_partial_key : nullptr, member_key, query, T, d, r,
                             eps, h, lse, stream, "lrar_block_phase2_assemble");
}

namespace {

int block_phase2_impl(int variant, int in_dtype, int pre_dtype, int out_dtype, const void *h_pre,
                      const float *lse_pre, const void *prev, const void *partial, const void *prev_key,
                      const void *partial_key, const float *query, int64_t T, int d, int r, float eps, void *h,
                      float *lse, void *stream, const char *name) {
    if (variant == LRAR_FULL)
        return fail(LRAR_ERR_UNSUPPORTED, "the two-phase block path serves low-rank keys (sliced, projected)");
    int rc = check_shape(variant, in_dtype, 1, T, d, r, eps);
    if (rc) return rc;
    if (!dtype_ok(pre_dtype) || !dtype_ok(out_dtype)) return fail(LRAR_ERR_INVALID_ARG, "unknown dtype");
    if (T == 0) return LRAR_OK;
    if (!h_pre || !lse_pre || !partial || !query || !h)
        return fail(LRAR_ERR_INVALID_ARG, "h_pre, lse_pre, partial, query and h are required");
    if (variant == LRAR_PROJECTED && !partial_key)
        return fail(LRAR_ERR_INVALID_ARG, "the partial summary's projected key is required");
    if (!aligned16(h_pre) || !aligned16(partial) || !aligned16(h) || !aligned4(lse_pre) || !aligned4(query) ||
        (lse && !aligned4(lse)) || (variant == LRAR_PROJECTED && !aligned4(partial_key)))
        return fail(LRAR_ERR_ALIGNMENT, "tensors must be 16-byte aligned (lse, query and keys 4-byte)");
    lrar::BlockPh2Args a;
    a.variant = variant;
    a.in_dtype = in_dtype;
    a.pre_dtype = pre_dtype;
    a.out_dtype = out_dtype;
    a.h_pre = h_pre;
    a.lse_pre = lse_pre;
    a.partial = partial;
    a.pkeys = variant == LRAR_PROJECTED ? partial_key : nullptr;
    a.prev = prev;
    a.prev_keys = variant == LRAR_PROJECTED ? prev_key : nullptr;
    a.query = query;
    a.T = T;
    a.d = d;
    a.r = r;
    a.eps = eps;
    a.h = h;
    a.lse = lse;
    cudaError_t e = lrar::launch_block_phase2(a, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, name);
    return LRAR_OK;
}

}  // namespace

namespace {

int project_impl(int tile, int in_dtype, const void *a, const void *w, int64_t T, int m, int d, int r, void *o,
                 void *keys, int *status, void *stream) {
    if (!dtype_ok(in_dtype)) return fail(LRAR_ERR_INVALID_ARG, "unknown input dtype %d", in_dtype);
    if (in_dtype != LRAR_BF16) return fail(LRAR_ERR_UNSUPPORTED, "lrar_project takes bfloat16 operands");
    if (T < 0 || m < 1 || d < 0 || r < 0 || d + r < 1)
        return fail(LRAR_ERR_INVALID_ARG, "need T >= 0, m >= 1, d >= 0, r >= 0, d + r >= 1 (got T=%lld m=%d d=%d r=%d)",
                    (long long)T, m, d, r);
    if ((int64_t)d + r > 65535 * 176LL || T > (int64_t)0x7fffffff)
        return fail(LRAR_ERR_UNSUPPORTED, "projection too large (T < 2^31, d + r <= 65535 * 176)");
    if (m % 8 || d % 8 || r % 8) return fail(LRAR_ERR_ALIGNMENT, "m, d and r must be multiples of 8");
    if (!a || !w) return fail(LRAR_ERR_INVALID_ARG, "a and w are required");
    if ((d > 0 && !o) || (r > 0 && !keys)) return fail(LRAR_ERR_INVALID_ARG, "o (d > 0) and keys (r > 0) are required");
    if (!aligned16(a) || !aligned16(w) || (o && !aligned16(o)) || (keys && !aligned16(keys)))
        return fail(LRAR_ERR_ALIGNMENT, "a, w, o and keys must be 16-byte aligned");
    if (status && !aligned4(status)) return fail(LRAR_ERR_ALIGNMENT, "status must be 4-byte aligned");
    if (tile != 0 && !lrar::project_tile_ok(tile))
        return fail(LRAR_ERR_INVALID_ARG,
                    "tile must be 160, 176, 192, 224, 240 or 256, or 2000 plus one of them (got %d)", tile);
    if (T == 0) return LRAR_OK;
    return lrar::launch_project(a, w, T, m, d, r, o, keys, status, tile, static_cast<cudaStream_t>(stream));
}

}  // namespace

LRAR_API int lrar_project(int in_dtype, const void *a, const void *w, int64_t T, int m, int d, int r, void *o,
                          void *keys, int *status, void *stream) {
    return project_impl(0, in_dtype, a, w, T, m, d, r, o, keys, status, stream);
}

LRAR_API int lrar_test_project_tile(int tile, int in_dtype, const void *a, const void *w, int64_t T, int m, int d,
                                    int r, void *o, void *keys, int *status, void *stream) {
    if (tile == 0)
        return fail(LRAR_ERR_INVALID_ARG, "tile must be 160, 176, 192, 224, 240 or 256, or 2000 plus one of them (got 0)");
    return project_impl(tile, in_dtype, a, w, T, m, d, r, o, keys, status, stream);
}

LRAR_API int lrar_block_accumulate(int dst_dtype, void *dst, int src_dtype, const void *src, int64_t count,
                                   float alpha, float beta, void *stream) {
    if (!dtype_ok(dst_dtype) || !dtype_ok(src_dtype)) return fail(LRAR_ERR_INVALID_ARG, "unknown dtype");
    if (count < 0) return fail(LRAR_ERR_INVALID_ARG, "count must be >= 0");
    if (!isfinite(alpha) || !isfinite(beta)) return fail(LRAR_ERR_INVALID_ARG, "alpha and beta must be finite");
    if (count == 0) return LRAR_OK;
    if (!dst || !src) return fail(LRAR_ERR_INVALID_ARG, "dst and src are required");
    if ((reinterpret_cast<uintptr_t>(dst) % esize(dst_dtype)) || (reinterpret_cast<uintptr_t>(src) % esize(src_dtype)))
        return fail(LRAR_ERR_ALIGNMENT, "dst and src must be aligned to their element size");
    cudaError_t e = lrar::launch_block_accumulate(dst_dtype, dst, src_dtype, src, count, alpha, beta,
                                                  static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "lrar_block_accumulate");
    return LRAR_OK;
}
