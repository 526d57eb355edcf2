// lrar_launch.h -- host-side launch interface between the C ABI (lrar_api.cu)
// and the kernel translation units.  Arguments arrive here already validated.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace lrar {

enum { kFull = 0, kSliced = 1, kProjected = 2 };
enum { kF32 = 0, kBF16 = 1 };

// Source tables: entry i is the base of source i's row-major [T, width]
// matrix, so row x of source i starts at p[i] + x * width elements.  A stacked
// [n, T, width] buffer is the table base + i * T * width.
constexpr int kMaxTab = 128;
struct SrcTab {
    const void *p[kMaxTab];
};

struct FwdArgs {
    int variant, in_dtype, out_dtype;
    const void *const *values;  // host array of n source pointers
    const void *const *keys;    // host array of n P-LR key pointers (P-LR only)
    const float *query;  // may be null when n == 1
    int n;
    int64_t T;
    int d, r;
    float eps;
    void *h;
    float *lse;  // may be null
};

struct BwdArgs {
    int variant, in_dtype, grad_dtype, h_dtype;
    const void *const *values;  // host arrays of n pointers, as in FwdArgs
    const void *const *keys;
    const float *query;
    int n;
    int64_t T;
    int d, r;
    float eps;
    const void *dh;
    const void *h;
    const float *lse;
    void *const *dvalues;  // host arrays of n gradient pointers (dkeys: P-LR only)
    void *const *dkeys;
    float *dq;
    int accumulate;
    float *partials;  // workspace: [kMaxPartials][rq] floats
    int *status;      // optional: LRAR_STATUS_LSE_MISMATCH is ORed in by kernels that take alpha from lse
};

struct BlockPh1Args {
    int variant, in_dtype, pre_dtype;
    const void *const *values;  // host array of n pointers: completed sources, [T, d] each
    const void *const *keys;    // host array of n P-LR key pointers ([T, r] each), or null
    const float *queries;       // [c, r]
    int n, c;
    int64_t T;
    int d, r;
    float eps;
    void *h_pre;     // [c, T, d]
    float *lse_pre;  // [c, T]
    int *status;     // optional: LRAR_STATUS_WAIT_TIMEOUT is ORed in when a key wait gives up
    long long wait_cycles;  // bound of each key wait (SM clock cycles)
    bool stall;      // test hook: key waits wait on a barrier nothing completes
};

// Bound of a kernel's waits on its own asynchronous copies: about 2 s at the
// GB300's 2.07 GHz SM clock, far beyond any copy's latency.
constexpr long long kWaitCycles = 4LL << 30;

// Whether a phase-1 launch with these arguments stages keys in shared memory
// (and so waits for bulk copies).
bool block_phase1_stages_keys(const BlockPh1Args &a);

struct BlockPh2Args {
    int variant, in_dtype, pre_dtype, out_dtype;
    const void *h_pre;     // [T, d] of one site
    const float *lse_pre;  // [T]
    const void *partial;   // partial-block summary [T, d] (assembling: the newest member's output, replaced by it)
    const void *pkeys;     // its P-LR key [T, r] (likewise)
    const void *prev = nullptr;       // assembling: the running sum before the member [T, d], else null
    const void *prev_keys = nullptr;  // and its P-LR key [T, r]
    const float *query;    // [r]
    int64_t T;
    int d, r;
    float eps;
    void *h;     // [T, d]
    float *lse;  // [T] or null
};

cudaError_t launch_block_phase1(const BlockPh1Args &a, cudaStream_t s);
cudaError_t launch_block_phase2(const BlockPh2Args &a, cudaStream_t s);

// Sets the calling thread's lrar_last_error() message; returns `code`.
int record_error(int code, const char *message);

// Every argument check of lrar_backward on a stacked buffer except those of
// the workspace, in the same order and with the same messages; launches
// nothing.  LRAR_OK for T == 0 once the scalar arguments are valid.
int check_backward(int variant, int in_dtype, int grad_dtype, const void *values, const void *keys,
                   const float *query, int n_src, int64_t T, int d, int r, float eps, const void *dh, const void *h,
                   int h_dtype, const float *lse, const void *dvalues, const void *dkeys, const float *dq,
                   int accumulate, const int *status);

// P-LR fused output projection on the tensor cores (lrar_proj.cu); returns an
// LRAR status (argument checks done by the caller).
// tile: 0 picks the width from the shape, else one of the compiled widths.
int launch_project(const void *a, const void *w, int64_t T, int m, int d, int r, void *o, void *keys, int *status,
                   int tile, cudaStream_t s);
bool project_tile_ok(int tile);

// Largest d one warp covers (the kernels keep a whole token row per warp).
int max_width(int in_dtype);

cudaError_t launch_forward(const FwdArgs &a, cudaStream_t s);
// Routing diagnostics (a.h unused): neff [T] and/or mean_alpha [n] (the latter
// through `partials`, [kMaxPartials][n] floats).
cudaError_t launch_diagnostics(const FwdArgs &a, float *neff, float *mean_alpha, float *partials, cudaStream_t s);
// out[j] (+)= sum_b partials[b][j] for b < nparts, in a fixed order.
cudaError_t launch_partial_sum(const float *partials, int nparts, int width, float *out, int accumulate,
                               cudaStream_t s);
cudaError_t launch_backward(const BwdArgs &a, cudaStream_t s);
cudaError_t launch_block_accumulate(int dst_dtype, void *dst, int src_dtype, const void *src, int64_t count,
                                    float alpha, float beta, cudaStream_t s);

// Resident CTAs of `kernel` per SM times the SM count of the current device,
// capped by `cap`.
int persistent_grid(const void *kernel, int threads, size_t smem, int64_t work_ctas, int cap);

// Launches kernel with programmatic stream serialization, so that it can be
// scheduled while the previous kernel in the stream finishes (every kernel of
// the library waits for its predecessor with griddepcontrol.wait before it
// touches global memory).  Errors are returned and kept for cudaGetLastError.
template <typename... K, typename... A>
inline cudaError_t launch_pdl(void (*kernel)(K...), dim3 grid, dim3 block, size_t smem, cudaStream_t s, A &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<A &&>(args)...);
}

}  // namespace lrar
