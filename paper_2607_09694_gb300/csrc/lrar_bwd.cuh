// lrar_bwd.cuh -- the backward kernels' launch parameters, shared by the
// translation units that hold backward kernels (lrar_bwd.cu, lrar_bwd_fixed.cu).
#pragma once

#include "lrar.h"
#include "lrar_device.cuh"
#include "lrar_launch.h"

namespace lrar {

struct BwdParams {
    SrcTab vt, kt, dvt, dkt;  // values, P-LR keys and their gradients, one matrix per source
    const void *dh, *h;
    const float *query, *lse;
    float *partials;
    int *status;  // optional: LRAR_STATUS_LSE_MISMATCH when a token's weights from lse do not sum to 1
    int64_t T;
    int n, d, r;
    float eps, inv_r;
    int sliced, key_vec, accumulate, h_bf16;
};

// Weights taken from a supplied lse sum to 1 up to fp32 rounding when the lse
// belongs to the same values and query; a sum further than this from 1 marks
// an lse of other inputs.
constexpr float kLseSumTol = 1e-3f;

__device__ __forceinline__ void check_alpha_sum(const BwdParams &p, float asum, int lane) {
    if (lane == 0 && p.status && !(fabsf(asum - 1.f) <= kLseSumTol)) atomicOr(p.status, LRAR_STATUS_LSE_MISMATCH);
}

// The fixed-shape sliced backward (lrar_bwd_fixed.cu): launches it and sets
// launched when the call's shape is one it was compiled for.
cudaError_t launch_bwd_fixed(const BwdParams &p, const BwdArgs &a, bool &launched, cudaStream_t s);

}  // namespace lrar
