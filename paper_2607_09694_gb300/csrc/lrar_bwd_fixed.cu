// lrar_bwd_fixed.cu -- the sliced-key backward with the forward's lse for
// bfloat16 rows of a fixed width (chain rule through Eq. 8-10 and 14 of arxiv
// 2607.09694; the paper prints no gradient formulas):
//
//   alpha_i = exp(s_i - lse),  g_i = <dh, o_i>,  gbar = sum_i alpha_i g_i,
//   ds_i = alpha_i (g_i - gbar),  dL/do_i = alpha_i dh  (+ dL/dk_i on the slice),
//   dL/dk_i = ds_i rho_i (q - (s_i / r) kbar_i),  dL/dq = sum ds_i kbar_i.
//
// One pass over the values, as in the generic one-pass kernels of lrar_bwd.cu,
// with the row width D and the key rank R fixed at compile time, so that every
// lane's vectors, the lanes holding the key slice and every loop bound are
// constants.  g_i takes its products straight from the packed bfloat16 words
// (fma.rn.f32.bf16: the product of two bfloat16 values is exact in fp32 and
// the sum is rounded once, the same value as fmaf of the widened operands), so
// neither the row nor dh is widened for it; dh is widened once per token for
// the gradient rows.  The gradient rows are bitwise those of the generic
// kernels; dq is their fixed-order sum over the same grid when accumulating (the
// writing generic kernel runs one CTA per SM, so its dq sums in another order).
//
// Two CTAs per SM.  Shared memory: ring [kWarps][S][P][V][32] cells (P = 2
// planes, value and old gradient, when accumulating) | q [R] | dq [kWarps][R] |
// tables [kWarps][2][n4] (alpha, g) | per warp: key stash [n][NV] cells and the
// token's dh slice [NV] cells.
#include "lrar.h"
#include "lrar_bwd.cuh"
#include "lrar_device.cuh"
#include "lrar_launch.h"

namespace lrar {

// g0 += lo(a) lo(b), g1 += hi(a) hi(b) for two packed bfloat16 pairs.
__device__ __forceinline__ void fma_bf16x2(float &g0, float &g1, uint32_t a, uint32_t b) {
    asm("{\n\t.reg .b16 al, ah, bl, bh;\n\tmov.b32 {al, ah}, %2;\n\tmov.b32 {bl, bh}, %3;\n\t"
        "fma.rn.f32.bf16 %0, al, bl, %0;\n\tfma.rn.f32.bf16 %1, ah, bh, %1;\n\t}"
        : "+f"(g0), "+f"(g1)
        : "r"(a), "r"(b));
}

template <int D, int R, int S, bool ACC> struct FixedShape {
    static constexpr int E = 8;                 // bfloat16 elements per 16-byte vector
    static constexpr int V = D / (32 * E);      // vectors per lane
    static constexpr int NV = R / E;            // lanes holding a row's key slice
    static constexpr int LEAD = 32 - NV;        // first of them; the slice is in vector V - 1
    static constexpr int KST = 32 / NV;         // sources per round of the slice pass
    static constexpr int P = ACC ? 2 : 1;       // ring planes
    static_assert(D % (32 * E) == 0 && R % E == 0 && 32 % NV == 0 && D % R == 0, "fixed shapes only");
    static size_t smem(int n) {
        const int n4 = round_up(n, 4);
        return (size_t)kWarps * S * P * V * 32 * 16 + sizeof(float) * (size_t)R * (1 + kWarps) +
               (size_t)kWarps * (sizeof(float) * 2 * n4 + (size_t)16 * NV * (n + 1));
    }
};

template <int D, int R, int S, bool ACC>
__global__ void __launch_bounds__(kThreads, 2) bwd_slr_fixed_kernel(const __grid_constant__ BwdParams p) {
    pdl_enter();
    using Sh = FixedShape<D, R, S, ACC>;
    constexpr int E = Sh::E, V = Sh::V, NV = Sh::NV, LEAD = Sh::LEAD, KST = Sh::KST, P = Sh::P;
    constexpr int TAIL0 = D - R;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int n4 = round_up(p.n, 4);
    float *q_s = reinterpret_cast<float *>(smem_raw + (size_t)kWarps * S * P * V * 32 * 16);
    float *dq_all = q_s + R;            // [kWarps][R]
    float *tab = dq_all + kWarps * R;   // [kWarps][2][n4]
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    float *a_s = tab + warp * 2 * n4;
    float *g_s = a_s + n4;
    const uint32_t stash_w = smem_u32(tab + kWarps * 2 * n4) + (uint32_t)(warp * NV * (p.n + 1) * 16);
    const uint32_t dhs_w = stash_w + (uint32_t)(p.n * NV * 16);
    const uint32_t ring_w = smem_u32(smem_raw) + (uint32_t)(warp * S * P * V * 32 * 16) + 16u * lane;
    for (int j = threadIdx.x; j < R; j += kThreads) q_s[j] = p.query ? p.query[j] : 0.f;
    __syncthreads();

    const bf16 *__restrict__ dh = static_cast<const bf16 *>(p.dh);
    const int64_t nwarps = (int64_t)gridDim.x * kWarps;
    const int kvi = lane - LEAD;
    const bool has_key = kvi >= 0;  // this lane's last vector is a slice vector
    const bool full_last = lane < LEAD;  // its last vector lies before the slice
    float qv[E];
#pragma unroll
    for (int t = 0; t < E; ++t) qv[t] = has_key ? q_s[kvi * E + t] : 0.f;
    // slice pass: lane takes slice vector kp of sources lane / NV, lane / NV + KST, ...
    const int kp = lane % NV, j0 = kp * E;
    float qs[E];
#pragma unroll
    for (int t = 0; t < E; ++t) qs[t] = q_s[j0 + t];
    float dq_r[E];
#pragma unroll
    for (int t = 0; t < E; ++t) dq_r[t] = 0.f;

    // the ring: this lane's next copies are its vectors of source ii's row of token ix
    const int64_t x0 = (int64_t)blockIdx.x * kWarps + warp;
    int64_t ix = x0;
    int ii = 0;
    uint32_t wcell = ring_w;  // the stage the next copies go to
    const uint32_t ring_end = ring_w + (uint32_t)(S * P * V * 32 * 16);
    auto issue = [&]() {
        if (ix < p.T) {
            const bf16 *row = static_cast<const bf16 *>(p.vt.p[ii]) + ix * D + lane * E;
#pragma unroll
            for (int v = 0; v < V; ++v) cp_async16(wcell + (uint32_t)(v * 32 * 16), row + v * 32 * E);
            if (ACC) {
                const bf16 *old = static_cast<const bf16 *>(p.dvt.p[ii]) + ix * D + lane * E;
#pragma unroll
                for (int v = 0; v < V; ++v)  // the slice's old value is re-read with the slice
                    if (v < V - 1 || full_last) cp_async16(wcell + (uint32_t)((V + v) * 32 * 16), old + v * 32 * E);
            }
            if (++ii == p.n) {
                ii = 0;
                ix += nwarps;
            }
        }
        cp_async_commit();
        wcell += (uint32_t)(P * V * 32 * 16);
        if (wcell == ring_end) wcell = ring_w;
    };
#pragma unroll
    for (int st = 0; st < S - 1; ++st) issue();
    uint32_t rcell = ring_w;  // the stage of the next row to use

    for (int64_t x = x0; x < p.T; x += nwarps) {
        Frag<bf16, E> dhr[V];
        float dv[V][E];
#pragma unroll
        for (int v = 0; v < V; ++v) {
            dhr[v].load_nc(dh + x * D + (lane + 32 * v) * E);
            dhr[v].get(dv[v]);
        }
        const float lse = __ldg(p.lse + x);
        if (has_key) st_shared16(dhs_w + (uint32_t)(kvi * 16), dhr[V - 1].a);

        float asum = 0.f;
        for (int i = 0; i < p.n; ++i) {
            issue();
            cp_async_wait<S - 1>();  // this lane's copies of row i have landed
            Frag<bf16, E> f[V];
#pragma unroll
            for (int v = 0; v < V; ++v) f[v].a = ld_shared16(rcell + (uint32_t)(v * 32 * 16));
            float g0 = 0.f, g1 = 0.f;
#pragma unroll
            for (int v = 0; v < V; ++v) {
                fma_bf16x2(g0, g1, dhr[v].a.x, f[v].a.x);
                fma_bf16x2(g0, g1, dhr[v].a.y, f[v].a.y);
                fma_bf16x2(g0, g1, dhr[v].a.z, f[v].a.z);
                fma_bf16x2(g0, g1, dhr[v].a.w, f[v].a.w);
            }
            float ss = 0.f, qk = 0.f;
            if (has_key) {
                float o[E];
                f[V - 1].get(o);
#pragma unroll
                for (int t = 0; t < E; ++t) {
                    ss = fmaf(o[t], o[t], ss);
                    qk = fmaf(qv[t], o[t], qk);
                }
                st_shared16(stash_w + (uint32_t)((i * NV + kvi) * 16), f[V - 1].a);
            }
#pragma unroll
            for (int off = 1; off < NV; off <<= 1) {  // the slice lanes form an aligned group
                ss += __shfl_xor_sync(0xffffffffu, ss, off);
                qk += __shfl_xor_sync(0xffffffffu, qk, off);
            }
            const float rho = rsqrtf(fmaf(ss, p.inv_r, p.eps));
            const float s = __shfl_sync(0xffffffffu, rho * qk, LEAD);
            // one source weighs exactly 1 (a softmax over one score), however s rounds against lse
            const float a = p.n == 1 ? 1.f : expf(s - lse);
            asum += a;
            bf16 *drow = static_cast<bf16 *>(const_cast<void *>(p.dvt.p[i])) + x * D + lane * E;
#pragma unroll
            for (int v = 0; v < V; ++v) {
                if (v < V - 1 || full_last) {
                    float w[E];
                    if (ACC) {
                        Frag<bf16, E> of;
                        of.a = ld_shared16(rcell + (uint32_t)((V + v) * 32 * 16));
                        of.get(w);
                    }
#pragma unroll
                    for (int t = 0; t < E; ++t) w[t] = ACC ? fmaf(a, dv[v][t], w[t]) : a * dv[v][t];
                    Frag<bf16, E> out;
                    out.set(w);
                    out.store(drow + v * 32 * E);
                }
            }
            const float g = warp_sum(g0 + g1);
            if (lane == LEAD) {
                a_s[i] = a;
                g_s[i] = g;
            }
            rcell += (uint32_t)(P * V * 32 * 16);
            if (rcell == ring_end) rcell = ring_w;
        }
        __syncwarp();  // stash, tables and the dh slice are visible to the whole warp
        check_alpha_sum(p, asum, lane);

        float part = 0.f;
        for (int k = lane; k < p.n; k += 32) part = fmaf(a_s[k], g_s[k], part);
        const float gbar = warp_sum(part);
        float dhv[E];
        {
            Frag<bf16, E> hf;
            hf.a = ld_shared16(dhs_w + (uint32_t)(kp * 16));
            hf.get(dhv);
        }
        // sources k = lane / NV + m KST: the old slices of a batch are loaded together
        constexpr int B = 4;
        for (int kb = lane / NV; kb - (lane / NV) < p.n; kb += KST * B) {
            Frag<bf16, E> of[B];
#pragma unroll
            for (int m = 0; m < B; ++m) {
                const int k = kb + m * KST;
                if (ACC && k < p.n) of[m].load(static_cast<const bf16 *>(p.dvt.p[k]) + x * D + TAIL0 + j0);
                else of[m].zero();
            }
#pragma unroll
            for (int m = 0; m < B; ++m) {
                const int k = kb + m * KST;  // the NV lanes of source k are consecutive: an aligned group
                Frag<bf16, E> kf;
                if (k < p.n) kf.a = ld_shared16(stash_w + (uint32_t)((k * NV + kp) * 16));
                else kf.zero();
                float kv[E], w[E];
                kf.get(kv);
                of[m].get(w);
                float ss = 0.f, qk = 0.f;
#pragma unroll
                for (int t = 0; t < E; ++t) {
                    ss = fmaf(kv[t], kv[t], ss);
                    qk = fmaf(qs[t], kv[t], qk);
                }
#pragma unroll
                for (int off = 1; off < NV; off <<= 1) {
                    ss += __shfl_xor_sync(0xffffffffu, ss, off);
                    qk += __shfl_xor_sync(0xffffffffu, qk, off);
                }
                if (k < p.n) {
                    const float rho = rsqrtf(fmaf(ss, p.inv_r, p.eps));
                    const float s = rho * qk;
                    const float a = a_s[k];
                    const float ds = a * (g_s[k] - gbar);
                    const float c1 = ds * rho, c2 = s * p.inv_r;
#pragma unroll
                    for (int t = 0; t < E; ++t) {
                        const float kbar = rho * kv[t];
                        const float dk = c1 * (qs[t] - c2 * kbar);
                        dq_r[t] = fmaf(ds, kbar, dq_r[t]);
                        w[t] += fmaf(a, dhv[t], dk);
                    }
                    Frag<bf16, E> out;
                    out.set(w);
                    out.store(static_cast<bf16 *>(const_cast<void *>(p.dvt.p[k])) + x * D + TAIL0 + j0);
                }
            }
        }
        __syncwarp();  // the next token overwrites stash, tables and dh slice
    }
    cp_async_wait_all();
    // lanes sharing a slice vector combine their dq parts with a fixed butterfly
#pragma unroll
    for (int t = 0; t < E; ++t)
#pragma unroll
        for (int off = NV; off < 32; off <<= 1) dq_r[t] += __shfl_xor_sync(0xffffffffu, dq_r[t], off);
    if (lane < NV)
#pragma unroll
        for (int t = 0; t < E; ++t) dq_all[warp * R + j0 + t] = dq_r[t];
    __syncthreads();
    for (int j = threadIdx.x; j < R; j += kThreads) {
        float acc = 0.f;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) acc += dq_all[w * R + j];
        p.partials[(int64_t)blockIdx.x * R + j] = acc;
    }
}

namespace {

template <int D, int R, int S, bool ACC>
cudaError_t go_fixed(const BwdParams &p, const BwdArgs &a, bool &launched, cudaStream_t s) {
    using Sh = FixedShape<D, R, S, ACC>;
    const size_t smem = Sh::smem(a.n);
    int dev = 0, per_sm = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&per_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev);
    if (2 * (smem + 1024) > (size_t)per_sm) return cudaSuccess;  // two CTAs per SM (1 KB reserved each), else not used
    const void *k = (const void *)bwd_slr_fixed_kernel<D, R, S, ACC>;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int grid = persistent_grid(k, kThreads, smem, (a.T + kWarps - 1) / kWarps, kMaxPartials);
    launch_pdl(bwd_slr_fixed_kernel<D, R, S, ACC>, grid, kThreads, smem, s, p);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    launched = true;
    return launch_partial_sum(a.partials, grid, R, a.dq, a.accumulate, s);
}

}  // namespace

// The fixed-shape kernel serves bfloat16 sliced keys with the forward's lse at
// (d, r) = (1024, 16); `launched` stays false for every other call.
cudaError_t launch_bwd_fixed(const BwdParams &p, const BwdArgs &a, bool &launched, cudaStream_t s) {
    launched = false;
    if (a.variant != kSliced || a.in_dtype != kBF16 || a.grad_dtype != kBF16 || !a.lse) return cudaSuccess;
    if (a.d == 1024 && a.r == 16)
        return a.accumulate ? go_fixed<1024, 16, 3, true>(p, a, launched, s) : go_fixed<1024, 16, 5, false>(p, a, launched, s);
    return cudaSuccess;
}

}  // namespace lrar
