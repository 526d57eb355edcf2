// lrar_block.cu -- Block AttnRes two-phase batched sites (§3.5 of arxiv
// 2607.09694) for low-rank keys.
//
// The c read sites inside one block see the same completed sources (embedding
// and completed block summaries, Eq. 5) plus a partial-block summary that
// grows by one output per site (Eq. 6).  Queries are static, so:
//
//   phase 1  one pass over the n completed sources serves all c queries: per
//            token and site j, lse_j = log sum_i exp(s_ij) and the normalised
//            mix h_pre_j = sum_i exp(s_ij - lse_j) o_i;
//   phase 2  at site j the partial summary b_P (score s_P) joins by the online
//            softmax update lse = log(exp(lse_j) + exp(s_P)),
//            h = exp(lse_j - lse) h_pre_j + exp(s_P - lse) b_P.
//
// The result is the site's mix over [completed sources, b_P] (Eq. 8-10).
// Phase 1 tiles a token's row over warps: warp (g, ch) of a CTA owns the
// 32 x 16-byte chunk ch of token g's rows and keeps c accumulators per element.
#include "lrar_device.cuh"
#include "lrar_launch.h"

namespace lrar {

constexpr int kPh1MaxSites = 8;  // queries per phase-1 launch (more are split by the host)

struct Ph1Params {
    const void *values, *keys;
    const float *queries;  // [c][r]
    void *h_pre;           // [c][T][d]
    float *lse_pre;        // [c][T]
    int64_t T, site_stride;  // site_stride: elements between sites in h_pre (T * d)
    int n, c, d, r, chunks;
    float eps, inv_r;
    int sliced, key_vec;
};

template <typename Tin, typename Tout>
__global__ void __launch_bounds__(kThreads) block_phase1_kernel(const Ph1Params p) {
    constexpr int E = VecE<Tin>::value;
    constexpr int U = 4;  // rows in flight per lane
    extern __shared__ float smem[];
    const int rp = round_up(p.r, 4);
    float *q_s = smem;                             // [c][r]
    float *a_s = q_s + kPh1MaxSites * rp;          // [kWarps][c][n]: scores, then weights
    float *lse_s = a_s + kWarps * kPh1MaxSites * p.n;  // [kWarps][c]
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int G = kWarps / p.chunks;  // tokens per CTA pass
    const int g = warp / p.chunks, ch = warp % p.chunks;
    for (int j = threadIdx.x; j < p.c * p.r; j += kThreads) q_s[(j / p.r) * rp + j % p.r] = p.queries[j];
    __syncthreads();

    const Tin *__restrict__ values = static_cast<const Tin *>(p.values);
    const Tin *__restrict__ keys = static_cast<const Tin *>(p.keys);
    Tout *__restrict__ h_pre = static_cast<Tout *>(p.h_pre);
    const int e = (ch * 32 + lane) * E;  // this lane's first element of the row
    float *ag = a_s + g * kPh1MaxSites * p.n;

    for (int64_t base = (int64_t)blockIdx.x * G; base < p.T; base += (int64_t)gridDim.x * G) {
        const int64_t x = base + g;
        if (ch == 0 && x < p.T) {
            // Eq. (8)-(9) for all c queries: lane i scores source i
            for (int i = lane; i < p.n; i += 32) {
                const Tin *kp = p.sliced ? values + ((int64_t)i * p.T + x) * p.d + (p.d - p.r)
                                         : keys + ((int64_t)i * p.T + x) * p.r;
                float ss = 0.f, qk[kPh1MaxSites];
#pragma unroll
                for (int j = 0; j < kPh1MaxSites; ++j) qk[j] = 0.f;
                for (int jj = 0; jj < p.r; ++jj) {
                    const float k = to_f(__ldg(kp + jj));
                    ss = fmaf(k, k, ss);
#pragma unroll
                    for (int j = 0; j < kPh1MaxSites; ++j)
                        if (j < p.c) qk[j] = fmaf(q_s[j * rp + jj], k, qk[j]);
                }
                const float rho = rsqrtf(fmaf(ss, p.inv_r, p.eps));
#pragma unroll
                for (int j = 0; j < kPh1MaxSites; ++j)
                    if (j < p.c) ag[j * p.n + i] = rho * qk[j];
            }
            __syncwarp();
            for (int j = 0; j < p.c; ++j) {
                float m = -INFINITY;
                for (int i = lane; i < p.n; i += 32) m = fmaxf(m, ag[j * p.n + i]);
                m = warp_max(m);
                float z = 0.f;
                for (int i = lane; i < p.n; i += 32) z += expf(ag[j * p.n + i] - m);
                z = warp_sum(z);
                __syncwarp();
                for (int i = lane; i < p.n; i += 32) ag[j * p.n + i] = expf(ag[j * p.n + i] - m) / z;
                if (lane == 0) lse_s[g * kPh1MaxSites + j] = m + logf(z);
                __syncwarp();
            }
        }
        __syncthreads();
        if (x < p.T) {
            float acc[kPh1MaxSites][E];
#pragma unroll
            for (int j = 0; j < kPh1MaxSites; ++j)
#pragma unroll
                for (int t = 0; t < E; ++t) acc[j][t] = 0.f;
            const Tin *row0 = values + x * p.d + e;
            for (int i0 = 0; i0 < p.n; i0 += U) {
                Frag<Tin, E> f[U];
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    if (i0 + u < p.n && e < p.d) f[u].load_nc(row0 + (int64_t)(i0 + u) * p.T * p.d);
                    else f[u].zero();
                }
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    if (i0 + u < p.n) {
                        float o[E];
                        f[u].get(o);
#pragma unroll
                        for (int j = 0; j < kPh1MaxSites; ++j) {
                            if (j < p.c) {
                                const float w = ag[j * p.n + i0 + u];
#pragma unroll
                                for (int t = 0; t < E; ++t) acc[j][t] = fmaf(w, o[t], acc[j][t]);
                            }
                        }
                    }
                }
            }
            if (e < p.d) {
#pragma unroll
                for (int j = 0; j < kPh1MaxSites; ++j) {
                    if (j < p.c) {
                        Frag<Tout, E> out;
                        out.set(acc[j]);
                        out.store(h_pre + (int64_t)j * p.site_stride + x * p.d + e);
                    }
                }
            }
            if (ch == 0 && lane < p.c) p.lse_pre[(int64_t)lane * p.T + x] = lse_s[g * kPh1MaxSites + lane];
        }
        __syncthreads();
    }
}

struct Ph2Params {
    const void *h_pre, *partial, *pkeys;
    const float *lse_pre, *query;
    void *h;
    float *lse;
    int64_t T;
    int d, r;
    float eps, inv_r;
    int sliced;
};

// Phase 2: one warp per token merges h_pre with the partial-block summary.
template <typename Tin, typename Tp, typename Tout, int V>
__global__ void __launch_bounds__(kThreads) block_phase2_kernel(const Ph2Params p) {
    constexpr int E = VecE<Tin>::value;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const Tin *__restrict__ part = static_cast<const Tin *>(p.partial);
    const Tin *__restrict__ pkeys = static_cast<const Tin *>(p.pkeys);
    const Tp *__restrict__ h_pre = static_cast<const Tp *>(p.h_pre);
    Tout *__restrict__ h = static_cast<Tout *>(p.h);
    const int64_t nwarps = (int64_t)gridDim.x * kWarps;
    for (int64_t x = (int64_t)blockIdx.x * kWarps + warp; x < p.T; x += nwarps) {
        // score of the partial summary, Eq. (8)-(9)
        const Tin *kp = p.sliced ? part + x * p.d + (p.d - p.r) : pkeys + x * p.r;
        float ss = 0.f, qk = 0.f;
        for (int j = lane; j < p.r; j += 32) {
            const float k = to_f(__ldg(kp + j));
            ss = fmaf(k, k, ss);
            qk = fmaf(__ldg(p.query + j), k, qk);
        }
        ss = warp_sum(ss);
        qk = warp_sum(qk);
        const float sP = rsqrtf(fmaf(ss, p.inv_r, p.eps)) * qk;
        const float lp = __ldg(p.lse_pre + x);
        const float M = fmaxf(lp, sP);
        const float lse = M + logf(expf(lp - M) + expf(sP - M));
        const float w1 = expf(lp - lse), w2 = expf(sP - lse);
#pragma unroll
        for (int v = 0; v < V; ++v) {
            const int e = (lane + 32 * v) * E;
            if (e < p.d) {
                Frag<Tin, E> fb;
                fb.load_nc(part + x * p.d + e);
                Frag<Tp, E> fh;
                fh.load_nc(h_pre + x * p.d + e);
                float b[E], hp[E], o[E];
                fb.get(b);
                fh.get(hp);
#pragma unroll
                for (int t = 0; t < E; ++t) o[t] = fmaf(w2, b[t], w1 * hp[t]);
                Frag<Tout, E> out;
                out.set(o);
                out.store(h + x * p.d + e);
            }
        }
        if (lane == 0 && p.lse) p.lse[x] = lse;
    }
}

// --------------------------------------------------------------- launch ----
template <typename Tin, typename Tout>
static cudaError_t launch_ph1_t(const BlockPh1Args &a, cudaStream_t s) {
    constexpr int E = VecE<Tin>::value;
    const int chunks_needed = (a.d + 32 * E - 1) / (32 * E);
    int chunks = 1;
    while (chunks < chunks_needed) chunks *= 2;  // 1, 2, 4 or 8 (validated: d <= 8 * 32 * E)
    Ph1Params p;
    p.values = a.values;
    p.keys = a.keys;
    p.T = a.T;
    p.site_stride = a.T * (int64_t)a.d;
    p.n = a.n;
    p.d = a.d;
    p.r = a.r;
    p.chunks = chunks;
    p.eps = a.eps;
    p.inv_r = 1.f / (float)a.r;
    p.sliced = a.variant == kSliced;
    p.key_vec = 0;
    const size_t smem = sizeof(float) * ((size_t)kPh1MaxSites * round_up(a.r, 4) +
                                         (size_t)kWarps * kPh1MaxSites * a.n + (size_t)kWarps * kPh1MaxSites);
    const void *k = (const void *)block_phase1_kernel<Tin, Tout>;
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
    }
    const int G = kWarps / chunks;
    const int grid = persistent_grid(k, kThreads, smem, (a.T + G - 1) / G, 1 << 30);
    for (int j0 = 0; j0 < a.c; j0 += kPh1MaxSites) {  // groups of at most 8 queries
        p.c = a.c - j0 < kPh1MaxSites ? a.c - j0 : kPh1MaxSites;
        p.queries = a.queries + (size_t)j0 * a.r;
        p.h_pre = static_cast<char *>(a.h_pre) + (size_t)j0 * p.site_stride * sizeof(Tout);
        p.lse_pre = a.lse_pre + (size_t)j0 * a.T;
        block_phase1_kernel<Tin, Tout><<<grid, kThreads, smem, s>>>(p);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

cudaError_t launch_block_phase1(const BlockPh1Args &a, cudaStream_t s) {
    if (a.in_dtype == kBF16)
        return a.pre_dtype == kBF16 ? launch_ph1_t<bf16, bf16>(a, s) : launch_ph1_t<bf16, float>(a, s);
    return a.pre_dtype == kBF16 ? launch_ph1_t<float, bf16>(a, s) : launch_ph1_t<float, float>(a, s);
}

template <typename Tin, typename Tp, typename Tout, int V>
static cudaError_t launch_ph2_t(const BlockPh2Args &a, cudaStream_t s) {
    Ph2Params p;
    p.h_pre = a.h_pre;
    p.partial = a.partial;
    p.pkeys = a.pkeys;
    p.lse_pre = a.lse_pre;
    p.query = a.query;
    p.h = a.h;
    p.lse = a.lse;
    p.T = a.T;
    p.d = a.d;
    p.r = a.r;
    p.eps = a.eps;
    p.inv_r = 1.f / (float)a.r;
    p.sliced = a.variant == kSliced;
    const void *k = (const void *)block_phase2_kernel<Tin, Tp, Tout, V>;
    const int grid = persistent_grid(k, kThreads, 0, (a.T + kWarps - 1) / kWarps, 1 << 30);
    block_phase2_kernel<Tin, Tp, Tout, V><<<grid, kThreads, 0, s>>>(p);
    return cudaGetLastError();
}

template <typename Tin, typename Tp, typename Tout>
static cudaError_t launch_ph2_w(const BlockPh2Args &a, cudaStream_t s) {
    constexpr int E = VecE<Tin>::value;
    const int vecs = (a.d + E - 1) / E;
    if (vecs <= 32) return launch_ph2_t<Tin, Tp, Tout, 1>(a, s);
    if (vecs <= 64) return launch_ph2_t<Tin, Tp, Tout, 2>(a, s);
    if (vecs <= 128) return launch_ph2_t<Tin, Tp, Tout, 4>(a, s);
    return launch_ph2_t<Tin, Tp, Tout, 8>(a, s);
}

template <typename Tin, typename Tp>
static cudaError_t launch_ph2_o(const BlockPh2Args &a, cudaStream_t s) {
    return a.out_dtype == kBF16 ? launch_ph2_w<Tin, Tp, bf16>(a, s) : launch_ph2_w<Tin, Tp, float>(a, s);
}

cudaError_t launch_block_phase2(const BlockPh2Args &a, cudaStream_t s) {
    if (a.in_dtype == kBF16)
        return a.pre_dtype == kBF16 ? launch_ph2_o<bf16, bf16>(a, s) : launch_ph2_o<bf16, float>(a, s);
    return a.pre_dtype == kBF16 ? launch_ph2_o<float, bf16>(a, s) : launch_ph2_o<float, float>(a, s);
}

}  // namespace lrar
