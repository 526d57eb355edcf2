// lrar_fwd.cu -- forward depth-attention mix, Eq. (8)-(10) of arxiv 2607.09694.
//
// One warp owns one token row at a time (grid-stride over tokens, persistent
// grid sized to the resident CTAs of the device).  Lane l holds the 16-byte
// vectors l, l+32, ... of the row, so every load instruction of a warp covers
// 512 contiguous bytes of one source row.
//
// Low-rank keys (SLICED, PROJECTED): a routing stage reads the n r-dim keys
// (lane i scores source i), takes the softmax with two warp reductions and
// leaves alpha in shared memory; the value stage then streams the n full-width
// value rows once and accumulates in fp32 registers.
//
// Full keys (AttnRes, r = d): the key is the whole value row, so the score of a
// source is known only once its row is loaded.  The kernel streams each row
// once with an online softmax (running max, rescaled accumulator), so the
// values are read exactly once.
#include "lrar_device.cuh"
#include "lrar_launch.h"

namespace lrar {

struct FwdParams {
    SrcTab vt, kt;  // value and P-LR key tables
    const float *query;
    void *h;
    float *lse;
    int64_t T;
    int n, d, r;
    float eps, inv_r;
    int sliced;   // key = last r coordinates of the value row
    int key_vec;  // keys can be read as aligned 16-byte vectors
    int chunks;   // warps per token row (low-rank forward): each mixes one 32 x V-vector chunk
};

// Staged keys in shared memory: key i of a token occupies `per` = r / E
// 16-byte cells from cell i * per, piece c stored at cell i * per + key_swz(i, c).
// The routing lane of source i reads the pieces of key i one at a time; the
// swizzle spreads the eight lanes of a 16-byte access phase over all banks
// (a power-of-two per; other widths are stored in order).
__device__ __forceinline__ int key_swz(int i, int c, int per) {
    if (per & (per - 1)) return c;
    return per >= 8 ? c ^ (i & 7) : c ^ ((i * per >> 3) & (per - 1));
}

// sum_j k_j^2 and sum_j q_j k_j of one key of r elements.
// With sw >= 0, kp points at a key staged in shared memory by stage_keys for
// source sw, its pieces in key_swz order.
template <typename Tin>
__device__ __forceinline__ void key_stats(const Tin *__restrict__ kp, int r, const float *__restrict__ q_s,
                                          bool vec, float &ss, float &qk, int sw = -1) {
    ss = 0.f;
    qk = 0.f;
    if (vec) {
        constexpr int E = VecE<Tin>::value;
        for (int j = 0; j < r; j += E) {
            Frag<Tin, E> f;
            if (sw >= 0) f.a = *reinterpret_cast<const uint4 *>(kp + key_swz(sw, j / E, r / E) * E);
            else f.load_nc(kp + j);
            float k[E];
            f.get(k);
#pragma unroll
            for (int t = 0; t < E; ++t) {
                ss = fmaf(k[t], k[t], ss);
                qk = fmaf(q_s[j + t], k[t], qk);
            }
        }
    } else {
        for (int j = 0; j < r; ++j) {
            const float k = to_f(__ldg(kp + j));
            ss = fmaf(k, k, ss);
            qk = fmaf(q_s[j], k, qk);
        }
    }
}

// Routing stage for token x (Eq. 8-9): lane owns sources lane + 32k.
// Leaves alpha_i in a_s[i] (and s_i, rho_i in s_s, rho_s when non-null);
// returns lse = log sum_i exp(s_i) in every lane.
// With kb_s, the token's keys are read from that shared buffer [n][r] (filled
// by stage_keys) instead of global memory.
template <typename Tin>
__device__ __forceinline__ float lr_route(const SrcTab &vt, const SrcTab &kt, int n, int d, int r, float eps,
                                          float inv_r, int sliced, int key_vec,
                                          int64_t x, int lane, const float *__restrict__ q_s, float *a_s, float *s_s,
                                          float *rho_s, const Tin *kb_s = nullptr) {
    float s_reg[kSrcRegs];
    float m = -INFINITY;
#pragma unroll
    for (int k = 0; k < kSrcRegs; ++k) {
        const int i = lane + 32 * k;
        float s = -INFINITY;
        if (i < n) {
            float ss, qk;
            if (kb_s) {
                key_stats<Tin>(kb_s + i * r, r, q_s, true, ss, qk, i);
            } else {
                const Tin *kp = sliced ? src_row<Tin>(vt, i, x, d) + (d - r) : src_row<Tin>(kt, i, x, r);
                key_stats<Tin>(kp, r, q_s, key_vec != 0, ss, qk);
            }
            const float rho = rsqrtf(fmaf(ss, inv_r, eps));
            s = rho * qk;
            if (s_s) {
                s_s[i] = s;
                rho_s[i] = rho;
            }
        }
        s_reg[k] = s;
        m = fmaxf(m, s);
    }
    m = warp_max(m);
    float z = 0.f;
#pragma unroll
    for (int k = 0; k < kSrcRegs; ++k) {
        const int i = lane + 32 * k;
        const float e = (i < n) ? expf(s_reg[k] - m) : 0.f;
        s_reg[k] = e;
        z += e;
    }
    z = warp_sum(z);
    const float inv_z = 1.f / z;
#pragma unroll
    for (int k = 0; k < kSrcRegs; ++k) {
        const int i = lane + 32 * k;
        if (i < n) a_s[i] = s_reg[k] * inv_z;
    }
    return m + logf(z);
}

template <typename Tin, typename Tout, int V>
__device__ __forceinline__ void store_row(Tout *__restrict__ hrow, int d, int lane, const float *acc, float scale) {
    constexpr int E = VecE<Tin>::value;
#pragma unroll
    for (int v = 0; v < V; ++v) {
        const int e = (lane + 32 * v) * E;
        if (e < d) {
            float o[E];
#pragma unroll
            for (int t = 0; t < E; ++t) o[t] = acc[v * E + t] * scale;
            Frag<Tout, E> f;
            f.set(o);
            f.store(hrow + e);
        }
    }
}

// Copy the n keys of token x (aligned 16-byte vectors) into the warp's shared
// buffer kbuf with cp.async, one commit group; consecutive lanes take
// consecutive pieces, so each instruction covers whole keys.  The caller waits
// and syncs the warp before the routing lanes read them.
template <typename Tin>
__device__ __forceinline__ void stage_keys(const SrcTab &vt, const SrcTab &kt, int n, int d, int r, int sliced,
                                           int64_t x, int lane, uint32_t kbuf) {
    constexpr int E = VecE<Tin>::value;
    const int per = r / E;
    const bool pow2 = (per & (per - 1)) == 0;
    const int sh = 31 - __clz(per);
    for (int j = lane; j < n * per; j += 32) {
        const int i = pow2 ? j >> sh : j / per, c = j - i * per;
        const Tin *src = (sliced ? src_row<Tin>(vt, i, x, d) + (d - r) : src_row<Tin>(kt, i, x, r)) + c * E;
        cp_async16(kbuf + 16u * (uint32_t)(i * per + key_swz(i, c, per)), src);
    }
    cp_async_commit();
}

// ------------------------------------------------- low-rank keys (LR) ----
// KS: each warp stages its next token's keys in shared memory with cp.async
// while it mixes the current token's last rows (kPrefetchRows before the end),
// so the routing reads no global memory on its critical path.
constexpr int kPrefetchRows = 8;

template <typename Tin, typename Tout, int V, int U, bool KS>
__global__ void __launch_bounds__(kThreads, (V <= 4 ? 2 : 1)) fwd_lr_kernel(const __grid_constant__ FwdParams p) {
    pdl_enter();
    constexpr int E = VecE<Tin>::value;
    extern __shared__ float smem[];
    float *q_s = smem;                                         // [r]
    float *a_all = smem + round_up(p.r, 4);                    // [kWarps][kMaxSources]
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    float *a_s = a_all + warp * kMaxSources;
    const int kb_elems = round_up(p.n * p.r, 16 / (int)sizeof(Tin));  // per warp, whole 16-byte cells
    Tin *kb_s = reinterpret_cast<Tin *>(a_all + kWarps * kMaxSources) + warp * kb_elems;
    for (int j = threadIdx.x; j < p.r; j += kThreads) q_s[j] = p.query ? p.query[j] : 0.f;
    __syncthreads();

    const int64_t nwarps = (int64_t)gridDim.x * kWarps;
    const int64_t items = p.T * p.chunks;

    // item = (token, chunk): rows wider than one warp's V vectors are split
    // across warps, each of which recomputes the (cheap) routing of its token
    const uint32_t kbuf = smem_u32(kb_s);
    const int pf_at = p.n > kPrefetchRows ? (p.n - kPrefetchRows) / U * U : 0;
    if (KS && (int64_t)blockIdx.x * kWarps + warp < items)
        stage_keys<Tin>(p.vt, p.kt, p.n, p.d, p.r, p.sliced, ((int64_t)blockIdx.x * kWarps + warp) / p.chunks,
                        lane, kbuf);
    for (int64_t it = (int64_t)blockIdx.x * kWarps + warp; it < items; it += nwarps) {
        const int64_t x = it / p.chunks;
        const int e0 = (int)(it - x * p.chunks) * 32 * V * E;  // first element of this chunk
        const int dc = p.d - e0;                               // elements from the chunk start to the row end
        if (KS) {
            cp_async_wait_all();
            __syncwarp();  // every lane's pieces are visible to the warp
        }
        // the token's first rows do not depend on the weights: their loads go out
        // before the routing, so the two latencies overlap
        const int pre = p.n < U ? p.n : U;
        Frag<Tin, E> f0[U][V];
#pragma unroll
        for (int u = 0; u < U; ++u)
#pragma unroll
            for (int v = 0; v < V; ++v) {
                const int e = (lane + 32 * v) * E;
                if (u < pre && e < dc) f0[u][v].load_nc(src_row<Tin>(p.vt, u, x, p.d) + e0 + e);
                else f0[u][v].zero();
            }
        const float lse = lr_route<Tin>(p.vt, p.kt, p.n, p.d, p.r, p.eps, p.inv_r, p.sliced, p.key_vec, x,
                                        lane, q_s, a_s, nullptr, nullptr, KS ? kb_s : nullptr);
        if (lane == 0 && p.lse && e0 == 0) p.lse[x] = lse;
        __syncwarp();  // a_s written; kb_s free for the next token
        bool staged = !KS || it + nwarps >= items;
        auto stage_next = [&]() {
            stage_keys<Tin>(p.vt, p.kt, p.n, p.d, p.r, p.sliced, (it + nwarps) / p.chunks, lane, kbuf);
            staged = true;
        };

        // Eq. (10): h = sum_i alpha_i o_i, fp32 accumulation.
        float acc[V * E];
#pragma unroll
        for (int t = 0; t < V * E; ++t) acc[t] = 0.f;
#pragma unroll
        for (int u = 0; u < U; ++u) {
            if (u < pre) {
                const float a = a_s[u];
#pragma unroll
                for (int v = 0; v < V; ++v) {
                    float o[E];
                    f0[u][v].get(o);
#pragma unroll
                    for (int t = 0; t < E; ++t) acc[v * E + t] = fmaf(a, o[t], acc[v * E + t]);
                }
            }
        }
        int i = pre;
        if (!staged && pf_at < i) stage_next();  // the staging point falls among the preloaded rows
        for (; i + U <= p.n; i += U) {
            if (!staged && i == pf_at) stage_next();
            Frag<Tin, E> f[U][V];
#pragma unroll
            for (int u = 0; u < U; ++u)
#pragma unroll
                for (int v = 0; v < V; ++v) {
                    const int e = (lane + 32 * v) * E;
                    if (e < dc) f[u][v].load_nc(src_row<Tin>(p.vt, i + u, x, p.d) + e0 + e);
                    else f[u][v].zero();
                }
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const float a = a_s[i + u];
#pragma unroll
                for (int v = 0; v < V; ++v) {
                    float o[E];
                    f[u][v].get(o);
#pragma unroll
                    for (int t = 0; t < E; ++t) acc[v * E + t] = fmaf(a, o[t], acc[v * E + t]);
                }
            }
        }
        for (; i < p.n; ++i) {
            const float a = a_s[i];
#pragma unroll
            for (int v = 0; v < V; ++v) {
                const int e = (lane + 32 * v) * E;
                Frag<Tin, E> f;
                if (e < dc) f.load_nc(src_row<Tin>(p.vt, i, x, p.d) + e0 + e);
                else f.zero();
                float o[E];
                f.get(o);
#pragma unroll
                for (int t = 0; t < E; ++t) acc[v * E + t] = fmaf(a, o[t], acc[v * E + t]);
            }
        }
        if (!staged) stage_next();
        store_row<Tin, Tout, V>(static_cast<Tout *>(p.h) + x * p.d + e0, dc, lane, acc, 1.f);
        __syncwarp();  // a_s is rewritten for the next token
    }
    if (KS) cp_async_wait_all();
}

// ------------------------------------------------------- full keys -------
template <typename Tin, int V>
__device__ __forceinline__ void full_row_step(const Frag<Tin, VecE<Tin>::value> *f, const float *__restrict__ q_s,
                                              int lane, float inv_d, float eps, float &m, float &z, float *acc) {
    constexpr int E = VecE<Tin>::value;
    float o[V * E];
    float ss = 0.f, qo = 0.f;
#pragma unroll
    for (int v = 0; v < V; ++v) f[v].get(o + v * E);
#pragma unroll
    for (int v = 0; v < V; ++v) {
        float qv[E];
        q_get<E>(q_s, v, lane, qv);  // q is zero past d
#pragma unroll
        for (int t = 0; t < E; ++t) {
            if constexpr (V * E <= 32) {  // packed pairs pay where the row fits 32 values per lane
                fma2(ss, qo, o[v * E + t], qv[t], o[v * E + t], o[v * E + t]);  // o.o, q.o
            } else {
                ss = fmaf(o[v * E + t], o[v * E + t], ss);
                qo = fmaf(qv[t], o[v * E + t], qo);
            }
        }
    }
    ss = warp_sum(ss);
    qo = warp_sum(qo);
    const float s = rsqrtf(fmaf(ss, inv_d, eps)) * qo;  // Eq. (2) with RMSNorm(o_i) as the key
    if (s > m) {                                        // warp-uniform: s is identical in all lanes
        const float c = expf(m - s);
        z *= c;
#pragma unroll
        for (int t = 0; t < V * E; ++t) acc[t] *= c;
        m = s;
    }
    const float w = expf(s - m);
    z += w;
    if constexpr (V * E <= 32) {
#pragma unroll
        for (int t = 0; t < V * E; t += 2) fma2(acc[t], acc[t + 1], w, w, o[t], o[t + 1]);
    } else {
#pragma unroll
        for (int t = 0; t < V * E; ++t) acc[t] = fmaf(w, o[t], acc[t]);
    }
}

// One warp per token; each lane streams its own 16-byte vectors of the source
// rows through a per-lane cp.async ring in shared memory (it reads back only
// what it copied, so the wait_group alone orders the two), S - 1 rows ahead.
// The ring runs across tokens: the next token's first rows travel while this
// one finishes.  Scores and the mix use the online softmax of full_row_step.
template <typename Tin, typename Tout, int V, int S>
__global__ void __launch_bounds__(kThreads, (V * VecE<Tin>::value <= 32 ? 2 : 1))
    fwd_full_kernel(const __grid_constant__ FwdParams p) {
    pdl_enter();
    constexpr int E = VecE<Tin>::value;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    float *q_s = reinterpret_cast<float *>(smem_raw + (size_t)kWarps * S * V * 32 * 16);  // [32 V E] (q_slot), zero past d
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int j = threadIdx.x; j < 32 * V * E; j += kThreads) q_s[q_slot<E>(j)] = (p.query && j < p.d) ? p.query[j] : 0.f;
    __syncthreads();
    const uint32_t ring_w = smem_u32(smem_raw) + (uint32_t)(warp * S * V * 32 * 16) + 16u * lane;
    const int64_t nwarps = (int64_t)gridDim.x * kWarps;
    const float inv_d = 1.f / (float)p.d;
    const int64_t x0 = (int64_t)blockIdx.x * kWarps + warp;

    int64_t ix = x0;  // next row to copy: source ii of token ix
    int ii = 0;
    auto cell = [&](int st, int v) -> uint32_t { return ring_w + (uint32_t)((st * V + v) * 32 * 16); };
    auto issue = [&](int st) {
        if (ix < p.T) {
            const Tin *row = src_row<Tin>(p.vt, ii, ix, p.d);
#pragma unroll
            for (int v = 0; v < V; ++v) {
                const int e = (lane + 32 * v) * E;
                if (e < p.d) cp_async16(cell(st, v), row + e);
            }
            if (++ii == p.n) {
                ii = 0;
                ix += nwarps;
            }
        }
        cp_async_commit();
    };
#pragma unroll
    for (int st = 0; st < S - 1; ++st) issue(st);
    int st_c = 0, st_i = S - 1;

    for (int64_t x = x0; x < p.T; x += nwarps) {
        float acc[V * E];
#pragma unroll
        for (int t = 0; t < V * E; ++t) acc[t] = 0.f;
        float m = -INFINITY, z = 0.f;
        for (int i = 0; i < p.n; ++i) {
            issue(st_i);
            cp_async_wait<S - 1>();  // this lane's copies of row i have landed
            Frag<Tin, E> f[V];
#pragma unroll
            for (int v = 0; v < V; ++v) {
                const int e = (lane + 32 * v) * E;
                if (e < p.d) f[v].a = ld_shared16(cell(st_c, v));
                else f[v].zero();
            }
            full_row_step<Tin, V>(f, q_s, lane, inv_d, p.eps, m, z, acc);
            st_c = (st_c + 1 == S) ? 0 : st_c + 1;
            st_i = (st_i + 1 == S) ? 0 : st_i + 1;
        }
        store_row<Tin, Tout, V>(static_cast<Tout *>(p.h) + x * p.d, p.d, lane, acc, 1.f / z);
        if (lane == 0 && p.lse) p.lse[x] = m + logf(z);
    }
    cp_async_wait_all();
}

// ------------------------------------------------------------- launch ----
static void fill_tables(FwdParams &p, const FwdArgs &a) {
    for (int i = 0; i < kMaxTab; ++i) {
        p.vt.p[i] = i < a.n ? a.values[i] : nullptr;
        p.kt.p[i] = (i < a.n && a.keys) ? a.keys[i] : nullptr;
    }
}

#ifndef LRAR_STAGE_KEYS
#define LRAR_STAGE_KEYS 1
#endif
constexpr bool kStageKeys = LRAR_STAGE_KEYS;
constexpr size_t kStageKeyBytes = 12 * 1024;  // per warp

template <typename Tin, typename Tout, int V>
static cudaError_t launch_fwd_t(const FwdArgs &a, cudaStream_t s, int chunks = 1) {
    constexpr int U = V >= 8 ? 1 : (V == 4 ? 2 : 4);
    FwdParams p;
    fill_tables(p, a);
    p.query = a.query;
    p.h = a.h;
    p.lse = a.lse;
    p.T = a.T;
    p.n = a.n;
    p.d = a.d;
    p.r = a.r;
    p.eps = a.eps;
    p.inv_r = 1.f / (float)a.r;
    p.sliced = a.variant == kSliced;
    p.chunks = chunks;
    constexpr int esz = sizeof(Tin);
    if (a.variant == kSliced)
        p.key_vec = ((a.r * esz) % 16 == 0) && (((a.d - a.r) * esz) % 16 == 0);
    else
        p.key_vec = (a.r * esz) % 16 == 0;  // every key matrix is 16-byte aligned (checked by the API)
    const int64_t work = (a.T * chunks + kWarps - 1) / kWarps;
    if (a.variant == kFull) {
        constexpr int S = FullStages<V, 1, 24>::value;
        const size_t smem = (size_t)kWarps * S * V * 32 * 16 + sizeof(float) * 32 * V * VecE<Tin>::value;
        const void *k = (const void *)fwd_full_kernel<Tin, Tout, V, S>;
        if (smem > 48 * 1024) {
            cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            if (e != cudaSuccess) return e;
        }
        const int grid = persistent_grid(k, kThreads, smem, work, 1 << 30);
        launch_pdl(fwd_full_kernel<Tin, Tout, V, S>, grid, kThreads, smem, s, p);
    } else {
        // Keys staged in shared memory when rows are split over warps (each warp
        // routes its token, so routing weighs twice as much), the keys are whole
        // aligned vectors and a warp's buffer leaves room for two CTAs per SM.
        // At one warp per row staging measured neutral to slightly slower.
        const size_t kb = (size_t)round_up(a.n * a.r, 16 / esz) * esz;
        const bool ks = kStageKeys && chunks > 1 && p.key_vec && kb <= kStageKeyBytes;
        const size_t smem = sizeof(float) * (round_up(a.r, 4) + kWarps * kMaxSources) + (ks ? kWarps * kb : 0);
        const void *k = ks ? (const void *)fwd_lr_kernel<Tin, Tout, V, U, true>
                           : (const void *)fwd_lr_kernel<Tin, Tout, V, U, false>;
        if (smem > 48 * 1024) {
            cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            if (e != cudaSuccess) return e;
        }
        const int grid = persistent_grid(k, kThreads, smem, work, 1 << 30);
        if (ks) launch_pdl(fwd_lr_kernel<Tin, Tout, V, U, true>, grid, kThreads, smem, s, p);
        else launch_pdl(fwd_lr_kernel<Tin, Tout, V, U, false>, grid, kThreads, smem, s, p);
    }
    return cudaGetLastError();
}

template <typename Tin, typename Tout>
static cudaError_t launch_fwd_w(const FwdArgs &a, cudaStream_t s) {
    constexpr int E = VecE<Tin>::value;
    const int vecs = (a.d + E - 1) / E;  // 16-byte vectors per row
    if (vecs <= 32) return launch_fwd_t<Tin, Tout, 1>(a, s);
    if (vecs <= 64) return launch_fwd_t<Tin, Tout, 2>(a, s);
    if (vecs <= 128) return launch_fwd_t<Tin, Tout, 4>(a, s);
    if (a.variant != kFull) return launch_fwd_t<Tin, Tout, 4>(a, s, (vecs + 127) / 128);  // rows split over warps
    return launch_fwd_t<Tin, Tout, 8>(a, s);
}

// ------------------------------------------------- routing diagnostics ----
// §4.5-4.6: per token, N_eff = exp(H(alpha)) with H = -sum_i alpha_i log alpha_i
// (Eq. 16, 0 log 0 = 0); per site, alpha averaged over the T tokens.  Routing is
// that of the forward (low-rank keys: lr_route; full keys: each value row is
// read once for its score).  Each CTA writes one row of mean partials (already
// divided by T) for a fixed-order sum.
template <typename Tin, int V>
__global__ void __launch_bounds__(kThreads)
    diag_kernel(const __grid_constant__ FwdParams p, float *neff, float *partials, int full) {
    pdl_enter();
    constexpr int E = VecE<Tin>::value;
    extern __shared__ float smem[];
    float *q_s = smem;                                    // [r]
    float *a_all = smem + round_up(p.r, 4);               // [kWarps][kMaxSources]
    float *m_all = a_all + kWarps * kMaxSources;          // [kWarps][kMaxSources] running mean
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    float *a_s = a_all + warp * kMaxSources;
    float *m_s = m_all + warp * kMaxSources;
    for (int j = threadIdx.x; j < p.r; j += kThreads) q_s[j] = p.query ? p.query[j] : 0.f;
    for (int j = threadIdx.x; j < kWarps * kMaxSources; j += kThreads) m_all[j] = 0.f;
    __syncthreads();

    const int64_t nwarps = (int64_t)gridDim.x * kWarps;
    const float inv_T = 1.f / (float)p.T;
    for (int64_t x = (int64_t)blockIdx.x * kWarps + warp; x < p.T; x += nwarps) {
        if (!full) {
            lr_route<Tin>(p.vt, p.kt, p.n, p.d, p.r, p.eps, p.inv_r, p.sliced, p.key_vec, x, lane, q_s, a_s,
                          nullptr, nullptr);
        } else {
            for (int i = 0; i < p.n; ++i) {  // score of source i from its whole row (r = d)
                const Tin *row = src_row<Tin>(p.vt, i, x, p.d);
                float ss = 0.f, qo = 0.f;
#pragma unroll
                for (int v = 0; v < V; ++v) {
                    const int e = (lane + 32 * v) * E;
                    if (e < p.d) {
                        Frag<Tin, E> f;
                        f.load_nc(row + e);
                        float o[E];
                        f.get(o);
#pragma unroll
                        for (int t = 0; t < E; ++t) {
                            ss = fmaf(o[t], o[t], ss);
                            qo = fmaf(q_s[e + t], o[t], qo);
                        }
                    }
                }
                ss = warp_sum(ss);
                qo = warp_sum(qo);
                if (lane == 0) a_s[i] = rsqrtf(fmaf(ss, p.inv_r, p.eps)) * qo;  // score, softmax below
            }
            __syncwarp();
            float m = -INFINITY;
            for (int i = lane; i < p.n; i += 32) m = fmaxf(m, a_s[i]);
            m = warp_max(m);
            float z = 0.f;
            for (int i = lane; i < p.n; i += 32) z += expf(a_s[i] - m);
            z = warp_sum(z);
            __syncwarp();
            for (int i = lane; i < p.n; i += 32) a_s[i] = expf(a_s[i] - m) / z;
        }
        __syncwarp();
        float hp = 0.f;
        for (int i = lane; i < p.n; i += 32) {
            const float a = a_s[i];
            if (a > 0.f) hp -= a * logf(a);
            m_s[i] = fmaf(a, inv_T, m_s[i]);  // coordinate i belongs to this lane alone
        }
        const float H = warp_sum(hp);
        if (lane == 0 && neff) neff[x] = expf(H);
        __syncwarp();
    }
    __syncthreads();
    if (partials)
        for (int i = threadIdx.x; i < p.n; i += kThreads) {
            float acc = 0.f;
#pragma unroll
            for (int w = 0; w < kWarps; ++w) acc += m_all[w * kMaxSources + i];
            partials[(int64_t)blockIdx.x * p.n + i] = acc;
        }
}

template <typename Tin, int V>
static cudaError_t launch_diag_t(const FwdArgs &a, float *neff, float *mean_alpha, float *partials, cudaStream_t s) {
    FwdParams p;
    fill_tables(p, a);
    p.query = a.query;
    p.h = nullptr;
    p.lse = nullptr;
    p.T = a.T;
    p.n = a.n;
    p.d = a.d;
    p.r = a.r;
    p.eps = a.eps;
    p.inv_r = 1.f / (float)a.r;
    p.sliced = a.variant == kSliced;
    p.chunks = 1;
    constexpr int esz = sizeof(Tin);
    if (a.variant == kSliced)
        p.key_vec = ((a.r * esz) % 16 == 0) && (((a.d - a.r) * esz) % 16 == 0);
    else
        p.key_vec = (a.r * esz) % 16 == 0;  // every key matrix is 16-byte aligned (checked by the API)
    const size_t smem = sizeof(float) * (round_up(a.r, 4) + 2 * kWarps * kMaxSources);
    const void *k = (const void *)diag_kernel<Tin, V>;
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
    }
    const int grid = persistent_grid(k, kThreads, smem, (a.T + kWarps - 1) / kWarps, kMaxPartials);
    launch_pdl(diag_kernel<Tin, V>, grid, kThreads, smem, s, p, neff, mean_alpha ? partials : nullptr, a.variant == kFull);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess || !mean_alpha) return e;
    return launch_partial_sum(partials, grid, a.n, mean_alpha, 0, s);
}

template <typename Tin>
static cudaError_t launch_diag_w(const FwdArgs &a, float *neff, float *mean_alpha, float *partials, cudaStream_t s) {
    constexpr int E = VecE<Tin>::value;
    const int vecs = (a.d + E - 1) / E;
    if (vecs <= 32) return launch_diag_t<Tin, 1>(a, neff, mean_alpha, partials, s);
    if (vecs <= 64) return launch_diag_t<Tin, 2>(a, neff, mean_alpha, partials, s);
    if (vecs <= 128) return launch_diag_t<Tin, 4>(a, neff, mean_alpha, partials, s);
    return launch_diag_t<Tin, 8>(a, neff, mean_alpha, partials, s);
}

cudaError_t launch_diagnostics(const FwdArgs &a, float *neff, float *mean_alpha, float *partials, cudaStream_t s) {
    return a.in_dtype == kBF16 ? launch_diag_w<bf16>(a, neff, mean_alpha, partials, s)
                               : launch_diag_w<float>(a, neff, mean_alpha, partials, s);
}

cudaError_t launch_forward(const FwdArgs &a, cudaStream_t s) {
    if (a.in_dtype == kBF16)
        return a.out_dtype == kBF16 ? launch_fwd_w<bf16, bf16>(a, s) : launch_fwd_w<bf16, float>(a, s);
    return a.out_dtype == kBF16 ? launch_fwd_w<float, bf16>(a, s) : launch_fwd_w<float, float>(a, s);
}

}  // namespace lrar
