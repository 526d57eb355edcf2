// lrar_bwd.cu -- backward of the depth-attention mix (chain rule through
// Eq. 8-10 of arxiv 2607.09694; the paper prints no gradient formulas):
//
//   g_i = <dh, o_i>,  gbar = sum_i alpha_i g_i,  ds_i = alpha_i (g_i - gbar)
//   dL/do_i = alpha_i dh,   dL/dq = sum ds_i kbar_i
//   dL/dk_i = ds_i rho_i (q - (s_i / r) kbar_i),   rho_i = (mean k_i^2 + eps)^-1/2
//
// Every value row is read once and every gradient row written once.
//
// Low-rank keys: (1) the routing stage recomputes s, rho, alpha from the r-dim
// keys; (2) the value pass streams o_i, forms g_i with a warp reduction and
// writes dL/do_i = alpha_i dh (+ the old value when accumulating) for every
// 16-byte vector that does not lie wholly in the key slice; (3) the key pass,
// with gbar known, forms ds_i and dL/dk_i lane-per-key-coordinate, writes the
// key slice of dvalues (SLICED: alpha_i dh + dL/dk_i in one rounding) or dkeys
// (PROJECTED), and accumulates dq.  Sliced keys with the forward's lse and
// written gradients skip (1) and fold (3) into the same pass
// (bwd_slr_onepass_kernel): alpha_i = exp(s_i - lse) from the row's own slice.
//
// Full keys (r = d): ds_i needs gbar before row i can be written, and gbar =
// <dh, h> because h = sum_i alpha_i o_i, so a single pass needs the forward's
// h and lse: per row, three warp reductions (g_i, |o_i|^2, q.o_i) give s_i,
// rho_i, alpha_i = exp(s_i - lse), ds_i, and the whole gradient row
//   alpha_i dh + ds_i rho_i q - ds_i rho_i^2 (s_i / d) o_i.
//
// dq: each warp accumulates its tokens, each CTA writes one partial row to the
// workspace, and a second kernel sums the partials in CTA order, so dq is
// bitwise reproducible on a given device.
#include <type_traits>

#include "lrar.h"
#include "lrar_bwd.cuh"
#include "lrar_device.cuh"
#include "lrar_launch.h"

namespace lrar {

// Routing stage, identical arithmetic to the forward's (see lrar_fwd.cu).
template <typename Tin>
__device__ __forceinline__ void key_stats_b(const Tin *__restrict__ kp, int r, const float *__restrict__ q_s,
                                            bool vec, float &ss, float &qk) {
    ss = 0.f;
    qk = 0.f;
    if (vec) {
        constexpr int E = VecE<Tin>::value;
        for (int j = 0; j < r; j += E) {
            Frag<Tin, E> f;
            f.load_nc(kp + j);
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

template <typename Tin>
__device__ __forceinline__ void lr_route_b(const BwdParams &p, int64_t x, int lane, const float *__restrict__ q_s,
                                           float *a_s, float *s_s, float *rho_s) {
    float s_reg[kSrcRegs];
    float m = -INFINITY;
#pragma unroll
    for (int k = 0; k < kSrcRegs; ++k) {
        const int i = lane + 32 * k;
        float s = -INFINITY;
        if (i < p.n) {
            const Tin *kp = p.sliced ? src_row<Tin>(p.vt, i, x, p.d) + (p.d - p.r) : src_row<Tin>(p.kt, i, x, p.r);
            float ss, qk;
            key_stats_b<Tin>(kp, p.r, q_s, p.key_vec != 0, ss, qk);
            const float rho = rsqrtf(fmaf(ss, p.inv_r, p.eps));
            s = rho * qk;
            s_s[i] = s;
            rho_s[i] = rho;
        }
        s_reg[k] = s;
        m = fmaxf(m, s);
    }
    m = warp_max(m);
    float z = 0.f;
#pragma unroll
    for (int k = 0; k < kSrcRegs; ++k) {
        const int i = lane + 32 * k;
        const float e = (i < p.n) ? expf(s_reg[k] - m) : 0.f;
        s_reg[k] = e;
        z += e;
    }
    z = warp_sum(z);
    const float inv_z = 1.f / z;
#pragma unroll
    for (int k = 0; k < kSrcRegs; ++k) {
        const int i = lane + 32 * k;
        if (i < p.n) a_s[i] = s_reg[k] * inv_z;
    }
}

// One value row of the low-rank backward (phase 2): returns the lane's part of g_i.
// Vectors wholly inside the key slice (e >= skip0) are left to the key pass; in
// the one vector that straddles the slice start (tail0), the slice elements keep
// their old value here and receive alpha_i dh + dL/dk_i in the key pass, so every
// element is rounded once.
template <typename Tin, typename Tg, int V, bool ACC>
__device__ __forceinline__ float lr_bwd_row(const Frag<Tin, VecE<Tin>::value> *f,
                                            const Frag<Tg, VecE<Tin>::value> *old,
                                            const Frag<Tin, VecE<Tin>::value> *dhr, float a, Tg *__restrict__ drow,
                                            int tail0, int skip0, int lane) {
    constexpr int E = VecE<Tin>::value;
    float gp = 0.f;
#pragma unroll
    for (int v = 0; v < V; ++v) {
        const int e = (lane + 32 * v) * E;
        float o[E], dhv[E];
        f[v].get(o);
        dhr[v].get(dhv);
#pragma unroll
        for (int t = 0; t < E; ++t) gp = fmaf(dhv[t], o[t], gp);
        if (e < skip0) {
            float w[E];
            if (ACC) old[v].get(w);
            else
#pragma unroll
                for (int t = 0; t < E; ++t) w[t] = 0.f;
            if (e + E <= tail0) {
#pragma unroll
                for (int t = 0; t < E; ++t) w[t] = fmaf(a, dhv[t], w[t]);
            } else {
#pragma unroll
                for (int t = 0; t < E; ++t)
                    if (e + t < tail0) w[t] = fmaf(a, dhv[t], w[t]);
            }
            Frag<Tg, E> out;
            out.set(w);
            out.store(drow + e);
        }
    }
    return gp;
}

template <typename Tin, typename Tg, int V, int U, bool ACC>
__global__ void __launch_bounds__(kThreads, (V <= 4 ? 2 : 1)) bwd_lr_kernel(const __grid_constant__ BwdParams p) {
    pdl_enter();
    constexpr int E = VecE<Tin>::value;
    extern __shared__ float smem[];
    const int rp = round_up(p.r, 4);
    float *q_s = smem;                                   // [r]
    float *dq_all = q_s + rp;                            // [kWarps][r]
    float *tab = dq_all + kWarps * rp;                   // [kWarps][4][kMaxSources]
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    float *dq_s = dq_all + warp * rp;
    float *a_s = tab + warp * 4 * kMaxSources;
    float *s_s = a_s + kMaxSources;
    float *rho_s = s_s + kMaxSources;
    float *g_s = rho_s + kMaxSources;  // g_i, then ds_i
    for (int j = threadIdx.x; j < p.r; j += kThreads) q_s[j] = p.query ? p.query[j] : 0.f;
    for (int j = threadIdx.x; j < kWarps * rp; j += kThreads) dq_all[j] = 0.f;
    __syncthreads();

    const Tin *__restrict__ dh = static_cast<const Tin *>(p.dh);
    const int64_t nwarps = (int64_t)gridDim.x * kWarps;
    const int tail0 = p.sliced ? p.d - p.r : p.d;  // first key coordinate inside the value row
    const int skip0 = round_up(tail0, E);          // vectors starting here lie wholly in the key slice

    for (int64_t x = (int64_t)blockIdx.x * kWarps + warp; x < p.T; x += nwarps) {
        // (1) routing: s_i, rho_i, alpha_i
        lr_route_b<Tin>(p, x, lane, q_s, a_s, s_s, rho_s);
        __syncwarp();

        // (2) value pass; dh stays packed in registers and widens per use
        Frag<Tin, E> dhr[V];
#pragma unroll
        for (int v = 0; v < V; ++v) {
            const int e = (lane + 32 * v) * E;
            if (e < p.d) dhr[v].load_nc(dh + x * p.d + e);
            else dhr[v].zero();
        }
        const int64_t row_off = x * p.d;
        const int wend = p.d < skip0 ? p.d : skip0;
        int i = 0;
        for (; i + U <= p.n; i += U) {
            Frag<Tin, E> f[U][V];
            Frag<Tg, E> old[U][V];
#pragma unroll
            for (int u = 0; u < U; ++u)
#pragma unroll
                for (int v = 0; v < V; ++v) {
                    const int e = (lane + 32 * v) * E;
                    if (e < p.d) f[u][v].load_nc(src_row<Tin>(p.vt, i + u, x, p.d) + e);
                    else f[u][v].zero();
                    if (ACC && e < skip0) old[u][v].load(dst_row<Tg>(p.dvt, i + u, x, p.d) + e);
                    else old[u][v].zero();
                }
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const float gp = lr_bwd_row<Tin, Tg, V, ACC>(f[u], old[u], dhr, a_s[i + u],
                                                             dst_row<Tg>(p.dvt, i + u, x, p.d), tail0, wend, lane);
                const float g = warp_sum(gp);
                if (lane == 0) g_s[i + u] = g;
            }
        }
        for (; i < p.n; ++i) {
            Frag<Tin, E> f[V];
            Frag<Tg, E> old[V];
#pragma unroll
            for (int v = 0; v < V; ++v) {
                const int e = (lane + 32 * v) * E;
                if (e < p.d) f[v].load_nc(src_row<Tin>(p.vt, i, x, p.d) + e);
                else f[v].zero();
                if (ACC && e < skip0) old[v].load(dst_row<Tg>(p.dvt, i, x, p.d) + e);
                else old[v].zero();
            }
            const float gp = lr_bwd_row<Tin, Tg, V, ACC>(f, old, dhr, a_s[i], dst_row<Tg>(p.dvt, i, x, p.d), tail0,
                                                         wend, lane);
            const float g = warp_sum(gp);
            if (lane == 0) g_s[i] = g;
        }
        __syncwarp();

        // (3) key pass: gbar, ds_i, dL/dk_i, dq
        float part = 0.f;
        for (int k = lane; k < p.n; k += 32) part = fmaf(a_s[k], g_s[k], part);
        const float gbar = warp_sum(part);
        __syncwarp();
        for (int k = lane; k < p.n; k += 32) g_s[k] = a_s[k] * (g_s[k] - gbar);
        __syncwarp();
        for (int j = lane; j < p.r; j += 32) {
            const float qj = q_s[j];
            const int c = tail0 + j;  // coordinate of key element j inside the value row (SLICED)
            const float dh_c = p.sliced ? to_f(__ldg(dh + row_off + c)) : 0.f;
            float dqj = 0.f;
#pragma unroll 4
            for (int k = 0; k < p.n; ++k) {
                const float rho = rho_s[k], s = s_s[k], ds = g_s[k];
                float kij;
                if (p.sliced) kij = to_f(__ldg(src_row<Tin>(p.vt, k, x, p.d) + c));
                else kij = to_f(__ldg(src_row<Tin>(p.kt, k, x, p.r) + j));
                const float kbar = rho * kij;
                const float dk = ds * rho * (qj - s * p.inv_r * kbar);
                dqj = fmaf(ds, kbar, dqj);
                if (p.sliced) {
                    // c < skip0: the value pass stored the old value (or 0) here
                    Tg *dp = dst_row<Tg>(p.dvt, k, x, p.d) + c;
                    const float base = (c < skip0 || p.accumulate) ? to_f(*dp) : 0.f;
                    *dp = from_f<Tg>(base + fmaf(a_s[k], dh_c, dk));
                } else {
                    Tg *dp = dst_row<Tg>(p.dkt, k, x, p.r) + j;
                    *dp = from_f<Tg>(p.accumulate ? to_f(*dp) + dk : dk);
                }
            }
            dq_s[j] += dqj;  // coordinate j belongs to this lane alone
        }
        __syncwarp();
    }
    __syncthreads();
    for (int j = threadIdx.x; j < p.r; j += kThreads) {
        float acc = 0.f;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) acc += dq_all[w * rp + j];
        p.partials[(int64_t)blockIdx.x * p.r + j] = acc;
    }
}

// Low-rank keys with a per-lane async-copy ring (gradient type = input type):
// the value pass reads rows of o (and, when accumulating, of the old gradient)
// from shared memory, filled by cp.async S - 1 rows ahead across token
// boundaries, so the loads in flight no longer drain between rows and cost no
// registers.  Routing and key pass are those of bwd_lr_kernel.
#ifndef LRAR_BWD_PIPE
#define LRAR_BWD_PIPE 1
#endif
#ifndef LRAR_KEY_BATCH
#define LRAR_KEY_BATCH 8
#endif
constexpr int kKeyBatch = LRAR_KEY_BATCH;  // key-pass loads a lane keeps in flight
#ifndef LRAR_VEC_KEYPASS
#define LRAR_VEC_KEYPASS 1
#endif
constexpr bool kVecKeyPass = LRAR_VEC_KEYPASS;
template <int V, bool ACC> struct BwdStages {
#ifdef LRAR_BWD_STAGES
    static constexpr int value = LRAR_BWD_STAGES;
#else
    static constexpr int value = V >= 8 ? (ACC ? 2 : 3) : (ACC ? 3 : 5);
#endif
};

// Key pass with 16-byte vectors, for keys that are whole aligned vectors
// (key_vec) and whose row of NV = r / E vectors divides 32: lane l owns vector
// jv = l mod NV of the key rows of sources l / NV, l / NV + 32 / NV, ...; it
// loads a key vector and an old-gradient vector per source, writes the new
// gradient vector, and keeps E dq parts that the lanes sharing jv combine with
// a fixed butterfly.  S-LR slices are vector-aligned here, so no element of
// the slice was touched by the value pass.
template <typename T, bool ACC>
__device__ __forceinline__ void key_pass_vec(const BwdParams &p, const T *__restrict__ dh, int64_t x, int lane,
                                             int tail0, const float *__restrict__ q_s, const float *a_s,
                                             const float *s_s, const float *rho_s, const float *ds_s, float *dq_s) {
    constexpr int E = VecE<T>::value;
    constexpr int B = 4;  // sources per batch and lane
    const int NV = p.r / E;
    const int jv = lane % NV, kst = 32 / NV;
    const int j0 = jv * E;
    const int64_t row_off = x * p.d;
    float dqv[E];
#pragma unroll
    for (int t = 0; t < E; ++t) dqv[t] = 0.f;
    for (int kb = lane / NV; kb < p.n; kb += kst * B) {
        Frag<T, E> kf[B], of[B];
#pragma unroll
        for (int m = 0; m < B; ++m) {
            const int k = kb + m * kst;
            if (k < p.n) {
                if (p.sliced) {
                    kf[m].load_nc(src_row<T>(p.vt, k, x, p.d) + tail0 + j0);
                    if (ACC) of[m].load(dst_row<T>(p.dvt, k, x, p.d) + tail0 + j0);
                    else of[m].zero();
                } else {
                    kf[m].load_nc(src_row<T>(p.kt, k, x, p.r) + j0);
                    if (ACC) of[m].load(dst_row<T>(p.dkt, k, x, p.r) + j0);
                    else of[m].zero();
                }
            }
        }
#pragma unroll
        for (int m = 0; m < B; ++m) {
            const int k = kb + m * kst;
            if (k < p.n) {
                const float rho = rho_s[k], s = s_s[k], ds = ds_s[k], a = a_s[k];
                const float c1 = ds * rho, c2 = s * p.inv_r;
                float kv[E], w[E], dhv[E];
                kf[m].get(kv);
                of[m].get(w);
                if (p.sliced) {  // dh of the slice, re-read from L1 per source
                    Frag<T, E> f;
                    f.a = __ldg(reinterpret_cast<const uint4 *>(dh + row_off + tail0 + j0));
                    f.get(dhv);
                }
#pragma unroll
                for (int t = 0; t < E; ++t) {
                    const float kbar = rho * kv[t];
                    const float dk = c1 * (q_s[j0 + t] - c2 * kbar);
                    dqv[t] = fmaf(ds, kbar, dqv[t]);
                    w[t] += p.sliced ? fmaf(a, dhv[t], dk) : dk;
                }
                Frag<T, E> out;
                out.set(w);
                if (p.sliced) out.store(dst_row<T>(p.dvt, k, x, p.d) + tail0 + j0);
                else out.store(dst_row<T>(p.dkt, k, x, p.r) + j0);
            }
        }
    }
#pragma unroll
    for (int t = 0; t < E; ++t) {
        float v = dqv[t];
        for (int off = NV; off < 32; off <<= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
        if (lane < NV) dq_s[j0 + t] += v;
    }
}

// Key pass of one token (low-rank keys), with ds_i already in ds_s: writes the
// key slice of dvalues (S-LR: old + alpha_i dh + dL/dk_i, one rounding) or the
// key gradients (P-LR), and adds sum_i ds_i kbar_i into dq_s.  When r divides
// 32 or is a multiple of 32, every lane works and keeps kKeyBatch (key, old
// gradient) loads in flight; lanes that share a coordinate combine their dq
// parts with a fixed butterfly.  Other widths take one coordinate per lane.
template <typename T, bool ACC>
__device__ __forceinline__ void key_pass(const BwdParams &p, const T *__restrict__ dh, int64_t x, int lane, int tail0,
                                         int skip0, const float *__restrict__ q_s, const float *a_s,
                                         const float *s_s, const float *rho_s, const float *ds_s, float *dq_s) {
    const int64_t row_off = x * p.d;
    const bool shared_j = (32 % p.r) == 0;  // 32/r lanes per coordinate
    const bool multi_j = (p.r % 32) == 0;   // r/32 coordinates per lane
    if (shared_j || multi_j) {
        const int kstep = shared_j ? 32 / p.r : 1;
        const int jn = shared_j ? 1 : p.r / 32;
        for (int t = 0; t < jn; ++t) {
            const int j = shared_j ? lane % p.r : lane + 32 * t;
            const float qj = q_s[j];
            const int c = tail0 + j;
            const float dh_c = p.sliced ? to_f(__ldg(dh + row_off + c)) : 0.f;
            const bool rd_old = p.sliced ? (c < skip0 || ACC) : ACC;
            float dqj = 0.f;
            for (int kb = shared_j ? lane / p.r : 0; kb < p.n; kb += kstep * kKeyBatch) {
                float kv[kKeyBatch], ov[kKeyBatch];
#pragma unroll
                for (int m = 0; m < kKeyBatch; ++m) {
                    const int k = kb + m * kstep;
                    kv[m] = ov[m] = 0.f;
                    if (k < p.n) {
                        if (p.sliced) {
                            kv[m] = to_f(__ldg(src_row<T>(p.vt, k, x, p.d) + c));
                            if (rd_old) ov[m] = to_f(dst_row<T>(p.dvt, k, x, p.d)[c]);
                        } else {
                            kv[m] = to_f(__ldg(src_row<T>(p.kt, k, x, p.r) + j));
                            if (rd_old) ov[m] = to_f(dst_row<T>(p.dkt, k, x, p.r)[j]);
                        }
                    }
                }
#pragma unroll
                for (int m = 0; m < kKeyBatch; ++m) {
                    const int k = kb + m * kstep;
                    if (k < p.n) {
                        const float rho = rho_s[k], s = s_s[k], ds = ds_s[k];
                        const float kbar = rho * kv[m];
                        const float dk = ds * rho * (qj - s * p.inv_r * kbar);
                        dqj = fmaf(ds, kbar, dqj);
                        if (p.sliced)
                            dst_row<T>(p.dvt, k, x, p.d)[c] = from_f<T>(ov[m] + fmaf(a_s[k], dh_c, dk));
                        else
                            dst_row<T>(p.dkt, k, x, p.r)[j] = from_f<T>(ov[m] + dk);
                    }
                }
            }
            if (shared_j) {  // lanes l and l ^ (r, 2r, ..., 16) share j: fixed-order butterfly
                for (int off = p.r; off < 32; off <<= 1) dqj += __shfl_xor_sync(0xffffffffu, dqj, off);
                if (lane < p.r) dq_s[j] += dqj;
            } else {
                dq_s[j] += dqj;
            }
        }
    } else {
        for (int j = lane; j < p.r; j += 32) {
            const float qj = q_s[j];
            const int c = tail0 + j;
            const float dh_c = p.sliced ? to_f(__ldg(dh + row_off + c)) : 0.f;
            float dqj = 0.f;
#pragma unroll 4
            for (int k = 0; k < p.n; ++k) {
                const float rho = rho_s[k], s = s_s[k], ds = ds_s[k];
                float kij;
                if (p.sliced) kij = to_f(__ldg(src_row<T>(p.vt, k, x, p.d) + c));
                else kij = to_f(__ldg(src_row<T>(p.kt, k, x, p.r) + j));
                const float kbar = rho * kij;
                const float dk = ds * rho * (qj - s * p.inv_r * kbar);
                dqj = fmaf(ds, kbar, dqj);
                if (p.sliced) {
                    T *dp = dst_row<T>(p.dvt, k, x, p.d) + c;
                    const float base = (c < skip0 || ACC) ? to_f(*dp) : 0.f;
                    *dp = from_f<T>(base + fmaf(a_s[k], dh_c, dk));
                } else {
                    T *dp = dst_row<T>(p.dkt, k, x, p.r) + j;
                    *dp = from_f<T>(ACC ? to_f(*dp) + dk : dk);
                }
            }
            dq_s[j] += dqj;
        }
    }
}

template <typename T, int V, int S, bool ACC, bool VK>
__global__ void __launch_bounds__(kThreads, V >= 8 ? 1 : 2) bwd_lr_pipe_kernel(const __grid_constant__ BwdParams p) {
    pdl_enter();
    constexpr int E = VecE<T>::value;
    constexpr int P = ACC ? 2 : 1;  // planes per stage: o, old gradient
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int rp = round_up(p.r, 4);
    uint4 *ring = reinterpret_cast<uint4 *>(smem_raw);  // [kWarps][S][P][V][32] cells
    float *q_s = reinterpret_cast<float *>(smem_raw + (size_t)kWarps * S * P * V * 32 * 16);
    float *dq_all = q_s + rp;             // [kWarps][r]
    float *tab = dq_all + kWarps * rp;    // [kWarps][4][kMaxSources]
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    float *dq_s = dq_all + warp * rp;
    float *a_s = tab + warp * 4 * kMaxSources;
    float *s_s = a_s + kMaxSources;
    float *rho_s = s_s + kMaxSources;
    float *g_s = rho_s + kMaxSources;  // g_i, then ds_i
    const uint32_t ring_w = smem_u32(ring + (size_t)warp * S * P * V * 32) + 16u * lane;
    for (int j = threadIdx.x; j < p.r; j += kThreads) q_s[j] = p.query ? p.query[j] : 0.f;
    for (int j = threadIdx.x; j < kWarps * rp; j += kThreads) dq_all[j] = 0.f;
    __syncthreads();

    const T *__restrict__ dh = static_cast<const T *>(p.dh);
    const int64_t nwarps = (int64_t)gridDim.x * kWarps;
    const int tail0 = p.sliced ? p.d - p.r : p.d;
    const int skip0 = round_up(tail0, E);
    const int wend = p.d < skip0 ? p.d : skip0;  // vectors below wend are written by the value pass
    const int64_t x0 = (int64_t)blockIdx.x * kWarps + warp;

    int64_t ix = x0;  // next row to copy: source ii of token ix
    int ii = 0;
    auto cell = [&](int st, int plane, int v) -> uint32_t {
        return ring_w + (uint32_t)((((st * P + plane) * V + v) * 32) * 16);
    };
    auto issue = [&](int st) {
        if (ix < p.T) {
            const T *row = src_row<T>(p.vt, ii, ix, p.d);
            const T *old = ACC ? dst_row<T>(p.dvt, ii, ix, p.d) : nullptr;
#pragma unroll
            for (int v = 0; v < V; ++v) {
                const int e = (lane + 32 * v) * E;
                if (e < p.d) cp_async16(cell(st, 0, v), row + e);
                if (ACC && e < wend) cp_async16(cell(st, P - 1, v), old + e);
            }
            if (++ii == p.n) {
                ii = 0;
                ix += nwarps;
            }
        }
        cp_async_commit();
    };
    Frag<T, E> dhr[V];  // dh of the token being processed (loaded one token ahead)
    auto load_dh = [&](int64_t xx) {
#pragma unroll
        for (int v = 0; v < V; ++v) {
            const int e = (lane + 32 * v) * E;
            if (e < p.d && xx < p.T) dhr[v].load_nc(dh + xx * p.d + e);
            else dhr[v].zero();
        }
    };
    load_dh(x0);
#pragma unroll
    for (int st = 0; st < S - 1; ++st) issue(st);
    int st_c = 0, st_i = S - 1;

    for (int64_t x = x0; x < p.T; x += nwarps) {
        lr_route_b<T>(p, x, lane, q_s, a_s, s_s, rho_s);
        __syncwarp();

        for (int i = 0; i < p.n; ++i) {
            issue(st_i);
            cp_async_wait<S - 1>();  // this lane's copies of row i have landed
            Frag<T, E> f[V];
            Frag<T, E> old[V];
#pragma unroll
            for (int v = 0; v < V; ++v) {
                const int e = (lane + 32 * v) * E;
                if (e < p.d) f[v].a = ld_shared16(cell(st_c, 0, v));
                else f[v].zero();
                if (ACC && e < wend) old[v].a = ld_shared16(cell(st_c, P - 1, v));
                else old[v].zero();
            }
            const float gp = lr_bwd_row<T, T, V, ACC>(f, old, dhr, a_s[i], dst_row<T>(p.dvt, i, x, p.d),
                                                      tail0, wend, lane);
            const float g = warp_sum(gp);
            if (lane == 0) g_s[i] = g;
            st_c = (st_c + 1 == S) ? 0 : st_c + 1;
            st_i = (st_i + 1 == S) ? 0 : st_i + 1;
        }
        // this token's dh is dead now: the next token's travels during the key pass
        load_dh(x + nwarps);
        __syncwarp();

        float part = 0.f;
        for (int k = lane; k < p.n; k += 32) part = fmaf(a_s[k], g_s[k], part);
        const float gbar = warp_sum(part);
        __syncwarp();
        for (int k = lane; k < p.n; k += 32) g_s[k] = a_s[k] * (g_s[k] - gbar);
        __syncwarp();
        if (VK)  // chosen on the host (vector_key_pass): only one pass is compiled in
            key_pass_vec<T, ACC>(p, dh, x, lane, tail0, q_s, a_s, s_s, rho_s, g_s, dq_s);
        else
            key_pass<T, ACC>(p, dh, x, lane, tail0, skip0, q_s, a_s, s_s, rho_s, g_s, dq_s);
        __syncwarp();
    }
    cp_async_wait_all();
    __syncthreads();
    for (int j = threadIdx.x; j < p.r; j += kThreads) {
        float acc = 0.f;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) acc += dq_all[w * rp + j];
        p.partials[(int64_t)blockIdx.x * p.r + j] = acc;
    }
}

// -------------------------------------------------------------- full keys
// One source row of the full-key backward, with lse and gbar = <dh, h> known:
// alpha_i, g_i = <dh, o_i>, ds_i (Eq. 11-12), and the value gradient
// alpha_i dh + ds_i rho_i (q - (s_i / d) kbar_i) written in one pass (the key
// is the value, Eq. 13).  Returns alpha_i (warp-uniform).  Operands stay packed and are unpacked one vector at
// a time; q_s (laid out by q_slot) is zero past d.  dq accumulates in dqf: V * E registers, or with
// DQS the warp's d floats in shared memory.
template <typename Tin, typename Tg, int V, bool DQS = false>
__device__ __forceinline__ float full_bwd_row(const Frag<Tin, VecE<Tin>::value> *f,
                                             const Frag<Tg, VecE<Tin>::value> *old,
                                             const Frag<Tin, VecE<Tin>::value> *dhr,
                                             const float *__restrict__ q_s, float *dqf, float gbar, float lse,
                                             float inv_d, float eps, Tg *__restrict__ drow, int d, int lane,
                                             bool accumulate) {
    constexpr int E = VecE<Tin>::value;
    float g = 0.f, ss = 0.f, qo = 0.f;
#pragma unroll
    for (int v = 0; v < V; ++v) {  // vectors past d are zero in f, dh and q
        float o[E], dv[E], qv[E];
        f[v].get(o);
        dhr[v].get(dv);
        q_get<E>(q_s, v, lane, qv);
#pragma unroll
        for (int t = 0; t < E; ++t) {
            if constexpr (!DQS) {  // packed pairs pay where dq stays in registers
                fma2(ss, qo, o[t], qv[t], o[t], o[t]);  // o.o, q.o
            } else {
                ss = fmaf(o[t], o[t], ss);
                qo = fmaf(qv[t], o[t], qo);
            }
            g = fmaf(dv[t], o[t], g);
        }
    }
    g = warp_sum(g);
    ss = warp_sum(ss);
    qo = warp_sum(qo);
    const float rho = rsqrtf(fmaf(ss, inv_d, eps));
    const float s = rho * qo;
    const float a = expf(s - lse);
    const float ds = a * (g - gbar);
    const float c1 = ds * rho;             // coefficient of q
    const float c2 = c1 * rho * s * inv_d;  // coefficient of o_i
#pragma unroll
    for (int v = 0; v < V; ++v) {
        const int e = (lane + 32 * v) * E;
        if (e < d) {
            float o[E], dv[E], w[E], qv[E];
            f[v].get(o);
            dhr[v].get(dv);
            q_get<E>(q_s, v, lane, qv);
            if (accumulate) old[v].get(w);
            else
#pragma unroll
                for (int t = 0; t < E; ++t) w[t] = 0.f;
            if constexpr (!DQS) {
#pragma unroll
                for (int t = 0; t < E; t += 2) {
                    fma2(w[t], w[t + 1], a, a, dv[t], dv[t + 1]);
                    fma2(w[t], w[t + 1], c1, c1, qv[t], qv[t + 1]);
                    fma2(w[t], w[t + 1], -c2, -c2, o[t], o[t + 1]);
                    fma2(dqf[v * E + t], dqf[v * E + t + 1], c1, c1, o[t], o[t + 1]);
                }
            } else {
#pragma unroll
                for (int t = 0; t < E; ++t) {
                    w[t] = fmaf(a, dv[t], w[t]);
                    w[t] = fmaf(c1, qv[t], w[t]);
                    w[t] = fmaf(-c2, o[t], w[t]);
                    dqf[e + t] = fmaf(c1, o[t], dqf[e + t]);  // this warp's row in shared memory
                }
            }
            Frag<Tg, E> out;
            out.set(w);
            out.store(drow + e);
        }
    }
    return a;
}

// gbar = <dh, h> = sum_i alpha_i g_i for one token, from the saved output.
template <typename Tin, int V>
__device__ __forceinline__ float full_gbar(const BwdParams &p, const Frag<Tin, VecE<Tin>::value> *dhr, int64_t x,
                                           int lane) {
    constexpr int E = VecE<Tin>::value;
    float gb = 0.f;
#pragma unroll
    for (int v = 0; v < V; ++v) {
        const int e = (lane + 32 * v) * E;
        if (e >= p.d) continue;
        float dv[E], hv[E];
        dhr[v].get(dv);
        if (p.h_bf16) {
            Frag<bf16, E> hf;
            hf.load_nc(static_cast<const bf16 *>(p.h) + x * p.d + e);
            hf.get(hv);
        } else {
            Frag<float, E> hf;
            hf.load_nc(static_cast<const float *>(p.h) + x * p.d + e);
            hf.get(hv);
        }
#pragma unroll
        for (int t = 0; t < E; ++t) gb = fmaf(dv[t], hv[t], gb);
    }
    return warp_sum(gb);
}

// Write the CTA's dq partial (sum over its warps, fixed order) from each warp's
// register accumulator dqf; scratch holds kWarps * round_up(d, 4) floats.
template <typename Tin, int V, bool DQS = false>
__device__ __forceinline__ void full_dq_partial(const BwdParams &p, const float *dqf, float *scratch, int lane,
                                                int warp) {
    constexpr int E = VecE<Tin>::value;
    const int dp4 = DQS ? 32 * V * E : round_up(p.d, 4);  // with DQS the rows are already in scratch
    float *dq_s = scratch + warp * dp4;
    if (!DQS)
#pragma unroll
        for (int v = 0; v < V; ++v) {
            const int e = (lane + 32 * v) * E;
            if (e < p.d)
#pragma unroll
                for (int t = 0; t < E; ++t) dq_s[e + t] = dqf[v * E + t];
        }
    __syncthreads();
    for (int j = threadIdx.x; j < p.d; j += kThreads) {
        float acc = 0.f;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) acc += scratch[w * dp4 + j];
        p.partials[(int64_t)blockIdx.x * p.d + j] = acc;
    }
}

// Bytes of the per-warp rings (cells of 16 bytes per lane), at least the dq
// scratch of full_dq_partial that reuses them.
__host__ __device__ inline size_t full_ring_bytes(int cells, int d) {
    const size_t ring = (size_t)kWarps * cells * 32 * 16, dq = sizeof(float) * (size_t)kWarps * round_up(d, 4);
    return ring > dq ? ring : dq;
}

// Full keys, one dtype for inputs and gradients: one warp per token, source
// rows (and old gradients when accumulating) streamed through the per-lane
// cp.async ring of the forward, S - 1 rows ahead and across tokens.  One CTA
// per SM: dq, dh and a row stay in registers, and the deep ring keeps enough
// bytes in flight for eight warps.
template <typename T, int V, int S, bool ACC>
__global__ void __launch_bounds__(kThreads, 1) bwd_full_pipe_kernel(const __grid_constant__ BwdParams p) {
    pdl_enter();
    constexpr int E = VecE<T>::value;
    constexpr int P = ACC ? 2 : 1;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    constexpr bool DQS = V * E > 32;  // dq in shared memory past 32 registers
    const size_t ring_bytes = full_ring_bytes(S * P * V, p.d);
    float *q_s = reinterpret_cast<float *>(smem_raw + ring_bytes);  // [32 V E] (q_slot), zero past d
    // dq partials: per warp rows of 32 V E floats after q_s (DQS), else the drained ring
    float *scratch = DQS ? q_s + 32 * V * E : reinterpret_cast<float *>(smem_raw);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int j = threadIdx.x; j < 32 * V * E; j += kThreads) q_s[q_slot<E>(j)] = (p.query && j < p.d) ? p.query[j] : 0.f;
    if (DQS)
        for (int j = threadIdx.x; j < kWarps * 32 * V * E; j += kThreads) scratch[j] = 0.f;
    __syncthreads();
    const uint32_t ring_w = smem_u32(smem_raw) + (uint32_t)(warp * S * P * V * 32 * 16) + 16u * lane;

    const T *__restrict__ dh = static_cast<const T *>(p.dh);
    const int64_t nwarps = (int64_t)gridDim.x * kWarps;
    const float inv_d = 1.f / (float)p.d;
    const int64_t x0 = (int64_t)blockIdx.x * kWarps + warp;

    int64_t ix = x0;
    int ii = 0;
    auto cell = [&](int st, int plane, int v) -> uint32_t {
        return ring_w + (uint32_t)((((st * P + plane) * V + v) * 32) * 16);
    };
    auto issue = [&](int st) {
        if (ix < p.T) {
            const T *row = src_row<T>(p.vt, ii, ix, p.d);
            const T *old = ACC ? dst_row<T>(p.dvt, ii, ix, p.d) : nullptr;
#pragma unroll
            for (int v = 0; v < V; ++v) {
                const int e = (lane + 32 * v) * E;
                if (e < p.d) {
                    cp_async16(cell(st, 0, v), row + e);
                    if (ACC) cp_async16(cell(st, P - 1, v), old + e);
                }
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
    float dq_r[DQS ? 1 : V * E];
#pragma unroll
    for (int t = 0; t < (DQS ? 1 : V * E); ++t) dq_r[t] = 0.f;
    float *dqf = DQS ? scratch + warp * 32 * V * E : dq_r;

    for (int64_t x = x0; x < p.T; x += nwarps) {
        const int64_t row_off = x * p.d;
        Frag<T, E> dhr[V];
#pragma unroll
        for (int v = 0; v < V; ++v) {
            const int e = (lane + 32 * v) * E;
            if (e < p.d) dhr[v].load_nc(dh + row_off + e);
            else dhr[v].zero();
        }
        const float gbar = full_gbar<T, V>(p, dhr, x, lane);
        const float lse = __ldg(p.lse + x);
        float asum = 0.f;
        for (int i = 0; i < p.n; ++i) {
            issue(st_i);
            cp_async_wait<S - 1>();
            Frag<T, E> f[V], old[V];
#pragma unroll
            for (int v = 0; v < V; ++v) {
                const int e = (lane + 32 * v) * E;
                if (e < p.d) f[v].a = ld_shared16(cell(st_c, 0, v));
                else f[v].zero();
                if (ACC && e < p.d) old[v].a = ld_shared16(cell(st_c, P - 1, v));
                else old[v].zero();
            }
            asum += full_bwd_row<T, T, V, DQS>(f, old, dhr, q_s, dqf, gbar, lse, inv_d, p.eps,
                                               dst_row<T>(p.dvt, i, x, p.d), p.d, lane, ACC);
            st_c = (st_c + 1 == S) ? 0 : st_c + 1;
            st_i = (st_i + 1 == S) ? 0 : st_i + 1;
        }
        check_alpha_sum(p, asum, lane);
    }
    cp_async_wait_all();
    __syncthreads();  // every warp is done with the ring before it becomes dq scratch
    full_dq_partial<T, V, DQS>(p, dqf, scratch, lane, warp);
}

// ---------------------------------------------------- sliced, one pass ----
// Sliced keys, one dtype for inputs and gradients, with the forward's lse: the
// key of row i is that row's last r coordinates, so the row streamed for the
// value gradient carries its key and no routing stage is needed.  The
// NV = r / E lanes holding the slice (one 16-byte vector each; an aligned
// group of lanes because NV divides 32 and r divides d) form |k_i|^2 and
// q.k_i with a butterfly over the group, which gives rho_i, s_i and
// alpha_i = exp(s_i - lse).  Every lane writes alpha_i dh (+ old) for its
// vectors before the slice, and the slice lanes park the row's key vector
// (and old gradient vector) in a per-warp stash in shared memory.  After the
// token's last row gbar = sum_i alpha_i g_i is exact, and all 32 lanes finish
// the slices from the stash (ds_i, dL/dk_i, old + alpha_i dh + dL/dk_i in one
// rounding, dq) as key_pass_vec does from global memory.  Every value row and
// every gradient row crosses HBM once.  The launcher runs the writing form
// (ACC = false); see launch_bwd_t for the accumulating one.
//
// Shared memory: ring [kWarps][S][P][V][32] cells | q [rp] | dq [kWarps][rp] |
// tables [kWarps][4][n4] (alpha, s, rho, g) | per warp: stash [n][P][NV]
// cells and the token's dh slice [NV] cells.
template <int V, bool ACC> struct OnePassStages {
    static constexpr int raw = 40 / (V * (ACC ? 2 : 1));  // a ring of about 160 KB per CTA
    static constexpr int value = raw < 2 ? 2 : (raw > 8 ? 8 : raw);
};

inline size_t onepass_smem(int S, int P, int V, int n, int r, int nv) {
    const int rp = round_up(r, 4), n4 = round_up(n, 4);
    return (size_t)kWarps * S * P * V * 32 * 16 + sizeof(float) * (size_t)rp * (1 + kWarps) +
           (size_t)kWarps * (sizeof(float) * 4 * n4 + (size_t)16 * nv * (n * P + 1));
}

template <typename T, int V, int S, bool ACC>
__global__ void __launch_bounds__(kThreads, 1) bwd_slr_onepass_kernel(const __grid_constant__ BwdParams p) {
    pdl_enter();
    constexpr int E = VecE<T>::value;
    constexpr int P = ACC ? 2 : 1;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int rp = round_up(p.r, 4), n4 = round_up(p.n, 4);
    const int nv = p.r / E;
    float *q_s = reinterpret_cast<float *>(smem_raw + (size_t)kWarps * S * P * V * 32 * 16);
    float *dq_all = q_s + rp;           // [kWarps][rp]
    float *tab = dq_all + kWarps * rp;  // [kWarps][4][n4]
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    float *a_s = tab + warp * 4 * n4;
    float *s_s = a_s + n4;
    float *rho_s = s_s + n4;
    float *g_s = rho_s + n4;
    const uint32_t stash_w = smem_u32(tab + kWarps * 4 * n4) + (uint32_t)(warp * nv * (p.n * P + 1) * 16);
    const uint32_t dhs_w = stash_w + (uint32_t)(p.n * P * nv * 16);
    const uint32_t ring_w = smem_u32(smem_raw) + (uint32_t)(warp * S * P * V * 32 * 16) + 16u * lane;
    for (int j = threadIdx.x; j < p.r; j += kThreads) q_s[j] = p.query ? p.query[j] : 0.f;
    __syncthreads();

    const T *__restrict__ dh = static_cast<const T *>(p.dh);
    const int64_t nwarps = (int64_t)gridDim.x * kWarps;
    const int tail0 = p.d - p.r;  // a whole number of vectors
    const int tv0 = tail0 / E;    // first slice vector of a row
    const int lead = tv0 % 32;    // lanes lead .. lead + nv - 1 hold the slice, all in register slot vk
    const int vk = tv0 / 32;
    const int kvi = lane - lead;
    const bool has_key = kvi >= 0 && kvi < nv;
    const int qi = has_key ? kvi * E : 0;  // r >= E, so q_s[qi + t] is in range for every lane
    float qv[E];
#pragma unroll
    for (int t = 0; t < E; ++t) qv[t] = has_key ? q_s[qi + t] : 0.f;
    // slice pass: lane takes slice vector kp of sources lane / nv, lane / nv + kst, ...
    const int kp = lane % nv, kst = 32 / nv, j0 = kp * E;
    float dq_r[E];
#pragma unroll
    for (int t = 0; t < E; ++t) dq_r[t] = 0.f;
    auto stash = [&](int i, int plane, int c) -> uint32_t {
        return stash_w + (uint32_t)(((i * P + plane) * nv + c) * 16);
    };

    const int64_t x0 = (int64_t)blockIdx.x * kWarps + warp;
    int64_t ix = x0;  // next row to copy: source ii of token ix
    int ii = 0;
    auto cell = [&](int st, int plane, int v) -> uint32_t {
        return ring_w + (uint32_t)((((st * P + plane) * V + v) * 32) * 16);
    };
    auto issue = [&](int st) {
        if (ix < p.T) {
            const T *row = src_row<T>(p.vt, ii, ix, p.d);
            const T *old = ACC ? dst_row<T>(p.dvt, ii, ix, p.d) : nullptr;
#pragma unroll
            for (int v = 0; v < V; ++v) {
                const int e = (lane + 32 * v) * E;
                if (e < p.d) {
                    cp_async16(cell(st, 0, v), row + e);
                    if (ACC) cp_async16(cell(st, P - 1, v), old + e);
                }
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
        const int64_t row_off = x * p.d;
        Frag<T, E> dhr[V];
#pragma unroll
        for (int v = 0; v < V; ++v) {
            const int e = (lane + 32 * v) * E;
            if (e < p.d) dhr[v].load_nc(dh + row_off + e);
            else dhr[v].zero();
        }
        const float lse = __ldg(p.lse + x);
#pragma unroll
        for (int v = 0; v < V; ++v)
            if (v == vk && has_key) st_shared16(dhs_w + (uint32_t)(kvi * 16), dhr[v].a);

        float asum = 0.f;
        for (int i = 0; i < p.n; ++i) {
            issue(st_i);
            cp_async_wait<S - 1>();  // this lane's copies of row i have landed
            Frag<T, E> f[V], old[V];
#pragma unroll
            for (int v = 0; v < V; ++v) {
                const int e = (lane + 32 * v) * E;
                if (e < p.d) f[v].a = ld_shared16(cell(st_c, 0, v));
                else f[v].zero();
                if (ACC && e < p.d) old[v].a = ld_shared16(cell(st_c, P - 1, v));
                else old[v].zero();
            }
            float g0 = 0.f, g1 = 0.f, ss = 0.f, qk = 0.f;
#pragma unroll
            for (int v = 0; v < V; ++v) {  // vectors past d are zero
                float o[E], dv[E];
                f[v].get(o);
                dhr[v].get(dv);
#pragma unroll
                for (int t = 0; t < E; t += 2) fma2(g0, g1, dv[t], dv[t + 1], o[t], o[t + 1]);
                if (v == vk && has_key) {
#pragma unroll
                    for (int t = 0; t < E; ++t) {
                        ss = fmaf(o[t], o[t], ss);
                        qk = fmaf(qv[t], o[t], qk);
                    }
                    st_shared16(stash(i, 0, kvi), f[v].a);
                    if (ACC) st_shared16(stash(i, 1, kvi), old[v].a);
                }
            }
            for (int off = 1; off < nv; off <<= 1) {  // the slice group is aligned: partners stay inside
                ss += __shfl_xor_sync(0xffffffffu, ss, off);
                qk += __shfl_xor_sync(0xffffffffu, qk, off);
            }
            const float rho = rsqrtf(fmaf(ss, p.inv_r, p.eps));
            const float s = __shfl_sync(0xffffffffu, rho * qk, lead);
            // one source weighs exactly 1 (a softmax over one score), however s rounds against lse
            const float a = p.n == 1 ? 1.f : expf(s - lse);
            asum += a;
            T *drow = dst_row<T>(p.dvt, i, x, p.d);
#pragma unroll
            for (int v = 0; v < V; ++v) {
                const int e = (lane + 32 * v) * E;
                if (e < tail0) {
                    float dv[E], w[E];
                    dhr[v].get(dv);
                    if (ACC) old[v].get(w);
                    else
#pragma unroll
                        for (int t = 0; t < E; ++t) w[t] = 0.f;
#pragma unroll
                    for (int t = 0; t < E; ++t) w[t] = fmaf(a, dv[t], w[t]);
                    Frag<T, E> out;
                    out.set(w);
                    out.store(drow + e);
                }
            }
            const float g = warp_sum(g0 + g1);
            if (lane == lead) {
                a_s[i] = a;
                s_s[i] = s;
                rho_s[i] = rho;
                g_s[i] = g;
            }
            st_c = (st_c + 1 == S) ? 0 : st_c + 1;
            st_i = (st_i + 1 == S) ? 0 : st_i + 1;
        }
        __syncwarp();  // stash, tables and the dh slice are visible to the whole warp
        check_alpha_sum(p, asum, lane);

        float part = 0.f;
        for (int k = lane; k < p.n; k += 32) part = fmaf(a_s[k], g_s[k], part);
        const float gbar = warp_sum(part);
        float dhv[E];
        {
            Frag<T, E> hf;
            hf.a = ld_shared16(dhs_w + (uint32_t)(kp * 16));
            hf.get(dhv);
        }
        for (int k = lane / nv; k < p.n; k += kst) {
            Frag<T, E> kf, of;
            kf.a = ld_shared16(stash(k, 0, kp));
            if (ACC) of.a = ld_shared16(stash(k, 1, kp));
            else of.zero();
            const float a = a_s[k], s = s_s[k], rho = rho_s[k];
            const float ds = a * (g_s[k] - gbar);
            const float c1 = ds * rho, c2 = s * p.inv_r;
            float kv[E], w[E];
            kf.get(kv);
            of.get(w);
#pragma unroll
            for (int t = 0; t < E; ++t) {
                const float kbar = rho * kv[t];
                const float dk = c1 * (q_s[j0 + t] - c2 * kbar);
                dq_r[t] = fmaf(ds, kbar, dq_r[t]);
                w[t] += fmaf(a, dhv[t], dk);
            }
            Frag<T, E> out;
            out.set(w);
            out.store(dst_row<T>(p.dvt, k, x, p.d) + tail0 + j0);
        }
        __syncwarp();  // the next token overwrites stash, tables and dh slice
    }
    cp_async_wait_all();
    // lanes sharing a slice vector combine their dq parts with a fixed butterfly
#pragma unroll
    for (int t = 0; t < E; ++t)
        for (int off = nv; off < 32; off <<= 1) dq_r[t] += __shfl_xor_sync(0xffffffffu, dq_r[t], off);
    if (lane < nv)
#pragma unroll
        for (int t = 0; t < E; ++t) dq_all[warp * rp + j0 + t] = dq_r[t];
    __syncthreads();
    for (int j = threadIdx.x; j < p.r; j += kThreads) {
        float acc = 0.f;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) acc += dq_all[w * rp + j];
        p.partials[(int64_t)blockIdx.x * p.r + j] = acc;
    }
}

// Sliced keys, gradients accumulated, with the forward's lse: the one-pass
// structure of bwd_slr_onepass_kernel sized for two CTAs per SM, so that
// sixteen warps share each SM.  The ring carries the value row and the old
// gradient row (3 stages); only each row's key vector is parked in the stash,
// and the tables hold alpha_i and g_i alone: after the token's last row the
// slice lanes recompute rho_i and s_i from the stashed key (the same fixed
// butterfly as in the value pass, so bitwise the same values) and re-read the
// old gradient of the slice, which the ring brought through L2 moments before.
//
// Shared memory: ring [kWarps][S][2][V][32] cells | q [rp] | dq [kWarps][rp] |
// tables [kWarps][2][n4] (alpha, g) | per warp: stash [n][nv] cells and the
// token's dh slice [nv] cells.
inline size_t onepass_acc_smem(int S, int V, int n, int r, int nv) {
    const int rp = round_up(r, 4), n4 = round_up(n, 4);
    return (size_t)kWarps * S * 2 * V * 32 * 16 + sizeof(float) * (size_t)rp * (1 + kWarps) +
           (size_t)kWarps * (sizeof(float) * 2 * n4 + (size_t)16 * nv * (n + 1));
}

template <typename T, int V, int S>
__global__ void __launch_bounds__(kThreads, V >= 8 ? 1 : 2) bwd_slr_onepass_acc_kernel(const __grid_constant__ BwdParams p) {
    pdl_enter();
    constexpr int E = VecE<T>::value;
    constexpr int P = 2;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int rp = round_up(p.r, 4), n4 = round_up(p.n, 4);
    const int nv = p.r / E;
    float *q_s = reinterpret_cast<float *>(smem_raw + (size_t)kWarps * S * P * V * 32 * 16);
    float *dq_all = q_s + rp;           // [kWarps][rp]
    float *tab = dq_all + kWarps * rp;  // [kWarps][2][n4]
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    float *a_s = tab + warp * 2 * n4;
    float *g_s = a_s + n4;
    const uint32_t stash_w = smem_u32(tab + kWarps * 2 * n4) + (uint32_t)(warp * nv * (p.n + 1) * 16);
    const uint32_t dhs_w = stash_w + (uint32_t)(p.n * nv * 16);
    const uint32_t ring_w = smem_u32(smem_raw) + (uint32_t)(warp * S * P * V * 32 * 16) + 16u * lane;
    for (int j = threadIdx.x; j < p.r; j += kThreads) q_s[j] = p.query ? p.query[j] : 0.f;
    __syncthreads();

    const T *__restrict__ dh = static_cast<const T *>(p.dh);
    const int64_t nwarps = (int64_t)gridDim.x * kWarps;
    const int tail0 = p.d - p.r;  // a whole number of vectors
    const int tv0 = tail0 / E;    // first slice vector of a row
    const int lead = tv0 % 32;    // lanes lead .. lead + nv - 1 hold the slice, all in register slot vk
    const int vk = tv0 / 32;
    const int kvi = lane - lead;
    const bool has_key = kvi >= 0 && kvi < nv;
    float qv[E];
#pragma unroll
    for (int t = 0; t < E; ++t) qv[t] = has_key ? q_s[kvi * E + t] : 0.f;
    // slice pass: lane takes slice vector kp of sources lane / nv, lane / nv + kst, ...
    const int kp = lane % nv, kst = 32 / nv, j0 = kp * E;
    float qs[E];
#pragma unroll
    for (int t = 0; t < E; ++t) qs[t] = q_s[j0 + t];
    float dq_r[E];
#pragma unroll
    for (int t = 0; t < E; ++t) dq_r[t] = 0.f;

    const int64_t x0 = (int64_t)blockIdx.x * kWarps + warp;
    int64_t ix = x0;  // next row to copy: source ii of token ix
    int ii = 0;
    auto cell = [&](int st, int plane, int v) -> uint32_t {
        return ring_w + (uint32_t)((((st * P + plane) * V + v) * 32) * 16);
    };
    auto issue = [&](int st) {
        if (ix < p.T) {
            const T *row = src_row<T>(p.vt, ii, ix, p.d);
            const T *old = dst_row<T>(p.dvt, ii, ix, p.d);
#pragma unroll
            for (int v = 0; v < V; ++v) {
                const int e = (lane + 32 * v) * E;
                if (e < p.d) cp_async16(cell(st, 0, v), row + e);
                if (e < tail0) cp_async16(cell(st, 1, v), old + e);  // the slice's old value is re-read later
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
        const int64_t row_off = x * p.d;
        Frag<T, E> dhr[V];
#pragma unroll
        for (int v = 0; v < V; ++v) {
            const int e = (lane + 32 * v) * E;
            if (e < p.d) dhr[v].load_nc(dh + row_off + e);
            else dhr[v].zero();
        }
        const float lse = __ldg(p.lse + x);
#pragma unroll
        for (int v = 0; v < V; ++v)
            if (v == vk && has_key) st_shared16(dhs_w + (uint32_t)(kvi * 16), dhr[v].a);

        float asum = 0.f;
        for (int i = 0; i < p.n; ++i) {
            issue(st_i);
            cp_async_wait<S - 1>();  // this lane's copies of row i have landed
            Frag<T, E> f[V];
#pragma unroll
            for (int v = 0; v < V; ++v) {
                const int e = (lane + 32 * v) * E;
                if (e < p.d) f[v].a = ld_shared16(cell(st_c, 0, v));
                else f[v].zero();
            }
            float g0 = 0.f, g1 = 0.f, ss = 0.f, qk = 0.f;
#pragma unroll
            for (int v = 0; v < V; ++v) {  // vectors past d are zero
                float o[E], dv[E];
                f[v].get(o);
                dhr[v].get(dv);
#pragma unroll
                for (int t = 0; t < E; t += 2) fma2(g0, g1, dv[t], dv[t + 1], o[t], o[t + 1]);
                if (v == vk && has_key) {
#pragma unroll
                    for (int t = 0; t < E; ++t) {
                        ss = fmaf(o[t], o[t], ss);
                        qk = fmaf(qv[t], o[t], qk);
                    }
                    st_shared16(stash_w + (uint32_t)((i * nv + kvi) * 16), f[v].a);
                }
            }
            for (int off = 1; off < nv; off <<= 1) {  // the slice group is aligned: partners stay inside
                ss += __shfl_xor_sync(0xffffffffu, ss, off);
                qk += __shfl_xor_sync(0xffffffffu, qk, off);
            }
            const float rho = rsqrtf(fmaf(ss, p.inv_r, p.eps));
            const float s = __shfl_sync(0xffffffffu, rho * qk, lead);
            // one source weighs exactly 1 (a softmax over one score), however s rounds against lse
            const float a = p.n == 1 ? 1.f : expf(s - lse);
            asum += a;
            T *drow = dst_row<T>(p.dvt, i, x, p.d);
#pragma unroll
            for (int v = 0; v < V; ++v) {
                const int e = (lane + 32 * v) * E;
                if (e < tail0) {
                    Frag<T, E> of;
                    of.a = ld_shared16(cell(st_c, 1, v));
                    float dv[E], w[E];
                    dhr[v].get(dv);
                    of.get(w);
#pragma unroll
                    for (int t = 0; t < E; ++t) w[t] = fmaf(a, dv[t], w[t]);
                    Frag<T, E> out;
                    out.set(w);
                    out.store(drow + e);
                }
            }
            const float g = warp_sum(g0 + g1);
            if (lane == lead) {
                a_s[i] = a;
                g_s[i] = g;
            }
            st_c = (st_c + 1 == S) ? 0 : st_c + 1;
            st_i = (st_i + 1 == S) ? 0 : st_i + 1;
        }
        __syncwarp();  // stash, tables and the dh slice are visible to the whole warp
        check_alpha_sum(p, asum, lane);

        float part = 0.f;
        for (int k = lane; k < p.n; k += 32) part = fmaf(a_s[k], g_s[k], part);
        const float gbar = warp_sum(part);
        float dhv[E];
        {
            Frag<T, E> hf;
            hf.a = ld_shared16(dhs_w + (uint32_t)(kp * 16));
            hf.get(dhv);
        }
        // sources k = lane / nv + m kst: the old slices of a batch are loaded together
        constexpr int B = 4;
        for (int kb = lane / nv; kb - (lane / nv) < p.n; kb += kst * B) {
            Frag<T, E> of[B];
#pragma unroll
            for (int m = 0; m < B; ++m) {
                const int k = kb + m * kst;
                if (k < p.n) of[m].load(dst_row<T>(p.dvt, k, x, p.d) + tail0 + j0);
                else of[m].zero();
            }
#pragma unroll
            for (int m = 0; m < B; ++m) {
                const int k = kb + m * kst;  // the nv lanes of source k are consecutive: an aligned group
                Frag<T, E> kf;
                if (k < p.n) kf.a = ld_shared16(stash_w + (uint32_t)((k * nv + kp) * 16));
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
                for (int off = 1; off < nv; off <<= 1) {
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
                    Frag<T, E> out;
                    out.set(w);
                    out.store(dst_row<T>(p.dvt, k, x, p.d) + tail0 + j0);
                }
            }
        }
        __syncwarp();  // the next token overwrites stash, tables and dh slice
    }
    cp_async_wait_all();
    // lanes sharing a slice vector combine their dq parts with a fixed butterfly
#pragma unroll
    for (int t = 0; t < E; ++t)
        for (int off = nv; off < 32; off <<= 1) dq_r[t] += __shfl_xor_sync(0xffffffffu, dq_r[t], off);
    if (lane < nv)
#pragma unroll
        for (int t = 0; t < E; ++t) dq_all[warp * rp + j0 + t] = dq_r[t];
    __syncthreads();
    for (int j = threadIdx.x; j < p.r; j += kThreads) {
        float acc = 0.f;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) acc += dq_all[w * rp + j];
        p.partials[(int64_t)blockIdx.x * p.r + j] = acc;
    }
}

// Full keys with gradients in another dtype than the inputs: rows loaded into
// registers, U at a time.
template <typename Tin, typename Tg, int V, int U>
__global__ void __launch_bounds__(kThreads, (V <= 2 ? 2 : 1)) bwd_full_kernel(const __grid_constant__ BwdParams p) {
    pdl_enter();
    constexpr int E = VecE<Tin>::value;
    extern __shared__ float smem[];
    float *q_s = smem;                    // [32 V E] (q_slot), zero past d
    float *scratch = q_s + 32 * V * E;    // [kWarps][round_up(d, 4)], used once at the end
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int j = threadIdx.x; j < 32 * V * E; j += kThreads) q_s[q_slot<E>(j)] = (p.query && j < p.d) ? p.query[j] : 0.f;
    __syncthreads();

    const Tin *__restrict__ dh = static_cast<const Tin *>(p.dh);
    const int64_t nwarps = (int64_t)gridDim.x * kWarps;
    const float inv_d = 1.f / (float)p.d;
    float dqf[V * E];
#pragma unroll
    for (int t = 0; t < V * E; ++t) dqf[t] = 0.f;

    for (int64_t x = (int64_t)blockIdx.x * kWarps + warp; x < p.T; x += nwarps) {
        const int64_t row_off = x * p.d;
        Frag<Tin, E> dhr[V];
#pragma unroll
        for (int v = 0; v < V; ++v) {
            const int e = (lane + 32 * v) * E;
            if (e < p.d) dhr[v].load_nc(dh + row_off + e);
            else dhr[v].zero();
        }
        const float gbar = full_gbar<Tin, V>(p, dhr, x, lane);
        const float lse = __ldg(p.lse + x);
        float asum = 0.f;
        int i = 0;
        for (; i + U <= p.n; i += U) {
            Frag<Tin, E> f[U][V];
            Frag<Tg, E> old[U][V];
#pragma unroll
            for (int u = 0; u < U; ++u)
#pragma unroll
                for (int v = 0; v < V; ++v) {
                    const int e = (lane + 32 * v) * E;
                    if (e < p.d) f[u][v].load_nc(src_row<Tin>(p.vt, i + u, x, p.d) + e);
                    else f[u][v].zero();
                    if (p.accumulate && e < p.d) old[u][v].load(dst_row<Tg>(p.dvt, i + u, x, p.d) + e);
                    else old[u][v].zero();
                }
#pragma unroll
            for (int u = 0; u < U; ++u)
                asum += full_bwd_row<Tin, Tg, V>(f[u], old[u], dhr, q_s, dqf, gbar, lse, inv_d, p.eps,
                                                 dst_row<Tg>(p.dvt, i + u, x, p.d), p.d, lane, p.accumulate);
        }
        for (; i < p.n; ++i) {
            Frag<Tin, E> f[V];
            Frag<Tg, E> old[V];
#pragma unroll
            for (int v = 0; v < V; ++v) {
                const int e = (lane + 32 * v) * E;
                if (e < p.d) f[v].load_nc(src_row<Tin>(p.vt, i, x, p.d) + e);
                else f[v].zero();
                if (p.accumulate && e < p.d) old[v].load(dst_row<Tg>(p.dvt, i, x, p.d) + e);
                else old[v].zero();
            }
            asum += full_bwd_row<Tin, Tg, V>(f, old, dhr, q_s, dqf, gbar, lse, inv_d, p.eps,
                                             dst_row<Tg>(p.dvt, i, x, p.d), p.d, lane, p.accumulate);
        }
        check_alpha_sum(p, asum, lane);
    }
    full_dq_partial<Tin, V>(p, dqf, scratch, lane, warp);
}

// Fixed-order sum of the CTA partials, dq[j] (+)= sum_b partials[b][j]: one
// warp per coordinate, lane l sums partials l, l+32, ... and a fixed butterfly
// combines the lanes, so the result depends only on the number of partials.
__global__ void dq_reduce_kernel(const float *__restrict__ partials, int nparts, int rq, float *dq, int accumulate) {
    pdl_enter();
    const int j = (int)((blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5);
    const int lane = threadIdx.x & 31;
    if (j >= rq) return;  // whole warps leave together (blockDim is a multiple of 32)
    float acc = 0.f;
    for (int b = lane; b < nparts; b += 32) acc += partials[(int64_t)b * rq + j];
    acc = warp_sum(acc);
    if (lane == 0) dq[j] = accumulate ? dq[j] + acc : acc;
}

cudaError_t launch_partial_sum(const float *partials, int nparts, int width, float *out, int accumulate,
                               cudaStream_t s) {
    launch_pdl(dq_reduce_kernel, (width + 7) / 8, 256, 0, s, partials, nparts, width, out, accumulate);
    return cudaGetLastError();
}

// ------------------------------------------------------------- launch ----
// Rows in flight per lane in the low-rank value pass (registers: V vectors of
// values, and as many of old gradients when accumulating, per row).
#ifndef LRAR_BWD_U_ACC
#define LRAR_BWD_U_ACC 2
#endif
#ifndef LRAR_BWD_U_NOACC
#define LRAR_BWD_U_NOACC 4
#endif
template <int V, bool ACC> struct BwdRows {
    static constexpr int value = V >= 8 ? (ACC ? 1 : 2)
                                        : V == 4 ? (ACC ? LRAR_BWD_U_ACC : LRAR_BWD_U_NOACC) : (ACC ? 4 : 8);
};

template <typename Tin, typename Tg, int V>
static cudaError_t launch_bwd_t(const BwdArgs &a, cudaStream_t s) {
    constexpr int U = V >= 4 ? 1 : (V == 2 ? 2 : 4);
    // wider gradients than inputs double the old-gradient registers per row
    constexpr int UA = sizeof(Tg) > sizeof(Tin) ? (BwdRows<V, true>::value + 1) / 2 : BwdRows<V, true>::value;
    BwdParams p;
    for (int i = 0; i < kMaxTab; ++i) {
        const bool in = i < a.n;
        p.vt.p[i] = in ? a.values[i] : nullptr;
        p.kt.p[i] = (in && a.keys) ? a.keys[i] : nullptr;
        p.dvt.p[i] = in ? a.dvalues[i] : nullptr;
        p.dkt.p[i] = (in && a.dkeys) ? a.dkeys[i] : nullptr;
    }
    p.dh = a.dh;
    p.h = a.h;
    p.query = a.query;
    p.lse = a.lse;
    p.partials = a.partials;
    p.status = a.status;
    p.T = a.T;
    p.n = a.n;
    p.d = a.d;
    p.r = a.r;
    p.eps = a.eps;
    p.inv_r = 1.f / (float)a.r;
    p.sliced = a.variant == kSliced;
    p.accumulate = a.accumulate;
    p.h_bf16 = a.h_dtype == kBF16;
    constexpr int esz = sizeof(Tin);
    if (a.variant == kSliced)
        p.key_vec = ((a.r * esz) % 16 == 0) && (((a.d - a.r) * esz) % 16 == 0);
    else
        p.key_vec = (a.r * esz) % 16 == 0;  // every key matrix is 16-byte aligned (checked by the API)
    // Vector key pass (key_pass_vec) when the keys are whole aligned vectors whose
    // row divides a warp, except for accumulating keys of fewer than four vectors,
    // where the scalar batches measured slightly faster.
    constexpr int E = VecE<Tin>::value;
    const bool vk = kVecKeyPass && p.key_vec && a.r % E == 0 && 32 % (a.r / E) == 0 && (!a.accumulate || a.r / E >= 4);
    const int64_t work = (a.T + kWarps - 1) / kWarps;
    const void *k;
    size_t smem;
    int rq;
    constexpr bool kPipe = LRAR_BWD_PIPE && std::is_same<Tin, Tg>::value;
    // Sliced keys with the forward's lse: one pass over the values when the
    // slice is whole vectors forming an aligned lane group (r / E divides 32,
    // r divides d) and the per-warp stash fits in shared memory -- the
    // fixed-shape kernel at (d, r) = (1024, 16), else bwd_slr_onepass_acc_kernel
    // (accumulating) or bwd_slr_onepass_kernel (writing).  Other calls take the
    // routing + value pass + key pass kernel (bwd_lr_pipe_kernel).
    if constexpr (kPipe) {
        bool launched = false;
        cudaError_t ef = launch_bwd_fixed(p, a, launched, s);
        if (ef != cudaSuccess || launched) return ef;
        constexpr int OSN = OnePassStages<V, false>::value;
        const int nvk = a.r / E;
        // accumulating: the one-pass kernel when it fits two CTAs per SM (one at
        // eight vectors per lane, where the other kernels run one CTA per SM too).
        // At eight vectors per lane (d = 2048) it wins at few sources and loses
        // at many (fraction of the copy peak, one-pass against routing + value
        // pass + key pass: n = 2: 0.82 / 0.65, n = 5: 0.94 / 0.84, n = 9: 0.97 /
        // 0.96, n = 17: 0.96 / 0.99), so there it serves n <= 9.
        constexpr int kAccMaxSources = V >= 8 ? 9 : kMaxSources;
        if (a.variant == kSliced && a.lse && a.accumulate && p.key_vec && nvk >= 1 && nvk <= 32 && 32 % nvk == 0 &&
            a.d % a.r == 0 && a.n <= kAccMaxSources) {
            constexpr int OSA = 3;
            const size_t smem2 = onepass_acc_smem(OSA, V, a.n, a.r, nvk);
            const void *k2 = (const void *)bwd_slr_onepass_acc_kernel<Tin, V, OSA>;
            int dev = 0, per_sm = 0, optin = 0;
            cudaGetDevice(&dev);
            cudaDeviceGetAttribute(&per_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev);
            cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
            constexpr int kCtas = V >= 8 ? 1 : 2;  // CTAs per SM (1 KB reserved per CTA)
            if (kCtas * (smem2 + 1024) <= (size_t)per_sm && smem2 <= (size_t)optin) {
                cudaError_t e = cudaFuncSetAttribute(k2, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem2);
                if (e != cudaSuccess) return e;
                const int grid = persistent_grid(k2, kThreads, smem2, work, kMaxPartials);
                launch_pdl(bwd_slr_onepass_acc_kernel<Tin, V, OSA>, grid, kThreads, smem2, s, p);
                e = cudaGetLastError();
                if (e != cudaSuccess) return e;
                launch_pdl(dq_reduce_kernel, (a.r + 7) / 8, 256, 0, s, a.partials, grid, a.r, a.dq, a.accumulate);
                return cudaGetLastError();
            }
        }
        if (a.variant == kSliced && a.lse && !a.accumulate && p.key_vec && nvk >= 1 && nvk <= 32 &&
            32 % nvk == 0 && a.d % a.r == 0) {
            const size_t smem1 = onepass_smem(OSN, 1, V, a.n, a.r, nvk);
            int dev = 0, optin = 0;
            cudaGetDevice(&dev);
            cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
            if (smem1 <= (size_t)optin) {
                const void *k1 = (const void *)bwd_slr_onepass_kernel<Tin, V, OSN, false>;
                cudaError_t e = cudaFuncSetAttribute(k1, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem1);
                if (e != cudaSuccess) return e;
                const int grid = persistent_grid(k1, kThreads, smem1, work, kMaxPartials);
                launch_pdl(bwd_slr_onepass_kernel<Tin, V, OSN, false>, grid, kThreads, smem1, s, p);
                e = cudaGetLastError();
                if (e != cudaSuccess) return e;
                launch_pdl(dq_reduce_kernel, (a.r + 7) / 8, 256, 0, s, a.partials, grid, a.r, a.dq, a.accumulate);
                return cudaGetLastError();
            }
        }
    }
    constexpr int SA = BwdStages<V, true>::value, SN = BwdStages<V, false>::value;
    // with dq in shared memory (V E > 32) the rings leave it room
    constexpr int FB = V * E > 32 ? 32 : 48;
    constexpr int FSA = FullStages<V, 2, FB>::value, FSN = FullStages<V, 1, FB>::value;
    if (a.variant == kFull) {
        if (kPipe) {
            k = a.accumulate ? (const void *)bwd_full_pipe_kernel<Tin, V, FSA, true>
                             : (const void *)bwd_full_pipe_kernel<Tin, V, FSN, false>;
            smem = full_ring_bytes(a.accumulate ? FSA * 2 * V : FSN * V, a.d) +
                   sizeof(float) * 32 * V * E * (V * E > 32 ? 1 + kWarps : 1);
        } else {
            k = (const void *)bwd_full_kernel<Tin, Tg, V, U>;
            smem = sizeof(float) * (32 * V * E + (size_t)kWarps * round_up(a.d, 4));
        }
        rq = a.d;
    } else if (kPipe) {
        if (vk)
            k = a.accumulate ? (const void *)bwd_lr_pipe_kernel<Tin, V, SA, true, true>
                             : (const void *)bwd_lr_pipe_kernel<Tin, V, SN, false, true>;
        else
            k = a.accumulate ? (const void *)bwd_lr_pipe_kernel<Tin, V, SA, true, false>
                             : (const void *)bwd_lr_pipe_kernel<Tin, V, SN, false, false>;
        smem = (size_t)kWarps * (a.accumulate ? SA * 2 : SN) * V * 32 * 16 +
               sizeof(float) * ((size_t)round_up(a.r, 4) * (1 + kWarps) + (size_t)kWarps * 4 * kMaxSources);
        rq = a.r;
    } else {
        k = a.accumulate ? (const void *)bwd_lr_kernel<Tin, Tg, V, UA, true>
                         : (const void *)bwd_lr_kernel<Tin, Tg, V, BwdRows<V, false>::value, false>;
        smem = sizeof(float) * ((size_t)round_up(a.r, 4) * (1 + kWarps) + (size_t)kWarps * 4 * kMaxSources);
        rq = a.r;
    }
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
    }
    const int grid = persistent_grid(k, kThreads, smem, work, kMaxPartials);
    if (a.variant == kFull && kPipe && a.accumulate)
        launch_pdl(bwd_full_pipe_kernel<Tin, V, FSA, true>, grid, kThreads, smem, s, p);
    else if (a.variant == kFull && kPipe)
        launch_pdl(bwd_full_pipe_kernel<Tin, V, FSN, false>, grid, kThreads, smem, s, p);
    else if (a.variant == kFull)
        launch_pdl(bwd_full_kernel<Tin, Tg, V, U>, grid, kThreads, smem, s, p);
    else if (kPipe && a.accumulate && vk)
        launch_pdl(bwd_lr_pipe_kernel<Tin, V, SA, true, true>, grid, kThreads, smem, s, p);
    else if (kPipe && a.accumulate)
        launch_pdl(bwd_lr_pipe_kernel<Tin, V, SA, true, false>, grid, kThreads, smem, s, p);
    else if (kPipe && vk)
        launch_pdl(bwd_lr_pipe_kernel<Tin, V, SN, false, true>, grid, kThreads, smem, s, p);
    else if (kPipe)
        launch_pdl(bwd_lr_pipe_kernel<Tin, V, SN, false, false>, grid, kThreads, smem, s, p);
    else if (a.accumulate)
        launch_pdl(bwd_lr_kernel<Tin, Tg, V, UA, true>, grid, kThreads, smem, s, p);
    else
        launch_pdl(bwd_lr_kernel<Tin, Tg, V, BwdRows<V, false>::value, false>, grid, kThreads, smem, s, p);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    launch_pdl(dq_reduce_kernel, (rq + 7) / 8, 256, 0, s, a.partials, grid, rq, a.dq, a.accumulate);
    return cudaGetLastError();
}

template <typename Tin, typename Tg>
static cudaError_t launch_bwd_w(const BwdArgs &a, cudaStream_t s) {
    constexpr int E = VecE<Tin>::value;
    const int vecs = (a.d + E - 1) / E;
    if (vecs <= 32) return launch_bwd_t<Tin, Tg, 1>(a, s);
    if (vecs <= 64) return launch_bwd_t<Tin, Tg, 2>(a, s);
    if (vecs <= 128) return launch_bwd_t<Tin, Tg, 4>(a, s);
    return launch_bwd_t<Tin, Tg, 8>(a, s);
}

cudaError_t launch_backward(const BwdArgs &a, cudaStream_t s) {
    if (a.in_dtype == kBF16)
        return a.grad_dtype == kBF16 ? launch_bwd_w<bf16, bf16>(a, s) : launch_bwd_w<bf16, float>(a, s);
    return a.grad_dtype == kBF16 ? launch_bwd_w<float, bf16>(a, s) : launch_bwd_w<float, float>(a, s);
}

// ------------------------------------------------------ block assembly ---
// dst = beta * dst + alpha * src over count elements, 8 per thread-step.
template <typename Td, typename Ts>
__global__ void block_acc_kernel(Td *__restrict__ dst, const Ts *__restrict__ src, int64_t count, float alpha,
                                 float beta, int vec) {
    pdl_enter();
    const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t nthreads = (int64_t)gridDim.x * blockDim.x;
    const int64_t groups = vec ? count / 8 : 0;
    for (int64_t gi = tid; gi < groups; gi += nthreads) {
        const int64_t e = gi * 8;
        Frag<Ts, 8> fs;
        fs.load_nc(src + e);
        float sv[8], w[8];
        fs.get(sv);
        if (beta != 0.f) {
            Frag<Td, 8> fd;
            fd.load(dst + e);
            fd.get(w);
#pragma unroll
            for (int t = 0; t < 8; ++t) w[t] = fmaf(alpha, sv[t], beta * w[t]);
        } else {
#pragma unroll
            for (int t = 0; t < 8; ++t) w[t] = alpha * sv[t];
        }
        Frag<Td, 8> out;
        out.set(w);
        out.store(dst + e);
    }
    for (int64_t e = groups * 8 + tid; e < count; e += nthreads) {
        const float sv = to_f(src[e]);
        const float w = beta != 0.f ? fmaf(alpha, sv, beta * to_f(dst[e])) : alpha * sv;
        dst[e] = from_f<Td>(w);
    }
}

template <typename Td, typename Ts>
static cudaError_t launch_acc_t(void *dst, const void *src, int64_t count, float alpha, float beta, cudaStream_t s) {
    const int vec = ((reinterpret_cast<uintptr_t>(dst) | reinterpret_cast<uintptr_t>(src)) & 15) == 0;
    const int threads = 256;
    const int64_t groups = vec ? count / 8 : count;
    const int grid = persistent_grid((const void *)block_acc_kernel<Td, Ts>, threads, 0,
                                     (groups + threads - 1) / threads, 1 << 30);
    launch_pdl(block_acc_kernel<Td, Ts>, grid, threads, 0, s, static_cast<Td *>(dst), static_cast<const Ts *>(src), count,
                                                       alpha, beta, vec);
    return cudaGetLastError();
}

cudaError_t launch_block_accumulate(int dst_dtype, void *dst, int src_dtype, const void *src, int64_t count,
                                    float alpha, float beta, cudaStream_t s) {
    if (dst_dtype == kBF16)
        return src_dtype == kBF16 ? launch_acc_t<bf16, bf16>(dst, src, count, alpha, beta, s)
                                  : launch_acc_t<bf16, float>(dst, src, count, alpha, beta, s);
    return src_dtype == kBF16 ? launch_acc_t<float, bf16>(dst, src, count, alpha, beta, s)
                              : launch_acc_t<float, float>(dst, src, count, alpha, beta, s);
}

}  // namespace lrar
