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
//
// Phase 1 tiles a token's row over the warps of a group: warp (g, ch) of a CTA
// owns the 32 x 16-byte chunk ch of token g's rows and keeps up to 8
// accumulators per element, one per site, so every row read serves all the
// block's sites.  Tokens go through a three-stage pipeline, one stage per pass
// and one named barrier per pass: the chunk warps score token p + 2 (split by
// source: each warp scores its sources against every query), take the softmax
// of token p + 1 (split by query), and mix token p.
#include <algorithm>
#include <type_traits>

#include "lrar.h"
#include "lrar_device.cuh"
#include "lrar_launch.h"
#include "lrar_sm100.cuh"

namespace lrar {

constexpr int kPh1MaxSites = 8;  // queries per phase-1 launch (more are split by the host)
constexpr int kPh1Stages = 16;   // ring depth of phase 1 (rows in flight per lane + 1; a power of two)
static_assert((kPh1Stages & (kPh1Stages - 1)) == 0, "the ring index wraps with a mask");

struct Ph1Params {
    SrcTab vt, kt;         // completed sources [T, d] each; P-LR keys [T, r] each
    int qpl;               // queries per lane of the per-source scoring (1 or 2); 0: scoring split by query
    const float *queries;  // [c][r]
    void *h_pre;           // [c][T][d]
    float *lse_pre;        // [c][T]
    int64_t T, site_stride;  // site_stride: elements between sites in h_pre (T * d)
    int n, c, d, r, chunks;
    float eps, inv_r;
    int sliced, key_vec;
    int *status;            // optional: LRAR_STATUS_WAIT_TIMEOUT when a key wait gives up
    long long wait_cycles;  // bound of each key wait
    int stall;              // test hook: key waits go to a barrier that never completes
    int tw;                 // weights kernel on the tensor cores: tokens per warp chunk
};

// Coordinate t of query j (zero past c and r), read from the caller's array.
__device__ __forceinline__ float q_init(const Ph1Params &p, int j, int t) {
    return (j < p.c && t < p.r) ? p.queries[j * p.r + t] : 0.f;
}

__device__ __forceinline__ void group_sync(int id, int threads) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}

// Key of source i at token x: the last r coordinates of the row (S-LR, Eq. 14)
// or the P-LR key row.
template <typename Tin>
__device__ __forceinline__ const Tin *ph1_key(const Ph1Params &p, int i, int64_t x) {
    return p.sliced ? src_row<Tin>(p.vt, i, x, p.d) + (p.d - p.r) : src_row<Tin>(p.kt, i, x, p.r);
}

// Staged keys of one token: key i at byte i * kstride of a group's buffer
// (r * sizeof(Tin) bytes, then 16 bytes of padding against bank conflicts).
template <typename Tin>
__host__ __device__ __forceinline__ int ph1_kstride(int r) {
    return r * (int)sizeof(Tin) + 16;
}

// Copy token x's n keys into a group buffer with bulk copies counted on bar
// (one warp: lane 0 announces the bytes, lane i copies key i).
template <typename Tin>
__device__ __forceinline__ void ph1_stage(const Ph1Params &p, int64_t x, int lane, uint32_t kbuf, uint32_t bar) {
    const uint32_t kbytes = (uint32_t)(p.r * (int)sizeof(Tin));
    if (lane == 0) sm100::mbar_arrive_expect_tx(bar, kbytes * (uint32_t)p.n);
    __syncwarp();
    for (int i = lane; i < p.n; i += 32)
        sm100::bulk_load(kbuf + (uint32_t)(i * ph1_kstride<Tin>(p.r)), ph1_key<Tin>(p, i, x), kbytes, bar);
}

// Scores of token x for QW queries j = j0, j0 + jstep, ... (Eq. 8-9), by one
// warp: s_ij goes to aw[i * kPh1MaxSites + j].  Keys that are whole 16-byte
// vectors and whose row of nv = r / E vectors divides a warp are scored lane
// per (source, key vector): each lane forms its vector's part of |k_i|^2 and of
// q_j . k_i, and the nv lanes of a source combine them with a fixed butterfly.
// Other keys take a lane per source.  kb_s: the token's keys staged in shared
// memory (null: read from global memory).
template <typename Tin, int QW>
__device__ __forceinline__ void ph1_scores(const Ph1Params &p, const float *__restrict__ q_s, int rp, int64_t x,
                                           int lane, int j0, int jstep, float *aw, const unsigned char *kb_s) {
    constexpr int E = VecE<Tin>::value;
    const int nv = p.r / E;
    if (p.key_vec && nv <= 32 && (32 % nv) == 0) {
        const int per = 32 / nv;  // sources per round
        const int v = lane % nv;
        for (int i0 = 0; i0 < p.n; i0 += per) {
            const int i = i0 + lane / nv;
            float k[E];
            if (i < p.n) {
                Frag<Tin, E> f;
                if (kb_s) f.a = *reinterpret_cast<const uint4 *>(kb_s + i * ph1_kstride<Tin>(p.r) + v * 16);
                else f.load_nc(ph1_key<Tin>(p, i, x) + v * E);
                f.get(k);
            } else {
#pragma unroll
                for (int t = 0; t < E; ++t) k[t] = 0.f;
            }
            float ss = 0.f, qk[QW];
#pragma unroll
            for (int t = 0; t < E; ++t) ss = fmaf(k[t], k[t], ss);
#pragma unroll
            for (int u = 0; u < QW; ++u) {
                qk[u] = 0.f;
                const float *qj = q_s + (j0 + u * jstep) * rp + v * E;
#pragma unroll
                for (int t = 0; t < E; t += 4) {
                    const float4 q4 = *reinterpret_cast<const float4 *>(qj + t);
                    qk[u] = fmaf(q4.x, k[t], qk[u]);
                    qk[u] = fmaf(q4.y, k[t + 1], qk[u]);
                    qk[u] = fmaf(q4.z, k[t + 2], qk[u]);
                    qk[u] = fmaf(q4.w, k[t + 3], qk[u]);
                }
            }
            for (int off = 1; off < nv; off <<= 1) {  // the source's lanes form an aligned group
                ss += __shfl_xor_sync(0xffffffffu, ss, off);
#pragma unroll
                for (int u = 0; u < QW; ++u) qk[u] += __shfl_xor_sync(0xffffffffu, qk[u], off);
            }
            if (v == 0 && i < p.n) {
                const float rho = rsqrtf(fmaf(ss, p.inv_r, p.eps));
#pragma unroll
                for (int u = 0; u < QW; ++u) aw[i * kPh1MaxSites + j0 + u * jstep] = rho * qk[u];
            }
        }
    } else {
        for (int i = lane; i < p.n; i += 32) {
            const Tin *kp = ph1_key<Tin>(p, i, x);
            float ss = 0.f, qk[QW];
#pragma unroll
            for (int u = 0; u < QW; ++u) qk[u] = 0.f;
            for (int t = 0; t < p.r; ++t) {
                const float kt = to_f(__ldg(kp + t));
                ss = fmaf(kt, kt, ss);
#pragma unroll
                for (int u = 0; u < QW; ++u) qk[u] = fmaf(q_s[(j0 + u * jstep) * rp + t], kt, qk[u]);
            }
            const float rho = rsqrtf(fmaf(ss, p.inv_r, p.eps));
#pragma unroll
            for (int u = 0; u < QW; ++u) aw[i * kPh1MaxSites + j0 + u * jstep] = rho * qk[u];
        }
    }
}

// Scores of token x split by query (keys that are not whole vectors, or too
// many queries per lane for the per-source split): this warp's queries
// j = ch, ch + chunks, ... < c against every source, into sc.
template <typename Tin>
__device__ __forceinline__ void ph1_scores_by_query(const Ph1Params &p, const float *__restrict__ q_s, int rp,
                                                    int64_t x, int ch, int lane, float *sc, const unsigned char *kb_s) {
    const int nq = ch < p.c ? (p.c - ch + p.chunks - 1) / p.chunks : 0;
    switch (nq) {  // queries of this warp: 8 / chunks when c = 8
        case 0: break;
        case 1: ph1_scores<Tin, 1>(p, q_s, rp, x, lane, ch, p.chunks, sc, kb_s); break;
        case 2: ph1_scores<Tin, 2>(p, q_s, rp, x, lane, ch, p.chunks, sc, kb_s); break;
        case 3: ph1_scores<Tin, 3>(p, q_s, rp, x, lane, ch, p.chunks, sc, kb_s); break;
        case 4: ph1_scores<Tin, 4>(p, q_s, rp, x, lane, ch, p.chunks, sc, kb_s); break;
        default: ph1_scores<Tin, 8>(p, q_s, rp, x, lane, ch, p.chunks, sc, kb_s); break;  // 5..8: chunks == 1
    }
}

// Scores of token x split by source (keys that are whole 16-byte vectors, nv =
// r / E of them dividing a warp): this warp scores sources i = chunks - 1 - ch,
// 2 chunks - 1 - ch, ... against every query.  Lane l holds key vector v = l % nv and the queries
// j = l / nv + u (32 / nv), u < QPL, whose vector v it reads from qv_s (float4
// t of query slot u at qv_s[(u E / 4 + t) 32 + l], conflict-free);
// the nv lanes of a source combine |k_i|^2 and the q_j . k_i parts with a fixed
// butterfly, the same arithmetic in the same order as the split by query, and
// lane v = 0 writes s_ij = rho_i (q_j . k_i) to sc[i * kPh1MaxSites + j].
template <typename Tin, int QPL>
__device__ __forceinline__ void ph1_scores_by_source(const Ph1Params &p, const float4 *__restrict__ qv_s, int64_t x,
                                                     int ch, int lane, float *sc, const unsigned char *kb_s) {
    constexpr int E = VecE<Tin>::value;
    const int nv = p.r / E;
    const int v = lane % nv, qg = lane / nv, gstep = 32 / nv;
    // sources chunks - 1 - ch, 2 chunks - 1 - ch, ...: warp 0, which also stages the
    // keys, is the last to take a second source
    for (int i = p.chunks - 1 - ch; i < p.n; i += p.chunks) {  // warp-uniform
        Frag<Tin, E> f;
        if (kb_s) f.a = *reinterpret_cast<const uint4 *>(kb_s + i * ph1_kstride<Tin>(p.r) + v * 16);
        else f.load_nc(ph1_key<Tin>(p, i, x) + v * E);
        float k[E];
        f.get(k);
        float ss = 0.f, qk[QPL];
#pragma unroll
        for (int t = 0; t < E; ++t) ss = fmaf(k[t], k[t], ss);
#pragma unroll
        for (int u = 0; u < QPL; ++u) {
            qk[u] = 0.f;
#pragma unroll
            for (int t = 0; t < E; t += 4) {
                const float4 q4 = qv_s[(u * (E / 4) + t / 4) * 32 + lane];
                qk[u] = fmaf(q4.x, k[t], qk[u]);
                qk[u] = fmaf(q4.y, k[t + 1], qk[u]);
                qk[u] = fmaf(q4.z, k[t + 2], qk[u]);
                qk[u] = fmaf(q4.w, k[t + 3], qk[u]);
            }
        }
        for (int off = 1; off < nv; off <<= 1) {  // the source's lanes form an aligned group
            ss += __shfl_xor_sync(0xffffffffu, ss, off);
#pragma unroll
            for (int u = 0; u < QPL; ++u) qk[u] += __shfl_xor_sync(0xffffffffu, qk[u], off);
        }
        if (v == 0) {
            const float rho = rsqrtf(fmaf(ss, p.inv_r, p.eps));
#pragma unroll
            for (int u = 0; u < QPL; ++u) {
                const int j = qg + u * gstep;
                if (j < p.c) sc[i * kPh1MaxSites + j] = rho * qk[u];
            }
        }
    }
}

// Softmax of token x (Eq. 10) for the queries j = ch, ch + chunks, ... < c:
// weights alpha_ij = exp(s_ij - lse_j) to aw[i * kPh1MaxSites + j], lse_j to
// lse_pre, from the scores in sc.
__device__ __forceinline__ void ph1_softmax(const Ph1Params &p, int64_t x, int ch, int lane, const float *sc,
                                            float *aw) {
    for (int j = ch; j < p.c; j += p.chunks) {
        float m = -INFINITY;
        for (int i = lane; i < p.n; i += 32) m = fmaxf(m, sc[i * kPh1MaxSites + j]);
        m = warp_max(m);
        float z = 0.f;
        for (int i = lane; i < p.n; i += 32) z += expf(sc[i * kPh1MaxSites + j] - m);
        z = warp_sum(z);
        for (int i = lane; i < p.n; i += 32) aw[i * kPh1MaxSites + j] = expf(sc[i * kPh1MaxSites + j] - m) / z;
        if (lane == 0) p.lse_pre[(int64_t)j * p.T + x] = m + logf(z);
    }
}

// One row of phase 1's mix: acc_j (+)= alpha_ij o_i for the sites j < c, the
// row in f and its weights at aw[j] (FIRST: acc_j = alpha_ij o_i, used with
// all eight sites only).
template <typename Tin, int E, bool C8, bool FIRST>
__device__ __forceinline__ void ph1_row(float (&acc)[kPh1MaxSites][E], const Frag<Tin, E> &f,
                                        const float *__restrict__ aw, int c) {
    float o[E], w[kPh1MaxSites];
    f.get(o);
    const float4 w0 = *reinterpret_cast<const float4 *>(aw);
    const float4 w1 = *reinterpret_cast<const float4 *>(aw + 4);
    w[0] = w0.x, w[1] = w0.y, w[2] = w0.z, w[3] = w0.w, w[4] = w1.x, w[5] = w1.y, w[6] = w1.z, w[7] = w1.w;
#pragma unroll
    for (int j = 0; j < kPh1MaxSites; ++j) {
        if (C8 || j < c) {
#pragma unroll
            for (int t = 0; t < E; t += 2) {
                if (FIRST) {
                    const float2 m = __fmul2_rn(make_float2(w[j], w[j]), make_float2(o[t], o[t + 1]));
                    acc[j][t] = m.x;
                    acc[j][t + 1] = m.y;
                } else {
                    fma2(acc[j][t], acc[j][t + 1], w[j], w[j], o[t], o[t + 1]);
                }
            }
        }
    }
}

// Phase 1 (§3.5): in pass p a token group's warps score the group's token
// p + 2, take the softmax of token p + 1 and mix the n rows of token p into c
// sites; scores and weights pass through shared memory (double-buffered by
// token), and the pass ends at the group's named barrier.
//   Rows stream through a per-lane cp.async ring (each lane copies and reads
//   back its own 16-byte vector of every row), S - 1 rows ahead and across
//   tokens, so the next token's rows travel while this one is mixed.
//   KS: each group's keys are staged three tokens ahead in shared memory with
//   bulk copies (double-buffered, one mbarrier per buffer) by the group's warp
//   0, so scoring reads no global memory.  Each warp's wait for them is
//   bounded (p.wait_cycles) and decided for the whole warp; one that runs out
//   ORs LRAR_STATUS_WAIT_TIMEOUT into *p.status and raises the CTA's abort
//   flag, after which no warp waits again and no group issues another copy.
//   A copy into a buffer follows the barrier that ends the pass in which its
//   previous token was waited for, so a give-up is always seen before the
//   buffer is reused, and each buffer holds at most one phase that no wait
//   confirmed; the issuing warp waits (bounded) for that one before the CTA
//   exits, so no copy lands in released shared memory.  A launch that gave up
//   writes outputs that are not valid.
//   C8: exactly eight sites (compile-time loop bounds); else p.c <= 8.
//   FULLW: every lane's vector lies inside the row (d = chunks * 32 * E).
template <typename Tin, typename Tout, int S, bool KS, bool C8, bool FULLW>
__global__ void __launch_bounds__(kThreads, 2) block_phase1_kernel(const __grid_constant__ Ph1Params p) {
    pdl_enter();
    constexpr int E = VecE<Tin>::value;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int rp = round_up(p.r, 4);
    const int G = kWarps / p.chunks;  // token groups per CTA
    const int kbuf_bytes = KS ? round_up(p.n * ph1_kstride<Tin>(p.r), 16) : 0;  // one token's keys
    unsigned char *kb_all = smem_raw + (size_t)kWarps * S * 32 * 16;           // [G][2][kbuf_bytes]
    uint64_t *kbar_all = reinterpret_cast<uint64_t *>(kb_all + (size_t)G * 2 * kbuf_bytes);  // [G][2]
    int *conf_all = reinterpret_cast<int *>(kbar_all + (KS ? 2 * G : 0));     // [G][2] phases seen complete
    // q_s starts 16-byte aligned: the barriers and counters take round_up(G * 2 * 12, 16) bytes
    float *q_s = reinterpret_cast<float *>(reinterpret_cast<unsigned char *>(kbar_all) +
                                           (KS ? round_up(G * 2 * (8 + 4), 16) : 0));  // [8][rp], zero past c and r
    float *a_all = q_s + kPh1MaxSites * rp;  // [G][2][n][8]: weights, double-buffered by token
    float *s_all = a_all + (size_t)G * 2 * kPh1MaxSites * p.n;  // [G][2][n][8]: scores, double-buffered by token
    float4 *qv_s = reinterpret_cast<float4 *>(s_all + (size_t)G * 2 * kPh1MaxSites * p.n);  // [2][E / 4][32]
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int g = warp / p.chunks, ch = warp % p.chunks;
    const int nthr = p.chunks * 32;  // threads of a token group (named barrier 1 + g)
    __shared__ int abort_s;           // set once a key wait of this CTA gave up
    __shared__ __align__(8) uint64_t never_bar;  // test hook: a barrier nothing arrives on
    volatile int *abort = &abort_s;
    for (int j = threadIdx.x; j < kPh1MaxSites * rp; j += kThreads) {
        const int jj = j / rp, t = j % rp;
        q_s[j] = (jj < p.c && t < p.r) ? p.queries[jj * p.r + t] : 0.f;
    }
    if (threadIdx.x < 2 * (E / 4) * 32) {  // per-lane query vectors of the per-source split
        const int l = threadIdx.x % 32, ut = threadIdx.x / 32, u = ut / (E / 4), t4 = ut % (E / 4);
        const int nvq = p.qpl ? p.r / E : 1;
        const int j = l / nvq + u * (32 / nvq), t = (l % nvq) * E + 4 * t4;
        const bool ok = u < p.qpl && j < kPh1MaxSites;
        qv_s[threadIdx.x] = ok ? make_float4(q_init(p, j, t), q_init(p, j, t + 1), q_init(p, j, t + 2), q_init(p, j, t + 3))
                               : make_float4(0.f, 0.f, 0.f, 0.f);
    }
    if (KS && threadIdx.x < 2 * G) {
        sm100::mbar_init(smem_u32(kbar_all + threadIdx.x), 1);
        conf_all[threadIdx.x] = 0;
        sm100::mbar_fence_init();
    }
    if (threadIdx.x == 0) {
        abort_s = 0;
        if (KS) {
            sm100::mbar_init(smem_u32(&never_bar), 1);
            sm100::mbar_fence_init();
        }
    }
    __syncthreads();

    Tout *__restrict__ h_pre = static_cast<Tout *>(p.h_pre);
    const int e = (ch * 32 + lane) * E;  // this lane's first element of the row
    float *aw0 = a_all + (size_t)g * 2 * kPh1MaxSites * p.n;
    float *sc0 = s_all + (size_t)g * 2 * kPh1MaxSites * p.n;
    auto awb = [&](int q) { return aw0 + (q & 1) * kPh1MaxSites * p.n; };  // weights of the group's token q
    auto scb = [&](int q) { return sc0 + (q & 1) * kPh1MaxSites * p.n; };  // scores of the group's token q
    const int64_t stride = (int64_t)gridDim.x * G;
    const uint32_t ring_w = smem_u32(smem_raw) + (uint32_t)(warp * S * 32 * 16) + 16u * lane;
    unsigned char *kb0 = kb_all + (size_t)g * 2 * kbuf_bytes;
    int *conf = conf_all + 2 * g;
    auto kbuf = [&](int b) { return smem_u32(kb0 + b * kbuf_bytes); };
    auto kbar = [&](int b) { return smem_u32(kbar_all + 2 * g + b); };
    // token q of this group (x0 + q * stride) uses key buffer q % 2, for the (q / 2)-th time
    auto kwait = [&](int q) {
        if (__any_sync(0xffffffffu, *abort != 0)) return;  // the CTA gave up: no further waits
        const uint32_t bar = p.stall ? smem_u32(&never_bar) : kbar(q & 1);
        const uint32_t par = p.stall ? 0u : (uint32_t)(q >> 1) & 1u;
        if (__all_sync(0xffffffffu, sm100::mbar_wait(bar, par, p.wait_cycles, abort))) {
            if (lane == 0 && ch == 0) conf[q & 1] = (q >> 1) + 1;
        } else if (lane == 0) {
            *abort = 1;
            if (p.status) atomicOr(p.status, LRAR_STATUS_WAIT_TIMEOUT);
        }
    };
    uint32_t issued0 = 0u, issued1 = 0u;  // the issuing warp's phases per buffer
    auto stage = [&](int64_t xx, int b) {  // warp 0 of the group, unless the CTA gave up
        if (__any_sync(0xffffffffu, *abort != 0)) return;
        ph1_stage<Tin>(p, xx, lane, kbuf(b), kbar(b));
        if (b) ++issued1;
        else ++issued0;
    };
    auto score = [&](int q, int64_t xx) {  // token q = xx of the group: this warp's share of the scores
        if (KS) kwait(q);
        const unsigned char *kb = KS ? kb0 + (q & 1) * kbuf_bytes : nullptr;
        if (p.qpl == 2) ph1_scores_by_source<Tin, 2>(p, qv_s, xx, ch, lane, scb(q), kb);
        else if (p.qpl == 1) ph1_scores_by_source<Tin, 1>(p, qv_s, xx, ch, lane, scb(q), kb);
        else ph1_scores_by_query<Tin>(p, q_s, rp, xx, ch, lane, scb(q), kb);
    };

    int64_t x = (int64_t)blockIdx.x * G + g;
    // the ring: this lane's next copy is its vector of source ii's row at element
    // offset xoff (the group's token times d, plus e); rows_left copies remain
    const bool cp_lane = FULLW || e < p.d;
    const int64_t xstep = stride * p.d;
    int64_t xoff = x * p.d + e;
    int ii = 0;
    int rows_left = x < p.T ? (int)((p.T - x + stride - 1) / stride) * p.n : 0;  // warp-uniform
    uint32_t wslot = ring_w;  // shared address the next copy goes to
    const uint32_t ring_end = ring_w + 16u * 32u * S;
    auto issue = [&]() {
        if (rows_left > 0) {
            if (cp_lane) cp_async16(wslot, static_cast<const Tin *>(p.vt.p[ii]) + xoff);
            --rows_left;
            if (++ii == p.n) {
                ii = 0;
                xoff += xstep;
            }
        }
        cp_async_commit();
        wslot += 16u * 32u;
        if (wslot == ring_end) wslot = ring_w;
    };
#pragma unroll
    for (int st = 0; st < S - 1; ++st) issue();
    uint32_t rslot = ring_w;  // shared address of the next row to read
    // Within a token each row is read from the ring one row ahead of its use:
    // with K rows of the stream mixed before the token, K + S - 1 + i copies
    // have been issued when row K + i is read, and the wait that leaves at most
    // S - 2 of them pending means rows up to K + i have landed.  Each copy
    // refills the slot of a row whose value a multiply-add has already used.
    Frag<Tin, E> f;
    auto read_row = [&]() {
        if (cp_lane) f.a = ld_shared16(rslot);
        else f.zero();
        rslot += 16u * 32u;
        if (rslot == ring_end) rslot = ring_w;
    };
    auto next_row = [&]() {
        issue();
        cp_async_wait<S - 2>();
        read_row();
    };

    // prologue: token 0 scored; then token 1 scored and token 0's softmax
    if (KS && ch == 0) {
        if (x < p.T) stage(x, 0);
        if (x + stride < p.T) stage(x + stride, 1);
    }
    if (x < p.T) score(0, x);
    group_sync(1 + g, nthr);
    if (KS && ch == 0 && x + 2 * stride < p.T) stage(x + 2 * stride, 0);  // buffer 0 held token 0, scored above
    if (x < p.T) ph1_softmax(p, x, ch, lane, scb(0), awb(0));
    if (x + stride < p.T) score(1, x + stride);
    group_sync(1 + g, nthr);
    for (int pass = 0; (int64_t)blockIdx.x * G + pass * stride < p.T; ++pass, x += stride) {
        const float *aw = awb(pass);
        // key buffer (pass + 1) % 2 held token pass + 1, scored before the last barrier
        if (KS && ch == 0 && x + 3 * stride < p.T) stage(x + 3 * stride, (pass + 1) & 1);
        if (x + stride < p.T) ph1_softmax(p, x + stride, ch, lane, scb(pass + 1), awb(pass + 1));
        if (x + 2 * stride < p.T) score(pass + 2, x + 2 * stride);
        if (x < p.T) {
            // the next row is read from the ring before this row's multiply-adds,
            // so its shared-memory latency overlaps them; row 0 starts the
            // accumulators with a product (the value of a multiply-add onto zero)
            float acc[kPh1MaxSites][E];
            cp_async_wait<S - 2>();
            read_row();
            if (C8) {
                ph1_row<Tin, E, C8, true>(acc, f, aw, p.c);
            } else {  // fewer sites: zero, then every row as a multiply-add (fewer live values)
#pragma unroll
                for (int j = 0; j < kPh1MaxSites; ++j)
#pragma unroll
                    for (int t = 0; t < E; ++t) acc[j][t] = 0.f;
                ph1_row<Tin, E, C8, false>(acc, f, aw, p.c);
            }
            for (int i = 1; i < p.n; ++i) {
                next_row();
                ph1_row<Tin, E, C8, false>(acc, f, aw + i * kPh1MaxSites, p.c);
            }
            issue();  // the stream stays S - 1 copies ahead of the next token's first row
            if (FULLW || e < p.d) {
                Tout *hp = h_pre + x * p.d + e;
#pragma unroll
                for (int j = 0; j < kPh1MaxSites; ++j) {
                    if (C8 || j < p.c) {
                        Frag<Tout, E> out;
                        out.set(acc[j]);
                        out.store(hp + (int64_t)j * p.site_stride);
                    }
                }
            }
        }
        group_sync(1 + g, nthr);  // next weights and scores complete; this pass's weights free for reuse
    }
    cp_async_wait_all();
    if (KS && ch == 0)  // drain: the one phase per buffer a give-up may have left unconfirmed
        for (int b = 0; b < 2; ++b) {
            const uint32_t iss = b ? issued1 : issued0, done = (uint32_t)conf[b];
            if (iss > done && !__all_sync(0xffffffffu, sm100::mbar_wait(kbar(b), (iss - 1u) & 1u, p.wait_cycles)) &&
                lane == 0 && p.status)
                atomicOr(p.status, LRAR_STATUS_WAIT_TIMEOUT);
        }
}

// ----------------------------------------------------- split phase 1 ----
// Phase 1 in two kernels, for shapes whose weights fit one row of h_pre:
//   block_weights_kernel (bf16 keys of depth 16..64: block_weights_mma_kernel,
//       the scores on the tensor cores)  computes s_ij (Eq. 8-9) for every
//       completed source i and site j, the softmax over i (Eq. 10) and lse_j,
//       writes lse_j to lse_pre and alpha_ij as fp32 at float i * 8 + j of the
//       token's row of the last site's h_pre, which serves as scratch;
//   block_mix_kernel  the mix of phase 1 with those weights: in pass p a token
//       group copies token p + 1's weights from that row into shared memory and
//       mixes token p, whose row the last site then overwrites with its h_pre.
//       Its first source rows stream in while the weights kernel finishes.
// The mix carries no scoring, so its instructions go to the row stream and
// the multiply-adds.

// The fp32 weight row of token x: the start of the last site's h_pre row.
template <typename Tout>
__device__ __forceinline__ float *ph1_weight_row(const Ph1Params &p, int64_t x) {
    return reinterpret_cast<float *>(static_cast<Tout *>(p.h_pre) + (int64_t)(p.c - 1) * p.site_stride + x * p.d);
}

// Scores of kWTok tokens at once (keys that are whole 16-byte vectors whose
// nv = r / E vectors divide a warp): lane (source i0 + l / nv, vector l % nv)
// loads its key vector of every round and token before any arithmetic, so the
// loads of all of them are in flight together; then, round by round, |k|^2 and
// the eight q_j . k products (a fixed butterfly over the nv lanes, the
// arithmetic of ph1_scores) give s_ij = rho_i (q_j . k_i) in sc[t][i][j].
constexpr int kWTok = 2;     // tokens per warp and iteration of the weights kernel
constexpr int kWRounds = 4;  // source rounds whose key vectors are held at once
template <typename Tin>
__device__ __forceinline__ void ph1_scores_batch(const Ph1Params &p, const float *__restrict__ q_s, int rp,
                                                 const int64_t (&xs)[kWTok], int lane, float *sc) {
    constexpr int E = VecE<Tin>::value;
    const int nv = p.r / E, per = 32 / nv, v = lane % nv, so = lane / nv;
    for (int i0 = 0; i0 < p.n; i0 += kWRounds * per) {
        Frag<Tin, E> k[kWTok][kWRounds];
#pragma unroll
        for (int t = 0; t < kWTok; ++t)
#pragma unroll
            for (int rr = 0; rr < kWRounds; ++rr) {
                const int i = i0 + rr * per + so;
                if (xs[t] < p.T && i < p.n) k[t][rr].load_nc(ph1_key<Tin>(p, i, xs[t]) + v * E);
                else k[t][rr].zero();
            }
#pragma unroll
        for (int t = 0; t < kWTok; ++t)
#pragma unroll
            for (int rr = 0; rr < kWRounds; ++rr) {
                const int i = i0 + rr * per + so;
                if (i0 + rr * per >= p.n) break;  // warp-uniform
                float kv[E];
                k[t][rr].get(kv);
                float ss = 0.f, qk[kPh1MaxSites];
#pragma unroll
                for (int e = 0; e < E; ++e) ss = fmaf(kv[e], kv[e], ss);
#pragma unroll
                for (int j = 0; j < kPh1MaxSites; ++j) {
                    qk[j] = 0.f;
                    const float *qj = q_s + j * rp + v * E;
#pragma unroll
                    for (int e = 0; e < E; e += 4) {
                        const float4 q4 = *reinterpret_cast<const float4 *>(qj + e);
                        qk[j] = fmaf(q4.x, kv[e], qk[j]);
                        qk[j] = fmaf(q4.y, kv[e + 1], qk[j]);
                        qk[j] = fmaf(q4.z, kv[e + 2], qk[j]);
                        qk[j] = fmaf(q4.w, kv[e + 3], qk[j]);
                    }
                }
                for (int off = 1; off < nv; off <<= 1) {  // the source's lanes form an aligned group
                    ss += __shfl_xor_sync(0xffffffffu, ss, off);
#pragma unroll
                    for (int j = 0; j < kPh1MaxSites; ++j) qk[j] += __shfl_xor_sync(0xffffffffu, qk[j], off);
                }
                if (v == 0 && i < p.n) {
                    const float rho = rsqrtf(fmaf(ss, p.inv_r, p.eps));
#pragma unroll
                    for (int j = 0; j < kPh1MaxSites; ++j) sc[(t * p.n + i) * kPh1MaxSites + j] = rho * qk[j];
                }
            }
    }
}

template <typename Tin, typename Tout>
__global__ void __launch_bounds__(kThreads) block_weights_kernel(const __grid_constant__ Ph1Params p) {
    pdl_enter();
    extern __shared__ __align__(16) float wsm[];
    const int rp = round_up(p.r, 4);
    float *q_s = wsm;                                       // [8][rp], zero past c and r
    float *sc_all = q_s + kPh1MaxSites * rp;                // [kWarps][kWTok][n][8]
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int j = threadIdx.x; j < kPh1MaxSites * rp; j += kThreads) {
        const int jj = j / rp, t = j % rp;
        q_s[j] = (jj < p.c && t < p.r) ? p.queries[jj * p.r + t] : 0.f;
    }
    __syncthreads();
    float *sc = sc_all + (size_t)warp * kWTok * kPh1MaxSites * p.n;
    const int nv = p.key_vec ? p.r / VecE<Tin>::value : 0;
    const bool batch = nv >= 1 && nv <= 32 && 32 % nv == 0;
    const int j = lane >> 2, slot = lane & 3;  // softmax: lane (j, slot) takes sources slot, slot + 4, ...
    const int64_t wstride = (int64_t)gridDim.x * kWarps;
    for (int64_t x0 = ((int64_t)blockIdx.x * kWarps + warp) * kWTok; x0 < p.T; x0 += wstride * kWTok) {
        int64_t xs[kWTok];
#pragma unroll
        for (int t = 0; t < kWTok; ++t) xs[t] = x0 + t;
        if (batch) {
            ph1_scores_batch<Tin>(p, q_s, rp, xs, lane, sc);
        } else {
            for (int t = 0; t < kWTok; ++t)
                if (xs[t] < p.T) ph1_scores<Tin, kPh1MaxSites>(p, q_s, rp, xs[t], lane, 0, 1, sc + t * p.n * kPh1MaxSites, nullptr);
        }
        __syncwarp();
#pragma unroll
        for (int t = 0; t < kWTok; ++t) {
            if (xs[t] >= p.T) break;  // warp-uniform
            const float *st = sc + t * p.n * kPh1MaxSites;
            float m = -INFINITY;
            for (int i = slot; i < p.n; i += 4) m = fmaxf(m, st[i * kPh1MaxSites + j]);
            m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, 1));
            m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, 2));
            float z = 0.f;
            for (int i = slot; i < p.n; i += 4) z += expf(st[i * kPh1MaxSites + j] - m);
            z += __shfl_xor_sync(0xffffffffu, z, 1);
            z += __shfl_xor_sync(0xffffffffu, z, 2);
            float *wrow = ph1_weight_row<Tout>(p, xs[t]);
            if (j < p.c) {
                for (int i = slot; i < p.n; i += 4) wrow[i * kPh1MaxSites + j] = expf(st[i * kPh1MaxSites + j] - m) / z;
                if (slot == 0) p.lse_pre[(int64_t)j * p.T + xs[t]] = m + logf(z);
            }
        }
        __syncwarp();  // the scores are rewritten for the next tokens
    }
}

// ---------------------------------------------- weights on the tensor cores ----
// With bf16 keys of depth r = 16 KS the scores of a chunk of tokens are one
// small contraction: rows are the chunk's (token, source) pairs, columns the
// c <= 8 queries.  It runs as m16n8k16 MMAs.  Each fp32 query coordinate is
// split exactly into three bf16 parts q = q1 + q2 + q3 (each part the bf16
// rounding of what the previous ones leave, so that together they carry q's
// 24-bit significand); every bf16 product q_u k is exact and the MMA sums in
// fp32, so s_ij = rho_i (q_j . k_i) comes out with fp32 accuracy.  The depth
// index is permuted so that lane t of a quad holds one contiguous quarter of a
// key row (depth 4 KS t ... 4 KS t + 4 KS - 1): depth 4 KS t + 4 s + {0, 1} is
// column {2t, 2t + 1} of k-step s and 4 KS t + 4 s + {2, 3} column
// {2t + 8, 2t + 9}; the queries take the same permutation, which leaves the
// contraction unchanged.  |k_i|^2 comes from the same registers (mixed-precision
// multiply-adds, then the quad's four lanes).
__device__ __forceinline__ void mma_bf16_16816(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                               uint32_t b0, uint32_t b1) {
    asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// ss += lo^2 + hi^2 of a bf16 pair (exact products, fp32 sums).
__device__ __forceinline__ void sumsq_bf16x2(float &ss, uint32_t w) {
    asm("{\n\t.reg .b16 l, h;\n\tmov.b32 {l, h}, %1;\n\t"
        "fma.rn.f32.bf16 %0, l, l, %0;\n\tfma.rn.f32.bf16 %0, h, h, %0;\n\t}"
        : "+f"(ss)
        : "r"(w));
}

// The three bf16 parts of x (x = u0 + u1 + u2 up to 2^-27 |x|).
__device__ __forceinline__ void split3_bf16(float x, bf16 (&u)[3]) {
#pragma unroll
    for (int k = 0; k < 3; ++k) {
        u[k] = __float2bfloat16_rn(x);
        x -= __bfloat162float(u[k]);  // exact: the rounding error of a bf16 rounding is an fp32 number
    }
}

__device__ __forceinline__ uint32_t pack_bf16(bf16 lo, bf16 hi) {
    return (uint32_t)__bfloat16_as_ushort(lo) | ((uint32_t)__bfloat16_as_ushort(hi) << 16);
}

template <typename Tout, int KS>
__global__ void __launch_bounds__(kThreads, 2) block_weights_mma_kernel(const __grid_constant__ Ph1Params p) {
    pdl_enter();
    constexpr int W = 2 * KS;                  // bf16 pairs of a key row per lane
    constexpr int G = KS >= 3 ? 4 : 8 / KS;    // tiles of 16 pairs whose rows are loaded together
    extern __shared__ __align__(16) float wsm[];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int g = lane >> 2, t4 = lane & 3;
    const int tw = p.tw, n = p.n;
    float *sc = wsm + (size_t)warp * tw * n * kPh1MaxSites;  // [tw * n][8] scores of the warp's chunk
    // B fragments: query g's depth quarter t4, three parts each
    uint32_t qb[3][KS][2];
#pragma unroll
    for (int s = 0; s < KS; ++s)
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int e = 4 * KS * t4 + 4 * s + 2 * h;
            bf16 u0[3], u1[3];
            split3_bf16(g < p.c ? p.queries[g * p.r + e] : 0.f, u0);
            split3_bf16(g < p.c ? p.queries[g * p.r + e + 1] : 0.f, u1);
#pragma unroll
            for (int k = 0; k < 3; ++k) qb[k][s][h] = pack_bf16(u0[k], u1[k]);
        }
    const uint64_t magic = 0xFFFFFFFFull / (uint32_t)n + 1;  // P / n = (P * magic) >> 32 for P < 2^32 / n
    const int64_t nchunks = (p.T + tw - 1) / tw;
    for (int64_t ch = (int64_t)blockIdx.x * kWarps + warp; ch < nchunks; ch += (int64_t)gridDim.x * kWarps) {
        const int64_t x0 = ch * tw;
        const int tcount = (int)(p.T - x0 < tw ? p.T - x0 : tw);
        const int np = tcount * n;  // pairs (token u, source i) at u * n + i
        for (int tile0 = 0; tile0 * 16 < np; tile0 += G) {
            uint32_t w[G][2][W];  // rows g and g + 8 of each tile
#pragma unroll
            for (int gi = 0; gi < G; ++gi)
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int P = (tile0 + gi) * 16 + g + 8 * h;
                    if (P < np) {
                        const int u = (int)(((uint64_t)P * magic) >> 32), i = P - u * n;
                        const bf16 *kr = ph1_key<bf16>(p, i, x0 + u) + 4 * KS * t4;
                        if constexpr (KS % 2 == 0) {
#pragma unroll
                            for (int v = 0; v < KS / 2; ++v) {
                                const uint4 q4 = ld_nc16(kr + 8 * v);
                                w[gi][h][4 * v] = q4.x; w[gi][h][4 * v + 1] = q4.y;
                                w[gi][h][4 * v + 2] = q4.z; w[gi][h][4 * v + 3] = q4.w;
                            }
                        } else {
#pragma unroll
                            for (int v = 0; v < KS; ++v) {
                                const uint2 q2 = ld_nc8(kr + 4 * v);
                                w[gi][h][2 * v] = q2.x; w[gi][h][2 * v + 1] = q2.y;
                            }
                        }
                    } else {
#pragma unroll
                        for (int v = 0; v < W; ++v) w[gi][h][v] = 0u;
                    }
                }
#pragma unroll
            for (int gi = 0; gi < G; ++gi) {
                const int P0 = (tile0 + gi) * 16 + g;
                if ((tile0 + gi) * 16 >= np) break;  // warp-uniform
                float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                for (int k = 2; k >= 0; --k)  // smallest parts first
#pragma unroll
                    for (int s = 0; s < KS; ++s)
                        mma_bf16_16816(acc, w[gi][0][2 * s], w[gi][1][2 * s], w[gi][0][2 * s + 1], w[gi][1][2 * s + 1],
                                       qb[k][s][0], qb[k][s][1]);
                float ss0 = 0.f, ss1 = 0.f;
#pragma unroll
                for (int v = 0; v < W; ++v) {
                    sumsq_bf16x2(ss0, w[gi][0][v]);
                    sumsq_bf16x2(ss1, w[gi][1][v]);
                }
                ss0 += __shfl_xor_sync(0xffffffffu, ss0, 1);
                ss1 += __shfl_xor_sync(0xffffffffu, ss1, 1);
                ss0 += __shfl_xor_sync(0xffffffffu, ss0, 2);
                ss1 += __shfl_xor_sync(0xffffffffu, ss1, 2);
                const float rho0 = rsqrtf(fmaf(ss0, p.inv_r, p.eps)), rho1 = rsqrtf(fmaf(ss1, p.inv_r, p.eps));
                if (P0 < np)
                    *reinterpret_cast<float2 *>(sc + P0 * kPh1MaxSites + 2 * t4) = make_float2(rho0 * acc[0], rho0 * acc[1]);
                if (P0 + 8 < np)
                    *reinterpret_cast<float2 *>(sc + (P0 + 8) * kPh1MaxSites + 2 * t4) =
                        make_float2(rho1 * acc[2], rho1 * acc[3]);
            }
        }
        __syncwarp();
        // softmax over the sources: lane (u0, j) takes tokens u0, u0 + 4, ... of the chunk for query j
        const int j = lane & 7;
        for (int u = lane >> 3; u < tcount; u += 4) {
            float *st = sc + u * n * kPh1MaxSites + j;
            float m = -INFINITY;
            for (int i = 0; i < n; ++i) m = fmaxf(m, st[i * kPh1MaxSites]);
            float z = 0.f;
            for (int i = 0; i < n; ++i) {
                const float e = expf(st[i * kPh1MaxSites] - m);
                st[i * kPh1MaxSites] = e;
                z += e;
            }
            if (j < p.c) {
                float *wrow = ph1_weight_row<Tout>(p, x0 + u);
                for (int i = 0; i < n; ++i) wrow[i * kPh1MaxSites + j] = st[i * kPh1MaxSites] / z;
                p.lse_pre[(int64_t)j * p.T + x0 + u] = m + logf(z);
            }
        }
        __syncwarp();  // the scores are rewritten for the next chunk
    }
}

template <typename Tin, typename Tout, int S, bool C8, bool FULLW>
__global__ void __launch_bounds__(kThreads, 2) block_mix_kernel(const __grid_constant__ Ph1Params p) {
    constexpr int E = VecE<Tin>::value;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int G = kWarps / p.chunks;  // token groups per CTA
    float *a_all = reinterpret_cast<float *>(smem_raw + (size_t)kWarps * S * 32 * 16);  // [G][2][n][8]
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int g = warp / p.chunks, ch = warp % p.chunks;
    const int nthr = p.chunks * 32;
    const int gt = ch * 32 + lane;  // thread index within the group
    Tout *__restrict__ h_pre = static_cast<Tout *>(p.h_pre);
    const int e = (ch * 32 + lane) * E;
    float *aw0 = a_all + (size_t)g * 2 * kPh1MaxSites * p.n;
    auto awb = [&](int q) { return aw0 + (q & 1) * kPh1MaxSites * p.n; };
    const int n4 = p.n * kPh1MaxSites / 4;  // 16-byte pieces of a token's weights
    auto fetch = [&](int q, int64_t xx) {   // token q = xx of the group: its weights into shared memory
        const float4 *src = reinterpret_cast<const float4 *>(ph1_weight_row<Tout>(p, xx));
        float4 *dst = reinterpret_cast<float4 *>(awb(q));
        for (int t = gt; t < n4; t += nthr) dst[t] = src[t];
    };
    const int64_t stride = (int64_t)gridDim.x * G;
    const uint32_t ring_w = smem_u32(smem_raw) + (uint32_t)(warp * S * 32 * 16) + 16u * lane;

    int64_t x = (int64_t)blockIdx.x * G + g;
    const bool cp_lane = FULLW || e < p.d;
    const int64_t xstep = stride * p.d;
    int64_t xoff = x * p.d + e;
    int ii = 0;
    int rows_left = x < p.T ? (int)((p.T - x + stride - 1) / stride) * p.n : 0;  // warp-uniform
    uint32_t wslot = ring_w;
    const uint32_t ring_end = ring_w + 16u * 32u * S;
    auto issue = [&]() {
        if (rows_left > 0) {
            if (cp_lane) cp_async16(wslot, static_cast<const Tin *>(p.vt.p[ii]) + xoff);
            --rows_left;
            if (++ii == p.n) {
                ii = 0;
                xoff += xstep;
            }
        }
        cp_async_commit();
        wslot += 16u * 32u;
        if (wslot == ring_end) wslot = ring_w;
    };
#pragma unroll
    for (int st = 0; st < S - 1; ++st) issue();
    // The first rows stream in before the wait: they are completed sources,
    // written before the weights kernel that precedes this grid began, and that
    // kernel lets this grid start only after its own wait on its predecessors.
    // The weights, that kernel's output, are read after the wait.
    pdl_wait();
    pdl_launch_dependents();
    uint32_t rslot = ring_w;
    Frag<Tin, E> f;
    auto read_row = [&]() {
        if (cp_lane) f.a = ld_shared16(rslot);
        else f.zero();
        rslot += 16u * 32u;
        if (rslot == ring_end) rslot = ring_w;
    };
    auto next_row = [&]() {
        issue();
        cp_async_wait<S - 2>();
        read_row();
    };

    if (x < p.T) fetch(0, x);
    group_sync(1 + g, nthr);
    for (int pass = 0; (int64_t)blockIdx.x * G + pass * stride < p.T; ++pass, x += stride) {
        const float *aw = awb(pass);
        // token pass + 1's weights: its h_pre rows are written only in the next pass
        if (x + stride < p.T) fetch(pass + 1, x + stride);
        if (x < p.T) {
            float acc[kPh1MaxSites][E];
            cp_async_wait<S - 2>();
            read_row();
            if (C8) {
                ph1_row<Tin, E, C8, true>(acc, f, aw, p.c);
            } else {
#pragma unroll
                for (int j = 0; j < kPh1MaxSites; ++j)
#pragma unroll
                    for (int t = 0; t < E; ++t) acc[j][t] = 0.f;
                ph1_row<Tin, E, C8, false>(acc, f, aw, p.c);
            }
            for (int i = 1; i < p.n; ++i) {
                next_row();
                ph1_row<Tin, E, C8, false>(acc, f, aw + i * kPh1MaxSites, p.c);
            }
            issue();  // the stream stays S - 1 copies ahead of the next token's first row
            if (FULLW || e < p.d) {
                Tout *hp = h_pre + x * p.d + e;
#pragma unroll
                for (int j = 0; j < kPh1MaxSites; ++j) {
                    if (C8 || j < p.c) {
                        Frag<Tout, E> out;
                        out.set(acc[j]);
                        out.store(hp + (int64_t)j * p.site_stride);
                    }
                }
            }
        }
        group_sync(1 + g, nthr);  // next weights copied; this token's weight row is overwritten
    }
    cp_async_wait_all();
}

struct Ph2Params {
    const void *h_pre, *partial, *pkeys;
    const void *prev, *prev_keys;  // assembling: the running sum before the member (then partial / pkeys are
                                   // the member's output / key, replaced by the sum)
    const float *lse_pre, *query;
    void *h;
    float *lse;
    int64_t T;
    int d, r;
    float eps, inv_r;
    int sliced;
};

// Phase 2: one warp per token merges h_pre with the partial-block summary.
// Each lane reads its elements of h_pre (and lane 0 lse_pre) before it writes
// the same elements of h (and lse), so h may be h_pre and lse may be lse_pre.
// Assembling (p.prev set), the partial summary is first formed from the
// running sum before the newest member and that member's output (Eq. 6): the
// fp32 sum rounded once to the stack type, as lrar_block_accumulate forms it,
// written over the member and used as read back.
template <typename Tin, typename Tp, typename Tout, int V>
__global__ void __launch_bounds__(kThreads) block_phase2_kernel(const Ph2Params p) {
    pdl_enter();
    constexpr int E = VecE<Tin>::value;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const Tin *__restrict__ part = static_cast<const Tin *>(p.partial);
    const Tin *__restrict__ pkeys = static_cast<const Tin *>(p.pkeys);
    const Tp *h_pre = static_cast<const Tp *>(p.h_pre);  // may alias h: no __restrict__
    Tout *h = static_cast<Tout *>(p.h);
    const int64_t nwarps = (int64_t)gridDim.x * kWarps;
    for (int64_t x = (int64_t)blockIdx.x * kWarps + warp; x < p.T; x += nwarps) {
        // both rows first: their loads travel while the partial summary is scored
        Frag<Tin, E> fb[V];
        Frag<Tp, E> fh[V];
        if (p.prev) {
            Frag<Tin, E> fp[V];
#pragma unroll
            for (int v = 0; v < V; ++v) {
                const int e = (lane + 32 * v) * E;
                if (e < p.d) {
                    fb[v].load(part + x * p.d + e);  // coherent: the member row is rewritten below
                    fp[v].load_nc(static_cast<const Tin *>(p.prev) + x * p.d + e);
                    fh[v].load(h_pre + x * p.d + e);
                } else {
                    fb[v].zero();
                    fp[v].zero();
                    fh[v].zero();
                }
            }
#pragma unroll
            for (int v = 0; v < V; ++v) {
                const int e = (lane + 32 * v) * E;
                if (e < p.d) {
                    float m[E], b[E];
                    fb[v].get(m);
                    fp[v].get(b);
#pragma unroll
                    for (int t = 0; t < E; ++t) b[t] += m[t];
                    fb[v].set(b);  // rounded once: the partial summary as stored
                    fb[v].store(const_cast<Tin *>(part) + x * p.d + e);
                }
            }
        } else {
#pragma unroll
            for (int v = 0; v < V; ++v) {
                const int e = (lane + 32 * v) * E;
                if (e < p.d) {
                    fb[v].load_nc(part + x * p.d + e);
                    fh[v].load(h_pre + x * p.d + e);  // coherent: h may be h_pre (in place)
                } else {
                    fb[v].zero();
                    fh[v].zero();
                }
            }
        }
        // score of the partial summary, Eq. (8)-(9); an S-LR key is the tail of
        // the summary row already in registers
        float ss = 0.f, qk = 0.f;
        if (p.sliced) {
            const int k0 = p.d - p.r;
#pragma unroll
            for (int v = 0; v < V; ++v) {
                const int e = (lane + 32 * v) * E;
                if (e + E > k0 && e < p.d) {
                    float b[E];
                    fb[v].get(b);
#pragma unroll
                    for (int t = 0; t < E; ++t)
                        if (e + t >= k0) {
                            ss = fmaf(b[t], b[t], ss);
                            qk = fmaf(__ldg(p.query + (e + t - k0)), b[t], qk);
                        }
                }
            }
        } else if (p.prev_keys) {
            Tin *kp = const_cast<Tin *>(pkeys) + x * p.r;
            const Tin *pp = static_cast<const Tin *>(p.prev_keys) + x * p.r;
            for (int j = lane; j < p.r; j += 32) {
                const Tin kr = from_f<Tin>(to_f(pp[j]) + to_f(kp[j]));
                kp[j] = kr;
                const float k = to_f(kr);
                ss = fmaf(k, k, ss);
                qk = fmaf(__ldg(p.query + j), k, qk);
            }
        } else {
            const Tin *kp = pkeys + x * p.r;
            for (int j = lane; j < p.r; j += 32) {
                const float k = to_f(__ldg(kp + j));
                ss = fmaf(k, k, ss);
                qk = fmaf(__ldg(p.query + j), k, qk);
            }
        }
        ss = warp_sum(ss);
        qk = warp_sum(qk);
        const float sP = rsqrtf(fmaf(ss, p.inv_r, p.eps)) * qk;
        const float lp = p.lse_pre[x];  // coherent: lse may be lse_pre (in place)
        const float M = fmaxf(lp, sP);
        const float lse = M + logf(expf(lp - M) + expf(sP - M));
        const float w1 = expf(lp - lse), w2 = expf(sP - lse);
#pragma unroll
        for (int v = 0; v < V; ++v) {
            const int e = (lane + 32 * v) * E;
            if (e < p.d) {
                float b[E], hp[E], o[E];
                fb[v].get(b);
                fh[v].get(hp);
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
// Keys as whole 16-byte vectors (vector loads, and bulk copies when staged).
template <typename Tin>
static bool ph1_key_vec(const BlockPh1Args &a) {
    constexpr int esz = sizeof(Tin);
    if ((a.r * esz) % 16) return false;
    if (a.variant == kSliced) return ((a.d - a.r) * esz) % 16 == 0;
    for (int i = 0; i < a.n; ++i)  // every key matrix (the API checks 16-byte alignment of the tables)
        if (reinterpret_cast<uintptr_t>(a.keys[i]) & 15) return false;
    return true;
}

// A token's keys are staged in shared memory when they are whole vectors and fit 4 KB.
template <typename Tin>
static bool ph1_stages_keys_t(const BlockPh1Args &a) {
    const size_t kbuf_bytes = (size_t)round_up(a.n * ph1_kstride<Tin>(a.r), 16);
    return ph1_key_vec<Tin>(a) && kbuf_bytes <= 4096;
}

bool block_phase1_stages_keys(const BlockPh1Args &a) {
    return a.in_dtype == kBF16 ? ph1_stages_keys_t<bf16>(a) : ph1_stages_keys_t<float>(a);
}

// Dynamic shared memory of a phase-1 launch (layout of block_phase1_kernel).
static size_t ph1_smem(int S, bool ks, int G, int n, int r, int kstride) {
    const size_t kbuf = ks ? (size_t)round_up(n * kstride, 16) : 0;
    return (size_t)kWarps * S * 32 * 16 + (size_t)G * 2 * kbuf + (ks ? (size_t)round_up(G * 2 * (8 + 4), 16) : 0) +
           sizeof(float) * ((size_t)kPh1MaxSites * round_up(r, 4) + (size_t)G * 4 * kPh1MaxSites * n) +
           2 * 2 * 32 * sizeof(float4);  // per-lane query vectors
}

template <typename Tin, typename Tout, bool KS, bool FAST>
static cudaError_t ph1_go(const Ph1Params &p, int grid, size_t smem, cudaStream_t s) {
    constexpr int S = kPh1Stages;
    launch_pdl(block_phase1_kernel<Tin, Tout, S, KS, FAST, FAST>, grid, kThreads, smem, s, p);
    return cudaGetLastError();
}

template <typename Tin, typename Tout>
static cudaError_t launch_ph1_t(const BlockPh1Args &a, cudaStream_t s) {
    constexpr int E = VecE<Tin>::value;
    constexpr int S = kPh1Stages;
    const int chunks_needed = (a.d + 32 * E - 1) / (32 * E);
    int chunks = 1;
    while (chunks < chunks_needed) chunks *= 2;  // 1, 2, 4 or 8 (validated: d <= 8 * 32 * E)
    Ph1Params p;
    p.tw = 1;
    for (int i = 0; i < kMaxTab; ++i) {
        p.vt.p[i] = i < a.n ? a.values[i] : nullptr;
        p.kt.p[i] = (i < a.n && a.keys) ? a.keys[i] : nullptr;
    }
    p.T = a.T;
    p.site_stride = a.T * (int64_t)a.d;
    p.n = a.n;
    p.d = a.d;
    p.r = a.r;
    p.chunks = chunks;
    p.eps = a.eps;
    p.inv_r = 1.f / (float)a.r;
    p.sliced = a.variant == kSliced;
    p.status = a.status;
    p.wait_cycles = a.wait_cycles;
    p.stall = a.stall ? 1 : 0;
    p.key_vec = ph1_key_vec<Tin>(a);
    {  // per-source scoring: keys as whole vectors, nv dividing a warp, at most 2 queries per lane
        const int nv = a.r / E, c8 = a.c < kPh1MaxSites ? a.c : kPh1MaxSites;
        const int qpl = (nv >= 1 && nv <= 32 && 32 % nv == 0) ? (c8 + 32 / nv - 1) / (32 / nv) : 99;
        p.qpl = (p.key_vec && a.r % E == 0 && qpl <= 2) ? qpl : 0;
    }
    const int G = kWarps / chunks;
    const bool ks = ph1_stages_keys_t<Tin>(a);  // keys staged in shared memory
    const bool fullw = a.d == chunks * 32 * E;  // every lane's vector inside the row
    const size_t smem = ph1_smem(S, ks, G, a.n, a.r, ph1_kstride<Tin>(a.r));
    // every variant this call may launch: 8 sites on whole rows (fast), or the rest
    const void *k_fast = ks ? (const void *)block_phase1_kernel<Tin, Tout, S, true, true, true>
                            : (const void *)block_phase1_kernel<Tin, Tout, S, false, true, true>;
    const void *k_gen = ks ? (const void *)block_phase1_kernel<Tin, Tout, S, true, false, false>
                           : (const void *)block_phase1_kernel<Tin, Tout, S, false, false, false>;
    if (smem > 48 * 1024)
        for (const void *kk : {k_fast, k_gen}) {
            cudaError_t e = cudaFuncSetAttribute(kk, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            if (e != cudaSuccess) return e;
        }
    const int grid = persistent_grid(k_gen, kThreads, smem, (a.T + G - 1) / G, 1 << 30);
    // split phase 1 (weights kernel, then the mix) when a token's weights fit the
    // last site's row of h_pre; the stall test hook keeps the key-staging kernel
    const bool split = !a.stall && (size_t)a.n * kPh1MaxSites * sizeof(float) <= (size_t)a.d * sizeof(Tout);
    size_t smem_w =
        sizeof(float) * ((size_t)kPh1MaxSites * round_up(a.r, 4) + (size_t)kWarps * kWTok * kPh1MaxSites * a.n);
    const size_t smem_m = (size_t)kWarps * S * 32 * 16 + sizeof(float) * (size_t)G * 2 * kPh1MaxSites * a.n;
    // bf16 keys of depth 16, 32, 48 or 64 as whole vectors: scores on the tensor cores
    const int kst = (a.r % 16 == 0 && a.r <= 64) ? a.r / 16 : 0;  // k-steps of the MMA
    const bool mma = std::is_same<Tin, bf16>::value && p.key_vec && kst > 0;
    const void *kw = !mma ? (const void *)block_weights_kernel<Tin, Tout>
                   : kst == 1 ? (const void *)block_weights_mma_kernel<Tout, 1>
                   : kst == 2 ? (const void *)block_weights_mma_kernel<Tout, 2>
                   : kst == 3 ? (const void *)block_weights_mma_kernel<Tout, 3>
                             : (const void *)block_weights_mma_kernel<Tout, 4>;
    // tokens per warp chunk: enough chunks for every resident warp, at most 16, scores within 8 KB a warp
    const int tw_max = std::max(1, std::min(16, 256 / a.n));
    if (mma) smem_w = sizeof(float) * (size_t)kWarps * tw_max * kPh1MaxSites * a.n;
    const void *km_fast = (const void *)block_mix_kernel<Tin, Tout, S, true, true>;
    const void *km_gen = (const void *)block_mix_kernel<Tin, Tout, S, false, false>;
    int grid_w = 0, grid_m = 0;
    if (split) {
        for (const void *kk : {kw, km_fast, km_gen}) {
            const size_t sm = kk == kw ? smem_w : smem_m;
            cudaError_t e = cudaFuncSetAttribute(kk, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
            if (e != cudaSuccess) return e;
        }
        if (mma) {
            const int64_t slots = (int64_t)persistent_grid(kw, kThreads, smem_w, 1 << 30, 1 << 30) * kWarps;
            p.tw = (int)std::max<int64_t>(1, std::min<int64_t>(tw_max, (a.T + slots - 1) / slots));
            const int64_t nchunks = (a.T + p.tw - 1) / p.tw;
            grid_w = (int)std::min<int64_t>(slots / kWarps, (nchunks + kWarps - 1) / kWarps);
        } else {
            grid_w = persistent_grid(kw, kThreads, smem_w, (a.T + kWarps * kWTok - 1) / (kWarps * kWTok), 1 << 30);
        }
        grid_m = persistent_grid(km_gen, kThreads, smem_m, (a.T + G - 1) / G, 1 << 30);
    }
    for (int j0 = 0; j0 < a.c; j0 += kPh1MaxSites) {  // groups of at most 8 queries
        p.c = a.c - j0 < kPh1MaxSites ? a.c - j0 : kPh1MaxSites;
        p.queries = a.queries + (size_t)j0 * a.r;
        p.h_pre = static_cast<char *>(a.h_pre) + (size_t)j0 * p.site_stride * sizeof(Tout);
        p.lse_pre = a.lse_pre + (size_t)j0 * a.T;
        const bool fast = p.c == kPh1MaxSites && fullw;
        cudaError_t e;
        if (split) {
            if (!mma) launch_pdl(block_weights_kernel<Tin, Tout>, grid_w, kThreads, smem_w, s, p);
            else if (kst == 1) launch_pdl(block_weights_mma_kernel<Tout, 1>, grid_w, kThreads, smem_w, s, p);
            else if (kst == 2) launch_pdl(block_weights_mma_kernel<Tout, 2>, grid_w, kThreads, smem_w, s, p);
            else if (kst == 3) launch_pdl(block_weights_mma_kernel<Tout, 3>, grid_w, kThreads, smem_w, s, p);
            else launch_pdl(block_weights_mma_kernel<Tout, 4>, grid_w, kThreads, smem_w, s, p);
            if ((e = cudaGetLastError()) != cudaSuccess) return e;
            if (fast) launch_pdl(block_mix_kernel<Tin, Tout, S, true, true>, grid_m, kThreads, smem_m, s, p);
            else launch_pdl(block_mix_kernel<Tin, Tout, S, false, false>, grid_m, kThreads, smem_m, s, p);
            if ((e = cudaGetLastError()) != cudaSuccess) return e;
            continue;
        }
        if (ks) e = fast ? ph1_go<Tin, Tout, true, true>(p, grid, smem, s) : ph1_go<Tin, Tout, true, false>(p, grid, smem, s);
        else e = fast ? ph1_go<Tin, Tout, false, true>(p, grid, smem, s) : ph1_go<Tin, Tout, false, false>(p, grid, smem, s);
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
    p.prev = a.prev;
    p.prev_keys = a.prev_keys;
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
    launch_pdl(block_phase2_kernel<Tin, Tp, Tout, V>, grid, kThreads, 0, s, p);
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
