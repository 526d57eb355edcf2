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
// Phase 1 tiles a token's row over the warps of a group: warp (g, ch) of a CTA
// owns the 32 x 16-byte chunk ch of token g's rows and keeps c accumulators per
// element.  The chunk warps split the c queries for scoring and share the
// weights through shared memory (double-buffered, one named barrier per pass),
// and each pass scores the next token while the current token's rows load.
#include "lrar.h"
#include "lrar_device.cuh"
#include "lrar_launch.h"
#include "lrar_sm100.cuh"

namespace lrar {

constexpr int kPh1MaxSites = 8;  // queries per phase-1 launch (more are split by the host)
constexpr int kPh1Stages = 12;   // ring depth of phase 1 (rows in flight per lane + 1)

struct Ph1Params {
    const void *values, *keys;
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
};

__device__ __forceinline__ void group_sync(int id, int threads) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}

// Scores of token x for the queries j = ch, ch + chunks, ... (Eq. 8-9): lane i
// takes source i; then the softmax of each of those queries over the n sources.
// Weights go to aw[j * n + i], lse_j to the output.
template <typename Tin>
__device__ __forceinline__ float ph1_dot(const Tin *__restrict__ kp, const float *__restrict__ qj, int r, bool vec,
                                         float *ss) {
    constexpr int E = VecE<Tin>::value;
    float qk = 0.f, s2 = 0.f;
    if (vec) {
#pragma unroll 4
        for (int jj = 0; jj < r; jj += E) {
            Frag<Tin, E> f;
            f.load_nc(kp + jj);
            float k[E];
            f.get(k);
#pragma unroll
            for (int t = 0; t < E; ++t) {
                s2 = fmaf(k[t], k[t], s2);
                qk = fmaf(qj[jj + t], k[t], qk);
            }
        }
    } else {
        for (int jj = 0; jj < r; ++jj) {
            const float k = to_f(__ldg(kp + jj));
            s2 = fmaf(k, k, s2);
            qk = fmaf(qj[jj], k, qk);
        }
    }
    if (ss) *ss = s2;
    return qk;
}

// The same over a key staged in shared memory (whole 16-byte vectors).
template <typename Tin>
__device__ __forceinline__ float ph1_dot_s(const Tin *kp, const float *__restrict__ qj, int r, float *ss) {
    constexpr int E = VecE<Tin>::value;
    float qk = 0.f, s2 = 0.f;
#pragma unroll 4
    for (int jj = 0; jj < r; jj += E) {
        Frag<Tin, E> f;
        f.a = *reinterpret_cast<const uint4 *>(kp + jj);
        float k[E];
        f.get(k);
#pragma unroll
        for (int t = 0; t < E; ++t) {
            s2 = fmaf(k[t], k[t], s2);
            qk = fmaf(qj[jj + t], k[t], qk);
        }
    }
    if (ss) *ss = s2;
    return qk;
}

// Staged keys of one token: key i at byte i * kstride of a group's buffer
// (r * sizeof(Tin) bytes, then 16 bytes of padding against bank conflicts).
template <typename Tin>
__device__ __forceinline__ int ph1_kstride(int r) {
    return r * (int)sizeof(Tin) + 16;
}

// Copy token x's n keys into a group buffer with bulk copies counted on bar
// (one warp: lane 0 announces the bytes, lane i copies key i).
template <typename Tin>
__device__ __forceinline__ void ph1_stage(const Ph1Params &p, int64_t x, int lane, uint32_t kbuf, uint32_t bar) {
    const Tin *__restrict__ values = static_cast<const Tin *>(p.values);
    const Tin *__restrict__ keys = static_cast<const Tin *>(p.keys);
    const uint32_t kbytes = (uint32_t)(p.r * (int)sizeof(Tin));
    if (lane == 0) sm100::mbar_arrive_expect_tx(bar, kbytes * (uint32_t)p.n);
    __syncwarp();
    for (int i = lane; i < p.n; i += 32) {
        const Tin *kp = p.sliced ? values + ((int64_t)i * p.T + x) * p.d + (p.d - p.r)
                                 : keys + ((int64_t)i * p.T + x) * p.r;
        sm100::bulk_load(kbuf + (uint32_t)(i * ph1_kstride<Tin>(p.r)), kp, kbytes, bar);
    }
}

// Scores of token x for the queries j = ch, ch + chunks, ... (Eq. 8-9): lane i
// takes source i, reading its key from kb_s (staged) or global memory; then the
// softmax of each of those queries over the n sources.  Weights go to
// aw[i * kPh1MaxSites + j] (a source's weights for every query side by side),
// lse_j to the output.
template <typename Tin>
__device__ __forceinline__ void ph1_score(const Ph1Params &p, const float *__restrict__ q_s, int rp, int64_t x,
                                          int ch, int lane, float *aw, const unsigned char *kb_s = nullptr) {
    const Tin *__restrict__ values = static_cast<const Tin *>(p.values);
    const Tin *__restrict__ keys = static_cast<const Tin *>(p.keys);
    if (ch < p.c)
        for (int i = lane; i < p.n; i += 32) {
            float ss, qk0;
            const Tin *kp;
            if (kb_s) {
                kp = reinterpret_cast<const Tin *>(kb_s + i * ph1_kstride<Tin>(p.r));
                qk0 = ph1_dot_s<Tin>(kp, q_s + ch * rp, p.r, &ss);
            } else {
                kp = p.sliced ? values + ((int64_t)i * p.T + x) * p.d + (p.d - p.r) : keys + ((int64_t)i * p.T + x) * p.r;
                qk0 = ph1_dot<Tin>(kp, q_s + ch * rp, p.r, p.key_vec != 0, &ss);
            }
            const float rho = rsqrtf(fmaf(ss, p.inv_r, p.eps));
            aw[i * kPh1MaxSites + ch] = rho * qk0;
            for (int j = ch + p.chunks; j < p.c; j += p.chunks)  // further queries of this warp (small d)
                aw[i * kPh1MaxSites + j] = rho * (kb_s ? ph1_dot_s<Tin>(kp, q_s + j * rp, p.r, nullptr)
                                              : ph1_dot<Tin>(kp, q_s + j * rp, p.r, p.key_vec != 0, nullptr));
        }
    __syncwarp();
    for (int j = ch; j < p.c; j += p.chunks) {
        float m = -INFINITY;
        for (int i = lane; i < p.n; i += 32) m = fmaxf(m, aw[i * kPh1MaxSites + j]);
        m = warp_max(m);
        float z = 0.f;
        for (int i = lane; i < p.n; i += 32) z += expf(aw[i * kPh1MaxSites + j] - m);
        z = warp_sum(z);
        __syncwarp();
        for (int i = lane; i < p.n; i += 32) aw[i * kPh1MaxSites + j] = expf(aw[i * kPh1MaxSites + j] - m) / z;
        if (lane == 0) p.lse_pre[(int64_t)j * p.T + x] = m + logf(z);
        __syncwarp();
    }
}

// Rows stream through a per-lane cp.async ring (each lane copies and reads
// back its own 16-byte vector of every row), S - 1 rows ahead and across
// tokens, so the loads of the next token's rows overlap this token's mix.
// KS: each group's keys are staged two tokens ahead in shared memory with
// bulk copies (double-buffered, one mbarrier per buffer), so scoring reads no
// global memory.  Each wait for them is bounded (p.wait_cycles) and decided
// for the whole warp; one that runs out ORs LRAR_STATUS_WAIT_TIMEOUT into
// *p.status and raises the CTA's abort flag, after which no warp waits again
// and no group issues another copy (a group's copy into a buffer follows the
// barrier that ends the pass in which its warps waited for that buffer's
// previous token, so a give-up is seen before the buffer is reused).  The
// issuing warp counts the phases it issued and saw complete per buffer (at
// most one per buffer is left unconfirmed after a give-up) and waits, bounded,
// for that one before the CTA exits, so no copy lands in freed shared memory.
// The outputs of a launch that gave up are not valid.
// C8: exactly eight sites per launch (compile-time loop bounds); else p.c <= 8.
template <typename Tin, typename Tout, int S, bool KS, bool C8>
__global__ void __launch_bounds__(kThreads, 2) block_phase1_kernel(const __grid_constant__ Ph1Params p) {
    constexpr int E = VecE<Tin>::value;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int rp = round_up(p.r, 4);
    const int G_ = kWarps / p.chunks;
    const int kbuf_bytes = KS ? round_up(p.n * ph1_kstride<Tin>(p.r), 16) : 0;  // one token's keys
    unsigned char *kb_all = smem_raw + (size_t)kWarps * S * 32 * 16;           // [G][2][kbuf_bytes]
    uint64_t *kbar_all = reinterpret_cast<uint64_t *>(kb_all + (size_t)G_ * 2 * kbuf_bytes);  // [G][2]
    float *q_s = reinterpret_cast<float *>(kbar_all + (KS ? 2 * G_ : 0));       // [c][r]
    float *a_all = q_s + kPh1MaxSites * rp;  // [G][2][n][kPh1MaxSites]: weights, double-buffered by pass
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int G = kWarps / p.chunks;  // tokens per CTA pass
    const int g = warp / p.chunks, ch = warp % p.chunks;
    const int nthr = p.chunks * 32;   // threads of a token group (named barrier 1 + g)
    __shared__ int abort_s;           // set once a key wait of this CTA gave up
    __shared__ __align__(8) uint64_t never_bar;  // test hook: a barrier nothing arrives on
    volatile int *abort = &abort_s;
    for (int j = threadIdx.x; j < p.c * p.r; j += kThreads) q_s[(j / p.r) * rp + j % p.r] = p.queries[j];
    if (KS && threadIdx.x < 2 * G) {
        sm100::mbar_init(smem_u32(kbar_all + threadIdx.x), 1);
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

    const Tin *__restrict__ values = static_cast<const Tin *>(p.values);
    Tout *__restrict__ h_pre = static_cast<Tout *>(p.h_pre);
    const int e = (ch * 32 + lane) * E;  // this lane's first element of the row
    float *aw0 = a_all + (size_t)g * 2 * kPh1MaxSites * p.n;
    const int64_t stride = (int64_t)gridDim.x * G;
    const uint32_t ring_w = smem_u32(smem_raw) + (uint32_t)(warp * S * 32 * 16) + 16u * lane;
    unsigned char *kb0 = kb_all + (size_t)g * 2 * kbuf_bytes;
    auto kbuf = [&](int b) { return smem_u32(kb0 + b * kbuf_bytes); };
    auto kbar = [&](int b) { return smem_u32(kbar_all + 2 * g + b); };
    // token q of this group (x0 + q * stride) uses key buffer q % 2, for the (q / 2)-th time;
    // the issuing warp (ch == 0) counts phases issued and seen complete per buffer
    uint32_t issued0 = 0u, issued1 = 0u, seen0 = 0u, seen1 = 0u;
    auto kwait = [&](int q) {
        if (__any_sync(0xffffffffu, *abort != 0)) return;  // the CTA gave up: no further waits (warp-uniform)
        const uint32_t bar = p.stall ? smem_u32(&never_bar) : kbar(q & 1);
        const uint32_t par = p.stall ? 0u : (uint32_t)(q >> 1) & 1u;
        const bool ok = __all_sync(0xffffffffu, sm100::mbar_wait(bar, par, p.wait_cycles, abort));
        if (ok) {
            if (ch == 0) {
                if (q & 1) seen1 = (uint32_t)(q >> 1) + 1u;
                else seen0 = (uint32_t)(q >> 1) + 1u;
            }
        } else if (lane == 0) {
            *abort = 1;
            if (p.status) atomicOr(p.status, LRAR_STATUS_WAIT_TIMEOUT);
        }
    };
    // the issuing warp stages token xx into buffer b unless the CTA gave up (warp-uniform)
    auto stage = [&](int64_t xx, int b) {
        if (__any_sync(0xffffffffu, *abort != 0)) return;
        ph1_stage<Tin>(p, xx, lane, kbuf(b), kbar(b));
        if (b) ++issued1;
        else ++issued0;
    };

    int64_t x = (int64_t)blockIdx.x * G + g;
    int64_t ix = x;  // next row to copy: source ii of token ix
    int ii = 0;
    auto issue = [&](int st) {
        if (ix < p.T) {
            if (e < p.d) cp_async16(ring_w + 16u * 32u * st, values + ((int64_t)ii * p.T + ix) * p.d + e);
            if (++ii == p.n) {
                ii = 0;
                ix += stride;
            }
        }
        cp_async_commit();
    };
#pragma unroll
    for (int st = 0; st < S - 1; ++st) issue(st);
    int st_c = 0, st_i = S - 1;

    if (KS && ch == 0) {
        if (x < p.T) stage(x, 0);
        if (x + stride < p.T) stage(x + stride, 1);
    }
    if (x < p.T) {
        if (KS) kwait(0);
        ph1_score<Tin>(p, q_s, rp, x, ch, lane, aw0, KS ? kb0 : nullptr);
    }
    group_sync(1 + g, nthr);
    for (int pass = 0; (int64_t)blockIdx.x * G + pass * stride < p.T; ++pass, x += stride) {
        const float *aw = aw0 + (pass & 1) * kPh1MaxSites * p.n;
        float *aw_next = aw0 + ((pass + 1) & 1) * kPh1MaxSites * p.n;
        // buffer pass % 2 held token `pass`, scored by every warp before the last barrier
        if (KS && ch == 0 && x + 2 * stride < p.T) stage(x + 2 * stride, pass & 1);
        if (x + stride < p.T) {
            if (KS) kwait(pass + 1);
            ph1_score<Tin>(p, q_s, rp, x + stride, ch, lane, aw_next, KS ? kb0 + ((pass + 1) & 1) * kbuf_bytes : nullptr);
        }
        if (x < p.T) {
            float acc[kPh1MaxSites][E];
#pragma unroll
            for (int j = 0; j < kPh1MaxSites; ++j)
#pragma unroll
                for (int t = 0; t < E; ++t) acc[j][t] = 0.f;
            for (int i = 0; i < p.n; ++i) {
                issue(st_i);
                cp_async_wait<S - 1>();  // this lane's copy of row i has landed
                Frag<Tin, E> f;
                if (e < p.d) f.a = ld_shared16(ring_w + 16u * 32u * st_c);
                else f.zero();
                st_c = (st_c + 1 == S) ? 0 : st_c + 1;
                st_i = (st_i + 1 == S) ? 0 : st_i + 1;
                float o[E], w[kPh1MaxSites];
                f.get(o);
                const float4 w0 = *reinterpret_cast<const float4 *>(aw + i * kPh1MaxSites);
                const float4 w1 = *reinterpret_cast<const float4 *>(aw + i * kPh1MaxSites + 4);
                w[0] = w0.x, w[1] = w0.y, w[2] = w0.z, w[3] = w0.w, w[4] = w1.x, w[5] = w1.y, w[6] = w1.z, w[7] = w1.w;
#pragma unroll
                for (int j = 0; j < kPh1MaxSites; ++j) {
                    if (C8 || j < p.c) {
#pragma unroll
                        for (int t = 0; t < E; t += 2) fma2(acc[j][t], acc[j][t + 1], w[j], w[j], o[t], o[t + 1]);
                    }
                }
            }
            if (e < p.d) {
#pragma unroll
                for (int j = 0; j < kPh1MaxSites; ++j) {
                    if (C8 || j < p.c) {
                        Frag<Tout, E> out;
                        out.set(acc[j]);
                        out.store(h_pre + (int64_t)j * p.site_stride + x * p.d + e);
                    }
                }
            }
        }
        group_sync(1 + g, nthr);  // next weights complete; this pass's weights free for reuse
    }
    cp_async_wait_all();
    if (KS && ch == 0)  // drain: the one phase per buffer a give-up may have left unconfirmed
        for (int b = 0; b < 2; ++b) {
            const uint32_t iss = b ? issued1 : issued0, done = b ? seen1 : seen0;
            if (iss > done && !__all_sync(0xffffffffu, sm100::mbar_wait(kbar(b), (iss - 1u) & 1u, p.wait_cycles)) &&
                lane == 0 && p.status)
                atomicOr(p.status, LRAR_STATUS_WAIT_TIMEOUT);
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
        // both rows first: their loads travel while the partial summary is scored
        Frag<Tin, E> fb[V];
        Frag<Tp, E> fh[V];
#pragma unroll
        for (int v = 0; v < V; ++v) {
            const int e = (lane + 32 * v) * E;
            if (e < p.d) {
                fb[v].load_nc(part + x * p.d + e);
                fh[v].load_nc(h_pre + x * p.d + e);
            } else {
                fb[v].zero();
                fh[v].zero();
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
        const float lp = __ldg(p.lse_pre + x);
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
    return (a.r * esz) % 16 == 0 && (a.variant == kSliced ? ((a.d - a.r) * esz) % 16 == 0
                                                          : (reinterpret_cast<uintptr_t>(a.keys) & 15) == 0);
}

// A token's keys are staged in shared memory when they are whole vectors and fit 4 KB.
template <typename Tin>
static bool ph1_stages_keys_t(const BlockPh1Args &a) {
    const size_t kbuf_bytes = (size_t)round_up(a.n * (a.r * (int)sizeof(Tin) + 16), 16);
    return ph1_key_vec<Tin>(a) && kbuf_bytes <= 4096;
}

bool block_phase1_stages_keys(const BlockPh1Args &a) {
    return a.in_dtype == kBF16 ? ph1_stages_keys_t<bf16>(a) : ph1_stages_keys_t<float>(a);
}

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
    p.status = a.status;
    p.wait_cycles = a.wait_cycles;
    p.stall = a.stall ? 1 : 0;
    p.key_vec = ph1_key_vec<Tin>(a);
    const int G = kWarps / chunks;
    constexpr int S = kPh1Stages;
    const int kstride = a.r * (int)sizeof(Tin) + 16;
    const size_t kbuf_bytes = (size_t)round_up(a.n * kstride, 16);
    const bool ks = ph1_stages_keys_t<Tin>(a);  // keys staged in shared memory
    const size_t smem = (size_t)kWarps * S * 32 * 16 + (ks ? (size_t)G * 2 * (kbuf_bytes + 8) : 0) +
                        sizeof(float) * ((size_t)kPh1MaxSites * round_up(a.r, 4) + (size_t)G * 2 * kPh1MaxSites * a.n);
    const void *k = ks ? (const void *)block_phase1_kernel<Tin, Tout, S, true, true>
                       : (const void *)block_phase1_kernel<Tin, Tout, S, false, true>;  // same resources for C8 or not
    if (smem > 48 * 1024) {  // every variant this call may launch (8 sites, or the rest)
        const void *ks_all[4] = {(const void *)block_phase1_kernel<Tin, Tout, S, true, true>,
                                 (const void *)block_phase1_kernel<Tin, Tout, S, true, false>,
                                 (const void *)block_phase1_kernel<Tin, Tout, S, false, true>,
                                 (const void *)block_phase1_kernel<Tin, Tout, S, false, false>};
        for (const void *kk : ks_all) {
            cudaError_t e = cudaFuncSetAttribute(kk, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            if (e != cudaSuccess) return e;
        }
    }
    const int grid = persistent_grid(k, kThreads, smem, (a.T + G - 1) / G, 1 << 30);
    for (int j0 = 0; j0 < a.c; j0 += kPh1MaxSites) {  // groups of at most 8 queries
        p.c = a.c - j0 < kPh1MaxSites ? a.c - j0 : kPh1MaxSites;
        p.queries = a.queries + (size_t)j0 * a.r;
        p.h_pre = static_cast<char *>(a.h_pre) + (size_t)j0 * p.site_stride * sizeof(Tout);
        p.lse_pre = a.lse_pre + (size_t)j0 * a.T;
        const bool c8 = p.c == kPh1MaxSites;
        if (ks && c8) block_phase1_kernel<Tin, Tout, S, true, true><<<grid, kThreads, smem, s>>>(p);
        else if (ks) block_phase1_kernel<Tin, Tout, S, true, false><<<grid, kThreads, smem, s>>>(p);
        else if (c8) block_phase1_kernel<Tin, Tout, S, false, true><<<grid, kThreads, smem, s>>>(p);
        else block_phase1_kernel<Tin, Tout, S, false, false><<<grid, kThreads, smem, s>>>(p);
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
