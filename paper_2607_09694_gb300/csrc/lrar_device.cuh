// lrar_device.cuh -- device helpers shared by the depth-mix kernels:
// 16-byte streaming loads, bf16 <-> f32 packing, warp reductions.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "lrar_launch.h"

namespace lrar {

constexpr int kWarps = 8;                 // warps per CTA
constexpr int kThreads = kWarps * 32;
constexpr int kMaxSources = 128;          // LRAR_MAX_SOURCES
static_assert(kMaxSources == kMaxTab, "source tables hold every source");
constexpr int kSrcRegs = kMaxSources / 32;
constexpr int kMaxPartials = 1024;        // CTAs whose dq partials the workspace holds

typedef __nv_bfloat16 bf16;

// Elements of T in one 16-byte vector.
template <typename T> struct VecE;
template <> struct VecE<float> { static constexpr int value = 4; };
template <> struct VecE<bf16> { static constexpr int value = 8; };

// ---------------------------------------------------------------- loads ----
// Read-only, streamed once: bypass L1 allocation.
__device__ __forceinline__ uint4 ld_nc16(const void *p) {
    uint4 v;
    asm("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
        : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
        : "l"(p));
    return v;
}
__device__ __forceinline__ uint2 ld_nc8(const void *p) {
    uint2 v;
    asm("ld.global.nc.L1::no_allocate.v2.u32 {%0, %1}, [%2];" : "=r"(v.x), "=r"(v.y) : "l"(p));
    return v;
}
// Coherent loads/stores (data the same kernel writes).
__device__ __forceinline__ uint4 ld16(const void *p) { return *reinterpret_cast<const uint4 *>(p); }
__device__ __forceinline__ uint2 ld8(const void *p) { return *reinterpret_cast<const uint2 *>(p); }
__device__ __forceinline__ void st16(void *p, uint4 v) { *reinterpret_cast<uint4 *>(p) = v; }
__device__ __forceinline__ void st8(void *p, uint2 v) { *reinterpret_cast<uint2 *>(p) = v; }

// Asynchronous global -> shared copies of 16 bytes (L2 only).  Each lane
// copies and later reads its own cells, so completing its own groups
// (cp.async.wait_group) is the only synchronisation needed.
__device__ __forceinline__ void cp_async16(uint32_t smem_addr, const void *gptr) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_addr), "l"(gptr) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N> __device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;" ::: "memory"); }
__device__ __forceinline__ uint4 ld_shared16(uint32_t smem_addr) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "r"(smem_addr)
                 : "memory");
    return v;
}
__device__ __forceinline__ void st_shared16(uint32_t smem_addr, uint4 v) {
    asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(smem_addr), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
                 : "memory");
}
__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// ------------------------------------------------------------- packing ----
// A bfloat16 is the upper half of a binary32 word, so widening is a shift.
__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }
__device__ __forceinline__ uint32_t bf_pack(float lo, float hi) {
    __nv_bfloat162 b = __floats2bfloat162_rn(lo, hi);  // round to nearest even
    return *reinterpret_cast<uint32_t *>(&b);
}

__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(bf16 v) { return __bfloat162float(v); }
template <typename T> __device__ __forceinline__ T from_f(float v);
template <> __device__ __forceinline__ float from_f<float>(float v) { return v; }
template <> __device__ __forceinline__ bf16 from_f<bf16>(float v) { return __float2bfloat16_rn(v); }

// E consecutive elements of type T held as raw words.
template <typename T, int E> struct Frag;

template <> struct Frag<bf16, 8> {
    uint4 a;
    __device__ __forceinline__ void load_nc(const bf16 *p) { a = ld_nc16(p); }
    __device__ __forceinline__ void load(const bf16 *p) { a = ld16(p); }
    __device__ __forceinline__ void store(bf16 *p) const { st16(p, a); }
    __device__ __forceinline__ void zero() { a = make_uint4(0, 0, 0, 0); }
    __device__ __forceinline__ void get(float *f) const {
        f[0] = bf_lo(a.x); f[1] = bf_hi(a.x); f[2] = bf_lo(a.y); f[3] = bf_hi(a.y);
        f[4] = bf_lo(a.z); f[5] = bf_hi(a.z); f[6] = bf_lo(a.w); f[7] = bf_hi(a.w);
    }
    // consecutive pairs, as the operands of packed fp32 arithmetic
    __device__ __forceinline__ void get2(float2 *f) const {
        f[0] = make_float2(bf_lo(a.x), bf_hi(a.x)); f[1] = make_float2(bf_lo(a.y), bf_hi(a.y));
        f[2] = make_float2(bf_lo(a.z), bf_hi(a.z)); f[3] = make_float2(bf_lo(a.w), bf_hi(a.w));
    }
    __device__ __forceinline__ void set(const float *f) {
        a.x = bf_pack(f[0], f[1]); a.y = bf_pack(f[2], f[3]);
        a.z = bf_pack(f[4], f[5]); a.w = bf_pack(f[6], f[7]);
    }
    __device__ __forceinline__ void set2(const float2 *f) {
        a.x = bf_pack(f[0].x, f[0].y); a.y = bf_pack(f[1].x, f[1].y);
        a.z = bf_pack(f[2].x, f[2].y); a.w = bf_pack(f[3].x, f[3].y);
    }
};

template <> struct Frag<bf16, 4> {
    uint2 a;
    __device__ __forceinline__ void load_nc(const bf16 *p) { a = ld_nc8(p); }
    __device__ __forceinline__ void load(const bf16 *p) { a = ld8(p); }
    __device__ __forceinline__ void store(bf16 *p) const { st8(p, a); }
    __device__ __forceinline__ void zero() { a = make_uint2(0, 0); }
    __device__ __forceinline__ void get(float *f) const {
        f[0] = bf_lo(a.x); f[1] = bf_hi(a.x); f[2] = bf_lo(a.y); f[3] = bf_hi(a.y);
    }
    __device__ __forceinline__ void set(const float *f) { a.x = bf_pack(f[0], f[1]); a.y = bf_pack(f[2], f[3]); }
    __device__ __forceinline__ void get2(float2 *f) const {
        f[0] = make_float2(bf_lo(a.x), bf_hi(a.x)); f[1] = make_float2(bf_lo(a.y), bf_hi(a.y));
    }
    __device__ __forceinline__ void set2(const float2 *f) { a.x = bf_pack(f[0].x, f[0].y); a.y = bf_pack(f[1].x, f[1].y); }
};

template <> struct Frag<float, 4> {
    uint4 a;
    __device__ __forceinline__ void load_nc(const float *p) { a = ld_nc16(p); }
    __device__ __forceinline__ void load(const float *p) { a = ld16(p); }
    __device__ __forceinline__ void store(float *p) const { st16(p, a); }
    __device__ __forceinline__ void zero() { a = make_uint4(0, 0, 0, 0); }
    __device__ __forceinline__ void get(float *f) const {
        f[0] = __uint_as_float(a.x); f[1] = __uint_as_float(a.y);
        f[2] = __uint_as_float(a.z); f[3] = __uint_as_float(a.w);
    }
    __device__ __forceinline__ void get2(float2 *f) const {
        f[0] = make_float2(__uint_as_float(a.x), __uint_as_float(a.y));
        f[1] = make_float2(__uint_as_float(a.z), __uint_as_float(a.w));
    }
    __device__ __forceinline__ void set(const float *f) {
        a.x = __float_as_uint(f[0]); a.y = __float_as_uint(f[1]);
        a.z = __float_as_uint(f[2]); a.w = __float_as_uint(f[3]);
    }
    __device__ __forceinline__ void set2(const float2 *f) {
        a.x = __float_as_uint(f[0].x); a.y = __float_as_uint(f[0].y);
        a.z = __float_as_uint(f[1].x); a.w = __float_as_uint(f[1].y);
    }
};

template <> struct Frag<float, 8> {
    Frag<float, 4> lo, hi;
    __device__ __forceinline__ void load_nc(const float *p) { lo.load_nc(p); hi.load_nc(p + 4); }
    __device__ __forceinline__ void load(const float *p) { lo.load(p); hi.load(p + 4); }
    __device__ __forceinline__ void store(float *p) const { lo.store(p); hi.store(p + 4); }
    __device__ __forceinline__ void zero() { lo.zero(); hi.zero(); }
    __device__ __forceinline__ void get(float *f) const { lo.get(f); hi.get(f + 4); }
    __device__ __forceinline__ void set(const float *f) { lo.set(f); hi.set(f + 4); }
    __device__ __forceinline__ void get2(float2 *f) const { lo.get2(f); hi.get2(f + 2); }
    __device__ __forceinline__ void set2(const float2 *f) { lo.set2(f); hi.set2(f + 2); }
};

// ---------------------------------------------------- dependent launch ---
// Every kernel of the library is launched with programmatic stream
// serialization (launch_pdl): it may be scheduled while the kernel before it
// in the stream is still running, and waits here, before its first access to
// global memory, until that kernel has completed and its writes are visible;
// it then lets the next kernel be scheduled in turn.  Only the launch and the
// CTAs' set-up overlap; in a kernel launched without the attribute both
// instructions return at once.
__device__ __forceinline__ void pdl_enter() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// The same two steps apart, for a kernel that starts reading inputs written
// before its predecessor began (never its predecessor's own outputs) ahead of
// the wait.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_dependents() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// ----------------------------------------------------------- reductions ---
// xor butterflies leave the identical bit pattern in every lane.
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

__host__ __device__ __forceinline__ int round_up(int a, int b) { return (a + b - 1) / b * b; }

// Ring stages per warp for the full-key passes: about B * 4 KB of rows in
// flight per CTA (P planes of V 16-byte vectors per lane and stage), at least
// two.  B = 24 for two CTAs per SM, 48 for one.
template <int V, int P, int B> struct FullStages {
    static constexpr int raw = B / (V * P);
    static constexpr int value = raw < 2 ? 2 : (raw > 8 ? 8 : raw);
};

// The query of a full-key row in shared memory, laid out so that a lane reads
// the E coordinates of its vector v as E / 4 bank-conflict-free 16-byte loads:
// row element e = (lane + 32 v) E + t sits at float ((v E/4 + t/4) 32 + lane) 4 + t % 4.
template <int E> __device__ __forceinline__ int q_slot(int e) {
    const int v = e / (32 * E), lane = (e / E) % 32, t = e % E;
    return ((v * (E / 4) + t / 4) * 32 + lane) * 4 + (t % 4);
}
template <int E> __device__ __forceinline__ void q_get(const float *__restrict__ q_s, int v, int lane, float *qv) {
#pragma unroll
    for (int k = 0; k < E / 4; ++k) {
        const float4 a = *reinterpret_cast<const float4 *>(q_s + ((v * (E / 4) + k) * 32 + lane) * 4);
        qv[4 * k] = a.x;
        qv[4 * k + 1] = a.y;
        qv[4 * k + 2] = a.z;
        qv[4 * k + 3] = a.w;
    }
}

// Row x of source i (width elements per row) in a source table.
template <typename T>
__device__ __forceinline__ const T *src_row(const SrcTab &t, int i, int64_t x, int width) {
    return static_cast<const T *>(t.p[i]) + x * width;
}
template <typename T>
__device__ __forceinline__ T *dst_row(const SrcTab &t, int i, int64_t x, int width) {
    return static_cast<T *>(const_cast<void *>(t.p[i])) + x * width;
}

// Two fp32 fused multiply-adds in one packed instruction (d_k = a_k b_k + d_k,
// each rounded to nearest even: the same results as two fmaf).
__device__ __forceinline__ void fma2(float &d0, float &d1, float a0, float a1, float b0, float b1) {
    const float2 r = __ffma2_rn(make_float2(a0, a1), make_float2(b0, b1), make_float2(d0, d1));
    d0 = r.x;
    d1 = r.y;
}

}  // namespace lrar
