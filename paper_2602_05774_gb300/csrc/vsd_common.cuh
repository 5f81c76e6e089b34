// vsd_common.cuh -- low-level device helpers for the VSD E-step / M-step
// kernels (sm_103a): cache-hinted 128-bit loads and stores, bf16/f32 unpacking,
// warp reductions, the exponent scale of a temperature, bounded waits.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "vsd.h"

namespace vsd {

constexpr int kThreads = 128;            // threads of every block-level pass
constexpr int kWarps = kThreads / 32;
constexpr int kLoads = 4;                // 16-byte vectors per lane per chunk per tensor
#ifndef VSD_STAGES
#define VSD_STAGES 2
#endif
constexpr int kStages = VSD_STAGES;      // TMA ring depth per warp (chunks in flight)
constexpr double kLog2e = 1.4426950408889634073599246810019;
constexpr double kLn2 = 0.69314718055994530941723212145818;

template <typename T> struct Traits;
template <> struct Traits<float> {
    static constexpr int kPerVec = 4;
    static constexpr uint32_t kNegInf = 0xFF800000u;
};
template <> struct Traits<__nv_bfloat16> {
    static constexpr int kPerVec = 8;
    static constexpr uint32_t kNegInf = 0xFF80FF80u;  // two bf16 -inf
};
// A chunk is what one warp holds in registers at a time: 32 lanes x kLoads
// vectors = 2 KB of one tensor (1024 bf16 or 512 f32 logits).
template <typename T> __host__ __device__ constexpr int chunk_elems() {
    return 32 * kLoads * Traits<T>::kPerVec;
}

// exp(x / T) = 2^(x * c) with c = log2(e) / T.
struct TempScale {
    float c;        // log2(e)/T rounded to float
    float T;
    double Td;
    double invTd;   // 1/T
};

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// ---------------------------------------------------------------- loads
__device__ __forceinline__ uint64_t policy_evict_first() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}
__device__ __forceinline__ uint64_t policy_evict_last() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
    return p;
}
__device__ __forceinline__ uint64_t policy_evict_normal() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_normal.b64 %0, 1.0;" : "=l"(p));
    return p;
}

// Read-only 128-bit load that bypasses L1 and carries an L2 eviction policy.
__device__ __forceinline__ uint4 ld_stream(const void* p, uint64_t pol) {
    uint4 r;
    asm("ld.global.nc.L1::no_allocate.L2::cache_hint.v4.u32 {%0,%1,%2,%3}, [%4], %5;"
        : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
        : "l"(p), "l"(pol));
    return r;
}

// 128-bit store with an L2 eviction policy.
__device__ __forceinline__ void st_stream(void* p, uint4 v, uint64_t pol) {
    asm volatile("st.global.L1::no_allocate.L2::cache_hint.v4.u32 [%0], {%1,%2,%3,%4}, %5;"
                 :: "l"(p), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w), "l"(pol) : "memory");
}

// Coherent (L1-bypassing) loads of data written by other blocks of the same grid.
template <typename U> __device__ __forceinline__ U ld_cg(const U* p) { return __ldcg(p); }

__device__ __forceinline__ int ld_acquire(const int* p) {
    int v;
    asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void st_release(int* p, int v) {
    asm volatile("st.release.gpu.global.b32 [%0], %1;" :: "l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ uint64_t global_timer_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Scalar element load (for rows that are not 16-byte aligned).
__device__ __forceinline__ uint32_t raw_elem(const float* row, int64_t v) {
    return __float_as_uint(__ldg(row + v));
}
__device__ __forceinline__ uint32_t raw_elem(const __nv_bfloat16* row, int64_t v) {
    return (uint32_t)__ldg(reinterpret_cast<const unsigned short*>(row) + v);
}
__device__ __forceinline__ float elem_value(const float* row, int64_t v) { return __ldg(row + v); }
__device__ __forceinline__ float elem_value(const __nv_bfloat16* row, int64_t v) {
    return __uint_as_float(raw_elem(row, v) << 16);
}

// Load chunk c of a row into registers: lane l, vector k holds elements
// c*CE + k*32*PV + l*PV + [0, PV).  Elements at or beyond V read as -inf.
template <typename T, bool VEC>
__device__ __forceinline__ void load_chunk(const T* row, int64_t V, int c, int lane, uint64_t pol,
                                           uint4 (&buf)[kLoads]) {
    constexpr int PV = Traits<T>::kPerVec;
    const int64_t base = (int64_t)c * chunk_elems<T>() + lane * PV;
#pragma unroll
    for (int k = 0; k < kLoads; ++k) {
        const int64_t v0 = base + (int64_t)k * 32 * PV;
        if constexpr (VEC) {
            if (v0 < V) {
                buf[k] = ld_stream(row + v0, pol);
            } else {
                buf[k] = make_uint4(Traits<T>::kNegInf, Traits<T>::kNegInf, Traits<T>::kNegInf,
                                    Traits<T>::kNegInf);
            }
        } else {
            uint32_t w[4];
            if constexpr (PV == 4) {
#pragma unroll
                for (int e = 0; e < 4; ++e)
                    w[e] = (v0 + e < V) ? raw_elem(row, v0 + e) : Traits<T>::kNegInf;
            } else {
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    uint32_t lo = (v0 + 2 * e < V) ? raw_elem(row, v0 + 2 * e) : 0xFF80u;
                    uint32_t hi = (v0 + 2 * e + 1 < V) ? raw_elem(row, v0 + 2 * e + 1) : 0xFF80u;
                    w[e] = lo | (hi << 16);
                }
            }
            buf[k] = make_uint4(w[0], w[1], w[2], w[3]);
        }
    }
}

template <typename T> __device__ __forceinline__ void unpack(const uint4& v, float* f);
template <> __device__ __forceinline__ void unpack<float>(const uint4& v, float* f) {
    f[0] = __uint_as_float(v.x); f[1] = __uint_as_float(v.y);
    f[2] = __uint_as_float(v.z); f[3] = __uint_as_float(v.w);
}
template <> __device__ __forceinline__ void unpack<__nv_bfloat16>(const uint4& v, float* f) {
    f[0] = __uint_as_float(v.x << 16); f[1] = __uint_as_float(v.x & 0xFFFF0000u);
    f[2] = __uint_as_float(v.y << 16); f[3] = __uint_as_float(v.y & 0xFFFF0000u);
    f[4] = __uint_as_float(v.z << 16); f[5] = __uint_as_float(v.z & 0xFFFF0000u);
    f[6] = __uint_as_float(v.w << 16); f[7] = __uint_as_float(v.w & 0xFFFF0000u);
}

// Max over one 16-byte vector (NaN elements are ignored here; they surface
// through the exponential sums).
template <typename T> __device__ __forceinline__ float vec_max(const uint4& v);
template <> __device__ __forceinline__ float vec_max<float>(const uint4& v) {
    return fmaxf(fmaxf(__uint_as_float(v.x), __uint_as_float(v.y)),
                 fmaxf(__uint_as_float(v.z), __uint_as_float(v.w)));
}
template <> __device__ __forceinline__ float vec_max<__nv_bfloat16>(const uint4& v) {
    __nv_bfloat162 a = *reinterpret_cast<const __nv_bfloat162*>(&v.x);
    __nv_bfloat162 b = *reinterpret_cast<const __nv_bfloat162*>(&v.y);
    __nv_bfloat162 c = *reinterpret_cast<const __nv_bfloat162*>(&v.z);
    __nv_bfloat162 d = *reinterpret_cast<const __nv_bfloat162*>(&v.w);
    __nv_bfloat162 m = __hmax2(__hmax2(a, b), __hmax2(c, d));
    return fmaxf(__low2float(m), __high2float(m));
}

// ---------------------------------------------------------------- TMA / mbarrier
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" :: "r"(smem_u32(bar)), "r"(count)
                 : "memory");
}
// Make initialised barriers visible to the async (TMA) proxy.
__device__ __forceinline__ void mbar_init_fence() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
// Order this thread's earlier generic accesses to shared memory before later
// async-proxy (TMA) writes to it.
__device__ __forceinline__ void fence_proxy_async() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;"
                 :: "r"(smem_u32(bar)), "r"(bytes) : "memory");
}
// 1-D bulk copy global -> shared (TMA), completion counted on `bar`.  Both
// addresses 16-byte aligned, bytes a multiple of 16.
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar,
                                         uint64_t pol) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1], %2, [%3], %4;"
        :: "r"(smem_u32(dst)), "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(pol) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok) : "r"(smem_u32(bar)), "r"(parity) : "memory");
    return ok != 0;
}

// 16-byte asynchronous copy global -> shared that bypasses registers; with
// valid = false nothing is read and the 16 bytes are zero-filled.
__device__ __forceinline__ void cp_async16(void* dst, const void* src, bool valid) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;"
                 :: "r"(smem_u32(dst)), "l"(src), "r"(valid ? 16u : 0u) : "memory");
}
// Wait for all of this thread's cp.async copies.
__device__ __forceinline__ void cp_async_wait_all() {
    asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
}

// ---------------------------------------------------------------- packed f32x2
// Blackwell executes two float32 add/sub/mul in one instruction on a 64-bit
// register pair; each lane of the pair is an ordinary IEEE round-to-nearest op.
__device__ __forceinline__ uint64_t f2(float lo, float hi) {
    uint64_t r;
    asm("mov.b64 %0, {%1,%2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}
__device__ __forceinline__ void f2split(uint64_t v, float& lo, float& hi) {
    asm("mov.b64 {%0,%1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t f2sub(uint64_t a, uint64_t b) {
    uint64_t d;
    asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}
__device__ __forceinline__ uint64_t f2mul(uint64_t a, uint64_t b) {
    uint64_t d;
    asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}
__device__ __forceinline__ uint64_t f2add(uint64_t a, uint64_t b) {
    uint64_t d;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}
// The logits of one 16-byte vector as packed pairs (element 2i in the low half).
template <typename T> __device__ __forceinline__ void vec_pairs(const uint4& v, uint64_t* p);
template <> __device__ __forceinline__ void vec_pairs<float>(const uint4& v, uint64_t* p) {
    p[0] = f2(__uint_as_float(v.x), __uint_as_float(v.y));
    p[1] = f2(__uint_as_float(v.z), __uint_as_float(v.w));
}
__device__ __forceinline__ uint64_t bf16x2_pair(uint32_t u) {
    return f2(__uint_as_float(u << 16), __uint_as_float(u & 0xFFFF0000u));
}
template <> __device__ __forceinline__ void vec_pairs<__nv_bfloat16>(const uint4& v, uint64_t* p) {
    p[0] = bf16x2_pair(v.x);
    p[1] = bf16x2_pair(v.y);
    p[2] = bf16x2_pair(v.z);
    p[3] = bf16x2_pair(v.w);
}
// 2^{(v - m) c} of a packed pair: the same per-element arithmetic as the
// scalar ex2((v - m) * c).
__device__ __forceinline__ uint64_t f2_mass(uint64_t v2, uint64_t m2, uint64_t c2) {
    float lo, hi;
    f2split(f2mul(f2sub(v2, m2), c2), lo, hi);
    return f2(ex2(lo), ex2(hi));
}
// Max over a lane's chunk vectors (NaN elements are ignored here; they surface
// through the exponential sums).
template <typename T> __device__ __forceinline__ float lane_max(const uint4 (&buf)[kLoads]);
template <> __device__ __forceinline__ float lane_max<float>(const uint4 (&buf)[kLoads]) {
    float m = -INFINITY;
#pragma unroll
    for (int k = 0; k < kLoads; ++k)
        m = fmaxf(fmaxf(m, fmaxf(__uint_as_float(buf[k].x), __uint_as_float(buf[k].y))),
                  fmaxf(__uint_as_float(buf[k].z), __uint_as_float(buf[k].w)));
    return m;
}
template <> __device__ __forceinline__ float lane_max<__nv_bfloat16>(const uint4 (&buf)[kLoads]) {
    const __nv_bfloat162* w = reinterpret_cast<const __nv_bfloat162*>(&buf[0]);
    __nv_bfloat162 m = w[0];
#pragma unroll
    for (int i = 1; i < 4 * kLoads; ++i) m = __hmax2(m, w[i]);
    return fmaxf(__low2float(m), __high2float(m));
}

// ---------------------------------------------------------------- warps
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ double warp_sum(double v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
// Inclusive prefix sum over the lanes of a warp.
__device__ __forceinline__ float warp_incl_scan(float v, int lane) {
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        float n = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += n;
    }
    return v;
}
__device__ __forceinline__ double warp_incl_scan(double v, int lane) {
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        double n = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += n;
    }
    return v;
}

}  // namespace vsd
