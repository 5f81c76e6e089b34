// vsd_tc.cuh -- PTX wrappers for the tensor-core kernels on sm_103a (the
// draft LM head and its backward): 2-D TMA loads into shared memory, the
// shared-memory descriptor of a K-major bf16 tile in the 128-byte swizzle,
// tcgen05.mma / commit / ld, fences, and bounded mbarrier waits.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "vsd.h"
#include "vsd_common.cuh"

namespace vsd_lm {

using vsd::global_timer_ns;
using vsd::mbar_expect_tx;
using vsd::mbar_init;
using vsd::mbar_init_fence;
using vsd::mbar_try_wait;
using vsd::smem_u32;

// ---------------------------------------------------------------- PTX wrappers
// 2-D tiled TMA load global -> shared, completion counted on `bar`.  x is the
// inner (K) coordinate in elements, y the row.
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y,
                                            uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];"
        :: "r"(smem_u32(dst)), "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y),
           "r"(smem_u32(bar))
        : "memory");
}

// Shared-memory matrix descriptor of a K-major bf16 tile written by TMA with
// the 128-byte swizzle: rows of 128 bytes, 8-row groups 1024 bytes apart
// (stride byte offset), the leading byte offset unused for this layout,
// descriptor version 1, swizzle mode 2 (128 bytes).  The tile base is
// 1024-byte aligned, so the base-offset field is 0; a K step of 16 elements
// inside the 128-byte row advances the start address by 32 bytes.
__device__ __forceinline__ uint64_t sdesc_sw128(uint32_t saddr) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);  // bits 0-13: start address / 16
    d |= (uint64_t)1 << 16;                    // bits 16-29: leading byte offset / 16
    d |= (uint64_t)(1024 >> 4) << 32;          // bits 32-45: stride byte offset / 16
    d |= (uint64_t)1 << 46;                    // bits 46-48: version
    d |= (uint64_t)2 << 61;                    // bits 61-63: 128-byte swizzle
    return d;
}

// Instruction descriptor, kind::f16: fp32 accumulator, bf16 A and B, both
// K-major, an M x N tile.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N) {
    return (1u << 4)                    // D format f32
           | (1u << 7)                  // A format bf16
           | (1u << 10)                 // B format bf16
           | ((uint32_t)(N >> 3) << 17) // N / 8
           | ((uint32_t)(M >> 4) << 24);// M / 16
}

__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                         uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}"
        :: "r"(d_tmem), "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Arrive on `bar` once every tcgen05.mma this thread issued so far is done.
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];"
        :: "r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// 32 consecutive fp32 columns of this thread's TMEM lane.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32"
        " {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15,"
        " %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31},"
        " [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
          "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
          "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
          "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Bounded wait for the completion of the barrier phase with parity `parity`;
// gives up when another thread of the CTA has (*err set) or after timeout_ns
// (then sets *err and the timeout bit of the status word).
__device__ __forceinline__ bool wait_phase_err(uint64_t* bar, uint32_t parity, int* err,
                                               uint64_t timeout_ns, int* status) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    for (;;) {
        if (mbar_try_wait(bar, parity)) return true;
        if (*(volatile int*)err) return false;
        if (global_timer_ns() - t0 > timeout_ns) {
            *err = 1;
            atomicOr(status, VSD_STATUS_TIMEOUT);
            return false;
        }
    }
}

// Bounded wait that ignores the error flag (winding down after an error: the
// copies and MMAs already issued must finish before the CTA exits).
__device__ __forceinline__ void wait_phase_drain(uint64_t* bar, uint32_t parity,
                                                 uint64_t timeout_ns) {
    const uint64_t t0 = global_timer_ns();
    while (!mbar_try_wait(bar, parity))
        if (global_timer_ns() - t0 > timeout_ns) return;
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" :: "r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ uint32_t pack_bf16(uint32_t lo, uint32_t hi) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(__uint_as_float(lo), __uint_as_float(hi));
    return *reinterpret_cast<const uint32_t*>(&h);
}


// Tensor map of a row-major bf16 matrix [rows][cols] read in boxes of
// box_rows x box_cols, swizzled in swizzle_bytes (128, 64 or 0 for none; the
// box row, box_cols * 2 bytes, at most that wide); out-of-range elements read
// as zero (vsd_lmhead.cu).
bool make_map_box(CUtensorMap* m, const void* base, int rows, int cols, int box_cols,
                  int box_rows, int swizzle_bytes);

}  // namespace vsd_lm
