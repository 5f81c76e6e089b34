// vsd_lmhead.cu -- the draft model's LM head on the tensor cores:
// logits[M][N] = hidden[M][K] . weight[N][K]^T, bf16 inputs, fp32 accumulation
// in tensor memory (TMEM), bf16 logits out (the draft head that produces q,
// paper Sec. 5 implementation details).  Then the fused E-step + M-step on those
// logits (vsd_lmhead_estep_mstep).
//
// One persistent CTA per SM computes 128 x 256 output tiles:
//   warp 0   TMA producer: 128 x 64 hidden and 256 x 64 weight tiles (128-byte
//            swizzle) into a 4-stage shared-memory ring;
//   warp 1   MMA issuer: one thread issues tcgen05.mma (kind::f16, M=128,
//            N=256, K=16) into one of two TMEM accumulators (2 x 256 columns);
//            tcgen05.commit frees a ring stage / hands a finished accumulator on;
//   warps 2-5 epilogue: tcgen05.ld of the accumulator (each warp its 32 TMEM
//            lanes = 32 tile rows), rounding to bf16, 16-byte stores, and, for
//            the fused E-step, each row's chunk statistics of the rounded
//            logits (max, sum 2^{(x - max) c}) over 1024-column chunks.
// The epilogue of one tile overlaps the main loop of the next.  Every wait is
// bounded; a wait that runs out sets VSD_STATUS_TIMEOUT in the status word and
// the CTA winds down (waiting, again bounded, for its copies and MMAs in
// flight) and frees its tensor memory.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>
#include <string.h>

#include <mutex>

#include "vsd.h"
#include "vsd_common.cuh"
#include "vsd_tc.cuh"

namespace vsd_lm {

using vsd::global_timer_ns;
using vsd::mbar_expect_tx;
using vsd::mbar_init;
using vsd::mbar_init_fence;
using vsd::mbar_try_wait;
using vsd::smem_u32;

#ifndef VSD_LM_BN
#define VSD_LM_BN 256
#endif
#ifndef VSD_LM_STAGES
#define VSD_LM_STAGES 4
#endif
constexpr int BM = 128, BN = VSD_LM_BN, BK = 64;  // BK bf16 = one 128-byte swizzle row
constexpr int kStages = VSD_LM_STAGES;
constexpr int kThreads = 192;
constexpr int kABytes = BM * BK * 2;  // 16 KB
constexpr int kBBytes = BN * BK * 2;  // 32 KB
constexpr int kStageBytes = kABytes + kBBytes;
constexpr int kTmemCols = 2 * BN;  // two fp32 accumulators of 128 lanes x BN columns

struct Bars {
    uint64_t full[kStages];   // TMA bytes landed in stage s
    uint64_t empty[kStages];  // the MMAs reading stage s are done
    uint64_t acc_full[2];     // accumulator b holds a finished tile
    uint64_t acc_empty[2];    // the epilogue has read accumulator b (4 arrivals)
    uint64_t drain;           // the MMA warp's final commit
    uint64_t timeout_ns;      // bound of every wait (the call's wait timeout)
    uint32_t tmem_base;
    int err;
};
constexpr size_t kSmemBytes = 1024 /* alignment slack */ + kStages * kStageBytes + sizeof(Bars);

// (PTX wrappers: vsd_tc.cuh)
constexpr uint32_t kIdesc = idesc_bf16(BM, BN);

__device__ __forceinline__ bool wait_phase(uint64_t* bar, uint32_t parity, Bars* sb,
                                           int* status) {
    return wait_phase_err(bar, parity, &sb->err, sb->timeout_ns, status);
}
// The same wait by a whole warp, with one outcome for all its lanes (a lane
// that gave up while another saw the phase complete would split the warp
// between the loop's __syncwarp and the final __syncthreads).
__device__ __forceinline__ bool wait_phase_warp(uint64_t* bar, uint32_t parity, Bars* sb,
                                                int* status) {
    return __all_sync(0xffffffffu, wait_phase(bar, parity, sb, status));
}

// Work is cut into units of one 128-row M tile by one 1024-column chunk (the
// E-step's chunk of bf16 logits): kTilesPerChunk consecutive 128 x 256 tiles,
// computed by one CTA in turn, so that its epilogue threads (one per row) can
// carry a row's running (max, sum 2^{(x - max) c}) over the chunk.  Units are
// numbered with the M tile fastest, so the CTAs working at the same time share
// the same few weight tiles (read from DRAM once, then from L2) and the hidden
// states stay in L2 throughout.
constexpr int kChunkCols = 1024;
constexpr int kTilesPerChunk = kChunkCols / BN;
static_assert(kChunkCols % BN == 0, "a chunk is a whole number of tiles");

// Chunk statistics of the logits for the E-step (a1 of the hot path): for
// row r and chunk ch, tab[r * stride + ch].xy = (max, sum 2^{(x - max) c}) of
// the bf16-rounded logits x of the chunk, c = log2(e) / T.
struct ChunkStatsOut {
    float4* tab;   // null: none
    int stride;    // float4 entries per row
    float c;
};

__global__ void __launch_bounds__(kThreads, 1)
    k_lmhead(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
             __nv_bfloat16* __restrict__ out, int M, int N, int K, int* status,
             uint64_t timeout_ns, ChunkStatsOut cs) {
    extern __shared__ unsigned char dsm_raw[];
    unsigned char* dsm = dsm_raw + ((1024u - (smem_u32(dsm_raw) & 1023u)) & 1023u);
    Bars* sb = reinterpret_cast<Bars*>(dsm + kStages * kStageBytes);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int mt = (M + BM - 1) / BM, ntn = (N + BN - 1) / BN;
    const int nchunks = (ntn + kTilesPerChunk - 1) / kTilesPerChunk;
    const int nunits = mt * nchunks, nk = (K + BK - 1) / BK;
    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&sb->full[s], 1);
            mbar_init(&sb->empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&sb->acc_full[b], 1);
            mbar_init(&sb->acc_empty[b], 4);
        }
        mbar_init(&sb->drain, 1);
        sb->err = 0;
        sb->timeout_ns = timeout_ns;
        mbar_init_fence();
    }
    if (warp == 1) {  // the whole warp allocates the two accumulators
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                     :: "r"(smem_u32(&sb->tmem_base)), "r"(kTmemCols) : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sb->tmem_base;

    if (warp == 0) {
        // ------------------------------------------------------ TMA producer
        if (lane == 0) {
            uint32_t it = 0;
            bool ok = true;
            for (int u = blockIdx.x; ok && u < nunits && !*(volatile int*)&sb->err;
                 u += gridDim.x) {
                const int m0 = (u % mt) * BM, nt0 = (u / mt) * kTilesPerChunk;
                const int nt1 = min(nt0 + kTilesPerChunk, ntn);
                for (int nt = nt0; ok && nt < nt1; ++nt) {
                    const int n0 = nt * BN;
                    for (int kb = 0; kb < nk; ++kb) {
                        const int s = (int)(it % kStages);
                        const uint32_t round = it / kStages;
                        if (round > 0 && !wait_phase(&sb->empty[s], (round - 1) & 1u, sb, status)) {
                            ok = false;
                            break;
                        }
                        unsigned char* a = dsm + s * kStageBytes;
                        mbar_expect_tx(&sb->full[s], kStageBytes);
                        tma_load_2d(a, &tmA, kb * BK, m0, &sb->full[s]);
                        tma_load_2d(a + kABytes, &tmB, kb * BK, n0, &sb->full[s]);
                        ++it;
                    }
                }
            }
            // the last copies issued have landed before the CTA may exit
            for (uint32_t j = it > (uint32_t)kStages ? it - kStages : 0; j < it; ++j)
                wait_phase_drain(&sb->full[j % kStages], (j / kStages) & 1u, timeout_ns);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------ MMA issuer
        if (lane == 0) {
            uint32_t it = 0;
            int lt = 0;
            bool ok = true;
            for (int u = blockIdx.x; ok && u < nunits && !*(volatile int*)&sb->err;
                 u += gridDim.x) {
                const int nt0 = (u / mt) * kTilesPerChunk, nt1 = min(nt0 + kTilesPerChunk, ntn);
                for (int nt = nt0; ok && nt < nt1; ++nt, ++lt) {
                    const int buf = lt & 1;
                    const uint32_t use = (uint32_t)lt >> 1;
                    if (use > 0 && !wait_phase(&sb->acc_empty[buf], (use - 1) & 1u, sb, status)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t d = tmem + (uint32_t)(buf * BN);
                    for (int kb = 0; kb < nk; ++kb) {
                        const int s = (int)(it % kStages);
                        if (!wait_phase(&sb->full[s], (it / kStages) & 1u, sb, status)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint32_t a = smem_u32(dsm + s * kStageBytes), b = a + kABytes;
#pragma unroll
                        for (int k = 0; k < BK / 16; ++k)
                            mma_bf16(d, sdesc_sw128(a + 32u * k), sdesc_sw128(b + 32u * k),
                                     kIdesc, (kb | k) != 0 ? 1u : 0u);
                        mma_commit(&sb->empty[s]);  // frees the stage once these MMAs are done
                        ++it;
                    }
                    if (!ok) break;
                    mma_commit(&sb->acc_full[buf]);
                }
            }
            // every MMA this thread issued is complete once this arrives
            mma_commit(&sb->drain);
            wait_phase_drain(&sb->drain, 0, timeout_ns);
        }
    } else {
        // ------------------------------------------------------ epilogue
        const int q = warp & 3;  // this warp may access TMEM lanes 32q .. 32q + 31
        int lt = 0;
        bool ok = true;
        for (int u = blockIdx.x; ok && u < nunits; u += gridDim.x) {
            const int m0 = (u % mt) * BM, ch = u / mt;
            const int nt0 = ch * kTilesPerChunk, nt1 = min(nt0 + kTilesPerChunk, ntn);
            const int row = m0 + 32 * q + lane;
            float rm = -INFINITY, rs = 0.f;  // the row's running chunk statistics
            for (int nt = nt0; nt < nt1; ++nt, ++lt) {
                const int buf = lt & 1;
                const uint32_t use = (uint32_t)lt >> 1;
                if (!wait_phase_warp(&sb->acc_full[buf], use & 1u, sb, status)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const int n0 = nt * BN;
                const uint32_t taddr = tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(buf * BN);
#pragma unroll 1
                for (int c = 0; c < BN / 32; ++c) {
                    uint32_t r[32];
                    tmem_ld32(taddr + 32u * c, r);
                    const int col = n0 + 32 * c;
                    if (row < M && col < N) {
                        __nv_bfloat16* o = out + (size_t)row * N + col;
                        uint32_t w[16];
#pragma unroll
                        for (int i = 0; i < 16; ++i) w[i] = pack_bf16(r[2 * i], r[2 * i + 1]);
#pragma unroll
                        for (int v = 0; v < 4; ++v)
                            if (col + 8 * v < N)
                                *reinterpret_cast<uint4*>(o + 8 * v) =
                                    make_uint4(w[4 * v], w[4 * v + 1], w[4 * v + 2], w[4 * v + 3]);
                        if (cs.tab) {
                            // the rounded logits of the group, then the running
                            // (max, sum) rescaled to the new maximum
                            float f[32];
#pragma unroll
                            for (int i = 0; i < 16; ++i) {
                                f[2 * i] = __uint_as_float(w[i] << 16);
                                f[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
                            }
                            float gm = -INFINITY;
#pragma unroll
                            for (int i = 0; i < 32; ++i)
                                if (col + i < N) gm = fmaxf(gm, f[i]);
                            const float nm = fmaxf(rm, gm);
                            if (nm > -INFINITY) {
                                float acc = rs * vsd::ex2((rm - nm) * cs.c);
#pragma unroll
                                for (int i = 0; i < 32; ++i)
                                    if (col + i < N) acc += vsd::ex2((f[i] - nm) * cs.c);
                                rs = acc;
                                rm = nm;
                            }
                        }
                    }
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&sb->acc_empty[buf]);
            }
            if (ok && cs.tab && row < M)
                reinterpret_cast<float2*>(cs.tab + (size_t)row * cs.stride + ch)[0] =
                    make_float2(rm, rs);
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;"
                     :: "r"(tmem), "r"(kTmemCols) : "memory");
    }
}

// ---------------------------------------------------------------- host side
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

// cuTensorMapEncodeTiled through the runtime's driver entry point (no link
// against the driver library).
EncodeTiledFn encode_fn() {
    static std::once_flag once;
    static EncodeTiledFn fn = nullptr;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    });
    return fn;
}

// Tensor map of a row-major bf16 matrix [rows][cols] read in boxes of
// box_rows x 64 columns with the 128-byte swizzle; out-of-range elements read
// as zero (they add nothing to a dot product).
bool make_map_box(CUtensorMap* m, const void* base, int rows, int cols, int box_cols,
                  int box_rows, int swizzle_bytes) {
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    const cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    const cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
    const cuuint32_t box[2] = {(cuuint32_t)box_cols, (cuuint32_t)box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
               box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
               swizzle_bytes == 128  ? CU_TENSOR_MAP_SWIZZLE_128B
               : swizzle_bytes == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                                     : CU_TENSOR_MAP_SWIZZLE_NONE,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
           CUDA_SUCCESS;
}

bool make_map(CUtensorMap* m, const void* base, int rows, int cols, int box_rows) {
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    const cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    const cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
    const cuuint32_t box[2] = {(cuuint32_t)BK, (cuuint32_t)box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
               box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
           CUDA_SUCCESS;
}

}  // namespace vsd_lm

namespace vsd {

bool lmhead_shape_ok(const void* hidden, const void* weight, const void* logits, int M, int N,
                     int K) {
    if (!hidden || !weight || !logits) return false;
    if (M < 1 || N < 8 || K < 8) return false;
    if (N % 8 || K % 8) return false;  // 16-byte rows for TMA and for the stores
    if (((uintptr_t)hidden | (uintptr_t)weight | (uintptr_t)logits) & 15) return false;
    return true;
}

cudaError_t lmhead_gemm(const void* hidden, const void* weight, int M, int N, int K, void* logits,
                        int* status, uint64_t timeout_ns, cudaStream_t s, float4* chunk_tab,
                        int chunk_stride, float chunk_c) {
    using vsd_lm::k_lmhead;
    using vsd_lm::make_map;
    CUtensorMap ta, tb;
    if (!make_map(&ta, hidden, M, K, vsd_lm::BM) || !make_map(&tb, weight, N, K, vsd_lm::BN))
        return cudaErrorInvalidValue;
    int dev = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    {  // the shared-memory opt-in, once per device
        static std::mutex mu;
        static bool done[256];
        std::lock_guard<std::mutex> lock(mu);
        if (dev < 0 || dev >= 256) return cudaErrorInvalidDevice;
        if (!done[dev]) {
            e = cudaFuncSetAttribute(k_lmhead, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)vsd_lm::kSmemBytes);
            if (e != cudaSuccess) return e;
            done[dev] = true;
        }
    }
    const long long ntn = (N + vsd_lm::BN - 1) / vsd_lm::BN;
    const long long nunits = (long long)((M + vsd_lm::BM - 1) / vsd_lm::BM) *
                             ((ntn + vsd_lm::kTilesPerChunk - 1) / vsd_lm::kTilesPerChunk);
#ifndef VSD_LM_CTAS_PER_SM
#define VSD_LM_CTAS_PER_SM 1
#endif
    const long long slots = (long long)sms * VSD_LM_CTAS_PER_SM;
    const int grid = (int)(nunits < slots ? nunits : slots);
    const vsd_lm::ChunkStatsOut cs{chunk_tab, chunk_stride, chunk_c};
    // (qualified: the enclosing namespace has a kThreads of its own)
    k_lmhead<<<grid, vsd_lm::kThreads, vsd_lm::kSmemBytes, s>>>(
        ta, tb, static_cast<__nv_bfloat16*>(logits), M, N, K, status, timeout_ns, cs);
    return cudaGetLastError();
}

}  // namespace vsd
