// vsd_kernels_impl.cuh -- kernels and launchers for one logit dtype VSD_T.
// Included once by vsd_kernels_f32.cu and once by vsd_kernels_bf16.cu.
#pragma once

#include "vsd_launch.h"

namespace vsd {

// Dynamic shared memory: [Ring (vector rows)] [chunk table].
template <bool VEC>
__device__ __forceinline__ void smem_views(unsigned char* dsm, Ring*& rg, float4*& tab) {
    if (VEC) {
        rg = reinterpret_cast<Ring*>(dsm);
        tab = reinterpret_cast<float4*>(dsm + sizeof(Ring));
        ring_init(rg);
    } else {
        rg = nullptr;
        tab = reinterpret_cast<float4*>(dsm);
    }
}

// ------------------------------------------------------------ separate kernels
template <typename T, bool VEC>
__global__ void __launch_bounds__(kThreads) k_sample(Problem<T> P) {
    extern __shared__ __align__(128) unsigned char dsm[];
    __shared__ RowShared sh;
    Ring* rg;
    float4* tab;
    smem_views<VEC>(dsm, rg, tab);
    const int r = blockIdx.x;
    row_pass<T, VEC, false, kSampleToken, false>(P, r, rg, tab, sh);
    if (threadIdx.x == 0) {
        const RowRec rec = P.rows[r];
        P.out.tokens[r] = rec.tok;
        P.out.logq_tok[r] = rec.lq_tok;
        if (P.out.row_stats)
            reinterpret_cast<float4*>(P.out.row_stats)[r] =
                make_float4(rec.mx, (float)rec.lzx, 0.f, 0.f);
    }
}

template <typename T, bool VEC, bool TREE>
__global__ void __launch_bounds__(kThreads) k_rows_verify(Problem<T> P) {
    extern __shared__ __align__(128) unsigned char dsm[];
    __shared__ RowShared sh;
    Ring* rg;
    float4* tab;
    smem_views<VEC>(dsm, rg, tab);
    if (TREE)
        row_pass<T, VEC, true, kNoToken, false>(P, blockIdx.x, rg, tab, sh);
    else
        row_pass<T, VEC, true, kGivenToken, true>(P, blockIdx.x, rg, tab, sh);
}

template <typename T, bool VEC>
__global__ void __launch_bounds__(kThreads) k_paths(Problem<T> P) {
    extern __shared__ __align__(128) unsigned char dsm[];
    __shared__ PathShared sh;
    Ring* rg;
    float4* tab;
    smem_views<VEC>(dsm, rg, tab);
    path_pass<T, VEC>(P, blockIdx.x, rg, tab, sh);
}

template <typename T, bool VEC>
__global__ void __launch_bounds__(kThreads) k_tree(Problem<T> P) {
    extern __shared__ __align__(128) unsigned char dsm[];
    __shared__ TreeShared sh;
    Ring* rg;
    float4* tab;
    smem_views<VEC>(dsm, rg, tab);
    tree_pass<T, VEC>(P, blockIdx.x, rg, tab, sh);
}

template <typename T>
__global__ void __launch_bounds__(kThreads)
    k_weights(Problem<T> P, EStepView E, float* weights, float* loss) {
    __shared__ WeightsShared sh;
    __shared__ int last;
    weights_pass<T>(P, E, blockIdx.x, weights, loss, sh);
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        last = atomicAdd(P.prefix_done, 1) == P.B - 1;
        if (last) {
            __threadfence();
            loss_mean(loss, P.B);
        }
    }
}

template <typename T, bool VEC, typename G>
__global__ void __launch_bounds__(kThreads) k_grad(Problem<T> P, const float4* rstats, G* grad) {
    grad_pass<T, VEC, G>(P, blockIdx.x, rstats, grad);
}

// ------------------------------------------------------------ fused kernel
// Bounded wait for a flag set by another block; gives up after timeout_ns or
// as soon as another wait has timed out (status bit), never spins forever.
__device__ __forceinline__ bool wait_flag(const int* flag, int* status, uint64_t timeout_ns) {
    if (ld_acquire(flag)) return true;
    const uint64_t t0 = global_timer_ns();
    for (;;) {
        if (ld_acquire(flag)) return true;
        if (*(volatile int*)status & VSD_STATUS_TIMEOUT) return false;
        if (global_timer_ns() - t0 > timeout_ns) return false;
        __nanosleep(1000);
    }
}

// Persistent E-step + M-step.  Each block repeatedly takes the next work item:
// a gradient row of the oldest prefix whose M-step is already published, if
// any is left; otherwise the next logit row (rows in prefix order).  A row item
// streams one draft/target row; the block that completes the last row of a
// path runs its path pass; the block that completes the last path of a
// prefix runs the prefix's M-step and publishes it.  A block waits (bounded)
// only once every row has been claimed; claimed rows are finished by running
// blocks that never wait, so progress does not depend on residency.  Gradient
// rows follow their prefix closely, so the draft rows they re-read are still
// in L2.
#ifndef VSD_FUSED_MIN_BLOCKS
#define VSD_FUSED_MIN_BLOCKS 4
#endif
template <typename T, bool VEC, typename G>
__global__ void __launch_bounds__(kThreads, VSD_FUSED_MIN_BLOCKS) k_fused(Problem<T> P, G* grad) {
    extern __shared__ __align__(128) unsigned char dsm[];
    __shared__ union {
        RowShared row;
        PathShared path;
        WeightsShared w;
    } sh;
    Ring* rg;
    float4* tab;
    smem_views<VEC>(dsm, rg, tab);
    __shared__ int s_kind, s_idx, s_flag;
    const int Pp = P.K * P.D;
    const int B = P.B;
    const EStepView E{P.es.tok, P.es.corr, P.es.lq_tok, P.es.lq_corr,
                      P.es.lk, P.es.lkc, P.es.lkr};
    for (;;) {
        if (threadIdx.x == 0) {
            int kind = 0, idx = 0;  // 0: finished, 1: logit row, 2: gradient row
            int g = *(volatile int*)P.grad_head;
            for (;;) {
                if (*(volatile int*)P.status & VSD_STATUS_TIMEOUT) break;  // stop after a failed wait
                while (g < B && ld_acquire(P.ready + g)) {
                    const int t = atomicAdd(P.grad_cnt + g, 1);
                    if (t < Pp) { kind = 2; idx = g * Pp + t; break; }
                    atomicMax(P.grad_head, g + 1);
                    ++g;
                }
                if (kind) break;
                const int t = atomicAdd(P.ticket, 1);
                if (t < P.R) { kind = 1; idx = t; break; }
                if (g >= B) break;
                if (!wait_flag(P.ready + g, P.status, P.timeout_ns)) {
                    atomicOr(P.status, VSD_STATUS_TIMEOUT);
                    break;
                }
            }
            s_kind = kind;
            s_idx = idx;
        }
        __syncthreads();
        const int kind = s_kind, r = s_idx;
        __syncthreads();
        if (kind == 0) break;
        if (kind == 1) {
            const int prefix = r / Pp;
            row_pass<T, VEC, true, kSampleToken, true>(P, r, rg, tab, sh.row);
            const int path = r / P.D;
            if (threadIdx.x == 0) {
                __threadfence();
                s_flag = atomicAdd(P.path_cnt + path, 1) == P.D - 1;
                if (s_flag) __threadfence();
            }
            __syncthreads();
            if (s_flag) {
                path_pass<T, VEC>(P, path, rg, tab, sh.path);
                __syncthreads();
                if (threadIdx.x == 0) {
                    __threadfence();
                    s_flag = atomicAdd(P.prefix_cnt + prefix, 1) == P.K - 1;
                    if (s_flag) __threadfence();
                }
                __syncthreads();
                if (s_flag) {
                    weights_pass<T>(P, E, prefix, P.out.weights, P.out.loss, sh.w);
                    __syncthreads();
                    if (threadIdx.x == 0) {
                        __threadfence();
                        if (!P.inject_wait_fault) st_release(P.ready + prefix, 1);
                        if (atomicAdd(P.prefix_done, 1) == P.B - 1) {
                            __threadfence();
                            loss_mean(P.out.loss, P.B);
                        }
                    }
                }
            }
        } else {
            grad_pass<T, VEC, G>(P, r, P.rstats, grad);
        }
        __syncthreads();
    }
}

// ------------------------------------------------------------ launchers
template <typename K>
static cudaError_t prep(K kernel, size_t smem) {
    if (smem > 48 * 1024)
        return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)smem);
    return cudaSuccess;
}

template <>
cudaError_t Launch<VSD_T>::sample(const Problem<VSD_T>& P, bool vec, cudaStream_t s) {
    const size_t smem = stream_smem_bytes(P.nch, vec);
    if (vec) {
        cudaError_t e = prep(k_sample<VSD_T, true>, smem);
        if (e) return e;
        k_sample<VSD_T, true><<<P.R, kThreads, smem, s>>>(P);
    } else {
        cudaError_t e = prep(k_sample<VSD_T, false>, smem);
        if (e) return e;
        k_sample<VSD_T, false><<<P.R, kThreads, smem, s>>>(P);
    }
    return cudaGetLastError();
}

template <>
cudaError_t Launch<VSD_T>::rows_verify(const Problem<VSD_T>& P, bool vec, bool tree,
                                       cudaStream_t s) {
    const size_t smem = stream_smem_bytes(P.nch, vec);
#define VSD_ROWS(V_, T_)                                              \
    do {                                                              \
        cudaError_t e = prep(k_rows_verify<VSD_T, V_, T_>, smem);     \
        if (e) return e;                                              \
        k_rows_verify<VSD_T, V_, T_><<<P.R, kThreads, smem, s>>>(P);  \
    } while (0)
    if (vec && tree) VSD_ROWS(true, true);
    else if (vec) VSD_ROWS(true, false);
    else if (tree) VSD_ROWS(false, true);
    else VSD_ROWS(false, false);
#undef VSD_ROWS
    return cudaGetLastError();
}

template <>
cudaError_t Launch<VSD_T>::paths(const Problem<VSD_T>& P, bool vec, cudaStream_t s) {
    const size_t smem = stream_smem_bytes(P.nch, vec);
    const int npaths = P.B * P.K;
    if (vec) {
        cudaError_t e = prep(k_paths<VSD_T, true>, smem);
        if (e) return e;
        k_paths<VSD_T, true><<<npaths, kThreads, smem, s>>>(P);
    } else {
        cudaError_t e = prep(k_paths<VSD_T, false>, smem);
        if (e) return e;
        k_paths<VSD_T, false><<<npaths, kThreads, smem, s>>>(P);
    }
    return cudaGetLastError();
}

template <>
cudaError_t Launch<VSD_T>::tree(const Problem<VSD_T>& P, bool vec, cudaStream_t s) {
    const size_t smem = stream_smem_bytes(P.nch, vec);
    if (vec) {
        cudaError_t e = prep(k_tree<VSD_T, true>, smem);
        if (e) return e;
        k_tree<VSD_T, true><<<P.B, kThreads, smem, s>>>(P);
    } else {
        cudaError_t e = prep(k_tree<VSD_T, false>, smem);
        if (e) return e;
        k_tree<VSD_T, false><<<P.B, kThreads, smem, s>>>(P);
    }
    return cudaGetLastError();
}

template <>
cudaError_t Launch<VSD_T>::weights(const Problem<VSD_T>& P, const EStepView& E, float* weights,
                                   float* loss, cudaStream_t s) {
    k_weights<VSD_T><<<P.B, kThreads, 0, s>>>(P, E, weights, loss);
    return cudaGetLastError();
}

template <>
cudaError_t Launch<VSD_T>::grad(const Problem<VSD_T>& P, bool vec, const float4* rstats,
                                void* grad, bool grad_bf16, cudaStream_t s) {
#define VSD_GRAD(V_, G_) \
    k_grad<VSD_T, V_, G_><<<P.R, kThreads, 0, s>>>(P, rstats, reinterpret_cast<G_*>(grad))
    if (vec && grad_bf16) VSD_GRAD(true, __nv_bfloat16);
    else if (vec) VSD_GRAD(true, float);
    else if (grad_bf16) VSD_GRAD(false, __nv_bfloat16);
    else VSD_GRAD(false, float);
#undef VSD_GRAD
    return cudaGetLastError();
}

template <>
cudaError_t Launch<VSD_T>::fused(const Problem<VSD_T>& P, bool vec, void* grad, bool grad_bf16,
                                 int ctas, cudaStream_t s) {
    const size_t smem = stream_smem_bytes(P.nch, vec);
#define VSD_FUSED(V_, G_)                                                              \
    do {                                                                               \
        cudaError_t e = prep(k_fused<VSD_T, V_, G_>, smem);                            \
        if (e) return e;                                                               \
        k_fused<VSD_T, V_, G_><<<ctas, kThreads, smem, s>>>(P, reinterpret_cast<G_*>(grad)); \
    } while (0)
    if (vec && grad_bf16) VSD_FUSED(true, __nv_bfloat16);
    else if (vec) VSD_FUSED(true, float);
    else if (grad_bf16) VSD_FUSED(false, __nv_bfloat16);
    else VSD_FUSED(false, float);
#undef VSD_FUSED
    return cudaGetLastError();
}

template <>
int Launch<VSD_T>::fused_blocks_per_sm(const Problem<VSD_T>& P, bool vec, bool grad_bf16) {
    const size_t smem = stream_smem_bytes(P.nch, vec);
    // the attribute must allow this much before the occupancy query counts it
    if (vec && grad_bf16) prep(k_fused<VSD_T, true, __nv_bfloat16>, smem);
    else if (vec) prep(k_fused<VSD_T, true, float>, smem);
    else if (grad_bf16) prep(k_fused<VSD_T, false, __nv_bfloat16>, smem);
    else prep(k_fused<VSD_T, false, float>, smem);
    int n = 0;
    cudaError_t e;
    if (vec && grad_bf16)
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_fused<VSD_T, true, __nv_bfloat16>, kThreads, smem);
    else if (vec)
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_fused<VSD_T, true, float>, kThreads, smem);
    else if (grad_bf16)
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_fused<VSD_T, false, __nv_bfloat16>, kThreads, smem);
    else
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_fused<VSD_T, false, float>, kThreads, smem);
    if (e != cudaSuccess || n < 1) return 1;
    return n;
}

template struct Launch<VSD_T>;

}  // namespace vsd
