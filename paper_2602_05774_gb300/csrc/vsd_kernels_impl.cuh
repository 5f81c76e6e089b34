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

// End of a path (block): epilogue, then the prefix counter; the block that
// completes the prefix's last path runs its M-step and publishes it.
template <typename T>
__device__ void finish_path(const Problem<T>& P, const EStepView& E, int path, int A, int resid,
                            WeightsShared& wsh, int* s_flag) {
    path_epilogue<T>(P, path, A, resid);
    __syncthreads();
    const int prefix = path / P.K;
    if (threadIdx.x == 0) {
        __threadfence();
        *s_flag = atomicAdd(P.prefix_cnt + prefix, 1) == P.K - 1;
        if (*s_flag) __threadfence();
    }
    __syncthreads();
    if (*s_flag) {
        weights_pass<T>(P, E, prefix, P.out.weights, P.out.loss, wsh);
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

// Persistent E-step + M-step over row segments (segc chunks of a row).  Each
// block repeatedly takes, in this order of priority:
//   1. a residual segment from the queue (residual draws gate a prefix's M-step),
//   2. a gradient segment of the oldest prefix whose M-step is published,
//   3. the next logit-row segment (rows in prefix order).
// A row segment streams its chunks of the draft and target rows into the
// row's table in global memory; the block completing a row's last segment
// runs the row tail; the block completing a path's last row finds its
// accepted length and queues the residual row's segments (or, if every token
// was accepted, ends the path); the block completing a path's last residual
// segment draws the residual token and ends the path; the block ending a
// prefix's last path runs the M-step and publishes it.  Claimed work never
// waits; a block with nothing to claim polls (bounded by the wait timeout),
// so progress does not depend on residency.  Splitting rows lets a prefix be
// published soon after its rows are read, so its gradient segments re-read
// draft rows that are still in L2.
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
    __shared__ int s_kind, s_idx, s_flag;
    Ring* rg;
    float4* tab;
    smem_views<VEC>(dsm, rg, tab);
    constexpr int CE = chunk_elems<T>();
    const int Pp = P.K * P.D;
    const int B = P.B, D = P.D, nseg = P.nseg, segc = P.segc, nch = P.nch;
    const int row_items = P.R * nseg;
    const int grad_items = Pp * nseg;  // per prefix
    const int64_t V = P.V;
    const float c = P.ts.c;
    const EStepView E{P.es.tok, P.es.corr, P.es.lq_tok, P.es.lq_corr,
                      P.es.lk, P.es.lkc, P.es.lkr};
    for (;;) {
        if (threadIdx.x == 0) {
            int kind = 0, idx = 0;  // 0 finished, 1 row, 2 gradient, 3 residual segment
            uint64_t idle_since = 0;
            int g = *(volatile int*)P.grad_head;
            for (;;) {
                // independent reads first (one round trip), then at most one
                // attempt per kind of work
                const int h = *(volatile int*)P.resq_head;
                const int tl = *(volatile int*)P.resq_tail;
                const int tk = *(volatile int*)P.ticket;
                const int rdy = g < B ? ld_acquire(P.ready + g) : 0;
                if (h < tl && atomicCAS(P.resq_head, h, h + 1) == h) {
                    if (!wait_flag(P.resq_flag + h, P.status, P.timeout_ns)) {
                        atomicOr(P.status, VSD_STATUS_TIMEOUT);
                        break;
                    }
                    kind = 3;
                    idx = ld_cg(P.resq + h);
                    break;
                }
                if (rdy) {
                    const int t = atomicAdd(P.grad_cnt + g, 1);
                    if (t < grad_items) { kind = 2; idx = g * grad_items + t; break; }
                    atomicMax(P.grad_head, g + 1);
                    ++g;
                    continue;
                }
                if (tk < row_items) {
                    const int t = atomicAdd(P.ticket, 1);
                    if (t < row_items) { kind = 1; idx = t; break; }
                }
                if (g >= B) break;  // every gradient segment has been claimed
                if (*(volatile int*)P.status & VSD_STATUS_TIMEOUT) break;
                if (h < tl) continue;  // residual work is pending: try again at once
                const uint64_t now = global_timer_ns();
                if (idle_since == 0) {
                    idle_since = now;
                } else if (now - idle_since > P.timeout_ns) {
                    atomicOr(P.status, VSD_STATUS_TIMEOUT);
                    break;
                }
                __nanosleep(1000);
            }
            s_kind = kind;
            s_idx = idx;
        }
        __syncthreads();
        const int kind = s_kind, it = s_idx;
        __syncthreads();
        if (kind == 0) break;
        if (kind == 1) {  // ------------------------------------- row segment
            const int r = it / nseg, seg = it - r * nseg;
            const int c0 = seg * segc, c1 = min(nch, c0 + segc);
            const T* x = P.draft + (int64_t)r * V;
            const T* y = P.target + (int64_t)r * V;
            float4* rtab = P.gtab + (int64_t)r * P.nch_ws;
            // The draft row is read again for the gradient: ask L2 to keep it.
            stream_tables<T, VEC, true>(rg, x, y, V, c0, c1, rtab, c, policy_evict_last(),
                                        policy_evict_first(), P.status);
            __syncthreads();
            if (threadIdx.x == 0) {
                __threadfence();
                s_flag = atomicAdd(P.row_seg_cnt + r, 1) == nseg - 1;
                if (s_flag) __threadfence();
            }
            __syncthreads();
            if (!s_flag) continue;
            for (int ch = threadIdx.x; ch < nch; ch += kThreads) tab[ch] = ld_cg(rtab + ch);
            __syncthreads();
            row_tail<T, VEC, true, kSampleToken, true>(P, r, tab, sh.row);
            __syncthreads();
            const int path = r / D;
            if (threadIdx.x == 0) {
                __threadfence();
                s_flag = atomicAdd(P.path_cnt + path, 1) == D - 1;
                if (s_flag) __threadfence();
            }
            __syncthreads();
            if (!s_flag) continue;
            path_head<T>(P, path, sh.path);
            __syncthreads();
            const int A = sh.path.A;
            if (A < D && !sh.path.rec.flags) {
                if (threadIdx.x == 0) {  // queue the residual row's segments
                    P.path_A[path] = A;
                    const int base = atomicAdd(P.resq_tail, nseg);
                    for (int sg = 0; sg < nseg; ++sg) P.resq[base + sg] = path * nseg + sg;
                    __threadfence();
                    for (int sg = 0; sg < nseg; ++sg) st_release(P.resq_flag + base + sg, 1);
                }
            } else {
                finish_path<T>(P, E, path, A, -1, sh.w, &s_flag);
            }
        } else if (kind == 3) {  // ------------------------- residual segment
            const int path = it / nseg, seg = it - path * nseg;
            const int c0 = seg * segc, c1 = min(nch, c0 + segc);
            if (threadIdx.x == 0) {
                sh.path.A = ld_cg(P.path_A + path);
                sh.path.rec = ld_cg(P.rows + path * D + sh.path.A);
            }
            __syncthreads();
            const int A = sh.path.A;
            const int rA = path * D + A;
            const RowRec rec = sh.path.rec;
            const T* x = P.draft + (int64_t)rA * V;
            const T* y = P.target + (int64_t)rA * V;
            float4* rtab = P.gtab + (int64_t)rA * P.nch_ws;  // row A's table is free again
            const MassRes mr{rec.mx, rec.my, (float)exp(-rec.lzx), (float)exp(-rec.lzy), c};
            stream_residual<T, VEC>(rg, x, y, V, c0, c1, rtab, mr, P.status);
            __syncthreads();
            if (threadIdx.x == 0) {
                __threadfence();
                s_flag = atomicAdd(P.res_seg_cnt + path, 1) == nseg - 1;
                if (s_flag) __threadfence();
            }
            __syncthreads();
            if (!s_flag) continue;
            for (int ch = threadIdx.x; ch < nch; ch += kThreads) tab[ch] = ld_cg(rtab + ch);
            __syncthreads();
            const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
            if (warp == 0) {
                const double Rt = table_total(tab, nch, 0, 0.f, c, lane);
                int tok = -1;
                if (Rt > 0.0) {
                    const float u = __ldg(P.u_correct + rA);
                    const Located loc = table_locate(tab, nch, 0, 0.f, c, (double)u * Rt, lane);
                    if (loc.ch >= 0)
                        tok = warp_rescan<T, VEC, true, true>(x, y, V, loc.ch, loc.tc, mr, lane,
                                                              policy_evict_normal());
                }
                if (lane == 0) sh.path.resid = tok < V ? tok : -1;
            }
            __syncthreads();
            finish_path<T>(P, E, path, A, sh.path.resid, sh.w, &s_flag);
        } else {  // ------------------------------------------ gradient segment
            const int b = it / grad_items, t = it - b * grad_items;
            const int r = b * Pp + t / nseg, seg = t % nseg;
            const int64_t e0 = (int64_t)seg * segc * CE;
            const int64_t e1 = min(V, e0 + (int64_t)segc * CE);
            grad_pass_range<T, VEC, G>(P, r, e0, e1, P.rstats, grad);
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
