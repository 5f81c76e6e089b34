// vsd_kernels_impl.cuh -- kernels and launchers for one logit dtype VSD_T.
// Included once by vsd_kernels_f32.cu and once by vsd_kernels_bf16.cu.
#pragma once

#include "vsd_launch.h"

namespace vsd {

// Dynamic shared memory: [Ring (vector rows)] [chunk table].
template <bool VEC>
__device__ __forceinline__ void smem_views(unsigned char* dsm, Ring*& rg, float4*& tab,
                                           uint64_t timeout_ns) {
    if (VEC) {
        rg = reinterpret_cast<Ring*>(dsm);
        tab = reinterpret_cast<float4*>(dsm + sizeof(Ring));
        ring_init(rg, timeout_ns);
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
    smem_views<VEC>(dsm, rg, tab, P.timeout_ns);
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

template <typename T, bool VEC>
__global__ void __launch_bounds__(kThreads) k_rows_verify(Problem<T> P) {
    extern __shared__ __align__(128) unsigned char dsm[];
    __shared__ RowShared sh;
    Ring* rg;
    float4* tab;
    smem_views<VEC>(dsm, rg, tab, P.timeout_ns);
    row_pass<T, VEC, true, kGivenToken, true>(P, blockIdx.x, rg, tab, sh);
}

// Rows along supplied greedy reference paths (Algorithm 2's z-bar): per row
// the target's argmax and log min(1, p/q) there (row_pass with the argmax).
template <typename T, bool VEC>
__global__ void __launch_bounds__(kThreads) k_ref_rows(Problem<T> P) {
    extern __shared__ __align__(128) unsigned char dsm[];
    __shared__ RowShared sh;
    Ring* rg;
    float4* tab;
    smem_views<VEC>(dsm, rg, tab, P.timeout_ns);
    row_pass<T, VEC, true, kNoToken, true>(P, blockIdx.x, rg, tab, sh);
}

// log kappa(z-bar_{<=l}) of reference path b: the prefix sums over its rows
// of log min(1, p/q) at the argmax (one warp per path, Eq. 2).
template <typename T>
__global__ void k_ref_scan(Problem<T> P, float* out) {
    const int b = blockIdx.x, lane = threadIdx.x & 31;
    double carry = 0.0;
    for (int d0 = 0; d0 < P.D; d0 += 32) {
        const int d = d0 + lane;
        double la = 0.0;
        if (d < P.D) {
            const RowRec rec = P.rows[(int64_t)b * P.D + d];
            la = (rec.flags || rec.ref < 0) ? -INFINITY : (double)rec.la_ref;
        }
        const double inc = carry + warp_incl_scan(la, lane);
        if (d < P.D) out[(int64_t)b * P.D + d] = (float)inc;
        carry = __shfl_sync(0xffffffffu, inc, 31);
    }
}

template <typename T, bool VEC>
__global__ void __launch_bounds__(kThreads) k_paths(Problem<T> P) {
    extern __shared__ __align__(128) unsigned char dsm[];
    __shared__ PathShared sh;
    Ring* rg;
    float4* tab;
    smem_views<VEC>(dsm, rg, tab, P.timeout_ns);
    path_pass<T, VEC>(P, blockIdx.x, rg, tab, sh);
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

// Residual queue: producers reserve slots (resq_tail), write the items,
// release each slot's flag and then add the items to resq_avail.  A consumer
// reserves one published item with one atomic on resq_avail (returned at once
// if none was left) and takes the next slot with one atomic on resq_head, so
// claims pipeline in L2 instead of queueing behind a compare-and-swap.  The
// slot may belong to a producer that reserved it but has not released it yet
// (it is running, past its reservation): a bounded wait on the flag.
// Callers look at resq_avail first.  Returns the item, -1 if none was left,
// -2 if the wait ran out (status bit set).
__device__ __forceinline__ int take_residual(int* head, int* avail, const int* flags,
                                             const int* items, int* status,
                                             uint64_t timeout_ns) {
    if (atomicSub(avail, 1) <= 0) {
        atomicAdd(avail, 1);
        return -1;
    }
    const int h = atomicAdd(head, 1);
    if (!wait_flag(flags + h, status, timeout_ns)) {
        atomicOr(status, VSD_STATUS_TIMEOUT);
        return -2;
    }
    return ld_cg(items + h);
}

__device__ __forceinline__ void publish_residuals(int* tail, int* avail, int* flags, int* items,
                                                  int first, int n, bool sem) {
    const int base = atomicAdd(tail, n);
    for (int i = 0; i < n; ++i) items[base + i] = first + i;
    __threadfence();
    for (int i = 0; i < n; ++i) st_release(flags + base + i, 1);
    if (sem) atomicAdd(avail, n);
}

// The fused kernel's block: kWarps streaming warps (threads 0 .. kThreads-1)
// that only move logits, and one control warp (the last) that claims work,
// keeps the counters and runs every per-row, per-path and per-prefix step.
constexpr int kFusedThreads = kThreads + 32;
#ifndef VSD_SLOTS
#define VSD_SLOTS 2
#endif
constexpr int kSlots = VSD_SLOTS;  // jobs handed to the streaming warps ahead of time
// Named barriers (0 is __syncthreads): slot s is FULL (1 + s) when the control
// warp has written a job into it, DONE (1 + kSlots + s) when the streaming
// warps have finished that job.
__device__ __forceinline__ int bar_full(int s) { return 1 + s; }
__device__ __forceinline__ int bar_done(int s) { return 1 + kSlots + s; }
constexpr int kStreamBar = 1 + 2 * kSlots;  // the streaming warps among themselves
__device__ __forceinline__ void named_sync(int id) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(kFusedThreads) : "memory");
}
__device__ __forceinline__ void named_arrive(int id) {
    asm volatile("bar.arrive %0, %1;" ::"r"(id), "r"(kFusedThreads) : "memory");
}

enum JobKind { kJobEnd = 0, kJobRow = 1, kJobGrad = 2, kJobResidual = 3 };
struct Job {
    int kind;
    int r;       // the row streamed (residual: row A of the path)
    int item;    // row segment or residual item index
    int c0, c1;  // chunk range of the segment
    int path, A;
    MassRes mr;  // residual segment: the row's normalisers
};

// Claim the next job (lane 0 of the control warp), in this order of priority:
//   1. a residual segment from the queue (residual draws gate a prefix's M-step),
//   2. a gradient segment of the oldest prefix whose M-step is published,
//   3. the next logit-row segment (rows in prefix order).
// With wait = false returns false at once when nothing is available; with
// wait = true polls (bounded by the wait timeout) until a job or the end.
// The caller may only wait when it has no job in flight whose follow-up steps
// it still owes, so that no block waits on work that it holds itself.
template <typename T>
__device__ bool claim_job(const Problem<T>& P, bool wait, int& g, Job& j) {
    const int B = P.B, nseg = P.nseg, segc = P.segc;
    const int row_items = P.R * nseg;
    uint64_t idle_since = 0;
    j.kind = kJobEnd;
    for (;;) {
        // independent reads first (one round trip), then at most one attempt
        // per kind of work
        const int tk = *(volatile int*)P.ticket;
        const int rdy = g < B ? ld_acquire(P.ready + g) : 0;
        int it = -1, av;
        if (P.resq_sem) {  // short rows: claims must not queue (the chain bounds the kernel)
            av = *(volatile int*)P.resq_avail > 0;
            if (av)
                it = take_residual(P.resq_head, P.resq_avail, P.resq_flag, P.resq, P.status,
                                   P.timeout_ns);
        } else {  // long rows: one compare-and-swap, fewer round trips per claim
            const int h = *(volatile int*)P.resq_head;
            const int tl = *(volatile int*)P.resq_tail;
            av = h < tl;
            if (av && atomicCAS(P.resq_head, h, h + 1) == h) {
                it = wait_flag(P.resq_flag + h, P.status, P.timeout_ns) ? ld_cg(P.resq + h) : -2;
                if (it == -2) atomicOr(P.status, VSD_STATUS_TIMEOUT);
            }
        }
        if (it == -2) return true;  // a wait ran out: end
        if (it >= 0) {
            const int path = it / nseg, seg = it - path * nseg;
            const int A = ld_cg(P.path_A + path);
            const int rA = path * P.D + A;
            const RowRec rec = ld_cg(P.rows + rA);
            j.kind = kJobResidual;
            j.item = it;
            j.path = path;
            j.A = A;
            j.r = rA;
            j.c0 = seg * segc;
            j.c1 = min(P.nch, j.c0 + segc);
            j.mr = MassRes{rec.mx, rec.my, rec.izx, rec.izy, P.ts.c};
            return true;
        }
        if (rdy) {
            const int gn = P.gnseg, gs = P.gsegc;
            const int t = atomicAdd(P.grad_cnt + g, 1);
            if (t < P.K * P.D * gn) {
                const int seg = t % gn;
                j.kind = kJobGrad;
                j.r = g * P.K * P.D + t / gn;
                j.c0 = seg * gs;
                j.c1 = min(P.nch, j.c0 + gs);
                return true;
            }
            atomicMax(P.grad_head, g + 1);
            ++g;
            continue;
        }
        if (tk < row_items) {
            const int t = atomicAdd(P.ticket, 1);
            if (t < row_items) {
                const int seg = t % nseg;
                j.kind = kJobRow;
                j.item = t;
                j.r = t / nseg;
                j.c0 = seg * segc;
                j.c1 = min(P.nch, j.c0 + segc);
                return true;
            }
        }
        if (g >= B) return true;  // every gradient segment has been claimed: end
        if (*(volatile int*)P.status & VSD_STATUS_TIMEOUT) return true;
        if (!wait) return false;
        if (av) continue;  // residual work is pending: try again at once
        const uint64_t now = global_timer_ns();
        if (idle_since == 0) {
            idle_since = now;
        } else if (now - idle_since > P.timeout_ns) {
            atomicOr(P.status, VSD_STATUS_TIMEOUT);
            return true;
        }
        __nanosleep(1000);
    }
}

// Last-finisher counter (control warp): lane 0 adds one to *cnt after a fence
// and every lane learns whether it completed the count n (n = 1: no counter).
__device__ __forceinline__ bool warp_count_last(int* cnt, int n, int lane) {
    if (n == 1) return true;
    int last = 0;
    if (lane == 0) {
        __threadfence();
        last = atomicAdd(cnt, 1) == n - 1;
        if (last) __threadfence();
    }
    return __shfl_sync(0xffffffffu, last, 0) != 0;
}

// Shared memory of the control warp.
union CtlShared {
    WeightsShared w;
    RescanBuf rb;
};

// End of a path (control warp): epilogue, then the prefix counter; the warp
// that completes the prefix's last path runs its M-step and publishes it.
template <typename T>
__device__ void finish_path_warp(const Problem<T>& P, const EStepView& E, int path, int A,
                                 int resid, bool have_rl, float rlq, float rla, CtlShared& cs,
                                 int lane) {
    path_epilogue_warp<T>(P, path, A, resid, lane, have_rl, rlq, rla);
    __syncwarp();
    const int prefix = path / P.K;
    if (!warp_count_last(P.prefix_cnt + prefix, P.K, lane)) return;
    weights_warp<T>(P, E, prefix, P.out.weights, P.out.loss, cs.w, lane);
    __syncwarp();
    if (lane == 0) {
        __threadfence();
        if (!P.inject_wait_fault) st_release(P.ready + prefix, 1);
        if (atomicAdd(P.prefix_done, 1) == P.B - 1) {
            __threadfence();
            loss_mean(P.out.loss, P.B);
        }
    }
}

// What the control warp does after the streaming warps finished job j.
template <typename T, bool VEC, bool KL>
__device__ void post_job(const Problem<T>& P, const EStepView& E, const Job& j, float4* tab,
                         CtlShared& cs, int lane) {
    const int D = P.D, nseg = P.nseg, nch = P.nch;
    if (j.kind == kJobRow) {
        const int r = j.r;
        if (!warp_count_last(P.row_seg_cnt + r, nseg, lane)) return;
        if (!P.stream_tails) row_tail_warp<T, VEC, KL>(P, r, tab, cs.rb, lane);
        __syncwarp();
        const int path = r / D;
        if (!warp_count_last(P.path_cnt + path, D, lane)) return;
        const int A = path_accept_len<T>(P, path, lane);
        const int flags = A < D ? ld_cg(P.rows + path * D + A).flags : 0;
        // T = 0: the residual is the target's argmax, the row's p-draw: no
        // residual row to read
        if (A < D && !flags && !P.greedy) {
            if (lane == 0) {  // queue the residual row's segments
                P.path_A[path] = A;
                publish_residuals(P.resq_tail, P.resq_avail, P.resq_flag, P.resq, path * nseg,
                                  nseg, P.resq_sem != 0);
            }
        } else {
            finish_path_warp<T>(P, E, path, A, -1, false, 0.f, 0.f, cs, lane);
        }
    } else if (j.kind == kJobResidual) {
        if (!warp_count_last(P.res_seg_cnt + j.path, nseg, lane)) return;
        const int rA = j.r;
        const int64_t V = P.V;
        const T* x = P.draft + (int64_t)rA * V;
        const T* y = P.target + (int64_t)rA * V;
        const float c = P.ts.c;
        // one round trip: row A's residual table, record and uniform
        const float u = __ldg(P.u_correct + rA);
        const RowRec rec = ld_cg(P.rows + rA);
        const float4* rtab = P.gtab + (int64_t)rA * P.nch_ws;
        for (int ch = lane; ch < nch; ch += 32) tab[ch] = ld_cg(rtab + ch);
        __syncwarp();
        const TableSum Rt = table_sum(tab, nch, 0, 0.f, c, lane);
        int tok = -1;
        Located loc{-1, 0.f};
        if (Rt.Z > 0.0) loc = table_locate(tab, nch, 0, 0.f, c, Rt, u, lane);
        uint4 bx[kLoads], by[kLoads];
        if (loc.ch >= 0) {
            if (VEC) {  // one round trip for both rows' chunks
                chunk_async<T>(cs.rb.c[0], x, V, loc.ch, lane);
                chunk_async<T>(cs.rb.c[1], y, V, loc.ch, lane);
                cp_async_wait_all();
                __syncwarp();
                chunk_from_smem<T>(cs.rb.c[0], V, loc.ch, lane, bx);
                chunk_from_smem<T>(cs.rb.c[1], V, loc.ch, lane, by);
            } else {
                load_chunk<T, VEC>(x, V, loc.ch, lane, policy_evict_normal(), bx);
                load_chunk<T, VEC>(y, V, loc.ch, lane, policy_evict_normal(), by);
            }
            tok = rescan_regs<T, true, true>(bx, by, loc.ch, loc.tc, j.mr, lane);
        }
        if (tok >= V) tok = -1;
        float rlq = 0.f, rla = 0.f;
        if (tok >= 0) {
            const float xv = VEC ? smem_elem(cs.rb.c[0], loc.ch, tok, x) : elem_value(x, tok);
            const float yv = VEC ? smem_elem(cs.rb.c[1], loc.ch, tok, y) : elem_value(y, tok);
            token_logs_vals(xv, yv, rec, P.ts.invTd, &rlq, &rla);
        }
        __syncwarp();
        finish_path_warp<T>(P, E, j.path, j.A, tok, tok >= 0, rlq, rla, cs, lane);
    }
}

// Persistent E-step + M-step over row segments (segc chunks of a row).  The
// streaming warps run the jobs that the control warp hands them through
// kSlots shared-memory slots:
//   row segment: its chunks of the draft and target rows into the row's
//     table in global memory;
//   residual segment: its chunks of row A's residual mass into row A's table;
//   gradient segment: its chunks of the draft row into the gradient row.
// The control warp claims jobs ahead, and after each job does its counter:
// the block completing a row's last segment runs the row tail; the block
// completing a path's last row finds its accepted length and queues the
// residual row's segments (or, if every token was accepted, ends the path);
// the block completing a path's last residual segment draws the residual
// token and ends the path; the block ending a prefix's last path runs the
// M-step and publishes it.  So the streaming warps never wait for a claim or
// a tail unless there is no work.  Claimed work never waits for other
// blocks; a block with nothing to claim polls (bounded by the wait timeout),
// so progress does not depend on residency.  Splitting rows lets a prefix be
// published soon after its rows are read, so its gradient segments re-read
// draft rows that are still in L2.
#ifndef VSD_FUSED_MIN_BLOCKS
#define VSD_FUSED_MIN_BLOCKS 4
#endif
// KL: VSD (KL), the rows' top-K terms (a separate instantiation, so that the
// plain kernel's code is unchanged by them).
template <typename T, bool VEC, typename G, bool KL>
__global__ void __launch_bounds__(kFusedThreads, VSD_FUSED_MIN_BLOCKS)
    k_fused(Problem<T> P, G* grad) {
    extern __shared__ __align__(128) unsigned char dsm[];
    __shared__ CtlShared cs;
    __shared__ Job slots[kSlots];
    __shared__ KlRec kslot[kSlots];  // VSD (KL): the top-K terms of a gradient job's row
    __shared__ RowShared rsh;
    Ring* rg;
    float4* tab;
    smem_views<VEC>(dsm, rg, tab, P.timeout_ns);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (warp < kWarps) {  // ------------------------------- streaming warps
        for (int i = 0;; ++i) {
            const int s = i % kSlots;
            named_sync(bar_full(s));
            const Job j = slots[s];
            if (j.kind == kJobEnd) break;
            const int64_t V = P.V;
            const T* x = P.draft + (int64_t)j.r * V;
            if (j.kind == kJobRow) {
                // The draft row is read again for the gradient: ask L2 to keep it.
                float4* rtab = P.gtab + (int64_t)j.r * P.nch_ws;
                bool both = true;
                if constexpr (VEC) {
                    if (P.xtab_given) {  // the LM head wrote the draft's statistics
                        stream_target_tables<T>(rg, P.target + (int64_t)j.r * V, V, j.c0, j.c1,
                                                rtab, P.ts.c, policy_evict_first(), P.status);
                        both = false;
                    }
                }
                if (both)  // (with no gradient jobs the draft row is read once)
                    stream_tables<T, VEC, true>(rg, x, P.target + (int64_t)j.r * V, V, j.c0,
                                                j.c1, rtab, P.ts.c,
                                                P.gnseg ? policy_evict_last() : policy_evict_first(),
                                                policy_evict_first(), P.status);
                if (P.stream_tails) {  // short rows: the tail here, three draws at once
                    asm volatile("bar.sync %0, %1;" ::"r"(kStreamBar), "r"(kThreads) : "memory");
                    row_tail<T, VEC, true, kSampleToken, true, kStreamBar, KL>(
                        P, j.r, rtab, rsh, VEC ? &rg->data[kWarps - 1][0][0][0] : nullptr);
                }
            } else if (j.kind == kJobResidual) {
                // row A's table was consumed by its row tail: reuse it
                stream_residual<T, VEC>(rg, x, P.target + (int64_t)j.r * V, V, j.c0, j.c1,
                                        P.gtab + (int64_t)j.r * P.nch_ws, j.mr, P.status);
            } else {
                stream_grad<T, VEC, G, KL>(rg, P, j.r, j.c0, j.c1, grad, KL ? &kslot[s] : nullptr);
            }
            __syncwarp();
            named_arrive(bar_done(s));
        }
        return;
    }
    // ------------------------------------------------------------ control warp
    const EStepView E{P.es.tok, P.es.corr, P.es.lq_tok, P.es.lq_corr,
                      P.es.lk, P.es.lkc, P.es.lkr};
    int g = *(volatile int*)P.grad_head;
    int head = 0, tail = 0, inflight = 0;
    bool ended = false;
    __shared__ Job cur;
    // Fill the free slots.  A claim may wait only when no job is in flight
    // (then no follow-up step is owed either).
    auto fill = [&]() {
        while (!ended && inflight < kSlots) {
            int got = 0;
            if (lane == 0) got = claim_job<T>(P, inflight == 0, g, slots[tail % kSlots]) ? 1 : 0;
            got = __shfl_sync(0xffffffffu, got, 0);
            if (!got) break;
            __syncwarp();
            const int kind = slots[tail % kSlots].kind;
            if (KL && kind == kJobGrad) {  // the row's top-K terms for the streaming warps
                const int4* src = reinterpret_cast<const int4*>(P.klr + slots[tail % kSlots].r);
                if (lane < (int)(sizeof(KlRec) / 16))
                    reinterpret_cast<int4*>(&kslot[tail % kSlots])[lane] = __ldcg(src + lane);
                __syncwarp();
            }
            named_arrive(bar_full(tail % kSlots));
            ++tail;
            if (kind == kJobEnd) {
                ended = true;
                break;
            }
            ++inflight;
        }
    };
    for (;;) {
        fill();
        if (inflight == 0) break;
        const int s = head % kSlots;
        named_sync(bar_done(s));
        if (lane == 0) cur = slots[s];
        __syncwarp();
        ++head;
        --inflight;
        if (cur.kind != kJobGrad) post_job<T, VEC, KL>(P, E, cur, tab, cs, lane);
        __syncwarp();
    }
}

// ------------------------------------------------------------ fused tree kernel
// Tree verification in one launch of plain 128-thread blocks, R + tail
// blocks.  Each block first takes a ticket: a ticket below R is a node row
// (its tables and p-draw, then its children's acceptance; a leaf's row is
// skipped unless row statistics are requested); the block completing a
// tree's last row runs the per-node pass for that tree (its shared memory is
// the idle ring), queues the tree's residual rows and, when the bonus token
// needs the row of a leaf that was skipped, runs that row's pass itself as
// one more of the tree's items.  After its row a block takes queued residual
// rows (the rejected children's draws) while any are ready; the block
// completing a tree's last item writes its bonus token.  A block whose
// ticket is R or more was started after every row had
// been claimed, so every job it may wait for is held by a running block: it
// waits for residual rows (bounded, status bit on expiry) until every tree is
// done.
template <typename T>
__device__ int claim_residual(const Problem<T>& P, bool wait) {
    uint64_t idle_since = 0;
    for (;;) {
        const int it = *(volatile int*)P.resq_avail > 0
                           ? take_residual(P.resq_head, P.resq_avail, P.resq_flag, P.resq,
                                           P.status, P.timeout_ns)
                           : -1;
        if (it >= 0) return it;
        if (it == -2) return -1;
        if (!wait) return -1;
        if (*(volatile int*)P.prefix_done >= P.B) return -1;
        if (*(volatile int*)P.status & VSD_STATUS_TIMEOUT) return -1;
        const uint64_t now = global_timer_ns();
        if (idle_since == 0) {
            idle_since = now;
        } else if (now - idle_since > P.timeout_ns) {
            atomicOr(P.status, VSD_STATUS_TIMEOUT);
            return -1;
        }
        __nanosleep(1000);
    }
}

template <typename T, bool VEC>
__global__ void __launch_bounds__(kThreads) k_tree_fused(Problem<T> P) {
    extern __shared__ __align__(128) unsigned char dsm[];
    __shared__ RowShared sh;
    __shared__ int s_t, s_last, s_tok, s_cnt, s_leaf;
    Ring* rg;
    float4* tab;
    smem_views<VEC>(dsm, rg, tab, P.timeout_ns);
    // The per-node pass runs between streams: on the vector path its shared
    // memory is the ring's data (no copy is in flight then), else it follows
    // the chunk table.
    static_assert(sizeof(TreeShared) <= sizeof(Ring::data), "TreeShared fits the ring");
    TreeShared* tsh = VEC ? reinterpret_cast<TreeShared*>(rg->data)
                          : reinterpret_cast<TreeShared*>(tab + P.nch);
    const int N = P.N;
    if (threadIdx.x == 0) s_t = atomicAdd(P.ticket, 1);
    __syncthreads();
    const int t = s_t;
    if (t < P.R) {
        const int b = t / N, u = t - b * N;
        // A leaf's row is needed only for the bonus token (taken later if at
        // all) and for the row statistics output.
        int need = P.tout.row_stats != nullptr;
        for (int n = u + 1 + threadIdx.x; n < N && !need; n += kThreads)
            need = __ldg(P.parent + (int64_t)b * N + n) == u;
        if (__syncthreads_or(need)) {
            row_pass<T, VEC, true, kNoToken, false>(P, t, rg, tab, sh);
            __syncthreads();
            tree_children<T>(P, b, u);
            __syncthreads();
        }
        if (threadIdx.x == 0) {
            __threadfence();
            s_last = atomicAdd(P.path_cnt + b, 1) == N - 1;
            if (s_last) __threadfence();
        }
        __syncthreads();
        if (s_last) {
            tree_nodes<T>(P, b, *tsh);
            __syncthreads();
            if (threadIdx.x == 0) {
                const int cnt = ld_cg(P.tcount + b);
                const int best = ld_cg(P.tout.deepest + b);
                const int child = best >= 0 ? ld_cg(P.tlist + b * N + N - 1) : 0;
                // a leaf's row not read yet that the bonus token needs
                const int leaf = (best >= 0 && child < 0 && !P.tout.row_stats) ? b * N + best : -1;
                s_cnt = cnt;
                s_leaf = leaf;
                if (cnt > 0) {  // queue the tree's residual rows (list positions)
                    // the leaf's row pass here counts as one more of the tree's items
                    if (leaf >= 0) atomicSub(P.res_seg_cnt + b, 1);
                    publish_residuals(P.resq_tail, P.resq_avail, P.resq_flag, P.resq, b * N,
                                      cnt, true);
                }
            }
            __syncthreads();
            const int cnt = s_cnt, leaf = s_leaf;
            if (leaf >= 0) {  // while other blocks take the residual rows
                row_pass<T, VEC, true, kNoToken, false>(P, leaf, rg, tab, sh);
                __syncthreads();
            }
            if (threadIdx.x == 0) {
                bool done = cnt == 0;
                if (!done && leaf >= 0) {
                    __threadfence();
                    done = atomicAdd(P.res_seg_cnt + b, 1) == cnt - 1;
                }
                if (done) {
                    __threadfence();
                    tree_bonus<T>(P, b);
                    __threadfence();
                    atomicAdd(P.prefix_done, 1);
                }
            }
            __syncthreads();
        }
    }
    const bool wait = t >= P.R;
    for (;;) {
        if (threadIdx.x == 0) s_t = claim_residual<T>(P, wait);
        __syncthreads();
        const int item = s_t;
        if (item < 0) break;
        const int b = item / N;
        tree_residual_row<T, VEC>(P, b, ld_cg(P.tlist + item), rg, tab, &s_tok);
        if (threadIdx.x == 0) {
            __threadfence();
            if (atomicAdd(P.res_seg_cnt + b, 1) == ld_cg(P.tcount + b) - 1) {
                __threadfence();
                tree_bonus<T>(P, b);
                __threadfence();
                atomicAdd(P.prefix_done, 1);
            }
        }
        __syncthreads();
    }
}

// ------------------------------------------------------------ launchers
// Static plus dynamic shared memory above 48 KB needs the kernel's opt-in
// (made once per kernel and device).
template <typename K>
static cudaError_t prep(K kernel, size_t smem) {
    return ensure_dyn_smem(reinterpret_cast<const void*>(kernel), smem);
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
cudaError_t Launch<VSD_T>::rows_verify(const Problem<VSD_T>& P, bool vec, cudaStream_t s) {
    const size_t smem = stream_smem_bytes(P.nch, vec);
    auto kern = vec ? k_rows_verify<VSD_T, true> : k_rows_verify<VSD_T, false>;
    cudaError_t e = prep(kern, smem);
    if (e) return e;
    kern<<<P.R, kThreads, smem, s>>>(P);
    return cudaGetLastError();
}

template <>
cudaError_t Launch<VSD_T>::reference(const Problem<VSD_T>& P, bool vec, float* out,
                                     cudaStream_t s) {
    const size_t smem = stream_smem_bytes(P.nch, vec);
    auto kern = vec ? k_ref_rows<VSD_T, true> : k_ref_rows<VSD_T, false>;
    cudaError_t e = prep(kern, smem);
    if (e) return e;
    kern<<<P.R, kThreads, smem, s>>>(P);
    e = cudaGetLastError();
    if (e) return e;
    k_ref_scan<VSD_T><<<P.B, 32, 0, s>>>(P, out);
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

#ifndef VSD_TREE_TAIL_PER_SM
#define VSD_TREE_TAIL_PER_SM 1
#endif
template <>
cudaError_t Launch<VSD_T>::tree(const Problem<VSD_T>& P, bool vec, cudaStream_t s) {
    // one block per node row, then tail blocks for the last trees' residual rows
    const size_t smem = stream_smem_bytes(P.nch, vec) + (vec ? 0 : sizeof(TreeShared));
    auto kern = vec ? k_tree_fused<VSD_T, true> : k_tree_fused<VSD_T, false>;
    cudaError_t e = prep(kern, smem);
    if (e) return e;
    long long tail = (long long)device_sm_count() * VSD_TREE_TAIL_PER_SM;
    const long long most = (long long)P.B * (P.N - 1);  // residual rows at most
    if (tail > most) tail = most;
    if (tail < 1) tail = 1;
    kern<<<(unsigned)(P.R + tail), kThreads, smem, s>>>(P);
    return cudaGetLastError();
}

template <>
cudaError_t Launch<VSD_T>::tree_seq(const Problem<VSD_T>& P, bool vec, cudaStream_t s) {
    const size_t smem = stream_smem_bytes(P.nch, vec);
    auto rows = vec ? k_tree_rows<VSD_T, true, false> : k_tree_rows<VSD_T, false, false>;
    cudaError_t e = prep(rows, smem);
    if (e) return e;
    rows<<<P.R, kThreads, smem, s>>>(P);
    if ((e = cudaGetLastError())) return e;
    const size_t sm2 = sizeof(TreeSeqShared) + table_smem_bytes(P.nch);
    auto seq = vec ? k_tree_seq<VSD_T, true> : k_tree_seq<VSD_T, false>;
    if ((e = prep(seq, sm2))) return e;
    seq<<<P.B, kThreads, sm2, s>>>(P);
    return cudaGetLastError();
}

template <>
cudaError_t Launch<VSD_T>::tree_em(const Problem<VSD_T>& P, bool vec,
                                   const vsd_tree_em_outputs& o, void* grad, bool grad_bf16,
                                   cudaStream_t s) {
    const size_t smem = stream_smem_bytes(P.nch, vec);
    auto rows = vec ? k_tree_rows<VSD_T, true, true> : k_tree_rows<VSD_T, false, true>;
    cudaError_t e = prep(rows, smem);
    if (e) return e;
    rows<<<P.R, kThreads, smem, s>>>(P);
    if ((e = cudaGetLastError())) return e;
    if ((e = prep(k_tree_em<VSD_T>, sizeof(TreeEmShared)))) return e;
    k_tree_em<VSD_T><<<P.B, kThreads, sizeof(TreeEmShared), s>>>(P, o);
    if ((e = cudaGetLastError())) return e;
#define VSD_TGRAD(V_, G_) \
    k_tree_grad<VSD_T, V_, G_><<<P.R, kThreads, 0, s>>>(P, reinterpret_cast<G_*>(grad))
    if (vec && grad_bf16) VSD_TGRAD(true, __nv_bfloat16);
    else if (vec) VSD_TGRAD(true, float);
    else if (grad_bf16) VSD_TGRAD(false, __nv_bfloat16);
    else VSD_TGRAD(false, float);
#undef VSD_TGRAD
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
    const bool kl = P.kl_topk != 0;
#define VSD_FUSED(V_, G_, KL_)                                                         \
    do {                                                                               \
        cudaError_t e = prep(k_fused<VSD_T, V_, G_, KL_>, smem);                       \
        if (e) return e;                                                               \
        k_fused<VSD_T, V_, G_, KL_><<<ctas, kFusedThreads, smem, s>>>(                 \
            P, reinterpret_cast<G_*>(grad));                                           \
    } while (0)
#define VSD_FUSED_KL(V_, G_)                 \
    do {                                     \
        if (kl) VSD_FUSED(V_, G_, true);     \
        else VSD_FUSED(V_, G_, false);       \
    } while (0)
    if (vec && grad_bf16) VSD_FUSED_KL(true, __nv_bfloat16);
    else if (vec) VSD_FUSED_KL(true, float);
    else if (grad_bf16) VSD_FUSED_KL(false, __nv_bfloat16);
    else VSD_FUSED_KL(false, float);
#undef VSD_FUSED_KL
#undef VSD_FUSED
    return cudaGetLastError();
}

template <>
int Launch<VSD_T>::fused_blocks_per_sm(const Problem<VSD_T>& P, bool vec, bool grad_bf16) {
    const size_t smem = stream_smem_bytes(P.nch, vec);
    const bool kl = P.kl_topk != 0;
#define VSD_K(V_, G_) (kl ? reinterpret_cast<const void*>(k_fused<VSD_T, V_, G_, true>) \
                          : reinterpret_cast<const void*>(k_fused<VSD_T, V_, G_, false>))
    const void* k = vec ? (grad_bf16 ? VSD_K(true, __nv_bfloat16) : VSD_K(true, float))
                        : (grad_bf16 ? VSD_K(false, __nv_bfloat16) : VSD_K(false, float));
#undef VSD_K
    const int n = blocks_per_sm(k, kFusedThreads, smem);
    return n < 1 ? 1 : n;
}

template struct Launch<VSD_T>;

}  // namespace vsd
