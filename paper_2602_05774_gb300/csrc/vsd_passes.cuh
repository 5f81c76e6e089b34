// vsd_passes.cuh -- block-level passes of the VSD E-step / M-step (arxiv
// 2602.05774) on sm_103a.  Each pass is a __device__ function run by one block
// of kThreads threads; the separate-kernel entry points and the fused
// persistent kernel call the same functions.
//
//   row_pass     one streaming read of a draft row (and its target row):
//                per-chunk (max, sum-exp) tables in shared memory, the row's
//                log-partitions, inverse-CDF draws from q (z~, Algorithm 1) and
//                from p (used after the first rejection), the target argmax
//                (greedy reference of Algorithm 2), and the log-probabilities
//                of those tokens (Eq. 1 needs p and q at a token).
//   path_pass    per proposal path: acceptance (Eq. 1), accepted length,
//                survival/expected length (Eqs. 9-11), the residual draw
//                norm(max(0, p - q)) at the first rejection (Sec. 3; one more
//                streaming read of that row), the corrected path z', and the
//                log-kappa prefix sums (Eq. 2) of z~, z' and the reference.
//   weights_pass per prefix: o~, o' (Algorithm 2 with w(l) = w_base^l), beta
//                (Eq. beta), zeta (Eq. zeta), N_b, loss_b (Eq. advance), and
//                the per-row gradient coefficients.
//   grad_pass    one streaming read of a draft row and write of its gradient:
//                grad[v] = g q(v) - c0 [v = t0] - c1 [v = t1].
//   tree_nodes / tree_residual_row / tree_bonus   per draft tree: acceptance
//                per node at its parent's row, the AND-scan along parent
//                pointers, log kappa, the deepest node; the residual draws at
//                each accepted parent of rejected nodes (one block per such
//                row); the bonus token.
#pragma once

#include "vsd_common.cuh"

namespace vsd {

// --------------------------------------------------------------- records
struct __align__(16) RowRec {  // one logit row after row_pass (workspace)
    double lzx, lzy;         // ln sum_v exp((v - max)/T) of the q and p rows
    float mx, my;            // row maxima (exact input values)
    float izx, izy;          // 1 / sum_v exp((v - max)/T) in float (0 if the row is invalid)
    int tok;                 // z~ (drawn from q, or given); -1 if none
    float lq_tok, la_tok;    // log q(z~), log alpha(z~) = min(0, log p - log q)
    int ps;                  // draw from p with u_correct
    float lq_ps, la_ps;
    int ref;                 // argmax of the target row
    float la_ref;
    int flags;               // 1: invalid row, 2: invalid given token
    int pad[3];
};
static_assert(sizeof(RowRec) == 80, "RowRec layout");

struct __align__(16) Coef {     // grad[v] = g q(v) - c0 [v == t0] - c1 [v == t1]
    float g;
    int t0;
    float c0;
    int t1;
    float c1;
    float pad0, pad1, pad2;
};
static_assert(sizeof(Coef) == 32, "Coef layout");

// VSD (KL), Eq. klv: the top-K renormalised cross-entropy of one row and its
// gradient, which touches only the K selected tokens.
constexpr int kMaxKlTop = 16;
struct __align__(16) KlRec {
    int tok[kMaxKlTop];     // the K tokens of highest target probability (lowest index on ties)
    float coef[kMaxKlTop];  // their gradient terms, kl_weight / (B K T) (q^ - p^)
    float loss;             // L_topK of the row
    int n;                  // entries used (0: the row has no term)
    int pad[2];
};
static_assert(sizeof(KlRec) == 144, "KlRec layout");

// Coherent loads of records written by other blocks of the same grid.
template <typename U>
__device__ __forceinline__ U ld_cg_rec(const U* p) {
    static_assert(sizeof(U) % 16 == 0, "record size");
    U r;
    const int4* src = reinterpret_cast<const int4*>(p);
    int4* dst = reinterpret_cast<int4*>(&r);
#pragma unroll
    for (int i = 0; i < (int)(sizeof(U) / 16); ++i) dst[i] = __ldcg(src + i);
    return r;
}
__device__ __forceinline__ RowRec ld_cg(const RowRec* p) { return ld_cg_rec(p); }
__device__ __forceinline__ KlRec ld_cg(const KlRec* p) { return ld_cg_rec(p); }
__device__ __forceinline__ Coef ld_cg(const Coef* p) { return ld_cg_rec(p); }

// E-step results the M-step reads (structure of arrays, [R] each).
struct EStepView {
    const int32_t* tok;      // z~
    const int32_t* corr;     // z'
    const float* lq_tok;     // log q(z~_d)
    const float* lq_corr;    // log q(z'_d)
    const float* lk;         // log kappa(z~_{<=l})
    const float* lkc;        // log kappa(z'_{<=l})
    const float* lkr;        // log kappa(z-bar_{<=l})
};

struct EStepStore {          // same arrays, writable (workspace copy)
    int32_t* tok;
    int32_t* corr;
    float* lq_tok;
    float* lq_corr;
    float* lk;
    float* lkc;
    float* lkr;
};

template <typename T>
struct Problem {
    const T* draft;
    const T* target;
    int B, K, D, N;          // N: nodes per tree (tree layout)
    int64_t V;
    int R;                   // rows
    int nch;                 // chunks per row
    TempScale ts;
    const float* u_draft;
    const float* u_accept;
    const float* u_correct;
    const float* ref_logkappa;    // [B][D] or null
    const int32_t* given_tokens;  // [R] or null (draft sampling)
    const int32_t* parent;        // tree [B][N]
    double w_base, tau_car;
    double wl[64];  // w(l) = w_base^l for l = 1 .. D (App. F), computed on the host
    float wlf[64];  // the same in float
    double inv_tau;  // 1 / tau_car
    float inv_tau_f;
    int zeta_mode;
    int kl_topk;                  // VSD (KL): K of Eq. klv, 0 = no top-K term
    double kl_weight;             // its weight in the loss
    double kl_scale;              // kl_weight / (B K T), the gradient factor
    KlRec* klr;                   // [R] the rows' terms
    int grad_bf16;
    int inject_wait_fault;
    uint64_t timeout_ns;
    // workspace
    int* status;
    int* ticket;
    int* prefix_done;
    int* path_cnt;                // [B*K]
    int* prefix_cnt;              // [B]
    int* ready;                   // [B]
    int* grad_cnt;                // [B] gradient rows claimed per prefix
    int* grad_head;               // oldest prefix that may have unclaimed gradient rows
    RowRec* rows;                 // [R]
    float4* rstats;               // [R] m_q, logZ_q, m_p, logZ_p (float copy of rows[])
    EStepStore es;                // [R] each
    Coef* coef;                   // [R]
    double2* wscr;                // [R] M-step scratch
    // fused kernel: rows, residual rows and gradient rows are split into
    // segments of segc chunks (nseg per row)
    int segc, nseg, nch_ws;       // nch_ws: row stride of gtab (>= nch)
    int gsegc, gnseg;             // gradient jobs: chunks per segment, segments per row
    float4* gtab;                 // [R][nch_ws] per-chunk tables of each row
    int* row_seg_cnt;             // [R] segments of a row completed
    int* res_seg_cnt;             // [B*K] residual segments of a path completed
    int stream_tails;             // fused kernel: the streaming warps run the row tails
    int greedy;                   // T = 0: every decision takes the argmax limit of
                                  // Eq. 1's distributions; ts holds temperature 1,
                                  // the M-step's
    int xtab_given;               // fused kernel: gtab[r][ch].xy (the draft's chunk
                                  // statistics) were written by the LM head's epilogue
    int* path_A;                  // [B*K] accepted length of a path
    struct TreeNodeRec* tnode;    // trees beyond independent verification: [R] node records
    struct TreeCoef* tcoef;       // [R] each node's gradient terms at its parent's row
    float* tg;                    // [R] each row's dense gradient factor
    int* tbad;                    // [B] the tree failed its checks
    int* tlist;                   // tree layout: [R] residual rows of each tree (its rows' slots)
    int* tcount;                  // tree layout: [B] length of each tree's list
    float* tla;                   // tree layout: [R] log alpha of each node's token
    int* resq;                    // [B*K*nseg] residual segment items (path*nseg + seg);
                                  // trees: [B*N] positions b*N + i in the residual list
    int* resq_flag;               // item written
    int* resq_head;               // next item to take
    int* resq_tail;               // next free slot
    int* resq_avail;              // items published and not yet reserved (may dip below 0)
    int resq_sem;                 // fused kernel claims residual items through resq_avail
    // outputs (device, caller-owned; null = not written)
    vsd_linear_outputs out;
    vsd_tree_outputs tout;
};

// --------------------------------------------------------------- masses
// exp((v - m)/T) for a chunk-relative frame m; a frame of -inf (chunk of -inf
// logits) is replaced by 0 so that the masses are exactly 0, not NaN.
__device__ __forceinline__ float frame_of(float m) { return m == -INFINITY ? 0.f : m; }
__device__ __forceinline__ float mass_rel(float f, float mm, float c) { return ex2((f - mm) * c); }

// Chunk statistics of one tensor: (max, sum_v 2^{(v - max) c}) over the warp's chunk.
template <typename T>
__device__ __forceinline__ float2 chunk_stats(const uint4 (&buf)[kLoads], float c) {
    constexpr int NP = Traits<T>::kPerVec / 2;
    const float m = warp_max(lane_max<T>(buf));
    const float mm = frame_of(m);
    const uint64_t mm2 = f2(mm, mm), c2 = f2(c, c);
    uint64_t acc0 = f2(0.f, 0.f), acc1 = acc0;
#pragma unroll
    for (int k = 0; k < kLoads; ++k) {
        uint64_t pr[NP];
        vec_pairs<T>(buf[k], pr);
#pragma unroll
        for (int i = 0; i < NP; ++i) {
            const uint64_t e2 = f2_mass(pr[i], mm2, c2);
            if (i & 1) acc1 = f2add(acc1, e2);
            else acc0 = f2add(acc0, e2);
        }
    }
    float lo, hi;
    f2split(f2add(acc0, acc1), lo, hi);
    return make_float2(m, warp_sum(lo + hi));
}

// --------------------------------------------------------------- TMA ring
// Every warp owns kStages slots, each holding one chunk of the draft row and
// one of the target row.  The warp's lane 0 issues 1-D bulk copies (TMA) up
// to kStages chunks ahead; all lanes wait on the slot's mbarrier, read their
// own vectors, and the slot is refilled once the warp has read it.  Each warp
// produces and consumes its own slots, so no block-wide synchronisation is
// involved.  A stream of one row only (no target) uses the same memory as
// 2 kStages single-chunk slots, so it keeps as many bytes in flight.  Each
// layout has its own barriers and its own count of consumed chunks (pos2 for
// two rows, pos1 for one; slot = pos % stages, phase = (pos / stages) & 1),
// which persist across calls; a call consumes every chunk it issues, so the
// two layouts never hold a buffer at the same time.
struct Ring {
    uint4 data[kWarps][kStages][2][kLoads * 32];
    uint64_t bar2[kWarps][kStages];
    uint64_t bar1[kWarps][2 * kStages];
    int pos2[kWarps];
    int pos1[kWarps];
    int broken[kWarps];  // a wait ran out: no further waits or copies in this block
    uint64_t timeout_ns; // bound of every slot wait (the call's wait timeout)
};

// Every thread of the block calls it; warps beyond the streaming warps (the
// fused kernel's control warp) own no ring slots.
__device__ __forceinline__ void ring_init(Ring* rg, uint64_t timeout_ns) {
    if (threadIdx.x == 0) rg->timeout_ns = timeout_ns;
    if ((threadIdx.x & 31) == 0 && (threadIdx.x >> 5) < kWarps) {
        const int w = threadIdx.x >> 5;
        for (int st = 0; st < kStages; ++st) mbar_init(&rg->bar2[w][st], 1);
        for (int st = 0; st < 2 * kStages; ++st) mbar_init(&rg->bar1[w][st], 1);
        rg->pos2[w] = 0;
        rg->pos1[w] = 0;
        rg->broken[w] = 0;
        mbar_init_fence();
    }
    __syncthreads();
}

// Bounded wait on a slot; false (and the timeout status bit) if it ran out.
__device__ __forceinline__ bool ring_wait(uint64_t* bar, uint32_t parity, int* status,
                                          uint64_t timeout_ns) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    for (;;) {
        if (mbar_try_wait(bar, parity)) return true;
        if (global_timer_ns() - t0 > timeout_ns) {
            atomicOr(status, VSD_STATUS_TIMEOUT);
            return false;
        }
    }
}

// Warp-level stream of this warp's chunks (ch0 + warp, ch0 + warp + kWarps,
// ... < ch1) of row x (and y) through the ring; consume(ch, bx, by) gets each
// chunk in registers (positions at or beyond V read as -inf).  Rows must be
// 16-byte aligned with V * sizeof(T) a multiple of 16.
template <typename T, bool HAS_Y, class Consume>
__device__ __forceinline__ void ring_stream(Ring* rg, const T* x, const T* y, int64_t V, int ch0,
                                            int ch1, uint64_t polx, uint64_t poly, int* status,
                                            Consume&& consume) {
    constexpr int PV = Traits<T>::kPerVec;
    constexpr int CE = chunk_elems<T>();
    constexpr int NS = HAS_Y ? kStages : 2 * kStages;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    uint64_t* bars = HAS_Y ? rg->bar2[warp] : rg->bar1[warp];
    int* posp = HAS_Y ? &rg->pos2[warp] : &rg->pos1[warp];
    // slot q: the x and y halves of stage q (two rows), or half q & 1 of
    // stage q >> 1 (one row)
    auto xbuf = [&](int q) -> uint4* {
        return HAS_Y ? rg->data[warp][q][0] : rg->data[warp][q >> 1][q & 1];
    };
    const int nrange = ch1 - ch0;
    const int nj = nrange > warp ? (nrange - warp + kWarps - 1) / kWarps : 0;
    const int cfirst = ch0 + warp, cstride = kWarps;
    const int pos = *posp;
    bool broken = rg->broken[warp] != 0;
    const uint64_t timeout_ns = rg->timeout_ns;
    auto issue = [&](int j) {
        const int ch = cfirst + j * cstride;
        const int slot = (pos + j) % NS;
        const int64_t e0 = (int64_t)ch * CE;
        const int64_t ne = V - e0 < CE ? V - e0 : CE;
        const uint32_t bytes = (uint32_t)(ne * (int64_t)sizeof(T));
        uint64_t* bar = &bars[slot];
        fence_proxy_async();
        mbar_expect_tx(bar, HAS_Y ? 2 * bytes : bytes);
        bulk_g2s(xbuf(slot), x + e0, bytes, bar, polx);
        if (HAS_Y) bulk_g2s(rg->data[warp][slot][1], y + e0, bytes, bar, poly);
    };
    if (lane == 0)
        for (int j = 0; j < nj && j < NS; ++j) issue(j);
    for (int j = 0; j < nj; ++j) {
        const int slot = (pos + j) % NS;
        const uint32_t parity = (uint32_t)((pos + j) / NS) & 1u;
        bool ok = broken ? false : ring_wait(&bars[slot], parity, status, timeout_ns);
        broken = __any_sync(0xffffffffu, !ok);
        const int ch = cfirst + j * cstride;
        const int64_t e0 = (int64_t)ch * CE;
        const uint4* sx = xbuf(slot);
        uint4 bx[kLoads], by[kLoads];
        if (e0 + CE <= V) {  // full chunk (all but possibly the row's last)
#pragma unroll
            for (int k = 0; k < kLoads; ++k) {
                bx[k] = sx[k * 32 + lane];
                if (HAS_Y) by[k] = rg->data[warp][slot][1][k * 32 + lane];
            }
        } else {
#pragma unroll
            for (int k = 0; k < kLoads; ++k) {
                const bool in = e0 + (int64_t)k * 32 * PV + lane * PV < V;
                const uint4 ninf = make_uint4(Traits<T>::kNegInf, Traits<T>::kNegInf,
                                              Traits<T>::kNegInf, Traits<T>::kNegInf);
                bx[k] = in ? sx[k * 32 + lane] : ninf;
                if (HAS_Y) by[k] = in ? rg->data[warp][slot][1][k * 32 + lane] : ninf;
            }
        }
        __syncwarp();
        if (lane == 0 && !broken && j + NS < nj) issue(j + NS);
        consume(ch, bx, by);
    }
    __syncwarp();
    if (lane == 0) {
        *posp = pos + nj;
        rg->broken[warp] = broken ? 1 : 0;
    }
    __syncwarp();
}

// Stream chunks [ch0, ch1) of a row (and optionally its target row) once,
// filling tab[c] = (max_x, sum_x, max_y, sum_y) for each chunk c (tab is a
// shared-memory table or a row's table in global memory).  Warps take chunks
// round-robin and keep the next chunks' loads in flight.
template <typename T, bool VEC, bool HAS_Y>
__device__ __forceinline__ void stream_tables(Ring* rg, const T* x, const T* y, int64_t V, int ch0,
                                              int ch1, float4* tab, float c, uint64_t polx,
                                              uint64_t poly, int* status) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if constexpr (VEC) {
        ring_stream<T, HAS_Y>(rg, x, y, V, ch0, ch1, polx, poly, status,
                              [&](int ch, const uint4 (&bx)[kLoads], const uint4 (&by)[kLoads]) {
                                  const float2 sx = chunk_stats<T>(bx, c);
                                  float2 sy = make_float2(0.f, 0.f);
                                  if (HAS_Y) sy = chunk_stats<T>(by, c);
                                  if (lane == 0) tab[ch] = make_float4(sx.x, sx.y, sy.x, sy.y);
                              });
        return;
    }
    int ch = ch0 + warp;
    uint4 bx[kLoads], by[kLoads];
    if (ch < ch1) {
        load_chunk<T, VEC>(x, V, ch, lane, polx, bx);
        if (HAS_Y) load_chunk<T, VEC>(y, V, ch, lane, poly, by);
    }
    while (ch < ch1) {
        const int cn = ch + kWarps;
        uint4 nx[kLoads], ny[kLoads];
        if (cn < ch1) {
            load_chunk<T, VEC>(x, V, cn, lane, polx, nx);
            if (HAS_Y) load_chunk<T, VEC>(y, V, cn, lane, poly, ny);
        }
        const float2 sx = chunk_stats<T>(bx, c);
        float2 sy = make_float2(0.f, 0.f);
        if (HAS_Y) sy = chunk_stats<T>(by, c);
        if (lane == 0) tab[ch] = make_float4(sx.x, sx.y, sy.x, sy.y);
#pragma unroll
        for (int k = 0; k < kLoads; ++k) {
            bx[k] = nx[k];
            if (HAS_Y) by[k] = ny[k];
        }
        ch = cn;
    }
}

// The target half of a row's chunk table when the draft half is given (the LM
// head's epilogue wrote it): tab[ch].zw = (max, sum) of target chunk ch, for
// ch in [ch0, ch1), one streaming read of the target row through the ring.
template <typename T>
__device__ __forceinline__ void stream_target_tables(Ring* rg, const T* y, int64_t V, int ch0,
                                                     int ch1, float4* tab, float c, uint64_t pol,
                                                     int* status) {
    const int lane = threadIdx.x & 31;
    ring_stream<T, false>(rg, y, nullptr, V, ch0, ch1, pol, pol, status,
                          [&](int ch, const uint4 (&by)[kLoads], const uint4 (&)[kLoads]) {
                              const float2 sy = chunk_stats<T>(by, c);
                              if (lane == 0) reinterpret_cast<float2*>(tab + ch)[1] = sy;
                          });
}

__device__ __forceinline__ float2 tab_ms(const float4& t, int comp) {
    return comp == 0 ? make_float2(t.x, t.y) : make_float2(t.z, t.w);
}

// Row max over the table (warp).
__device__ __forceinline__ float table_max(const float4* tab, int nch, int comp, int lane) {
    float M = -INFINITY;
    for (int ch = lane; ch < nch; ch += 32) M = fmaxf(M, tab_ms(tab[ch], comp).x);
    return warp_max(M);
}

// --------------------------------------------------------------- table sums
// The weight of chunk c in the row frame Mm is w_c = s_c 2^{(m_c - Mm) c}.
// Tables are summed in exact 64-bit fixed point, w_c 2^E rounded down, with E
// set from the largest weight so that it keeps at least 50 significant bits
// and no sum of up to 2048 weights overflows.  Integer sums are exact and do
// not depend on their order, so a total and the prefix sums that search it
// agree, and none of it runs on the slow FP64 pipe.

__device__ __forceinline__ float chunk_scale(const float4* tab, int ch, int comp, float Mm,
                                             float c) {
    return ex2((frame_of(tab_ms(tab[ch], comp).x) - Mm) * c);
}

// floor(s sc 2^E) for finite s, sc >= 0, by integer arithmetic on the two
// 24-bit significands.
__device__ __forceinline__ long long fixed_prod(float s, float sc, int E) {
    if (!(s > 0.f) || !(sc > 0.f)) return 0;
    const unsigned bs = __float_as_uint(s), bc = __float_as_uint(sc);
    const int xs = (bs >> 23) & 0xFF, xc = (bc >> 23) & 0xFF;
    const unsigned long long ms = xs ? ((bs & 0x7FFFFFu) | 0x800000u) : (bs & 0x7FFFFFu);
    const unsigned long long mc = xc ? ((bc & 0x7FFFFFu) | 0x800000u) : (bc & 0x7FFFFFu);
    const int sh = (xs ? xs : 1) + (xc ? xc : 1) - 300 + E;  // s sc 2^E = ms mc 2^sh
    const unsigned long long pm = ms * mc;                   // < 2^48
    if (sh >= 0) return (long long)(pm << min(sh, 15));
    return sh > -64 ? (long long)(pm >> -sh) : 0;
}

// floor(u Zi) for Zi >= 0 (exact, 128-bit product); u >= 1 or NaN gives Zi
// (no chunk is crossed), u <= 0 gives 0.
__device__ __forceinline__ long long fixed_scale(long long Zi, float u) {
    if (!(u < 1.f)) return Zi;
    if (!(u > 0.f)) return 0;
    const unsigned bu = __float_as_uint(u);
    const int xu = (bu >> 23) & 0xFF;
    const unsigned long long mu = xu ? ((bu & 0x7FFFFFu) | 0x800000u) : (bu & 0x7FFFFFu);
    const int k = 150 - (xu ? xu : 1);  // u = mu 2^-k, k >= 24
    const unsigned long long Z = (unsigned long long)Zi;
    const unsigned long long lo = Z * mu, hi = __umul64hi(Z, mu);
    if (k >= 128) return 0;
    if (k >= 64) return (long long)(hi >> (k - 64));
    return (long long)((hi << (64 - k)) | (lo >> k));
}

// 2^-E as a double (|E| <= 1000).
__device__ __forceinline__ double pow2_neg(int E) {
    return __longlong_as_double((long long)(1023 - E) << 52);
}

__device__ __forceinline__ long long warp_sum_ll(long long v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ long long warp_incl_scan_ll(long long v, int lane) {
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const long long n = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += n;
    }
    return v;
}

// Whether t sc 2^E <= num exactly, for finite t, sc >= 0 and num >= 0 (integer
// arithmetic on the two 24-bit significands).
__device__ __forceinline__ bool prod_le(float t, float sc, int E, long long num) {
    if (!(t > 0.f) || !(sc > 0.f)) return true;
    const unsigned bt = __float_as_uint(t), bc = __float_as_uint(sc);
    const int xt = (bt >> 23) & 0xFF, xc = (bc >> 23) & 0xFF;
    const unsigned long long mt = xt ? ((bt & 0x7FFFFFu) | 0x800000u) : (bt & 0x7FFFFFu);
    const unsigned long long mc = xc ? ((bc & 0x7FFFFFu) | 0x800000u) : (bc & 0x7FFFFFu);
    const unsigned long long pm = mt * mc;  // t sc 2^E = pm 2^sh
    const int sh = (xt ? xt : 1) + (xc ? xc : 1) - 300 + E;
    const unsigned long long n = (unsigned long long)num;
    if (sh >= 0) return sh < 64 && pm <= (n >> sh);
    const int k = -sh;
    if (k >= 64) return n >= 1;
    const unsigned long long q = pm >> k, r = pm & ((1ull << k) - 1ull);
    return q < n || (q == n && r == 0);
}

// The largest float t >= 0 with t sc <= num 2^-E (num >= 0, sc > 0): a float
// estimate, then exact tests one float step at a time.
__device__ __forceinline__ float fixed_quotient_rd(long long num, float sc, int E) {
    const float nf = (float)(int)(num >> 32) * 4294967296.f + (float)(unsigned)(num & 0xFFFFFFFFull);
    float t = ldexpf(nf, -E) / sc;
    if (!(t >= 0.f)) t = 0.f;
    if (t > 3.0e38f) t = 3.0e38f;
    for (int i = 0; i < 16 && !prod_le(t, sc, E, num); ++i) t = nextafterf(t, 0.f);
    for (int i = 0; i < 16; ++i) {
        const float up = nextafterf(t, INFINITY);
        if (!prod_le(up, sc, E, num)) break;
        t = up;
    }
    return t;
}

// A table total: Z = Zi 2^-E (NaN if a weight is not finite).
struct TableSum {
    long long Zi;
    int E;
    double Z;
};

// Sum of the chunk weights of one table component (warp).
__device__ __forceinline__ TableSum table_sum(const float4* tab, int nch, int comp, float Mm,
                                              float c, int lane) {
    float wm = 0.f;
    bool bad = false;
    for (int ch = lane; ch < nch; ch += 32) {
        const float w = tab_ms(tab[ch], comp).y * chunk_scale(tab, ch, comp, Mm, c);
        bad |= !(w < INFINITY) && !(w == 0.f);
        wm = fmaxf(wm, w);
    }
    bad = __any_sync(0xffffffffu, bad);
    wm = warp_max(wm);
    TableSum r{0, 0, 0.0};
    if (bad) {
        r.Z = __longlong_as_double(0x7FF8000000000000ll);  // NaN
        return r;
    }
    if (!(wm > 0.f)) return r;
    r.E = 50 - ilogbf(wm);
    long long acc = 0;
    for (int ch = lane; ch < nch; ch += 32)
        acc += fixed_prod(tab_ms(tab[ch], comp).y, chunk_scale(tab, ch, comp, Mm, c), r.E);
    r.Zi = warp_sum_ll(acc);
    r.Z = (double)r.Zi * pow2_neg(r.E);
    return r;
}

// Find the chunk where the running weight first exceeds ti = floor(u Zi).
// Returns the chunk and the threshold in that chunk's own frame, rounded down
// to a float (a float running mass exceeds the exact threshold if and only if
// it exceeds this float); if no chunk crosses, the last chunk with weight and
// an infinite threshold (the rescan then takes its last token with mass).
struct Located {
    int ch;
    float tc;
};
__device__ __forceinline__ Located table_locate(const float4* tab, int nch, int comp, float Mm,
                                                float c, const TableSum& S, float u, int lane) {
    const long long ti = fixed_scale(S.Zi, u);
    long long base = 0;
    int last = -1;
    for (int g = 0; g < nch; g += 32) {
        const int ch = g + lane;
        float sc = 1.f;
        long long w = 0;
        if (ch < nch) {
            sc = chunk_scale(tab, ch, comp, Mm, c);
            w = fixed_prod(tab_ms(tab[ch], comp).y, sc, S.E);
        }
        const long long inc = warp_incl_scan_ll(w, lane);
        const unsigned hit = __ballot_sync(0xffffffffu, ch < nch && base + inc > ti);
        const unsigned pos = __ballot_sync(0xffffffffu, ch < nch && w > 0);
        if (hit) {
            const int L = __ffs(hit) - 1;
            const long long before = __shfl_sync(0xffffffffu, base + inc - w, L);
            const float scL = __shfl_sync(0xffffffffu, sc, L);
            // the threshold in the chunk's frame, (ti - before) 2^-E / sc,
            // rounded down to a float
            return Located{g + L, fixed_quotient_rd(ti - before, scL, S.E)};
        }
        if (pos) last = g + 31 - __clz(pos);
        base += __shfl_sync(0xffffffffu, inc, 31);
    }
    return Located{last, INFINITY};
}

// Scan chunk ch (in registers: bx, by as load_chunk gives them) in token order
// and return the first token of positive mass whose running mass exceeds tc
// (the chunk-frame threshold); if none does, the last token with mass; -1 if
// the chunk has no mass.  Only tokens of positive mass can be returned, so
// masked positions (at or beyond V) never are.  mass(fx, fy) gives a token's
// mass.
template <typename T, bool NEED_X, bool NEED_Y, class Mass>
__device__ __forceinline__ int rescan_regs(const uint4 (&bx)[kLoads], const uint4 (&by)[kLoads],
                                           int ch, float tc, const Mass& mass, int lane) {
    constexpr int PV = Traits<T>::kPerVec;
    float carry = 0.f;
    int last = -1;
    const int64_t base = (int64_t)ch * chunk_elems<T>();
#pragma unroll
    for (int k = 0; k < kLoads; ++k) {
        float fx[PV], fy[PV], m[PV];
        if (NEED_X) unpack<T>(bx[k], fx);
        if (NEED_Y) unpack<T>(by[k], fy);
        float run = 0.f;
        int lastpos = -1;
#pragma unroll
        for (int e = 0; e < PV; ++e) {
            m[e] = mass(NEED_X ? fx[e] : 0.f, NEED_Y ? fy[e] : 0.f);
            run += m[e];
            if (m[e] > 0.f) lastpos = e;
        }
        const float incl = warp_incl_scan(run, lane);
        float excl = __shfl_up_sync(0xffffffffu, incl, 1);
        if (lane == 0) excl = 0.f;
        const float tot = __shfl_sync(0xffffffffu, incl, 31);
        int epos = -1;
        float acc = carry + excl;
#pragma unroll
        for (int e = 0; e < PV; ++e) {
            acc += m[e];
            if (epos < 0 && m[e] > 0.f && acc > tc) epos = e;
        }
        const unsigned hit = __ballot_sync(0xffffffffu, epos >= 0);
        if (hit) {
            const int L = __ffs(hit) - 1;
            const int e = __shfl_sync(0xffffffffu, epos, L);
            return (int)(base + (int64_t)k * 32 * PV + L * PV + e);
        }
        const unsigned pos = __ballot_sync(0xffffffffu, lastpos >= 0);
        if (pos) {
            const int L = 31 - __clz(pos);
            const int lp = __shfl_sync(0xffffffffu, lastpos, L);
            last = (int)(base + (int64_t)k * 32 * PV + L * PV + lp);
        }
        carry += tot;
    }
    return last;
}

// rescan_regs on chunk ch loaded from global memory.
template <typename T, bool VEC, bool NEED_X, bool NEED_Y, class Mass>
__device__ __forceinline__ int warp_rescan(const T* x, const T* y, int64_t V, int ch, float tc,
                                           const Mass& mass, int lane, uint64_t pol) {
    uint4 bx[kLoads], by[kLoads];
    if (NEED_X) load_chunk<T, VEC>(x, V, ch, lane, pol, bx);
    if (NEED_Y) load_chunk<T, VEC>(y, V, ch, lane, pol, by);
    return rescan_regs<T, NEED_X, NEED_Y>(bx, by, ch, tc, mass, lane);
}

struct MassX {
    float mm, c;
    __device__ float operator()(float fx, float) const { return mass_rel(fx, mm, c); }
};
struct MassY {
    float mm, c;
    __device__ float operator()(float, float fy) const { return mass_rel(fy, mm, c); }
};
// Residual mass max(0, p(v) - q(v)) with p and q normalised by 1/Z factors.
struct MassRes {
    float mx, my, izx, izy, c;
    __device__ float operator()(float fx, float fy) const {
        const float p = ex2((fy - my) * c) * izy;
        const float q = ex2((fx - mx) * c) * izx;
        return fmaxf(p - q, 0.f);
    }
};

// Inverse-CDF draw from the distribution of one table component (warp).
// S is the table total; returns the token (or -1 if the row has no mass).
template <typename T, bool VEC>
__device__ __forceinline__ int warp_sample(const T* x, const T* y, int64_t V, const float4* tab,
                                           int nch, int comp, float M, const TableSum& S, float u,
                                           float c, int lane, uint64_t pol) {
    const Located loc = table_locate(tab, nch, comp, frame_of(M), c, S, u, lane);
    if (loc.ch < 0) return -1;
    const float mm = frame_of(tab_ms(tab[loc.ch], comp).x);
    if (comp == 0)
        return warp_rescan<T, VEC, true, false>(x, y, V, loc.ch, loc.tc, MassX{mm, c}, lane, pol);
    return warp_rescan<T, VEC, false, true>(x, y, V, loc.ch, loc.tc, MassY{mm, c}, lane, pol);
}

// First chunk whose target maximum equals the row max M (warp; -1 if none).
__device__ __forceinline__ int table_first_max(const float4* tab, int nch, float M, int comp = 1) {
    for (int g = 0; g < nch; g += 32) {
        const int cc = g + (threadIdx.x & 31);
        const unsigned hit =
            __ballot_sync(0xffffffffu, cc < nch && tab_ms(tab[cc], comp).x == M);
        if (hit) return g + __ffs(hit) - 1;
    }
    return -1;
}

// Lowest index of chunk ch (target chunk in registers) whose logit equals M
// (warp; -1 if none).
template <typename T>
__device__ __forceinline__ int first_max_regs(const uint4 (&by)[kLoads], int ch, float M) {
    constexpr int PV = Traits<T>::kPerVec;
    const int lane = threadIdx.x & 31;
    const int64_t base = (int64_t)ch * chunk_elems<T>();
#pragma unroll
    for (int k = 0; k < kLoads; ++k) {
        float f[PV];
        unpack<T>(by[k], f);
        int e0 = PV;
#pragma unroll
        for (int e = PV - 1; e >= 0; --e)
            if (f[e] == M) e0 = e;
        const unsigned hit = __ballot_sync(0xffffffffu, e0 < PV);
        if (hit) {
            const int L = __ffs(hit) - 1;
            const int e = __shfl_sync(0xffffffffu, e0, L);
            return (int)(base + (int64_t)k * 32 * PV + L * PV + e);
        }
    }
    return -1;
}

// Lowest index whose target logit equals the row max M (warp).
template <typename T, bool VEC>
__device__ __forceinline__ int warp_first_max(const T* y, int64_t V, const float4* tab, int nch,
                                              float M, int lane, uint64_t pol, int comp = 1) {
    const int ch = table_first_max(tab, nch, M, comp);
    if (ch < 0) return -1;
    uint4 by[kLoads];
    load_chunk<T, VEC>(y, V, ch, lane, pol, by);
    return first_max_regs<T>(by, ch, M);
}

__device__ __forceinline__ bool row_ok(float M, double Z) {
    return M > -INFINITY && M < INFINITY && Z > 0.0 && Z < INFINITY;
}

// log q and log alpha = min(0, log p - log q) of token v (Eq. 1), in double.
// The same from the token's draft and target logits xv, yv.
__device__ __forceinline__ void token_logs_vals(float xv, float yv, const RowRec& rec, double invT,
                                                float* lq, float* la) {
    const double lqd = ((double)xv - (double)rec.mx) * invT - rec.lzx;
    const double lpd = ((double)yv - (double)rec.my) * invT - rec.lzy;
    const double d = lpd - lqd;
    *lq = (float)lqd;
    *la = (float)(d >= 0.0 ? 0.0 : d);
}
template <typename T>
__device__ __forceinline__ void token_logs(const T* x, const T* y, int v, const RowRec& rec,
                                           double invT, float* lq, float* la) {
    token_logs_vals(elem_value(x, v), elem_value(y, v), rec, invT, lq, la);
}

// --------------------------------------------------------------- row pass
enum XMode { kNoToken = 0, kSampleToken = 1, kGivenToken = 2 };

// One of the row's three table-driven results (warp; every lane returns the
// same values): which = 0 the draft statistics and z~ (drawn from q with
// u_draft, or read from given_tokens), 1 the target statistics and the draw
// from p with u_correct, 2 the lowest-index argmax of the target.
struct RowTask {
    float M;
    TableSum S;
    int tok;
};
template <typename T, bool VEC, int XMODE>
__device__ __forceinline__ RowTask row_task(const Problem<T>& P, int r, const float4* tab,
                                            int which, int lane) {
    const int64_t V = P.V;
    const T* x = P.draft + (int64_t)r * V;
    const T* y = P.target + (int64_t)r * V;
    const float c = P.ts.c;
    const uint64_t pol = policy_evict_normal();
    RowTask t;
    t.M = table_max(tab, P.nch, which == 0 ? 0 : 1, lane);
    t.S = TableSum{0, 0, 0.0};
    t.tok = -1;
    if (which == 2) {
        if (t.M > -INFINITY) t.tok = warp_first_max<T, VEC>(y, V, tab, P.nch, t.M, lane, pol);
        if (t.tok >= V) t.tok = -1;
        return t;
    }
    t.S = table_sum(tab, P.nch, which, frame_of(t.M), c, lane);
    if (which == 0) {
        if (XMODE == kSampleToken) {
            if (row_ok(t.M, t.S.Z))
                t.tok = P.greedy ? warp_first_max<T, VEC>(x, V, tab, P.nch, t.M, lane, pol, 0)
                                 : warp_sample<T, VEC>(x, y, V, tab, P.nch, 0, t.M, t.S,
                                                       __ldg(P.u_draft + r), c, lane, pol);
            if (t.tok >= V) t.tok = -1;
        } else if (XMODE == kGivenToken) {
            t.tok = __ldg(P.given_tokens + r);
        }
    } else {
        // (no uniforms for the p-draw: the reference rows of
        // vsd_reference_logkappa need only the argmax)
        if (row_ok(t.M, t.S.Z) && (P.greedy || P.u_correct))
            t.tok = P.greedy ? warp_first_max<T, VEC>(y, V, tab, P.nch, t.M, lane, pol)
                             : warp_sample<T, VEC>(x, y, V, tab, P.nch, 1, t.M, t.S,
                                                   __ldg(P.u_correct + r), c, lane, pol);
        if (t.tok >= V) t.tok = -1;
    }
    return t;
}

// The row record from the three tasks (warp): lanes 0..2 take the log q and
// log alpha of z~, of the p-draw and of the argmax; lane 0 writes rows[r] and
// rstats[r].
// vals(which, v, xv, yv) gives the draft and target logits of token v (the
// draw `which`).
template <typename T, bool HAS_Y, int XMODE, bool ARGMAX, class Vals>
__device__ __forceinline__ void row_finish(const Problem<T>& P, int r, const RowTask& tx,
                                           const RowTask& ty, int ref, int lane, const Vals& vals) {
    const int64_t V = P.V;
    const double invT = P.ts.invTd;
    const bool okx = row_ok(tx.M, tx.S.Z);
    const bool oky = HAS_Y ? row_ok(ty.M, ty.S.Z) : true;
    const bool ok = okx && oky;
    // the two logarithms at once, on lanes 0 and 1
    const double lz = log(lane == 0 ? tx.S.Z : ty.S.Z);
    const double lzx0 = __shfl_sync(0xffffffffu, lz, 0), lzy0 = __shfl_sync(0xffffffffu, lz, 1);
    const double lzx = okx ? lzx0 : 0.0;
    const double lzy = (HAS_Y && oky) ? lzy0 : 0.0;
    const int tok = XMODE == kNoToken ? -1 : tx.tok;
    const bool tok_ok = tok >= 0 && tok < V;
    float lq = -INFINITY, la = -INFINITY;
    if (lane < 3) {
        const int v = lane == 0 ? tok : (lane == 1 ? ty.tok : ref);
        const bool want = lane == 0 || (HAS_Y && (lane == 1 || ARGMAX));
        if (want && ok && v >= 0 && v < V) {
            RowRec tmp;
            tmp.mx = tx.M;
            tmp.lzx = lzx;
            tmp.my = HAS_Y ? ty.M : 0.f;
            tmp.lzy = lzy;
            float xv, yv;
            vals(lane, v, xv, yv);
            if (HAS_Y)
                token_logs_vals(xv, yv, tmp, invT, &lq, &la);
            else
                lq = (float)(((double)xv - (double)tmp.mx) * invT - tmp.lzx);
        }
    }
    if (P.greedy && lane < 3 && la > -INFINITY) {
        // T = 0: alpha is 1 where the token is the target's argmax (the
        // p-draw and the reference are), else 0 (one-hot limits)
        la = (lane == 0 && tok != ref) ? -INFINITY : 0.f;
    }
    const float lq1 = __shfl_sync(0xffffffffu, lq, 1), la1 = __shfl_sync(0xffffffffu, la, 1);
    const float la2 = __shfl_sync(0xffffffffu, la, 2);
    if (lane == 0) {
        RowRec rec;
        rec.mx = tx.M;
        rec.lzx = lzx;
        rec.my = HAS_Y ? ty.M : 0.f;
        rec.lzy = lzy;
        rec.izx = okx ? 1.f / (float)tx.S.Z : 0.f;
        rec.izy = (HAS_Y && oky) ? 1.f / (float)ty.S.Z : 0.f;
        rec.pad[0] = rec.pad[1] = rec.pad[2] = 0;
        rec.flags = ok ? 0 : 1;
        if (!ok) atomicOr(P.status, VSD_STATUS_BAD_ROW);
        if (!ok && P.kl_topk) {  // an invalid row has no top-K term
            P.klr[r].n = 0;
            P.klr[r].loss = 0.f;
            if (P.out.kl_loss) P.out.kl_loss[r] = 0.f;
        }
        int t = tok;
        if (XMODE == kGivenToken && !tok_ok) {
            atomicOr(P.status, VSD_STATUS_BAD_TOKEN);
            t = -1;
            rec.flags |= 2;
        }
        rec.tok = t;
        rec.lq_tok = (ok && t >= 0) ? lq : -INFINITY;
        rec.la_tok = (ok && t >= 0) ? la : -INFINITY;
        rec.ps = (HAS_Y && ok) ? ty.tok : -1;
        rec.lq_ps = (HAS_Y && ok) ? lq1 : -INFINITY;
        rec.la_ps = (HAS_Y && ok) ? la1 : -INFINITY;
        rec.ref = (HAS_Y && ARGMAX && ok) ? ref : -1;
        rec.la_ref = (HAS_Y && ARGMAX && ok) ? la2 : -INFINITY;
        P.rows[r] = rec;
        P.rstats[r] = make_float4(rec.mx, (float)rec.lzx, rec.my, (float)rec.lzy);
    }
}

struct RowShared {
    RowTask t[3];
};

// VSD (KL): the row's top-K term of Eq. klv (defined below).
template <typename T, bool VEC>
__device__ void kl_select(const Problem<T>& P, int r, const float4* tab, int nch, uint4* buf,
                          int npair, bool ok, int lane);

// The per-row work once the row's chunk table tab[0..nch) is complete
// (block, or with BAR > 0 the kThreads threads 0 .. kThreads-1 that meet at
// named barrier BAR): warps 0, 1 and 2 take the three tasks at once, warp 0
// then writes the record.
template <typename T, bool VEC, bool HAS_Y, int XMODE, bool ARGMAX, int BAR = 0, bool KL = false>
__device__ void row_tail(const Problem<T>& P, int r, const float4* tab, RowShared& sh,
                         uint4* klbuf = nullptr) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (warp == 0 || (HAS_Y && (warp == 1 || (ARGMAX && warp == 2)))) {
        const RowTask t = row_task<T, VEC, XMODE>(P, r, tab, warp, lane);
        if (lane == 0) sh.t[warp] = t;
    } else if (KL && HAS_Y && warp == 3) {
        // VSD (KL): the top-K term on the fourth warp (an invalid row's term
        // is cleared by row_finish)
        kl_select<T, VEC>(P, r, tab, P.nch, klbuf, 2, true, lane);
    }
    if (BAR == 0)
        __syncthreads();
    else
        asm volatile("bar.sync %0, %1;" ::"r"(BAR), "r"(kThreads) : "memory");
    if (warp == 0) {
        RowTask ty = sh.t[1];
        if (!HAS_Y) ty = RowTask{0.f, TableSum{0, 0, 0.0}, -1};
        const int ref = (HAS_Y && ARGMAX) ? sh.t[2].tok : -1;
        const T* x = P.draft + (int64_t)r * P.V;
        const T* y = HAS_Y ? P.target + (int64_t)r * P.V : nullptr;
        row_finish<T, HAS_Y, XMODE, ARGMAX>(P, r, sh.t[0], ty, ref, lane,
                                            [&](int, int v, float& xv, float& yv) {
                                                xv = elem_value(x, v);
                                                yv = HAS_Y ? elem_value(y, v) : 0.f;
                                            });
    }
}

// Chunk ch of a row into a shared-memory buffer with cp.async (warp; rows
// 16-byte aligned).  Vectors at or beyond V are not read.
template <typename T>
__device__ __forceinline__ void chunk_async(uint4* buf, const T* row, int64_t V, int ch,
                                            int lane) {
    constexpr int PV = Traits<T>::kPerVec;
    const int64_t base = (int64_t)ch * chunk_elems<T>() + lane * PV;
#pragma unroll
    for (int k = 0; k < kLoads; ++k) {
        const int64_t v0 = base + (int64_t)k * 32 * PV;
        cp_async16(buf + k * 32 + lane, row + (v0 < V ? v0 : 0), v0 < V);
    }
}
// The chunk in registers as load_chunk gives it (positions at or beyond V
// read as -inf).
template <typename T>
__device__ __forceinline__ void chunk_from_smem(const uint4* buf, int64_t V, int ch, int lane,
                                                uint4 (&b)[kLoads]) {
    constexpr int PV = Traits<T>::kPerVec;
    const int64_t base = (int64_t)ch * chunk_elems<T>() + lane * PV;
#pragma unroll
    for (int k = 0; k < kLoads; ++k)
        b[k] = base + (int64_t)k * 32 * PV < V
                   ? buf[k * 32 + lane]
                   : make_uint4(Traits<T>::kNegInf, Traits<T>::kNegInf, Traits<T>::kNegInf,
                                Traits<T>::kNegInf);
}
// Logit v of a buffer holding chunk ch.
__device__ __forceinline__ float smem_elem(const uint4* buf, int ch, int v, const float*) {
    return reinterpret_cast<const float*>(buf)[v - ch * chunk_elems<float>()];
}
__device__ __forceinline__ float smem_elem(const uint4* buf, int ch, int v, const __nv_bfloat16*) {
    return __bfloat162float(
        reinterpret_cast<const __nv_bfloat16*>(buf)[v - ch * chunk_elems<__nv_bfloat16>()]);
}

// --------------------------------------------------------------- VSD (KL)
// The top-Kt tokens of the target row r (largest logit, lowest index on ties:
// p's order at any T > 0) and the terms of Eq. klv on them (warp): p^ and q^
// renormalised on those tokens, L = -sum p^ log q^, and the gradient
// kl_scale (q^ - p^) of each token (log q^ = x/T - log sum over the tokens, so
// the vocabulary's partition cancels and no other logit has a gradient).
//
// Only a chunk whose target maximum reaches the Kt-th largest chunk maximum
// can hold a selected token (Kt chunk maxima are that large, so the Kt-th
// largest logit is too).  The warp reads those chunks of both rows in
// increasing order, skipping a chunk whose maximum cannot beat the current
// Kt-th entry, and keeps the running list sorted by (logit desc, index asc)
// in lanes 0 .. Kt-1.  buf stages npair chunk pairs in shared memory (null:
// loads into registers, one pair at a time).  ok = false (an invalid row)
// writes an empty term.
template <typename T, bool VEC>
__device__ void kl_select(const Problem<T>& P, int r, const float4* tab, int nch, uint4* buf,
                          int npair, bool ok, int lane) {
    constexpr int PV = Traits<T>::kPerVec;
    constexpr int CE = chunk_elems<T>();
    constexpr unsigned FULL = 0xffffffffu;
    const int64_t V = P.V;
    const T* x = P.draft + (int64_t)r * V;
    const T* y = P.target + (int64_t)r * V;
    KlRec* dst = P.klr + r;
    const int Kt = (int)min((int64_t)P.kl_topk, V);
    if (!ok) {
        if (lane == 0) {
            dst->n = 0;
            dst->loss = 0.f;
            if (P.out.kl_loss) P.out.kl_loss[r] = 0.f;
        }
        return;
    }
    // the Kt-th largest chunk maximum (order: value desc, chunk asc)
    float tv = INFINITY, tk = -INFINITY;
    int tch = -1;
    for (int k = 0; k < Kt; ++k) {
        float bv = -INFINITY;
        int bc = 0x7fffffff;
        for (int ch = lane; ch < nch; ch += 32) {
            const float v = tab[ch].z;
            const bool after = v < tv || (v == tv && ch > tch);
            if (after && (v > bv || (v == bv && ch < bc))) {
                bv = v;
                bc = ch;
            }
        }
#pragma unroll
        for (int o = 16; o; o >>= 1) {
            const float ov = __shfl_xor_sync(FULL, bv, o);
            const int oc = __shfl_xor_sync(FULL, bc, o);
            if (ov > bv || (ov == bv && oc < bc)) {
                bv = ov;
                bc = oc;
            }
        }
        if (bc == 0x7fffffff) {  // fewer chunks than Kt: every chunk is a candidate
            tk = -INFINITY;
            break;
        }
        tv = bv;
        tch = bc;
        tk = bv;
    }
    float lv = -INFINITY, lx = 0.f;  // lane i < Kt: entry i (target logit, draft logit, index)
    int li = 0x7fffffff;
    int cnt = 0;
    float thv = -INFINITY;
    int thi = 0x7fffffff;
    auto insert = [&](float v, int idx, float xv) {
        const bool above = lane < cnt && (lv > v || (lv == v && li < idx));
        const int pos = __popc(__ballot_sync(FULL, above));
        if (pos >= Kt) return;
        const float pv = __shfl_up_sync(FULL, lv, 1);
        const int pi = __shfl_up_sync(FULL, li, 1);
        const float px = __shfl_up_sync(FULL, lx, 1);
        if (lane > pos) {
            lv = pv;
            li = pi;
            lx = px;
        }
        if (lane == pos) {
            lv = v;
            li = idx;
            lx = xv;
        }
        cnt = min(cnt + 1, Kt);
        if (cnt == Kt) {
            thv = __shfl_sync(FULL, lv, Kt - 1);
            thi = __shfl_sync(FULL, li, Kt - 1);
        }
    };
    auto scan_chunk = [&](int ch, const uint4 (&bx)[kLoads], const uint4 (&by)[kLoads]) {
#pragma unroll
        for (int k = 0; k < kLoads; ++k) {
            float fx[PV], fy[PV];
            unpack<T>(bx[k], fx);
            unpack<T>(by[k], fy);
#pragma unroll
            for (int e = 0; e < PV; ++e) {
                const int idx = ch * CE + k * 32 * PV + lane * PV + e;
                const bool c = idx < V && (cnt < Kt || fy[e] > thv || (fy[e] == thv && idx < thi));
                for (unsigned m = __ballot_sync(FULL, c); m; m &= m - 1) {
                    const int L = __ffs(m) - 1;
                    insert(__shfl_sync(FULL, fy[e], L), __shfl_sync(FULL, idx, L),
                           __shfl_sync(FULL, fx[e], L));
                }
            }
        }
    };
    const int np = (VEC && buf) ? max(1, min(npair, 3)) : 1;
    const uint64_t pol = policy_evict_normal();
    int ch0 = 0;
    for (;;) {
        int cand[3] = {-1, -1, -1};
        int nc = 0;
        while (nc < np && ch0 < nch) {
            const int ch = ch0 + lane;
            const float mxc = ch < nch ? tab[ch].z : -INFINITY;
            const bool want = ch < nch && mxc >= tk && (cnt < Kt || mxc > thv);
            unsigned bal = __ballot_sync(FULL, want);
            while (bal && nc < np) {
                cand[nc++] = ch0 + __ffs(bal) - 1;
                bal &= bal - 1;
            }
            ch0 = bal ? ch0 + __ffs(bal) - 1 : ch0 + 32;
        }
        if (nc == 0) break;
        if (VEC && buf) {
            for (int j = 0; j < nc; ++j) {
                chunk_async<T>(buf + (2 * j) * kLoads * 32, x, V, cand[j], lane);
                chunk_async<T>(buf + (2 * j + 1) * kLoads * 32, y, V, cand[j], lane);
            }
            cp_async_wait_all();
            __syncwarp();
            for (int j = 0; j < nc; ++j) {
                uint4 bx[kLoads], by[kLoads];
                chunk_from_smem<T>(buf + (2 * j) * kLoads * 32, V, cand[j], lane, bx);
                chunk_from_smem<T>(buf + (2 * j + 1) * kLoads * 32, V, cand[j], lane, by);
                scan_chunk(cand[j], bx, by);
            }
            __syncwarp();
        } else {
            uint4 bx[kLoads], by[kLoads];
            load_chunk<T, VEC>(x, V, cand[0], lane, pol, bx);
            load_chunk<T, VEC>(y, V, cand[0], lane, pol, by);
            scan_chunk(cand[0], bx, by);
        }
    }
    // Eq. klv on the selected tokens (fp64; the list is sorted, lane 0 holds
    // the largest target logit)
    const bool mine = lane < Kt;
    const double invT = P.ts.invTd;
    const double y0 = (double)__shfl_sync(FULL, lv, 0);
    const double xm = (double)warp_max(mine ? lx : -INFINITY);
    const double ep = mine ? exp(((double)lv - y0) * invT) : 0.0;
    const double eq = mine ? exp(((double)lx - xm) * invT) : 0.0;
    const double Sp = warp_sum(ep), Sq = warp_sum(eq);
    const double ph = ep / Sp;
    const double lqh = ((double)lx - xm) * invT - log(Sq);
    const double L = warp_sum((mine && ph > 0.0) ? -ph * lqh : 0.0);
    if (mine) {
        dst->tok[lane] = li;
        dst->coef[lane] = (float)(P.kl_scale * (exp(lqh) - ph));
    }
    if (lane == 0) {
        dst->loss = (float)L;
        dst->n = Kt;
        if (P.out.kl_loss) P.out.kl_loss[r] = (float)L;
    }
}

// Shared memory of the fused kernel's control warp: the six chunks a row tail
// rescans, or the M-step's scratch (never both at once).
struct RescanBuf {
    uint4 c[6][kLoads * 32];
};

// The row tail of row r by one warp (the fused kernel's control warp) with
// its memory accesses batched, because each dependent round trip to memory
// is slow while the streaming warps keep DRAM busy: one round trip for the
// row's table (from global memory into tab) and its uniforms, then the three
// draws' table work, then one round trip (cp.async) for the draft and target
// chunks at the three chunks the draws rescan, which also hold the logits of
// the tokens they return.  Same tokens and record as row_tail.
template <typename T, bool VEC, bool KL = false>
__device__ void row_tail_warp(const Problem<T>& P, int r, float4* tab, RescanBuf& rb, int lane) {
    const int64_t V = P.V;
    const int nch = P.nch;
    const T* x = P.draft + (int64_t)r * V;
    const T* y = P.target + (int64_t)r * V;
    const float c = P.ts.c;
    const float ud = __ldg(P.u_draft + r), uc = __ldg(P.u_correct + r);
    const float4* rtab = P.gtab + (int64_t)r * P.nch_ws;
    for (int ch = lane; ch < nch; ch += 32) tab[ch] = ld_cg(rtab + ch);
    __syncwarp();
    RowTask tx{table_max(tab, nch, 0, lane), TableSum{0, 0, 0.0}, -1};
    tx.S = table_sum(tab, nch, 0, frame_of(tx.M), c, lane);
    RowTask ty{table_max(tab, nch, 1, lane), TableSum{0, 0, 0.0}, -1};
    ty.S = table_sum(tab, nch, 1, frame_of(ty.M), c, lane);
    Located lx{-1, 0.f}, ly{-1, 0.f};
    const int ca = ty.M > -INFINITY ? table_first_max(tab, nch, ty.M) : -1;
    if (P.greedy) {  // T = 0: the argmax of each row (first chunk holding its maximum)
        if (row_ok(tx.M, tx.S.Z)) lx.ch = table_first_max(tab, nch, tx.M, 0);
        if (row_ok(ty.M, ty.S.Z)) ly.ch = ca;
    } else {
        if (row_ok(tx.M, tx.S.Z)) lx = table_locate(tab, nch, 0, frame_of(tx.M), c, tx.S, ud, lane);
        if (row_ok(ty.M, ty.S.Z)) ly = table_locate(tab, nch, 1, frame_of(ty.M), c, ty.S, uc, lane);
    }
    const int chs[3] = {lx.ch, ly.ch, ca};
    if (VEC) {
#pragma unroll
        for (int w = 0; w < 3; ++w)
            if (chs[w] >= 0) {
                chunk_async<T>(rb.c[2 * w], x, V, chs[w], lane);
                chunk_async<T>(rb.c[2 * w + 1], y, V, chs[w], lane);
            }
        cp_async_wait_all();
        __syncwarp();
    }
    const uint64_t pol = policy_evict_normal();
    uint4 b[kLoads];
    if (lx.ch >= 0) {
        if (VEC) chunk_from_smem<T>(rb.c[0], V, lx.ch, lane, b);
        else load_chunk<T, VEC>(x, V, lx.ch, lane, pol, b);
        const float mm = frame_of(tab_ms(tab[lx.ch], 0).x);
        tx.tok = P.greedy ? first_max_regs<T>(b, lx.ch, tx.M)
                          : rescan_regs<T, true, false>(b, b, lx.ch, lx.tc, MassX{mm, c}, lane);
        if (tx.tok >= V) tx.tok = -1;
    }
    if (ly.ch >= 0) {
        if (VEC) chunk_from_smem<T>(rb.c[3], V, ly.ch, lane, b);
        else load_chunk<T, VEC>(y, V, ly.ch, lane, pol, b);
        const float mm = frame_of(tab_ms(tab[ly.ch], 1).x);
        ty.tok = P.greedy ? first_max_regs<T>(b, ly.ch, ty.M)
                          : rescan_regs<T, false, true>(b, b, ly.ch, ly.tc, MassY{mm, c}, lane);
        if (ty.tok >= V) ty.tok = -1;
    }
    int ref = -1;
    if (ca >= 0) {
        if (VEC) chunk_from_smem<T>(rb.c[5], V, ca, lane, b);
        else load_chunk<T, VEC>(y, V, ca, lane, pol, b);
        ref = first_max_regs<T>(b, ca, ty.M);
        if (ref >= V) ref = -1;
    }
    row_finish<T, true, kSampleToken, true>(P, r, tx, ty, ref, lane,
                                            [&](int w, int v, float& xv, float& yv) {
                                                if (VEC) {
                                                    xv = smem_elem(rb.c[2 * w], chs[w], v, x);
                                                    yv = smem_elem(rb.c[2 * w + 1], chs[w], v, y);
                                                } else {
                                                    xv = elem_value(x, v);
                                                    yv = elem_value(y, v);
                                                }
                                            });
    if (KL) {  // VSD (KL): the row's top-K term, staged through the rescan buffers
        __syncwarp();
        kl_select<T, VEC>(P, r, tab, nch, rb.c[0], 3,
                          row_ok(tx.M, tx.S.Z) && row_ok(ty.M, ty.S.Z), lane);
    }
}

// Streams row r of the draft (and, with HAS_Y, of the target) once, then runs
// row_tail.  XMODE: whether z~ is drawn from q with u_draft, read from
// given_tokens, or absent (trees).  ARGMAX: locate the greedy reference token.
template <typename T, bool VEC, bool HAS_Y, int XMODE, bool ARGMAX>
__device__ void row_pass(const Problem<T>& P, int r, Ring* rg, float4* tab, RowShared& sh) {
    const int64_t V = P.V;
    const T* x = P.draft + (int64_t)r * V;
    const T* y = HAS_Y ? P.target + (int64_t)r * V : nullptr;
    // The draft row is read again by the gradient pass: ask L2 to keep it.
    stream_tables<T, VEC, HAS_Y>(rg, x, y, V, 0, P.nch, tab, P.ts.c, policy_evict_last(),
                                 policy_evict_first(), P.status);
    __syncthreads();
    row_tail<T, VEC, HAS_Y, XMODE, ARGMAX>(P, r, tab, sh);
}

// --------------------------------------------------------------- residual
// Stream rows x, y once more and fill tab[c].y with the chunk sums of the
// residual mass max(0, p - q).
template <typename T>
__device__ __forceinline__ float residual_chunk(const uint4 (&bx)[kLoads], const uint4 (&by)[kLoads],
                                               const MassRes& mr) {
    constexpr int NP = Traits<T>::kPerVec / 2;
    const uint64_t mx2 = f2(mr.mx, mr.mx), my2 = f2(mr.my, mr.my), c2 = f2(mr.c, mr.c);
    const uint64_t izx2 = f2(mr.izx, mr.izx), izy2 = f2(mr.izy, mr.izy);
    float acc = 0.f;
#pragma unroll
    for (int k = 0; k < kLoads; ++k) {
        uint64_t px[NP], py[NP];
        vec_pairs<T>(bx[k], px);
        vec_pairs<T>(by[k], py);
#pragma unroll
        for (int i = 0; i < NP; ++i) {
            const uint64_t q2 = f2mul(f2_mass(px[i], mx2, c2), izx2);
            const uint64_t p2 = f2mul(f2_mass(py[i], my2, c2), izy2);
            float lo, hi;
            f2split(f2sub(p2, q2), lo, hi);
            acc += fmaxf(lo, 0.f) + fmaxf(hi, 0.f);
        }
    }
    return warp_sum(acc);
}

template <typename T, bool VEC>
__device__ void stream_residual(Ring* rg, const T* x, const T* y, int64_t V, int ch0, int ch1,
                                float4* tab, const MassRes& mr, int* status) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint64_t pol = policy_evict_normal();
    if constexpr (VEC) {
        ring_stream<T, true>(rg, x, y, V, ch0, ch1, pol, pol, status,
                             [&](int ch, const uint4 (&bx)[kLoads], const uint4 (&by)[kLoads]) {
                                 const float t = residual_chunk<T>(bx, by, mr);
                                 if (lane == 0) tab[ch] = make_float4(0.f, t, 0.f, 0.f);
                             });
        return;
    }
    int ch = ch0 + warp;
    uint4 bx[kLoads], by[kLoads];
    if (ch < ch1) {
        load_chunk<T, VEC>(x, V, ch, lane, pol, bx);
        load_chunk<T, VEC>(y, V, ch, lane, pol, by);
    }
    while (ch < ch1) {
        const int cn = ch + kWarps;
        uint4 nx[kLoads], ny[kLoads];
        if (cn < ch1) {
            load_chunk<T, VEC>(x, V, cn, lane, pol, nx);
            load_chunk<T, VEC>(y, V, cn, lane, pol, ny);
        }
        const float t = residual_chunk<T>(bx, by, mr);
        if (lane == 0) tab[ch] = make_float4(0.f, t, 0.f, 0.f);
#pragma unroll
        for (int k = 0; k < kLoads; ++k) {
            bx[k] = nx[k];
            by[k] = ny[k];
        }
        ch = cn;
    }
}

// Residual draw norm(max(0, p - q)) at row r with uniform u (block).  Returns
// -1 when the residual has no mass.
template <typename T, bool VEC>
__device__ int residual_draw(const Problem<T>& P, int r, const RowRec& rec, float u, Ring* rg,
                             float4* tab, int* out) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t V = P.V;
    const T* x = P.draft + (int64_t)r * V;
    const T* y = P.target + (int64_t)r * V;
    const float c = P.ts.c;
    const MassRes mr{rec.mx, rec.my, rec.izx, rec.izy, c};
    stream_residual<T, VEC>(rg, x, y, V, 0, P.nch, tab, mr, P.status);
    __syncthreads();
    if (warp == 0) {
        const TableSum Rt = table_sum(tab, P.nch, 0, 0.f, c, lane);
        int tok = -1;
        if (Rt.Z > 0.0) {
            const Located loc = table_locate(tab, P.nch, 0, 0.f, c, Rt, u, lane);
            if (loc.ch >= 0)
                tok = warp_rescan<T, VEC, true, true>(x, y, V, loc.ch, loc.tc, mr, lane,
                                                      policy_evict_normal());
        }
        if (tok >= V) tok = -1;
        if (lane == 0) *out = tok;
    }
    __syncthreads();
    const int tok = *out;
    __syncthreads();
    return tok;
}

// --------------------------------------------------------------- path pass
struct PathShared {
    int A;
    int resid;
    RowRec rec;
};

// Linear proposal path (b, s) = path: rows path*D .. path*D + D - 1.
// The accepted length A of the path (warp; first rejection by ballot).
template <typename T>
__device__ __forceinline__ int path_accept_len(const Problem<T>& P, int path, int lane) {
    const int D = P.D;
    const int r0 = path * D;
    int A = D;
    for (int d0 = 0; d0 < D; d0 += 32) {
        const int d = d0 + lane;
        bool rej = false;
        if (d < D) {
            const RowRec rec = ld_cg(P.rows + r0 + d);
            const float a = rec.flags ? 0.f : expf(rec.la_tok);
            rej = rec.flags || !(__ldg(P.u_accept + r0 + d) <= a);
        }
        const unsigned bal = __ballot_sync(0xffffffffu, rej);
        if (bal && A == D) A = d0 + __ffs(bal) - 1;
    }
    return A;
}

// path_head (warp 0): the accepted length A and, if A < D, the record of
// row A.  Written to sh.A, sh.rec.
template <typename T>
__device__ void path_head(const Problem<T>& P, int path, PathShared& sh) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (warp == 0) {
        const int A = path_accept_len<T>(P, path, lane);
        if (lane == 0) {
            sh.A = A;
            if (A < P.D) sh.rec = ld_cg(P.rows + path * P.D + A);
        }
    }
}

// path_epilogue_warp (one warp): given A and the residual token at row A (-1: none
// or no residual mass), the corrected path, alpha', the log-kappa prefix sums
// of z~, z' and the reference (Eq. 2, warp scans), E[A] (Eq. 11); writes the
// E-step view and the requested outputs.
// have_rl: rlq, rla are the log q and log alpha of the residual token (else
// they are read from the logits).
template <typename T>
__device__ void path_epilogue_warp(const Problem<T>& P, int path, int A, int resid, int lane,
                                   bool have_rl = false, float rlq = 0.f, float rla = 0.f) {
    const int D = P.D;
    const int r0 = path * D;
    {
        const int b = path / P.K;
        const double NEG = -INFINITY;
        const int64_t V = P.V;
        const vsd_linear_outputs& o = P.out;
        double ck = 0.0, ckc = 0.0, ckr = 0.0, EA = 0.0;
        for (int d0 = 0; d0 < D; d0 += 32) {
            const int d = d0 + lane;
            const bool act = d < D;
            const int r = r0 + (act ? d : 0);
            RowRec rec;
            if (act) rec = ld_cg(P.rows + r);
            float a = 0.f;
            double tk = 0.0, tkc = 0.0, tkr = 0.0;
            bool acc = false;
            int zc = -1;
            float lqc = -INFINITY, lac = -INFINITY;
            if (act) {
                a = rec.flags ? 0.f : expf(rec.la_tok);  // alpha (Eq. 1)
                acc = !rec.flags && __ldg(P.u_accept + r) <= a;
                if (d < A) {
                    zc = rec.tok; lqc = rec.lq_tok; lac = rec.la_tok;
                } else if (d == A) {
                    zc = resid >= 0 ? resid : rec.ps;  // no residual mass: draw from p
                    if (zc == rec.ps) {
                        lqc = rec.lq_ps; lac = rec.la_ps;
                    } else if (have_rl) {
                        lqc = rlq; lac = rla;
                    } else {
                        token_logs(P.draft + (int64_t)r * V, P.target + (int64_t)r * V, zc, rec,
                                   P.ts.invTd, &lqc, &lac);
                    }
                } else {
                    zc = rec.ps; lqc = rec.lq_ps; lac = rec.la_ps;
                }
                if (rec.flags) { zc = -1; lqc = lac = -INFINITY; }
                tk = rec.flags ? NEG : (double)rec.la_tok;
                tkc = zc >= 0 ? (double)lac : NEG;
                tkr = rec.ref >= 0 ? (double)rec.la_ref : NEG;
            }
            // prefix sums over l (Eq. 2): log kappa of z~, z' and the reference
            const double lk = ck + warp_incl_scan(tk, lane);
            const double lkc = ckc + warp_incl_scan(tkc, lane);
            double lkr = ckr + warp_incl_scan(tkr, lane);
            if (P.ref_logkappa && act) lkr = (double)__ldg(P.ref_logkappa + (int64_t)b * D + d);
            EA += warp_sum(act ? (double)expf((float)lk) : 0.0);  // Eq. 11
            const int lastl = min(31, D - 1 - d0);
            ck = __shfl_sync(0xffffffffu, lk, lastl);
            ckc = __shfl_sync(0xffffffffu, lkc, lastl);
            ckr = __shfl_sync(0xffffffffu, ckr + warp_incl_scan(tkr, lane), lastl);
            if (act) {
                P.es.tok[r] = rec.tok;
                P.es.corr[r] = zc;
                P.es.lq_tok[r] = rec.lq_tok;
                P.es.lq_corr[r] = lqc;
                P.es.lk[r] = (float)lk;
                P.es.lkc[r] = (float)lkc;
                P.es.lkr[r] = (float)lkr;
                if (o.tokens) o.tokens[r] = rec.tok;
                if (o.logq_tok) o.logq_tok[r] = rec.lq_tok;
                if (o.alpha) o.alpha[r] = a;
                if (o.accept) o.accept[r] = acc ? 1 : 0;
                if (o.corr_tokens) o.corr_tokens[r] = zc;
                if (o.logq_corr) o.logq_corr[r] = lqc;
                if (o.alpha_corr) o.alpha_corr[r] = zc >= 0 ? expf(lac) : 0.f;
                if (o.logkappa) o.logkappa[r] = (float)lk;
                if (o.logkappa_corr) o.logkappa_corr[r] = (float)lkc;
                if (o.logkappa_ref) o.logkappa_ref[r] = (float)lkr;
                if (o.ref_tokens) o.ref_tokens[r] = rec.ref;
                if (o.row_stats)
                    reinterpret_cast<float4*>(o.row_stats)[r] =
                        make_float4(rec.mx, (float)rec.lzx, rec.my, (float)rec.lzy);
            }
        }
        if (lane == 0) {
            if (o.accept_len) o.accept_len[path] = A;
            if (o.expected_len) o.expected_len[path] = (float)EA;
        }
    }
}

template <typename T>
__device__ void path_epilogue(const Problem<T>& P, int path, int A, int resid) {
    if ((threadIdx.x >> 5) == 0) path_epilogue_warp<T>(P, path, A, resid, threadIdx.x & 31);
}


// The whole path (block): head, the residual draw at the first rejection (one
// more streaming read of that row), epilogue.
template <typename T, bool VEC>
__device__ void path_pass(const Problem<T>& P, int path, Ring* rg, float4* tab, PathShared& sh) {
    const int D = P.D;
    const int r0 = path * D;
    path_head<T>(P, path, sh);
    __syncthreads();
    const int A = sh.A;
    int resid = -1;
    if (A < D && !sh.rec.flags)
        resid = residual_draw<T, VEC>(P, r0 + A, sh.rec, __ldg(P.u_correct + r0 + A), rg, tab,
                                      &sh.resid);
    path_epilogue<T>(P, path, A, resid);
}

// --------------------------------------------------------------- weights
// The M-step reads its prefix's E-step view in tiles of (s, l) entries, all
// proposals s and a run of positions l, so that each tile costs one round
// trip to memory.  Within a tile the entries are processed in parallel
// wherever the arithmetic allows, because double-precision latency, not
// work, bounds a single warp here.
constexpr int kMTile = 256;
constexpr int kLqE = 32;  // fixed-point scale 2^-32 of the M-step's sums
struct WeightsShared {
    // per proposal: running sums over l of log q(z~) and log q(z') (fixed point)
    long long lqt[256], lqc[256];
    // the tile: entry e = s * nd + (l - l0)
    float lq[kMTile];    // log q(z~); then the CAR weight
    float lqcz[kMTile];  // log q(z')
    unsigned char ot[kMTile], pc[kMTile];  // o~, and whether z' passes
    int tok[kMTile], corr[kMTile];
    long long elqt[kMTile];  // running sum of log q(z~) at the entry
    long long elqc[kMTile];  // running sum of log q(z'); then the term o'(1 - o~)
    long long et0[kMTile];   // the term o'(o~ - beta zeta)
    // per position of the tile
    int n1[64], n0[64];          // proposals with o' != 0 and o~ = 1, with o' != 0
    long long lmax[64];          // max over proposals of the running log q(z~)
    unsigned long long zs[64];   // sum of the CAR weights (fixed point, 2^-40)
    float rz[64];                // 1 / that sum
    float beta[64][3];           // leave-one-out beta for (o', o~) = (w, 1), (w, 0), (0, 0)
    float cmax[64];              // zeta_mode 0: exp(lmax) / tau
};

// x 2^E rounded toward zero, |x| clamped to 2^20 (a non-finite log-probability
// of an invalid row becomes -2^20); exact for |x| >= 2^(23-E).
__device__ __forceinline__ long long to_fixed(float x, int E) {
    float a = fabsf(x);
    if (!(a <= 1048576.f)) a = 1048576.f;
    const long long m = fixed_prod(a, 1.f, E);
    return (x < 0.f || x != x) ? -m : m;
}
// q 2^-E as a float (two 32-bit conversions: relative error below 2^-23).
__device__ __forceinline__ float from_fixed(long long q, int E) {
    const float hi = (float)(int)(q >> 32) * 4294967296.f;
    const float lo = (float)(unsigned)(q & 0xFFFFFFFFull);
    return ldexpf(hi + lo, -E);
}

// f(e) for the entries e = lane, lane + 32, ... < ne, four at a time so that
// their independent loads and double-precision chains overlap.
template <class F>
__device__ __forceinline__ void each_entry(int ne, int lane, F&& f) {
    for (int e0 = lane; e0 < ne; e0 += 128) {
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int e = e0 + 32 * u;
            if (e < ne) f(e);
        }
    }
}

// Load the tile of positions [d0, d0 + nd) of prefix b (warp).  TERMS: the
// per-entry terms written by the forward sweep (from wscr) instead of the
// scores.
template <typename T, bool TERMS>
__device__ __forceinline__ void mstep_tile(const Problem<T>& P, const EStepView& E, int b, int d0,
                                           int nd, WeightsShared& sh, int lane) {
    const int K = P.K, D = P.D;
    each_entry(K * nd, lane, [&](int e) {
        const int s = e / nd, r = (b * K + s) * D + d0 + (e - s * nd);
        sh.tok[e] = ld_cg(E.tok + r);
        sh.corr[e] = ld_cg(E.corr + r);
        if (TERMS) {
            const double2 tm = ld_cg(P.wscr + r);
            sh.et0[e] = to_fixed((float)tm.x, kLqE);
            sh.elqc[e] = to_fixed((float)tm.y, kLqE);
        } else {
            const float lkr = ld_cg(E.lkr + r);
            sh.ot[e] = ld_cg(E.lk + r) >= lkr ? 1 : 0;
            sh.pc[e] = ld_cg(E.lkc + r) >= lkr ? 1 : 0;
            sh.lq[e] = ld_cg(E.lq_tok + r);
            sh.lqcz[e] = ld_cg(E.lq_corr + r);
        }
    });
    __syncwarp();
}

// M-step of prefix b by one warp (K <= 256, D <= 64).  Writes coef[] for the
// prefix's rows, the optional weights table and loss_out[b].  No dependent
// double-precision chains (GB300's FP64 latency would dominate): sums over l
// and over entries are exact 64-bit fixed-point sums of float terms, the CAR
// weights come from exact differences of those sums, and every reduction is
// exact, so the result does not depend on the order of the entries.
template <typename T>
__device__ void weights_warp(const Problem<T>& P, const EStepView& E, int b, float* weights_out,
                             float* loss_out, WeightsShared& sh, int lane) {
    const int K = P.K, D = P.D;
    const int dt = max(1, min(D, kMTile / K));
    const bool one_tile = dt >= D;
    const float inv_tau = P.inv_tau_f;
    for (int s = lane; s < K; s += 32) sh.lqt[s] = sh.lqc[s] = 0;
    long long Jq = 0, Nq = 0;  // this lane's parts of J and N (fixed point, 2^-24)
    for (int d0 = 0; d0 < D; d0 += dt) {
        const int nd = min(dt, D - d0);
        const int ne = K * nd;
        mstep_tile<T, false>(P, E, b, d0, nd, sh, lane);
        // running sums of log q over l, per proposal: the fixed-point terms
        // for every entry at once, then integer adds along l
        each_entry(ne, lane, [&](int e) {
            sh.elqt[e] = to_fixed(sh.lq[e], kLqE);
            sh.elqc[e] = to_fixed(sh.lqcz[e], kLqE);
        });
        __syncwarp();
        for (int s = lane; s < K; s += 32) {
            long long a = sh.lqt[s], q = sh.lqc[s];
            for (int dd = 0; dd < nd; ++dd) {
                const int e = s * nd + dd;
                a += sh.elqt[e];
                q += sh.elqc[e];
                sh.elqt[e] = a;
                sh.elqc[e] = q;
            }
            sh.lqt[s] = a;
            sh.lqc[s] = q;
        }
        for (int dd = lane; dd < nd; dd += 32) {
            sh.n1[dd] = sh.n0[dd] = 0;
            sh.lmax[dd] = (long long)0x8000000000000000ull;
            sh.zs[dd] = 0;
        }
        __syncwarp();
        // per position: the counts behind beta and the largest running log q,
        // gathered from every entry at once with shared-memory integer atomics
        each_entry(ne, lane, [&](int e) {
            const int dd = e % nd;
            // Algorithm 2 scores z~ (o~); Algorithm 1 keeps z~ if it passes,
            // else z', so o' = w(l) when either passes
            const bool ot = sh.ot[e], op = ot || sh.pc[e];
            if (op) {
                atomicAdd(&sh.n0[dd], 1);
                if (ot) atomicAdd(&sh.n1[dd], 1);
            }
            atomicMax(&sh.lmax[dd], sh.elqt[e]);
        });
        __syncwarp();
        if (P.zeta_mode == 0)  // exp(lmax) / tau, with the float split hi + lo of lmax
            for (int dd = lane; dd < nd; dd += 32) {
                const long long m = sh.lmax[dd];
                const float hi = from_fixed(m, kLqE);
                const float lo = from_fixed(m - to_fixed(hi, kLqE), kLqE);
                sh.cmax[dd] = expf(hi) * (1.f + lo) * inv_tau;
            }
        __syncwarp();
        // CAR weights (Eq. zeta) relative to the proposal with the largest
        // logit: exp((Q_s - Q_max) / tau) with Q = q(z~_{1:l}) (zeta_mode 0:
        // Q_s - Q_max = Q_max expm1(d)) or Q = log q(z~_{1:l}) (zeta_mode 1:
        // Q_s - Q_max = d), d = the exact difference of the running sums
        each_entry(ne, lane, [&](int e) {
            const int dd = e % nd;
            const float d = from_fixed(sh.elqt[e] - sh.lmax[dd], kLqE);
            const float arg = P.zeta_mode == 0 ? sh.cmax[dd] * expm1f(d) : d * inv_tau;
            const float ez = expf(arg);
            sh.lq[e] = ez;
            // at most 1: exact sum at 2^-40
            const long long z = fixed_prod(ez, 1.f, 40);
            if (z) atomicAdd(&sh.zs[dd], (unsigned long long)z);
        });
        __syncwarp();
        // per position, in parallel: 1 / sum, and beta (Eq. beta, leave-one-out:
        // o' is w(l) or 0, so both of its sums are w(l) times a count)
        for (int dd = lane; dd < nd; dd += 32) {
            const int n1 = sh.n1[dd], n0 = sh.n0[dd];
            const float zs = (float)(long long)sh.zs[dd] * 0x1p-40f;
            sh.rz[dd] = zs > 0.f ? 1.f / zs : 0.f;
            sh.beta[dd][0] = n0 - 1 > 0 ? (float)(n1 - 1) / (float)(n0 - 1) : 0.f;
            sh.beta[dd][1] = n0 - 1 > 0 ? (float)n1 / (float)(n0 - 1) : 0.f;
            sh.beta[dd][2] = n0 > 0 ? (float)n1 / (float)n0 : 0.f;
        }
        __syncwarp();
        // per entry, in parallel: zeta, the objective terms (Eq. advance) and
        // the per-l gradient terms o'(o~ - beta zeta), o'(1 - o~)
        each_entry(ne, lane, [&](int e) {
            const int s = e / nd, dd = e - s * nd, d = d0 + dd;
            const bool otb = sh.ot[e], opb = otb || sh.pc[e];
            const float w = P.wlf[d];
            const float beta = sh.beta[dd][opb ? (otb ? 0 : 1) : 2];
            const float zeta = sh.lq[e] * sh.rz[dd];
            if (opb) {
                const float lqt = from_fixed(sh.elqt[e], kLqE);
                const float lqz = otb ? lqt : from_fixed(sh.elqc[e], kLqE);
                Jq += to_fixed(w * (lqz - beta * zeta * lqt), 24);
                Nq += to_fixed(w, 24);
            }
            const float t0 = opb ? w * ((otb ? 1.f : 0.f) - beta * zeta) : 0.f;
            const float t1 = (opb && !otb) ? w : 0.f;
            sh.et0[e] = to_fixed(t0, kLqE);
            sh.elqc[e] = to_fixed(t1, kLqE);
            const int r = (b * K + s) * D + d;
            if (!one_tile) P.wscr[r] = make_double2(t0, t1);
            if (weights_out) {
                float4* wo = reinterpret_cast<float4*>(weights_out) + ((int64_t)b * D + d) * K + s;
                *wo = make_float4(otb ? 1.f : 0.f, opb ? w : 0.f, beta, zeta);
            }
        });
        __syncwarp();
    }
    const float J = from_fixed(warp_sum_ll(Jq), 24), N = from_fixed(warp_sum_ll(Nq), 24);
    const float scale = N > 0.f ? 1.f / ((float)P.B * N * P.ts.T) : 0.f;
    // suffix sums over l, from the last tile back (lqt, lqc now hold c0, c1)
    for (int s = lane; s < K; s += 32) sh.lqt[s] = sh.lqc[s] = 0;
    for (int d0 = ((D - 1) / dt) * dt; d0 >= 0; d0 -= dt) {
        const int nd = min(dt, D - d0);
        if (!one_tile) {
            __syncwarp();
            mstep_tile<T, true>(P, E, b, d0, nd, sh, lane);
        }
        // integer adds along l from the end, then every entry's coefficients
        // at once
        for (int s = lane; s < K; s += 32) {
            long long c0 = sh.lqt[s], c1 = sh.lqc[s];
            for (int dd = nd - 1; dd >= 0; --dd) {
                const int e = s * nd + dd;
                c0 += sh.et0[e];
                c1 += sh.elqc[e];
                sh.et0[e] = c0;
                sh.elqc[e] = c1;
            }
            sh.lqt[s] = c0;
            sh.lqc[s] = c1;
        }
        __syncwarp();
        each_entry(K * nd, lane, [&](int e) {
            const int s = e / nd, dd = e - s * nd;
            const long long c0 = sh.et0[e], c1 = sh.elqc[e];
            Coef cf;
            cf.t0 = sh.tok[e];
            cf.t1 = sh.corr[e];
            const float g = from_fixed(c0 + c1, kLqE) * scale;
            if (cf.t1 == cf.t0) {
                cf.c0 = g;
                cf.c1 = 0.f;
                cf.t1 = -1;
            } else {
                cf.c0 = from_fixed(c0, kLqE) * scale;
                cf.c1 = from_fixed(c1, kLqE) * scale;
            }
            cf.g = g;
            cf.pad0 = cf.pad1 = cf.pad2 = 0.f;
            P.coef[(b * K + s) * D + d0 + dd] = cf;
        });
    }
    float klterm = 0.f;
    if (P.kl_topk) {  // VSD (KL): + kl_weight (1/K) sum of the prefix's rows' top-K terms
        double sk = 0.0;
        for (int i = lane; i < K * D; i += 32) sk += (double)ld_cg(&P.klr[b * K * D + i].loss);
        klterm = (float)(P.kl_weight / (double)K * warp_sum(sk));
    }
    if (lane == 0) loss_out[b] = (N > 0.f ? -J / N : 0.f) + klterm;
}

// The M-step by a block: warp 0 runs weights_warp (the same bits as the fused
// kernel's control warp).
template <typename T>
__device__ void weights_pass(const Problem<T>& P, const EStepView& E, int b, float* weights_out,
                             float* loss_out, WeightsShared& sh) {
    if ((threadIdx.x >> 5) == 0) weights_warp<T>(P, E, b, weights_out, loss_out, sh, threadIdx.x & 31);
}

// Mean of loss[0..B) into loss[B], summed in order (one thread).
__device__ __forceinline__ void loss_mean(float* loss, int B) {
    double s = 0.0;
    for (int b = 0; b < B; ++b) s += (double)ld_cg(loss + b);
    loss[B] = (float)(s / (double)B);
}

// --------------------------------------------------------------- gradient
// grad[r][v] = g q_r(v) - c0 [v = t0] - c1 [v = t1], q_r(v) = 2^{(x_v - m) c} / Z.
template <typename T, typename G, int PV>
__device__ __forceinline__ void grad_store(G* g, int64_t v0, const float (&o)[PV], uint64_t pol) {
    if constexpr (sizeof(G) == 2) {
        uint32_t w[PV / 2];
#pragma unroll
        for (int e = 0; e < PV / 2; ++e) {
            __nv_bfloat162 h = __floats2bfloat162_rn(o[2 * e], o[2 * e + 1]);
            w[e] = *reinterpret_cast<uint32_t*>(&h);
        }
        if constexpr (PV == 8)
            st_stream(g + v0, make_uint4(w[0], w[1], w[2], w[3]), pol);
        else  // f32 logits, bf16 gradient: 8 bytes per vector
            *reinterpret_cast<uint2*>(g + v0) = make_uint2(w[0], w[1]);
    } else {
        st_stream(g + v0, make_uint4(__float_as_uint(o[0]), __float_as_uint(o[1]),
                                     __float_as_uint(o[2]), __float_as_uint(o[3])),
                  pol);
        if constexpr (PV == 8)  // bf16 logits, f32 gradient: a second store
            st_stream(g + v0 + 4, make_uint4(__float_as_uint(o[4]), __float_as_uint(o[5]),
                                             __float_as_uint(o[6]), __float_as_uint(o[7])),
                      pol);
    }
}

// Gradient of elements [e0, e1) of row r (block).  On the vector path e0 and
// e1 are multiples of the vector width.
template <typename T, bool VEC, typename G>
__device__ void grad_pass_range(const Problem<T>& P, int r, int64_t e0, int64_t e1,
                                const float4* rstats, G* grad, const KlRec* kl = nullptr) {
    constexpr int PV = Traits<T>::kPerVec;
    constexpr int U = 8;  // vectors per batch per thread (two batches in flight)
    const int64_t V = P.V;
    const T* x = P.draft + (int64_t)r * V;
    G* g = grad + (int64_t)r * V;
    const float4 st = ld_cg(rstats + r);
    const Coef cf = ld_cg(P.coef + r);
    const float c = P.ts.c;
    const float mx = st.x;
    const float gq = (float)((double)cf.g * exp(-(double)st.y));
    const uint64_t pol = policy_evict_first();
    if constexpr (VEC) {
        constexpr int NP = PV / 2;
        const uint64_t mx2 = f2(mx, mx), c2 = f2(c, c), gq2 = f2(gq, gq);
        const int nvec = (int)(e1 / PV);
        const int ib = (int)(e0 / PV) + threadIdx.x;
        uint4 cur[U], nxt[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int i = ib + u * kThreads;
            if (i < nvec) cur[u] = ld_stream(x + (int64_t)i * PV, pol);
        }
        for (int i0 = ib; i0 < nvec; i0 += kThreads * U) {
            // the next batch is in flight while this one is computed and stored
            const int in = i0 + kThreads * U;
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int i = in + u * kThreads;
                if (i < nvec) nxt[u] = ld_stream(x + (int64_t)i * PV, pol);
            }
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int i = i0 + u * kThreads;
                if (i >= nvec) break;
                const int v0 = i * PV;
                uint64_t pr[NP];
                vec_pairs<T>(cur[u], pr);
                float o[PV];
#pragma unroll
                for (int k = 0; k < NP; ++k)
                    f2split(f2mul(f2_mass(pr[k], mx2, c2), gq2), o[2 * k], o[2 * k + 1]);
                // the sparse terms touch at most two positions of the row
                if ((unsigned)(cf.t0 - v0) < (unsigned)PV) {
#pragma unroll
                    for (int e = 0; e < PV; ++e)
                        if (v0 + e == cf.t0) o[e] -= cf.c0;
                }
                if ((unsigned)(cf.t1 - v0) < (unsigned)PV) {
#pragma unroll
                    for (int e = 0; e < PV; ++e)
                        if (v0 + e == cf.t1) o[e] -= cf.c1;
                }
                grad_store<T, G, PV>(g, v0, o, pol);
            }
#pragma unroll
            for (int u = 0; u < U; ++u) cur[u] = nxt[u];
        }
    } else {
        const int nkl = kl ? min(max(kl->n, 0), kMaxKlTop) : 0;
        for (int64_t v = e0 + threadIdx.x; v < e1; v += kThreads) {
            float val = gq * ex2((elem_value(x, v) - mx) * c);
            if (v == cf.t0) val -= cf.c0;
            if (v == cf.t1) val -= cf.c1;
            for (int k = 0; k < nkl; ++k)
                if (v == kl->tok[k]) val += kl->coef[k];
            if constexpr (sizeof(G) == 2)
                g[v] = __float2bfloat16_rn(val);
            else
                g[v] = val;
        }
    }
}

// Gradient of chunks [c0, c1) of row r (warp level, through the ring; the
// streaming warps of the fused kernel).  Same arithmetic as grad_pass_range.
// KL: the row has top-K terms (VSD (KL)) in kl; without them the loop is the
// plain one.
template <typename T, bool VEC, typename G, bool KL = false>
__device__ void stream_grad(Ring* rg, const Problem<T>& P, int r, int c0, int c1, G* grad,
                            const KlRec* kl = nullptr) {
    constexpr int PV = Traits<T>::kPerVec;
    constexpr int CE = chunk_elems<T>();
    const int64_t V = P.V;
    if constexpr (!VEC) {
        grad_pass_range<T, VEC, G>(P, r, (int64_t)c0 * CE, min(V, (int64_t)c1 * CE), P.rstats,
                                   grad, kl);
    } else {
        constexpr int NP = PV / 2;
        const int lane = threadIdx.x & 31;
        const T* x = P.draft + (int64_t)r * V;
        G* g = grad + (int64_t)r * V;
        const RowRec rec = ld_cg(P.rows + r);
        const Coef cf = ld_cg(P.coef + r);
        const float c = P.ts.c;
        const float gq = cf.g * rec.izx;  // g / Z
        const uint64_t pol = policy_evict_first();
        const uint64_t mx2 = f2(rec.mx, rec.mx), c2 = f2(c, c), gq2 = f2(gq, gq);
        const int nkl = KL ? min(max(kl->n, 0), kMaxKlTop) : 0;
        // VSD (KL): which of the row's top-K terms fall in chunk ch (a
        // warp-uniform mask; called where the warp is converged)
        auto kl_mask = [&](int ch) -> unsigned {
            if (!KL || !nkl) return 0u;
            const bool in = lane < nkl && (unsigned)(kl->tok[lane] - ch * CE) < (unsigned)CE;
            return __ballot_sync(0xffffffffu, in);
        };
        // the sparse terms touch at most two positions of the row, plus the
        // top-K terms of the chunk
        auto emit = [&](int64_t v0, float (&o)[PV], unsigned km) {
            if ((uint64_t)(cf.t0 - v0) < (uint64_t)PV) {
#pragma unroll
                for (int e = 0; e < PV; ++e)
                    if (v0 + e == cf.t0) o[e] -= cf.c0;
            }
            if ((uint64_t)(cf.t1 - v0) < (uint64_t)PV) {
#pragma unroll
                for (int e = 0; e < PV; ++e)
                    if (v0 + e == cf.t1) o[e] -= cf.c1;
            }
            for (unsigned m = KL ? km : 0u; m; m &= m - 1) {
                const int k = __ffs(m) - 1;
                const int t = kl->tok[k];
                if ((uint64_t)(t - v0) < (uint64_t)PV) {
                    const float ck = kl->coef[k];
#pragma unroll
                    for (int e = 0; e < PV; ++e)
                        if (v0 + e == t) o[e] += ck;
                }
            }
            grad_store<T, G, PV>(g, v0, o, pol);
        };
        if (cf.g == 0.f && isfinite(rec.mx)) {
            // No dense part: g q(v) is +0 for every mass in [0, 1], so the
            // draft row is not read (rows no objective term reaches).
            const int warp = threadIdx.x >> 5;
            for (int ch = c0 + warp; ch < c1; ch += kWarps) {
                const unsigned km = kl_mask(ch);
#pragma unroll
                for (int k = 0; k < kLoads; ++k) {
                    const int64_t v0 = (int64_t)ch * CE + (int64_t)k * 32 * PV + lane * PV;
                    if (v0 >= V) break;
                    float o[PV];
#pragma unroll
                    for (int e = 0; e < PV; ++e) o[e] = 0.f;
                    emit(v0, o, km);
                }
            }
            return;
        }
        ring_stream<T, false>(
            rg, x, nullptr, V, c0, c1, pol, pol, P.status,
            [&](int ch, const uint4 (&bx)[kLoads], const uint4 (&)[kLoads]) {
                const unsigned km = kl_mask(ch);
#pragma unroll
                for (int k = 0; k < kLoads; ++k) {
                    const int64_t v0 = (int64_t)ch * CE + (int64_t)k * 32 * PV + lane * PV;
                    if (v0 >= V) break;
                    uint64_t pr[NP];
                    vec_pairs<T>(bx[k], pr);
                    float o[PV];
#pragma unroll
                    for (int q = 0; q < NP; ++q)
                        f2split(f2mul(f2_mass(pr[q], mx2, c2), gq2), o[2 * q], o[2 * q + 1]);
                    emit(v0, o, km);
                }
            });
    }
}

template <typename T, bool VEC, typename G>
__device__ void grad_pass(const Problem<T>& P, int r, const float4* rstats, G* grad) {
    grad_pass_range<T, VEC, G>(P, r, 0, P.V, rstats, grad);
}

// --------------------------------------------------------------- tree pass
struct TreeShared {
    int bad, deepest, maxdepth;
    unsigned char acc[1024], pacc[1024], hasrej[1024];
    int par[1024];
    int depth[1024];
    float la[1024];
    double lk[1024];
};

// The children of node u of tree b at row u (block, right after the row's
// pass, while the row is still in L2): alpha, the accept bit (Eq. 1) and log
// alpha of each child's token, for the per-node pass; and the row's
// statistics output.
template <typename T>
__device__ void tree_children(const Problem<T>& P, int b, int u) {
    const int N = P.N;
    const int64_t V = P.V;
    const int n0 = b * N, r = n0 + u;
    const int32_t* par = P.parent + (int64_t)n0;
    const vsd_tree_outputs& o = P.tout;
    if (threadIdx.x == 0 && o.row_stats)
        reinterpret_cast<float4*>(o.row_stats)[r] = ld_cg(P.rstats + r);
    for (int n = u + 1 + threadIdx.x; n < N; n += kThreads) {
        if (__ldg(par + n) != u) continue;
        const RowRec rec = ld_cg(P.rows + r);
        const int tok = __ldg(P.given_tokens + n0 + n);
        float la = -INFINITY;
        if (tok < 0 || tok >= V) {
            atomicOr(P.status, VSD_STATUS_BAD_TOKEN);
        } else if (!rec.flags) {
            float lq;
            token_logs(P.draft + (int64_t)r * V, P.target + (int64_t)r * V, tok, rec,
                       P.ts.invTd, &lq, &la);
        }
        const float a = expf(la);
        const bool acc = la > -INFINITY && __ldg(P.u_accept + n0 + n) <= a;
        o.alpha[n0 + n] = a;
        o.accept[n0 + n] = acc ? 1 : 0;
        P.tla[n0 + n] = la;
    }
}

// Tree verification, one draft tree b of N nodes per block; rows of tree b
// are b*N .. b*N + N - 1, row n is the distribution node n's children were
// drafted from (App. E tree).  This pass:
//   1. every node, in parallel: alpha and the accept bit of its token against
//      its parent's row (Eq. 1);
//   2. in node order (parents come first): the accepted-path bit and the
//      depth; then log kappa level by level (each node adds its log alpha to
//      its parent's); the deepest accepted node;
//   3. the list of residual rows (accepted nodes with a rejected child) for
//      tree_residual_row, in tlist[b*N ..], its length in tcount[b]; the first
//      child of the deepest accepted node (or -1) in tlist[b*N + N - 1], a
//      slot the list never reaches (node N - 1 has no children).
template <typename T>
__device__ void tree_nodes(const Problem<T>& P, int b, TreeShared& sh) {
    const int N = P.N;
    const int n0 = b * N;
    const int32_t* par = P.parent + (int64_t)n0;
    const vsd_tree_outputs& o = P.tout;
    // parents into shared memory; a tree is valid if node 0 is the root and
    // every other node's parent precedes it
    int badl = 0;
    for (int n = threadIdx.x; n < N; n += kThreads) {
        const int pn = __ldg(par + n);
        sh.par[n] = pn;
        badl |= n == 0 ? pn != -1 : (pn < 0 || pn >= n);
    }
    const int bad = __syncthreads_or(badl);
    if (bad) {
        if (threadIdx.x == 0) atomicOr(P.status, VSD_STATUS_BAD_TREE);
        for (int n = threadIdx.x; n < N; n += kThreads) {
            o.alpha[n0 + n] = 0.f;
            o.accept[n0 + n] = 0;
            o.path_accept[n0 + n] = 0;
            o.logkappa[n0 + n] = -INFINITY;
            o.corr_tokens[n0 + n] = -1;
        }
        if (threadIdx.x == 0) {
            o.deepest[b] = -1;
            o.accept_len[b] = -1;
            o.bonus[b] = -1;
            P.tcount[b] = 0;
        }
        return;
    }
    // 1. per node: log alpha and the accept bit from the parents' row blocks
    for (int n = threadIdx.x; n < N; n += kThreads) {
        sh.la[n] = n > 0 ? ld_cg(P.tla + n0 + n) : 0.f;
        sh.acc[n] = n > 0 ? ld_cg(o.accept + n0 + n) : 1;
        sh.hasrej[n] = 0;
    }
    __syncthreads();
    // 2. accepted-path bits, depths, the deepest accepted node
    if (threadIdx.x == 0) {
        sh.pacc[0] = 1;
        sh.depth[0] = 0;
        sh.lk[0] = 0.0;
        int deepest = 0, maxd = 0;
        for (int n = 1; n < N; ++n) {
            const int pn = sh.par[n];
            sh.pacc[n] = (unsigned char)(sh.acc[n] && sh.pacc[pn]);
            sh.depth[n] = sh.depth[pn] + 1;
            maxd = max(maxd, sh.depth[n]);
            if (sh.pacc[n] && sh.depth[n] > sh.depth[deepest]) deepest = n;
        }
        sh.deepest = deepest;
        sh.maxdepth = maxd;
        int first = -1;
        for (int n = deepest + 1; n < N && first < 0; ++n)
            if (sh.par[n] == deepest) first = n;
        P.tlist[n0 + N - 1] = first;
        o.alpha[n0] = 1.f;
        o.accept[n0] = 1;
        o.path_accept[n0] = 1;
        o.logkappa[n0] = 0.f;
        o.corr_tokens[n0] = -1;
        o.deepest[b] = deepest;
        o.accept_len[b] = sh.depth[deepest];
    }
    __syncthreads();
    for (int L = 1; L <= sh.maxdepth; ++L) {  // log kappa along each branch (Eq. 2)
        for (int n = threadIdx.x; n < N; n += kThreads)
            if (sh.depth[n] == L) sh.lk[n] = sh.lk[sh.par[n]] + (double)sh.la[n];
        __syncthreads();
    }
    for (int n = 1 + threadIdx.x; n < N; n += kThreads) {
        o.path_accept[n0 + n] = sh.pacc[n];
        o.logkappa[n0 + n] = (float)sh.lk[n];
        o.corr_tokens[n0 + n] = -1;
        const int pn = sh.par[n];
        if (sh.pacc[pn] && !sh.pacc[n]) sh.hasrej[pn] = 1;
    }
    __syncthreads();
    // 3. the residual rows, in node order
    if (threadIdx.x == 0) {
        int k = 0;
        for (int u = 0; u < N; ++u)
            if (sh.pacc[u] && sh.hasrej[u]) P.tlist[n0 + k++] = u;
        P.tcount[b] = k;
    }
}

// Residual row of node u of tree b (block): stream the row's residual
// max(0, p - q) (Sec. 3) and draw each rejected child's token with the
// child's own uniform; if the residual has no mass, a draw from p instead.
template <typename T, bool VEC>
__device__ void tree_residual_row(const Problem<T>& P, int b, int u, Ring* rg, float4* tab,
                                  int* s_tok) {
    const int N = P.N;
    const int64_t V = P.V;
    const int n0 = b * N;
    const int nch = P.nch;
    const int32_t* par = P.parent + (int64_t)n0;
    const vsd_tree_outputs& o = P.tout;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const float c = P.ts.c;
    const uint64_t pol = policy_evict_normal();
    const int r = n0 + u;
    const RowRec rec = ld_cg(P.rows + r);
    if (rec.flags) return;
    const T* x = P.draft + (int64_t)r * V;
    const T* y = P.target + (int64_t)r * V;
    const MassRes mr{rec.mx, rec.my, rec.izx, rec.izy, c};
    stream_residual<T, VEC>(rg, x, y, V, 0, nch, tab, mr, P.status);
    __syncthreads();
    {  // every warp computes the total; the rejected children are shared out
        const TableSum Rt = table_sum(tab, nch, 0, 0.f, c, lane);
        if (threadIdx.x == 0) *s_tok = Rt.Z > 0.0;
        int k = 0;
        if (Rt.Z > 0.0)
            for (int n = u + 1; n < N; ++n) {
                if (__ldg(par + n) != u || ld_cg(o.path_accept + n0 + n)) continue;
                if (k++ % kWarps != warp) continue;
                const Located loc =
                    table_locate(tab, nch, 0, 0.f, c, Rt, __ldg(P.u_correct + n0 + n), lane);
                int tok = -1;
                if (loc.ch >= 0)
                    tok = warp_rescan<T, VEC, true, true>(x, y, V, loc.ch, loc.tc, mr, lane, pol);
                if (lane == 0) o.corr_tokens[n0 + n] = tok < V ? tok : -1;
            }
    }
    __syncthreads();
    if (!*s_tok) {  // no residual mass: each rejected child draws from p
        stream_tables<T, VEC, false>(rg, y, nullptr, V, 0, nch, tab, c, pol, pol, P.status);
        __syncthreads();
        const float M = table_max(tab, nch, 0, lane);
        const TableSum S = table_sum(tab, nch, 0, frame_of(M), c, lane);
        int k = 0;
        for (int n = u + 1; n < N; ++n) {
            if (__ldg(par + n) != u || ld_cg(o.path_accept + n0 + n)) continue;
            if (k++ % kWarps != warp) continue;
            const int tok = row_ok(M, S.Z)
                                ? warp_sample<T, VEC>(y, nullptr, V, tab, nch, 0, M, S,
                                                      __ldg(P.u_correct + n0 + n), c, lane, pol)
                                : -1;
            if (lane == 0) o.corr_tokens[n0 + n] = tok < V ? tok : -1;
        }
    }
    __syncthreads();
}

// The bonus token of tree b: the residual (or p) draw of the deepest accepted
// node's first child, or, at a leaf, the p-draw at its row (one thread).
template <typename T>
__device__ void tree_bonus(const Problem<T>& P, int b) {
    const int N = P.N;
    const int n0 = b * N;
    const vsd_tree_outputs& o = P.tout;
    const int best = ld_cg(o.deepest + b);
    if (best < 0) return;  // invalid tree: already written
    const int child = ld_cg(P.tlist + n0 + N - 1);
    o.bonus[b] = child >= 0 ? ld_cg(o.corr_tokens + n0 + child) : ld_cg(P.rows + n0 + best).ps;
}

}  // namespace vsd
