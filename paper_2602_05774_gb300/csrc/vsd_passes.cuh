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
//   tree_pass    per draft tree: acceptance per node at its parent's row, the
//                AND-scan along parent pointers, log kappa, residual draws at
//                the parents of first-rejected nodes, deepest node, bonus.
#pragma once

#include "vsd_common.cuh"

namespace vsd {

// --------------------------------------------------------------- records
struct __align__(16) RowRec {  // one logit row after row_pass (workspace)
    double lzx, lzy;         // ln sum_v exp((v - max)/T) of the q and p rows
    float mx, my;            // row maxima (exact input values)
    int tok;                 // z~ (drawn from q, or given); -1 if none
    float lq_tok, la_tok;    // log q(z~), log alpha(z~) = min(0, log p - log q)
    int ps;                  // draw from p with u_correct
    float lq_ps, la_ps;
    int ref;                 // argmax of the target row
    float la_ref;
    int flags;               // 1: invalid row, 2: invalid given token
};
static_assert(sizeof(RowRec) == 64, "RowRec layout");

struct __align__(16) Coef {     // grad[v] = g q(v) - c0 [v == t0] - c1 [v == t1]
    float g;
    int t0;
    float c0;
    int t1;
    float c1;
    float pad0, pad1, pad2;
};
static_assert(sizeof(Coef) == 32, "Coef layout");

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
    int zeta_mode;
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
    float4* gtab;                 // [R][nch_ws] per-chunk tables of each row
    int* row_seg_cnt;             // [R] segments of a row completed
    int* res_seg_cnt;             // [B*K] residual segments of a path completed
    int* path_A;                  // [B*K] accepted length of a path
    int* resq;                    // [B*K*nseg] residual segment items (path*nseg + seg)
    int* resq_flag;               // [B*K*nseg] item written
    int* resq_head;               // next item to take
    int* resq_tail;               // next free slot
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
// involved.  pos[w] counts the chunks warp w has consumed (slot = pos %
// kStages, barrier phase = (pos / kStages) & 1) and persists across rows.
struct Ring {
    uint4 data[kWarps][kStages][2][kLoads * 32];
    uint64_t bar[kWarps][kStages];
    int pos[kWarps];
    int broken[kWarps];  // a wait ran out: no further waits or copies in this block
};

__device__ __forceinline__ void ring_init(Ring* rg) {
    if ((threadIdx.x & 31) == 0) {
        const int w = threadIdx.x >> 5;
        for (int st = 0; st < kStages; ++st) mbar_init(&rg->bar[w][st], 1);
        rg->pos[w] = 0;
        rg->broken[w] = 0;
        mbar_init_fence();
    }
    __syncthreads();
}

// Bounded wait on a slot; false (and the timeout status bit) if it ran out.
__device__ __forceinline__ bool ring_wait(uint64_t* bar, uint32_t parity, int* status) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    for (;;) {
        if (mbar_try_wait(bar, parity)) return true;
        if (global_timer_ns() - t0 > 2000000000ull) {
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
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nrange = ch1 - ch0;
    const int nj = nrange > warp ? (nrange - warp + kWarps - 1) / kWarps : 0;
    const int pos = rg->pos[warp];
    bool broken = rg->broken[warp] != 0;
    auto issue = [&](int j) {
        const int ch = ch0 + warp + j * kWarps;
        const int slot = (pos + j) % kStages;
        const int64_t e0 = (int64_t)ch * CE;
        const int64_t ne = V - e0 < CE ? V - e0 : CE;
        const uint32_t bytes = (uint32_t)(ne * (int64_t)sizeof(T));
        uint64_t* bar = &rg->bar[warp][slot];
        fence_proxy_async();
        mbar_expect_tx(bar, HAS_Y ? 2 * bytes : bytes);
        bulk_g2s(rg->data[warp][slot][0], x + e0, bytes, bar, polx);
        if (HAS_Y) bulk_g2s(rg->data[warp][slot][1], y + e0, bytes, bar, poly);
    };
    if (lane == 0)
        for (int j = 0; j < nj && j < kStages; ++j) issue(j);
    for (int j = 0; j < nj; ++j) {
        const int slot = (pos + j) % kStages;
        const uint32_t parity = (uint32_t)((pos + j) / kStages) & 1u;
        bool ok = broken ? false : ring_wait(&rg->bar[warp][slot], parity, status);
        broken = __any_sync(0xffffffffu, !ok);
        const int ch = ch0 + warp + j * kWarps;
        const int64_t e0 = (int64_t)ch * CE;
        uint4 bx[kLoads], by[kLoads];
        if (e0 + CE <= V) {  // full chunk (all but possibly the row's last)
#pragma unroll
            for (int k = 0; k < kLoads; ++k) {
                bx[k] = rg->data[warp][slot][0][k * 32 + lane];
                if (HAS_Y) by[k] = rg->data[warp][slot][1][k * 32 + lane];
            }
        } else {
#pragma unroll
            for (int k = 0; k < kLoads; ++k) {
                const bool in = e0 + (int64_t)k * 32 * PV + lane * PV < V;
                const uint4 ninf = make_uint4(Traits<T>::kNegInf, Traits<T>::kNegInf,
                                              Traits<T>::kNegInf, Traits<T>::kNegInf);
                bx[k] = in ? rg->data[warp][slot][0][k * 32 + lane] : ninf;
                if (HAS_Y) by[k] = in ? rg->data[warp][slot][1][k * 32 + lane] : ninf;
            }
        }
        __syncwarp();
        if (lane == 0 && !broken && j + kStages < nj) issue(j + kStages);
        consume(ch, bx, by);
    }
    __syncwarp();
    if (lane == 0) {
        rg->pos[warp] = pos + nj;
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

__device__ __forceinline__ float2 tab_ms(const float4& t, int comp) {
    return comp == 0 ? make_float2(t.x, t.y) : make_float2(t.z, t.w);
}

// Row max over the table (warp).
__device__ __forceinline__ float table_max(const float4* tab, int nch, int comp, int lane) {
    float M = -INFINITY;
    for (int ch = lane; ch < nch; ch += 32) M = fmaxf(M, tab_ms(tab[ch], comp).x);
    return warp_max(M);
}

// Weight of chunk ch in the row frame Mm: s_c 2^{(m_c - Mm) c}.
__device__ __forceinline__ double chunk_weight(const float4* tab, int ch, int comp, float Mm,
                                               float c, float* scale_out) {
    const float2 ms = tab_ms(tab[ch], comp);
    const float sc = ex2((frame_of(ms.x) - Mm) * c);
    if (scale_out) *scale_out = sc;
    return (double)ms.y * (double)sc;
}

// Sum of the chunk weights in a fixed order (groups of 32 chunks, warp scan).
__device__ __forceinline__ double table_total(const float4* tab, int nch, int comp, float Mm,
                                              float c, int lane) {
    double base = 0.0;
    for (int g = 0; g < nch; g += 32) {
        const int ch = g + lane;
        const double w = ch < nch ? chunk_weight(tab, ch, comp, Mm, c, nullptr) : 0.0;
        const double inc = warp_incl_scan(w, lane);
        base += __shfl_sync(0xffffffffu, inc, 31);
    }
    return base;
}

// Find the chunk where the running weight first exceeds t (same order and
// arithmetic as table_total).  Returns the chunk and the threshold in that
// chunk's own frame; if no chunk crosses (rounding), the last chunk with
// weight and an infinite threshold (the rescan then takes its last token
// with mass).
struct Located { int ch; double tc; };
__device__ __forceinline__ Located table_locate(const float4* tab, int nch, int comp, float Mm,
                                                float c, double t, int lane) {
    double base = 0.0;
    int last = -1;
    for (int g = 0; g < nch; g += 32) {
        const int ch = g + lane;
        float sc = 1.f;
        const double w = ch < nch ? chunk_weight(tab, ch, comp, Mm, c, &sc) : 0.0;
        const double inc = warp_incl_scan(w, lane);
        const unsigned hit = __ballot_sync(0xffffffffu, ch < nch && base + inc > t);
        const unsigned pos = __ballot_sync(0xffffffffu, ch < nch && w > 0.0);
        if (hit) {
            const int L = __ffs(hit) - 1;
            const double before = __shfl_sync(0xffffffffu, base + inc - w, L);
            const float scL = __shfl_sync(0xffffffffu, sc, L);
            return Located{g + L, (t - before) / (double)scL};
        }
        if (pos) last = g + 31 - __clz(pos);
        base += __shfl_sync(0xffffffffu, inc, 31);
    }
    return Located{last, INFINITY};
}

// Scan chunk ch in token order and return the first token of positive mass
// whose running mass exceeds tc (the chunk-frame threshold); if none does,
// the last token with mass; -1 if the chunk has no mass.  Only tokens of
// positive mass can be returned, so masked positions (at or beyond V) never
// are.  mass(fx, fy) gives a token's mass.
template <typename T, bool VEC, bool NEED_X, bool NEED_Y, class Mass>
__device__ __forceinline__ int warp_rescan(const T* x, const T* y, int64_t V, int ch, double tc,
                                           const Mass& mass, int lane, uint64_t pol) {
    constexpr int PV = Traits<T>::kPerVec;
    uint4 bx[kLoads], by[kLoads];
    if (NEED_X) load_chunk<T, VEC>(x, V, ch, lane, pol, bx);
    if (NEED_Y) load_chunk<T, VEC>(y, V, ch, lane, pol, by);
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
            if (epos < 0 && m[e] > 0.f && (double)acc > tc) epos = e;
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
// Z is the table total; returns the token (or -1 if the row has no mass).
template <typename T, bool VEC>
__device__ __forceinline__ int warp_sample(const T* x, const T* y, int64_t V, const float4* tab,
                                           int nch, int comp, float M, double Z, float u,
                                           float c, int lane, uint64_t pol) {
    const float Mm = frame_of(M);
    const double t = (double)u * Z;
    const Located loc = table_locate(tab, nch, comp, Mm, c, t, lane);
    if (loc.ch < 0) return -1;
    const float mm = frame_of(tab_ms(tab[loc.ch], comp).x);
    if (comp == 0)
        return warp_rescan<T, VEC, true, false>(x, y, V, loc.ch, loc.tc, MassX{mm, c}, lane, pol);
    return warp_rescan<T, VEC, false, true>(x, y, V, loc.ch, loc.tc, MassY{mm, c}, lane, pol);
}

// Lowest index whose target logit equals the row max M (warp).
template <typename T, bool VEC>
__device__ __forceinline__ int warp_first_max(const T* y, int64_t V, const float4* tab, int nch,
                                              float M, int lane, uint64_t pol) {
    int ch = -1;
    for (int g = 0; g < nch && ch < 0; g += 32) {
        const int cc = g + lane;
        const unsigned hit = __ballot_sync(0xffffffffu, cc < nch && tab[cc].z == M);
        if (hit) ch = g + __ffs(hit) - 1;
    }
    if (ch < 0) return -1;
    constexpr int PV = Traits<T>::kPerVec;
    uint4 by[kLoads];
    load_chunk<T, VEC>(y, V, ch, lane, pol, by);
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

__device__ __forceinline__ bool row_ok(float M, double Z) {
    return M > -INFINITY && M < INFINITY && Z > 0.0 && Z < INFINITY;
}

// log q and log alpha = min(0, log p - log q) of token v (Eq. 1), in double.
template <typename T>
__device__ __forceinline__ void token_logs(const T* x, const T* y, int v, const RowRec& rec,
                                           double invT, float* lq, float* la) {
    const double lqd = ((double)elem_value(x, v) - (double)rec.mx) * invT - rec.lzx;
    const double lpd = ((double)elem_value(y, v) - (double)rec.my) * invT - rec.lzy;
    const double d = lpd - lqd;
    *lq = (float)lqd;
    *la = (float)(d >= 0.0 ? 0.0 : d);
}

// --------------------------------------------------------------- row pass
struct RowShared {
    float Mx, My;
    double Zx, Zy, lzx, lzy;
    int tok, ps, ref;
    float lq[3], la[3];
};

enum XMode { kNoToken = 0, kSampleToken = 1, kGivenToken = 2 };

// The per-row work once the row's chunk table tab[0..nch) is complete in
// shared memory (block): row statistics, the draws, the argmax, the token
// log-probabilities; writes rows[r] and rstats[r].
template <typename T, bool VEC, bool HAS_Y, int XMODE, bool ARGMAX>
__device__ void row_tail(const Problem<T>& P, int r, const float4* tab, RowShared& sh) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t V = P.V;
    const T* x = P.draft + (int64_t)r * V;
    const T* y = HAS_Y ? P.target + (int64_t)r * V : nullptr;
    const float c = P.ts.c;
    const uint64_t pol = policy_evict_normal();
    if (warp == 0) {
        const float M = table_max(tab, P.nch, 0, lane);
        const double Z = table_total(tab, P.nch, 0, frame_of(M), c, lane);
        int tok = -1;
        if (XMODE == kSampleToken) {
            if (row_ok(M, Z))
                tok = warp_sample<T, VEC>(x, y, V, tab, P.nch, 0, M, Z, __ldg(P.u_draft + r), c,
                                          lane, pol);
        } else if (XMODE == kGivenToken) {
            tok = __ldg(P.given_tokens + r);
        }
        if (XMODE == kSampleToken && (tok < 0 || tok >= V)) tok = -1;
        if (lane == 0) {
            sh.Mx = M;
            sh.Zx = Z;
            sh.lzx = row_ok(M, Z) ? log(Z) : 0.0;
            sh.tok = tok;
        }
    } else if (HAS_Y && warp == 1) {
        const float M = table_max(tab, P.nch, 1, lane);
        const double Z = table_total(tab, P.nch, 1, frame_of(M), c, lane);
        int ps = -1;
        if (row_ok(M, Z))
            ps = warp_sample<T, VEC>(x, y, V, tab, P.nch, 1, M, Z, __ldg(P.u_correct + r), c,
                                     lane, pol);
        if (ps >= V) ps = -1;
        if (lane == 0) {
            sh.My = M;
            sh.Zy = Z;
            sh.lzy = row_ok(M, Z) ? log(Z) : 0.0;
            sh.ps = ps;
        }
    } else if (HAS_Y && ARGMAX && warp == 2) {
        const float M = table_max(tab, P.nch, 1, lane);
        const int ref =
            (M > -INFINITY) ? warp_first_max<T, VEC>(y, V, tab, P.nch, M, lane, pol) : -1;
        if (lane == 0) sh.ref = ref < V ? ref : -1;
    }
    __syncthreads();
    // log q and log alpha of z~, of the p-draw and of the argmax: one lane each.
    const double invT = P.ts.invTd;
    const bool okx = row_ok(sh.Mx, sh.Zx);
    const bool oky = HAS_Y ? row_ok(sh.My, sh.Zy) : true;
    const bool ok = okx && oky;
    const int tok = XMODE == kNoToken ? -1 : sh.tok;
    const bool tok_ok = tok >= 0 && tok < V;
    if (threadIdx.x < 3) {
        const int which = threadIdx.x;
        const int v = which == 0 ? tok : (which == 1 ? sh.ps : sh.ref);
        float lq = -INFINITY, la = -INFINITY;
        const bool want = which == 0 || (HAS_Y && (which == 1 || ARGMAX));
        if (want && ok && v >= 0 && v < V) {
            RowRec tmp;
            tmp.mx = sh.Mx;
            tmp.lzx = sh.lzx;
            tmp.my = HAS_Y ? sh.My : 0.f;
            tmp.lzy = HAS_Y ? sh.lzy : 0.0;
            if (HAS_Y)
                token_logs(x, y, v, tmp, invT, &lq, &la);
            else
                lq = (float)(((double)elem_value(x, v) - (double)tmp.mx) * invT - tmp.lzx);
        }
        sh.lq[which] = lq;
        sh.la[which] = la;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        RowRec rec;
        rec.mx = sh.Mx;
        rec.lzx = okx ? sh.lzx : 0.0;
        rec.my = HAS_Y ? sh.My : 0.f;
        rec.lzy = (HAS_Y && oky) ? sh.lzy : 0.0;
        rec.flags = ok ? 0 : 1;
        if (!ok) atomicOr(P.status, VSD_STATUS_BAD_ROW);
        int t = tok;
        if (XMODE == kGivenToken && !tok_ok) {
            atomicOr(P.status, VSD_STATUS_BAD_TOKEN);
            t = -1;
            rec.flags |= 2;
        }
        rec.tok = t;
        rec.lq_tok = (ok && t >= 0) ? sh.lq[0] : -INFINITY;
        rec.la_tok = (ok && t >= 0) ? sh.la[0] : -INFINITY;
        rec.ps = (HAS_Y && ok) ? sh.ps : -1;
        rec.lq_ps = (HAS_Y && ok) ? sh.lq[1] : -INFINITY;
        rec.la_ps = (HAS_Y && ok) ? sh.la[1] : -INFINITY;
        rec.ref = (HAS_Y && ARGMAX && ok) ? sh.ref : -1;
        rec.la_ref = (HAS_Y && ARGMAX && ok) ? sh.la[2] : -INFINITY;
        P.rows[r] = rec;
        P.rstats[r] = make_float4(rec.mx, (float)rec.lzx, rec.my, (float)rec.lzy);
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
    const MassRes mr{rec.mx, rec.my, (float)exp(-rec.lzx), (float)exp(-rec.lzy), c};
    stream_residual<T, VEC>(rg, x, y, V, 0, P.nch, tab, mr, P.status);
    __syncthreads();
    if (warp == 0) {
        const double Rt = table_total(tab, P.nch, 0, 0.f, c, lane);
        int tok = -1;
        if (Rt > 0.0) {
            const Located loc = table_locate(tab, P.nch, 0, 0.f, c, (double)u * Rt, lane);
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

// Inverse-CDF draw from p at row r with uniform u (block; streams the target row).
template <typename T, bool VEC>
__device__ int p_draw(const Problem<T>& P, int r, float u, Ring* rg, float4* tab, int* out) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t V = P.V;
    const T* y = P.target + (int64_t)r * V;
    const float c = P.ts.c;
    const uint64_t pol = policy_evict_normal();
    stream_tables<T, VEC, false>(rg, y, nullptr, V, 0, P.nch, tab, c, pol, pol, P.status);
    __syncthreads();
    if (warp == 0) {
        const float M = table_max(tab, P.nch, 0, lane);
        const double Z = table_total(tab, P.nch, 0, frame_of(M), c, lane);
        const int tok = row_ok(M, Z) ? warp_sample<T, VEC>(y, nullptr, V, tab, P.nch, 0, M, Z, u,
                                                          c, lane, pol)
                                     : -1;
        if (lane == 0) *out = tok < V ? tok : -1;
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
// path_head (warp 0): the accepted length A (first rejection by ballot) and,
// if A < D, the record of row A.  Written to sh.A, sh.rec.
template <typename T>
__device__ void path_head(const Problem<T>& P, int path, PathShared& sh) {
    const int D = P.D;
    const int r0 = path * D;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (warp == 0) {
        int A = D;
        for (int d0 = 0; d0 < D; d0 += 32) {
            const int d = d0 + lane;
            bool rej = false;
            if (d < D) {
                const RowRec rec = ld_cg(P.rows + r0 + d);
                const double a = rec.flags ? 0.0 : exp((double)rec.la_tok);
                rej = rec.flags || !((double)__ldg(P.u_accept + r0 + d) <= a);
            }
            const unsigned bal = __ballot_sync(0xffffffffu, rej);
            if (bal && A == D) A = d0 + __ffs(bal) - 1;
        }
        if (lane == 0) {
            sh.A = A;
            if (A < D) sh.rec = ld_cg(P.rows + r0 + A);
        }
    }
}

// path_epilogue (warp 0): given A and the residual token at row A (-1: none
// or no residual mass), the corrected path, alpha', the log-kappa prefix sums
// of z~, z' and the reference (Eq. 2, warp scans), E[A] (Eq. 11); writes the
// E-step view and the requested outputs.
template <typename T>
__device__ void path_epilogue(const Problem<T>& P, int path, int A, int resid) {
    const int D = P.D;
    const int r0 = path * D;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (warp == 0) {
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
            double a = 0.0, tk = 0.0, tkc = 0.0, tkr = 0.0;
            bool acc = false;
            int zc = -1;
            float lqc = -INFINITY, lac = -INFINITY;
            if (act) {
                a = rec.flags ? 0.0 : exp((double)rec.la_tok);
                acc = !rec.flags && (double)__ldg(P.u_accept + r) <= a;
                if (d < A) {
                    zc = rec.tok; lqc = rec.lq_tok; lac = rec.la_tok;
                } else if (d == A) {
                    zc = resid >= 0 ? resid : rec.ps;  // no residual mass: draw from p (R10)
                    if (zc == rec.ps) {
                        lqc = rec.lq_ps; lac = rec.la_ps;
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
            EA += warp_sum(act ? exp(lk) : 0.0);  // Eq. 11
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
                if (o.alpha) o.alpha[r] = (float)a;
                if (o.accept) o.accept[r] = acc ? 1 : 0;
                if (o.corr_tokens) o.corr_tokens[r] = zc;
                if (o.logq_corr) o.logq_corr[r] = lqc;
                if (o.alpha_corr) o.alpha_corr[r] = zc >= 0 ? (float)exp((double)lac) : 0.f;
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
struct WeightsShared {
    double ot[256], op[256], lqt[256], lqc[256], cq[256];
    float ez[256];
    double red[kThreads];
    double w, cmax;
};

__device__ __forceinline__ double block_sum(double v, double* red) {
    red[threadIdx.x] = v;
    __syncthreads();
    for (int o = kThreads / 2; o; o >>= 1) {
        if (threadIdx.x < o) red[threadIdx.x] += red[threadIdx.x + o];
        __syncthreads();
    }
    const double r = red[0];
    __syncthreads();
    return r;
}

// M-step of prefix b (block; proposals s strided over the threads, K <= 256).
// Writes coef[] for the prefix's rows, the optional weights table and
// loss_out[b].  Arithmetic in double.
template <typename T>
__device__ void weights_pass(const Problem<T>& P, const EStepView& E, int b, float* weights_out,
                             float* loss_out, WeightsShared& sh) {
    const int K = P.K, D = P.D;
    double Jp = 0.0, Np = 0.0;
    for (int s = threadIdx.x; s < K; s += kThreads) sh.lqt[s] = sh.lqc[s] = 0.0;
    for (int d = 0; d < D; ++d) {
        if (threadIdx.x == 0) sh.w = pow(P.w_base, (double)(d + 1));  // w(l), App. F
        __syncthreads();
        const double w = sh.w;
        for (int s = threadIdx.x; s < K; s += kThreads) {
            const int r = (b * K + s) * D + d;
            const double lk = ld_cg(E.lk + r), lkc = ld_cg(E.lkc + r), lkr = ld_cg(E.lkr + r);
            sh.lqt[s] += (double)ld_cg(E.lq_tok + r);
            sh.lqc[s] += (double)ld_cg(E.lq_corr + r);
            // Algorithm 2 scores z~; Algorithm 1 keeps z~ if it passes, else z'.
            const double ot = (lk >= lkr) ? 1.0 : 0.0;
            sh.ot[s] = ot;
            sh.op[s] = ot > 0.0 ? w : ((lkc >= lkr) ? w : 0.0);
            sh.cq[s] = (P.zeta_mode == 0 ? exp(sh.lqt[s]) : sh.lqt[s]) / P.tau_car;
        }
        __syncthreads();
        if (threadIdx.x < 32) {  // max of the CAR logits over the K proposals
            double m = -INFINITY;
            for (int j = threadIdx.x; j < K; j += 32) m = fmax(m, sh.cq[j]);
#pragma unroll
            for (int o = 16; o; o >>= 1) m = fmax(m, __shfl_xor_sync(0xffffffffu, m, o));
            if (threadIdx.x == 0) sh.cmax = m;
        }
        __syncthreads();
        for (int s = threadIdx.x; s < K; s += kThreads) sh.ez[s] = expf((float)(sh.cq[s] - sh.cmax));
        __syncthreads();
        for (int s = threadIdx.x; s < K; s += kThreads) {
            double num = 0.0, den = 0.0, Zs = 0.0;
            for (int j = 0; j < K; ++j) {
                if (j != s) { num += sh.op[j] * sh.ot[j]; den += sh.op[j]; }
                Zs += (double)sh.ez[j];
            }
            const double beta = den > 0.0 ? num / den : 0.0;  // Eq. beta (leave-one-out)
            const double zeta = (double)sh.ez[s] / Zs;         // Eq. zeta
            const double ot = sh.ot[s], op = sh.op[s];
            const double lqz = ot > 0.0 ? sh.lqt[s] : sh.lqc[s];
            if (op != 0.0) Jp += op * (lqz - beta * zeta * sh.lqt[s]);  // Eq. advance
            Np += op;
            // per-l terms o'(o~ - beta zeta) and o'(1 - o~) of row (s, l-1)
            P.wscr[(b * K + s) * D + d] = make_double2(op * (ot - beta * zeta), op * (1.0 - ot));
            if (weights_out) {
                float4* wo = reinterpret_cast<float4*>(weights_out) + ((int64_t)b * D + d) * K + s;
                *wo = make_float4((float)ot, (float)op, (float)beta, (float)zeta);
            }
        }
        __syncthreads();
    }
    const double N = block_sum(Np, sh.red);
    const double J = block_sum(Jp, sh.red);
    const double scale = N > 0.0 ? 1.0 / ((double)P.B * N * P.ts.Td) : 0.0;
    for (int s = threadIdx.x; s < K; s += kThreads) {
        const int rbase = (b * K + s) * D;
        double c0 = 0.0, c1 = 0.0;
        for (int d = D - 1; d >= 0; --d) {
            const int r = rbase + d;
            const double2 tm = P.wscr[r];
            c0 += tm.x;
            c1 += tm.y;
            Coef cf;
            cf.t0 = ld_cg(E.tok + r);
            cf.t1 = ld_cg(E.corr + r);
            double k0 = c0 * scale, k1 = c1 * scale;
            if (cf.t1 == cf.t0) { k0 += k1; k1 = 0.0; cf.t1 = -1; }
            cf.g = (float)((c0 + c1) * scale);
            cf.c0 = (float)k0;
            cf.c1 = (float)k1;
            cf.pad0 = cf.pad1 = cf.pad2 = 0.f;
            P.coef[r] = cf;
        }
    }
    if (threadIdx.x == 0) loss_out[b] = (float)(N > 0.0 ? -J / N : 0.0);
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
                                const float4* rstats, G* grad) {
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
        for (int64_t v = e0 + threadIdx.x; v < e1; v += kThreads) {
            float val = gq * ex2((elem_value(x, v) - mx) * c);
            if (v == cf.t0) val -= cf.c0;
            if (v == cf.t1) val -= cf.c1;
            if constexpr (sizeof(G) == 2)
                g[v] = __float2bfloat16_rn(val);
            else
                g[v] = val;
        }
    }
}

template <typename T, bool VEC, typename G>
__device__ void grad_pass(const Problem<T>& P, int r, const float4* rstats, G* grad) {
    grad_pass_range<T, VEC, G>(P, r, 0, P.V, rstats, grad);
}

// --------------------------------------------------------------- tree pass
struct TreeShared {
    int bad, deepest, bonus, resid;
    double rt;
    RowRec rec;
    unsigned char pacc[1024];
    int depth[1024];
    double lk[1024];
};

// One draft tree per block; rows of tree b are b*N .. b*N + N - 1, row n is
// the distribution node n's children were drafted from (App. E tree).
template <typename T, bool VEC>
__device__ void tree_pass(const Problem<T>& P, int b, Ring* rg, float4* tab, TreeShared& sh) {
    const int N = P.N;
    const int64_t V = P.V;
    const int n0 = b * N;
    const int32_t* par = P.parent + (int64_t)n0;
    const vsd_tree_outputs& o = P.tout;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        int bad = (__ldg(par) != -1);
        for (int n = 1; n < N && !bad; ++n) {
            const int pn = __ldg(par + n);
            if (pn < 0 || pn >= n) bad = 1;
        }
        sh.bad = bad;
        if (bad) atomicOr(P.status, VSD_STATUS_BAD_TREE);
    }
    __syncthreads();
    if (o.row_stats)
        for (int n = threadIdx.x; n < N; n += kThreads)
            reinterpret_cast<float4*>(o.row_stats)[n0 + n] = ld_cg(P.rstats + n0 + n);
    if (sh.bad) {
        for (int n = threadIdx.x; n < N; n += kThreads) {
            o.alpha[n0 + n] = 0.f;
            o.accept[n0 + n] = 0;
            o.path_accept[n0 + n] = 0;
            o.logkappa[n0 + n] = -INFINITY;
            o.corr_tokens[n0 + n] = -1;
        }
        if (threadIdx.x == 0) { o.deepest[b] = -1; o.accept_len[b] = -1; o.bonus[b] = -1; }
        return;
    }
    if (threadIdx.x == 0) {
        o.alpha[n0] = 1.f; o.accept[n0] = 1; o.path_accept[n0] = 1; o.logkappa[n0] = 0.f;
        o.corr_tokens[n0] = -1;
        sh.pacc[0] = 1;
        sh.depth[0] = 0;
        double* lk = sh.lk;
        lk[0] = 0.0;
        int deepest = 0;
        for (int n = 1; n < N; ++n) {
            const int pn = __ldg(par + n);
            const RowRec rec = ld_cg(P.rows + n0 + pn);
            const int tok = __ldg(P.given_tokens + n0 + n);
            double la = -INFINITY;
            if (tok < 0 || tok >= V) {
                atomicOr(P.status, VSD_STATUS_BAD_TOKEN);
            } else if (!rec.flags) {
                float lq, laf;
                token_logs(P.draft + (int64_t)(n0 + pn) * V, P.target + (int64_t)(n0 + pn) * V,
                           tok, rec, P.ts.invTd, &lq, &laf);
                la = (double)laf;
            }
            const double a = exp(la);
            const bool acc = la > -INFINITY && (double)__ldg(P.u_accept + n0 + n) <= a;
            sh.pacc[n] = (unsigned char)(acc && sh.pacc[pn]);
            sh.depth[n] = sh.depth[pn] + 1;
            lk[n] = lk[pn] + la;
            o.alpha[n0 + n] = (float)a;
            o.accept[n0 + n] = acc ? 1 : 0;
            o.path_accept[n0 + n] = sh.pacc[n];
            o.logkappa[n0 + n] = (float)lk[n];
            o.corr_tokens[n0 + n] = -1;
            if (sh.pacc[n] && sh.depth[n] > sh.depth[deepest]) deepest = n;
        }
        sh.deepest = deepest;
    }
    __syncthreads();
    // Residual draws (Sec. 3): every node on an accepted path whose children
    // include rejected ones streams its row once; each rejected child then
    // draws with its own uniform.
    for (int u = 0; u < N; ++u) {
        if (!sh.pacc[u]) continue;
        int first = -1;
        for (int n = u + 1; n < N; ++n)
            if (__ldg(par + n) == u && !sh.pacc[n]) { first = n; break; }
        if (first < 0) continue;
        if (threadIdx.x == 0) sh.rec = ld_cg(P.rows + n0 + u);
        __syncthreads();
        if (sh.rec.flags) { __syncthreads(); continue; }
        const int r = n0 + u;
        const T* x = P.draft + (int64_t)r * V;
        const T* y = P.target + (int64_t)r * V;
        const float c = P.ts.c;
        const MassRes mr{sh.rec.mx, sh.rec.my, (float)exp(-sh.rec.lzx), (float)exp(-sh.rec.lzy),
                         c};
        stream_residual<T, VEC>(rg, x, y, V, 0, P.nch, tab, mr, P.status);
        __syncthreads();
        if (warp == 0) {
            const double Rt = table_total(tab, P.nch, 0, 0.f, c, lane);
            if (lane == 0) sh.rt = Rt;
            if (Rt > 0.0) {
                for (int n = first; n < N; ++n) {
                    if (__ldg(par + n) != u || sh.pacc[n]) continue;
                    const float un = __ldg(P.u_correct + n0 + n);
                    const Located loc =
                        table_locate(tab, P.nch, 0, 0.f, c, (double)un * Rt, lane);
                    int tok = -1;
                    if (loc.ch >= 0)
                        tok = warp_rescan<T, VEC, true, true>(x, y, V, loc.ch, loc.tc, mr, lane,
                                                              policy_evict_normal());
                    if (lane == 0) o.corr_tokens[n0 + n] = tok < V ? tok : -1;
                }
            }
        }
        __syncthreads();
        if (!(sh.rt > 0.0)) {
            // no residual mass: each rejected child draws from p (reading R10)
            for (int n = first; n < N; ++n) {
                if (__ldg(par + n) != u || sh.pacc[n]) continue;
                const int tok = p_draw<T, VEC>(P, r, __ldg(P.u_correct + n0 + n), rg, tab, &sh.resid);
                if (threadIdx.x == 0) o.corr_tokens[n0 + n] = tok;
            }
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        const int best = sh.deepest;
        o.deepest[b] = best;
        o.accept_len[b] = sh.depth[best];
        int bonus = -1;
        bool has_child = false;
        for (int n = best + 1; n < N; ++n)
            if (__ldg(par + n) == best) { bonus = o.corr_tokens[n0 + n]; has_child = true; break; }
        if (!has_child) bonus = ld_cg(P.rows + n0 + best).ps;  // leaf: p-draw at its row
        o.bonus[b] = bonus;
    }
}

}  // namespace vsd
