// vsd_api.cu -- the C ABI of include/vsd.h: argument checks, workspace layout
// and launch sequencing on the caller's stream.  Every compute step runs in
// the kernels of vsd_kernels_{f32,bf16}.cu; this file only marshals.
#include <math.h>
#include <stdlib.h>
#include <string.h>

#include <mutex>
#include <vector>

#include <cuda_runtime.h>

#include "vsd.h"
#include "vsd_launch.h"

namespace vsd {
namespace {

constexpr int kMaxV = 1 << 20;
constexpr int kMaxD = 64;
constexpr int kMaxK = 256;
constexpr int kMaxN = 1024;
constexpr int64_t kMaxRows = 1 << 24;
constexpr uint64_t kDefaultTimeoutNs = 2000000000ull;

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

struct WsLayout {
    size_t status, ticket, prefix_done, grad_head, resq_head, resq_tail, resq_avail;
    size_t path_cnt, prefix_cnt, ready, grad_cnt, row_seg_cnt, res_seg_cnt, resq_flag, zero_end;
    size_t rows, rstats, es_tok, es_corr, es_lq_tok, es_lq_corr, es_lk, es_lkc, es_lkr;
    size_t coef, wscr, path_A, resq, klr, gtab, tnode, tcoef, tg, tbad, bfac, total;
    int nch_ws, nseg_ws;
};

// Chunks per segment of the fused kernel's row and residual jobs, and of its
// gradient jobs.  Gradient jobs are cut finer: they need no follow-up step, and
// small ones let the last prefixes' gradients spread over every block instead
// of leaving most blocks idle at the end of the kernel.
#ifndef VSD_SEG_CHUNKS
#define VSD_SEG_CHUNKS 128
#endif
constexpr int kSegChunks = VSD_SEG_CHUNKS;
#ifndef VSD_GRAD_SEG_CHUNKS
#define VSD_GRAD_SEG_CHUNKS 16
#endif
constexpr int kGradSegChunks = VSD_GRAD_SEG_CHUNKS;
// Longest row (in chunks) whose tail the streaming warps run themselves.
#ifndef VSD_STREAM_TAIL_CHUNKS
#define VSD_STREAM_TAIL_CHUNKS 48
#endif
constexpr int kStreamTailChunks = VSD_STREAM_TAIL_CHUNKS;

// Upper bounds of the chunk count and segment count of a row over both logit
// dtypes (the smaller float32 chunk gives the larger count).
int chunks_upper(int V) { return (V + chunk_elems<float>() - 1) / chunk_elems<float>(); }

bool layout_ok(const vsd_layout& L) {
    if (L.B < 1 || L.V < 1 || L.V > kMaxV) return false;
    if (L.parent) {
        if (L.N < 1 || L.N > kMaxN) return false;
        if (L.tree_rule != VSD_TREE_INDEPENDENT && L.tree_rule != VSD_TREE_SEQUENTIAL)
            return false;
        return (int64_t)L.B * L.N <= kMaxRows;
    }
    if (L.K < 1 || L.K > kMaxK || L.D < 1 || L.D > kMaxD) return false;
    return (int64_t)L.B * L.K * L.D <= kMaxRows;
}

int64_t rows_of(const vsd_layout& L) {
    return L.parent ? (int64_t)L.B * L.N : (int64_t)L.B * L.K * L.D;
}

WsLayout ws_layout(const vsd_layout& L) {
    WsLayout w;
    const size_t R = (size_t)rows_of(L);
    const size_t npath = L.parent ? (size_t)L.B : (size_t)L.B * L.K;
    size_t o = 0;
    w.nch_ws = chunks_upper(L.V);
    w.nseg_ws = (w.nch_ws + kSegChunks - 1) / kSegChunks;
    const size_t nseg = (size_t)w.nseg_ws;
    // residual queue: segments of the paths' residual rows, or a tree's
    // residual rows (at most one per node)
    const size_t nq = L.parent ? R : npath * nseg;
    // hot counters on separate 256-byte lines (distinct L2 lines and slices)
    w.status = 0;
    w.ticket = 256;
    w.prefix_done = 512;
    w.grad_head = 768;
    w.resq_head = 1024;
    w.resq_tail = 1280;
    w.resq_avail = 1536;
    o = 1792;
    w.path_cnt = o; o = align256(o + 4 * npath);
    w.prefix_cnt = o; o = align256(o + 4 * (size_t)L.B);
    w.ready = o; o = align256(o + 4 * (size_t)L.B);
    w.grad_cnt = o; o = align256(o + 4 * (size_t)L.B);
    w.row_seg_cnt = o; o = align256(o + 4 * R);
    w.res_seg_cnt = o; o = align256(o + 4 * npath);
    w.resq_flag = o; o = align256(o + 4 * nq);
    w.zero_end = o;
    w.rows = o; o = align256(o + sizeof(RowRec) * R);
    w.rstats = o; o = align256(o + sizeof(float4) * R);
    w.es_tok = o; o = align256(o + 4 * R);
    w.es_corr = o; o = align256(o + 4 * R);
    w.es_lq_tok = o; o = align256(o + 4 * R);
    w.es_lq_corr = o; o = align256(o + 4 * R);
    w.es_lk = o; o = align256(o + 4 * R);
    w.es_lkc = o; o = align256(o + 4 * R);
    w.es_lkr = o; o = align256(o + 4 * R);
    w.coef = o; o = align256(o + sizeof(Coef) * R);
    w.wscr = o; o = align256(o + sizeof(double2) * R);
    w.path_A = o; o = align256(o + 4 * npath);
    w.resq = o; o = align256(o + 4 * nq);
    w.klr = o; o = align256(o + sizeof(KlRec) * R);
    w.gtab = o; o = align256(o + sizeof(float4) * R * (size_t)w.nch_ws);
    // trees: the node records, gradient terms and flags of the tree EM
    const size_t Rt = L.parent ? R : 0;
    w.tnode = o; o = align256(o + sizeof(TreeNodeRec) * Rt);
    w.tcoef = o; o = align256(o + sizeof(TreeCoef) * Rt);
    w.tg = o; o = align256(o + 4 * Rt);
    w.tbad = o; o = align256(o + (L.parent ? 4 * (size_t)L.B : 0));
    // linear layouts: the rows' packed factors of the LM head's backward
    w.bfac = o; o = align256(o + (L.parent ? 0 : lmhead_backward_fac_bytes((int)R)));
    w.total = o;
    return w;
}

template <typename U> U* at(void* ws, size_t off) {
    return reinterpret_cast<U*>(static_cast<char*>(ws) + off);
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

int num_sms() { return device_sm_count(); }

// T = 0 (greedy decoding) is served by the fused E-step + M-step, the LM
// head with it and the reference log kappa (greedy = true); the separate
// sampling, verification and M-step calls take T > 0.
vsd_status check_temperature(float T, bool greedy_ok = false) {
    if (T == 0.f) return greedy_ok ? VSD_OK : VSD_ERR_UNSUPPORTED;
    if (!(T > 0.f) || !isfinite(T)) return VSD_ERR_INVALID_ARG;
    return VSD_OK;
}

vsd_status check_ws(const vsd_layout& L, void* ws, size_t ws_bytes) {
    if (!ws) return VSD_ERR_WORKSPACE;
    if (!aligned16(ws)) return VSD_ERR_WORKSPACE;
    if (ws_bytes < ws_layout(L).total) return VSD_ERR_WORKSPACE;
    return VSD_OK;
}

vsd_status from_cuda(cudaError_t e) { return e == cudaSuccess ? VSD_OK : VSD_ERR_CUDA; }

vsd_params default_params(vsd_dtype dtype) {
    vsd_params p;
    p.w_base = 1.05;
    p.tau_car = 0.2;
    p.zeta_mode = 0;
    p.grad_dtype = dtype;
    p.wait_timeout_ns = kDefaultTimeoutNs;
    p.test_never_publish = 0;
    p.kl_weight = 0.0;
    p.kl_topk = 10;
    return p;
}

vsd_status check_params(const vsd_params& p) {
    if (!(p.w_base > 0.0) || !isfinite(p.w_base)) return VSD_ERR_INVALID_ARG;
    if (!(p.tau_car > 0.0)) return VSD_ERR_INVALID_ARG;  // +inf allowed: zeta = 1/K
    if (p.zeta_mode != 0 && p.zeta_mode != 1) return VSD_ERR_INVALID_ARG;
    if (p.grad_dtype != VSD_F32 && p.grad_dtype != VSD_BF16) return VSD_ERR_INVALID_ARG;
    if (!isfinite(p.kl_weight) || p.kl_weight < 0.0) return VSD_ERR_INVALID_ARG;
    if (p.kl_weight != 0.0 && (p.kl_topk < 1 || p.kl_topk > kMaxKlTop)) return VSD_ERR_INVALID_ARG;
    return VSD_OK;
}

// Fill the shape, temperature, workspace views of a problem.
// w(l) = w_base^l for l = 1 .. D, with the host's pow, and 1 / tau_car.
template <typename T>
void fill_wl(Problem<T>& P) {
    for (int d = 0; d < 64; ++d) {
        P.wl[d] = d < P.D ? pow(P.w_base, (double)(d + 1)) : 0.0;
        P.wlf[d] = (float)P.wl[d];
    }
    P.inv_tau = 1.0 / P.tau_car;
    P.inv_tau_f = (float)P.inv_tau;
}

template <typename T>
Problem<T> make_problem(const void* draft, const void* target, const vsd_layout& L, float T_,
                        void* ws) {
    Problem<T> P;
    memset(&P, 0, sizeof(P));
    P.draft = static_cast<const T*>(draft);
    P.target = static_cast<const T*>(target);
    P.B = L.B;
    P.K = L.parent ? 1 : L.K;
    P.D = L.parent ? 1 : L.D;
    P.N = L.parent ? L.N : 0;
    P.V = L.V;
    P.R = (int)rows_of(L);
    P.nch = (int)((L.V + chunk_elems<T>() - 1) / chunk_elems<T>());
    // T = 0: decisions by argmax, log q (and everything that uses it) at
    // temperature 1
    P.greedy = T_ == 0.f ? 1 : 0;
    const float Tq = T_ == 0.f ? 1.f : T_;
    P.ts.c = (float)(kLog2e / (double)Tq);
    P.ts.T = Tq;
    P.ts.Td = (double)Tq;
    P.ts.invTd = 1.0 / (double)Tq;
    P.parent = L.parent;
    P.w_base = 1.05;
    P.tau_car = 0.2;
    fill_wl(P);
    P.timeout_ns = kDefaultTimeoutNs;
    const WsLayout w = ws_layout(L);
    P.status = at<int>(ws, w.status);
    P.ticket = at<int>(ws, w.ticket);
    P.prefix_done = at<int>(ws, w.prefix_done);
    P.path_cnt = at<int>(ws, w.path_cnt);
    P.prefix_cnt = at<int>(ws, w.prefix_cnt);
    P.ready = at<int>(ws, w.ready);
    P.grad_cnt = at<int>(ws, w.grad_cnt);
    P.grad_head = at<int>(ws, w.grad_head);
    P.rows = at<RowRec>(ws, w.rows);
    P.rstats = at<float4>(ws, w.rstats);
    P.es.tok = at<int32_t>(ws, w.es_tok);
    P.es.corr = at<int32_t>(ws, w.es_corr);
    P.es.lq_tok = at<float>(ws, w.es_lq_tok);
    P.es.lq_corr = at<float>(ws, w.es_lq_corr);
    P.es.lk = at<float>(ws, w.es_lk);
    P.es.lkc = at<float>(ws, w.es_lkc);
    P.es.lkr = at<float>(ws, w.es_lkr);
    P.coef = at<Coef>(ws, w.coef);
    P.klr = at<KlRec>(ws, w.klr);
    P.wscr = at<double2>(ws, w.wscr);
    P.segc = kSegChunks;
    P.nseg = (P.nch + kSegChunks - 1) / kSegChunks;
    P.gsegc = kGradSegChunks;
    P.gnseg = (P.nch + kGradSegChunks - 1) / kGradSegChunks;
    P.nch_ws = w.nch_ws;
    P.gtab = at<float4>(ws, w.gtab);
    P.row_seg_cnt = at<int>(ws, w.row_seg_cnt);
    P.res_seg_cnt = at<int>(ws, w.res_seg_cnt);
    P.path_A = at<int>(ws, w.path_A);
    // the tree layout has no E-step view and no path lengths: their arrays
    // hold its residual lists and its nodes' log alpha
    P.stream_tails = 0;
    P.resq_sem = 1;
    P.tnode = L.parent ? at<TreeNodeRec>(ws, w.tnode) : nullptr;
    P.tcoef = L.parent ? at<TreeCoef>(ws, w.tcoef) : nullptr;
    P.tg = L.parent ? at<float>(ws, w.tg) : nullptr;
    P.tbad = L.parent ? at<int>(ws, w.tbad) : nullptr;
    P.tlist = at<int>(ws, w.es_tok);
    P.tcount = at<int>(ws, w.path_A);
    P.tla = at<float>(ws, w.es_lq_tok);
    P.resq = at<int>(ws, w.resq);
    P.resq_flag = at<int>(ws, w.resq_flag);
    P.resq_head = at<int>(ws, w.resq_head);
    P.resq_tail = at<int>(ws, w.resq_tail);
    P.resq_avail = at<int>(ws, w.resq_avail);
    return P;
}

template <typename T>
void set_params(Problem<T>& P, const vsd_params& p) {
    P.w_base = p.w_base;
    P.tau_car = p.tau_car;
    P.zeta_mode = p.zeta_mode;
    P.grad_bf16 = p.grad_dtype == VSD_BF16;
    P.timeout_ns = p.wait_timeout_ns ? p.wait_timeout_ns : kDefaultTimeoutNs;
    P.inject_wait_fault = p.test_never_publish;
    P.kl_weight = p.kl_weight;
    P.kl_topk = p.kl_weight != 0.0 ? p.kl_topk : 0;
    P.kl_scale = p.kl_weight / ((double)P.B * (double)P.K * P.ts.Td);
    fill_wl(P);
}

cudaError_t clear_counters(void* ws, const vsd_layout& L, cudaStream_t s) {
    return cudaMemsetAsync(ws, 0, ws_layout(L).zero_end, s);
}

bool vec_ok(const void* a, const void* b, const void* g, int V, size_t elem, size_t gelem) {
    if (!aligned16(a) || (b && !aligned16(b)) || (g && !aligned16(g))) return false;
    if (((size_t)V * elem) % 16 != 0) return false;
    if (g && ((size_t)V * gelem) % 16 != 0) return false;
    return true;
}


// ------------------------------------------------------------ per-device caches
std::mutex g_cache_mu;
struct SmemEntry { const void* kernel; int dev; size_t smem; };
struct OccEntry { const void* kernel; int dev; int threads; size_t smem; int blocks; };
std::vector<SmemEntry> g_smem;
std::vector<OccEntry> g_occ;
int g_sms[256];

}  // namespace

int device_sm_count() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 256) return 1;
    std::lock_guard<std::mutex> lock(g_cache_mu);
    if (g_sms[dev] == 0) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1)
            return 1;
        g_sms[dev] = n;
    }
    return g_sms[dev];
}

cudaError_t ensure_dyn_smem(const void* kernel, size_t smem) {
    if (smem == 0) return cudaSuccess;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(g_cache_mu);
    for (SmemEntry& x : g_smem)
        if (x.kernel == kernel && x.dev == dev) {
            if (x.smem >= smem) return cudaSuccess;
            e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            if (e == cudaSuccess) x.smem = smem;
            return e;
        }
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e == cudaSuccess) g_smem.push_back(SmemEntry{kernel, dev, smem});
    return e;
}

int blocks_per_sm(const void* kernel, int threads, size_t smem) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    {
        std::lock_guard<std::mutex> lock(g_cache_mu);
        for (const OccEntry& x : g_occ)
            if (x.kernel == kernel && x.dev == dev && x.threads == threads && x.smem == smem)
                return x.blocks;
    }
    if (ensure_dyn_smem(kernel, smem) != cudaSuccess) return 0;
    int n = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kernel, threads, smem) != cudaSuccess)
        return 0;
    std::lock_guard<std::mutex> lock(g_cache_mu);
    g_occ.push_back(OccEntry{kernel, dev, threads, smem, n});
    return n;
}

namespace {

// ------------------------------------------------------------ entry bodies
template <typename T>
vsd_status sample_impl(const void* draft, vsd_layout L, float T_, const float* u_draft,
                       int32_t* tokens, float* logq_tok, float* row_stats, void* ws,
                       cudaStream_t s) {
    Problem<T> P = make_problem<T>(draft, nullptr, L, T_, ws);
    P.u_draft = u_draft;
    P.out.tokens = tokens;
    P.out.logq_tok = logq_tok;
    P.out.row_stats = row_stats;
    const bool vec = vec_ok(draft, nullptr, nullptr, L.V, sizeof(T), 0);
    cudaError_t e = clear_counters(ws, L, s);
    if (e == cudaSuccess) e = Launch<T>::sample(P, vec, s);
    return from_cuda(e);
}

template <typename T>
vsd_status verify_impl(const void* draft, const void* target, vsd_layout L, float T_,
                       const int32_t* tokens, const float* u_accept, const float* u_correct,
                       const float* ref_logkappa, vsd_linear_outputs* out,
                       vsd_tree_outputs* tout, void* ws, cudaStream_t s) {
    Problem<T> P = make_problem<T>(draft, target, L, T_, ws);
    P.given_tokens = tokens;
    P.u_accept = u_accept;
    P.u_correct = u_correct;
    P.ref_logkappa = ref_logkappa;
    const bool vec = vec_ok(draft, target, nullptr, L.V, sizeof(T), 0);
    cudaError_t e = clear_counters(ws, L, s);
    if (L.parent) {
        P.tout = *tout;
        if (e == cudaSuccess)
            e = L.tree_rule == VSD_TREE_SEQUENTIAL ? Launch<T>::tree_seq(P, vec, s)
                                                   : Launch<T>::tree(P, vec, s);
    } else {
        P.out = *out;
        if (e == cudaSuccess) e = Launch<T>::rows_verify(P, vec, s);
        if (e == cudaSuccess) e = Launch<T>::paths(P, vec, s);
    }
    return from_cuda(e);
}

template <typename T>
vsd_status loss_impl(const void* draft, vsd_layout L, float T_, const vsd_linear_outputs* es,
                     const vsd_params& p, float* loss, void* grad, float* weights, void* ws,
                     cudaStream_t s) {
    Problem<T> P = make_problem<T>(draft, nullptr, L, T_, ws);
    set_params(P, p);
    const EStepView E{es->tokens, es->corr_tokens, es->logq_tok, es->logq_corr,
                      es->logkappa, es->logkappa_corr, es->logkappa_ref};
    const size_t gelem = P.grad_bf16 ? 2 : 4;
    const bool vec = vec_ok(draft, nullptr, grad, L.V, sizeof(T), gelem);
    cudaError_t e = clear_counters(ws, L, s);
    if (e == cudaSuccess) e = Launch<T>::weights(P, E, weights, loss, s);
    if (e == cudaSuccess)
        e = Launch<T>::grad(P, vec, reinterpret_cast<const float4*>(es->row_stats), grad,
                            P.grad_bf16, s);
    return from_cuda(e);
}

template <typename T>
vsd_status fused_impl(const void* draft, const void* target, vsd_layout L, float T_,
                      const float* u_draft, const float* u_accept, const float* u_correct,
                      const float* ref_logkappa, const vsd_params& p,
                      const vsd_linear_outputs* out, void* ws, cudaStream_t s,
                      bool clear = true, bool xtab_given = false) {
    Problem<T> P = make_problem<T>(draft, target, L, T_, ws);
    set_params(P, p);
    P.u_draft = u_draft;
    P.u_accept = u_accept;
    P.u_correct = u_correct;
    P.ref_logkappa = ref_logkappa;
    P.out = *out;
    const size_t gelem = P.grad_bf16 ? 2 : 4;
    const bool vec = vec_ok(draft, target, out->grad, L.V, sizeof(T), gelem);
    const int per_sm = Launch<T>::fused_blocks_per_sm(P, vec, P.grad_bf16);
    // rows of one short segment: the streaming warps run the row tails
    // themselves (three warps at once) instead of leaving them to the
    // control warp, which would otherwise bound the kernel
    P.stream_tails = (P.nseg == 1 && P.nch <= kStreamTailChunks) ? 1 : 0;
    // Residual claims: short rows through the counting semaphore (claims in
    // parallel: the per-prefix chain bounds those launches), long rows by one
    // compare-and-swap on the queue head (one round trip fewer per claim:
    // there the claims of the streaming jobs bound it).  Measured on GB300:
    // V=32000 0.107 vs 0.136 ms, V=128256 0.669 vs 0.642 ms.
    P.resq_sem = P.stream_tails;
    P.xtab_given = xtab_given ? 1 : 0;
    // no dense gradient asked for: no gradient jobs (the M-step's coefficients
    // stay in the workspace for vsd_lmhead_backward)
    if (!out->grad) P.gnseg = 0;
    const int64_t tickets = (int64_t)P.R * (P.nseg + P.gnseg);
    int ctas = per_sm * num_sms();
    if ((int64_t)ctas > tickets) ctas = (int)tickets;
    cudaError_t e = clear ? clear_counters(ws, L, s) : cudaSuccess;
    if (e == cudaSuccess) e = Launch<T>::fused(P, vec, out->grad, P.grad_bf16, ctas, s);
    return from_cuda(e);
}

}  // namespace
}  // namespace vsd

using namespace vsd;

extern "C" {

size_t vsd_workspace_bytes(vsd_layout layout) {
    if (!layout_ok(layout)) return 0;
    return ws_layout(layout).total;
}

vsd_status vsd_sample_paths(const void* draft, vsd_dtype dtype, vsd_layout layout, float T,
                            const float* u_draft, int32_t* tokens, float* logq_tok,
                            float* row_stats, void* ws, size_t ws_bytes, void* stream) {
    if (!layout_ok(layout) || layout.parent) return VSD_ERR_INVALID_ARG;
    if (!draft || !u_draft || !tokens || !logq_tok) return VSD_ERR_INVALID_ARG;
    if (dtype != VSD_F32 && dtype != VSD_BF16) return VSD_ERR_INVALID_ARG;
    vsd_status st = check_temperature(T);
    if (st) return st;
    if ((st = check_ws(layout, ws, ws_bytes))) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (dtype == VSD_F32)
        return sample_impl<float>(draft, layout, T, u_draft, tokens, logq_tok, row_stats, ws, s);
    return sample_impl<__nv_bfloat16>(draft, layout, T, u_draft, tokens, logq_tok, row_stats, ws,
                                      s);
}

vsd_status vsd_verify_paths(const void* draft, const void* target, vsd_dtype dtype,
                            vsd_layout layout, float T, const int32_t* tokens,
                            const float* u_accept, const float* u_correct,
                            const float* ref_logkappa, vsd_linear_outputs* out,
                            vsd_tree_outputs* tree_out, void* ws, size_t ws_bytes,
                            void* stream) {
    if (!layout_ok(layout)) return VSD_ERR_INVALID_ARG;
    if (!draft || !target || !tokens || !u_accept || !u_correct) return VSD_ERR_INVALID_ARG;
    if (dtype != VSD_F32 && dtype != VSD_BF16) return VSD_ERR_INVALID_ARG;
    if (layout.parent) {
        if (!tree_out || ref_logkappa) return VSD_ERR_INVALID_ARG;
        const vsd_tree_outputs& o = *tree_out;
        if (!o.alpha || !o.accept || !o.path_accept || !o.logkappa || !o.corr_tokens ||
            !o.deepest || !o.accept_len || !o.bonus)
            return VSD_ERR_INVALID_ARG;
    } else {
        if (!out || !out->accept_len || !out->corr_tokens || !out->logkappa)
            return VSD_ERR_INVALID_ARG;
    }
    vsd_status st = check_temperature(T);
    if (st) return st;
    if ((st = check_ws(layout, ws, ws_bytes))) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (dtype == VSD_F32)
        return verify_impl<float>(draft, target, layout, T, tokens, u_accept, u_correct,
                                  ref_logkappa, out, tree_out, ws, s);
    return verify_impl<__nv_bfloat16>(draft, target, layout, T, tokens, u_accept, u_correct,
                                      ref_logkappa, out, tree_out, ws, s);
}

vsd_status vsd_weighted_loss_fwd_bwd(const void* draft, vsd_dtype dtype, vsd_layout layout,
                                     float T, const vsd_linear_outputs* estep,
                                     const vsd_params* params, float* loss, void* grad,
                                     float* weights, void* ws, size_t ws_bytes, void* stream) {
    if (!layout_ok(layout) || layout.parent) return VSD_ERR_INVALID_ARG;
    if (!draft || !estep || !loss || !grad) return VSD_ERR_INVALID_ARG;
    if (!estep->tokens || !estep->corr_tokens || !estep->logq_tok || !estep->logq_corr ||
        !estep->logkappa || !estep->logkappa_corr || !estep->logkappa_ref || !estep->row_stats)
        return VSD_ERR_INVALID_ARG;
    if (dtype != VSD_F32 && dtype != VSD_BF16) return VSD_ERR_INVALID_ARG;
    vsd_status st = check_temperature(T);
    if (st) return st;
    const vsd_params p = params ? *params : default_params(dtype);
    if ((st = check_params(p))) return st;
    if (p.kl_weight != 0.0) return VSD_ERR_UNSUPPORTED;  // the top-K term needs the target rows
    if ((st = check_ws(layout, ws, ws_bytes))) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (dtype == VSD_F32)
        return loss_impl<float>(draft, layout, T, estep, p, loss, grad, weights, ws, s);
    return loss_impl<__nv_bfloat16>(draft, layout, T, estep, p, loss, grad, weights, ws, s);
}

vsd_status vsd_estep_mstep(const void* draft, const void* target, vsd_dtype dtype,
                           vsd_layout layout, float T, const float* u_draft,
                           const float* u_accept, const float* u_correct,
                           const float* ref_logkappa, const vsd_params* params,
                           vsd_linear_outputs* out, void* ws, size_t ws_bytes, void* stream) {
    if (!layout_ok(layout) || layout.parent) return VSD_ERR_INVALID_ARG;
    if (!draft || !target || !u_draft || !u_accept || !u_correct || !out)
        return VSD_ERR_INVALID_ARG;
    if (!out->tokens || !out->accept_len || !out->corr_tokens || !out->logkappa || !out->loss)
        return VSD_ERR_INVALID_ARG;
    if (dtype != VSD_F32 && dtype != VSD_BF16) return VSD_ERR_INVALID_ARG;
    vsd_status st = check_temperature(T, true);
    if (st) return st;
    const vsd_params p = params ? *params : default_params(dtype);
    if ((st = check_params(p))) return st;
    if ((st = check_ws(layout, ws, ws_bytes))) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (dtype == VSD_F32)
        return fused_impl<float>(draft, target, layout, T, u_draft, u_accept, u_correct,
                                 ref_logkappa, p, out, ws, s);
    return fused_impl<__nv_bfloat16>(draft, target, layout, T, u_draft, u_accept, u_correct,
                                     ref_logkappa, p, out, ws, s);
}

vsd_status vsd_tree_estep_mstep(const void* draft, const void* target, vsd_dtype dtype,
                                vsd_layout layout, float T, const int32_t* tokens,
                                const float* u_accept, const float* u_correct,
                                const vsd_params* params, vsd_tree_em_outputs* out, void* ws,
                                size_t ws_bytes, void* stream) {
    if (!layout_ok(layout) || !layout.parent) return VSD_ERR_INVALID_ARG;
    if (!draft || !target || !tokens || !u_accept || !u_correct || !out || !out->loss ||
        !out->grad)
        return VSD_ERR_INVALID_ARG;
    if (dtype != VSD_F32 && dtype != VSD_BF16) return VSD_ERR_INVALID_ARG;
    vsd_status st = check_temperature(T);
    if (st) return st;
    const vsd_params p = params ? *params : default_params(dtype);
    if ((st = check_params(p))) return st;
    if (p.kl_weight != 0.0) return VSD_ERR_UNSUPPORTED;
    if ((st = check_ws(layout, ws, ws_bytes))) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = clear_counters(ws, layout, s);
    if (e != cudaSuccess) return from_cuda(e);
    const size_t gelem = p.grad_dtype == VSD_BF16 ? 2 : 4;
    if (dtype == VSD_F32) {
        Problem<float> P = make_problem<float>(draft, target, layout, T, ws);
        set_params(P, p);
        P.given_tokens = tokens;
        P.u_accept = u_accept;
        P.u_correct = u_correct;
        e = Launch<float>::tree_em(P, vec_ok(draft, target, out->grad, layout.V, 4, gelem), *out,
                                   out->grad, P.grad_bf16, s);
    } else {
        Problem<__nv_bfloat16> P = make_problem<__nv_bfloat16>(draft, target, layout, T, ws);
        set_params(P, p);
        P.given_tokens = tokens;
        P.u_accept = u_accept;
        P.u_correct = u_correct;
        e = Launch<__nv_bfloat16>::tree_em(P, vec_ok(draft, target, out->grad, layout.V, 2, gelem),
                                           *out, out->grad, P.grad_bf16, s);
    }
    return from_cuda(e);
}

vsd_status vsd_lmhead_logits(const void* hidden, const void* weight, int32_t M, int32_t N,
                             int32_t K, void* logits, void* ws, size_t ws_bytes, void* stream) {
    if (!lmhead_shape_ok(hidden, weight, logits, M, N, K)) return VSD_ERR_INVALID_ARG;
    if (!ws || ws_bytes < 256 || ((uintptr_t)ws & 255)) return VSD_ERR_WORKSPACE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = cudaMemsetAsync(ws, 0, sizeof(int32_t), s);
    if (e == cudaSuccess)
        e = lmhead_gemm(hidden, weight, M, N, K, logits, static_cast<int*>(ws), kDefaultTimeoutNs, s);
    return from_cuda(e);
}

vsd_status vsd_lmhead_estep_mstep(const void* hidden, const void* weight, int32_t H,
                                  const void* target, vsd_layout layout, float T,
                                  const float* u_draft, const float* u_accept,
                                  const float* u_correct, const float* ref_logkappa,
                                  const vsd_params* params, void* draft_logits,
                                  vsd_linear_outputs* out, void* ws, size_t ws_bytes,
                                  void* stream) {
    if (!layout_ok(layout) || layout.parent) return VSD_ERR_INVALID_ARG;
    if (!target || !u_draft || !u_accept || !u_correct || !out) return VSD_ERR_INVALID_ARG;
    if (!out->tokens || !out->accept_len || !out->corr_tokens || !out->logkappa || !out->loss)
        return VSD_ERR_INVALID_ARG;
    const int64_t R = rows_of(layout);
    if (R > (1 << 30) || !lmhead_shape_ok(hidden, weight, draft_logits, (int)R, layout.V, H))
        return VSD_ERR_INVALID_ARG;
    vsd_status st = check_temperature(T, true);
    if (st) return st;
    const vsd_params p = params ? *params : default_params(VSD_BF16);
    if ((st = check_params(p))) return st;
    if ((st = check_ws(layout, ws, ws_bytes))) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    // the counters and the status word are cleared once, before both steps;
    // the GEMM's epilogue writes the draft half of every row's chunk table
    // (a1 for the draft), so the E-step streams only the target rows
    const WsLayout w = ws_layout(layout);
    const float c = (float)(kLog2e / (double)(T == 0.f ? 1.f : T));  // as make_problem's
    cudaError_t e = clear_counters(ws, layout, s);
    if (e == cudaSuccess)
        e = lmhead_gemm(hidden, weight, (int)R, layout.V, H, draft_logits, static_cast<int*>(ws),
                        p.wait_timeout_ns ? p.wait_timeout_ns : kDefaultTimeoutNs, s,
                        at<float4>(ws, w.gtab), w.nch_ws, c);
    if (e != cudaSuccess) return from_cuda(e);
    return fused_impl<__nv_bfloat16>(draft_logits, target, layout, T, u_draft, u_accept,
                                     u_correct, ref_logkappa, p, out, ws, s, false, true);
}

vsd_status vsd_lmhead_backward(const void* hidden, const void* weight, int32_t H,
                               const void* draft_logits, vsd_layout layout, float T,
                               const vsd_params* params, float* d_hidden, float* d_weight,
                               void* ws, size_t ws_bytes, void* stream) {
    if (!layout_ok(layout) || layout.parent) return VSD_ERR_INVALID_ARG;
    const int64_t R = rows_of(layout);
    if (R > (1 << 30) || !lmhead_shape_ok(hidden, weight, draft_logits, (int)R, layout.V, H))
        return VSD_ERR_INVALID_ARG;
    if (((uintptr_t)d_hidden | (uintptr_t)d_weight) & 15) return VSD_ERR_INVALID_ARG;
    vsd_status st = check_temperature(T, true);
    if (st) return st;
    const vsd_params p = params ? *params : default_params(VSD_BF16);
    if ((st = check_params(p))) return st;
    if ((st = check_ws(layout, ws, ws_bytes))) return st;
    if (!d_hidden && !d_weight) return VSD_OK;
    const WsLayout w = ws_layout(layout);
    cudaError_t e = lmhead_backward(
        hidden, weight, draft_logits, (int)R, layout.V, H, T, at<RowRec>(ws, w.rows),
        at<Coef>(ws, w.coef), p.kl_weight != 0.0 ? at<KlRec>(ws, w.klr) : nullptr,
        at<void>(ws, w.bfac), d_hidden, d_weight, at<int>(ws, w.status), p.wait_timeout_ns ? p.wait_timeout_ns : kDefaultTimeoutNs,
        static_cast<cudaStream_t>(stream));
    return from_cuda(e);
}

vsd_status vsd_reference_logkappa(const void* ref_draft, const void* ref_target, vsd_dtype dtype,
                                  int32_t B, int32_t D, int32_t V, float T, float* ref_logkappa,
                                  void* ws, size_t ws_bytes, void* stream) {
    const vsd_layout L{B, 1, D, V, 0, nullptr, 0};
    if (!layout_ok(L)) return VSD_ERR_INVALID_ARG;
    if (!ref_draft || !ref_target || !ref_logkappa) return VSD_ERR_INVALID_ARG;
    if (dtype != VSD_F32 && dtype != VSD_BF16) return VSD_ERR_INVALID_ARG;
    vsd_status st = check_temperature(T, true);
    if (st) return st;
    if ((st = check_ws(L, ws, ws_bytes))) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = clear_counters(ws, L, s);
    if (e != cudaSuccess) return from_cuda(e);
    if (dtype == VSD_F32) {
        Problem<float> P = make_problem<float>(ref_draft, ref_target, L, T, ws);
        e = Launch<float>::reference(P, vec_ok(ref_draft, ref_target, nullptr, V, 4, 0),
                                     ref_logkappa, s);
    } else {
        Problem<__nv_bfloat16> P = make_problem<__nv_bfloat16>(ref_draft, ref_target, L, T, ws);
        e = Launch<__nv_bfloat16>::reference(P, vec_ok(ref_draft, ref_target, nullptr, V, 2, 0),
                                             ref_logkappa, s);
    }
    return from_cuda(e);
}

vsd_status vsd_device_status(void* ws, void* stream, int32_t* status_bits) {
    if (!ws || !status_bits) return VSD_ERR_INVALID_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    int32_t v = 0;
    cudaError_t e = cudaMemcpyAsync(&v, ws, sizeof(v), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e == cudaSuccess) e = cudaMemsetAsync(ws, 0, sizeof(v), s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return VSD_ERR_CUDA;
    *status_bits = v;
    if (v & VSD_STATUS_TIMEOUT) return VSD_ERR_TIMEOUT;
    return v ? VSD_ERR_DEVICE_DATA : VSD_OK;
}

const char* vsd_status_string(vsd_status status) {
    switch (status) {
        case VSD_OK: return "ok";
        case VSD_ERR_INVALID_ARG: return "invalid argument";
        case VSD_ERR_UNSUPPORTED: return "unsupported request (temperature 0)";
        case VSD_ERR_CUDA: return "CUDA runtime error";
        case VSD_ERR_TIMEOUT: return "a device-side wait timed out";
        case VSD_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
        case VSD_ERR_DEVICE_DATA: return "device-side data check failed";
        case VSD_ERR_TOO_LARGE:
            return "problem needs more scratch than the built-in array of vsd_estep_mstep_noalloc";
    }
    return "unknown status";
}

const char* vsd_version(void) { return "0.2.0"; }

}  // extern "C"
