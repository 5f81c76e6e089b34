// vsd_tree.cuh -- draft trees beyond independent branch verification (App. E
// trees): the E-step + M-step with every node a latent proposal, and tree
// verification with the sequential sibling rule (lossless multi-draft).
//
//   k_tree_rows  one block per node row u: the row pass (tables, statistics,
//                the target's argmax, a draw from p with u's uniform), then
//                for every child x of u its token's test at u's row (Eq. 1,
//                each branch alone) and, for the EM, the draws a corrected
//                path may take at x: from p with x's uniform (below a
//                rejection) and from the residual norm(max(0, p - q)) (the
//                first rejection; one more read of the row when a child is
//                rejected).
//   k_tree_em    one block per tree: the accepted paths, the corrected path
//                z' of every node, the log-kappa sums along the root paths
//                (Eq. 2), o~ and o' (Algorithm 2), beta and zeta over the nodes
//                of one depth (Eqs. beta, zeta), the loss (Eq. advance) and
//                each node's gradient terms (sums over its subtree).
//   k_tree_grad  one block per row: grad = g q(v) minus the sparse terms of
//                the row's children (their tokens and corrected tokens).
//   k_tree_seq   one block per tree: the sequential sibling rule along the
//                accepted path, with one read of a row per rejected sibling.
#pragma once

#include "vsd_passes.cuh"

namespace vsd {

// What k_tree_rows leaves for a node x (at index b*N + x).
struct __align__(16) TreeNodeRec {
    float la;      // log alpha of x's token at its parent's row (the branch alone)
    float lq;      // log q of that token
    int acc;       // u_accept <= alpha
    int zp;        // draw from p at the parent's row with x's u_correct
    float lq_zp, la_zp;
    int zr;        // residual draw at the parent's row with x's u_correct (-1: none)
    float lq_zr, la_zr;
    int pad[3];
};
static_assert(sizeof(TreeNodeRec) == 48, "TreeNodeRec layout");

// A node's gradient terms at its parent's row, scaled by 1 / (B N_b T):
// -ct at its token t, -cz at its corrected token z (z = -1: none).
struct __align__(16) TreeCoef {
    int t;
    float ct;
    int z;
    float cz;
};
static_assert(sizeof(TreeCoef) == 16, "TreeCoef layout");

// ------------------------------------------------------------ k_tree_rows
template <typename T, bool VEC, bool EM>
__device__ void tree_row_children(const Problem<T>& P, int r, Ring* rg, float4* tab, int* s_any) {
    const int N = P.N;
    const int64_t V = P.V;
    const int b = r / N, u = r - b * N, n0 = b * N;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int32_t* par = P.parent + (int64_t)n0;
    const T* x = P.draft + (int64_t)r * V;
    const T* y = P.target + (int64_t)r * V;
    const float c = P.ts.c;
    const uint64_t pol = policy_evict_normal();
    const RowRec rec = ld_cg(P.rows + r);
    if (threadIdx.x == 0) *s_any = 0;
    __syncthreads();
    // the target's table for the draws from p (each warp, identical values)
    float My = 0.f;
    TableSum Sy{0, 0, 0.0};
    if (EM) {
        My = table_max(tab, P.nch, 1, lane);
        Sy = table_sum(tab, P.nch, 1, frame_of(My), c, lane);
    }
    int k = 0;
    for (int n = u + 1; n < N; ++n) {
        if (__ldg(par + n) != u) continue;
        if (k++ % kWarps != warp) continue;
        TreeNodeRec nr;
        nr.la = -INFINITY;
        nr.lq = -INFINITY;
        nr.zp = -1;
        nr.lq_zp = nr.la_zp = -INFINITY;
        nr.zr = -1;
        nr.lq_zr = nr.la_zr = -INFINITY;
        nr.pad[0] = nr.pad[1] = nr.pad[2] = 0;
        const int tok = __ldg(P.given_tokens + n0 + n);
        if (tok < 0 || tok >= V) {
            if (lane == 0) atomicOr(P.status, VSD_STATUS_BAD_TOKEN);
        } else if (!rec.flags) {
            token_logs(x, y, tok, rec, P.ts.invTd, &nr.lq, &nr.la);
        }
        nr.acc = nr.la > -INFINITY && __ldg(P.u_accept + n0 + n) <= expf(nr.la);
        if (EM && !rec.flags) {
            int zp = warp_sample<T, VEC>(x, y, V, tab, P.nch, 1, My, Sy,
                                         __ldg(P.u_correct + n0 + n), c, lane, pol);
            if (zp >= V) zp = -1;
            nr.zp = zp;
            if (zp >= 0) token_logs(x, y, zp, rec, P.ts.invTd, &nr.lq_zp, &nr.la_zp);
        }
        if (lane == 0) {
            P.tnode[n0 + n] = nr;
            if (!nr.acc) *s_any = 1;
        }
    }
    __syncthreads();
    if (!EM || !*s_any || rec.flags) return;
    // a child is rejected: the residual max(0, p - q) of the row, and each
    // rejected child's draw from it (or from p if it has no mass)
    const MassRes mr{rec.mx, rec.my, rec.izx, rec.izy, c};
    stream_residual<T, VEC>(rg, x, y, V, 0, P.nch, tab, mr, P.status);
    __syncthreads();
    const TableSum Rt = table_sum(tab, P.nch, 0, 0.f, c, lane);
    k = 0;
    for (int n = u + 1; n < N; ++n) {
        if (__ldg(par + n) != u) continue;
        if (k++ % kWarps != warp) continue;
        TreeNodeRec nr = P.tnode[n0 + n];  // written by this warp above
        if (nr.acc) continue;
        int zr = -1;
        if (Rt.Z > 0.0) {
            const Located loc =
                table_locate(tab, P.nch, 0, 0.f, c, Rt, __ldg(P.u_correct + n0 + n), lane);
            if (loc.ch >= 0)
                zr = warp_rescan<T, VEC, true, true>(x, y, V, loc.ch, loc.tc, mr, lane, pol);
            if (zr >= V) zr = -1;
        } else {
            zr = nr.zp;  // no residual mass: the draw from p with the same uniform
        }
        nr.zr = zr;
        if (zr >= 0) token_logs(x, y, zr, rec, P.ts.invTd, &nr.lq_zr, &nr.la_zr);
        if (lane == 0) P.tnode[n0 + n] = nr;
    }
}

template <typename T, bool VEC, bool EM>
__global__ void __launch_bounds__(kThreads) k_tree_rows(Problem<T> P) {
    extern __shared__ __align__(128) unsigned char dsm[];
    __shared__ RowShared sh;
    __shared__ int s_any;
    Ring* rg = nullptr;
    float4* tab;
    if (VEC) {
        rg = reinterpret_cast<Ring*>(dsm);
        tab = reinterpret_cast<float4*>(dsm + sizeof(Ring));
        ring_init(rg, P.timeout_ns);
    } else {
        tab = reinterpret_cast<float4*>(dsm);
    }
    const int r = blockIdx.x;
    row_pass<T, VEC, true, kNoToken, true>(P, r, rg, tab, sh);
    __syncthreads();
    tree_row_children<T, VEC, EM>(P, r, rg, tab, &s_any);
    if (threadIdx.x == 0 && P.tout.row_stats)
        reinterpret_cast<float4*>(P.tout.row_stats)[r] = ld_cg(P.rstats + r);
}

// ------------------------------------------------------------ shared helpers
struct TreeShared2 {
    int par[1024];
    int depth[1024];
    unsigned char pacc[1024];
    int maxd;
};

// Parents into shared memory and the tree's checks (parent[0] = -1, every
// other parent precedes its node); depths.  Returns false for a bad tree.
template <typename T>
__device__ bool tree_load(const Problem<T>& P, int b, TreeShared2& sh) {
    const int N = P.N;
    const int32_t* par = P.parent + (int64_t)b * N;
    int badl = 0;
    for (int n = threadIdx.x; n < N; n += kThreads) {
        const int pn = __ldg(par + n);
        sh.par[n] = pn;
        badl |= n == 0 ? pn != -1 : (pn < 0 || pn >= n);
    }
    const int bad = __syncthreads_or(badl);
    if (bad) return false;
    if (threadIdx.x == 0) {
        sh.depth[0] = 0;
        int maxd = 0;
        for (int n = 1; n < N; ++n) {
            sh.depth[n] = sh.depth[sh.par[n]] + 1;
            maxd = max(maxd, sh.depth[n]);
        }
        sh.maxd = maxd;
    }
    __syncthreads();
    return true;
}

// ------------------------------------------------------------ k_tree_em
// The M-step of one tree, in double precision on one thread (a tree has at
// most 1024 nodes; the arithmetic follows the proposals in node order, so the
// result does not depend on scheduling).  Scratch per node in shared memory.
struct TreeEmShared {
    TreeShared2 t;
    double lk[1024], lkc[1024], lkr[1024], lqt[1024], lqz[1024];
    double st[1024], sz[1024];   // subtree sums of the gradient terms
    float w[1024][4];            // o~, o', beta, zeta
    float lqzn[1024];            // log q of z'_x at its parent's row
    int z[1024];                 // corrected token z'_x
};

template <typename T>
__global__ void __launch_bounds__(kThreads) k_tree_em(Problem<T> P, vsd_tree_em_outputs o) {
    extern __shared__ __align__(16) unsigned char dsm[];
    TreeEmShared& sh = *reinterpret_cast<TreeEmShared*>(dsm);
    const int N = P.N, b = blockIdx.x, n0 = b * N;
    const bool ok = tree_load<T>(P, b, sh.t);
    if (!ok) {
        for (int n = threadIdx.x; n < N; n += kThreads) {
            P.tcoef[n0 + n] = TreeCoef{-1, 0.f, -1, 0.f};
            P.tg[n0 + n] = 0.f;
            if (o.corr_tokens) o.corr_tokens[n0 + n] = -1;
            if (o.weights)
                reinterpret_cast<float4*>(o.weights)[n0 + n] = make_float4(0.f, 0.f, 0.f, 0.f);
        }
        if (threadIdx.x == 0) {
            atomicOr(P.status, VSD_STATUS_BAD_TREE);
            P.tbad[b] = 1;
            o.loss[b] = 0.f;
        }
    } else if (threadIdx.x == 0) {
        P.tbad[b] = 0;
        const int* par = sh.t.par;
        const int* depth = sh.t.depth;
        // the E-step per node (R15): accepted paths, z', the sums along the paths
        sh.t.pacc[0] = 1;
        sh.lk[0] = sh.lkc[0] = sh.lkr[0] = sh.lqt[0] = sh.lqz[0] = 0.0;
        sh.z[0] = -1;
        sh.lqzn[0] = 0.f;
        for (int x = 1; x < N; ++x) {
            const int a = par[x];
            const TreeNodeRec nr = ld_cg_rec(P.tnode + n0 + x);
            const RowRec ra = ld_cg(P.rows + n0 + a);
            const int tok = __ldg(P.given_tokens + n0 + x);
            const bool pa = nr.acc && sh.t.pacc[a];
            sh.t.pacc[x] = pa;
            int zc;
            float lqz, laz;
            if (pa) {
                zc = tok; lqz = nr.lq; laz = nr.la;
            } else if (sh.t.pacc[a]) {  // the first rejection on the path: the residual
                zc = nr.zr; lqz = nr.lq_zr; laz = nr.la_zr;
            } else {                    // below a rejection: the draw from p
                zc = nr.zp; lqz = nr.lq_zp; laz = nr.la_zp;
            }
            if (zc < 0) { lqz = -INFINITY; laz = -INFINITY; }
            sh.z[x] = zc;
            sh.lqzn[x] = lqz;
            const double lar = (ra.flags || ra.ref < 0) ? -INFINITY : (double)ra.la_ref;
            sh.lk[x] = sh.lk[a] + (double)nr.la;
            sh.lkc[x] = sh.lkc[a] + (double)laz;
            sh.lkr[x] = sh.lkr[a] + lar;
            sh.lqt[x] = sh.lqt[a] + (double)nr.lq;
            sh.lqz[x] = sh.lqz[a] + (double)lqz;
        }
        // o~, o' (Algorithm 2 with w(depth))
        double Nb = 0.0;
        for (int n = 1; n < N; ++n) {
            // w(l) = w_base^l at the node's depth (trees may be deeper than the
            // host's table of w)
            const double wl = pow(P.w_base, (double)depth[n]);
            const bool ot = sh.lk[n] >= sh.lkr[n];
            const bool op = ot || sh.lkc[n] >= sh.lkr[n];
            sh.w[n][0] = ot ? 1.f : 0.f;
            sh.w[n][1] = op ? (float)wl : 0.f;
            Nb += op ? wl : 0.0;
        }
        // beta (leave-one-out) and zeta (softmax of q(z~)/tau, or log q in
        // zeta_mode 1) over the nodes of each depth
        for (int l = 1; l <= sh.t.maxd; ++l) {
            double num = 0.0, den = 0.0, cmax = -INFINITY;
            for (int n = 1; n < N; ++n) {
                if (depth[n] != l) continue;
                const double op = sh.w[n][1];
                num += op * sh.w[n][0];
                den += op;
                const double cq = (P.zeta_mode == 0 ? exp(sh.lqt[n]) : sh.lqt[n]) * P.inv_tau;
                cmax = fmax(cmax, cq);
            }
            double zs = 0.0;
            for (int n = 1; n < N; ++n) {
                if (depth[n] != l) continue;
                const double cq = (P.zeta_mode == 0 ? exp(sh.lqt[n]) : sh.lqt[n]) * P.inv_tau;
                zs += exp(cq - cmax);
            }
            for (int n = 1; n < N; ++n) {
                if (depth[n] != l) continue;
                const double op = sh.w[n][1];
                const double d1 = den - op, n1 = num - op * sh.w[n][0];
                sh.w[n][2] = d1 > 0.0 ? (float)(n1 / d1) : 0.f;
                const double cq = (P.zeta_mode == 0 ? exp(sh.lqt[n]) : sh.lqt[n]) * P.inv_tau;
                sh.w[n][3] = (float)(exp(cq - cmax) / zs);
            }
        }
        // the objective (Eq. advance), each proposal's terms, subtree sums
        // (the proposals whose path goes through a node)
        double J = 0.0;
        for (int n = 0; n < N; ++n) sh.st[n] = sh.sz[n] = 0.0;
        for (int n = 1; n < N; ++n) {
            const double ot = sh.w[n][0], op = sh.w[n][1];
            const double bz = (double)sh.w[n][2] * (double)sh.w[n][3];
            if (op == 0.0) continue;
            const double lqn = ot > 0.0 ? sh.lqt[n] : sh.lqz[n];
            J += op * (lqn - bz * sh.lqt[n]);
            sh.st[n] += op * (ot - bz);
            sh.sz[n] += op * (1.0 - ot);
        }
        for (int n = N - 1; n >= 1; --n) {  // children come after their parents
            sh.st[par[n]] += sh.st[n];
            sh.sz[par[n]] += sh.sz[n];
        }
        const double scale = Nb > 0.0 ? 1.0 / ((double)P.B * Nb * P.ts.Td) : 0.0;
        for (int n = 0; n < N; ++n) P.tg[n0 + n] = 0.f;
        o.loss[b] = Nb > 0.0 ? (float)(-J / Nb) : 0.f;
        for (int x = 1; x < N; ++x) {
            TreeCoef cf;
            cf.t = __ldg(P.given_tokens + n0 + x);
            cf.ct = (float)(sh.st[x] * scale);
            cf.z = sh.z[x];
            cf.cz = (float)(sh.sz[x] * scale);
            if (cf.z == cf.t) {
                cf.ct = (float)((sh.st[x] + sh.sz[x]) * scale);
                cf.z = -1;
                cf.cz = 0.f;
            }
            P.tcoef[n0 + x] = cf;
            P.tg[n0 + par[x]] += (float)((sh.st[x] + sh.sz[x]) * scale);
        }
    }
    __syncthreads();
    if (ok) {
        for (int n = threadIdx.x; n < N; n += kThreads) {
            if (o.corr_tokens) o.corr_tokens[n0 + n] = sh.z[n];
            if (o.weights)
                reinterpret_cast<float4*>(o.weights)[n0 + n] =
                    n ? make_float4(sh.w[n][0], sh.w[n][1], sh.w[n][2], sh.w[n][3])
                      : make_float4(0.f, 0.f, 0.f, 0.f);
            if (o.logq_tok) o.logq_tok[n0 + n] = n ? ld_cg(&P.tnode[n0 + n].lq) : 0.f;
            if (o.logq_corr) o.logq_corr[n0 + n] = sh.lqzn[n];
            if (o.logkappa) o.logkappa[n0 + n] = (float)sh.lk[n];
            if (o.logkappa_corr) o.logkappa_corr[n0 + n] = (float)sh.lkc[n];
            if (o.logkappa_ref) o.logkappa_ref[n0 + n] = (float)sh.lkr[n];
        }
    }
    if (threadIdx.x == 0) {
        __threadfence();
        if (atomicAdd(P.prefix_done, 1) == P.B - 1) {
            __threadfence();
            loss_mean(o.loss, P.B);
        }
    }
}

// ------------------------------------------------------------ k_tree_grad
// Row r of the gradient: g q(v) minus the sparse terms of r's children.  The
// terms are merged by token in a fixed order (sorted by token, then by child)
// so that the sums do not depend on scheduling.
constexpr int kTreeMaxTerms = 2048;
struct TreeGradShared {
    int tok[kTreeMaxTerms];
    float cf[kTreeMaxTerms];
    int skey[kTreeMaxTerms];
    float scf[kTreeMaxTerms];
    int n, nu;
};

template <typename T, bool VEC, typename G>
__global__ void __launch_bounds__(kThreads) k_tree_grad(Problem<T> P, G* grad) {
    __shared__ TreeGradShared sh;
    constexpr int PV = Traits<T>::kPerVec;
    const int N = P.N, r = blockIdx.x, b = r / N, u = r - b * N, n0 = b * N;
    const int64_t V = P.V;
    G* g = grad + (int64_t)r * V;
    const T* x = P.draft + (int64_t)r * V;
    const int32_t* par = P.parent + (int64_t)n0;
    if (threadIdx.x == 0) sh.n = 0;
    __syncthreads();
    const bool bad = ld_cg(P.tbad + b) != 0;
    if (!bad) {  // the children's terms
        for (int n = u + 1 + threadIdx.x; n < N; n += kThreads) {
            if (__ldg(par + n) != u) continue;
            const TreeCoef cf = ld_cg_rec(P.tcoef + n0 + n);
            const int slot = atomicAdd(&sh.n, cf.z >= 0 ? 2 : 1);
            // (order fixed below by the sort key: token, then child index)
            sh.tok[slot] = cf.t;
            sh.cf[slot] = cf.ct;
            sh.skey[slot] = 2 * n;
            if (cf.z >= 0) {
                sh.tok[slot + 1] = cf.z;
                sh.cf[slot + 1] = cf.cz;
                sh.skey[slot + 1] = 2 * n + 1;
            }
        }
    }
    __syncthreads();
    const int n = sh.n;
    // rank sort by (token, key) into scf/skey order: entry i goes to its rank
    __shared__ int rk_tok[kTreeMaxTerms];
    for (int i = threadIdx.x; i < n; i += kThreads) {
        int rank = 0;
        for (int j = 0; j < n; ++j)
            rank += sh.tok[j] < sh.tok[i] || (sh.tok[j] == sh.tok[i] && sh.skey[j] < sh.skey[i]);
        rk_tok[rank] = sh.tok[i];
        sh.scf[rank] = sh.cf[i];
    }
    __syncthreads();
    if (threadIdx.x == 0) {  // merge equal tokens, in order
        int m = 0;
        for (int i = 0; i < n; ++i) {
            if (m > 0 && sh.tok[m - 1] == rk_tok[i]) {
                sh.cf[m - 1] += sh.scf[i];
            } else {
                sh.tok[m] = rk_tok[i];
                sh.cf[m] = sh.scf[i];
                ++m;
            }
        }
        sh.nu = m;
    }
    __syncthreads();
    const int nu = sh.nu;
    // the first merged term at or after token v (binary search)
    auto first_at = [&](int64_t v) {
        int lo = 0, hi = nu;
        while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if ((int64_t)sh.tok[mid] < v) lo = mid + 1; else hi = mid;
        }
        return lo;
    };
    const float gr = bad ? 0.f : ld_cg(P.tg + r);
    const RowRec rec = ld_cg(P.rows + r);
    const float gq = (nu == 0 && gr == 0.f) ? 0.f : gr * rec.izx;
    const float mx = rec.mx, c = P.ts.c;
    const bool dense = gq != 0.f && isfinite(mx);
    if constexpr (VEC) {
        const uint64_t pol = policy_evict_first();
        const int nvec = (int)(V / PV);
        for (int i = threadIdx.x; i < nvec; i += kThreads) {
            const int64_t v0 = (int64_t)i * PV;
            float o[PV];
            if (dense) {
                float f[PV];
                unpack<T>(ld_stream(x + v0, pol), f);
#pragma unroll
                for (int e = 0; e < PV; ++e) o[e] = gq * ex2((f[e] - mx) * c);
            } else {
#pragma unroll
                for (int e = 0; e < PV; ++e) o[e] = 0.f;
            }
            if (nu) {
                for (int k = first_at(v0); k < nu && sh.tok[k] < v0 + PV; ++k) {
#pragma unroll
                    for (int e = 0; e < PV; ++e)
                        if (v0 + e == sh.tok[k]) o[e] -= sh.cf[k];
                }
            }
            grad_store<T, G, PV>(g, v0, o, pol);
        }
    } else {
        for (int64_t v = threadIdx.x; v < V; v += kThreads) {
            float val = dense ? gq * ex2((elem_value(x, v) - mx) * c) : 0.f;
            if (nu) {
                const int k = first_at(v);
                if (k < nu && sh.tok[k] == v) val -= sh.cf[k];
            }
            if constexpr (sizeof(G) == 2)
                g[v] = __float2bfloat16_rn(val);
            else
                g[v] = val;
        }
    }
}

// ------------------------------------------------------------ k_tree_seq
// The sequential sibling rule (lossless multi-draft) along the accepted path
// of one tree.  At node u with children c_1 .. c_m (node order) child i is
// accepted with probability min(1, p_i(t_i)/q_i(t_i)); after a rejection
// p_{i+1} = norm(max(0, p_i - q_i)) (p_i kept if that has no mass) and
// q_{i+1} = q_i without t_i, renormalised.  p_i at a point follows the
// recursion from the row's p and q and the normalisers found so far; each
// normaliser is one read of the row (chunk sums of max(0, p_i - q_i), summed
// exactly), and after the last rejection the correction token is drawn from
// that table.
struct SeqState {
    int nrem;              // children tried so far at this node
    int rem[1024];         // their tokens (removed from q)
    double S[1024];        // S[j]: normaliser of p_{j+2} (0: p kept)
    double Qs[1024];       // Qs[j]: remaining draft mass before the (j+1)-th child
};

struct TreeSeqShared {
    TreeShared2 t;
    SeqState st;
    int kids[1024];
    int nk;
    int cur, out_tok, leaf_bonus;
};

// p_i(v) and q_i(v) for the (i+1)-th child (i = children rejected so far),
// from the row's own p(v), q(v).
__device__ __forceinline__ void seq_point(const SeqState& st, int i, int64_t v, double p,
                                          double q, double& pi, double& qi) {
    pi = p;
    bool removed = false;
    for (int j = 0; j < i; ++j) {
        const double qj = removed ? 0.0 : (st.Qs[j] > 0.0 ? q / st.Qs[j] : 0.0);
        if (st.S[j] > 0.0) pi = fmax(0.0, pi - qj) / st.S[j];
        removed |= st.rem[j] == v;
    }
    qi = removed ? 0.0 : (st.Qs[i] > 0.0 ? q / st.Qs[i] : 0.0);
}

template <typename T, bool VEC>
__global__ void __launch_bounds__(kThreads) k_tree_seq(Problem<T> P) {
    extern __shared__ __align__(16) unsigned char dsm[];
    TreeSeqShared& sh = *reinterpret_cast<TreeSeqShared*>(dsm);
    float4* tab = reinterpret_cast<float4*>(dsm + sizeof(TreeSeqShared));
    const int N = P.N, b = blockIdx.x, n0 = b * N;
    const int64_t V = P.V;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const vsd_tree_outputs& o = P.tout;
    const float c = P.ts.c;
    if (!tree_load<T>(P, b, sh.t)) {
        for (int n = threadIdx.x; n < N; n += kThreads) {
            o.alpha[n0 + n] = 0.f;
            o.accept[n0 + n] = 0;
            o.path_accept[n0 + n] = 0;
            o.logkappa[n0 + n] = -INFINITY;
            o.corr_tokens[n0 + n] = -1;
        }
        if (threadIdx.x == 0) {
            atomicOr(P.status, VSD_STATUS_BAD_TREE);
            o.deepest[b] = -1;
            o.accept_len[b] = -1;
            o.bonus[b] = -1;
        }
        return;
    }
    for (int n = threadIdx.x; n < N; n += kThreads) {
        o.alpha[n0 + n] = n ? 0.f : 1.f;
        o.accept[n0 + n] = n ? 0 : 1;
        o.path_accept[n0 + n] = n ? 0 : 1;
        o.corr_tokens[n0 + n] = -1;
    }
    if (threadIdx.x == 0) {  // log kappa: the path validity (Eq. 2) of every node
        double* lk = sh.st.S;  // (scratch before the walk)
        lk[0] = 0.0;
        o.logkappa[n0] = 0.f;
        for (int n = 1; n < N; ++n) {
            lk[n] = lk[sh.t.par[n]] + (double)ld_cg(&P.tnode[n0 + n].la);
            o.logkappa[n0 + n] = (float)lk[n];
        }
        sh.cur = 0;
        sh.out_tok = -1;
    }
    __syncthreads();
    for (;;) {
        const int u = sh.cur;
        // the children of u, in node order
        if (threadIdx.x == 0) {
            int m = 0;
            for (int n = u + 1; n < N; ++n)
                if (sh.t.par[n] == u) sh.kids[m++] = n;
            sh.nk = m;
            sh.st.nrem = 0;
        }
        __syncthreads();
        const int m = sh.nk;
        if (m == 0) break;
        const int ru = n0 + u;
        const RowRec rec = ld_cg(P.rows + ru);
        const T* x = P.draft + (int64_t)ru * V;
        const T* y = P.target + (int64_t)ru * V;
        int next = -1;
        for (int i = 0; i < m; ++i) {
            const int ch = sh.kids[i];
            if (threadIdx.x == 0) {
                const int t = __ldg(P.given_tokens + n0 + ch);
                double alpha = 0.0;
                if (!rec.flags && t >= 0 && t < V) {
                    if (i == 0) sh.st.Qs[0] = 1.0;
                    const double p = exp(((double)elem_value(y, t) - rec.my) * P.ts.invTd - rec.lzy);
                    const double q = exp(((double)elem_value(x, t) - rec.mx) * P.ts.invTd - rec.lzx);
                    double pi, qi;
                    seq_point(sh.st, i, t, p, q, pi, qi);
                    alpha = qi > 0.0 ? fmin(1.0, pi / qi) : (pi > 0.0 ? 1.0 : 0.0);
                }
                const bool a = __ldg(P.u_accept + n0 + ch) <= alpha && !rec.flags;
                o.alpha[n0 + ch] = (float)alpha;
                o.accept[n0 + ch] = a ? 1 : 0;
                sh.st.rem[i] = t;
                if (a) {
                    o.path_accept[n0 + ch] = 1;
                    sh.cur = ch;
                    sh.st.nrem = -1;  // accepted
                } else {
                    sh.st.nrem = i + 1;
                    const double q_t = (t >= 0 && t < V && !rec.flags)
                        ? exp(((double)elem_value(x, t) - rec.mx) * P.ts.invTd - rec.lzx) : 0.0;
                    // the remaining draft mass once t_i is removed (t_i not removed before)
                    bool before = false;
                    for (int j = 0; j < i; ++j) before |= sh.st.rem[j] == t;
                    sh.st.Qs[i + 1] = sh.st.Qs[i] - (before ? 0.0 : q_t);
                }
            }
            __syncthreads();
            if (sh.st.nrem < 0) {
                next = sh.cur;
                break;
            }
            if (rec.flags) continue;
            // the normaliser of p_{i+2}: chunk sums of max(0, p_{i+1} - q_{i+1})
            // (one read of the row); the draw after the last rejection
            const int ii = i + 1;  // children rejected so far
            for (int chn = warp; chn < P.nch; chn += kWarps) {
                const uint64_t pol = policy_evict_normal();
                uint4 bx[kLoads], by[kLoads];
                load_chunk<T, VEC>(x, V, chn, lane, pol, bx);
                load_chunk<T, VEC>(y, V, chn, lane, pol, by);
                float acc = 0.f;
#pragma unroll
                for (int k = 0; k < kLoads; ++k) {
                    float fx[Traits<T>::kPerVec], fy[Traits<T>::kPerVec];
                    unpack<T>(bx[k], fx);
                    unpack<T>(by[k], fy);
#pragma unroll
                    for (int e = 0; e < Traits<T>::kPerVec; ++e) {
                        const int64_t v = (int64_t)chn * chunk_elems<T>() +
                                          k * 32 * Traits<T>::kPerVec + lane * Traits<T>::kPerVec + e;
                        if (v >= V) continue;
                        const double p = (double)(ex2((fy[e] - rec.my) * c) * rec.izy);
                        const double q = (double)(ex2((fx[e] - rec.mx) * c) * rec.izx);
                        double pi, qi;
                        seq_point(sh.st, ii - 1, v, p, q, pi, qi);
                        acc += (float)fmax(0.0, pi - qi);
                    }
                }
                acc = warp_sum(acc);
                if (lane == 0) tab[chn] = make_float4(0.f, acc, 0.f, 0.f);
            }
            __syncthreads();
            if (warp == 0) {
                const TableSum Rt = table_sum(tab, P.nch, 0, 0.f, c, lane);
                if (lane == 0) sh.st.S[ii - 1] = Rt.Z > 0.0 && Rt.Z < INFINITY ? Rt.Z : 0.0;
                if (i == m - 1) {  // every child rejected: the correction token
                    const float uc = __ldg(P.u_correct + n0 + ch);
                    int tok = -1;
                    if (Rt.Z > 0.0) {
                        const Located loc = table_locate(tab, P.nch, 0, 0.f, c, Rt, uc, lane);
                        if (loc.ch >= 0) {  // rescan the chunk in token order
                            float carry = 0.f;
                            const int64_t base = (int64_t)loc.ch * chunk_elems<T>();
                            int last = -1;
                            for (int64_t v0 = base; v0 < base + chunk_elems<T>() && tok < 0; v0 += 32) {
                                const int64_t v = v0 + lane;
                                float mv = 0.f;
                                if (v < V) {
                                    const double p = (double)(ex2((elem_value(y, v) - rec.my) * c) * rec.izy);
                                    const double q = (double)(ex2((elem_value(x, v) - rec.mx) * c) * rec.izx);
                                    double pi, qi;
                                    seq_point(sh.st, ii - 1, v, p, q, pi, qi);
                                    mv = (float)fmax(0.0, pi - qi);
                                }
                                const float incl = carry + warp_incl_scan(mv, lane);
                                const unsigned hit = __ballot_sync(0xffffffffu, mv > 0.f && incl > loc.tc);
                                const unsigned pos = __ballot_sync(0xffffffffu, mv > 0.f);
                                if (hit) tok = (int)(v0 + __ffs(hit) - 1);
                                else if (pos) last = (int)(v0 + 31 - __clz(pos));
                                carry = __shfl_sync(0xffffffffu, incl, 31);
                            }
                            if (tok < 0) tok = last;
                        }
                    } else {  // no residual mass: keep the last target distribution
                        tok = -2;
                    }
                    if (lane == 0) sh.out_tok = tok;
                }
            }
            __syncthreads();
            if (i == m - 1) {
                if (sh.out_tok == -2) {
                    // p_{m+1} = p_m: draw from it with the same uniform (a
                    // pass over the row's masses p_m, as above)
                    for (int chn = warp; chn < P.nch; chn += kWarps) {
                        const uint64_t pol = policy_evict_normal();
                        uint4 bx[kLoads], by[kLoads];
                        load_chunk<T, VEC>(x, V, chn, lane, pol, bx);
                        load_chunk<T, VEC>(y, V, chn, lane, pol, by);
                        float acc = 0.f;
#pragma unroll
                        for (int k = 0; k < kLoads; ++k) {
                            float fx[Traits<T>::kPerVec], fy[Traits<T>::kPerVec];
                            unpack<T>(bx[k], fx);
                            unpack<T>(by[k], fy);
#pragma unroll
                            for (int e = 0; e < Traits<T>::kPerVec; ++e) {
                                const int64_t v = (int64_t)chn * chunk_elems<T>() +
                                                  k * 32 * Traits<T>::kPerVec +
                                                  lane * Traits<T>::kPerVec + e;
                                if (v >= V) continue;
                                const double p = (double)(ex2((fy[e] - rec.my) * c) * rec.izy);
                                const double q = (double)(ex2((fx[e] - rec.mx) * c) * rec.izx);
                                double pi, qi;
                                seq_point(sh.st, ii - 1, v, p, q, pi, qi);
                                acc += (float)pi;
                            }
                        }
                        acc = warp_sum(acc);
                        if (lane == 0) tab[chn] = make_float4(0.f, acc, 0.f, 0.f);
                    }
                    __syncthreads();
                    if (warp == 0) {
                        const TableSum Pt = table_sum(tab, P.nch, 0, 0.f, c, lane);
                        const float uc = __ldg(P.u_correct + n0 + ch);
                        int tok = -1;
                        if (Pt.Z > 0.0) {
                            const Located loc = table_locate(tab, P.nch, 0, 0.f, c, Pt, uc, lane);
                            if (loc.ch >= 0) {
                                float carry = 0.f;
                                const int64_t base = (int64_t)loc.ch * chunk_elems<T>();
                                int last = -1;
                                for (int64_t v0 = base; v0 < base + chunk_elems<T>() && tok < 0; v0 += 32) {
                                    const int64_t v = v0 + lane;
                                    float mv = 0.f;
                                    if (v < V) {
                                        const double p = (double)(ex2((elem_value(y, v) - rec.my) * c) * rec.izy);
                                        const double q = (double)(ex2((elem_value(x, v) - rec.mx) * c) * rec.izx);
                                        double pi, qi;
                                        seq_point(sh.st, ii - 1, v, p, q, pi, qi);
                                        mv = (float)pi;
                                    }
                                    const float incl = carry + warp_incl_scan(mv, lane);
                                    const unsigned hit = __ballot_sync(0xffffffffu, mv > 0.f && incl > loc.tc);
                                    const unsigned pos = __ballot_sync(0xffffffffu, mv > 0.f);
                                    if (hit) tok = (int)(v0 + __ffs(hit) - 1);
                                    else if (pos) last = (int)(v0 + 31 - __clz(pos));
                                    carry = __shfl_sync(0xffffffffu, incl, 31);
                                }
                                if (tok < 0) tok = last;
                            }
                        }
                        if (lane == 0) sh.out_tok = tok;
                    }
                    __syncthreads();
                }
                if (threadIdx.x == 0) o.corr_tokens[n0 + ch] = sh.out_tok;
            }
        }
        if (next < 0) break;  // every child rejected: the path ends at u
        __syncthreads();
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        const int best = sh.cur;
        o.deepest[b] = best;
        o.accept_len[b] = sh.t.depth[best];
        o.bonus[b] = sh.nk > 0 ? sh.out_tok : ld_cg(P.rows + n0 + best).ps;
    }
}

}  // namespace vsd
