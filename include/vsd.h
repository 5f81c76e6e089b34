/*
 * vsd.h -- C ABI of the GB300 (sm_103a) library for the data-parallel hot path
 * of Variational Speculative Decoding (VSD, arxiv 2602.05774): the per-token,
 * vocabulary-wide work of its Monte-Carlo EM draft training.
 *
 * For each prefix x (index b), K draft paths of depth D are drawn from the
 * draft distribution q (Algorithm 1, E-step), every token is verified against
 * the target distribution p with the speculative-sampling rule of Eq. 1, the
 * accepted length and the path-level validity kappa (Eq. 2) are formed, the
 * oracle of Algorithm 2 scores each proposal, and the M-step's weighted
 * log-likelihood (Eq. advance, with the ARW coefficient of Eq. beta and the
 * CAR weight of Eq. zeta) is evaluated together with its gradient with respect
 * to the draft logits.  Names follow the paper: K is the paper's S (number of
 * latent proposals), D its L (sampling length), T the sampling temperature,
 * tau_car the CAR temperature tau.
 *
 * Conventions shared by every entry point
 *   - Every array argument is a DEVICE pointer owned by the caller, unless the
 *     argument says "host".  The library allocates nothing and keeps no pointer
 *     after a call returns.
 *   - Logit rows are row-major with the vocabulary contiguous.  Linear paths:
 *     rows [B][K][D][V], row r = (b*K + s)*D + d, R = B*K*D rows.  Trees: rows
 *     [B][N][V], row (b, n) is the distribution node n's children were drafted
 *     from.  q_r = softmax(draft_r / T), p_r = softmax(target_r / T) (Eq. 1).
 *   - Uniform random numbers are inputs (float32 in [0,1), one per row per
 *     use).  A uniform u >= 1 draws the last token with mass; u < 0 the first.
 *   - Work is enqueued asynchronously on `stream` (a cudaStream_t, NULL = the
 *     legacy default stream).  Argument checks are synchronous and return an
 *     error before anything is enqueued.  Data errors found on the device (a
 *     NaN or all -inf row, a token outside [0,V), a malformed tree, a wait that
 *     timed out) set bits of a status word in the workspace, readable with
 *     vsd_device_status(); the kernels never trap.
 *   - `ws` is caller-owned device scratch of at least vsd_workspace_bytes()
 *     bytes; calls sharing one workspace must be ordered on one stream.
 *   - Rows whose address is 16-byte aligned with V*sizeof(elem) a multiple of
 *     16 take the 128-bit vector path; any other shape takes a scalar path with
 *     identical results.
 *   - Limits: 1 <= V <= 1048576, 1 <= D <= 64, 1 <= K <= 256, 1 <= N <= 1024,
 *     B*K*D (or B*N) <= 16777216, T finite and > 0.
 *   - T = 0 (greedy decoding, the T in {0, 1} of the paper's evaluation) is
 *     served by vsd_estep_mstep, vsd_estep_mstep_noalloc,
 *     vsd_lmhead_estep_mstep and vsd_reference_logkappa: every decision takes
 *     the argmax limit of Eq. 1's distributions (z~ = argmax q, accepted iff
 *     it is argmax p, the correction is argmax p; lowest index on ties), and
 *     the M-step's log q, its gradient, zeta and the top-K term use the
 *     draft's distribution at temperature 1.  The other calls return
 *     VSD_ERR_UNSUPPORTED for T = 0.
 */
#ifndef VSD_H_
#define VSD_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    VSD_OK = 0,
    VSD_ERR_INVALID_ARG = 1, /* a size, pointer, dtype or parameter is invalid */
    VSD_ERR_UNSUPPORTED = 2, /* a valid request this call does not serve          */
    VSD_ERR_CUDA = 3,        /* a CUDA runtime call failed                        */
    VSD_ERR_TIMEOUT = 4,     /* a device-side wait gave up (vsd_device_status)    */
    VSD_ERR_WORKSPACE = 5,   /* workspace missing or smaller than required        */
    VSD_ERR_DEVICE_DATA = 6, /* a device-side data check failed (status bits)     */
    VSD_ERR_TOO_LARGE = 7    /* the problem needs more scratch than the library's
                                built-in array (vsd_estep_mstep_noalloc)           */
} vsd_status;

typedef enum { VSD_F32 = 0, VSD_BF16 = 1 } vsd_dtype;

/* Device status bits (vsd_device_status). */
#define VSD_STATUS_BAD_ROW 1     /* a logit row holds NaN/+inf or is all -inf   */
#define VSD_STATUS_TIMEOUT 2     /* a bounded device wait ran out               */
#define VSD_STATUS_BAD_TREE 4    /* parent[0] != -1 or parent[n] not in [0, n)  */
#define VSD_STATUS_BAD_TOKEN 8   /* a given token is outside [0, V)             */

/* Problem shape.  parent == NULL: linear paths, R = B*K*D rows, N unused.
 * parent != NULL: draft trees, device array [B][N] of parent indices
 * (parent[b][0] = -1, 0 <= parent[b][n] < n), R = B*N rows, K and D unused.
 * tree_rule (trees, vsd_verify_paths): VSD_TREE_INDEPENDENT verifies every
 * branch alone (a node is accepted when it and its ancestors pass their own
 * test); VSD_TREE_SEQUENTIAL is the lossless multi-draft rule: along the
 * accepted path a node's children are tried in node order, child i accepted
 * with probability min(1, p_i(t_i)/q_i(t_i)), where after each rejection
 * p_{i+1} = norm(max(0, p_i - q_i)) and q_{i+1} = q_i with t_i removed and
 * renormalised; the first accepted child continues the path, and when every
 * child is rejected the correction token is drawn from p_{m+1} with the last
 * child's u_correct.  The emitted token is then distributed as p whenever the
 * siblings are drawn from q without replacement. */
#define VSD_TREE_INDEPENDENT 0
#define VSD_TREE_SEQUENTIAL 1
typedef struct {
    int32_t B, K, D, V, N;
    const int32_t* parent;
    int32_t tree_rule;
} vsd_layout;

/* M-step parameters (App. F: w(l) = 1.05^l, tau = 0.2). */
typedef struct {
    double w_base;     /* w(l) = w_base^l, l = 1..D                                */
    double tau_car;    /* CAR temperature tau of Eq. zeta                          */
    int32_t zeta_mode; /* 0: softmax of q(z~_{<=l})/tau (as printed); 1: log q      */
    int32_t grad_dtype;/* vsd_dtype of the gradient output                         */
    uint64_t wait_timeout_ns; /* bound of every device wait; 0 = 2 s              */
    int32_t test_never_publish; /* test hook, normally 0: if nonzero the fused kernel
                                 never publishes a prefix's M-step, so every gradient
                                 wait runs out after wait_timeout_ns, no gradient row
                                 is written and VSD_STATUS_TIMEOUT is set            */
    double kl_weight;  /* VSD (KL) (App., Eq. klv): 0 = none; else loss_b gains
                          kl_weight (1/K) sum over the prefix's rows of the top-K
                          renormalised cross-entropy -sum_{x in top-K of p}
                          p^(x) log q^(x) (the paper gives no weight)       */
    int32_t kl_topk;   /* K of that term (the paper's 10), 1 <= kl_topk <= 16  */
} vsd_params;

/* Output arrays of the linear E-step / M-step (all device, caller-owned).
 * Per-row arrays have R entries, per-path arrays B*K.  A NULL member is
 * not written, except where an entry point lists it as required. */
typedef struct {
    int32_t* tokens;        /* [R] z~_d, the draft sample (Algorithm 1)              */
    float* logq_tok;        /* [R] log q_r(z~_d)                                      */
    float* alpha;           /* [R] min(1, p_r(z~_d)/q_r(z~_d)) (Eq. 1)                */
    uint8_t* accept;        /* [R] u_accept <= alpha                                  */
    int32_t* accept_len;    /* [B*K] A: number of leading accepted tokens             */
    int32_t* corr_tokens;   /* [R] z'_d: z~_d before the first rejection, a residual
                               token norm(max(0,p-q)) at it, p-samples after it      */
    float* logq_corr;       /* [R] log q_r(z'_d)                                      */
    float* alpha_corr;      /* [R] min(1, p/q) at z'_d                                */
    float* logkappa;        /* [R] log kappa(z~_{<=l}), l = d+1 (Eq. 2)               */
    float* logkappa_corr;   /* [R] log kappa(z'_{<=l})                                */
    float* logkappa_ref;    /* [R] log kappa of the greedy reference (Algorithm 2)    */
    int32_t* ref_tokens;    /* [R] argmax of the target row (lowest index on ties)    */
    float* expected_len;    /* [B*K] sum_{k<=D} S_k (Eq. 11)                          */
    float* row_stats;       /* [R][4] m_q, logZ_q, m_p, logZ_p with
                               log q(v) = (x_v - m_q)/T - logZ_q                     */
    float* weights;         /* [B][D][K][4] o~, o', beta, zeta (Alg. 1, Eq. beta/zeta)*/
    float* loss;            /* [B+1] loss_b = -J_b/N_b, then mean over b (Eq. advance)*/
    void* grad;             /* [R][V] d loss / d draft logits, params.grad_dtype;
                               NULL (fused calls): not written, the M-step's
                               coefficients stay in ws for vsd_lmhead_backward */
    float* kl_loss;         /* [R] the row's top-K term of Eq. klv (with kl_weight)   */
} vsd_linear_outputs;

/* Output arrays of tree verification (device, caller-owned), [B][N] unless noted. */
typedef struct {
    float* alpha;           /* min(1, p/q) of node n's token at its parent's row; root 1 */
    uint8_t* accept;        /* u_accept <= alpha; root 1                                 */
    uint8_t* path_accept;   /* node and all its ancestors accepted                       */
    float* logkappa;        /* sum of log alpha from the root to n                       */
    int32_t* corr_tokens;   /* residual token at the parent's row for a rejected node
                               whose parent is on an accepted path; -1 otherwise         */
    int32_t* deepest;       /* [B] deepest node on an accepted path (lowest index)       */
    int32_t* accept_len;    /* [B] depth of that node                                    */
    int32_t* bonus;         /* [B] token after the accepted path: the residual of the
                               deepest node's first child, or a p-sample at its row      */
    float* row_stats;       /* optional [B*N][4] as in vsd_linear_outputs; when NULL
                               the rows of leaves are not read (a leaf's row enters
                               the results only through the bonus token, for which
                               the deepest accepted leaf's row is read), and a leaf
                               row's invalid values then set no status bit        */
} vsd_tree_outputs;

/* Outputs of the E-step + M-step over draft trees (vsd_tree_estep_mstep;
 * device, caller-owned, [B][N] unless noted; node 0, the root, is no
 * proposal and holds zeros).  Every node n >= 1 is a latent proposal: the
 * tokens on its root path, of length depth(n). */
typedef struct {
    int32_t* corr_tokens;   /* z'_n: n's token on an accepted path, the residual
                               norm(max(0, p - q)) at the path's first rejected
                               node, a draw from p below it (each with n's own
                               u_correct, at n's parent's row); root -1          */
    float* logq_tok;        /* log q of n's token at its parent's row            */
    float* logq_corr;       /* log q of z'_n there                               */
    float* logkappa;        /* log kappa of the root path of n (Eq. 2)           */
    float* logkappa_corr;   /* of the corrected path                             */
    float* logkappa_ref;    /* of the greedy reference along the same rows
                               (each row's target argmax, Algorithm 2)           */
    float* weights;         /* [B][N][4] o~, o', beta, zeta; beta and zeta over
                               the nodes of one depth                            */
    float* loss;            /* [B+1] loss_b = -J_b/N_b (Eq. advance), then the mean */
    void* grad;             /* [B*N][V] d loss / d draft logits, params.grad_dtype:
                               row n collects the terms of every proposal whose
                               path goes through one of n's children; a leaf's
                               row is 0                                          */
} vsd_tree_em_outputs;

/* Bytes of device workspace the calls below need for `layout` (0 if invalid). */
size_t vsd_workspace_bytes(vsd_layout layout);

/* Draft sampling (Algorithm 1, z~ ~ q): for every linear row, the inverse-CDF
 * draw z~_r = min{v : u_draft_r < sum_{j<=v} q_r(j)} and log q_r(z~_r).
 * draft: [R][V] of `dtype`.  u_draft: [R].  Outputs: tokens [R], logq_tok [R],
 * row_stats optional [R][4] (the p columns are written as 0).  Linear layout only. */
vsd_status vsd_sample_paths(const void* draft, vsd_dtype dtype, vsd_layout layout, float T,
                            const float* u_draft, int32_t* tokens, float* logq_tok,
                            float* row_stats, void* ws, size_t ws_bytes, void* stream);

/* Verification (Eq. 1 per token; Sec. 3 residual correction; Eqs. 2, 9-11;
 * Algorithm 2's greedy reference).
 * Linear layout: tokens are the drafted z~ [R] (for example from
 * vsd_sample_paths); u_accept, u_correct [R]; ref_logkappa optional [B][D]
 * (NULL: the greedy reference of each path, read from the same rows).  Writes
 * every verification member of `out` that is non-NULL (required: accept_len,
 * corr_tokens, logkappa); tokens/logq_tok are copied through.
 * Tree layout: tokens [B][N] (node 0 ignored), u_accept, u_correct [B][N],
 * ref_logkappa must be NULL, results in `tree_out` (all members but row_stats
 * required); `out` is ignored. */
vsd_status vsd_verify_paths(const void* draft, const void* target, vsd_dtype dtype,
                            vsd_layout layout, float T, const int32_t* tokens,
                            const float* u_accept, const float* u_correct,
                            const float* ref_logkappa, vsd_linear_outputs* out,
                            vsd_tree_outputs* tree_out, void* ws, size_t ws_bytes,
                            void* stream);

/* M-step (Algorithm 1 M-step, Algorithm 2 utility, Eqs. beta, zeta, advance;
 * params->kl_weight must be 0 here, VSD_ERR_UNSUPPORTED otherwise):
 * from the E-step results in `estep` (tokens, corr_tokens, logq_tok, logq_corr,
 * logkappa, logkappa_corr, logkappa_ref, row_stats: all required) computes
 * o~, o', beta, zeta, loss_b = -J_b/N_b, their mean, and the gradient of the
 * mean loss with respect to the draft logits, with o~, o', beta, zeta, N_b held
 * constant.  loss [B+1] and grad [R][V] (params->grad_dtype) are required,
 * weights [B][D][K][4] optional.  Linear layout only. */
vsd_status vsd_weighted_loss_fwd_bwd(const void* draft, vsd_dtype dtype, vsd_layout layout,
                                     float T, const vsd_linear_outputs* estep,
                                     const vsd_params* params, float* loss, void* grad,
                                     float* weights, void* ws, size_t ws_bytes, void* stream);

/* The fused E-step + M-step (Algorithm 1, both steps, for all prefixes at
 * once; Algorithm 2 as the oracle; Eqs. 1, 2, 11, beta, zeta, advance): one
 * persistent kernel runs sampling, verification, utilities, weights, loss and
 * gradient over all prefixes, with the results of vsd_sample_paths,
 * vsd_verify_paths and vsd_weighted_loss_fwd_bwd.  Arguments as for those
 * calls: draft, target [R][V] of `dtype`; u_draft, u_accept, u_correct [R];
 * ref_logkappa optional [B][D]; params NULL for the defaults (App. F:
 * w(l) = 1.05^l, tau = 0.2).  Required members of `out`: tokens, accept_len,
 * corr_tokens, logkappa, loss; the rest are optional (grad NULL: the dense
 * gradient is not written, for a vsd_lmhead_backward that makes it on chip
 * from what the call leaves in ws).  Linear layout
 * only.  Errors: VSD_ERR_INVALID_ARG for a bad shape, pointer, dtype or
 * parameter, VSD_ERR_UNSUPPORTED for T = 0, VSD_ERR_WORKSPACE for a missing
 * or small workspace, VSD_ERR_CUDA if a launch fails; data errors on the
 * device go to the status word (vsd_device_status). */
vsd_status vsd_estep_mstep(const void* draft, const void* target, vsd_dtype dtype,
                           vsd_layout layout, float T, const float* u_draft,
                           const float* u_accept, const float* u_correct,
                           const float* ref_logkappa, const vsd_params* params,
                           vsd_linear_outputs* out, void* ws, size_t ws_bytes, void* stream);

/* The E-step + M-step over draft trees (App. E trees as the latent
 * proposals; Algorithm 1 and 2, Eqs. 1, 2, beta, zeta, advance on the trees'
 * root paths).  Each position x of a path is verified alone (Eq. 1 at x's
 * parent's row; the path validity of Eq. 2), the corrected path follows
 * Sec. 3 along the branch, o~ and o' use w(depth), beta and zeta run over the
 * proposals of one length (the nodes of one depth), and the loss and its
 * gradient are Eq. advance's.  Arguments as for vsd_verify_paths with a tree
 * layout (tokens [B][N], node 0 ignored; u_accept, u_correct [B][N]) plus
 * params (NULL: the defaults; kl_weight must be 0).  Required outputs: loss,
 * grad; the rest optional.  T > 0.  Errors as for vsd_estep_mstep. */
vsd_status vsd_tree_estep_mstep(const void* draft, const void* target, vsd_dtype dtype,
                                vsd_layout layout, float T, const int32_t* tokens,
                                const float* u_accept, const float* u_correct,
                                const vsd_params* params, vsd_tree_em_outputs* out, void* ws,
                                size_t ws_bytes, void* stream);

/* Allocation-free variant of vsd_estep_mstep; the paper has no counterpart.
 * For callers that cannot allocate device memory where they call the library
 * (a plugin given only its input and output pointers, a process whose device
 * memory belongs entirely to another allocator, a latency-critical loop where
 * cudaMalloc/cudaFree would synchronise the device).  Instead of a caller
 * workspace it uses a fixed array of VSD_NOALLOC_SCRATCH_BYTES in device memory
 * that the library owns; every GPU that loads the library holds that array until
 * the process exits.  Arguments, required outputs and results are those of
 * vsd_estep_mstep.
 *   - Limit: the layout's vsd_workspace_bytes() must not exceed
 *     VSD_NOALLOC_SCRATCH_BYTES (32 MiB: every linear layout of up to 4096 rows
 *     with V <= 200000; the B=32, K=16, D=8, V=128256 workload needs 17 MB);
 *     larger problems return VSD_ERR_TOO_LARGE before anything is enqueued.
 *   - The first call on a device looks up the array's device address with that
 *     device current (cudaGetSymbolAddress); make that first call before any
 *     stream capture.  The call allocates nothing.
 *   - All calls on a device share the one array, which keeps the last call's
 *     contents (each call clears the part that must start at zero).  Calls that
 *     overlap on the GPU -- on different streams, or from different host
 *     threads -- race on it; order them on one stream.
 *   - The address is looked up again when the device's context has changed
 *     (after a cudaDeviceReset, for example).
 *   - The device status word of these calls (timeouts, invalid rows) lives in
 *     that array: read it with vsd_noalloc_device_status(); argument and
 *     launch errors are returned as usual. */
#define VSD_NOALLOC_SCRATCH_BYTES (32u << 20)
vsd_status vsd_estep_mstep_noalloc(const void* draft, const void* target, vsd_dtype dtype,
                                   vsd_layout layout, float T, const float* u_draft,
                                   const float* u_accept, const float* u_correct,
                                   const float* ref_logkappa, const vsd_params* params,
                                   vsd_linear_outputs* out, void* stream);

/* vsd_device_status() for the calls of vsd_estep_mstep_noalloc on the current
 * device: waits for `stream`, then reads and clears the status word kept in
 * the library's array into *status_bits (host).  Allocates nothing.  Same
 * return codes as vsd_device_status(). */
vsd_status vsd_noalloc_device_status(void* stream, int32_t* status_bits);

/* The draft model's LM head, the layer that produces the draft logits q is
 * computed from (paper Sec. 5, implementation details: the draft head's output
 * layer):  logits[M][N] = hidden[M][K] . weight[N][K]^T.
 *   hidden  device, bf16, row-major [M][K] (K contiguous);
 *   weight  device, bf16, row-major [N][K] (the vocabulary-by-hidden matrix);
 *   logits  device, bf16, row-major [M][N], written (caller-owned);
 *   ws      device workspace of at least 256 bytes whose first word is the
 *           status word (the same as a vsd_estep_mstep workspace); cleared here.
 * Products are exact and summed in fp32 on the tensor cores, then rounded once
 * to bf16 (round to nearest even).  N and K must be multiples of 8 and the
 * three pointers 16-byte aligned (VSD_ERR_INVALID_ARG otherwise); M >= 1.
 * Asynchronous on `stream`; a device wait that runs out sets the timeout bit
 * of the status word (vsd_device_status). */
vsd_status vsd_lmhead_logits(const void* hidden, const void* weight, int32_t M, int32_t N,
                             int32_t K, void* logits, void* ws, size_t ws_bytes, void* stream);

/* The LM head followed by the fused E-step + M-step on its logits (config of
 * the draft head fused with the EM step):
 *   hidden        device, bf16 [R][H], R = B*K*D rows in the layout's row order;
 *   weight        device, bf16 [V][H];
 *   target        device, bf16 [R][V], the target logits;
 *   draft_logits  device, bf16 [R][V], receives the draft logits (caller-owned);
 * every other argument as for vsd_estep_mstep with dtype VSD_BF16 (linear
 * layouts only).  The status word of `ws` collects the bits of both steps. */
vsd_status vsd_lmhead_estep_mstep(const void* hidden, const void* weight, int32_t H,
                                  const void* target, vsd_layout layout, float T,
                                  const float* u_draft, const float* u_accept,
                                  const float* u_correct, const float* ref_logkappa,
                                  const vsd_params* params, void* draft_logits,
                                  vsd_linear_outputs* out, void* ws, size_t ws_bytes,
                                  void* stream);

/* The draft LM head's backward: the M-step's gradient (Algorithm 1, the
 * gradient of Eq. advance, plus VSD (KL)'s top-K term when params->kl_weight
 * is nonzero) carried from the draft logits into the head's input and weight:
 *   d_hidden[R][H] = G . weight        d_weight[V][H] = G^T . hidden
 * with G[r][v] the gradient with respect to draft_logits[r][v], the bf16 value
 * the preceding call writes to out->grad with grad_dtype VSD_BF16.  G is not
 * read from memory: it is made on chip from draft_logits and the row records
 * and M-step coefficients that call left in `ws`, so this call must follow a
 * vsd_lmhead_estep_mstep, or a vsd_estep_mstep with dtype VSD_BF16, on the
 * same draft_logits, layout (linear), T, params->kl_weight and workspace, with
 * nothing else run on that workspace in between.
 *   hidden, weight   device, bf16 [R][H] and [V][H], as for the LM head;
 *   draft_logits     device, bf16 [R][V];
 *   d_hidden         device, float [R][H], written; NULL to skip;
 *   d_weight         device, float [V][H], written; NULL to skip.
 * Products of bf16 values are exact and summed in fp32 on the tensor cores.
 * H and V must be multiples of 8 and the pointers 16-byte aligned
 * (VSD_ERR_INVALID_ARG); T >= 0 as given to the preceding call.  A device wait
 * that runs out sets the timeout bit of the status word of `ws`. */
vsd_status vsd_lmhead_backward(const void* hidden, const void* weight, int32_t H,
                               const void* draft_logits, vsd_layout layout, float T,
                               const vsd_params* params, float* d_hidden, float* d_weight,
                               void* ws, size_t ws_bytes, void* stream);

/* The greedy reference of Algorithm 2 from its own rows: the oracle's z-bar
 * is drawn from the greedy target policy, so its validity log kappa(z-bar)
 * needs the draft and target distributions along z-bar, which the caller
 * computes (teacher-forced on z-bar) and passes here.  Writes
 * ref_logkappa[b][l-1] = sum_{d < l} log min(1, p_d(v_d) / q_d(v_d)) with v_d
 * the target row's argmax (lowest index on ties; Eq. 2 on the greedy path),
 * ready to pass as `ref_logkappa` to vsd_estep_mstep / vsd_verify_paths.
 *   ref_draft, ref_target  device, [B][D][V] of `dtype`, the rows along z-bar;
 *   ref_logkappa           device, [B][D] float, written;
 *   T >= 0 (T = 0: the one-hot limits, so every entry is 0);
 *   ws of vsd_workspace_bytes({B, 1, D, V}) bytes.
 * Errors as for vsd_verify_paths. */
vsd_status vsd_reference_logkappa(const void* ref_draft, const void* ref_target, vsd_dtype dtype,
                                  int32_t B, int32_t D, int32_t V, float T, float* ref_logkappa,
                                  void* ws, size_t ws_bytes, void* stream);

/* Waits for `stream`, then reads and clears the device status word of `ws`
 * into *status_bits (host).  Returns VSD_ERR_TIMEOUT if the timeout bit is set,
 * VSD_ERR_DEVICE_DATA for any other bit, VSD_OK if none. */
vsd_status vsd_device_status(void* ws, void* stream, int32_t* status_bits);

/* A static English description of a status code. */
const char* vsd_status_string(vsd_status status);

/* Library version, "major.minor.patch". */
const char* vsd_version(void);

#ifdef __cplusplus
}
#endif

#endif /* VSD_H_ */
