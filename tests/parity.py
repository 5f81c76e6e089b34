"""Comparison of the CUDA path with the CPU oracle on the same seeded inputs.

Discrete results (sampled tokens, accept bits, accepted lengths, corrected
tokens, oracle utilities) must be bit-exact.  The one exception is a decision
the oracle reports within a margin of its boundary -- |u - alpha| or
|u - CDF boundary| < PROB_MARGIN, or a log-kappa comparison within
LOGK_MARGIN: there the two sides may disagree, and a disagreement outside the
margins fails.  What depends on a flipped decision is then compared as
follows, so that nothing the GPU computed goes unchecked:

  * row-local results (the draft token z~_d, its acceptance and alpha, log
    q(z~_d), the target argmax, the row statistics) depend only on their own
    row: they are compared on every row whose draft token agrees, and every
    draft-token or acceptance disagreement must itself be near its boundary;
  * path results (the corrected path z', log kappa of z~, z' and the
    reference, the accepted length, E[A]) are compared on each path up to
    its first disagreeing decision;
  * the M-step (o~, o', beta, zeta, the loss and the gradient) of a prefix
    with any disagreement is recomputed by the oracle's own M-step from the
    GPU's E-step results (its tokens and log kappas) and compared with that:
    the M-step is a function of those results, so the GPU's arithmetic is
    checked given its own decisions.  Prefixes without one are compared with
    the oracle's end-to-end result.

Without the inputs that conditional check needs, a prefix with a disagreement
is excluded from the M-step comparison, within exclusion_budget().
"""
import numpy as np

PROB_MARGIN = 1e-6
# log-kappa comparisons add D log-alpha terms, each carrying the float32
# rounding of a log-probability (|log p| <= ~20, 2^-24 relative) and of the
# log-partition; D * 2e-6 bounds their sum for D <= 64 with room to spare.
LOGK_MARGIN = 1e-5
LOSS_RTOL = 1e-5
ALPHA_ATOL = 2e-6

# Session-wide record of what the protocol excused, printed at the end of the
# run (tests/conftest.py).
SESSION = {"calls": 0, "prefixes": 0, "near_boundary_decisions": 0, "diverged_paths": 0,
           "conditional_prefixes": 0, "excluded_prefixes": 0, "trees": 0,
           "excluded_trees": 0}


def exclusion_budget(B):
    """How many prefixes (or trees) of one call may be left out of the M-step
    (tree) comparison when no conditional check is possible: one per ten
    (at least one for B >= 3), none for B <= 2, and never all of them."""
    if B <= 2:
        return 0
    return max(1, B // 10)


def diverged_path_budget(npaths):
    """Paths of one call whose decisions may flip near a boundary: at most one
    in twenty (at least two).  At V = 128256 under the Zipf recipe about a
    third of the draft mass sits on tokens whose CDF interval is narrower
    than PROB_MARGIN, so near-boundary draws are common there (hundreds per
    call) and a few of them flip between fp64 and the GPU's exact-table/float
    rescan arithmetic; a systematic error would flip far more, or flip
    outside the margins."""
    return max(2, npaths // 20)


def to_np(t):
    if hasattr(t, "detach"):
        t = t.detach()
        return t.float().cpu().numpy() if t.dtype.is_floating_point else t.cpu().numpy()
    return np.asarray(t)


def _get(gpu, name):
    return None if gpu.get(name) is None else to_np(gpu[name])


def _close_mask(name, g, o, atol, rtol, mask):
    """Assert |g - o| <= atol + rtol |o| where mask holds; a NaN or a lone
    infinity on either side fails."""
    g = np.asarray(g, dtype=np.float64).reshape(-1)
    o = np.asarray(o, dtype=np.float64).reshape(-1)
    mask = np.asarray(mask, bool).reshape(-1)
    both_inf = np.isinf(g) & np.isinf(o) & (np.sign(g) == np.sign(o))
    both_nan = np.isnan(g) & np.isnan(o)
    with np.errstate(invalid="ignore"):
        err = np.where(both_inf | both_nan, 0.0, np.abs(g - o))
    lim = atol + rtol * np.abs(np.where(np.isfinite(o), o, 0))
    badi = np.nonzero(~(err <= lim) & mask)[0]
    assert badi.size == 0, "%s off at %s: gpu %s oracle %s" % (
        name, badi[:8], g[badi[:8]], o[badi[:8]])


def _grad_rows(name, g_rows, o_rows, grad_dtype, scale):
    g = np.asarray(g_rows, dtype=np.float64)
    o = np.asarray(o_rows, dtype=np.float64)
    if grad_dtype == "bf16":
        lim = 2.0 ** -8 * np.abs(o) + 1e-6 * scale + 1e-30
    else:
        lim = 1e-5 * np.abs(o) + 1e-6 * scale + 1e-30
    err = np.abs(g - o)
    badr = np.nonzero((~(err <= lim)).any(axis=1))[0]
    assert badr.size == 0, "%s rows off: %s, max err %g (scale %g)" % (
        name, badr[:8], np.nanmax(err[badr]), scale)
    emax = float(err.max()) if err.size else 0.0
    # the max-abs bar for gradients (fp32); a bf16 gradient adds the rounding
    # of its largest entry, 2^-8 relative
    bar = 1e-3 + (2.0 ** -8 * scale if grad_dtype == "bf16" else 0.0)
    assert emax <= bar, "%s max-abs error %g (bar %g)" % (name, emax, bar)
    return emax


def _first_divergence(gpu, orc, B, K, D):
    """Per path, the first row whose decisions disagree (D if none), after
    checking that every disagreement that is not a consequence of an earlier
    one lies within its margin."""
    m = orc["margins"].reshape(B * K, D, 6)
    tok_g = _get(gpu, "tokens")
    tok_o = np.asarray(orc["tokens"])
    tmis = (tok_g.reshape(B * K, D) != tok_o.reshape(B * K, D)) if tok_g is not None \
        else np.zeros((B * K, D), bool)
    # every draft token is an independent draw from its own row
    far = tmis & ~(m[..., 0] < PROB_MARGIN)
    assert not far.any(), "draft token differs outside the margin at path/row %s (margin %s)" % (
        np.argwhere(far)[:4].tolist(), m[..., 0][far][:4])
    acc_g = _get(gpu, "accept")
    amis = np.zeros((B * K, D), bool)
    if acc_g is not None:
        amis = acc_g.reshape(B * K, D) != np.asarray(orc["accept"]).reshape(B * K, D)
        # an acceptance depends only on its row's token and uniform
        far = amis & ~tmis & ~(m[..., 1] < PROB_MARGIN)
        assert not far.any(), "accept differs outside the margin at %s (margin %s)" % (
            np.argwhere(far)[:4].tolist(), m[..., 1][far][:4])
    corr_g = _get(gpu, "corr_tokens")
    cmis = np.zeros((B * K, D), bool)
    if corr_g is not None:
        cmis = corr_g.reshape(B * K, D) != np.asarray(orc["corr_tokens"]).reshape(B * K, D)
    anymis = tmis | amis | cmis
    f = np.where(anymis.any(axis=1), anymis.argmax(axis=1), D)
    for p in np.nonzero(f < D)[0]:
        d = f[p]
        if tmis[p, d] or amis[p, d]:
            continue  # checked above
        # the first disagreement is the corrected token itself: its draw
        # (residual or target sample with the same uniform) must be near a
        # boundary
        assert m[p, d, 2] < PROB_MARGIN, \
            "corrected token differs outside the margin at path %d row %d (margin %g)" % (
                p, d, m[p, d, 2])
    return f, tmis


def _conditional_mstep(gpu, b, K, D, V, T, grad_dtype, mi, check_grad, scale):
    """The oracle's M-step (weights, loss_b, gradient rows) recomputed from
    the GPU's E-step results of prefix b and compared with the GPU's."""
    from oracle import oracle as orc_mod
    P = K * D
    rows = slice(b * P, (b + 1) * P)

    def rowsof(name):
        return to_np(gpu[name]).reshape(-1)[rows].astype(np.float64).reshape(K, D)

    lk, lkc, lkr = rowsof("logkappa"), rowsof("logkappa_corr"), rowsof("logkappa_ref")
    lqpath = np.cumsum(rowsof("logq_tok"), axis=1)
    w, N = orc_mod.prefix_weights(lk, lkc, lkr, lqpath, mi.get("w_base", 1.05),
                                  mi.get("tau_car", 0.2), mi.get("zeta_mode", 0))
    tok = to_np(gpu["tokens"]).reshape(-1)[rows]
    corr = to_np(gpu["corr_tokens"]).reshape(-1)[rows]
    draft = np.asarray(mi["draft_rows"](b), dtype=np.float32).reshape(K, D, V)
    J, g = orc_mod.prefix_objective(draft, T, tok, corr, w, N, mi["B_total"],
                                    want_grad=check_grad)
    lam = mi.get("kl_weight", 0.0)
    kl = 0.0
    if lam:  # VSD (KL): the rows' top-K terms depend on the logits alone
        target = np.asarray(mi["target_rows"](b), dtype=np.float32).reshape(K * D, V)
        dr = draft.reshape(K * D, V)
        for i in range(K * D):
            Li, toks, dl = orc_mod.topk_ce(dr[i], target[i], T, mi.get("kl_topk", 10))
            kl += Li
            if check_grad:
                g.reshape(K * D, V)[i, toks] += lam / (mi["B_total"] * K) * dl
    if gpu.get("weights") is not None:
        wg = to_np(gpu["weights"]).reshape(-1, D, K, 4)[b]
        assert np.array_equal(wg[..., 0], w[..., 0]), "o~ (conditional) prefix %d" % b
        assert np.allclose(wg[..., 1], w[..., 1], rtol=1e-6, atol=0), "o' (conditional)"
        assert np.allclose(wg[..., 2], w[..., 2], rtol=1e-5, atol=1e-6), "beta (conditional)"
        assert np.allclose(wg[..., 3], w[..., 3], rtol=1e-5, atol=1e-6), "zeta (conditional)"
    lo = (-J / N if N > 0 else 0.0) + lam * kl / K
    lg = float(to_np(gpu["loss"])[b])
    assert abs(lg - lo) <= LOSS_RTOL * max(1.0, abs(lo)), \
        "loss[%d] (conditional) gpu %r oracle %r" % (b, lg, lo)
    if check_grad and gpu.get("grad") is not None:
        gg = gpu["grad"]
        gb = gg[b * P * V:(b + 1) * P * V] if gg.ndim == 1 else gg[b * P:(b + 1) * P]
        return _grad_rows("grad (conditional)", to_np(gb).reshape(P, V), g.reshape(P, V),
                          grad_dtype, scale)
    return 0.0


def compare_linear(gpu, orc, B, K, D, V, T, grad_dtype="f32", check_grad=True, report=None,
                   check_mean=True, mstep_inputs=None, kl=False):
    """Assert parity of E-step/M-step outputs under the protocol above;
    returns the number of prefixes whose M-step was not compared end to end
    (checked conditionally, or excluded).

    mstep_inputs (optional) enables the conditional M-step check: a dict with
    draft_rows(b) -> the prefix's draft logits [K*D, V], B_total (the call's
    number of prefixes, which scales the gradient), and the call's w_base,
    tau_car, zeta_mode when not the defaults.  With check_mean=False the mean
    loss entry is not compared (a sub-batch of a larger call, see sub_batch).
    kl: the call ran VSD (KL) (the per-row top-K terms are compared too)."""
    f, tmis = _first_divergence(gpu, orc, B, K, D)
    npaths = B * K
    path_div = f < D
    ndiv = int(path_div.sum())
    assert ndiv <= diverged_path_budget(npaths) and ndiv < npaths, \
        "too many paths with a flipped decision: %d of %d" % (ndiv, npaths)
    dvec = np.arange(D)
    before_f = (dvec[None, :] < f[:, None]).reshape(-1)        # rows before the path's first flip
    tok_ok = ~tmis.reshape(-1)                                  # rows whose draft token agrees
    first_tok = np.where(tmis.any(axis=1), tmis.argmax(axis=1), D)
    before_tok = (dvec[None, :] < first_tok[:, None]).reshape(-1)

    def eq(name, mask):
        if gpu.get(name) is None:
            return
        g = to_np(gpu[name]).reshape(-1)
        o = np.asarray(orc[name]).reshape(-1)
        mism = np.nonzero((g != o) & mask)[0]
        assert mism.size == 0, "%s mismatches at %s: gpu %s oracle %s" % (
            name, mism[:8], g[mism[:8]], o[mism[:8]])

    def close(name, atol, rtol, mask):
        if gpu.get(name) is not None:
            _close_mask(name, to_np(gpu[name]), orc[name], atol, rtol, mask)

    # row-local results
    eq("tokens", tok_ok)
    eq("accept", tok_ok)
    eq("ref_tokens", np.ones(B * K * D, bool))
    close("alpha", ALPHA_ATOL, 0.0, tok_ok)
    close("logq_tok", 2e-5, 1e-6, tok_ok)
    close("logkappa_ref", LOGK_MARGIN, 1e-6, np.ones(B * K * D, bool))
    if kl:  # VSD (KL): the row's top-K term depends on its logits alone
        close("kl_loss", 1e-5, 1e-5, np.ones(B * K * D, bool))
    if gpu.get("row_stats") is not None:
        rs = to_np(gpu["row_stats"]).reshape(-1, 4).astype(np.float64)
        _close_mask("row lse q", rs[:, 0] / T + rs[:, 1], orc["row_lse"][:, 0], 2e-5, 1e-6,
                    np.ones(len(rs), bool))
        _close_mask("row lse p", rs[:, 2] / T + rs[:, 3], orc["row_lse"][:, 1], 2e-5, 1e-6,
                    np.ones(len(rs), bool))
    # path results, up to each path's first flipped decision
    eq("corr_tokens", before_f)
    close("alpha_corr", ALPHA_ATOL, 0.0, before_f)
    close("logq_corr", 2e-5, 1e-6, before_f)
    close("logkappa", LOGK_MARGIN, 1e-6, before_tok)
    close("logkappa_corr", LOGK_MARGIN, 1e-6, before_f)
    eq("accept_len", ~path_div)
    close("expected_len", 1e-5, 1e-5, first_tok == D)
    # the M-step: end to end where no path flipped, conditionally elsewhere
    pre_div = path_div.reshape(B, K).any(axis=1)
    m = orc["margins"].reshape(B, K, D, 6)
    if gpu.get("weights") is not None:
        w = to_np(gpu["weights"]).reshape(B, D, K, 4)
        ow = orc["weights"]
        for b in np.nonzero(~pre_div)[0]:
            for col, mcol in ((0, 3), (1, 4)):
                bad = np.argwhere(w[b][..., col] != ow[b][..., col].astype(np.float32))
                if bad.size == 0:
                    continue
                marg = m[b][bad[:, 1], bad[:, 0], mcol]
                assert (marg < LOGK_MARGIN).all(), \
                    "weight %d differs outside the margin in prefix %d" % (col, b)
                pre_div[b] = True  # an o~/o' comparison flipped near its boundary
    direct = ~pre_div
    near = int((np.minimum(np.minimum(orc["margins"][:, 0], orc["margins"][:, 1]),
                           orc["margins"][:, 2]) < PROB_MARGIN).sum()
               + (np.minimum(orc["margins"][:, 3], orc["margins"][:, 4]) < LOGK_MARGIN).sum())
    ncond = int(pre_div.sum())
    conditional = mstep_inputs is not None and all(
        gpu.get(n) is not None for n in ("logkappa", "logkappa_corr", "logkappa_ref",
                                         "logq_tok", "tokens", "corr_tokens", "loss"))
    if not conditional:
        assert ncond <= exclusion_budget(B) and ncond < B, \
            "too many prefixes with a flipped decision: %d of %d" % (ncond, B)
    SESSION["calls"] += 1
    SESSION["prefixes"] += B
    SESSION["near_boundary_decisions"] += near
    SESSION["diverged_paths"] += ndiv
    SESSION["conditional_prefixes" if conditional else "excluded_prefixes"] += ncond
    if report is not None:
        report.update(near_boundary_decisions=near, diverged_paths=ndiv,
                      conditional_prefixes=ncond if conditional else 0,
                      excluded_prefixes=0 if conditional else ncond)
    if gpu.get("weights") is not None:
        w = to_np(gpu["weights"]).reshape(B, D, K, 4)
        o = orc["weights"]
        assert np.array_equal(w[direct][..., 0], o[direct][..., 0]), "o~ mismatch"
        assert np.allclose(w[direct][..., 1], o[direct][..., 1], rtol=1e-6, atol=0), "o' mismatch"
        assert np.allclose(w[direct][..., 2], o[direct][..., 2], rtol=1e-5, atol=1e-6), \
            "beta mismatch"
        assert np.allclose(w[direct][..., 3], o[direct][..., 3], rtol=1e-5, atol=1e-6), \
            "zeta mismatch"
    if gpu.get("loss") is not None:
        lg = to_np(gpu["loss"]).astype(np.float64)
        lo = orc["loss"]
        for b in np.nonzero(direct)[0]:
            assert abs(lg[b] - lo[b]) <= LOSS_RTOL * max(1.0, abs(lo[b])), \
                "loss[%d] gpu %r oracle %r" % (b, lg[b], lo[b])
        if check_mean and (ncond == 0 or conditional):
            # the mean of the per-prefix losses, each checked above
            lm = float(np.mean(lg[:B])) if ncond else lo[B]
            assert abs(lg[B] - lm) <= LOSS_RTOL * max(1.0, abs(lm)), "mean loss"
    emax = 0.0
    scale = 0.0
    if check_grad and gpu.get("grad") is not None:
        g_all = gpu["grad"]
        o_all = orc["grad"].reshape(B * K * D, V)
        scale = float(np.abs(o_all).max()) if o_all.size else 0.0
        P = K * D
        for b in np.nonzero(direct)[0]:  # prefix blocks: full-size gradients are GBs in fp64
            gb = g_all[b * P * V:(b + 1) * P * V] if g_all.ndim == 1 else g_all[b * P:(b + 1) * P]
            emax = max(emax, _grad_rows("grad", to_np(gb).reshape(P, V),
                                        o_all[b * P:(b + 1) * P], grad_dtype, scale))
    if conditional:
        for b in np.nonzero(pre_div)[0]:
            emax = max(emax, _conditional_mstep(gpu, b, K, D, V, T, grad_dtype, mstep_inputs,
                                                check_grad, scale))
    if report is not None and check_grad:
        report["grad_max_abs_err"] = emax
    return ncond


def mstep_inputs(prob, B_total=None, w_base=1.05, tau_car=0.2, zeta_mode=0, kl_weight=0.0,
                 kl_topk=10):
    """The inputs of the conditional M-step check for a problem dict (draft and
    target logits [B*K*D, V] on any device), as compare_linear takes them."""
    P = prob["K"] * prob["D"]

    def rows(name):
        def get(b):
            return to_np(prob[name][b * P:(b + 1) * P]).astype(np.float32)
        return get

    return dict(draft_rows=rows("draft"), target_rows=rows("target") if "target" in prob else None,
                B_total=B_total or prob["B"], w_base=w_base, tau_car=tau_car,
                zeta_mode=zeta_mode, kl_weight=kl_weight, kl_topk=kl_topk)


def sub_batch(gpu, b0, b1, B, K, D):
    """The GPU outputs of prefixes b0 .. b1-1 of a call over B prefixes, shaped
    as a call over those prefixes alone.  The mean loss entry is replaced by
    prefix b0's loss (a sub-batch has its own mean); the gradient keeps the
    call's 1/B scale, so the caller rescales the oracle's gradient by
    (b1 - b0) / B."""
    P = K * D
    out = {}
    for n, t in gpu.items():
        if t is None:
            continue
        if n in ("accept_len", "expected_len"):
            out[n] = t[b0 * K:b1 * K]
        elif n == "weights":
            out[n] = t[b0:b1]
        elif n == "loss":
            out[n] = t[list(range(b0, b1)) + [b0]]
        elif n == "draft_logits":
            continue
        elif t.shape[0] == B * P:
            out[n] = t[b0 * P:b1 * P]
    return out


def compare_tree(gpu, orc, report=None):
    """Tree parity under the same protocol: a tree is excluded only if a
    near-boundary accept or residual draw went the other way."""
    m = orc["margins"]
    B = m.shape[0]
    div = np.zeros(B, bool)
    ga, oa = to_np(gpu["accept"]), orc["accept"]
    gc, oc = to_np(gpu["corr_tokens"]), orc["corr_tokens"]
    for b in range(B):
        bad = np.nonzero(ga[b] != oa[b])[0]
        if bad.size:
            assert (m[b, bad, 0] < PROB_MARGIN).all(), "accept differs outside the margin"
            div[b] = True
            continue
        bad = np.nonzero(gc[b] != oc[b])[0]
        if bad.size:
            assert (m[b, bad, 1] < PROB_MARGIN).all(), "residual differs outside the margin"
            div[b] = True
    ok = ~div
    SESSION["trees"] += B
    SESSION["excluded_trees"] += int(div.sum())
    if report is not None:
        report["excluded_trees"] = int(div.sum())
    assert div.sum() <= exclusion_budget(B) and div.sum() < B, \
        "too many diverged trees: %d of %d" % (int(div.sum()), B)
    for name in ("accept", "path_accept", "corr_tokens"):
        assert np.array_equal(to_np(gpu[name])[ok], orc[name][ok]), name
    for name in ("deepest", "accept_len", "bonus"):
        assert np.array_equal(to_np(gpu[name])[ok], orc[name][ok]), name
    gal = to_np(gpu["alpha"]).astype(np.float64)
    assert np.allclose(gal[ok], orc["alpha"][ok], atol=ALPHA_ATOL, rtol=0)
    gl = to_np(gpu["logkappa"]).astype(np.float64)
    ol = orc["logkappa"]
    sel = ok[:, None] & np.isfinite(ol)
    assert np.allclose(gl[sel], ol[sel], atol=LOGK_MARGIN, rtol=1e-6)
    # a path the oracle gives zero validity (log kappa = -inf) must be -inf too
    neg = ok[:, None] & np.isneginf(ol)
    assert np.all(np.isneginf(gl[neg])), "log kappa finite where the oracle has -inf"
    return int(div.sum())


def compare_tree_sequential(gpu, orc, report=None):
    """Tree parity under the sequential sibling rule.  The walk visits nodes in
    increasing index order, so the first (lowest-index) node where an accept
    bit or a correction token differs is the decision that flipped: it must be
    within its margin, and the tree is then excluded (budget)."""
    m = orc["margins"]
    B = m.shape[0]
    ga, oa = to_np(gpu["accept"]), orc["accept"]
    gc, oc = to_np(gpu["corr_tokens"]), orc["corr_tokens"]
    div = np.zeros(B, bool)
    for b in range(B):
        bad = np.nonzero((ga[b] != oa[b]) | (gc[b] != oc[b]))[0]
        if bad.size == 0:
            continue
        n = bad[0]
        marg = m[b, n, 0] if ga[b, n] != oa[b, n] else m[b, n, 1]
        assert marg < PROB_MARGIN, "tree %d: decision at node %d differs outside the margin (%g)" % (
            b, n, marg)
        div[b] = True
    ok = ~div
    SESSION["trees"] += B
    SESSION["excluded_trees"] += int(div.sum())
    if report is not None:
        report["excluded_trees"] = int(div.sum())
    assert div.sum() <= exclusion_budget(B) and div.sum() < B, \
        "too many diverged trees: %d of %d" % (int(div.sum()), B)
    for name in ("accept", "path_accept", "corr_tokens"):
        assert np.array_equal(to_np(gpu[name])[ok], orc[name][ok]), name
    for name in ("deepest", "accept_len", "bonus"):
        assert np.array_equal(to_np(gpu[name])[ok], orc[name][ok]), name
    _close_mask("alpha", to_np(gpu["alpha"])[ok], orc["alpha"][ok], ALPHA_ATOL, 1e-6,
                np.ones(orc["alpha"][ok].shape, bool))
    _close_mask("logkappa", to_np(gpu["logkappa"])[ok], orc["logkappa"][ok], LOGK_MARGIN, 1e-6,
                np.ones(orc["logkappa"][ok].shape, bool))
    return int(div.sum())


def compare_tree_em(gpu, orc, B, N, V, grad_dtype="bf16", report=None):
    """Parity of the tree EM: a tree where an accept decision, a corrected
    draw or an o~ comparison went the other way within its margin is
    excluded (budget); every other tree is compared in full."""
    m = orc["margins"]  # [B][N][3]: accept, z' draw, o~
    gz = to_np(gpu["corr_tokens"])
    gw = to_np(gpu["weights"]).reshape(B, N, 4)
    ow = orc["weights"]
    div = np.zeros(B, bool)
    for b in range(B):
        bad = np.nonzero(gz[b] != orc["corr_tokens"][b])[0]
        if bad.size:
            # z' differs: the draw itself, or an accept decision above it
            assert (np.minimum(m[b, :, 0], m[b, :, 1]) < PROB_MARGIN).any(), \
                "tree %d: corrected token differs at %s with no near-boundary decision" % (b, bad[:4])
            div[b] = True
            continue
        bad = np.nonzero(gw[b, :, 0] != ow[b, :, 0])[0]
        if bad.size:
            assert (m[b, bad, 2] < LOGK_MARGIN).all(), "tree %d: o~ differs outside the margin" % b
            div[b] = True
    ok = ~div
    SESSION["trees"] += B
    SESSION["excluded_trees"] += int(div.sum())
    if report is not None:
        report["excluded_trees"] = int(div.sum())
    assert div.sum() <= exclusion_budget(B) and div.sum() < B, \
        "too many diverged trees: %d of %d" % (int(div.sum()), B)
    full = np.ones((int(ok.sum()), N), bool)
    assert np.array_equal(gz[ok], orc["corr_tokens"][ok]), "z'"
    for name, atol in (("logq_tok", 2e-5), ("logq_corr", 2e-5), ("logkappa", LOGK_MARGIN),
                       ("logkappa_corr", LOGK_MARGIN), ("logkappa_ref", LOGK_MARGIN)):
        _close_mask(name, to_np(gpu[name])[ok], orc[name][ok], atol, 1e-6, full)
    assert np.array_equal(gw[ok][..., 0], ow[ok][..., 0]), "o~"
    assert np.allclose(gw[ok][..., 1], ow[ok][..., 1], rtol=1e-6, atol=0), "o'"
    assert np.allclose(gw[ok][..., 2], ow[ok][..., 2], rtol=1e-5, atol=1e-6), "beta"
    assert np.allclose(gw[ok][..., 3], ow[ok][..., 3], rtol=1e-5, atol=1e-6), "zeta"
    lg = to_np(gpu["loss"]).astype(np.float64)
    for b in np.nonzero(ok)[0]:
        assert abs(lg[b] - orc["loss"][b]) <= LOSS_RTOL * max(1.0, abs(orc["loss"][b])), \
            "loss[%d] gpu %r oracle %r" % (b, lg[b], orc["loss"][b])
    if not div.any():
        assert abs(lg[B] - orc["loss"][B]) <= LOSS_RTOL * max(1.0, abs(orc["loss"][B]))
    g_all = gpu["grad"]
    o_all = orc["grad"].reshape(B * N, V)
    scale = float(np.abs(o_all).max()) if o_all.size else 0.0
    emax = 0.0
    for b in np.nonzero(ok)[0]:
        emax = max(emax, _grad_rows("tree grad", to_np(g_all[b * N:(b + 1) * N]).reshape(N, V),
                                    o_all[b * N:(b + 1) * N], grad_dtype, scale))
    if report is not None:
        report["grad_max_abs_err"] = emax
    return int(div.sum())
