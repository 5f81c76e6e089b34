"""Comparison of the CUDA path with the CPU oracle on the same seeded inputs.

Discrete results (sampled tokens, accept bits, accepted lengths, corrected
tokens, oracle utilities) must be bit-exact.  The one exception is a decision
the oracle reports within a margin of its boundary -- |u - alpha| or
|u - CDF boundary| < PROB_MARGIN, or a log-kappa comparison within
LOGK_MARGIN: there the two sides may disagree.  A prefix in which such a
decision disagrees is excluded from every later comparison (its paths and its
M-step legitimately diverge) and counted; a disagreement outside the margins
fails the test.  Prefixes whose decisions all agree, near-boundary ones
included, are compared in full, floats to the tolerances below.
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
# run (tests/conftest.py): near-boundary decisions seen and prefixes excluded.
SESSION = {"calls": 0, "prefixes": 0, "near_boundary_decisions": 0, "excluded_prefixes": 0,
           "trees": 0, "excluded_trees": 0}


def exclusion_budget(B):
    """How many prefixes (or trees) of one call may be excluded.

    A prefix is excluded only when one of its decisions lies within the
    margin of its boundary and the two sides took it differently.  With the
    margins below, a decision falls inside one with probability of order
    1e-5 on these inputs, so an exclusion is rare; the budget allows one per
    ten prefixes (at least one for B >= 3) and none at all for B <= 2, so
    that every call compares at least one prefix in full and a call whose
    only prefixes are excluded fails."""
    if B <= 2:
        return 0
    return max(1, B // 10)


def to_np(t):
    if hasattr(t, "detach"):
        t = t.detach()
        return t.float().cpu().numpy() if t.dtype.is_floating_point else t.cpu().numpy()
    return np.asarray(t)


def _diverged_prefixes(gpu, orc, B, K, D):
    """Per prefix: True if a near-boundary decision disagrees; raises on a
    disagreement outside the margins."""
    m = orc["margins"].reshape(B, K, D, 6)
    div = np.zeros(B, bool)

    def check(name, col, thr, shape):
        if name not in gpu or gpu.get(name) is None:
            return
        g = to_np(gpu[name]).reshape(shape)
        o = np.asarray(orc[name]).reshape(shape)
        for b in range(B):
            if div[b]:
                continue
            bad = np.argwhere(g[b] != o[b])
            if bad.size == 0:
                continue
            marg = m[b][tuple(bad.T)][:, col] if col is not None else np.zeros(len(bad))
            far = marg >= thr
            assert not far.any(), "%s differs outside the margin in prefix %d at %s (margin %s)" % (
                name, b, bad[far][:4].tolist(), marg[far][:4])
            div[b] = True

    check("tokens", 0, PROB_MARGIN, (B, K, D))
    check("accept", 1, PROB_MARGIN, (B, K, D))
    if "ref_tokens" in gpu and gpu.get("ref_tokens") is not None:
        g = to_np(gpu["ref_tokens"]).reshape(B, K, D)
        o = np.asarray(orc["ref_tokens"]).reshape(B, K, D)
        for b in range(B):
            if not div[b]:
                assert np.array_equal(g[b], o[b]), "argmax differs in prefix %d" % b
    check("corr_tokens", 2, PROB_MARGIN, (B, K, D))
    if gpu.get("weights") is not None:
        w = to_np(gpu["weights"]).reshape(B, D, K, 4)
        ow = orc["weights"]
        for b in range(B):
            if div[b]:
                continue
            for col, mcol in ((0, 3), (1, 4)):
                bad = np.argwhere(w[b][..., col] != ow[b][..., col].astype(np.float32))
                if bad.size == 0:
                    continue
                marg = m[b][bad[:, 1], bad[:, 0], mcol]
                assert (marg < LOGK_MARGIN).all(), "weight %d differs outside the margin" % col
                div[b] = True
    return div


def compare_linear(gpu, orc, B, K, D, V, T, grad_dtype="f32", check_grad=True, report=None):
    """Assert parity of E-step/M-step outputs; returns the number of prefixes
    excluded because a near-boundary decision went the other way."""
    div = _diverged_prefixes(gpu, orc, B, K, D)
    ok = ~div
    rows_ok = np.repeat(ok, K * D)
    paths_ok = np.repeat(ok, K)
    nbad = int(div.sum())
    m = orc["margins"]
    near = int((np.minimum(np.minimum(m[:, 0], m[:, 1]), m[:, 2]) < PROB_MARGIN).sum()
               + (np.minimum(m[:, 3], m[:, 4]) < LOGK_MARGIN).sum())
    SESSION["calls"] += 1
    SESSION["prefixes"] += B
    SESSION["near_boundary_decisions"] += near
    SESSION["excluded_prefixes"] += nbad
    if report is not None:
        report["excluded_prefixes"] = nbad
        report["near_boundary_decisions"] = near
    assert nbad <= exclusion_budget(B) and nbad < B, \
        "too many diverged prefixes: %d of %d" % (nbad, B)

    def eq(name, mask=rows_ok):
        g = to_np(gpu[name]).reshape(-1)
        o = np.asarray(orc[name]).reshape(-1)
        mism = np.nonzero((g != o) & mask)[0]
        assert mism.size == 0, "%s mismatches at %s: gpu %s oracle %s" % (
            name, mism[:8], g[mism[:8]], o[mism[:8]])

    def close(name, atol, rtol=0.0, mask=rows_ok):
        g = to_np(gpu[name]).reshape(-1).astype(np.float64)
        o = np.asarray(orc[name], dtype=np.float64).reshape(-1)
        both_inf = np.isinf(g) & np.isinf(o) & (np.sign(g) == np.sign(o))
        both_nan = np.isnan(g) & np.isnan(o)
        with np.errstate(invalid="ignore"):
            err = np.where(both_inf | both_nan, 0.0, np.abs(g - o))
        lim = atol + rtol * np.abs(np.where(np.isfinite(o), o, 0))
        # written as "not within": a NaN or a lone infinity on either side fails
        badi = np.nonzero(~(err <= lim) & mask)[0]
        assert badi.size == 0, "%s off at %s: gpu %s oracle %s" % (
            name, badi[:8], g[badi[:8]], o[badi[:8]])

    for n in ("tokens", "accept", "corr_tokens", "ref_tokens"):
        if gpu.get(n) is not None:
            eq(n)
    eq("accept_len", mask=paths_ok)
    if gpu.get("alpha") is not None:
        close("alpha", ALPHA_ATOL)
    if gpu.get("alpha_corr") is not None:
        close("alpha_corr", ALPHA_ATOL)
    for n in ("logq_tok", "logq_corr"):
        if gpu.get(n) is not None:
            close(n, 2e-5, 1e-6)
    for n in ("logkappa", "logkappa_corr", "logkappa_ref"):
        if gpu.get(n) is not None:
            close(n, LOGK_MARGIN, 1e-6)
    if gpu.get("expected_len") is not None:
        close("expected_len", 1e-5, 1e-5, mask=paths_ok)
    if gpu.get("row_stats") is not None:
        rs = to_np(gpu["row_stats"]).reshape(-1, 4).astype(np.float64)
        lse_q = rs[:, 0] / T + rs[:, 1]
        lse_p = rs[:, 2] / T + rs[:, 3]
        assert np.allclose(lse_q, orc["row_lse"][:, 0], atol=2e-5, rtol=1e-6)
        assert np.allclose(lse_p, orc["row_lse"][:, 1], atol=2e-5, rtol=1e-6)
    if gpu.get("weights") is not None:
        w = to_np(gpu["weights"]).reshape(B, D, K, 4)
        o = orc["weights"]
        assert np.array_equal(w[ok][..., 0], o[ok][..., 0]), "o~ mismatch"
        assert np.allclose(w[ok][..., 1], o[ok][..., 1], rtol=1e-6, atol=0), "o' mismatch"
        assert np.allclose(w[ok][..., 2], o[ok][..., 2], rtol=1e-5, atol=1e-6), "beta mismatch"
        assert np.allclose(w[ok][..., 3], o[ok][..., 3], rtol=1e-5, atol=1e-6), "zeta mismatch"
    if gpu.get("loss") is not None:
        lg = to_np(gpu["loss"]).astype(np.float64)
        lo = orc["loss"]
        for b in np.nonzero(ok)[0]:
            assert abs(lg[b] - lo[b]) <= LOSS_RTOL * max(1.0, abs(lo[b])), \
                "loss[%d] gpu %r oracle %r" % (b, lg[b], lo[b])
        if nbad == 0:
            assert abs(lg[B] - lo[B]) <= LOSS_RTOL * max(1.0, abs(lo[B])), "mean loss"
    if check_grad and gpu.get("grad") is not None:
        g = to_np(gpu["grad"]).reshape(B * K * D, V).astype(np.float64)
        o = orc["grad"].reshape(B * K * D, V)
        scale = np.abs(o).max() if o.size else 0.0
        if grad_dtype == "bf16":
            lim = 2.0 ** -8 * np.abs(o) + 1e-6 * scale + 1e-30
        else:
            lim = 1e-5 * np.abs(o) + 1e-6 * scale + 1e-30
        err = np.abs(g - o)
        badr = np.nonzero((~(err <= lim)).any(axis=1) & rows_ok)[0]
        assert badr.size == 0, "grad rows off: %s, max err %g (scale %g)" % (
            badr[:8], err[badr].max(), scale)
        emax = float(err[rows_ok].max()) if rows_ok.any() else 0.0
        assert emax <= 1e-3  # max-abs bar for gradients
        if report is not None:
            report["grad_max_abs_err"] = emax
    return nbad


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
