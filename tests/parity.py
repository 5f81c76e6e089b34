"""Comparison of the CUDA path with the CPU oracle on the same seeded inputs.

Discrete results (tokens, accept bits, accepted lengths) must be bit-exact,
except in prefixes where the oracle reports a decision within a margin of its
boundary: |u - alpha| or |u - CDF boundary| < 1e-6 (probability scale), or
|log kappa - log kappa_ref| < LOGK_MARGIN (log scale).  Such prefixes are
excluded from the comparison and counted.  Floating-point results are held to
the tolerances below.
"""
import math

import numpy as np

PROB_MARGIN = 1e-6
# log-kappa comparisons add D log-alpha terms, each carrying the float32
# rounding of a log-probability (|log p| <= ~20, 2^-24 relative) and of the
# log-partition; D * 2e-6 bounds their sum for D <= 64 with room to spare.
LOGK_MARGIN = 1e-5
LOSS_RTOL = 1e-5
ALPHA_ATOL = 2e-6


def to_np(t):
    return t.detach().float().cpu().numpy() if t.dtype.is_floating_point else t.detach().cpu().numpy()


def flagged_prefixes(orc, B, K, D):
    m = orc["margins"].reshape(B, K * D, 6)
    prob = np.minimum(np.minimum(m[..., 0], m[..., 1]), m[..., 2])
    logk = np.minimum(m[..., 3], m[..., 4])
    bad = (prob < PROB_MARGIN).any(axis=1) | (logk < LOGK_MARGIN).any(axis=1)
    return bad


def compare_linear(gpu, orc, B, K, D, V, T, grad_dtype="f32", check_grad=True, report=None):
    """Assert parity of fused/verify outputs; returns the number of excluded prefixes."""
    bad = flagged_prefixes(orc, B, K, D)
    ok = ~bad
    rows_ok = np.repeat(ok, K * D)
    paths_ok = np.repeat(ok, K)
    nbad = int(bad.sum())
    if report is not None:
        report["excluded_prefixes"] = nbad
    assert nbad <= max(1, B // 10), "too many near-boundary prefixes: %d of %d" % (nbad, B)

    def eq(name, gname=None, mask=rows_ok):
        g = to_np(gpu[gname or name]).reshape(-1)
        o = np.asarray(orc[name]).reshape(-1)
        mism = np.nonzero((g != o) & mask)[0]
        assert mism.size == 0, "%s mismatches at %s: gpu %s oracle %s" % (
            name, mism[:8], g[mism[:8]], o[mism[:8]])

    def close(name, atol, rtol=0.0, mask=rows_ok, gname=None):
        g = to_np(gpu[gname or name]).reshape(-1).astype(np.float64)
        o = np.asarray(orc[name], dtype=np.float64).reshape(-1)
        both_inf = np.isinf(g) & np.isinf(o) & (np.sign(g) == np.sign(o))
        err = np.where(both_inf, 0.0, np.abs(g - o))
        lim = atol + rtol * np.abs(np.where(np.isinf(o), 0, o))
        badi = np.nonzero((err > lim) & mask)[0]
        assert badi.size == 0, "%s off at %s: gpu %s oracle %s" % (
            name, badi[:8], g[badi[:8]], o[badi[:8]])

    if "tokens" in gpu:
        eq("tokens")
    if "accept" in gpu:
        eq("accept")
    eq("accept_len", mask=paths_ok)
    eq("corr_tokens")
    if "ref_tokens" in gpu:
        eq("ref_tokens")
    if "alpha" in gpu:
        close("alpha", ALPHA_ATOL)
    if "alpha_corr" in gpu:
        close("alpha_corr", ALPHA_ATOL)
    if "logq_tok" in gpu:
        close("logq_tok", 2e-5, 1e-6)
    if "logq_corr" in gpu:
        close("logq_corr", 2e-5, 1e-6)
    close("logkappa", LOGK_MARGIN, 1e-6)
    for n in ("logkappa_corr", "logkappa_ref"):
        if n in gpu:
            close(n, LOGK_MARGIN, 1e-6)
    if "expected_len" in gpu:
        close("expected_len", 1e-5, 1e-5, mask=paths_ok)
    if "row_stats" in gpu:
        rs = to_np(gpu["row_stats"]).reshape(-1, 4).astype(np.float64)
        lse_q = rs[:, 0] / T + rs[:, 1]
        lse_p = rs[:, 2] / T + rs[:, 3]
        assert np.allclose(lse_q, orc["row_lse"][:, 0], atol=2e-5, rtol=1e-6)
        assert np.allclose(lse_p, orc["row_lse"][:, 1], atol=2e-5, rtol=1e-6)
    if "weights" in gpu and gpu.get("weights") is not None:
        w = to_np(gpu["weights"]).reshape(B, D, K, 4)
        o = orc["weights"]
        assert np.array_equal(w[ok][..., 0], o[ok][..., 0]), "o~ mismatch"
        assert np.allclose(w[ok][..., 1], o[ok][..., 1], rtol=1e-6, atol=0), "o' mismatch"
        assert np.allclose(w[ok][..., 2], o[ok][..., 2], rtol=1e-5, atol=1e-6), "beta mismatch"
        assert np.allclose(w[ok][..., 3], o[ok][..., 3], rtol=1e-5, atol=1e-6), "zeta mismatch"
    if "loss" in gpu and gpu.get("loss") is not None:
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
        badr = np.nonzero(((err > lim).any(axis=1)) & rows_ok)[0]
        assert badr.size == 0, "grad rows off: %s, max err %g (scale %g)" % (
            badr[:8], err[badr].max(), scale)
        # the benchmark spec bar: max-abs 1e-3
        assert (err[rows_ok] if rows_ok.any() else np.zeros(1)).max() <= 1e-3
        if report is not None:
            report["grad_max_abs_err"] = float(err[rows_ok].max()) if rows_ok.any() else 0.0
    return nbad


def compare_tree(gpu, orc):
    """Tree parity: exact bits/tokens except near-boundary trees, which are counted."""
    m = orc["margins"]
    bad = (np.minimum(m[..., 0], m[..., 1]) < PROB_MARGIN).any(axis=1)
    ok = ~bad
    assert bad.sum() <= max(1, len(bad) // 10)
    for name in ("accept", "path_accept", "corr_tokens"):
        g = to_np(gpu[name])
        assert np.array_equal(g[ok], orc[name][ok]), name
    for name in ("deepest", "accept_len", "bonus"):
        g = to_np(gpu[name])
        assert np.array_equal(g[ok], orc[name][ok]), name
    ga = to_np(gpu["alpha"]).astype(np.float64)
    assert np.allclose(ga[ok], orc["alpha"][ok], atol=ALPHA_ATOL, rtol=0)
    gl = to_np(gpu["logkappa"]).astype(np.float64)
    ol = orc["logkappa"]
    fin = np.isfinite(ol)
    assert np.allclose(gl[ok & fin], ol[ok & fin], atol=LOGK_MARGIN, rtol=1e-6)
    return int(bad.sum())
