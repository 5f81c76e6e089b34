"""Pins of the CPU oracle to facts fixed by the paper and by mathematics.

Every test here checks the oracle against something other than itself:
exact lattice enumerations over the uniforms with dyadic distributions (so the
expected probabilities are exact), closed forms from Sec. 4.4, special cases
that reduce to library routines (cross-entropy and its autograd), hand-derived
worked examples stored under tests/golden/, theorems of Sec. 4.4 checked by
brute force, and finite differences of the oracle's own objective.
"""
import json
import math
import os

import numpy as np
import pytest

GOLDEN = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "worked_examples.json")))

Q4 = np.array([1 / 2, 1 / 4, 1 / 8, 1 / 8])
P_UNI = np.array([1 / 4, 1 / 4, 1 / 4, 1 / 4])
P_B = np.array([1 / 8, 3 / 8, 1 / 4, 1 / 4])


def logits(prob, scale=1.0):
    return (scale * np.log(np.asarray(prob, dtype=np.float64))).astype(np.float32)


def lattice(M):
    return ((np.arange(M) + 0.5) / M).astype(np.float32)


def midpoint(prob, t):
    """A uniform that the inverse CDF maps to token t (middle of its interval)."""
    F = np.concatenate([[0.0], np.cumsum(prob)])
    return np.float32((F[t] + F[t + 1]) / 2)


# --------------------------------------------------------------------------
# Eq. 1 distributions and the inverse-CDF draw


def test_log_softmax_closed_forms(oracle):
    # equal logits -> uniform
    lp = oracle.log_softmax(np.full(7, 3.25, np.float32), 1.0)
    assert np.allclose(np.exp(lp), 1 / 7, rtol=0, atol=1e-15)
    # two tokens: softmax is the logistic function of the gap over T
    for T in (0.5, 1.0, 2.0):
        lp = oracle.log_softmax(np.array([0.0, 1.5], np.float32), T)
        assert abs(np.exp(lp[1]) - 1 / (1 + math.exp(-1.5 / T))) < 1e-15
    # temperature: logits c*x at T=c equal x at T=1
    x = np.random.default_rng(0).normal(size=33).astype(np.float32)
    a = oracle.log_softmax(x * 4, 4.0)
    b = oracle.log_softmax(x, 1.0)
    assert np.allclose(a, b, atol=1e-13)


def test_inverse_cdf_lattice_is_exact(oracle):
    M = 64
    counts = np.zeros(4)
    for u in lattice(M):
        v, m = oracle.sample(Q4, u)
        counts[v] += 1
        assert m > 0
    assert np.array_equal(counts / M, Q4)


def test_inverse_cdf_boundaries(oracle):
    # strict u < F(v): a uniform on a boundary goes to the next token
    assert oracle.sample([0.5, 0.5], 0.5)[0] == 1
    assert oracle.sample([0.5, 0.5], 0.0)[0] == 0
    # zero-probability tokens are never drawn
    assert oracle.sample([0.0, 0.5, 0.0, 0.5], 0.0)[0] == 1
    assert oracle.sample([0.0, 0.5, 0.0, 0.5], 0.5)[0] == 3
    # rounding that leaves no crossing picks the last token with mass
    assert oracle.sample([0.25, 0.25, 0.0], 0.75)[0] == 1


# --------------------------------------------------------------------------
# Sec. 3: the accept/resample mixture reproduces the target distribution


@pytest.mark.parametrize("T", [1.0, 2.0])
def test_mixture_reproduces_target_exactly(oracle, T):
    M = 16
    ud, ua, uc = np.meshgrid(lattice(M), lattice(M), lattice(M), indexing="ij")
    B = M ** 3
    draft = np.tile(logits(Q4, T), (B, 1))
    target = np.tile(logits(P_UNI, T), (B, 1))
    o = oracle.linear(draft, target, T, ud.ravel(), ua.ravel(), uc.ravel(), K=1, D=1,
                      want_grad=False)
    out = o["corr_tokens"]
    hist = np.bincount(out, minlength=4) / B
    assert np.array_equal(hist, P_UNI)
    # acceptance rate sum_v min(p, q)
    assert o["accept"].mean() == np.minimum(P_UNI, Q4).sum()
    # a residual token always has p > q, so its alpha is 1 and the corrected
    # path's log kappa is 0; an accepted token keeps its own alpha
    rej = o["accept"] == 0
    assert np.all(o["alpha_corr"][rej] == 1.0)
    assert np.all(o["logkappa_corr"][rej] == 0.0)
    assert np.array_equal(o["alpha_corr"][~rej], o["alpha"][~rej])
    assert np.allclose(o["logkappa_corr"], np.log(o["alpha_corr"]), rtol=0, atol=1e-15)
    assert set(np.unique(out[rej])) <= {2, 3}


def test_mixture_random_distributions(oracle):
    """Non-dyadic p, q: lattice histogram within the lattice's resolution of p."""
    rng = np.random.default_rng(5)
    V = 6
    xq = rng.normal(0, 1.5, V).astype(np.float32)
    xp = rng.normal(0, 1.5, V).astype(np.float32)
    M = 40
    ud, ua, uc = np.meshgrid(lattice(M), lattice(M), lattice(M), indexing="ij")
    B = M ** 3
    o = oracle.linear(np.tile(xq, (B, 1)), np.tile(xp, (B, 1)), 1.0, ud.ravel(), ua.ravel(),
                      uc.ravel(), K=1, D=1, want_grad=False)
    hist = np.bincount(o["corr_tokens"], minlength=V) / B
    p = np.exp(xp - xp.max()) / np.exp(xp - xp.max()).sum()
    assert np.abs(hist - p).max() < 4.0 / M


# --------------------------------------------------------------------------
# Sec. 4.4: survival S_k and the expected accepted length


def _three_step_rows():
    rows_q = [Q4, Q4, P_UNI]
    rows_p = [P_UNI, P_B, P_B]
    toks = [0, 0, 1]  # alphas 1/2, 1/4, 1
    return rows_q, rows_p, toks


def test_survival_and_expected_length(oracle):
    g = GOLDEN["expected_length_three_steps"]
    rows_q, rows_p, toks = _three_step_rows()
    M = 16
    a0, a1, a2 = np.meshgrid(lattice(M), lattice(M), lattice(M), indexing="ij")
    B = M ** 3
    draft = np.tile(np.stack([logits(r) for r in rows_q]), (B, 1))
    target = np.tile(np.stack([logits(r) for r in rows_p]), (B, 1))
    ud = np.tile([midpoint(rows_q[d], toks[d]) for d in range(3)], B)
    ua = np.stack([a0.ravel(), a1.ravel(), a2.ravel()], 1).ravel()
    uc = np.full(B * 3, 0.5, np.float32)
    o = oracle.linear(draft, target, 1.0, ud, ua, uc, K=1, D=3, want_grad=False)
    assert np.array_equal(o["tokens"].reshape(B, 3)[0], toks)
    A = o["accept_len"]
    for k in range(1, 4):
        assert np.mean(A >= k) == g["survival"][k - 1]
    assert np.mean(A) == g["expected_length"]
    assert np.allclose(o["expected_len"], g["expected_length"], atol=1e-14)
    assert np.allclose(np.exp(o["logkappa"].reshape(B, 3)), g["survival"], atol=1e-14)


def test_correction_after_first_rejection_samples_p(oracle):
    """Reading R3: residual at the first rejection, then p-samples."""
    M = 16
    c0, c1 = np.meshgrid(lattice(M), lattice(M), indexing="ij")
    B = M * M
    draft = np.tile(np.stack([logits(Q4), logits(Q4)]), (B, 1))
    target = np.tile(np.stack([logits(P_UNI), logits(P_B)]), (B, 1))
    ud = np.tile([midpoint(Q4, 0), midpoint(Q4, 0)], B)
    ua = np.full(2 * B, 0.99, np.float32)  # alpha_0 = 1/2 -> rejected, A = 0
    uc = np.stack([c0.ravel(), c1.ravel()], 1).ravel()
    o = oracle.linear(draft, target, 1.0, ud, ua, uc, K=1, D=2, want_grad=False)
    assert np.all(o["accept_len"] == 0)
    z = o["corr_tokens"].reshape(B, 2)
    assert np.array_equal(np.bincount(z[:, 0], minlength=4) / B, [0, 0, 0.5, 0.5])
    assert np.array_equal(np.bincount(z[:, 1], minlength=4) / B, P_B)


def test_accept_tie_and_full_acceptance(oracle):
    """u = alpha accepts (Eq. 1 text 'r <= alpha'); A = D keeps z' = z~."""
    rng = np.random.default_rng(1)
    K, D, V = 2, 3, 9
    x = rng.normal(0, 2, (K * D, V)).astype(np.float32)
    o = oracle.linear(x, x, 1.0, rng.random(K * D), np.ones(K * D), rng.random(K * D),
                      K=K, D=D, want_grad=False)
    assert np.all(o["alpha"] == 1.0) and np.all(o["accept"] == 1)
    assert np.all(o["accept_len"] == D)
    assert np.array_equal(o["corr_tokens"], o["tokens"])
    assert np.allclose(o["expected_len"], D)


def test_greedy_reference_tokens(oracle):
    """Algorithm 2 reference: argmax of the target row, lowest index on ties."""
    V = 8
    target = np.array([[0, 3, 1, 3, -2, 3, 0, 1]], np.float32)
    draft = np.zeros((1, V), np.float32)
    o = oracle.linear(draft, target, 1.0, [0.3], [0.3], [0.3], K=1, D=1, want_grad=False)
    assert o["ref_tokens"][0] == 1
    p = np.exp(target[0] - target[0].max()); p /= p.sum()
    assert abs(o["logkappa_ref"][0] - math.log(min(1.0, p[1] / (1 / V)))) < 1e-14


# --------------------------------------------------------------------------
# M-step special cases


def _ce_weighted(draft, T, tokens, weights):
    """Library cross-entropy with per-row weights, and its autograd."""
    torch = pytest.importorskip("torch")
    import torch.nn.functional as F
    x = torch.tensor(draft, dtype=torch.float64, requires_grad=True)
    ce = F.cross_entropy(x / T, torch.tensor(tokens, dtype=torch.int64), reduction="none")
    loss = (torch.tensor(weights, dtype=torch.float64) * ce).sum()
    loss.backward()
    return loss.item(), x.grad.numpy()


@pytest.mark.parametrize("D,T", [(1, 1.0), (4, 0.7)])
def test_single_proposal_is_weighted_cross_entropy(oracle, D, T):
    """K = 1: beta = 0 (empty leave-one-out sum), so Eq. advance reduces to the
    basic gradient (Eq. basic), a w(l)-weighted cross-entropy of the kept path."""
    rng = np.random.default_rng(2)
    B, V = 3, 11
    R = B * D
    draft = rng.normal(0, 2, (R, V)).astype(np.float32)
    target = (draft + rng.normal(0, 0.5, (R, V))).astype(np.float32)
    ref = np.full(B * D, -1e30, np.float32)  # every proposal passes the oracle
    o = oracle.linear(draft, target, T, rng.random(R), rng.random(R), rng.random(R), K=1, D=D,
                      ref_logkappa=ref)
    w = o["weights"]
    assert np.all(w[..., 0] == 1.0) and np.all(w[..., 2] == 0.0)
    wl = 1.05 ** np.arange(1, D + 1)
    assert np.allclose(w[:, :, 0, 1], wl)
    # row d of path is counted by every l >= d
    row_w = np.array([wl[d:].sum() for d in range(D)]) / wl.sum()
    loss, grad = _ce_weighted(draft, T, o["tokens"], np.tile(row_w, B) / B)
    assert abs(o["loss"][B] - loss) < 1e-12
    assert np.allclose(o["grad"], grad, atol=1e-14)


def test_draft_equals_target_closed_form(oracle):
    """draft == target: alpha = 1, o~ = 1, o' = w(l), beta = 1 (Sec. 4.3 'automatic
    early stopping'); with tau -> infinity zeta = 1/K, and the loss is the
    cross-entropy of z~ weighted by w(l)(1 - 1/K) / N_b."""
    rng = np.random.default_rng(3)
    B, K, D, V = 2, 3, 4, 13
    R = B * K * D
    x = rng.normal(0, 2, (R, V)).astype(np.float32)
    o = oracle.linear(x, x, 1.0, rng.random(R), rng.random(R), rng.random(R), K=K, D=D,
                      tau_car=1e30)
    w = o["weights"]
    wl = 1.05 ** np.arange(1, D + 1)
    assert np.all(w[..., 0] == 1.0)
    assert np.allclose(w[..., 1], wl[None, :, None])
    assert np.all(w[..., 2] == 1.0)
    assert np.allclose(w[..., 3], 1.0 / K)
    N = K * wl.sum()
    row_w = np.array([wl[d:].sum() for d in range(D)]) * (1 - 1 / K) / N
    loss, grad = _ce_weighted(x, 1.0, o["tokens"], np.tile(row_w, B * K) / B)
    assert abs(o["loss"][B] - loss) < 1e-12
    assert np.allclose(o["grad"], grad, atol=1e-14)


def _forced_rows(cases):
    """Rows for K proposals of depth 1: (q, p, token, u_accept) per proposal."""
    draft = np.stack([logits(c[0]) for c in cases])
    target = np.stack([logits(c[1]) for c in cases])
    ud = np.array([midpoint(c[0], c[2]) for c in cases], np.float32)
    ua = np.array([c[3] for c in cases], np.float32)
    return draft, target, ud, ua


@pytest.mark.parametrize("name,u1", [("beta_one_rejected", 0.99), ("beta_one_invalid", 0.01)])
def test_beta_worked_examples(oracle, name, u1):
    g = GOLDEN[name]
    cases = [(Q4, Q4, 1, 0.5), (Q4, P_UNI, 0, u1), (P_B, P_B, 2, 0.5)]
    draft, target, ud, ua = _forced_rows(cases)
    o = oracle.linear(draft, target, 1.0, ud, ua, np.full(3, 0.5, np.float32), K=3, D=1,
                      ref_logkappa=np.zeros(1, np.float32))
    w = o["weights"][0, 0]
    assert np.array_equal(w[:, 0], g["o_tilde"])
    assert np.allclose(w[:, 1], g["o_prime"], rtol=0, atol=1e-15)
    assert np.allclose(w[:, 2], g["beta"], rtol=0, atol=1e-15)


@pytest.mark.parametrize("mode,key", [(0, "zeta_prob"), (1, "zeta_logprob")])
def test_zeta_worked_example(oracle, mode, key):
    g = GOLDEN["zeta_two_paths"]
    cases = [(Q4, P_UNI, 0, 0.5), (Q4, P_UNI, 1, 0.5)]  # q(z~) = 1/2, 1/4
    draft, target, ud, ua = _forced_rows(cases)
    o = oracle.linear(draft, target, 1.0, ud, ua, np.full(2, 0.5, np.float32), K=2, D=1,
                      tau_car=0.2, zeta_mode=mode)
    assert np.allclose(o["weights"][0, 0, :, 3], g[key], rtol=0, atol=1e-7)


def test_zeta_uniform_limit(oracle):
    rng = np.random.default_rng(4)
    K, D, V = 5, 3, 10
    R = K * D
    x = rng.normal(0, 2, (R, V)).astype(np.float32)
    y = (x + rng.normal(0, 1, (R, V))).astype(np.float32)
    for mode in (0, 1):
        o = oracle.linear(x, y, 1.0, rng.random(R), rng.random(R), rng.random(R), K=K, D=D,
                          tau_car=1e300, zeta_mode=mode, want_grad=False)
        assert np.allclose(o["weights"][..., 3], 1.0 / K, atol=1e-12)


# --------------------------------------------------------------------------
# Gradient: finite differences of the objective with weights held fixed


def test_gradient_finite_differences(oracle):
    rng = np.random.default_rng(6)
    B, K, D, V, T = 2, 3, 3, 7, 0.8
    R = B * K * D
    # logits on a 2^-8 grid so that x +- h is exact in float32
    draft = (np.round(rng.normal(0, 1.5, (R, V)) * 256) / 256).astype(np.float32)
    target = (draft + np.round(rng.normal(0, 1.0, (R, V)) * 256) / 256).astype(np.float32)
    o = oracle.linear(draft, target, T, rng.random(R), rng.random(R), rng.random(R), K=K, D=D)
    assert np.allclose(o["grad"].sum(axis=1), 0.0, atol=1e-15)
    h = 2.0 ** -8
    for b in range(B):
        rows = slice(b * K * D, (b + 1) * K * D)
        wts = o["weights"][b]
        N = wts[..., 1].sum()
        tok = o["tokens"][rows]
        ctok = o["corr_tokens"][rows]
        x0 = draft[rows].reshape(K, D, V)
        J, g = oracle.prefix_objective(x0, T, tok, ctok, wts, N, B)
        assert abs(-J / N / B - o["loss"][b] / B) < 1e-13
        assert np.allclose(g.reshape(-1, V), o["grad"][rows], atol=1e-15)
        for (s, d, v) in [(0, 0, 0), (1, 2, 3), (2, 1, 6), (0, 2, tok[2])]:
            xp, xm = x0.copy(), x0.copy()
            xp[s, d, v] += h
            xm[s, d, v] -= h
            Jp, _ = oracle.prefix_objective(xp, T, tok, ctok, wts, N, B, want_grad=False)
            Jm, _ = oracle.prefix_objective(xm, T, tok, ctok, wts, N, B, want_grad=False)
            fd = -(Jp - Jm) / (2 * h) / N / B
            assert abs(fd - g[s, d, v]) < 1e-5 * max(1.0, abs(g[s, d, v]))


def test_reference_input_is_used(oracle):
    rng = np.random.default_rng(7)
    B, K, D, V = 2, 2, 3, 6
    R = B * K * D
    x = rng.normal(0, 2, (R, V)).astype(np.float32)
    y = (x + rng.normal(0, 1, (R, V))).astype(np.float32)
    ref = rng.normal(-1, 0.3, B * D).astype(np.float32)
    o = oracle.linear(x, y, 1.0, rng.random(R), rng.random(R), rng.random(R), K=K, D=D,
                      ref_logkappa=ref, want_grad=False)
    lkr = o["logkappa_ref"].reshape(B, K, D)
    assert np.allclose(lkr, ref.reshape(B, 1, D))
    ot = o["weights"][..., 0]  # [B, D, K]
    lk = o["logkappa"].reshape(B, K, D).transpose(0, 2, 1)
    assert np.array_equal(ot, (lk >= ref.reshape(B, D, 1)).astype(float))


# --------------------------------------------------------------------------
# Tree verification


def test_chain_tree_equals_linear_path(oracle):
    rng = np.random.default_rng(8)
    D, V = 6, 12
    x = rng.normal(0, 2, (D, V)).astype(np.float32)
    y = (x + rng.normal(0, 1, (D, V))).astype(np.float32)
    ud, ua, uc = rng.random(D), rng.random(D), rng.random(D)
    lin = oracle.linear(x, y, 1.0, ud, ua, uc, K=1, D=D, want_grad=False)
    N = D + 1
    xt = np.concatenate([x, np.zeros((1, V), np.float32)])
    yt = np.concatenate([y, np.zeros((1, V), np.float32)])
    parent = np.arange(-1, N - 1, dtype=np.int32)[None]
    tokens = np.concatenate([[0], lin["tokens"]])[None]
    tr = oracle.tree(xt, yt, 1.0, parent, tokens, np.concatenate([[0], ua])[None],
                     np.concatenate([[0], uc])[None])
    assert np.allclose(tr["alpha"][0, 1:], lin["alpha"])
    assert np.allclose(tr["logkappa"][0, 1:], lin["logkappa"])
    A = lin["accept_len"][0]
    assert tr["accept_len"][0] == A and tr["deepest"][0] == A
    if A < D:
        assert tr["corr_tokens"][0, A + 1] == lin["corr_tokens"][A]
        assert tr["bonus"][0] == lin["corr_tokens"][A]


def test_tree_acceptance_lattice(oracle):
    """P(node n on an accepted path) = product of alpha along its ancestors."""
    # root -> {1, 2}; 1 -> {3}; 3 -> {4}
    parent = np.array([-1, 0, 0, 1, 3], np.int32)
    N, V = 5, 4
    rq = [Q4, Q4, P_UNI, Q4, P_UNI]
    rp = [P_UNI, P_B, P_B, P_UNI, P_UNI]
    # node tokens drawn at the parent's row: node1 tok0 (alpha 1/2), node2 tok1
    # (alpha 1), node3 tok0 at row1 (alpha 1/4), node4 tok0 at row3 (alpha 1/2)
    tok = np.array([0, 0, 1, 0, 0], np.int32)
    M = 8
    grids = np.meshgrid(*([lattice(M)] * 4), indexing="ij")
    B = M ** 4
    ua = np.zeros((B, N), np.float32)
    for i in range(4):
        ua[:, i + 1] = grids[i].ravel()
    draft = np.tile(np.stack([logits(r) for r in rq]), (B, 1))
    target = np.tile(np.stack([logits(r) for r in rp]), (B, 1))
    tr = oracle.tree(draft, target, 1.0, np.tile(parent, (B, 1)), np.tile(tok, (B, 1)), ua,
                     np.full((B, N), 0.3, np.float32))
    pa = tr["path_accept"].mean(axis=0)
    assert np.array_equal(pa, [1, 1 / 2, 1, 1 / 8, 1 / 16])
    # deepest: node 4 (depth 3) when accepted, else 3, else 1 or 2 (lowest index)
    d = tr["accept_len"]
    assert np.mean(d == 3) == 1 / 16 and np.mean(d == 2) == 1 / 8 - 1 / 16
    assert np.all(tr["deepest"][d == 1] == np.where(tr["path_accept"][d == 1, 1] == 1, 1, 2))


def test_tree_residual_and_bonus_distributions(oracle):
    """Root with two leaf children, dyadic rows, a lattice over the uniforms:
    child 1 (token 0 at the root row, alpha = 1/2) is accepted half the time;
    when it is rejected its correction token follows norm(max(0, p - q)) of
    the root row; child 2 (alpha = 1) is always accepted; the bonus is the
    p-draw at the deepest accepted node's row (a leaf here: child 1 if
    accepted, else child 2), so it follows (P_B + P_UNI) / 2 (Sec. 3, App. E)."""
    parent = np.array([-1, 0, 0], np.int32)
    tok = np.array([0, 0, 2], np.int32)
    rq = [Q4, Q4, Q4]
    rp = [P_UNI, P_B, P_UNI]
    M = 8
    g = np.meshgrid(lattice(M), lattice(M), lattice(M), indexing="ij")
    B = M ** 3
    ua = np.zeros((B, 3), np.float32)
    uc = np.zeros((B, 3), np.float32)
    ua[:, 1] = g[0].ravel()
    ua[:, 2] = 0.999
    uc[:, 1] = g[1].ravel()
    uc[:, 2] = g[2].ravel()
    draft = np.tile(np.stack([logits(r) for r in rq]), (B, 1))
    target = np.tile(np.stack([logits(r) for r in rp]), (B, 1))
    tr = oracle.tree(draft, target, 1.0, np.tile(parent, (B, 1)), np.tile(tok, (B, 1)), ua, uc)
    acc1 = tr["path_accept"][:, 1] == 1
    assert acc1.mean() == 1 / 2 and (tr["path_accept"][:, 2] == 1).all()
    assert (tr["accept_len"] == 1).all()
    assert np.array_equal(tr["deepest"], np.where(acc1, 1, 2))
    # residual of the root row: max(0, P_UNI - Q4) = (0, 0, 1/8, 1/8), normalised
    c1 = tr["corr_tokens"][~acc1, 1]
    assert np.array_equal(np.bincount(c1, minlength=4) / c1.size, [0, 0, 1 / 2, 1 / 2])
    assert (tr["corr_tokens"][acc1, 1] == -1).all() and (tr["corr_tokens"][:, 2] == -1).all()
    bonus = np.bincount(tr["bonus"], minlength=4) / B
    assert np.array_equal(bonus, (P_B + P_UNI) / 2)


# --------------------------------------------------------------------------
# Sec. 4.4 theorems by brute force on a tabulated autoregressive toy model


def test_theorems_by_enumeration(oracle):
    rng = np.random.default_rng(9)
    V, D = 3, 3
    import itertools
    paths = list(itertools.product(range(V), repeat=D))
    # tabulated conditionals: one (q, p) row per prefix of length 0..D-1
    tab = {}
    for d in range(D):
        for pre in itertools.product(range(V), repeat=d):
            tab[pre] = (rng.normal(0, 1.5, V).astype(np.float32),
                        rng.normal(0, 1.5, V).astype(np.float32))
    sm = lambda x: np.exp(x - x.max()) / np.exp(x - x.max()).sum()
    draft = np.stack([tab[z[:d]][0] for z in paths for d in range(D)])
    target = np.stack([tab[z[:d]][1] for z in paths for d in range(D)])
    ud = np.array([midpoint(sm(tab[z[:d]][0].astype(np.float64)), z[d]) for z in paths
                   for d in range(D)], np.float32)
    B = len(paths)
    o = oracle.linear(draft, target, 1.0, ud, np.full(B * D, 0.5), np.full(B * D, 0.5), K=1,
                      D=D, want_grad=False)
    assert np.array_equal(o["tokens"].reshape(B, D), np.array(paths))
    logk = o["logkappa"].reshape(B, D)[:, -1]
    lq = o["logq_tok"].reshape(B, D).sum(1)
    lp_path = np.array([sum(np.log(sm(tab[z[:d]][1].astype(np.float64))[z[d]])
                            for d in range(D)) for z in paths])
    q = np.exp(lq)
    assert abs(q.sum() - 1) < 1e-12
    elbo = np.sum(q * (logk + lp_path - lq))
    A = np.sum(q * o["expected_len"])
    assert A >= D * math.exp(elbo)  # Theorem 1
    Z = np.sum(np.exp(lp_path) * np.exp(logk))
    qs = np.exp(lp_path) * np.exp(logk) / Z  # the valid-path posterior, Eq. 4
    elbo_star = np.sum(qs * (logk + lp_path - np.log(qs)))
    elbo_kl = np.sum(np.exp(lp_path) * logk)  # q = p
    assert abs(elbo_star - math.log(Z)) < 1e-12  # Theorem 2, equality
    assert elbo_star > elbo_kl  # Theorem 2, strict when kappa varies
    assert elbo <= elbo_star + 1e-12  # the posterior maximises the ELBO


# --------------------------------------------------------------------------
# The draft LM head (Sec. 5, the draft head's output layer) and bf16 rounding


def test_lmhead_one_hot_rows_pick_weight_columns(oracle):
    """A one-hot hidden state e_k gives logits W[:, k]; e_i + e_j gives the sum
    of two columns.  A transposed operand or a dropped term fails here."""
    rng = np.random.default_rng(5)
    V, H = 7, 5
    W = rng.integers(-9, 10, size=(V, H)).astype(np.float64) / 4
    hid = np.zeros((3, H))
    hid[0, 2] = 1.0
    hid[1, 4] = 1.0
    hid[2, 0] = hid[2, 3] = 1.0
    lg = oracle.lmhead_logits(hid, W)
    assert lg.shape == (3, V)
    assert np.array_equal(lg[0], W[:, 2])
    assert np.array_equal(lg[1], W[:, 4])
    assert np.array_equal(lg[2], W[:, 0] + W[:, 3])


def test_lmhead_closed_form_sums(oracle):
    """hidden = all ones, W[v, k] = v - k: logits[v] = H v - H (H - 1) / 2."""
    V, H = 6, 9
    W = np.subtract.outer(np.arange(V), np.arange(H)).astype(np.float64)
    lg = oracle.lmhead_logits(np.ones((2, H)), W)
    want = H * np.arange(V) - H * (H - 1) / 2
    assert np.array_equal(lg[0], want) and np.array_equal(lg[1], want)


def test_round_bf16_ties_to_even_and_matches_torch(oracle):
    one = 1.0
    # halfway cases: 1 + 2^-8 lies between 1 and 1 + 2^-7 -> even (1);
    # 1 + 3 * 2^-8 between 1 + 2^-7 and 1 + 2^-6 -> even (1 + 2^-6)
    x = np.array([one + 2.0**-8, one + 3 * 2.0**-8, -(one + 2.0**-8), 2.0**-9 * 3, 0.0])
    r = oracle.round_bf16(x)
    assert r.tolist() == [1.0, 1.0 + 2.0**-6, -1.0, 2.0**-9 * 3, 0.0]
    # on float32 inputs (no double rounding) it is torch's round-to-nearest-even cast
    torch = pytest.importorskip("torch")
    f = np.random.default_rng(3).standard_normal(20000).astype(np.float32) * 40
    want = torch.from_numpy(f).to(torch.bfloat16).float().numpy()
    assert np.array_equal(oracle.round_bf16(f.astype(np.float64)), want)


# --------------------------------------------------------------------------
# Algorithm 2's comparison log k(z) >= log k(z-bar): the margin the parity
# protocol uses to decide which disagreements it may excuse.  Each case is
# built by hand so that the answer is known without the oracle.


def test_decision_margin_unequal_sums_is_the_gap(oracle):
    assert oracle.decision_margin(-1.0, -1.5, [-1.0], [3], [-1.5], [4]) == 0.5
    assert oracle.decision_margin(-2.25, -0.25, [-2.25], [3]) == 2.0


def test_decision_margin_clipped_tie_is_smallest_ratio(oracle):
    # both sums 0: every ratio at a position where the tokens differ is >= 0,
    # so min(0, r) clips it; position 0 holds the same token on both paths and
    # cancels exactly (its ratios do not count)
    ra, ta = [-0.4, 0.7, 0.3], [5, 1, 2]
    rb, tb = [-0.4, 0.2, 0.9], [5, 7, 8]
    assert oracle.decision_margin(-0.4, -0.4, ra, ta, rb, tb) == 0.2
    # an input reference of 0 (rb = None): every ratio of the path counts
    assert oracle.decision_margin(0.0, 0.0, [0.6, 0.25], [1, 2]) == 0.25


def test_decision_margin_coincidental_tie_is_zero(oracle):
    # equal sums reached through an unclipped ratio at a differing position:
    # a rounding difference could flip the comparison, so the margin is 0
    ra, ta = [-0.3, 0.5], [1, 2]
    rb, tb = [-0.3, 0.5], [4, 2]
    assert oracle.decision_margin(-0.3, -0.3, ra, ta, rb, tb) == 0.0
    # the same when only the reference's ratio is unclipped
    assert oracle.decision_margin(-0.1, -0.1, [0.4, -0.1], [1, 2], [0.4, -0.1],
                                  [1, 3]) == 0.0


def test_decision_margin_input_reference_tie_is_zero(oracle):
    # an input reference b != 0 equal to the path's sum is a coincidence
    assert oracle.decision_margin(-0.75, -0.75, [0.5, -0.75], [1, 2]) == 0.0
    assert oracle.decision_margin(-0.75, -0.75, [-0.5, -0.25], [1, 2]) == 0.0


def test_margins_of_a_worked_prefix(oracle):
    """The margins the oracle reports for a prefix built by hand: path 0
    accepts both tokens with ratios >= 1 (log k = 0 = the greedy reference,
    every differing ratio clipped), so its o~ margin is the smaller ratio."""
    q = [0.5, 0.25, 0.125, 0.125]
    p = [0.125, 0.5, 0.25, 0.125]
    D = 2
    draft = np.stack([logits(q)] * D)
    target = np.stack([logits(p)] * D)
    # z~ = 1 at both positions (ratio 2), greedy reference = 1 as well -> the
    # paths are equal: every term cancels, the comparison is exact
    ud = np.array([midpoint(q, 1)] * D, np.float32)
    o = oracle.linear(draft, target, 1.0, ud, np.full(D, 0.5, np.float32),
                      np.full(D, 0.5, np.float32), K=1, D=D, want_grad=False)
    assert list(o["tokens"]) == [1, 1] and list(o["ref_tokens"]) == [1, 1]
    assert np.all(np.isinf(o["margins"][:, 3]))
    # z~ = 2 at both positions (ratio 2, clipped): log k = 0 = reference, and
    # the differing positions hold ratios log 2 on both sides
    ud = np.array([midpoint(q, 2)] * D, np.float32)
    o = oracle.linear(draft, target, 1.0, ud, np.full(D, 0.5, np.float32),
                      np.full(D, 0.5, np.float32), K=1, D=D, want_grad=False)
    assert list(o["tokens"]) == [2, 2]
    # (the logits hold log q, log p rounded to float32: ratios within 1e-7 of 2)
    assert np.allclose(o["margins"][:, 3], math.log(2), rtol=0, atol=1e-7)


# --------------------------------------------------------------------------
# VSD (KL): the top-10 renormalised term of Eq. klv (reading R11), pinned to
# torch's cross-entropy with probability targets and its autograd.


def _torch_topk_ce(xq, xp, T, k=10):
    """L and dL/dxq of Eq. klv by torch: top-k of the target (distinct values),
    renormalised softmaxes on them, cross-entropy with soft targets."""
    import torch
    q = torch.tensor(np.asarray(xq, np.float64), requires_grad=True)
    p = torch.tensor(np.asarray(xp, np.float64))
    idx = torch.topk(p, min(k, p.numel())).indices
    phat = torch.softmax(p[idx] / T, dim=0)
    L = torch.nn.functional.cross_entropy((q[idx] / T)[None], phat[None])
    L.backward()
    return float(L.detach()), set(idx.tolist()), q.grad.numpy()


@pytest.mark.parametrize("T", [1.0, 0.7])
def test_topk_ce_matches_torch(oracle, T):
    rng = np.random.default_rng(11)
    for V in (10, 37, 300):
        xq = rng.normal(0, 2, V).astype(np.float32)
        xp = (xq + rng.normal(0, 1, V)).astype(np.float32)
        L, tok, dl = oracle.topk_ce(xq, xp, T, 10)
        Lt, it, gt = _torch_topk_ce(xq, xp, T)
        assert set(tok.tolist()) == it
        assert abs(L - Lt) < 1e-12 * max(1.0, abs(Lt))
        full = np.zeros(V)
        full[tok] = dl
        assert np.allclose(full, gt, rtol=1e-10, atol=1e-14)  # zero outside the top 10
        # cross-entropy = KL(p^ || q^) + H(p^) >= H(p^)
        import torch
        ph = torch.softmax(torch.tensor(xp[tok].astype(np.float64)) / T, 0)
        lqh = torch.log_softmax(torch.tensor(xq[tok].astype(np.float64)) / T, 0)
        kl = float(torch.nn.functional.kl_div(lqh, ph, reduction="sum"))
        H = float(-(ph * torch.log(ph)).sum())
        assert abs(L - (kl + H)) < 1e-12 * max(1.0, abs(L)) and kl >= 0


def test_topk_ce_finite_differences(oracle):
    rng = np.random.default_rng(12)
    xq = rng.normal(0, 1, 40)
    xp = rng.normal(0, 1, 40).astype(np.float32)
    T = 0.8
    L, tok, dl = oracle.topk_ce(xq.astype(np.float32), xp, T, 10)
    # central differences in float64 on logits exactly representable in float32
    for k in (0, 4, 9):
        v = tok[k]
        h = 2.0 ** -10
        xa, xb = xq.astype(np.float32).copy(), xq.astype(np.float32).copy()
        xa[v] += np.float32(h)
        xb[v] -= np.float32(h)
        fd = (oracle.topk_ce(xa, xp, T, 10)[0] - oracle.topk_ce(xb, xp, T, 10)[0]) / (2 * h)
        assert abs(fd - dl[k]) < 1e-6
    other = [v for v in range(40) if v not in set(tok.tolist())][0]
    xa = xq.astype(np.float32).copy()
    xa[other] += np.float32(0.5)
    assert oracle.topk_ce(xa, xp, T, 10)[0] == L  # a logit outside the top 10 does not enter


def test_topk_ce_ties_and_degenerate_rows(oracle):
    # ties at the cut: the lowest indices are kept
    xp = np.zeros(20, np.float32)
    xq = np.arange(20, dtype=np.float32) / 10
    L, tok, dl = oracle.topk_ce(xq, xp, 1.0, 10)
    assert sorted(tok.tolist()) == list(range(10))
    xp = np.array([5, 1, 1, 1, 3, 1, 1, 1, 1, 1, 1, 1, 2], np.float32)
    tok = oracle.topk_ce(np.zeros(13, np.float32), xp, 1.0, 10)[1]
    assert sorted(tok.tolist()) == [0, 1, 2, 3, 4, 5, 6, 7, 8, 12]
    # draft = target: q^ = p^, so the gradient is 0 and L is the entropy of p^
    x = np.array([3.0, 1.0, 0.5, -1.0, 2.0, 0.0, -2.0, 1.5, 0.25, -0.5, -3.0, -4.0], np.float32)
    L, tok, dl = oracle.topk_ce(x, x, 1.0, 10)
    assert np.allclose(dl, 0.0, atol=1e-15)
    import torch
    ph = torch.softmax(torch.tensor(x[tok].astype(np.float64)), 0)
    assert abs(L - float(-(ph * torch.log(ph)).sum())) < 1e-12
    # fewer than 10 tokens: the whole vocabulary, i.e. the ordinary soft-target
    # cross-entropy of the full softmaxes
    xq = np.array([0.3, -1.2, 2.0, 0.7, -0.1, 1.1], np.float32)
    xp = np.array([1.0, 0.2, -0.4, 0.9, 2.2, -1.0], np.float32)
    L, tok, dl = oracle.topk_ce(xq, xp, 1.0, 10)
    full = torch.nn.functional.cross_entropy(torch.tensor(xq.astype(np.float64))[None],
                                             torch.softmax(torch.tensor(xp.astype(np.float64)), 0)[None])
    assert abs(L - float(full)) < 1e-12


def test_kl_term_enters_loss_and_gradient(oracle):
    """kl_weight lam adds lam/K sum_rows L_topk to each prefix's loss and
    lam/(B K) dL/dx to the gradient rows (R11), here with torch computing
    the added terms; the rest of the result is unchanged."""
    from paper_2602_05774_gb300 import inputs
    B, K, D, V, T, lam = 2, 3, 2, 64, 0.9, 0.37
    p = inputs.linear_problem(B, K, D, V, "f32", "gauss", seed=21)
    f = {k: p[k].numpy() for k in ("draft", "target", "u_draft", "u_accept", "u_correct")}
    args = (f["draft"], f["target"], T, f["u_draft"], f["u_accept"], f["u_correct"], K, D)
    o0 = oracle.linear(*args)
    o1 = oracle.linear(*args, kl_weight=lam)
    for n in ("tokens", "corr_tokens", "weights", "logkappa"):
        assert np.array_equal(o0[n], o1[n])
    dg = np.zeros_like(o0["grad"])
    add = np.zeros(B)
    for r in range(B * K * D):
        Lt, _, gt = _torch_topk_ce(f["draft"][r], f["target"][r], T)
        add[r // (K * D)] += lam / K * Lt
        dg[r] = lam / (B * K) * gt
        assert abs(o1["kl_loss"][r] - Lt) < 1e-12 * max(1.0, Lt)
    assert np.allclose(o1["loss"][:B], o0["loss"][:B] + add, rtol=1e-12, atol=1e-12)
    assert abs(o1["loss"][B] - o1["loss"][:B].mean()) < 1e-12
    assert np.allclose(o1["grad"], o0["grad"] + dg, rtol=1e-10, atol=1e-15)


# --------------------------------------------------------------------------
# Greedy decoding, T = 0 (reading R12), and a supplied greedy reference path
# (reading R13).


def _separated_problem(B, K, D, V, seed):
    """Rows whose logits are distinct integers (a permutation of 0..V-1 per
    row), so that at T = 0.01 every non-maximal token has probability below
    e^-100 and the T -> 0 limit is reached in double precision."""
    rng = np.random.default_rng(seed)
    R = B * K * D
    draft = np.stack([rng.permutation(V) for _ in range(R)]).astype(np.float32)
    target = np.stack([rng.permutation(V) for _ in range(R)]).astype(np.float32)
    # make about half the rows agree on the argmax
    agree = rng.random(R) < 0.5
    for r in np.nonzero(agree)[0]:
        i, j = int(np.argmax(draft[r])), int(np.argmax(target[r]))
        target[r, [i, j]] = target[r, [j, i]]
    u = [rng.uniform(0.01, 0.99, R).astype(np.float32) for _ in range(3)]
    return draft, target, u


def test_greedy_is_the_small_temperature_limit(oracle):
    B, K, D, V = 3, 4, 4, 40
    draft, target, (ud, ua, uc) = _separated_problem(B, K, D, V, 31)
    g = oracle.linear(draft, target, 0.0, ud, ua, uc, K, D)
    s = oracle.linear(draft, target, 0.01, ud, ua, uc, K, D)
    for n in ("tokens", "accept", "accept_len", "corr_tokens", "ref_tokens"):
        assert np.array_equal(g[n], s[n]), n
    assert np.array_equal(g["weights"][..., :2], s["weights"][..., :2])


def test_greedy_decisions_closed_form(oracle):
    B, K, D, V = 2, 3, 5, 30
    draft, target, (ud, ua, uc) = _separated_problem(B, K, D, V, 32)
    o = oracle.linear(draft, target, 0.0, ud, ua, uc, K, D)
    am_q = np.argmax(draft, axis=1)   # numpy keeps the first maximum
    am_p = np.argmax(target, axis=1)
    assert np.array_equal(o["tokens"], am_q)
    assert np.array_equal(o["accept"], (am_q == am_p).astype(np.uint8))
    acc = (am_q == am_p).reshape(B * K, D)
    A = np.where(acc.all(1), D, np.argmin(acc, axis=1))
    assert np.array_equal(o["accept_len"], A)
    d = np.arange(D)[None, :]
    corr = np.where(d < A[:, None], am_q.reshape(B * K, D), am_p.reshape(B * K, D))
    assert np.array_equal(o["corr_tokens"].reshape(B * K, D), corr)
    assert np.all(o["logkappa_corr"] == 0.0) and np.all(o["logkappa_ref"] == 0.0)
    w = o["weights"]  # [B][D][K][4]
    Al = A.reshape(B, K)
    for l in range(1, D + 1):
        assert np.array_equal(w[:, l - 1, :, 0], (l <= Al).astype(float))
        assert np.allclose(w[:, l - 1, :, 1], 1.05 ** l)


def test_greedy_ties_take_the_lowest_index(oracle):
    # two equal draft maxima (tokens 1 and 2) and two equal target maxima
    # (tokens 2 and 3): z~ = 1, argmax p = 2, so the token is rejected and the
    # corrected token is 2
    xq = np.array([[0.0, 3.0, 3.0, -1.0]], np.float32)
    xp = np.array([[0.0, 1.0, 2.0, 2.0]], np.float32)
    o = oracle.linear(xq, xp, 0.0, [0.5], [0.5], [0.5], K=1, D=1)
    assert o["tokens"][0] == 1 and o["accept"][0] == 0 and o["corr_tokens"][0] == 2
    assert o["ref_tokens"][0] == 2
    # supplied reference: target maxima at 0 and 1; the draft is confident on
    # 0 (ratio below 1) and not on 1 (ratio above 1), so the tie decides
    rq = np.array([[3.0, 0.0, 0.0, 0.0]], np.float32)
    rp = np.array([[2.0, 2.0, 1.0, 0.0]], np.float32)
    ref = oracle.reference_logkappa(rq, rp, 1.0, 1, 1)
    lq, lp = oracle.log_softmax(rq[0], 1.0), oracle.log_softmax(rp[0], 1.0)
    assert lp[0] - lq[0] < 0 and lp[1] - lq[1] > 0
    assert abs(ref[0, 0] - (lp[0] - lq[0])) < 1e-12


@pytest.mark.parametrize("accept", [True, False])
def test_greedy_single_proposal_is_cross_entropy_at_temperature_one(oracle, accept):
    import torch
    V = 12
    rng = np.random.default_rng(33)
    xq = rng.permutation(V).astype(np.float32) * 0.5
    xp = rng.permutation(V).astype(np.float32)
    i, j = int(np.argmax(xq)), int(np.argmax(xp))
    if accept:
        xp[[i, j]] = xp[[j, i]]
    o = oracle.linear(xq[None], xp[None], 0.0, [0.5], [0.5], [0.5], K=1, D=1)
    z = i if accept else int(np.argmax(xp))
    assert o["corr_tokens"][0] == z and o["accept"][0] == int(accept)
    x = torch.tensor(xq.astype(np.float64), requires_grad=True)
    ce = torch.nn.functional.cross_entropy(x[None], torch.tensor([z]))
    ce.backward()
    assert abs(o["loss"][0] - float(ce.detach())) < 1e-12
    assert np.allclose(o["grad"][0], x.grad.numpy(), atol=1e-15)


@pytest.mark.parametrize("T", [1.0, 0.7, 0.0])
def test_reference_rows_equal_the_per_path_reference(oracle, T):
    """With the reference rows equal to a path's own rows, log k(z-bar) of the
    supplied rows is the per-path reference (R4) the oracle forms."""
    from paper_2602_05774_gb300 import inputs
    B, D, V = 3, 4, 64
    p = inputs.linear_problem(B, 1, D, V, "f32", "gauss", seed=34)
    f = {k: p[k].numpy() for k in ("draft", "target", "u_draft", "u_accept", "u_correct")}
    o = oracle.linear(f["draft"], f["target"], T, f["u_draft"], f["u_accept"], f["u_correct"],
                      1, D, want_grad=False)
    ref = oracle.reference_logkappa(f["draft"], f["target"], T, B, D)
    assert np.array_equal(ref.reshape(-1), o["logkappa_ref"])
    if T == 0.0:
        assert np.all(ref == 0.0)


def test_reference_rows_worked_example(oracle):
    q1, p1 = [1 / 2, 1 / 4, 1 / 8, 1 / 8], [1 / 8, 1 / 2, 1 / 4, 1 / 8]      # v = 1, ratio 2
    q2, p2 = [1 / 8, 1 / 2, 1 / 4, 1 / 8], [1 / 4, 3 / 8, 1 / 4, 1 / 8]      # v = 1, ratio 3/4
    draft = np.stack([logits(q1), logits(q2)])
    target = np.stack([logits(p1), logits(p2)])
    ref = oracle.reference_logkappa(draft, target, 1.0, 1, 2)
    assert abs(ref[0, 0]) < 1e-7 and abs(ref[0, 1] - math.log(0.75)) < 1e-7


# --------------------------------------------------------------------------
# Trees: the sequential sibling rule (reading R14) and the tree EM (R15).


def _chain_tree(B, N, V, seed, same=False):
    rng = np.random.default_rng(seed)
    draft = rng.normal(0, 2, (B * N, V)).astype(np.float32)
    target = draft.copy() if same else (draft + rng.normal(0, 1, (B * N, V))).astype(np.float32)
    parent = np.tile(np.arange(-1, N - 1, dtype=np.int32), (B, 1))
    tokens = rng.integers(0, V, (B, N)).astype(np.int32)
    ua = rng.random((B, N)).astype(np.float32)
    uc = rng.random((B, N)).astype(np.float32)
    return draft, target, parent, tokens, ua, uc


def test_sequential_rule_on_chains_is_the_independent_rule(oracle):
    """With one child per node there is nothing to try in turn: the accepted
    path, the correction and the bonus are the independent rule's."""
    args = _chain_tree(6, 7, 40, 51)
    a = oracle.tree(*args[:2], 1.0, *args[2:], rule=0)
    s = oracle.tree(*args[:2], 1.0, *args[2:], rule=1)
    for n in ("path_accept", "deepest", "accept_len", "bonus", "corr_tokens", "logkappa"):
        assert np.array_equal(a[n], s[n]), n
    tried = np.zeros_like(a["accept"], bool)
    tried[:, 1:] = a["path_accept"][:, :-1] == 1  # a child is tried when its parent is accepted
    assert np.array_equal(a["accept"][tried], s["accept"][tried])
    assert np.array_equal(a["alpha"][tried], s["alpha"][tried])
    untried = ~tried[:, 1:]  # (the root is node 0)
    assert np.all(s["accept"][:, 1:][untried] == 0) and np.all(s["alpha"][:, 1:][untried] == 0)


def test_sequential_rule_is_lossless(oracle):
    """A root with three children drawn without replacement from q: the token
    the step emits (the accepted child's, or the correction when all are
    rejected) is distributed as p.  Monte Carlo over 2^18 seeded trees: every
    frequency within 5 standard errors of p, while the independent rule's
    first-accepted-or-residual output is visibly off."""
    V, m, n = 5, 3, 1 << 18
    rng = np.random.default_rng(52)
    xq = np.array([1.2, 0.3, -0.5, 0.9, -1.0], np.float32)
    xp = np.array([-0.4, 1.1, 0.6, -0.2, 0.2], np.float32)
    q = np.exp(oracle.log_softmax(xq))
    p = np.exp(oracle.log_softmax(xp))
    # children tokens: sequential draws from q without replacement
    g = -np.log(-np.log(rng.random((n, V))))
    toks = np.argsort(-(np.log(q)[None, :] + g), axis=1)[:, :m].astype(np.int32)
    N = m + 1
    draft = np.tile(xq, (n * N, 1))
    target = np.tile(xp, (n * N, 1))
    parent = np.tile(np.array([-1] + [0] * m, np.int32), (n, 1))
    tokens = np.concatenate([np.zeros((n, 1), np.int32), toks], axis=1)
    ua = rng.random((n, N)).astype(np.float32)
    uc = rng.random((n, N)).astype(np.float32)
    o = oracle.tree(draft, target, 1.0, parent, tokens, ua, uc, rule=1)
    out = np.where(o["deepest"] > 0, tokens[np.arange(n), o["deepest"]], o["bonus"])
    freq = np.bincount(out, minlength=V) / n
    se = np.sqrt(p * (1 - p) / n)
    assert np.all(np.abs(freq - p) < 5 * se), (freq, p)
    # (the Gumbel-top-k draws above are exactly sequential draws without replacement)
    assert abs(np.mean(toks[:, 0] == 0) - q[0]) < 5 * np.sqrt(q[0] * (1 - q[0]) / n)


def test_sequential_first_child_accepted_when_draft_is_target(oracle):
    B, N, V = 4, 6, 30
    rng = np.random.default_rng(53)
    x = rng.normal(0, 2, (B * N, V)).astype(np.float32)
    parent = np.tile(np.array([-1, 0, 0, 0, 1, 1], np.int32), (B, 1))
    tokens = rng.integers(0, V, (B, N)).astype(np.int32)
    o = oracle.tree(x, x, 1.0, parent, tokens, rng.random((B, N)).astype(np.float32),
                    rng.random((B, N)).astype(np.float32), rule=1)
    assert np.all(o["path_accept"][:, [1, 4]] == 1) and np.all(o["path_accept"][:, [2, 3, 5]] == 0)
    assert np.all(o["deepest"] == 4) and np.all(o["accept_len"] == 2)


def test_tree_em_of_shared_root_chains_is_the_linear_em(oracle):
    """K chains of depth D below one root, the root's row shared: the tree's
    proposals at depth l are the K linear paths' length-l proposals, so the
    tree EM equals the linear EM of K paths whose first rows coincide (the
    root row's gradient is the sum of the K first rows')."""
    from paper_2602_05774_gb300 import inputs
    K, D, V, T = 4, 3, 50, 0.8
    pr = inputs.linear_problem(1, K, D, V, "f32", "gauss", seed=56)
    f = {k: pr[k].numpy().copy() for k in ("draft", "target", "u_draft", "u_accept", "u_correct")}
    for s in range(1, K):  # the first rows of every path coincide
        f["draft"][s * D] = f["draft"][0]
        f["target"][s * D] = f["target"][0]
    lin = oracle.linear(f["draft"], f["target"], T, f["u_draft"], f["u_accept"], f["u_correct"],
                        K, D, w_base=1.1, tau_car=0.3)
    # the case exercises both o~ values and positions below a rejection
    assert set(np.unique(lin["weights"][..., 0])) == {0.0, 1.0}
    assert np.any(lin["accept_len"] < D - 1)
    N = 1 + K * D
    node = lambda s, j: 1 + (j - 1) * K + s  # node of path s at depth j >= 1
    parent = np.full(N, -1, np.int32)
    tokens = np.zeros(N, np.int32)
    ua = np.zeros(N, np.float32)
    uc = np.zeros(N, np.float32)
    draft = np.zeros((N, V), np.float32)
    target = np.zeros((N, V), np.float32)
    draft[0], target[0] = f["draft"][0], f["target"][0]
    for s in range(K):
        for j in range(1, D + 1):
            x = node(s, j)
            parent[x] = 0 if j == 1 else node(s, j - 1)
            r = s * D + j - 1
            tokens[x], ua[x], uc[x] = lin["tokens"][r], f["u_accept"][r], f["u_correct"][r]
            rr = s * D + min(j, D - 1)  # the row of node x: linear row (s, j); leaves any row
            draft[x], target[x] = f["draft"][rr], f["target"][rr]
    t = oracle.tree_em(draft, target, T, parent[None], tokens[None], ua[None], uc[None],
                       w_base=1.1, tau_car=0.3)
    for s in range(K):
        for j in range(1, D + 1):
            x, r = node(s, j), s * D + j - 1
            assert t["corr_tokens"][0, x] == lin["corr_tokens"][r]
            for n in ("logkappa", "logkappa_corr", "logkappa_ref", "logq_corr"):
                assert abs(t[n][0, x] - lin[n][r]) < 1e-12, n
            assert np.allclose(t["weights"][0, x], lin["weights"][0, j - 1, s], rtol=1e-12,
                               atol=1e-15)
    assert abs(t["loss"][0] - lin["loss"][0]) < 1e-12
    g = t["grad"]
    assert np.allclose(g[0], sum(lin["grad"][s * D] for s in range(K)), atol=1e-14)
    for s in range(K):
        for j in range(1, D):
            assert np.allclose(g[node(s, j)], lin["grad"][s * D + j], atol=1e-14)
        assert np.all(g[node(s, D)] == 0.0)  # a leaf's row carries no term


# --------------------------------------------------------------------------
# The LM head's backward: d hidden = G W, d weight = G^T H.


def test_lmhead_backward_one_hot_and_chain_rule(oracle):
    import torch
    rng = np.random.default_rng(61)
    R, V, H = 5, 7, 3
    h = rng.normal(size=(R, H))
    w = rng.normal(size=(V, H))
    # one-hot gradients pick rows and columns: G = e_(r,v) gives d hidden row r
    # = weight row v and d weight row v = hidden row r
    for r, v in ((0, 0), (3, 6), (4, 2)):
        G = np.zeros((R, V))
        G[r, v] = 1.0
        dh, dw = oracle.lmhead_backward(G, h, w)
        assert np.array_equal(dh[r], w[v]) and np.count_nonzero(dh.sum(1)) <= 1
        assert np.array_equal(dw[v], h[r]) and np.count_nonzero(dw.sum(1)) <= 1
    # the chain rule through torch's autograd of the forward
    G = rng.normal(size=(R, V))
    ht = torch.tensor(h, requires_grad=True)
    wt = torch.tensor(w, requires_grad=True)
    (ht @ wt.T).backward(torch.tensor(G))
    dh, dw = oracle.lmhead_backward(G, h, w)
    assert np.allclose(dh, ht.grad.numpy(), rtol=1e-13, atol=1e-13)
    assert np.allclose(dw, wt.grad.numpy(), rtol=1e-13, atol=1e-13)
