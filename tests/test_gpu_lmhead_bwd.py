"""GPU parity of the draft LM head's backward (vsd_lmhead_backward):
d_hidden = G . W and d_weight = G^T . hidden, with G the M-step gradient of
the draft logits made on chip from the E-step's records.

Three kinds of check:
  * exact: with W a (V x H, V <= H) identity, d_hidden[:, :V] is G itself
    (every fp32 sum has one nonzero product), so it must equal, bit for bit,
    the bf16 gradient the fused E-step + M-step wrote; with hidden an (R x H,
    R <= H) identity, d_weight[:, :R] = G^T likewise.  This pins every element
    of the on-chip gradient, sparse terms and tails included.
  * bound: on Gaussian inputs, each output lies within the fp32 summation
    bound K 2^-24 sum_k |a_k b_k| of the float64 product of the written bf16
    gradient with W (or hidden).
  * oracle: against oracle.lmhead_backward applied to the oracle's float64
    gradient, within the propagated per-element gradient tolerance (2^-8
    relative for the bf16 rounding plus 1e-6 of the gradient's scale) plus the
    summation bound, for prefixes whose decisions agree with the oracle's.
"""
import numpy as np
import pytest
import torch

from tests.parity import _first_divergence, compare_linear, mstep_inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def vsd():
    from paper_2602_05774_gb300 import build, vsd as v
    build.build_library()
    v.load()
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    return v


def _np(t):
    return t.detach().float().cpu().numpy().astype(np.float64)


def _problem(B, K, D, V, H, kind, seed):
    """kind "dh_exact": W = identity (V <= H), hidden Gaussian, so the draft
    logits are hidden[:, :V]; "dw_exact": hidden = identity (R <= H), W
    Gaussian, so draft logits[r][v] = W[v][r]; "gauss": both Gaussian."""
    from paper_2602_05774_gb300 import inputs
    R = B * K * D
    g = torch.Generator(device="cuda").manual_seed(seed)
    if kind == "dh_exact":
        assert V <= H
        w = torch.eye(V, H, device="cuda")
        h = torch.randn(R, H, generator=g, device="cuda") * 2.0
    elif kind == "dw_exact":
        assert R <= H
        h = torch.eye(R, H, device="cuda")
        w = torch.randn(V, H, generator=g, device="cuda") * 2.0
    else:
        h = torch.randn(R, H, generator=g, device="cuda")
        w = torch.randn(V, H, generator=g, device="cuda") * (2.0 / H ** 0.5)
    t = inputs.logits_spiked(R, V, 3.0, min(50, V), 8.0, "cuda", seed + 1) + \
        inputs.logits_gaussian(R, V, 1.0, "cuda", seed + 2)
    return dict(hidden=h.to(torch.bfloat16).contiguous(), weight=w.to(torch.bfloat16).contiguous(),
                target=t.to(torch.bfloat16).contiguous(),
                u_draft=inputs.uniforms(R, "cuda", seed + 3),
                u_accept=inputs.uniforms(R, "cuda", seed + 4),
                u_correct=inputs.uniforms(R, "cuda", seed + 5))


def _run(vsd, p, K, D, T, kl_weight=0.0):
    B = p["hidden"].shape[0] // (K * D)
    V = p["weight"].shape[0]
    lay = vsd.layout(B, K, D, V)
    ws = vsd.new_workspace(lay, "cuda")
    prm = vsd.params(like=p["target"], kl_weight=kl_weight)
    fw = vsd.lmhead_estep_mstep(p["hidden"], p["weight"], p["target"], p["u_draft"],
                                p["u_accept"], p["u_correct"], K, D, T, prm=prm, workspace=ws)
    bw = vsd.lmhead_backward(p["hidden"], p["weight"], fw["draft_logits"], K, D, T, ws, prm=prm)
    torch.cuda.synchronize()
    assert vsd.device_status(ws) == (0, 0)
    assert fw["grad"].dtype == torch.bfloat16
    return fw, bw


def _check_bound(G, A, got, name):
    """got = G . A within the fp32 summation bound (G, A float64, exact)."""
    want = G @ A
    bound = G.shape[1] * 2.0 ** -24 * (np.abs(G) @ np.abs(A)) + 1e-30
    err = np.abs(got - want)
    assert np.isfinite(got).all(), name
    assert (err <= bound).all(), "%s off by %g (bound %g)" % (
        name, err.max(), bound.flat[np.argmax(err - bound)])


# ragged R, V and H (tails of every tile and K block), several M and N tiles
SHAPES = [(2, 4, 4, 520, 520), (3, 5, 4, 1032, 1032), (2, 8, 8, 4104, 4104)]


@pytest.mark.parametrize("B,K,D,V,H", SHAPES)
@pytest.mark.parametrize("T", [1.0, 0.7])
def test_d_hidden_is_the_gradient_exactly(vsd, B, K, D, V, H, T):
    p = _problem(B, K, D, V, H, "dh_exact", 300 + V)
    fw, bw = _run(vsd, p, K, D, T)
    G = fw["grad"].float()
    dh = bw["d_hidden"]
    assert torch.equal(dh[:, :V], G), \
        "d_hidden differs from the written gradient at %s" % (
            torch.nonzero(dh[:, :V] != G)[:4].tolist())
    assert not dh[:, V:].any()
    _check_bound(_np(G).T, _np(p["hidden"]), _np(bw["d_weight"]), "d_weight")


@pytest.mark.parametrize("B,K,D,V,H", [(2, 4, 4, 520, 136), (3, 5, 4, 4104, 264),
                                       (4, 8, 8, 1032, 1032)])
@pytest.mark.parametrize("T", [1.0, 0.7])
def test_d_weight_is_the_gradient_exactly(vsd, B, K, D, V, H, T):
    R = B * K * D
    p = _problem(B, K, D, V, H, "dw_exact", 500 + V + R)
    fw, bw = _run(vsd, p, K, D, T)
    G = fw["grad"].float()
    dw = bw["d_weight"]
    assert torch.equal(dw[:, :R], G.T), \
        "d_weight differs from the written gradient at %s" % (
            torch.nonzero(dw[:, :R] != G.T)[:4].tolist())
    assert not dw[:, R:].any()
    _check_bound(_np(G), _np(p["weight"]), _np(bw["d_hidden"]), "d_hidden")


@pytest.mark.parametrize("kind", ["dh_exact", "dw_exact"])
def test_kl_terms_exactly(vsd, kind):
    """VSD (KL): the top-K terms enter the on-chip gradient as they enter the
    written one."""
    B, K, D, V, H = 2, 4, 4, 1032, 1032
    R = B * K * D
    p = _problem(B, K, D, V, H, kind, 77)
    fw, bw = _run(vsd, p, K, D, 1.0, kl_weight=0.5)
    G = fw["grad"].float()
    if kind == "dh_exact":
        assert torch.equal(bw["d_hidden"][:, :V], G)
    else:
        assert torch.equal(bw["d_weight"][:, :R], G.T)


@pytest.mark.parametrize("kind", ["dh_exact", "dw_exact"])
def test_greedy_exactly(vsd, kind):
    """T = 0: the gradient at temperature 1 along the argmax decisions."""
    B, K, D, V, H = 2, 4, 4, 520, 520
    R = B * K * D
    p = _problem(B, K, D, V, H, kind, 91)
    fw, bw = _run(vsd, p, K, D, 0.0)
    G = fw["grad"].float()
    if kind == "dh_exact":
        assert torch.equal(bw["d_hidden"][:, :V], G)
    else:
        assert torch.equal(bw["d_weight"][:, :R], G.T)


@pytest.mark.parametrize("B,K,D,V,H,T", [(3, 5, 4, 4104, 264, 1.0), (2, 8, 8, 8200, 1032, 0.7)])
def test_gaussian_within_bound(vsd, B, K, D, V, H, T):
    p = _problem(B, K, D, V, H, "gauss", 40 + V)
    fw, bw = _run(vsd, p, K, D, T)
    G = _np(fw["grad"])
    _check_bound(G, _np(p["weight"]), _np(bw["d_hidden"]), "d_hidden")
    _check_bound(G.T, _np(p["hidden"]), _np(bw["d_weight"]), "d_weight")


def _oracle_chain(oracle, fw, bw, p, B, K, D, V, T, prefixes, B_total):
    """d_hidden rows of the given prefixes (and, with every prefix given,
    d_weight) against oracle.lmhead_backward of the oracle's gradient, run
    on the oracle's own logits; prefixes whose decisions disagree with the
    oracle's are left out (at least one must remain)."""
    from tests.parity import sub_batch
    Hn, Wn = _np(p["hidden"]), _np(p["weight"])
    P = K * D
    checked = 0
    Go_all, agree_all = [], True
    for b in prefixes:
        rows = slice(b * P, (b + 1) * P)
        draft = oracle.round_bf16(oracle.lmhead_logits(Hn[rows], Wn))
        assert np.array_equal(_np(fw["draft_logits"][rows]), draft), b
        orc = oracle.linear(draft, p["target"][rows].float().cpu().numpy(), T,
                            p["u_draft"][rows].cpu().numpy(), p["u_accept"][rows].cpu().numpy(),
                            p["u_correct"][rows].cpu().numpy(), K, D)
        orc["grad"] = np.asarray(orc["grad"], np.float64).reshape(P, V) / B_total
        sub = sub_batch(fw, b, b + 1, B_total, K, D)
        compare_linear(sub, orc, 1, K, D, V, T, grad_dtype="bf16", check_mean=False,
                       mstep_inputs=mstep_inputs(dict(B=1, K=K, D=D, draft=draft),
                                                 B_total=B_total))
        f, _ = _first_divergence(sub, orc, 1, K, D)
        Go = orc["grad"]
        Go_all.append(Go)
        if not (f == D).all():
            agree_all = False
            continue
        G = _np(fw["grad"][rows])
        dh_o, _ = oracle.lmhead_backward(Go, None, Wn)
        tol_g = 2.0 ** -8 * np.abs(Go) + 1e-6 * np.abs(Go).max()
        lim = tol_g @ np.abs(Wn) + V * 2.0 ** -24 * (np.abs(G) @ np.abs(Wn)) + 1e-30
        err = np.abs(_np(bw["d_hidden"][rows]) - dh_o)
        assert (err <= lim).all(), "prefix %d: d_hidden vs oracle off by %g" % (b, err.max())
        checked += 1
    assert checked >= 1
    if agree_all and len(prefixes) == B_total:
        Go = np.concatenate(Go_all)
        G = _np(fw["grad"])
        _, dw_o = oracle.lmhead_backward(Go, Hn, None)
        tol_g = 2.0 ** -8 * np.abs(Go) + 1e-6 * np.abs(Go).max()
        lim = tol_g.T @ np.abs(Hn) + G.shape[0] * 2.0 ** -24 * (np.abs(G).T @ np.abs(Hn)) + 1e-30
        err = np.abs(_np(bw["d_weight"]) - dw_o)
        assert (err <= lim).all(), "d_weight vs oracle off by %g" % err.max()
    return checked


@pytest.mark.parametrize("B,K,D,V,H,T", [(3, 5, 4, 4104, 264, 1.0), (2, 8, 8, 8200, 1032, 0.7)])
def test_against_oracle(vsd, oracle, B, K, D, V, H, T):
    """Inputs whose float32 partial sums are exact, so the oracle's logits are
    the GPU's bit for bit and the oracle runs on its own logits."""
    from paper_2602_05774_gb300 import inputs
    p = inputs.lmhead_exact_problem(B, K, D, V, H, device="cuda", seed=610 + V)
    fw, bw = _run(vsd, p, K, D, T)
    _oracle_chain(oracle, fw, bw, p, B, K, D, V, T, range(B), B)


def test_skip_one_output(vsd):
    B, K, D, V, H = 2, 4, 4, 520, 264
    p = _problem(B, K, D, V, H, "gauss", 5)
    lay = vsd.layout(B, K, D, V)
    ws = vsd.new_workspace(lay, "cuda")
    fw = vsd.lmhead_estep_mstep(p["hidden"], p["weight"], p["target"], p["u_draft"],
                                p["u_accept"], p["u_correct"], K, D, 1.0, workspace=ws)
    both = vsd.lmhead_backward(p["hidden"], p["weight"], fw["draft_logits"], K, D, 1.0, ws)
    only_h = vsd.lmhead_backward(p["hidden"], p["weight"], fw["draft_logits"], K, D, 1.0, ws,
                                 d_weight=False)
    only_w = vsd.lmhead_backward(p["hidden"], p["weight"], fw["draft_logits"], K, D, 1.0, ws,
                                 d_hidden=False)
    torch.cuda.synchronize()
    assert set(only_h) == {"d_hidden"} and set(only_w) == {"d_weight"}
    assert torch.equal(both["d_hidden"], only_h["d_hidden"])
    assert torch.equal(both["d_weight"], only_w["d_weight"])


def test_full_size_sampled(vsd, oracle):
    """The lmhead workload (R = 64*8*8 = 4096, H = 4096, V = 32000) as the
    benchmark launches it, on inputs whose float32 partial sums are exact:
    d_hidden rows of three prefixes (first, middle, last) against the oracle's
    chain; sampled d_weight rows against the float64 product of the written
    gradient with hidden within the summation bound; every output finite;
    deterministic across two calls."""
    from paper_2602_05774_gb300 import inputs
    c = inputs.CONFIGS["lmhead"]
    B, K, D, V, H = c["B"], c["K"], c["D"], c["V"], c["H"]
    p = inputs.lmhead_exact_problem(B, K, D, V, H, device="cuda", seed=4242)
    lay = vsd.layout(B, K, D, V)
    ws = vsd.new_workspace(lay, "cuda")
    fw = vsd.lmhead_estep_mstep(p["hidden"], p["weight"], p["target"], p["u_draft"],
                                p["u_accept"], p["u_correct"], K, D, 1.0, workspace=ws)
    bw = vsd.lmhead_backward(p["hidden"], p["weight"], fw["draft_logits"], K, D, 1.0, ws)
    bw2 = vsd.lmhead_backward(p["hidden"], p["weight"], fw["draft_logits"], K, D, 1.0, ws)
    torch.cuda.synchronize()
    assert vsd.device_status(ws) == (0, 0)
    assert torch.equal(bw["d_hidden"], bw2["d_hidden"])
    assert torch.equal(bw["d_weight"], bw2["d_weight"])
    del bw2
    assert torch.isfinite(bw["d_hidden"]).all() and torch.isfinite(bw["d_weight"]).all()
    _oracle_chain(oracle, fw, bw, p, B, K, D, V, 1.0, (0, B // 2, B - 1), B)
    cols = torch.tensor([0, 1, 255, 256, 17000, 31998, 31999], device="cuda")
    Gc = _np(fw["grad"][:, cols]).T  # [7][R]
    _check_bound(Gc, _np(p["hidden"]), _np(bw["d_weight"][cols]), "d_weight")


@pytest.mark.parametrize("kl_weight", [0.0, 0.5])
def test_factored_step_without_dense_gradient(vsd, kl_weight):
    """The training step that never writes the dense gradient: the fused call
    with no grad output, then the backward from what it left in the
    workspace.  Every output equals the one of the step that writes the
    gradient, bit for bit."""
    B, K, D, V, H = 3, 5, 4, 4104, 264
    p = _problem(B, K, D, V, H, "gauss", 808)
    prm = vsd.params(like=p["target"], kl_weight=kl_weight)
    res = []
    for grad in (True, False):
        ws = vsd.new_workspace(vsd.layout(B, K, D, V), "cuda")
        fw = vsd.lmhead_estep_mstep(p["hidden"], p["weight"], p["target"], p["u_draft"],
                                    p["u_accept"], p["u_correct"], K, D, 1.0, prm=prm,
                                    workspace=ws, grad=grad)
        bw = vsd.lmhead_backward(p["hidden"], p["weight"], fw["draft_logits"], K, D, 1.0, ws,
                                 prm=prm)
        torch.cuda.synchronize()
        assert vsd.device_status(ws) == (0, 0)
        assert ("grad" in fw) == grad
        res.append((fw, bw))
    (f1, b1), (f2, b2) = res
    for name in f2:
        assert torch.equal(f1[name], f2[name]), name
    assert torch.equal(b1["d_hidden"], b2["d_hidden"])
    assert torch.equal(b1["d_weight"], b2["d_weight"])


def test_d_hidden_exactly_with_stream_k(vsd):
    """160 output tiles of 128 x 512 on the GPU's SMs: d_hidden is shared out
    by stream-K (tiles split between two CTAs and added into the zeroed
    output).  With W the identity it is still the written gradient bit for
    bit, and two calls give the same bits."""
    B, K, D, V, H = 64, 8, 8, 2560, 2560
    p = _problem(B, K, D, V, H, "dh_exact", 4321)
    fw, bw = _run(vsd, p, K, D, 1.0)
    G = fw["grad"].float()
    assert torch.equal(bw["d_hidden"][:, :V], G)
    ws = vsd.new_workspace(vsd.layout(B, K, D, V), "cuda")
    fw2 = vsd.lmhead_estep_mstep(p["hidden"], p["weight"], p["target"], p["u_draft"],
                                 p["u_accept"], p["u_correct"], K, D, 1.0, workspace=ws)
    a = vsd.lmhead_backward(p["hidden"], p["weight"], fw2["draft_logits"], K, D, 1.0, ws,
                            d_weight=False)
    b = vsd.lmhead_backward(p["hidden"], p["weight"], fw2["draft_logits"], K, D, 1.0, ws,
                            d_weight=False)
    torch.cuda.synchronize()
    assert torch.equal(a["d_hidden"], b["d_hidden"])
    assert torch.equal(a["d_hidden"], bw["d_hidden"])
