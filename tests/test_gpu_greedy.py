"""GPU parity of greedy decoding (T = 0, reading R12) through the fused
E-step + M-step and the LM head with it, and of the greedy reference from
supplied rows (vsd_reference_logkappa, reading R13), against the oracle."""
import numpy as np
import pytest
import torch

from tests.parity import compare_linear, mstep_inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def vsd():
    from paper_2602_05774_gb300 import build, vsd as v
    build.build_library()
    v.load()
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    return v


def _np32(t):
    return t.detach().float().cpu().numpy()


def _fused_vs_oracle(vsd, oracle, prob, grad_dtype, ref=None, lam=0.0):
    B, K, D, V = prob["B"], prob["K"], prob["D"], prob["V"]
    orc = oracle.linear(_np32(prob["draft"]), _np32(prob["target"]), 0.0, _np32(prob["u_draft"]),
                        _np32(prob["u_accept"]), _np32(prob["u_correct"]), K, D,
                        ref_logkappa=None if ref is None else _np32(ref), kl_weight=lam)
    p = {k: (v.cuda() if torch.is_tensor(v) else v) for k, v in prob.items()}
    prm = vsd.params(like=p["draft"], grad_dtype=torch.float32 if grad_dtype == "f32"
                     else torch.bfloat16, kl_weight=lam)
    ws = vsd.new_workspace(vsd.layout(B, K, D, V), "cuda")
    g = vsd.estep_mstep(p["draft"], p["target"], p["u_draft"], p["u_accept"], p["u_correct"], K,
                        D, 0.0, prm=prm, workspace=ws,
                        ref_logkappa=None if ref is None else ref.cuda())
    torch.cuda.synchronize()
    assert vsd.device_status(ws) == (0, 0)
    compare_linear(g, orc, B, K, D, V, 1.0, grad_dtype=grad_dtype, kl=lam > 0,
                   mstep_inputs=mstep_inputs(prob, kl_weight=lam))
    # the decisions of the greedy limit
    tok = g["tokens"].cpu().numpy()
    assert np.array_equal(tok, np.argmax(_np32(prob["draft"]), axis=1))
    assert np.isin(g["alpha"].cpu().numpy(), [0.0, 1.0]).all()
    assert torch.all(g["logkappa_corr"] == 0)
    return g, orc


CASES = [
    (2, 4, 4, 1024, "f32", "gauss"),
    (3, 4, 3, 32000, "bf16", "spiked"),   # short rows: the streaming warps' tails
    (1, 3, 2, 140000, "bf16", "zipf"),    # long rows in two segments: the control warp
    (2, 2, 2, 70001, "f32", "gauss"),     # scalar path
    (2, 3, 2, 33, "f32", "gauss"),
]


@pytest.mark.parametrize("B,K,D,V,dtype,kind", CASES)
def test_greedy_fused_matches_oracle(vsd, oracle, B, K, D, V, dtype, kind):
    from paper_2602_05774_gb300 import inputs
    prob = inputs.linear_problem(B, K, D, V, dtype, kind, seed=500 + V)
    # target = draft on a third of the rows, so that tokens are accepted too
    R = B * K * D
    same = torch.arange(R) % 3 == 0
    prob["target"][same] = prob["draft"][same]
    _fused_vs_oracle(vsd, oracle, prob, dtype)


def test_greedy_ties_and_kl(vsd, oracle):
    """bf16 rows with repeated maxima (the lowest index wins), with the top-K term."""
    B, K, D, V = 2, 3, 3, 4096
    R = B * K * D
    g = torch.Generator().manual_seed(9)
    draft = torch.randn(R, V, generator=g)
    target = draft + 0.3 * torch.randn(R, V, generator=g)
    for r in range(R):
        idx = torch.randperm(V, generator=g)[:3]
        draft[r, idx] = 6.0
        target[r, idx if r % 2 else idx[:1]] = 6.0
    prob = dict(B=B, K=K, D=D, V=V, draft=draft.to(torch.bfloat16),
                target=target.to(torch.bfloat16), u_draft=torch.rand(R, generator=g),
                u_accept=torch.rand(R, generator=g), u_correct=torch.rand(R, generator=g))
    _fused_vs_oracle(vsd, oracle, prob, "bf16", lam=0.5)


@pytest.mark.parametrize("dtype,T", [("f32", 1.0), ("bf16", 0.7), ("bf16", 0.0)])
def test_reference_logkappa_matches_oracle(vsd, oracle, dtype, T):
    from paper_2602_05774_gb300 import inputs
    B, D, V = 5, 6, 3000
    prob = inputs.linear_problem(B, 1, D, V, dtype, "spiked", seed=77)
    ref = vsd.reference_logkappa(prob["draft"].cuda(), prob["target"].cuda(), B, D, T)
    torch.cuda.synchronize()
    want = oracle.reference_logkappa(_np32(prob["draft"]), _np32(prob["target"]), T, B, D)
    got = ref.cpu().numpy().astype(np.float64)
    fin = np.isfinite(want)
    assert np.array_equal(np.isfinite(got), fin)
    assert np.allclose(got[fin], want[fin], atol=1e-5, rtol=1e-6)
    if T == 0.0:
        assert np.all(got == 0.0)


def test_reference_rows_feed_the_fused_step(vsd, oracle):
    """The reference computed from supplied rows, passed to the fused step,
    gives the oracle's result with the oracle's own reference as input."""
    from paper_2602_05774_gb300 import inputs
    B, K, D, V, T = 3, 4, 3, 3000, 1.0
    prob = inputs.linear_problem(B, K, D, V, "bf16", "spiked", seed=78)
    rows = inputs.linear_problem(B, 1, D, V, "bf16", "spiked", seed=79)
    ref = vsd.reference_logkappa(rows["draft"].cuda(), rows["target"].cuda(), B, D, T)
    want = oracle.reference_logkappa(_np32(rows["draft"]), _np32(rows["target"]), T, B, D)
    orc = oracle.linear(_np32(prob["draft"]), _np32(prob["target"]), T, _np32(prob["u_draft"]),
                        _np32(prob["u_accept"]), _np32(prob["u_correct"]), K, D,
                        ref_logkappa=want.astype(np.float32))
    p = {k: (v.cuda() if torch.is_tensor(v) else v) for k, v in prob.items()}
    g = vsd.estep_mstep(p["draft"], p["target"], p["u_draft"], p["u_accept"], p["u_correct"], K,
                        D, T, ref_logkappa=ref)
    torch.cuda.synchronize()
    compare_linear(g, orc, B, K, D, V, T, grad_dtype="bf16", mstep_inputs=mstep_inputs(prob))


def test_greedy_lmhead_matches_oracle(vsd, oracle):
    from paper_2602_05774_gb300 import inputs
    B, K, D, V, H = 3, 4, 4, 4104, 264
    p = inputs.lmhead_exact_problem(B, K, D, V, H, device="cuda", seed=88)
    ws = vsd.new_workspace(vsd.layout(B, K, D, V), "cuda")
    g = vsd.lmhead_estep_mstep(p["hidden"], p["weight"], p["target"], p["u_draft"],
                               p["u_accept"], p["u_correct"], K, D, 0.0, workspace=ws)
    assert vsd.device_status(ws) == (0, 0)
    H64 = p["hidden"].float().cpu().numpy().astype(np.float64)
    W64 = p["weight"].float().cpu().numpy().astype(np.float64)
    draft = oracle.round_bf16(oracle.lmhead_logits(H64, W64))
    assert np.array_equal(g["draft_logits"].float().cpu().numpy(), draft)
    orc = oracle.linear(draft, p["target"].float().cpu().numpy(), 0.0,
                        p["u_draft"].cpu().numpy(), p["u_accept"].cpu().numpy(),
                        p["u_correct"].cpu().numpy(), K, D)
    compare_linear(g, orc, B, K, D, V, 1.0, grad_dtype="bf16",
                   mstep_inputs=mstep_inputs(dict(B=B, K=K, D=D, draft=draft)))
