"""GPU parity of VSD (KL): the fused E-step + M-step with the top-K
renormalised term of Eq. klv (params.kl_weight != 0), against the oracle's
own top-K term (reading R11), on the shapes that take each code path: short
rows whose tails the streaming warps run (the term on the fourth warp), long
rows whose tails the control warp runs, several work segments per row, the
scalar (unaligned) path, fewer tokens than K, and ties at the cut."""
import numpy as np
import pytest
import torch

from tests.parity import compare_linear, mstep_inputs, to_np

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


def _run(vsd, oracle, prob, T, lam, topk, grad_dtype):
    B, K, D, V = prob["B"], prob["K"], prob["D"], prob["V"]
    orc = oracle.linear(_np32(prob["draft"]), _np32(prob["target"]), T, _np32(prob["u_draft"]),
                        _np32(prob["u_accept"]), _np32(prob["u_correct"]), K, D,
                        kl_weight=lam, kl_topk=topk)
    p = {k: (v.cuda() if torch.is_tensor(v) else v) for k, v in prob.items()}
    prm = vsd.params(like=p["draft"], grad_dtype=torch.float32 if grad_dtype == "f32"
                     else torch.bfloat16, kl_weight=lam, kl_topk=topk)
    ws = vsd.new_workspace(vsd.layout(B, K, D, V), "cuda")
    g = vsd.estep_mstep(p["draft"], p["target"], p["u_draft"], p["u_accept"], p["u_correct"], K,
                        D, T, prm=prm, workspace=ws)
    torch.cuda.synchronize()
    assert vsd.device_status(ws) == (0, 0)
    rep = {}
    compare_linear(g, orc, B, K, D, V, T, grad_dtype=grad_dtype, report=rep, kl=True,
                   mstep_inputs=mstep_inputs(prob, kl_weight=lam, kl_topk=topk))
    return g, orc


CASES = [
    # B, K, D, V, dtype, kind, T, topk
    (2, 4, 4, 1024, "f32", "gauss", 1.0, 10),       # tiny
    (3, 4, 3, 32000, "bf16", "spiked", 1.0, 10),    # short rows: the streaming warps' tail
    (2, 3, 3, 5000, "bf16", "zipf", 0.7, 16),
    (1, 3, 2, 140000, "bf16", "zipf", 1.0, 10),     # long rows, two segments: control warp
    (2, 2, 2, 70001, "f32", "gauss", 0.9, 10),      # scalar path (unaligned rows)
    (2, 3, 2, 33, "f32", "gauss", 1.0, 1),
    (2, 2, 3, 7, "f32", "gauss", 1.0, 10),          # fewer tokens than K
]


@pytest.mark.parametrize("B,K,D,V,dtype,kind,T,topk", CASES)
def test_kl_fused_matches_oracle(vsd, oracle, B, K, D, V, dtype, kind, T, topk):
    from paper_2602_05774_gb300 import inputs
    prob = inputs.linear_problem(B, K, D, V, dtype, kind, seed=300 + V + topk)
    _run(vsd, oracle, prob, T, 0.5, topk, dtype)


def test_kl_ties_at_the_cut(vsd, oracle):
    """Target rows whose top logits tie across the K-th place (bf16): the
    lowest indices are kept, as the oracle keeps them."""
    B, K, D, V = 2, 2, 2, 3000
    R = B * K * D
    g = torch.Generator().manual_seed(5)
    draft = torch.randn(R, V, generator=g)
    target = torch.randn(R, V, generator=g) * 0.5
    for r in range(R):  # 14 equal maxima spread over the row, three chunks apart
        idx = torch.randperm(V, generator=g)[:14]
        target[r, idx] = 4.0
    prob = dict(B=B, K=K, D=D, V=V, draft=draft.to(torch.bfloat16),
                target=target.to(torch.bfloat16), u_draft=torch.rand(R, generator=g),
                u_accept=torch.rand(R, generator=g), u_correct=torch.rand(R, generator=g))
    gpu, orc = _run(vsd, oracle, prob, 1.0, 1.0, 10, "bf16")
    # the gradient's support on each row holds the 10 lowest-index maxima
    tgt = prob["target"].float().numpy()
    for r in range(R):
        top = np.sort(np.nonzero(tgt[r] == 4.0)[0])[:10]
        _, tok, _ = oracle.topk_ce(prob["draft"][r].float().numpy(), tgt[r], 1.0, 10)
        assert sorted(tok.tolist()) == top.tolist()


def test_kl_vocab32k_workload(vsd, oracle):
    """The vocab32k workload (B=16, K=8, D=6, V=32000, bf16) with the term."""
    from paper_2602_05774_gb300 import inputs
    prob = inputs.config("vocab32k")
    g, orc = _run(vsd, oracle, prob, 1.0, 1.0, 10, "bf16")
    assert np.all(np.isfinite(to_np(g["kl_loss"])))
