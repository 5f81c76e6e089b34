"""GPU parity of the draft-tree extensions against the oracle: verification
with the sequential sibling rule (lossless multi-draft, reading R14) and the
E-step + M-step with every node a latent proposal (reading R15)."""
import numpy as np
import pytest
import torch

from tests.parity import compare_tree_em, compare_tree_sequential

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


def _cases():
    from paper_2602_05774_gb300 import inputs
    cases = [("tree60 x12", inputs.config("tree60", B=12)),
             ("small", inputs.tree_problem(3, 12, 4, 3, 777, seed=1)),
             ("ragged V", inputs.tree_problem(2, 30, 6, 5, 4097, seed=2)),
             ("root only", inputs.tree_problem(3, 1, 1, 1, 100, seed=5)),
             ("two nodes", inputs.tree_problem(1, 2, 1, 1, 9, seed=3))]
    # a chain and a star, f32
    g = torch.Generator().manual_seed(8)
    for name, par in (("chain", [-1, 0, 1, 2, 3, 4, 5, 6]), ("star", [-1] + [0] * 8)):
        B, N, V = 3, len(par), 300
        draft = torch.randn(B * N, V, generator=g) * 2.0
        target = draft + torch.randn(B * N, V, generator=g)
        parent = torch.tensor(par, dtype=torch.int32).view(1, N).repeat(B, 1)
        rows = (torch.arange(B).view(B, 1) * N + parent.clamp(min=0).long()).view(-1)
        top = draft.topk(8, dim=1).indices.to(torch.int32)
        tokens = top[rows, torch.randint(0, 8, (B * N,), generator=g)].view(B, N)
        tokens[:, 0] = 0
        cases.append((name, dict(B=B, N=N, V=V, draft=draft, target=target, parent=parent,
                                 tokens=tokens, u_accept=torch.rand(B, N, generator=g),
                                 u_correct=torch.rand(B, N, generator=g))))
    return cases


@pytest.mark.parametrize("T", [1.0, 0.8])
def test_tree_sequential_rule_matches_oracle(vsd, oracle, T):
    for name, prob in _cases():
        B, N = prob["parent"].shape
        orc = oracle.tree(_np32(prob["draft"]), _np32(prob["target"]), T, prob["parent"].numpy(),
                          prob["tokens"].numpy(), _np32(prob["u_accept"]),
                          _np32(prob["u_correct"]), rule=1)
        p = {k: (v.cuda() if torch.is_tensor(v) else v) for k, v in prob.items()}
        for stats in (True, False):
            g = vsd.verify_tree(p["draft"], p["target"], p["parent"], p["tokens"],
                                p["u_accept"], p["u_correct"], T,
                                out=vsd.tree_outputs(B, N, "cuda", stats),
                                rule=vsd.TREE_SEQUENTIAL)
            torch.cuda.synchronize()
            compare_tree_sequential(g, orc)
            # the accepted nodes form one chain from the root
            pa = g["path_accept"].cpu().numpy()
            par = prob["parent"].numpy()
            for b in range(B):
                kids = [n for n in range(1, N) if pa[b, n]]
                assert all(pa[b, par[b, n]] for n in kids)
                assert len({par[b, n] for n in kids}) == len(kids)


@pytest.mark.parametrize("T,grad", [(1.0, "bf16"), (0.7, "f32")])
def test_tree_em_matches_oracle(vsd, oracle, T, grad):
    for name, prob in _cases():
        B, N = prob["parent"].shape
        V = prob["draft"].shape[-1]
        orc = oracle.tree_em(_np32(prob["draft"]), _np32(prob["target"]), T,
                             prob["parent"].numpy(), prob["tokens"].numpy(),
                             _np32(prob["u_accept"]), _np32(prob["u_correct"]))
        p = {k: (v.cuda() if torch.is_tensor(v) else v) for k, v in prob.items()}
        prm = vsd.params(grad_dtype=torch.bfloat16 if grad == "bf16" else torch.float32)
        ws = vsd.new_workspace(vsd.layout(B, V=V, N=N, parent=p["parent"]), "cuda")
        g = vsd.tree_estep_mstep(p["draft"], p["target"], p["parent"], p["tokens"],
                                 p["u_accept"], p["u_correct"], T, prm=prm, workspace=ws)
        torch.cuda.synchronize()
        assert vsd.device_status(ws) == (0, 0), name
        compare_tree_em(g, orc, B, N, V, grad_dtype=grad)
        # each row's gradient sums to ~0 (softmax minus its sparse terms), up to
        # the rounding of its entries
        gr = g["grad"].float()
        rel = 2.0 ** -8 if grad == "bf16" else 1e-6
        assert torch.all(gr.sum(dim=1).abs() <= 1e-6 + rel * gr.abs().sum(dim=1))


def test_tree_em_bad_tree_is_flagged(vsd):
    """A tree whose parent array is malformed sets the tree status bit; its
    loss and gradient rows are 0 and the other trees are unaffected."""
    from paper_2602_05774_gb300 import inputs
    prob = inputs.tree_problem(3, 12, 4, 3, 500, seed=4)
    p = {k: (v.cuda() if torch.is_tensor(v) else v) for k, v in prob.items()}
    good = vsd.tree_estep_mstep(p["draft"], p["target"], p["parent"], p["tokens"], p["u_accept"],
                                p["u_correct"], 1.0)
    par = p["parent"].clone()
    par[1, 5] = 7  # a parent after its node
    ws = vsd.new_workspace(vsd.layout(3, V=500, N=12, parent=par), "cuda")
    g = vsd.tree_estep_mstep(p["draft"], p["target"], par, p["tokens"], p["u_accept"],
                             p["u_correct"], 1.0, workspace=ws)
    code, bits = vsd.device_status(ws)
    assert bits & vsd.STATUS_BAD_TREE
    assert g["loss"][1].item() == 0.0
    assert torch.all(g["grad"][12:24] == 0)
    for b in (0, 2):
        assert g["loss"][b].item() == good["loss"][b].item()
        assert torch.equal(g["grad"][12 * b:12 * (b + 1)], good["grad"][12 * b:12 * (b + 1)])
