"""GPU robustness: bounded waits that run out, device-side data checks,
determinism, prefix sharding, and the exact output distribution of the
accept/resample rule on a lattice of uniforms.  Nothing here faults or hangs
a GPU: failures are made on the host or by a flag that nothing sets, and the
kernels report them through the workspace status word."""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def vsd():
    from paper_2602_05774_gb300 import build, vsd as v
    build.build_library()
    v.load()
    return v


def _cuda(prob):
    return {k: (v.cuda() if torch.is_tensor(v) else v) for k, v in prob.items()}


def _run(vsd, p, T=1.0, **kw):
    out = vsd.estep_mstep(p["draft"], p["target"], p["u_draft"], p["u_accept"], p["u_correct"],
                          p["K"], p["D"], T, **kw)
    torch.cuda.synchronize()
    return out


def test_wait_timeout_is_reported_and_context_survives(vsd):
    from paper_2602_05774_gb300 import inputs
    p = _cuda(inputs.config("tiny"))
    lay = vsd.layout(p["B"], p["K"], p["D"], p["V"])
    ws = vsd.new_workspace(lay, "cuda")
    prm = vsd.params(grad_dtype=torch.float32, wait_timeout_ns=2_000_000, test_never_publish=1)
    _run(vsd, p, prm=prm, workspace=ws)
    code, bits = vsd.device_status(ws)
    assert code == 4 and bits & vsd.STATUS_TIMEOUT
    # the context is still usable and a normal call is clean
    out = _run(vsd, p, prm=vsd.params(grad_dtype=torch.float32), workspace=ws)
    code, bits = vsd.device_status(ws)
    assert code == 0 and bits == 0
    assert torch.isfinite(out["loss"]).all()


def test_nan_row_sets_status(vsd):
    from paper_2602_05774_gb300 import inputs
    p = _cuda(inputs.linear_problem(2, 2, 2, 300, "f32", "gauss", seed=3))
    p["draft"][3, 17] = float("nan")
    lay = vsd.layout(2, 2, 2, 300)
    ws = vsd.new_workspace(lay, "cuda")
    _run(vsd, p, workspace=ws)
    code, bits = vsd.device_status(ws)
    assert code == 6 and bits & vsd.STATUS_BAD_ROW


def test_bad_tree_and_bad_token_set_status(vsd):
    from paper_2602_05774_gb300 import inputs
    prob = inputs.tree_problem(2, 8, 3, 3, 500, seed=4)
    p = _cuda(prob)
    parent = p["parent"].clone()
    parent[1, 5] = 5  # not an earlier node
    lay = vsd.layout(2, V=500, N=8, parent=parent)
    ws = vsd.new_workspace(lay, "cuda")
    out = vsd.verify_tree(p["draft"], p["target"], parent, p["tokens"], p["u_accept"],
                          p["u_correct"], 1.0, workspace=ws)
    code, bits = vsd.device_status(ws)
    assert bits & vsd.STATUS_BAD_TREE
    assert out["deepest"][1].item() == -1 and out["deepest"][0].item() >= 0
    tok = p["tokens"].clone()
    tok[0, 3] = 500
    vsd.verify_tree(p["draft"], p["target"], p["parent"], tok, p["u_accept"], p["u_correct"],
                    1.0, workspace=ws)
    code, bits = vsd.device_status(ws)
    assert bits & vsd.STATUS_BAD_TOKEN


def test_deterministic(vsd):
    from paper_2602_05774_gb300 import inputs
    p = _cuda(inputs.config("vocab32k"))
    a = _run(vsd, p)
    b = _run(vsd, p)
    for k in a:
        assert torch.equal(a[k], b[k]), k


def test_prefix_sharding_matches_whole_batch(vsd):
    """Prefixes are independent (the decomposition a multi-GPU run shards by):
    two half batches give the whole batch's results, gradients scaled by the
    batch-size ratio (an exact power of two here)."""
    from paper_2602_05774_gb300 import inputs
    p = _cuda(inputs.config("vocab32k"))
    B, K, D = p["B"], p["K"], p["D"]
    full = _run(vsd, p)
    h = B // 2
    P = K * D
    for part in range(2):
        rows = slice(part * h * P, (part + 1) * h * P)
        q = dict(K=K, D=D, draft=p["draft"][rows].contiguous(),
                 target=p["target"][rows].contiguous(), u_draft=p["u_draft"][rows].contiguous(),
                 u_accept=p["u_accept"][rows].contiguous(),
                 u_correct=p["u_correct"][rows].contiguous())
        o = _run(vsd, q)
        for n in ("tokens", "accept", "corr_tokens", "ref_tokens", "alpha", "logkappa"):
            assert torch.equal(o[n], full[n][rows]), n
        paths = slice(part * h * K, (part + 1) * h * K)
        assert torch.equal(o["accept_len"], full["accept_len"][paths])
        assert torch.equal(o["loss"][:h], full["loss"][part * h:(part + 1) * h])
        assert torch.equal(o["grad"].float() * 0.5, full["grad"][rows].float())


def test_lattice_output_distribution_is_target(vsd):
    """Sec. 3: accept-or-resample outputs an exact sample of p.  Dyadic q, p and
    a midpoint lattice over the three uniforms make the histogram exact."""
    q = torch.tensor([1 / 2, 1 / 4, 1 / 8, 1 / 8], dtype=torch.float64)
    pp = torch.tensor([1 / 4, 1 / 4, 1 / 4, 1 / 4], dtype=torch.float64)
    M = 16
    lat = (torch.arange(M, dtype=torch.float64) + 0.5) / M
    ud, ua, uc = torch.meshgrid(lat, lat, lat, indexing="ij")
    Bn = M ** 3
    prob = dict(K=1, D=1, draft=q.log().float().repeat(Bn, 1), target=pp.log().float().repeat(Bn, 1),
                u_draft=ud.reshape(-1).float(), u_accept=ua.reshape(-1).float(),
                u_correct=uc.reshape(-1).float())
    o = _run(vsd, _cuda(prob), prm=vsd.params(grad_dtype=torch.float32))
    hist = torch.bincount(o["corr_tokens"].long().cpu(), minlength=4).double() / Bn
    assert torch.equal(hist, pp)
    assert o["accept"].double().mean().item() == 0.75
