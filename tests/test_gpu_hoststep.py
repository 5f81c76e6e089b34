"""The end-to-end helpers that feed the kernels from pinned host tensors
(HostStep, HostLMHeadStep, HostTreeStep) keep two device copies of the inputs
and overlap one call's copies with the previous call's kernels.  Run several
calls back to back on alternating inputs with no synchronisation between
them: every call must give what a direct call on device tensors gives."""
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def vsd():
    from paper_2602_05774_gb300 import build, vsd as v
    build.build_library()
    v.load()
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    return v


def _u(p):
    return torch.stack([p["u_draft"], p["u_accept"], p["u_correct"]])


def test_host_step_overlapped_calls(vsd):
    from paper_2602_05774_gb300 import inputs
    B, K, D, V, T = 2, 3, 4, 4096, 1.0
    probs = [inputs.linear_problem(B, K, D, V, "bf16", "spiked", seed=s) for s in (1, 2, 3)]
    want = []
    for p in probs:
        c = {k: (v.cuda() if torch.is_tensor(v) else v) for k, v in p.items()}
        o = vsd.estep_mstep(c["draft"], c["target"], c["u_draft"], c["u_accept"], c["u_correct"],
                            K, D, T)
        want.append((o["loss"].clone(), o["grad"].clone()))
    host = [(p["draft"].pin_memory(), p["target"].pin_memory(), _u(p).pin_memory()) for p in probs]
    hs = vsd.HostStep(B, K, D, V, torch.bfloat16, "cuda", prm=vsd.params(grad_dtype=torch.bfloat16))
    got = []
    for i in range(7):
        hs(*host[i % 3], T)
        got.append((hs.out["loss"].clone(), hs.out["grad"].clone()))  # queued after the call
    torch.cuda.synchronize()
    for i, (loss, grad) in enumerate(got):
        wl, wg = want[i % 3]
        assert torch.equal(loss, wl), i
        assert torch.equal(grad, wg), i
    # the returned pinned loss of the last call
    assert torch.equal(hs.loss_host[(7 - 1) % 2], want[(7 - 1) % 3][0].cpu())


def test_host_lmhead_step_overlapped_calls(vsd):
    from paper_2602_05774_gb300 import inputs
    B, K, D, V, H, T = 2, 4, 4, 4096, 256, 1.0
    probs = [inputs.lmhead_exact_problem(B, K, D, V, H, device="cpu", seed=s) for s in (4, 5)]
    weight = probs[0]["weight"].cuda()
    prm = vsd.params(grad_dtype=torch.bfloat16)
    want = []
    for p in probs:
        c = {k: (v.cuda() if torch.is_tensor(v) else v) for k, v in p.items()}
        o = vsd.lmhead_estep_mstep(c["hidden"], weight, c["target"], c["u_draft"], c["u_accept"],
                                   c["u_correct"], K, D, T, prm=prm)
        want.append((o["loss"].clone(), o["draft_logits"].clone()))
    host = [(p["hidden"].pin_memory(), p["target"].pin_memory(), _u(p).pin_memory()) for p in probs]
    hs = vsd.HostLMHeadStep(weight, B, K, D, V, prm=prm)
    got = []
    for i in range(5):
        hs(*host[i % 2], T)
        got.append((hs.out["loss"].clone(), hs.logits.clone()))
    torch.cuda.synchronize()
    for i, (loss, logits) in enumerate(got):
        assert torch.equal(logits, want[i % 2][1]), i
        assert torch.equal(loss, want[i % 2][0]), i


def test_host_tree_step_overlapped_calls(vsd):
    from paper_2602_05774_gb300 import inputs
    T = 0.9
    probs = [inputs.tree_problem(3, 20, 5, 4, 4096, seed=s) for s in (6, 7)]
    B, N, V = 3, 20, 4096
    names = ("draft", "target", "parent", "tokens", "u_accept", "u_correct")
    keys = ("accept_len", "deepest", "bonus", "corr_tokens", "accept", "logkappa")
    want = []
    for p in probs:
        c = {k: p[k].cuda() for k in names}
        o = vsd.verify_tree(c["draft"], c["target"], c["parent"], c["tokens"], c["u_accept"],
                            c["u_correct"], T)
        want.append({k: o[k].clone() for k in keys})
    host = [{k: p[k].pin_memory() for k in names} for p in probs]
    hs = vsd.HostTreeStep(B, N, V, torch.bfloat16, "cuda")
    got = []
    for i in range(5):
        hs(host[i % 2], T)
        got.append({k: hs.out[k].clone() for k in keys})
    torch.cuda.synchronize()
    for i, g in enumerate(got):
        for k in keys:
            assert torch.equal(g[k], want[i % 2][k]), (i, k)


def test_host_lmhead_training_step_overlapped_calls(vsd):
    """train=True: the draft head's training step from pinned host buffers (no
    dense gradient, then the backward) gives, call after call, the
    d_hidden / d_weight of the same calls made directly on device tensors."""
    from paper_2602_05774_gb300 import inputs
    B, K, D, V, H, T = 2, 4, 4, 4096, 256, 1.0
    probs = [inputs.lmhead_exact_problem(B, K, D, V, H, device="cpu", seed=s) for s in (8, 9)]
    weight = probs[0]["weight"].cuda()
    prm = vsd.params(grad_dtype=torch.bfloat16)
    want = []
    for p in probs:
        c = {k: (v.cuda() if torch.is_tensor(v) else v) for k, v in p.items()}
        ws = vsd.new_workspace(vsd.layout(B, K, D, V), "cuda")
        o = vsd.lmhead_estep_mstep(c["hidden"], weight, c["target"], c["u_draft"], c["u_accept"],
                                   c["u_correct"], K, D, T, prm=prm, workspace=ws, grad=False)
        b = vsd.lmhead_backward(c["hidden"], weight, o["draft_logits"], K, D, T, ws, prm=prm)
        want.append((o["loss"].clone(), b["d_hidden"].clone(), b["d_weight"].clone()))
    host = [(p["hidden"].pin_memory(), p["target"].pin_memory(), _u(p).pin_memory()) for p in probs]
    hs = vsd.HostLMHeadStep(weight, B, K, D, V, prm=prm, train=True)
    got = []
    for i in range(5):
        hs(*host[i % 2], T)
        got.append((hs.out["loss"].clone(), hs.d_hidden.clone(), hs.d_weight.clone()))
    torch.cuda.synchronize()
    assert vsd.device_status(hs.ws) == (0, 0)
    for i, g in enumerate(got):
        for a, b in zip(g, want[i % 2]):
            assert torch.equal(a, b), i
