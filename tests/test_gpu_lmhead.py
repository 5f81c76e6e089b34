"""GPU parity of the draft LM head on the tensor cores (vsd_lmhead_logits) and
of the LM head fused with the E-step + M-step (vsd_lmhead_estep_mstep).

The oracle computes the logits in float64 from the exact bf16 inputs and
rounds them once to bf16.  The GPU sums exact products in float32, so on
inputs whose partial sums are all exact in float32
(inputs.lmhead_exact_problem) both sides must give the same bf16 logits bit
for bit, and everything downstream is held to the usual parity protocol.  On
Gaussian inputs (the paper-shaped workload) each logit must lie within the
float32 summation bound K 2^-24 sum_k |h_k w_k| plus half a bf16 ulp of the
exact value.
"""
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


def _np(t):
    return t.detach().float().cpu().numpy().astype(np.float64)


def _exact_inputs(M, N, K, seed):
    g = torch.Generator(device="cuda").manual_seed(seed)
    h = torch.randint(-2, 3, (M, K), generator=g, device="cuda").to(torch.bfloat16)
    w = (torch.randint(-64, 65, (N, K), generator=g, device="cuda").float() / 256).to(
        torch.bfloat16)
    return h, w


def _gauss_inputs(M, N, K, seed):
    g = torch.Generator(device="cuda").manual_seed(seed)
    h = torch.randn(M, K, generator=g, device="cuda").to(torch.bfloat16)
    w = (torch.randn(N, K, generator=g, device="cuda") * 0.02).to(torch.bfloat16)
    return h, w


def _check_within_bound(oracle, h, w, got):
    H, W = _np(h), _np(w)
    exact = oracle.lmhead_logits(H, W)
    K = H.shape[1]
    bound = K * 2.0**-24 * (np.abs(H) @ np.abs(W).T)
    err = np.abs(_np(got) - exact)
    lim = bound + 2.0**-8 * (np.abs(exact) + bound)  # fp32 sums, then half a bf16 ulp
    assert (err <= lim).all(), "logit off by %g (limit %g)" % (err.max(), lim[err > lim][:1])
    # the one rounding is to nearest: almost every logit is the oracle's rounding
    same = np.mean(_np(got) == oracle.round_bf16(exact).astype(np.float64))
    assert same > 0.99, same


# one tile; ragged M, N and K (K tail read as zeros); many tiles per CTA
SHAPES = [(128, 256, 64), (300, 520, 200), (60, 4104, 264), (1000, 8192, 1024)]


@pytest.mark.parametrize("M,N,K", SHAPES)
def test_lmhead_exact_inputs_bit_exact(vsd, oracle, M, N, K):
    h, w = _exact_inputs(M, N, K, 11 + M)
    got = vsd.lmhead_logits(h, w)
    torch.cuda.synchronize()
    want = oracle.round_bf16(oracle.lmhead_logits(_np(h), _np(w)))
    assert np.array_equal(got.float().cpu().numpy(), want)


@pytest.mark.parametrize("M,N,K", [(300, 1032, 4096), (256, 512, 136)])
def test_lmhead_gaussian_within_fp32_bound(vsd, oracle, M, N, K):
    h, w = _gauss_inputs(M, N, K, 7 + K)
    got = vsd.lmhead_logits(h, w)
    torch.cuda.synchronize()
    _check_within_bound(oracle, h, w, got)


def test_lmhead_full_size_sampled_rows(vsd, oracle):
    """The lmhead workload (4096 x 4096 hidden, 32000 x 4096 weight) as the
    benchmark launches it; rows from the first, a middle and the last M tile
    are checked against the oracle."""
    from paper_2602_05774_gb300 import inputs
    p = inputs.config("lmhead", device="cuda")
    got = vsd.lmhead_logits(p["hidden"], p["weight"])
    torch.cuda.synchronize()
    rows = torch.tensor([0, 1, 77, 127, 128, 2049, 3000, 3967, 3968, 4094, 4095], device="cuda")
    _check_within_bound(oracle, p["hidden"][rows], p["weight"], got[rows])
    assert torch.isfinite(got.float()).all()


@pytest.mark.parametrize("B,K,D,V,H,T", [(2, 4, 4, 4096, 256, 1.0), (3, 5, 4, 4104, 264, 0.7)])
def test_lmhead_estep_mstep_matches_oracle(vsd, oracle, B, K, D, V, H, T):
    from paper_2602_05774_gb300 import inputs
    p = inputs.lmhead_exact_problem(B, K, D, V, H, device="cuda", seed=900 + V)
    ws = vsd.new_workspace(vsd.layout(B, K, D, V), "cuda")
    g = vsd.lmhead_estep_mstep(p["hidden"], p["weight"], p["target"], p["u_draft"],
                               p["u_accept"], p["u_correct"], K, D, T, workspace=ws)
    assert vsd.device_status(ws) == (0, 0)
    draft = oracle.round_bf16(oracle.lmhead_logits(_np(p["hidden"]), _np(p["weight"])))
    assert np.array_equal(g["draft_logits"].float().cpu().numpy(), draft)
    orc = oracle.linear(draft, p["target"].float().cpu().numpy(), T,
                        p["u_draft"].cpu().numpy(), p["u_accept"].cpu().numpy(),
                        p["u_correct"].cpu().numpy(), K, D)
    compare_linear(g, orc, B, K, D, V, T, grad_dtype="bf16",
                   mstep_inputs=mstep_inputs(dict(B=B, K=K, D=D, draft=draft)))


def test_lmhead_estep_mstep_full_size(vsd, oracle):
    """The lmhead workload's shape (R = 64*8*8 = 4096 rows, H = 4096, V =
    32000) through vsd_lmhead_estep_mstep, on inputs whose float32 partial
    sums are exact (so the oracle's logits are the GPU's bit for bit): the
    draft logits of three sampled prefixes (first, middle, last) are checked
    bit for bit, and those prefixes' E-step/M-step results against the oracle
    run on the oracle's own logits."""
    from paper_2602_05774_gb300 import inputs
    from tests.parity import sub_batch
    c = inputs.CONFIGS["lmhead"]
    B, K, D, V, H = c["B"], c["K"], c["D"], c["V"], c["H"]
    p = inputs.lmhead_exact_problem(B, K, D, V, H, device="cuda", seed=4242)
    ws = vsd.new_workspace(vsd.layout(B, K, D, V), "cuda")
    g = vsd.lmhead_estep_mstep(p["hidden"], p["weight"], p["target"], p["u_draft"],
                               p["u_accept"], p["u_correct"], K, D, 1.0, workspace=ws)
    assert vsd.device_status(ws) == (0, 0)
    assert torch.isfinite(g["loss"]).all()
    W = _np(p["weight"])
    P = K * D
    for b in (0, B // 2, B - 1):
        rows = slice(b * P, (b + 1) * P)
        draft = oracle.round_bf16(oracle.lmhead_logits(_np(p["hidden"][rows]), W))
        assert np.array_equal(g["draft_logits"][rows].float().cpu().numpy(), draft), b
        orc = oracle.linear(draft, p["target"][rows].float().cpu().numpy(), 1.0,
                            p["u_draft"][rows].cpu().numpy(), p["u_accept"][rows].cpu().numpy(),
                            p["u_correct"][rows].cpu().numpy(), K, D)
        orc["grad"] = orc["grad"] / B
        compare_linear(sub_batch(g, b, b + 1, B, K, D), orc, 1, K, D, V, 1.0,
                       grad_dtype="bf16", check_mean=False,
                       mstep_inputs=mstep_inputs(dict(B=1, K=K, D=D, draft=draft), B_total=B))
