"""CPU checks of the parity protocol itself (tests/parity.py): a comparison
that is handed a wrong GPU result must fail.  The "GPU" side here is the
oracle's own output cast to the GPU's output types, with one planted fault."""
import numpy as np
import pytest

from tests import parity


def _problem(oracle, B, K=3, D=3, V=300, seed=4):
    from paper_2602_05774_gb300 import inputs
    p = inputs.linear_problem(B, K, D, V, "f32", "gauss", seed=seed)
    f = {k: p[k].numpy() for k in ("draft", "target", "u_draft", "u_accept", "u_correct")}
    orc = oracle.linear(f["draft"], f["target"], 1.0, f["u_draft"], f["u_accept"],
                        f["u_correct"], K, D)
    gpu = {}
    for n in ("tokens", "accept_len", "corr_tokens", "ref_tokens"):
        gpu[n] = orc[n].astype(np.int32)
    gpu["accept"] = orc["accept"].astype(np.uint8)
    for n in ("alpha", "alpha_corr", "logq_tok", "logq_corr", "logkappa", "logkappa_corr",
              "logkappa_ref", "expected_len", "loss", "grad", "weights"):
        gpu[n] = orc[n].astype(np.float32)
    return gpu, orc, (B, K, D, V)


def _fails(gpu, orc, shape):
    B, K, D, V = shape
    with pytest.raises(AssertionError):
        parity.compare_linear(gpu, orc, B, K, D, V, 1.0, grad_dtype="f32")


def test_faithful_copy_passes(oracle):
    gpu, orc, shape = _problem(oracle, 4)
    B, K, D, V = shape
    rep = {}
    assert parity.compare_linear(gpu, orc, B, K, D, V, 1.0, grad_dtype="f32", report=rep) == 0
    assert rep["excluded_prefixes"] == 0


@pytest.mark.parametrize("name", ["alpha", "alpha_corr", "logq_tok", "logkappa",
                                  "logkappa_corr", "logkappa_ref", "expected_len", "loss"])
def test_nan_in_a_float_output_fails(oracle, name):
    gpu, orc, shape = _problem(oracle, 4)
    gpu[name] = gpu[name].copy()
    gpu[name].reshape(-1)[1] = np.nan
    _fails(gpu, orc, shape)


def test_lone_infinity_fails(oracle):
    gpu, orc, shape = _problem(oracle, 4)
    finite = np.nonzero(np.isfinite(orc["logkappa"]))[0]
    gpu["logkappa"] = gpu["logkappa"].copy()
    gpu["logkappa"][finite[0]] = -np.inf
    _fails(gpu, orc, shape)


def test_nan_in_gradient_fails(oracle):
    gpu, orc, shape = _problem(oracle, 4)
    gpu["grad"] = gpu["grad"].copy()
    gpu["grad"][2, 7] = np.nan
    _fails(gpu, orc, shape)


def test_token_off_the_boundary_fails(oracle):
    gpu, orc, shape = _problem(oracle, 4)
    r = int(np.argmax(orc["margins"][:, 0]))  # the decision farthest from a boundary
    gpu["tokens"] = gpu["tokens"].copy()
    gpu["tokens"][r] = (gpu["tokens"][r] + 1) % shape[3]
    _fails(gpu, orc, shape)


def _plant_near_boundary_divergence(gpu, orc, b, K, D, V):
    """Make prefix b's first draft sample a near-boundary decision that the
    GPU side took differently (the margin is the oracle's report)."""
    r = b * K * D
    orc["margins"] = orc["margins"].copy()
    orc["margins"][r, 0] = 1e-8
    gpu["tokens"] = gpu["tokens"].copy()
    gpu["tokens"][r] = (gpu["tokens"][r] + 1) % V


def test_excluded_prefix_is_counted(oracle):
    gpu, orc, shape = _problem(oracle, 12)
    B, K, D, V = shape
    _plant_near_boundary_divergence(gpu, orc, 5, K, D, V)
    rep = {}
    assert parity.compare_linear(gpu, orc, B, K, D, V, 1.0, grad_dtype="f32", report=rep) == 1
    assert rep["excluded_prefixes"] == 1 and rep["near_boundary_decisions"] >= 1


@pytest.mark.parametrize("B", [1, 2])
def test_small_call_may_exclude_nothing(oracle, B):
    """A call of one or two prefixes compares every prefix: excluding the only
    one (or half of two) would leave a wrong result unchecked."""
    gpu, orc, shape = _problem(oracle, B)
    _plant_near_boundary_divergence(gpu, orc, 0, *shape[1:])
    _fails(gpu, orc, shape)


def test_budget_is_one_in_ten(oracle):
    gpu, orc, shape = _problem(oracle, 12)
    B, K, D, V = shape
    for b in (1, 7):  # two of twelve: over the budget of one
        _plant_near_boundary_divergence(gpu, orc, b, K, D, V)
    _fails(gpu, orc, shape)
    assert parity.exclusion_budget(32) == 3 and parity.exclusion_budget(3) == 1
    assert parity.exclusion_budget(2) == 0 and parity.exclusion_budget(1) == 0


def _gpu_view(o):
    gpu = {}
    for n in ("tokens", "accept_len", "corr_tokens", "ref_tokens"):
        gpu[n] = o[n].astype(np.int32)
    gpu["accept"] = o["accept"].astype(np.uint8)
    for n in ("alpha", "alpha_corr", "logq_tok", "logq_corr", "logkappa", "logkappa_corr",
              "logkappa_ref", "expected_len", "loss", "grad", "weights"):
        gpu[n] = o[n].astype(np.float32)
    return gpu


@pytest.mark.parametrize("lam", [0.0, 0.4])
def test_flipped_draw_is_checked_conditionally(oracle, lam):
    """A consistent result that took one near-boundary draft draw the other
    way (the oracle itself run with that row's uniform moved across the CDF
    boundary by one float step) passes: the flipped path is compared up to
    the flip and the prefix's M-step conditionally; the same result with its
    loss changed fails."""
    from paper_2602_05774_gb300 import inputs
    B, K, D, V = 4, 3, 3, 300
    p = inputs.linear_problem(B, K, D, V, "f32", "gauss", seed=8)
    f = {k: p[k].numpy().copy() for k in ("draft", "target", "u_draft", "u_accept", "u_correct")}
    r = K * D + 1  # prefix 1, path 0, row 1
    q = np.exp(oracle.log_softmax(f["draft"][r], 1.0))
    F = float(np.cumsum(q)[10])
    below = np.float32(F)
    while float(below) >= F:
        below = np.nextafter(below, np.float32(0))
    above = np.nextafter(below, np.float32(1))
    assert float(below) < F <= float(above)
    f["u_draft"][r] = below
    orc = oracle.linear(f["draft"], f["target"], 1.0, f["u_draft"], f["u_accept"],
                        f["u_correct"], K, D, kl_weight=lam)
    f2 = dict(f)
    f2["u_draft"] = f["u_draft"].copy()
    f2["u_draft"][r] = above
    o2 = oracle.linear(f2["draft"], f2["target"], 1.0, f2["u_draft"], f2["u_accept"],
                       f2["u_correct"], K, D, kl_weight=lam)
    assert o2["tokens"][r] != orc["tokens"][r] and orc["margins"][r, 0] < parity.PROB_MARGIN
    gpu = _gpu_view(o2)
    P = K * D
    mi = dict(draft_rows=lambda b: f["draft"][b * P:(b + 1) * P],
              target_rows=lambda b: f["target"][b * P:(b + 1) * P], B_total=B, kl_weight=lam)
    gpu["kl_loss"] = o2["kl_loss"].astype(np.float32)
    rep = {}
    assert parity.compare_linear(gpu, orc, B, K, D, V, 1.0, grad_dtype="f32", report=rep,
                                 mstep_inputs=mi, kl=lam > 0) == 1
    assert rep["diverged_paths"] == 1 and rep["conditional_prefixes"] == 1
    bad = _gpu_view(o2)
    bad["loss"][1] += 1e-3
    with pytest.raises(AssertionError):
        parity.compare_linear(bad, orc, B, K, D, V, 1.0, grad_dtype="f32", mstep_inputs=mi)
    bad = _gpu_view(o2)
    bad["grad"][P + 2, 5] += 1e-3
    with pytest.raises(AssertionError):
        parity.compare_linear(bad, orc, B, K, D, V, 1.0, grad_dtype="f32", mstep_inputs=mi)
