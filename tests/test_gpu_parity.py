"""GPU parity: the CUDA path against the CPU oracle on the same seeded inputs.

Runs through the C ABI (Python binding).  Sizes span several chunks and a
ragged tail; the full vocab128k workload is checked on sampled prefixes, in
the launch configuration the benchmark times.
"""
import numpy as np
import pytest
import torch

from tests.parity import compare_linear, compare_tree, mstep_inputs, to_np

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


def run_oracle(oracle, prob, T, **kw):
    return oracle.linear(_np32(prob["draft"]), _np32(prob["target"]), T,
                         _np32(prob["u_draft"]), _np32(prob["u_accept"]),
                         _np32(prob["u_correct"]), prob["K"], prob["D"], **kw)


def to_cuda(prob):
    return {k: (v.cuda() if torch.is_tensor(v) else v) for k, v in prob.items()}


def fused(vsd, p, T, **kw):
    out = vsd.estep_mstep(p["draft"], p["target"], p["u_draft"], p["u_accept"], p["u_correct"],
                          p["K"], p["D"], T, **kw)
    torch.cuda.synchronize()
    return out


@pytest.mark.parametrize("T", [1.0, 0.7])
def test_tiny_fused_matches_oracle(vsd, oracle, T):
    from paper_2602_05774_gb300 import inputs
    prob = inputs.config("tiny")
    orc = run_oracle(oracle, prob, T)
    g = fused(vsd, to_cuda(prob), T)
    compare_linear(g, orc, prob["B"], prob["K"], prob["D"], prob["V"], T, grad_dtype="f32",
                   mstep_inputs=mstep_inputs(prob))


def test_vocab32k_fused_matches_oracle(vsd, oracle):
    from paper_2602_05774_gb300 import inputs
    prob = inputs.config("vocab32k")
    orc = run_oracle(oracle, prob, 1.0)
    g = fused(vsd, to_cuda(prob), 1.0)
    rep = {}
    compare_linear(g, orc, prob["B"], prob["K"], prob["D"], prob["V"], 1.0, grad_dtype="bf16",
                   report=rep, mstep_inputs=mstep_inputs(prob))


SHAPES = [
    # B, K, D, V, dtype, kind, T
    (1, 1, 1, 1, "f32", "gauss", 1.0),
    (2, 3, 2, 2, "f32", "gauss", 0.25),
    (3, 2, 3, 3, "bf16", "gauss", 2.0),
    (2, 5, 3, 7, "f32", "gauss", 1.0),
    (2, 4, 2, 8, "bf16", "gauss", 0.7),
    (1, 3, 5, 33, "f32", "gauss", 1.0),
    (2, 2, 3, 1000, "bf16", "gauss", 1.0),
    (2, 3, 4, 4097, "f32", "gauss", 0.7),
    (2, 3, 4, 4097, "bf16", "spiked", 1.0),
    (1, 7, 3, 5000, "bf16", "zipf", 1.0),
    (3, 1, 6, 2048, "bf16", "spiked", 1.0),
    (2, 16, 1, 1536, "f32", "gauss", 1.0),
    # rows longer than one work segment (several segments per row and per
    # residual row): V above 128 chunks of 1024 bf16 / 512 f32 values
    (1, 3, 3, 140000, "bf16", "zipf", 1.0),
    (2, 2, 2, 70001, "f32", "gauss", 0.9),
    (1, 2, 4, 262400, "bf16", "spiked", 1.0),
]


@pytest.mark.parametrize("B,K,D,V,dtype,kind,T", SHAPES)
def test_random_shapes_fused(vsd, oracle, B, K, D, V, dtype, kind, T):
    from paper_2602_05774_gb300 import inputs
    prob = inputs.linear_problem(B, K, D, V, dtype, kind, seed=1000 + V + 7 * K + D)
    orc = run_oracle(oracle, prob, T)
    g = fused(vsd, to_cuda(prob), T)
    compare_linear(g, orc, B, K, D, V, T, grad_dtype=dtype, mstep_inputs=mstep_inputs(prob))


@pytest.mark.parametrize("zeta_mode,ref", [(1, False), (0, True)])
def test_params_and_reference_input(vsd, oracle, zeta_mode, ref):
    from paper_2602_05774_gb300 import inputs
    prob = inputs.linear_problem(3, 4, 3, 3000, "bf16", "spiked", seed=77)
    refk = None
    if ref:
        refk = torch.linspace(-0.5, -3.0, 9).reshape(3, 3).float()
    orc = run_oracle(oracle, prob, 1.0, zeta_mode=zeta_mode, tau_car=0.5, w_base=1.2,
                     ref_logkappa=None if refk is None else refk.numpy())
    p = to_cuda(prob)
    prm = vsd.params(w_base=1.2, tau_car=0.5, zeta_mode=zeta_mode, grad_dtype=torch.float32)
    g = fused(vsd, p, 1.0, prm=prm, ref_logkappa=None if refk is None else refk.cuda())
    compare_linear(g, orc, 3, 4, 3, 3000, 1.0, grad_dtype="f32",
                   mstep_inputs=mstep_inputs(prob, w_base=1.2, tau_car=0.5, zeta_mode=zeta_mode))


def test_draft_equals_target(vsd, oracle):
    from paper_2602_05774_gb300 import inputs
    prob = inputs.linear_problem(2, 4, 4, 2500, "bf16", "gauss", seed=5)
    prob["target"] = prob["draft"].clone()
    orc = run_oracle(oracle, prob, 1.0)
    g = fused(vsd, to_cuda(prob), 1.0)
    assert np.all(to_np(g["alpha"]) == 1.0)
    assert np.all(to_np(g["accept_len"]) == 4)
    compare_linear(g, orc, 2, 4, 4, 2500, 1.0, grad_dtype="bf16", mstep_inputs=mstep_inputs(prob))


def test_one_token_rows(vsd, oracle):
    """All -inf logits but one token per row (and a few two-token rows)."""
    B, K, D, V = 2, 3, 3, 3000
    R = B * K * D
    gen = torch.Generator().manual_seed(3)
    draft = torch.full((R, V), float("-inf"))
    target = torch.full((R, V), float("-inf"))
    idx = torch.randint(0, V, (R,), generator=gen)
    draft[torch.arange(R), idx] = 1.0
    target[torch.arange(R), idx] = 2.0
    idx2 = torch.randint(0, V, (R,), generator=gen)
    target[torch.arange(R)[::2], idx2[::2]] = 1.5
    draft[torch.arange(R)[::3], idx2[::3]] = 0.5
    prob = dict(B=B, K=K, D=D, V=V, draft=draft, target=target,
                u_draft=torch.rand(R, generator=gen), u_accept=torch.rand(R, generator=gen),
                u_correct=torch.rand(R, generator=gen))
    orc = run_oracle(oracle, prob, 1.0)
    g = fused(vsd, to_cuda(prob), 1.0, prm=vsd.params(grad_dtype=torch.float32))
    compare_linear(g, orc, B, K, D, V, 1.0, grad_dtype="f32", mstep_inputs=mstep_inputs(prob))


def test_separate_entry_points(vsd, oracle):
    """sample -> verify -> weighted loss, each fed the oracle's own E-step results."""
    from paper_2602_05774_gb300 import inputs
    B, K, D, V, T = 3, 4, 3, 5000, 0.8
    prob = inputs.linear_problem(B, K, D, V, "bf16", "spiked", seed=11)
    orc = run_oracle(oracle, prob, T)
    p = to_cuda(prob)
    s = vsd.sample_paths(p["draft"], p["u_draft"], K, D, T)
    torch.cuda.synchronize()
    m = orc["margins"][:, 0] >= 1e-6
    assert np.array_equal(to_np(s["tokens"])[m], orc["tokens"][m])
    assert np.allclose(to_np(s["logq_tok"]), orc["logq_tok"], atol=2e-5, rtol=1e-6)
    tok = torch.from_numpy(orc["tokens"]).cuda()
    v = vsd.verify_paths(p["draft"], p["target"], tok, p["u_accept"], p["u_correct"], K, D, T)
    torch.cuda.synchronize()
    compare_linear(v, orc, B, K, D, V, T, check_grad=False)
    es = {n: torch.from_numpy(np.ascontiguousarray(orc[n])).cuda() for n in
          ("tokens", "corr_tokens")}
    for n in ("logq_tok", "logq_corr", "logkappa", "logkappa_corr", "logkappa_ref"):
        es[n] = torch.from_numpy(orc[n].astype(np.float32)).cuda()
    rs = to_np(v["row_stats"])  # statistics of the draft rows (inputs, not decisions)
    es["row_stats"] = torch.from_numpy(rs).cuda()
    lo = vsd.weighted_loss_fwd_bwd(p["draft"], es, K, D, T,
                                   prm=vsd.params(grad_dtype=torch.float32))
    torch.cuda.synchronize()
    res = dict(loss=lo["loss"], grad=lo["grad"], weights=lo["weights"],
               accept_len=torch.from_numpy(orc["accept_len"]),
               corr_tokens=torch.from_numpy(orc["corr_tokens"]),
               logkappa=torch.from_numpy(orc["logkappa"].astype(np.float32)))
    compare_linear(res, orc, B, K, D, V, T, grad_dtype="f32")


def test_tree60_matches_oracle(vsd, oracle):
    from paper_2602_05774_gb300 import inputs
    prob = inputs.config("tree60")
    B, N, V = prob["B"], prob["N"], prob["V"]
    orc = oracle.tree(_np32(prob["draft"]), _np32(prob["target"]), 1.0, prob["parent"].numpy(),
                      prob["tokens"].numpy(), _np32(prob["u_accept"]), _np32(prob["u_correct"]))
    p = to_cuda(prob)
    for stats in (True, False):  # without row statistics leaf rows are not read
        g = vsd.verify_tree(p["draft"], p["target"], p["parent"], p["tokens"], p["u_accept"],
                            p["u_correct"], 1.0, out=vsd.tree_outputs(B, N, "cuda", stats))
        torch.cuda.synchronize()
        compare_tree(g, orc)


def test_small_trees_matches_oracle(vsd, oracle):
    from paper_2602_05774_gb300 import inputs
    for (B, N, depth, topk, V, seed) in [(3, 12, 4, 3, 777, 1), (2, 30, 6, 5, 4096, 2),
                                         (1, 2, 1, 1, 9, 3)]:
        prob = inputs.tree_problem(B, N, depth, topk, V, seed=seed)
        orc = oracle.tree(_np32(prob["draft"]), _np32(prob["target"]), 0.9,
                          prob["parent"].numpy(), prob["tokens"].numpy(),
                          _np32(prob["u_accept"]), _np32(prob["u_correct"]))
        p = to_cuda(prob)
        for stats in (True, False):
            g = vsd.verify_tree(p["draft"], p["target"], p["parent"], p["tokens"],
                                p["u_accept"], p["u_correct"], 0.9,
                                out=vsd.tree_outputs(B, N, "cuda", stats))
            torch.cuda.synchronize()
            compare_tree(g, orc)



def _tree_case(B, N, V, parent, seed, same=False):
    """Random spiked logits (target = draft if same) for a given parent array,
    node tokens drawn among each parent row's 8 largest draft logits."""
    g = torch.Generator().manual_seed(seed)
    draft = torch.randn(B * N, V, generator=g) * 3.0
    target = draft.clone() if same else draft + torch.randn(B * N, V, generator=g)
    parent = torch.as_tensor(parent, dtype=torch.int32).view(1, N).repeat(B, 1)
    top = draft.topk(min(8, V), dim=1).indices.to(torch.int32)
    rows = (torch.arange(B).view(B, 1) * N + parent.clamp(min=0).long()).view(-1)
    pick = torch.randint(0, min(8, V), (B * N,), generator=g)
    tokens = top[rows, pick].view(B, N)
    tokens[:, 0] = 0
    return dict(B=B, N=N, V=V, draft=draft.to(torch.bfloat16), target=target.to(torch.bfloat16),
                parent=parent, tokens=tokens,
                u_accept=torch.rand(B, N, generator=g), u_correct=torch.rand(B, N, generator=g))


def test_tree_edge_shapes(vsd, oracle):
    """Root-only trees, the largest tree (1024 nodes), a chain whose every
    token is accepted (target = draft: no residual row, the bonus is the leaf
    row's p-draw) and a star (every node a child of the root)."""
    from paper_2602_05774_gb300 import inputs
    cases = [inputs.tree_problem(3, 1, 1, 1, 100, seed=5),
             inputs.tree_problem(2, 1024, 17, 8, 64, seed=6),
             _tree_case(2, 8, 50, [-1, 0, 1, 2, 3, 4, 5, 6], seed=7, same=True),
             _tree_case(3, 9, 300, [-1] + [0] * 8, seed=8)]
    for i, prob in enumerate(cases):
        orc = oracle.tree(_np32(prob["draft"]), _np32(prob["target"]), 1.0,
                          prob["parent"].numpy(), prob["tokens"].numpy(),
                          _np32(prob["u_accept"]), _np32(prob["u_correct"]))
        p = to_cuda(prob)
        B, N = prob["parent"].shape
        for stats in (True, False):  # without row statistics leaf rows are not read
            g = vsd.verify_tree(p["draft"], p["target"], p["parent"], p["tokens"],
                                p["u_accept"], p["u_correct"], 1.0,
                                out=vsd.tree_outputs(B, N, "cuda", stats))
            torch.cuda.synchronize()
            compare_tree(g, orc)
            if i == 2:  # the chain: every node accepted, so the accepted length is N - 1
                assert (g["accept_len"].cpu() == 7).all()



@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_tree_lattice_residual_and_bonus(vsd, oracle, dtype):
    """512 three-node trees (a root and two leaves) with dyadic rows and a
    lattice of uniforms: every bonus token is a draw at a leaf's row (the leaf
    row skipped without row statistics is read for it), and half the trees
    draw a residual token at the root row."""
    q4, uni, pb = [0.5, 0.25, 0.125, 0.125], [0.25] * 4, [0.125, 0.375, 0.25, 0.25]
    rows_q = np.log(np.array([q4, q4, q4]))
    rows_p = np.log(np.array([uni, pb, uni]))
    M, N, V = 8, 3, 4
    lat = (np.arange(M) + 0.5) / M
    g = np.meshgrid(lat, lat, lat, indexing="ij")
    B = M ** 3
    ua = np.zeros((B, N), np.float32)
    uc = np.zeros((B, N), np.float32)
    ua[:, 1], ua[:, 2] = g[0].ravel(), 0.999
    uc[:, 1], uc[:, 2] = g[1].ravel(), g[2].ravel()
    prob = dict(B=B, N=N, V=V,
                draft=torch.tensor(np.tile(rows_q, (B, 1)), dtype=torch.float32).to(dtype),
                target=torch.tensor(np.tile(rows_p, (B, 1)), dtype=torch.float32).to(dtype),
                parent=torch.tensor([[-1, 0, 0]] * B, dtype=torch.int32),
                tokens=torch.tensor([[0, 0, 2]] * B, dtype=torch.int32),
                u_accept=torch.from_numpy(ua), u_correct=torch.from_numpy(uc))
    orc = oracle.tree(_np32(prob["draft"]), _np32(prob["target"]), 1.0, prob["parent"].numpy(),
                      prob["tokens"].numpy(), ua, uc)
    p = to_cuda(prob)
    for stats in (True, False):
        g_ = vsd.verify_tree(p["draft"], p["target"], p["parent"], p["tokens"], p["u_accept"],
                             p["u_correct"], 1.0, out=vsd.tree_outputs(B, N, "cuda", stats))
        torch.cuda.synchronize()
        compare_tree(g_, orc)


def test_vocab128k_full_size_all_prefixes(vsd, oracle):
    """The benchmark's workload (B=32, K=16, D=8, V=128256, bf16) in the launch
    the benchmark times, T = 1: every prefix against the oracle over the whole
    batch (the oracle's own gradient scale 1/B matches the call's)."""
    from paper_2602_05774_gb300 import inputs
    prob = inputs.config("vocab128k", device="cuda")
    B, K, D, V = prob["B"], prob["K"], prob["D"], prob["V"]
    g = fused(vsd, prob, 1.0)
    rs = g["grad"].float().sum(dim=1)  # each gradient row sums to ~0
    assert torch.isfinite(g["loss"]).all() and rs.abs().max().item() < 1e-3
    orc = run_oracle(oracle, prob, 1.0)
    rep = {}
    compare_linear(g, orc, B, K, D, V, 1.0, grad_dtype="bf16", report=rep,
                   mstep_inputs=mstep_inputs(prob))
    print("vocab128k T=1: %s" % rep)


def test_vocab128k_last_published_prefixes(vsd, oracle):
    """T = 0.7, the four prefixes the fused kernel publishes last (their
    gradient segments are scheduled after every other prefix's), compared as
    a sub-batch of the full call."""
    from paper_2602_05774_gb300 import inputs
    from tests.parity import sub_batch
    prob = inputs.config("vocab128k", device="cuda")
    B, K, D, V = prob["B"], prob["K"], prob["D"], prob["V"]
    T = 0.7
    g = fused(vsd, prob, T)
    b0 = B - 4
    P = K * D
    rows = slice(b0 * P, B * P)
    sub = dict(B=4, K=K, D=D, V=V, draft=prob["draft"][rows], target=prob["target"][rows],
               u_draft=prob["u_draft"][rows], u_accept=prob["u_accept"][rows],
               u_correct=prob["u_correct"][rows])
    orc = run_oracle(oracle, sub, T)
    orc["grad"] = orc["grad"] * (4.0 / B)  # the call normalises over its B prefixes
    rep = {}
    compare_linear(sub_batch(g, b0, B, B, K, D), orc, 4, K, D, V, T, grad_dtype="bf16",
                   report=rep, check_mean=False, mstep_inputs=mstep_inputs(sub, B_total=B))
    print("vocab128k T=0.7 last prefixes: %s" % rep)
