"""Seeded synthetic inputs for the VSD E-step / M-step workloads.

This module only draws random numbers and lays them out; it holds none of the
method's arithmetic (no softmax, sampling, acceptance or weighting), so the
CPU oracle and the CUDA path can both consume its output.  Everything is drawn
with torch's seeded generators on the requested device, so the same (config,
seed, device) always yields the same bytes.  Logits are drawn in float32 and
rounded to bf16 (round-to-nearest-even) where the workload is bf16.

Workloads (the paper's draft/target distributions stand in for trained
EAGLE-3/MSD drafts on ShareGPT-style text; no model or dataset is used):

  tiny       B=2  K=4  D=4 V=1024   f32  draft~N(0,2^2), target=draft+N(0,0.5^2), T=1
  vocab32k   B=16 K=8  D=6 V=32000  bf16 draft~N(0,3^2) + 8 on 50 random tokens/row,
                                         target=draft+N(0,1), T=1
  vocab128k  B=32 K=16 D=8 V=128256 bf16 target logit of rank r = -1.1 ln r under a
                                         random permutation per row (Zipf s=1.1),
                                         draft=target+N(0,1.5^2), T in {0.7, 1.0}
  tree60     B=64 trees of N=60 nodes (depth<=7, top-8 expansion, rerank to 60),
             V=32000 bf16 rows as vocab32k
  lmhead     hidden [4096 x 4096] bf16 ~N(0,1), LM-head weight [32000 x 4096] bf16
             ~N(0,0.02^2) (nn.Linear layout: V rows of H), target as vocab32k

Rows are [B][K][D][V] (row r = (b*K + s)*D + d) for linear paths and [B][N][V]
for trees; uniforms are float32 in [0, 1), one per row and per use.
"""
import math

import torch

CONFIGS = {
    "tiny": dict(B=2, K=4, D=4, V=1024, dtype="f32", T=(1.0,)),
    "vocab32k": dict(B=16, K=8, D=6, V=32000, dtype="bf16", T=(1.0,)),
    "vocab128k": dict(B=32, K=16, D=8, V=128256, dtype="bf16", T=(0.7, 1.0)),
    "tree60": dict(B=64, N=60, depth=7, topk=8, V=32000, dtype="bf16", T=(1.0,)),
    "lmhead": dict(B=64, K=8, D=8, V=32000, H=4096, dtype="bf16", T=(1.0,)),
}

BASE_SEED = 20260205


def _gen(device, seed):
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def _cast(x, dtype):
    return x.to(torch.bfloat16) if dtype == "bf16" else x.to(torch.float32)


def uniforms(n, device, seed):
    """float32 uniforms in [0, 1)."""
    return torch.rand(n, generator=_gen(device, seed), device=device, dtype=torch.float32)


def logits_gaussian(R, V, sigma, device, seed):
    return torch.randn(R, V, generator=_gen(device, seed), device=device) * sigma


def logits_spiked(R, V, sigma, n_spike, spike, device, seed):
    """N(0, sigma^2) plus `spike` added on n_spike distinct random tokens per row."""
    g = _gen(device, seed)
    x = torch.randn(R, V, generator=g, device=device) * sigma
    idx = torch.rand(R, V, generator=g, device=device).topk(n_spike, dim=1).indices
    x.scatter_add_(1, idx, torch.full(idx.shape, float(spike), device=device))
    return x


def logits_zipf(R, V, s, device, seed, chunk=256):
    """Logit -s*ln(rank) with ranks assigned by a random permutation per row."""
    g = _gen(device, seed)
    out = torch.empty(R, V, device=device)
    base = -s * torch.log(torch.arange(1, V + 1, device=device, dtype=torch.float32))
    for r0 in range(0, R, chunk):
        r1 = min(R, r0 + chunk)
        perm = torch.rand(r1 - r0, V, generator=g, device=device).argsort(dim=1)
        out[r0:r1].scatter_(1, perm, base.expand(r1 - r0, V).contiguous())
    return out


def linear_problem(B, K, D, V, dtype="bf16", kind="gauss", device="cpu", seed=BASE_SEED,
                   draft_sigma=2.0, noise_sigma=0.5):
    """A linear-path problem: draft/target [B*K*D, V] and three uniform vectors.

    kind: 'gauss' (draft~N(0,draft_sigma^2), target=draft+noise),
          'spiked' (vocab32k recipe), 'zipf' (vocab128k recipe)."""
    R = B * K * D
    if kind == "gauss":
        d = logits_gaussian(R, V, draft_sigma, device, seed + 1)
        t = d + logits_gaussian(R, V, noise_sigma, device, seed + 2)
    elif kind == "spiked":
        d = logits_spiked(R, V, 3.0, min(50, V), 8.0, device, seed + 1)
        t = d + logits_gaussian(R, V, 1.0, device, seed + 2)
    elif kind == "zipf":
        t = logits_zipf(R, V, 1.1, device, seed + 2)
        d = t + logits_gaussian(R, V, 1.5, device, seed + 1)
    else:
        raise ValueError(kind)
    return dict(B=B, K=K, D=D, V=V, dtype=dtype,
                draft=_cast(d, dtype).contiguous(), target=_cast(t, dtype).contiguous(),
                u_draft=uniforms(R, device, seed + 3), u_accept=uniforms(R, device, seed + 4),
                u_correct=uniforms(R, device, seed + 5))


def config(name, device="cpu", seed=None, B=None):
    """The named workload (see the module docstring); B overrides the number of
    prefixes (trees) for small profiling runs of the same shapes."""
    c = dict(CONFIGS[name])
    if B is not None:
        c["B"] = int(B)
    idx = list(CONFIGS).index(name)
    seed = BASE_SEED + idx if seed is None else seed
    if name == "tiny":
        return linear_problem(c["B"], c["K"], c["D"], c["V"], "f32", "gauss", device, seed)
    if name == "vocab32k":
        return linear_problem(c["B"], c["K"], c["D"], c["V"], "bf16", "spiked", device, seed)
    if name == "vocab128k":
        return linear_problem(c["B"], c["K"], c["D"], c["V"], "bf16", "zipf", device, seed)
    if name == "tree60":
        return tree_problem(c["B"], c["N"], c["depth"], c["topk"], c["V"], device, seed)
    if name == "lmhead":
        return lmhead_problem(c["B"], c["K"], c["D"], c["V"], c["H"], device, seed)
    raise KeyError(name)


def tree_shapes(B, N, depth, topk, seed):
    """EAGLE-2-style draft-tree shapes (App. E): per layer the top-`topk` frontier
    nodes by score are expanded with `topk` children each; after `depth` layers
    all candidates are reranked by score and the best N-1 (plus the root) kept.
    Scores are seeded random log-probabilities (strictly decreasing along a
    path), so the kept set is ancestor-closed.  Nodes are ordered by (depth,
    score), so parent(n) < n.  Returns parent [B, N] (root -1) and each node's
    rank among its parent's candidates [B, N] (root 0)."""
    g = torch.Generator().manual_seed(int(seed))
    parents = torch.empty(B, N, dtype=torch.int32)
    ranks = torch.empty(B, N, dtype=torch.int32)
    for b in range(B):
        # candidate pool: (score, depth, parent_pool_index, rank)
        pool = [(0.0, 0, -1, 0)]
        frontier = [0]
        for dep in range(1, depth + 1):
            layer = []
            for pi in frontier:
                u = torch.rand(topk, generator=g).sort(descending=True).values
                sc = pool[pi][0]
                for k in range(topk):
                    sc_k = sc + math.log(max(float(u[k]), 1e-12)) - 1e-9 * (k + 1)
                    layer.append(len(pool))
                    pool.append((sc_k, dep, pi, k))
            layer.sort(key=lambda i: -pool[i][0])
            frontier = layer[:topk]
        if len(pool) < N:
            raise ValueError("depth %d and top-%d give %d candidates, fewer than N = %d"
                             % (depth, topk, len(pool), N))
        order = sorted(range(1, len(pool)), key=lambda i: -pool[i][0])[: N - 1]
        keep = [0] + sorted(order, key=lambda i: (pool[i][1], -pool[i][0]))
        pos = {pi: n for n, pi in enumerate(keep)}
        for n, pi in enumerate(keep):
            par = pool[pi][2]
            parents[b, n] = -1 if par < 0 else pos[par]
            ranks[b, n] = pool[pi][3]
    return parents, ranks


def tree_problem(B, N, depth, topk, V, device="cpu", seed=BASE_SEED, dtype="bf16"):
    """Tree verification workload: rows [B*N, V] (vocab32k recipe), parent [B, N],
    node tokens [B, N] (the rank-th largest draft logit of the parent's row, as a
    top-k expansion drafts them), uniforms [B, N]."""
    R = B * N
    d = logits_spiked(R, V, 3.0, min(50, V), 8.0, device, seed + 1)
    t = d + logits_gaussian(R, V, 1.0, device, seed + 2)
    draft, target = _cast(d, dtype).contiguous(), _cast(t, dtype).contiguous()
    parent, rank = tree_shapes(B, N, depth, topk, seed + 6)
    top = draft.float().topk(topk, dim=1).indices.to(torch.int32).cpu()  # [R, topk]
    rows = (torch.arange(B).view(B, 1) * N + parent.clamp(min=0).long()).view(-1)
    tokens = top[rows, rank.view(-1).long()].view(B, N)
    tokens[:, 0] = 0
    return dict(B=B, N=N, V=V, dtype=dtype, draft=draft, target=target,
                parent=parent.to(device), tokens=tokens.to(device),
                u_accept=uniforms(R, device, seed + 4).view(B, N),
                u_correct=uniforms(R, device, seed + 5).view(B, N))


def lmhead_problem(B, K, D, V, H, device="cpu", seed=BASE_SEED):
    """LM-head workload: hidden [R, H] ~N(0,1), weight [V, H] ~N(0, 0.02^2) (bf16),
    target logits [R, V] (vocab32k recipe, bf16), uniforms."""
    R = B * K * D
    hidden = torch.randn(R, H, generator=_gen(device, seed + 7), device=device).to(torch.bfloat16)
    weight = (torch.randn(V, H, generator=_gen(device, seed + 8), device=device) * 0.02).to(
        torch.bfloat16)
    t = logits_spiked(R, V, 3.0, min(50, V), 8.0, device, seed + 1) + logits_gaussian(
        R, V, 1.0, device, seed + 2)
    return dict(B=B, K=K, D=D, V=V, H=H, dtype="bf16", hidden=hidden.contiguous(),
                weight=weight.contiguous(), target=t.to(torch.bfloat16).contiguous(),
                u_draft=uniforms(R, device, seed + 3), u_accept=uniforms(R, device, seed + 4),
                u_correct=uniforms(R, device, seed + 5))


def lmhead_exact_problem(B, K, D, V, H, device="cpu", seed=BASE_SEED):
    """LM-head inputs whose products and partial sums are all exact in float32:
    hidden in {-2, ..., 2}, weight in {-64, ..., 64} / 256, so every product is
    a multiple of 2^-8 of magnitude at most 1/2 and every partial sum a
    multiple of 2^-8 below H/2: exact in float32 (24 bits) for H < 2^17.  Any
    summation order then gives the exact logits before the one rounding to
    bf16.  Target logits and uniforms as in lmhead_problem."""
    R = B * K * D
    g = _gen(device, seed + 9)
    hidden = torch.randint(-2, 3, (R, H), generator=g, device=device).to(torch.bfloat16)
    weight = (torch.randint(-64, 65, (V, H), generator=g, device=device).float() / 256.0).to(
        torch.bfloat16)
    t = logits_spiked(R, V, 3.0, min(50, V), 8.0, device, seed + 1) + logits_gaussian(
        R, V, 1.0, device, seed + 2)
    return dict(B=B, K=K, D=D, V=V, H=H, dtype="bf16", hidden=hidden.contiguous(),
                weight=weight.contiguous(), target=t.to(torch.bfloat16).contiguous(),
                u_draft=uniforms(R, device, seed + 3), u_accept=uniforms(R, device, seed + 4),
                u_correct=uniforms(R, device, seed + 5))
