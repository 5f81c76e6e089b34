"""Mutation check of the oracle's pins.

Each case below plants one plausible mistake in a copy of oracle/vsd_oracle.c
(a tie rule, a sign, an index, a dropped term, a swapped operand), compiles
that copy, and runs every pin of tests/test_oracle_pins.py against it: at
least one pin must fail.  A mutation no pin notices would mean that part of
the oracle is checked only against itself.  CPU only; gcc builds each copy in
well under a second.
"""
import inspect
import itertools
import os
import subprocess

import pytest

from oracle import oracle as oracle_mod
from oracle.build import SRC
from tests import test_oracle_pins as pins

# (name, text in vsd_oracle.c, replacement); the text must occur exactly once.
MUTATIONS = [
    ("accept tie goes to reject",
     "double u = (double)in->u_accept[r];\n                uint8_t a = (u <= alpha)",
     "double u = (double)in->u_accept[r];\n                uint8_t a = (u < alpha)"),
    ("inverse CDF takes the boundary", "        if (u < F) {", "        if (u <= F) {"),
    ("residual direction reversed",
     "                    for (int64_t v = 0; v < V; ++v) {\n"
     "                        double dv = p[v] - q[v];",
     "                    for (int64_t v = 0; v < V; ++v) {\n"
     "                        double dv = q[v] - p[v];"),
    ("w(l) off by one", "pow(w_base, (double)l)", "pow(w_base, (double)(l - 1))"),
    ("beta not leave-one-out", "        if (j == s) continue;\n", ""),
    ("beta denominator counts proposals", "den += op[j];", "den += 1.0;"),
    ("zeta modes swapped", "(mode == 0 ? exp(logq_path[j]) : logq_path[j])",
     "(mode == 1 ? exp(logq_path[j]) : logq_path[j])"),
    ("zeta multiplies by tau", "logq_path[j]) / tau;", "logq_path[j]) * tau;"),
    ("control-variate sign", "J += op * (logq_z - beta * zeta * logq_zt);",
     "J += op * (logq_z + beta * zeta * logq_zt);"),
    ("gradient of the correction term", "double c_neg = op * beta * zeta /",
     "double c_neg = -op * beta * zeta /"),
    ("o' of a substitute path dropped",
     "op[s] = oracle_utility(logkappa_corr[s * D + d], lkr, l, w_base);", "op[s] = 0.0;"),
    ("o' of a kept proposal is binary", "                op[s] = o_tilde; /* z = z~, o' = o(z~) */",
     "                op[s] = 1.0;"),
    ("greedy reference ties to the highest index",
     "                for (int64_t v = 1; v < V; ++v) if (xp[v] > xp[vb]) vb = v;",
     "                for (int64_t v = 1; v < V; ++v) if (xp[v] >= xp[vb]) vb = v;"),
    ("supplied reference ties to the highest index",
     "            int64_t vb = 0;\n            for (int64_t v = 1; v < V; ++v) if (xp[v] > xp[vb])",
     "            int64_t vb = 0;\n            for (int64_t v = 1; v < V; ++v) if (xp[v] >= xp[vb])"),
    ("expected length skips S_1", "for (int d = 0; d < D; ++d) EA += exp(lk[s * D + d]);",
     "for (int d = 1; d < D; ++d) EA += exp(lk[s * D + d]);"),
    ("after the first rejection draws from q",
     "                } else {\n                    zc = sample_inverse_cdf(p, V, "
     "(double)in->u_correct[r], &mg);\n                }",
     "                } else {\n                    zc = sample_inverse_cdf(q, V, "
     "(double)in->u_correct[r], &mg);\n                }"),
    ("log kappa of z' uses z~'s alpha", "lkc[s * D + d] = prev + log(ac);",
     "lkc[s * D + d] = prev + log(out->alpha[r]);"),
    ("loss not normalised by N", "double lb = N > 0.0 ? -J / N : 0.0;",
     "double lb = N > 0.0 ? -J : 0.0;"),
    ("tree acceptance not an AND-scan",
     "out->path_accept[n0 + n] = (uint8_t)(a && out->path_accept[rp]);",
     "out->path_accept[n0 + n] = (uint8_t)a;"),
    ("tree residual direction reversed",
     "                for (int64_t v = 0; v < V; ++v) {\n"
     "                    double dv = p[v] - q[v];",
     "                for (int64_t v = 0; v < V; ++v) {\n"
     "                    double dv = q[v] - p[v];"),
    ("tree bonus ignores the residual", "if (par[n] == best) { bonus = out->corr_tokens[n0 + n]; break; }",
     "if (par[n] == best) { break; }"),
    ("top-K ties to the highest index", "if (best < 0 || xp[v] > xp[best]) best = v;",
     "if (best < 0 || xp[v] >= xp[best]) best = v;"),
    ("top-K gradient sign", "dl[k] = (exp(lqh) - ph) / T;", "dl[k] = (ph - exp(lqh)) / T;"),
    ("top-K term not averaged over proposals", "lb += in->kl_weight * kl / (double)K;",
     "lb += in->kl_weight * kl;"),
    ("top-K gradient scale", "in->kl_weight / ((double)B * K) * dl[k];",
     "in->kl_weight / (double)B * dl[k];"),
    ("greedy ties to the last maximum", "for (int64_t v = 1; v < V; ++v) if (x[v] > x[m]) m = v;",
     "for (int64_t v = 1; v < V; ++v) if (x[v] >= x[m]) m = v;"),
    ("greedy M-step at another temperature", "const double T = greedy ? 1.0 : in->T;",
     "const double T = greedy ? 0.5 : in->T;"),
    ("greedy decisions from the softmax", "    if (greedy) {\n        greedy_one_hot(xq, V, q);",
     "    if (0) {\n        greedy_one_hot(xq, V, q);"),
    ("supplied reference ratio inverted", "            double ab = p[vb] / q[vb];\n            if (ab > 1.0) ab = 1.0;\n            acc += log(ab);",
     "            double ab = q[vb] / p[vb];\n            if (ab > 1.0) ab = 1.0;\n            acc += log(ab);"),
    ("sequential rule keeps the residual target", "                if (Rm > 0.0)\n                    for (int64_t v = 0; v < V; ++v) p[v] = res[v] / Rm;\n                q[t] = 0.0;",
     "                q[t] = 0.0;"),
    ("sequential rule keeps rejected siblings in q", "                q[t] = 0.0;\n                double Qs = 0.0;",
     "                double Qs = 0.0;"),
    ("sequential rule tries children of rejected nodes", "            if (!out->path_accept[n0 + u]) continue;\n            int last = -1;",
     "            int last = -1;"),
    ("tree EM beta over all proposals", "                if (depth[n] == l) {\n                    grp[m] = n;",
     "                if (depth[n] >= 1) {\n                    grp[m] = n;"),
    ("tree EM z' below a rejection is the residual", "            } else { /* below a rejection: a draw from p */\n                zc = sample_inverse_cdf(p, V,",
     "            } else { /* below a rejection: a draw from p */\n                zc = sample_inverse_cdf(q, V,"),
    ("tree EM weight of the parent's depth", "            const double o_tilde = oracle_utility(lk, lkr, depth[n], in->w_base);",
     "            const double o_tilde = oracle_utility(lk, lkr, depth[n] - 1, in->w_base);"),
    ("margin: unequal sums given no margin", "if (a != b) return fabs(a - b);",
     "if (a != b) return 0.0;"),
    ("margin: a clipped tie given no margin", "        if (ra[i] < m) m = ra[i];\n", ""),
    ("margin: identical tokens not cancelled",
     "        if (rb && ta[i] == tb[i]) continue; /* identical terms cancel exactly */\n", ""),
]


def _pin_calls():
    """Every pin of test_oracle_pins as (name, zero-argument callable)."""
    calls = []
    for name, fn in inspect.getmembers(pins, inspect.isfunction):
        if not name.startswith("test_") or fn.__module__ != pins.__name__:
            continue
        marks = [m for m in getattr(fn, "pytestmark", []) if m.name == "parametrize"]
        grids = []
        for m in marks:
            names = [n.strip() for n in m.args[0].split(",")] if isinstance(m.args[0], str) \
                else list(m.args[0])
            vals = [v if len(names) > 1 else (v,) for v in m.args[1]]
            grids.append([dict(zip(names, v)) for v in vals])
        for combo in itertools.product(*grids) if grids else [()]:
            kw = {}
            for d in combo:
                kw.update(d)
            calls.append((name, lambda fn=fn, kw=kw: fn(oracle_mod, **kw)))
    return calls


def _build(text, path):
    with open(path + ".c", "w") as f:
        f.write(text)
    subprocess.run(["gcc", "-O1", "-std=c99", "-fPIC", "-shared", "-fno-fast-math",
                    "-ffp-contract=off", path + ".c", "-o", path, "-lm"], check=True)


def test_unmutated_copy_passes_every_pin(tmp_path, oracle):
    path = str(tmp_path / "orig.so")
    _build(open(SRC).read(), path)
    with oracle_mod.using_library(path):
        for name, call in _pin_calls():
            call()


@pytest.mark.parametrize("name,old,new", MUTATIONS, ids=[m[0] for m in MUTATIONS])
def test_each_mutation_fails_a_pin(tmp_path, oracle, name, old, new):
    src = open(SRC).read()
    assert src.count(old) == 1, "mutation anchor must occur once: %r" % old
    path = str(tmp_path / "mut.so")
    _build(src.replace(old, new), path)
    caught = []
    with oracle_mod.using_library(path):
        for pin, call in _pin_calls():
            try:
                call()
            except (AssertionError, ValueError, IndexError, OverflowError, ZeroDivisionError):
                caught.append(pin)
                break
    assert caught, "no pin fails with the mutation %r" % name
