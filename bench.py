"""Benchmark of the fused VSD E-step + M-step (one persistent kernel per step).

Workload (default): vocab128k -- B=32 prefixes x K=16 proposals x D=8 depth,
V=128256, bf16 draft/target logits (Zipf-shaped target, draft = target +
N(0, 1.5^2)), temperatures alternating 0.7 / 1.0 between steps, synthetic and
seeded.  Inputs (2.1 GB) are larger than L2, so no flush is needed between
steps.  One step = one call of vsd_estep_mstep over the whole batch.

Prints ONE JSON line (rank 0).  `--impl reference` times the CPU oracle (the
reference implementation of this tier) on a bounded sample of the same
workload instead.
"""
import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import threading
import time

# The oracle baseline is single-threaded: keep numpy's BLAS (the oracle's LM
# head) on one core so that "cores": 1 holds.
for _v in ("OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS", "BLIS_NUM_THREADS"):
    os.environ.setdefault(_v, "1")

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = ("draft-logit rows/s and achieved HBM GB/s (fraction of GB300 roofline) for fused "
          "E/M step")
WORKLOADS = ("vocab128k", "vocab32k", "tiny", "lmhead", "tree60", "lmhead_train")


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=("ours", "reference"))
    ap.add_argument("--config", default="vocab128k", choices=WORKLOADS)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--prefixes", type=int, default=0,
                    help="run only the first B prefixes of the workload (small profiling "
                         "captures); 0 = all")
    return ap.parse_args()


def dist_env():
    from paper_2602_05774_gb300 import multirank
    return multirank.env()


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        d = json.load(open(path))
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def tensor_peak():
    """Measured cuBLAS bf16 throughput (burst: the GEMM is timed on its own)."""
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        d = json.load(open(path))
        return float(d["bf16_tflops"]), "measured"
    except Exception:
        return 1900.0, "fallback"


def _code_only(text):
    """Source text without comments and with whitespace collapsed: the hash
    below follows the code, not its comments."""
    text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
    text = re.sub(r"//[^\n]*", " ", text)
    return " ".join(text.split())


def kernel_source_hash():
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2602_05774_gb300", "csrc")
    for f in sorted(os.listdir(csrc)):
        h.update(_code_only(open(os.path.join(csrc, f)).read()).encode())
    h.update(_code_only(open(os.path.join(ROOT, "include", "vsd.h")).read()).encode())
    return h.hexdigest()[:16]


def ncu_traffic(workload, kernel="k_fused"):
    """DRAM bytes per launch of the roofline's kernel (k_fused; k_lmhead_bwd:
    per backward call) from the committed ncu summary, if it was taken on the
    current kernel sources; else None."""
    path = os.path.join(ROOT, "profiles", "%s_%s_traffic.json" % (kernel, workload))
    try:
        d = json.load(open(path))
        if d.get("kernel_source_hash") == kernel_source_hash():
            return float(d["dram_bytes_per_launch"])
    except Exception:
        pass
    return None


class ClockSampler:
    """nvidia-smi clocks and throttle reasons, sampled while the timed loop runs."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.rows = []
        self.proc = None
        self.thread = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
            time.sleep(0.25)
        except Exception:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.rows.append([c.strip() for c in line.split(",")])

    def __exit__(self, *a):
        if self.proc is not None:
            time.sleep(0.15)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.thread.join(timeout=2)

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for r in self.rows:
            try:
                sm.append(float(r[0]))
                mx.append(float(r[1]))
                for n, v in zip(names, r[4:8]):
                    if v.lower() == "active":
                        reasons.add(n)
            except Exception:
                continue
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx),
                "reasons": sorted(reasons), "samples": len(sm)}


def algorithmic_bytes(R, V, elem, gelem):
    """Bytes the method itself must move per step: draft and target logits read
    once, the gradient written once, three uniforms per row read once."""
    return R * V * (2 * elem + gelem) + R * 12


def oracle_sample(prob, rows, T):
    from oracle import oracle
    K, D, V = prob["K"], prob["D"], prob["V"]
    sub = {k: prob[k][:rows].float().cpu().numpy() for k in
           ("draft", "target", "u_draft", "u_accept", "u_correct")}
    k_paths = rows // D
    t0 = time.perf_counter()
    oracle.linear(sub["draft"], sub["target"], T, sub["u_draft"], sub["u_accept"],
                  sub["u_correct"], min(K, k_paths), D)
    return time.perf_counter() - t0


# ---------------------------------------------------------------- CPU baseline
# The oracle as it stands, on the host's cores: one unit (a prefix of the
# workload, or a tree) per process.  Workers draw their unit's inputs with the
# same recipe and their own seed (so nothing large crosses a pipe) and time
# only the oracle call.
_KIND = {"vocab128k": "zipf", "vocab32k": "spiked", "tiny": "gauss"}


def _cpu_unit(task):
    """(workload, unit index, T) -> seconds of the oracle on that unit."""
    name, i, T = task
    from paper_2602_05774_gb300 import inputs
    from oracle import oracle
    c = inputs.CONFIGS["lmhead" if name == "lmhead_train" else name]
    seed = inputs.BASE_SEED + 5000 + i
    if name == "tree60":
        p = inputs.config("tree60", device="cpu", seed=seed, B=1)
        f = {k: p[k].float().numpy() if p[k].is_floating_point() else p[k].numpy()
             for k in ("draft", "target", "parent", "tokens", "u_accept", "u_correct")}
        t0 = time.perf_counter()
        oracle.tree(f["draft"], f["target"], T, f["parent"], f["tokens"], f["u_accept"],
                    f["u_correct"])
        return time.perf_counter() - t0
    if name in ("lmhead", "lmhead_train"):
        p = inputs.lmhead_problem(1, c["K"], c["D"], c["V"], c["H"], device="cpu", seed=seed)
        h = p["hidden"].float().numpy()
        w = p["weight"].float().numpy()
        f = {k: p[k].float().numpy() for k in ("target", "u_draft", "u_accept", "u_correct")}
        t0 = time.perf_counter()
        draft = oracle.round_bf16(oracle.lmhead_logits(h, w))
        o = oracle.linear(draft, f["target"], T, f["u_draft"], f["u_accept"], f["u_correct"],
                          c["K"], c["D"])
        if name == "lmhead_train":  # the head's backward of this prefix's gradient
            oracle.lmhead_backward(o["grad"], h, w)
        return time.perf_counter() - t0
    p = inputs.linear_problem(1, c["K"], c["D"], c["V"], c["dtype"], _KIND[name], device="cpu",
                              seed=seed)
    f = {k: p[k].float().numpy() for k in ("draft", "target", "u_draft", "u_accept", "u_correct")}
    t0 = time.perf_counter()
    oracle.linear(f["draft"], f["target"], T, f["u_draft"], f["u_accept"], f["u_correct"],
                  c["K"], c["D"])
    return time.perf_counter() - t0


def host_cores():
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


def cpu_baseline(name, T, rows_per_unit, unit, max_workers=None):
    """The oracle single-core (one unit per repetition) and on every host core
    (one unit per core at once; at most max_workers), each the median of three
    repetitions, in rows/s.  A spawned pool: the GPU context of this process
    is not forked."""
    import multiprocessing as mp
    cores = host_cores() if max_workers is None else min(host_cores(), max_workers)
    _cpu_unit((name, 0, T))  # builds the oracle and warms the import
    single = [rows_per_unit / _cpu_unit((name, k, T)) for k in range(3)]
    ctx = mp.get_context("spawn")
    multi = []
    with ctx.Pool(cores) as pool:
        pool.map(_cpu_unit, [(name, 100 + k, T) for k in range(cores)])  # warm the workers
        for rep in range(3):
            secs = pool.map(_cpu_unit, [(name, 200 + rep * cores + k, T) for k in range(cores)])
            multi.append(rows_per_unit * cores / max(secs))
    return {"value": statistics.median(multi), "unit": "rows/s", "cores": cores,
            "kind": "oracle",
            "sample": "%s: %d %s(s) of %d rows at once, one per core, median of 3 (inputs drawn "
                      "with the same recipe and other seeds)" % (name, cores, unit, rows_per_unit),
            "single_core": {"value": statistics.median(single), "unit": "rows/s", "cores": 1,
                            "sample": "one %s of %d rows, median of 3" % (unit, rows_per_unit)},
            "nproc": os.cpu_count()}


def parity_sample(out, prob, B, K, D, T, prefixes):
    """The GPU's results on the first prefixes of the timed batch against the
    oracle on the same inputs: discrete decisions must agree except within
    the oracle's margins (counted), per-prefix losses within 1e-5."""
    import numpy as np
    from oracle import oracle
    P = K * D
    rows = prefixes * P
    sub = {k: prob[k][:rows].float().cpu().numpy() for k in
           ("draft", "target", "u_draft", "u_accept", "u_correct")}
    orc = oracle.linear(sub["draft"], sub["target"], T, sub["u_draft"], sub["u_accept"],
                        sub["u_correct"], K, D, want_grad=False)
    m = orc["margins"]
    near = int((np.minimum(np.minimum(m[:, 0], m[:, 1]), m[:, 2]) < 1e-6).sum()
               + (np.minimum(m[:, 3], m[:, 4]) < 1e-5).sum())
    res = {"prefixes": prefixes, "rows": rows, "near_boundary_decisions": near,
           "decision_mismatches": 0, "mismatches_outside_margin": 0, "max_loss_rel_err": 0.0}
    for name, col in (("tokens", 0), ("accept", 1), ("corr_tokens", 2)):
        g = out[name][:rows].cpu().numpy()
        bad = np.nonzero(g != orc[name])[0]
        res["decision_mismatches"] += int(bad.size)
        res["mismatches_outside_margin"] += int((m[bad, col] >= 1e-6).sum()) if name != "corr_tokens" else 0
    lg = out["loss"][:prefixes].cpu().double().numpy()
    rel = np.abs(lg - orc["loss"][:prefixes]) / np.maximum(1.0, np.abs(orc["loss"][:prefixes]))
    res["max_loss_rel_err"] = float(rel.max())
    return res


def run_reference(args):
    """The oracle, as it stands, on the host cores: each step a bounded sample
    (the first paths of one prefix) of the same workload."""
    rank, world, _ = dist_env()
    if rank != 0:
        return
    import torch
    from paper_2602_05774_gb300 import inputs
    from oracle.build import build_oracle
    build_oracle()
    c = inputs.CONFIGS[args.config]
    K, D, V = c["K"], c["D"], c["V"]
    # bounded sample: one path (D rows) of prefix 0 per step, on the CPU generator
    small = inputs.linear_problem(1, K, D, V, c["dtype"], {"vocab128k": "zipf",
                                  "vocab32k": "spiked", "tiny": "gauss"}[args.config],
                                  device="cpu", seed=inputs.BASE_SEED + 99)
    temps = c["T"]
    paths = 1
    rows = paths * D
    for i in range(args.warmup):
        oracle_sample(small, rows, temps[i % len(temps)])
    t = 0.0
    for i in range(args.steps):
        t += oracle_sample(small, rows, temps[i % len(temps)])
    ms = t / args.steps * 1e3
    val = rows / (ms / 1e3)
    line = {
        "impl": "reference", "metric": METRIC, "value": val, "unit": "rows/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded; same recipe)",
        "config": {"workload": args.config, "B": c["B"], "K": K, "D": D, "V": V,
                   "logits": c["dtype"], "temperatures": list(temps),
                   "sample_per_step": "%d path(s) x %d rows of one prefix" % (paths, D)},
        "cpu_baseline": {"value": val, "unit": "rows/s", "cores": 1, "kind": "oracle",
                         "sample": "%d rows per step (one path of one prefix)" % rows},
        "e2e": {"value": val, "unit": "rows/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def run_ours(args):
    import torch
    rank, world, local = dist_env()
    from paper_2602_05774_gb300 import multirank
    multirank.init(world, "nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_2602_05774_gb300 import build, inputs, vsd
    build.build_library()
    vsd.load()
    c = inputs.CONFIGS[args.config]
    seed = multirank.rank_seed(inputs.BASE_SEED + list(inputs.CONFIGS).index(args.config), rank)
    prob = inputs.config(args.config, device=dev, seed=seed, B=args.prefixes or None)
    torch.cuda.empty_cache()
    B, K, D, V = prob["B"], prob["K"], prob["D"], prob["V"]
    R = B * K * D
    temps = c["T"]
    elem = prob["draft"].element_size()
    prm = vsd.params(like=prob["draft"])
    gelem = 2 if prm.grad_dtype == vsd.VSD_BF16 else 4
    lay = vsd.layout(B, K, D, V)
    ws = vsd.new_workspace(lay, dev)
    gdt = torch.bfloat16 if gelem == 2 else torch.float32
    out = vsd.linear_outputs(B, K, D, V, dev, grad_dtype=gdt, full=True)

    def step(i):
        vsd.estep_mstep(prob["draft"], prob["target"], prob["u_draft"], prob["u_accept"],
                        prob["u_correct"], K, D, temps[i % len(temps)], prm=prm, workspace=ws,
                        out=out)

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize(dev)
    code, bits = vsd.device_status(ws)
    if code != 0:
        raise RuntimeError("device status %d (bits %d) after warm-up" % (code, bits))

    def barrier():
        multirank.barrier(world, dev)

    stream = torch.cuda.current_stream(dev)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    barrier()
    with ClockSampler(local) as clk:
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record(stream)
        for i in range(args.steps):
            ev[i][0].record(stream)
            step(i)
            ev[i][1].record(stream)
        t1.record(stream)
        barrier()
    total_ms = t0.elapsed_time(t1)
    launch_ms = statistics.mean(a.elapsed_time(b) for a, b in ev)
    total_ms = multirank.max_over_ranks(total_ms, world, dev)
    ms = total_ms / args.steps
    code, bits = vsd.device_status(ws)
    if code != 0:
        raise RuntimeError("device status %d (bits %d) after timing" % (code, bits))

    # end-to-end through the public API from pinned host buffers
    e2e = None
    if not args.no_e2e:
        hs = vsd.HostStep(B, K, D, V, prob["draft"].dtype, dev, prm=prm)
        h_draft = prob["draft"].cpu().pin_memory()
        h_target = prob["target"].cpu().pin_memory()
        h_u = torch.stack([prob["u_draft"], prob["u_accept"], prob["u_correct"]]).cpu().pin_memory()
        e_steps = max(3, min(args.steps, 30))
        for i in range(2):
            hs(h_draft, h_target, h_u, temps[i % len(temps)])
        barrier()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for i in range(e_steps):
            loss = hs(h_draft, h_target, h_u, temps[i % len(temps)])
        b.record(stream)
        barrier()
        e_ms = a.elapsed_time(b) / e_steps
        e_ms = multirank.max_over_ranks(e_ms, world, dev)
        e2e = {"value": multirank.job_rate(R, world, e_ms), "unit": "rows/s",
               "h2d_bytes_per_step": hs.h2d_bytes(), "d2h_bytes_per_step": hs.d2h_bytes(),
               "ms_per_step": e_ms, "steps": e_steps,
               "inputs": "double-buffered: a step's copies overlap the previous step's kernels"}
        torch.cuda.synchronize(dev)
        assert torch.isfinite(loss).all()
        del hs, h_draft, h_target, h_u

    if rank != 0:
        return
    peak, peak_kind = peaks()
    alg = algorithmic_bytes(R, V, elem, gelem)
    achieved = alg / (launch_ms / 1e3) / 1e9
    traffic = ncu_traffic(args.config)
    value = multirank.job_rate(R, world, ms)
    line = {
        "metric": METRIC, "value": value, "unit": "rows/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16" if elem == 2 else "f32",
        "data": "synthetic (seeded; Zipf target, noisy draft)",
        "config": {"workload": args.config, "B": B, "K": K, "D": D, "V": V,
                   "logits": "bf16" if elem == 2 else "f32",
                   "grad": "bf16" if gelem == 2 else "f32", "temperatures": list(temps),
                   "l2": "inputs larger than L2 (no flush)" if alg > 200e6 else "L2-resident",
                   "rows_per_gpu": R},
        "achieved_gbs": achieved,
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": traffic, "peak_kind": peak_kind,
                     "kernel": "k_fused", "algorithmic_bytes_per_launch": alg,
                     "launch_ms": launch_ms},
        "gpu_launches": args.steps,
        "clocks": clk.summary(),
    }
    if e2e is not None:
        line["e2e"] = e2e
    if world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(args.config, temps[-1], K * D, "prefix")
        # the GPU's results on two prefixes of the timed batch against the oracle
        step(len(temps) - 1)
        torch.cuda.synchronize(dev)
        line["parity_sample"] = parity_sample(out, prob, B, K, D, temps[-1], min(2, B))
    print(json.dumps(line), flush=True)



def oracle_lmhead_sample(prob, rows, T, train=False):
    """The oracle's LM head (fp64 matmul, one bf16 rounding) and E/M step on the
    first `rows` rows (train: and the head's backward of their gradient):
    seconds."""
    from oracle import oracle
    K, D = prob["K"], prob["D"]
    h = prob["hidden"][:rows].float().cpu().numpy()
    w = prob["weight"].float().cpu().numpy()
    sub = {k: prob[k][:rows].float().cpu().numpy() for k in
           ("target", "u_draft", "u_accept", "u_correct")}
    t0 = time.perf_counter()
    draft = oracle.round_bf16(oracle.lmhead_logits(h, w))
    o = oracle.linear(draft, sub["target"], T, sub["u_draft"], sub["u_accept"], sub["u_correct"],
                      min(K, rows // D), D)
    if train:
        oracle.lmhead_backward(o["grad"], h, w)
    return time.perf_counter() - t0


def run_reference_lmhead(args, train=False):
    """The oracle on the host cores for the LM-head workload: each step the LM
    head and E/M step of one path (D rows) of one prefix (train: and the
    head's backward)."""
    rank, world, _ = dist_env()
    if rank != 0:
        return
    from paper_2602_05774_gb300 import inputs
    from oracle.build import build_oracle
    build_oracle()
    c = inputs.CONFIGS["lmhead"]
    K, D, V, H = c["K"], c["D"], c["V"], c["H"]
    small = inputs.lmhead_problem(1, K, D, V, H, device="cpu", seed=inputs.BASE_SEED + 99)
    rows = D
    for i in range(args.warmup):
        oracle_lmhead_sample(small, rows, 1.0, train)
    t = sum(oracle_lmhead_sample(small, rows, 1.0, train) for _ in range(args.steps))
    ms = t / args.steps * 1e3
    val = rows / (ms / 1e3)
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": val, "unit": "rows/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded; same recipe)",
        "config": {"workload": "lmhead_train" if train else "lmhead", "B": c["B"], "K": K,
                   "D": D, "V": V, "H": H,
                   "sample_per_step": "1 path x %d rows of one prefix" % D},
        "cpu_baseline": {"value": val, "unit": "rows/s", "cores": 1, "kind": "oracle",
                         "sample": "%d rows per step (one path of one prefix)" % rows},
        "e2e": {"value": val, "unit": "rows/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }), flush=True)


def run_lmhead(args, train=False):
    """Config 5: the LM head on the tensor cores fused with the E/M step.  The
    step is vsd_lmhead_estep_mstep; the roofline is the GEMM's (tensor), timed
    on its own with CUDA events per launch.  train: the draft head's training
    step, vsd_lmhead_estep_mstep with no dense gradient, then
    vsd_lmhead_backward (d_hidden and d_weight from the factored gradient);
    the roofline is the backward's (tensor), timed per call."""
    import torch
    rank, world, local = dist_env()
    from paper_2602_05774_gb300 import multirank
    multirank.init(world, "nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_2602_05774_gb300 import build, inputs, vsd
    build.build_library()
    vsd.load()
    seed = multirank.rank_seed(inputs.BASE_SEED + list(inputs.CONFIGS).index("lmhead"), rank)
    prob = inputs.config("lmhead", device=dev, seed=seed, B=args.prefixes or None)
    B, K, D, V, H = prob["B"], prob["K"], prob["D"], prob["V"], prob["H"]
    R = B * K * D
    T = 1.0
    prm = vsd.params(like=prob["target"])
    ws = vsd.new_workspace(vsd.layout(B, K, D, V), dev)
    out = vsd.linear_outputs(B, K, D, V, dev, grad_dtype=torch.bfloat16, full=True,
                             grad=not train)
    dl = torch.empty(R, V, dtype=torch.bfloat16, device=dev)
    if train:
        d_hidden = torch.empty(R, H, dtype=torch.float32, device=dev)
        d_weight = torch.empty(V, H, dtype=torch.float32, device=dev)

    def backward(i):
        vsd.lmhead_backward(prob["hidden"], prob["weight"], dl, K, D, T, ws, prm=prm,
                            d_hidden=d_hidden, d_weight=d_weight)

    def step(i):
        vsd.lmhead_estep_mstep(prob["hidden"], prob["weight"], prob["target"], prob["u_draft"],
                               prob["u_accept"], prob["u_correct"], K, D, T, prm=prm,
                               workspace=ws, out=out, draft_logits=dl)
        if train:
            backward(i)

    def barrier():
        multirank.barrier(world, dev)

    def timed(fn, n):
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(n)]
        stream = torch.cuda.current_stream(dev)
        barrier()
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record(stream)
        for i in range(n):
            ev[i][0].record(stream)
            fn(i)
            ev[i][1].record(stream)
        t1.record(stream)
        barrier()
        return t0.elapsed_time(t1), statistics.mean(a.elapsed_time(b) for a, b in ev)

    for i in range(args.warmup):
        step(i)
    barrier()
    if vsd.device_status(ws)[0] != 0:
        raise RuntimeError("device status after warm-up: %s" % (vsd.device_status(ws),))
    with ClockSampler(local) as clk:
        total_ms, _ = timed(step, args.steps)
        gws = torch.zeros(256, dtype=torch.uint8, device=dev)
        if train:  # the backward alone, per call (the roofline's kernels)
            _, gemm_ms = timed(backward, args.steps)
        else:  # the GEMM alone, per launch (the roofline's kernel)
            for _ in range(3):
                vsd.lmhead_logits(prob["hidden"], prob["weight"], out=dl, workspace=gws)
            _, gemm_ms = timed(lambda i: vsd.lmhead_logits(prob["hidden"], prob["weight"],
                                                           out=dl, workspace=gws), args.steps)
    total_ms = multirank.max_over_ranks(total_ms, world, dev)
    ms = total_ms / args.steps
    if vsd.device_status(ws)[0] != 0 or vsd.device_status(gws)[0] != 0:
        raise RuntimeError("device status after timing")

    e2e = None
    if not args.no_e2e:  # the same step from pinned host buffers, loss read back
        h_hidden = prob["hidden"].cpu().pin_memory()
        h_target = prob["target"].cpu().pin_memory()
        h_u = torch.stack([prob["u_draft"], prob["u_accept"], prob["u_correct"]]).cpu().pin_memory()
        hs = vsd.HostLMHeadStep(prob["weight"], B, K, D, V, prm=prm, train=train)
        losses = []

        def e2e_step(i):
            losses.append(hs(h_hidden, h_target, h_u, T))

        e_steps = max(3, min(args.steps, 20))
        for i in range(2):
            e2e_step(i)
        e_total, _ = timed(e2e_step, e_steps)
        e_ms = multirank.max_over_ranks(e_total / e_steps, world, dev)
        e2e = {"value": multirank.job_rate(R, world, e_ms), "unit": "rows/s",
               "h2d_bytes_per_step": hs.h2d_bytes(), "d2h_bytes_per_step": hs.d2h_bytes(),
               "ms_per_step": e_ms, "steps": e_steps, "weights": "resident on the device",
               "inputs": "double-buffered: a step's copies overlap the previous step's kernels"}
        assert torch.isfinite(losses[-1]).all()
        del hs
    if rank != 0:
        return
    peak, peak_kind = tensor_peak()
    flops = (4.0 if train else 2.0) * R * V * H
    achieved = flops / (gemm_ms / 1e3) / 1e12
    line = {
        "metric": METRIC, "value": multirank.job_rate(R, world, ms), "unit": "rows/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded; hidden ~N(0,1), LM-head weight ~N(0,0.02^2), spiked target)",
        "config": {"workload": "lmhead_train" if train else "lmhead", "B": B, "K": K, "D": D,
                   "V": V, "H": H, "logits": "bf16",
                   "grad": "factored: made on chip by the backward, never in HBM" if train
                   else "bf16", "temperatures": [T],
                   "l2": "inputs larger than L2 (no flush)", "rows_per_gpu": R},
        "roofline": {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                     "frac": achieved / peak,
                     "traffic": ncu_traffic("lmhead_train", "k_lmhead_bwd") if train else None,
                     "peak_kind": peak_kind,
                     "kernel": "k_lmhead_bwd (d_hidden + d_weight)" if train else "k_lmhead",
                     "flops_per_launch": flops, "launch_ms": gemm_ms},
        # per step: GEMM, fused E/M (+ row factors, d_hidden, d_weight)
        "gpu_launches": (5 if train else 2) * args.steps,
        "clocks": clk.summary(),
    }
    if e2e is not None:
        line["e2e"] = e2e
    if world == 1 and not args.no_cpu_baseline:
        if train:  # the fp64 V x H product of each unit: four workers at most
            line["cpu_baseline"] = cpu_baseline(
                "lmhead_train", T, K * D,
                "prefix (LM head in fp64 + E/M step + the head's backward)", max_workers=4)
        else:
            line["cpu_baseline"] = cpu_baseline("lmhead", T, K * D,
                                                "prefix (LM head in fp64 + E/M step)")
    print(json.dumps(line), flush=True)


def oracle_tree_sample(prob, trees, T):
    """The oracle's tree verification of the first `trees` trees: seconds."""
    from oracle import oracle
    N = prob["parent"].shape[1]
    rows = trees * N
    t0 = time.perf_counter()
    oracle.tree(prob["draft"][:rows].float().cpu().numpy(),
                prob["target"][:rows].float().cpu().numpy(), T,
                prob["parent"][:trees].cpu().numpy(), prob["tokens"][:trees].cpu().numpy(),
                prob["u_accept"][:trees].cpu().numpy(), prob["u_correct"][:trees].cpu().numpy())
    return time.perf_counter() - t0


def run_reference_tree(args):
    """The oracle on the host cores for the tree workload: one tree per step."""
    rank, world, _ = dist_env()
    if rank != 0:
        return
    from paper_2602_05774_gb300 import inputs
    from oracle.build import build_oracle
    build_oracle()
    c = inputs.CONFIGS["tree60"]
    small = inputs.config("tree60", device="cpu", seed=inputs.BASE_SEED + 99, B=1)
    N = small["parent"].shape[1]
    for _ in range(args.warmup):
        oracle_tree_sample(small, 1, 1.0)
    t = sum(oracle_tree_sample(small, 1, 1.0) for _ in range(args.steps))
    ms = t / args.steps * 1e3
    val = N / (ms / 1e3)
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": val, "unit": "rows/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded; same recipe)",
        "config": {"workload": "tree60", "B": c["B"], "N": N, "V": c["V"],
                   "sample_per_step": "1 tree of %d nodes" % N},
        "cpu_baseline": {"value": val, "unit": "rows/s", "cores": 1, "kind": "oracle",
                         "sample": "one tree (%d rows) per step" % N},
        "e2e": {"value": val, "unit": "rows/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }), flush=True)


def run_tree(args):
    """Config 4: verification of B draft trees (vsd_verify_paths with a tree
    layout); HBM roofline on the two logit reads."""
    import torch
    rank, world, local = dist_env()
    from paper_2602_05774_gb300 import multirank
    multirank.init(world, "nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_2602_05774_gb300 import build, inputs, vsd
    build.build_library()
    vsd.load()
    seed = multirank.rank_seed(inputs.BASE_SEED + list(inputs.CONFIGS).index("tree60"), rank)
    prob = inputs.config("tree60", device=dev, seed=seed, B=args.prefixes or None)
    B, N = prob["parent"].shape
    V = prob["draft"].shape[-1]
    R = B * N
    T = 1.0
    ws = vsd.new_workspace(vsd.layout(B, V=V, N=N, parent=prob["parent"]), dev)
    # the verification outputs; no per-row statistics, so leaf rows are read
    # only where a bonus token needs one
    tout = vsd.tree_outputs(B, N, dev, row_stats=False)

    def step(i):
        return vsd.verify_tree(prob["draft"], prob["target"], prob["parent"], prob["tokens"],
                               prob["u_accept"], prob["u_correct"], T, workspace=ws, out=tout)

    def barrier():
        multirank.barrier(world, dev)

    for i in range(args.warmup):
        step(i)
    barrier()
    if vsd.device_status(ws)[0] != 0:
        raise RuntimeError("device status after warm-up: %s" % (vsd.device_status(ws),))
    stream = torch.cuda.current_stream(dev)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    with ClockSampler(local) as clk:
        barrier()
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record(stream)
        for i in range(args.steps):
            ev[i][0].record(stream)
            step(i)
            ev[i][1].record(stream)
        t1.record(stream)
        barrier()
    total_ms = t0.elapsed_time(t1)
    launch_ms = statistics.mean(a.elapsed_time(b) for a, b in ev)
    total_ms = multirank.max_over_ranks(total_ms, world, dev)
    ms = total_ms / args.steps
    if vsd.device_status(ws)[0] != 0:
        raise RuntimeError("device status after timing")
    e2e = None
    if not args.no_e2e:  # inputs from pinned host buffers, accepted lengths read back
        names = ("draft", "target", "parent", "tokens", "u_accept", "u_correct")
        host = {k: prob[k].cpu().pin_memory() for k in names}
        hs = vsd.HostTreeStep(B, N, V, prob["draft"].dtype, dev)

        def e2e_step(i):
            hs(host, T)

        e_steps = max(3, min(args.steps, 20))
        for i in range(2):
            e2e_step(i)
        barrier()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for i in range(e_steps):
            e2e_step(i)
        b.record(stream)
        barrier()
        e_ms = multirank.max_over_ranks(a.elapsed_time(b) / e_steps, world, dev)
        e2e = {"value": multirank.job_rate(R, world, e_ms), "unit": "rows/s",
               "h2d_bytes_per_step": hs.h2d_bytes(), "d2h_bytes_per_step": hs.d2h_bytes(),
               "ms_per_step": e_ms, "steps": e_steps,
               "inputs": "double-buffered: a step's copies overlap the previous step's kernels"}
        del hs
    if rank != 0:
        return
    peak, peak_kind = peaks()
    elem = prob["draft"].element_size()
    # rows the outputs need: both logit rows of every node with children, and
    # of the deepest accepted node when it is a leaf (its bonus token)
    par = prob["parent"].cpu()
    has_kids = torch.zeros(B, N, dtype=torch.bool)
    for b in range(B):
        kids = par[b, 1:]
        has_kids[b, kids[kids >= 0].long()] = True
    deepest = tout["deepest"].cpu()
    leaf_bonus = sum(1 for b in range(B)
                     if deepest[b] >= 0 and not bool(has_kids[b, int(deepest[b])]))
    rows_read = int(has_kids.sum()) + leaf_bonus
    alg = 2 * rows_read * V * elem + R * 16  # those rows once; token, parent, two uniforms
    achieved = alg / (launch_ms / 1e3) / 1e9
    line = {
        "metric": METRIC, "value": multirank.job_rate(R, world, ms), "unit": "rows/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16" if elem == 2 else "f32",
        "data": "synthetic (seeded; EAGLE-2-style trees, spiked logits)",
        "config": {"workload": "tree60", "B": B, "N": N, "V": V, "logits": "bf16",
                   "temperatures": [T], "l2": "inputs larger than L2 (no flush)",
                   "rows_per_gpu": R, "row_stats": "not requested",
                   "rows_read": rows_read},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": None, "peak_kind": peak_kind,
                     "kernel": "k_tree_fused",
                     "algorithmic_bytes_per_launch": alg, "launch_ms": launch_ms},
        "gpu_launches": args.steps,
        "clocks": clk.summary(),
    }
    if e2e is not None:
        line["e2e"] = e2e
    if world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline("tree60", T, N, "tree")
    print(json.dumps(line), flush=True)

def main():
    args = parse()
    if args.config in ("lmhead", "lmhead_train"):
        train = args.config == "lmhead_train"
        if args.impl == "reference":
            run_reference_lmhead(args, train)
        else:
            run_lmhead(args, train)
    elif args.config == "tree60":
        run_reference_tree(args) if args.impl == "reference" else run_tree(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
