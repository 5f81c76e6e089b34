"""The N-process path on CPU: two gloo ranks run the host logic the GPU runs
use (paper_2602_05774_gb300.multirank) with the oracle standing in for the
kernels.  Checks that the ranks draw different prefixes, that the job's time
is the slowest rank's, that the job rate counts every rank's rows, and that
sharding by prefix loses nothing: each rank's results equal the whole batch's
results for its prefixes (the method has no cross-prefix term; the gradient of
the mean loss differs only by the number of prefixes it averages over)."""
import multiprocessing as mp
import os
import socket

import numpy as np
import pytest

B_RANK, K, D, V, T = 2, 3, 2, 64, 0.9


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _run_oracle(prob):
    from oracle import oracle
    return oracle.linear(prob["draft"].numpy().astype(np.float64),
                         prob["target"].numpy().astype(np.float64), T,
                         prob["u_draft"].numpy(), prob["u_accept"].numpy(),
                         prob["u_correct"].numpy(), K, D)


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    try:
        import torch.distributed as dist
        from paper_2602_05774_gb300 import inputs, multirank
        r, w, _ = multirank.env()
        multirank.init(w, "gloo")
        seed = multirank.rank_seed(inputs.BASE_SEED, r)
        prob = inputs.linear_problem(B_RANK, K, D, V, "f32", "gauss", seed=seed)
        multirank.barrier(w)
        orc = _run_oracle(prob)
        fake_ms = 10.0 * (r + 1)  # rank r "took" 10 (r + 1) ms
        job_ms = multirank.max_over_ranks(fake_ms, w)
        rate = multirank.job_rate(B_RANK * K * D, w, job_ms)
        multirank.barrier(w)
        dist.destroy_process_group()
        q.put((r, dict(seed=seed, job_ms=job_ms, rate=rate,
                       loss=np.asarray(orc["loss"]), accept_len=np.asarray(orc["accept_len"]),
                       corr_tokens=np.asarray(orc["corr_tokens"]), grad=np.asarray(orc["grad"]))))
    except BaseException as e:  # report instead of hanging the parent
        q.put((rank, repr(e)))


def test_two_gloo_ranks_shard_by_prefix():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    got = {}
    try:
        for _ in range(world):
            r, res = q.get(timeout=240)
            got[r] = res
    finally:
        for p in procs:
            p.join(timeout=60)
            if p.is_alive():
                p.kill()
    for r in range(world):
        assert isinstance(got[r], dict), got[r]
    # different prefixes per rank; the job's time is the slowest rank's; the
    # rate counts every rank's rows
    assert got[0]["seed"] != got[1]["seed"]
    for r in range(world):
        assert got[r]["job_ms"] == 20.0
        assert got[r]["rate"] == pytest.approx(world * B_RANK * K * D / 0.020)
    # sharding loses nothing: the two ranks' prefixes as one batch give the
    # same per-prefix results
    import torch
    from paper_2602_05774_gb300 import inputs, multirank
    parts = [inputs.linear_problem(B_RANK, K, D, V, "f32", "gauss",
                                   seed=multirank.rank_seed(inputs.BASE_SEED, r))
             for r in range(world)]
    whole = dict(parts[0])
    for k in ("draft", "target", "u_draft", "u_accept", "u_correct"):
        whole[k] = torch.cat([p[k] for p in parts])
    whole["B"] = world * B_RANK
    orc = _run_oracle(whole)
    rows = B_RANK * K * D
    for r in range(world):
        assert np.array_equal(np.asarray(orc["loss"])[r * B_RANK:(r + 1) * B_RANK],
                              got[r]["loss"][:B_RANK])
        assert np.array_equal(np.asarray(orc["accept_len"])[r * B_RANK * K:(r + 1) * B_RANK * K],
                              got[r]["accept_len"])
        assert np.array_equal(np.asarray(orc["corr_tokens"])[r * rows:(r + 1) * rows],
                              got[r]["corr_tokens"])
        # the gradient is that of the mean loss over the prefixes a call sees:
        # per rank over B_RANK, in the whole batch over world * B_RANK (powers
        # of two, so the rescaling is exact)
        whole_rows = np.asarray(orc["grad"])[r * rows:(r + 1) * rows]
        assert np.array_equal(whole_rows * (world * B_RANK), got[r]["grad"] * B_RANK)
