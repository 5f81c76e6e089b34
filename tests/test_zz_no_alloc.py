"""The allocation-free entry point vsd_estep_mstep_noalloc.

It serves callers that cannot give the library device scratch memory (for
example a plugin that only receives input and output pointers, or a process
whose device memory is all owned by another allocator): the library uses its
own fixed array in device memory instead of a caller workspace.  The GPU test
calls it through the C ABI and checks that it gives the same results as
vsd_estep_mstep with a caller workspace, on consecutive calls with different
shapes, so that whatever one call leaves in the shared array cannot leak into
the next.  This file sorts last so that a run stopping at the first failure has
already run every other test.
"""
import ctypes as C

import pytest
import torch


@pytest.fixture(scope="module")
def vsd():
    from paper_2602_05774_gb300 import build, vsd as v
    build.build_library()
    v.load()
    return v


def test_rejects_layouts_beyond_the_scratch(vsd):
    """Host-side check, before any CUDA call: too large -> VSD_ERR_TOO_LARGE.
    Every pointer is NULL, so a call that got past the size check would be
    refused as an invalid argument before anything is launched."""
    lib = vsd.load()
    lay = vsd.layout(64, 64, 64, 1024)  # needs ~49 MB of scratch
    assert vsd.workspace_bytes(lay) > vsd.NOALLOC_SCRATCH_BYTES
    null = None
    outs = vsd.LinearOutputs(*([None] * len(vsd.LINEAR_FIELDS)))
    code = lib.vsd_estep_mstep_noalloc(null, null, 1, lay, 1.0, null, null, null, None, None,
                                       C.byref(outs), None)
    assert code == 7
    assert b"scratch" in lib.vsd_status_string(code)
    bad = vsd.layout(0, 1, 1, 8)
    assert lib.vsd_estep_mstep_noalloc(null, null, 1, bad, 1.0, null, null, null, None, None,
                                       C.byref(outs), None) == 1
    assert lib.vsd_noalloc_device_status(None, None) == 1


def _problem(kind):
    from paper_2602_05774_gb300 import inputs
    if kind == "vocab32k":
        p = inputs.config("vocab32k", device="cuda")
    else:
        p = inputs.linear_problem(3, 5, 4, 4097, "f32", "gauss", device="cuda", seed=404)
    return p


@pytest.mark.gpu
def test_noalloc_matches_workspace_entry_point(vsd):
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    for kind, T in (("vocab32k", 1.0), ("ragged", 0.7), ("vocab32k", 0.7)):
        p = _problem(kind)
        K, D = p["K"], p["D"]
        ref = vsd.estep_mstep(p["draft"], p["target"], p["u_draft"], p["u_accept"],
                              p["u_correct"], K, D, T)
        got = vsd.estep_mstep_noalloc(p["draft"], p["target"], p["u_draft"], p["u_accept"],
                                      p["u_correct"], K, D, T)
        torch.cuda.synchronize()
        assert ref.keys() == got.keys()
        for name in ref:
            # the same kernel on the same inputs is deterministic: equal bits
            assert torch.equal(ref[name], got[name]), (kind, T, name)
        assert torch.isfinite(got["loss"]).all()
        assert vsd.noalloc_device_status() == (0, 0)


@pytest.mark.gpu
def test_noalloc_status_word_reports_a_timeout(vsd):
    """The status word of the built-in array is readable: a call whose
    gradient waits are made to run out (the test hook, with a 2 ms bound)
    reports the timeout bit, and the next ordinary call reports none."""
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    p = _problem("ragged")
    K, D = p["K"], p["D"]
    prm = vsd.params(like=p["draft"], wait_timeout_ns=2_000_000, test_never_publish=1)
    vsd.estep_mstep_noalloc(p["draft"], p["target"], p["u_draft"], p["u_accept"],
                            p["u_correct"], K, D, 1.0, prm=prm)
    code, bits = vsd.noalloc_device_status()
    assert code == 4 and bits & vsd.STATUS_TIMEOUT
    vsd.estep_mstep_noalloc(p["draft"], p["target"], p["u_draft"], p["u_accept"],
                            p["u_correct"], K, D, 1.0)
    assert vsd.noalloc_device_status() == (0, 0)
