"""CPU checks of the C ABI: the library builds, loads and exports every symbol
that include/vsd.h declares; host-side argument checks return the documented
codes before anything touches a GPU (no compute call is made here)."""
import ctypes as C
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def vsd():
    from paper_2602_05774_gb300 import build, vsd as v
    build.build_library()
    v.load()
    return v


def declared_symbols():
    src = open(os.path.join(ROOT, "include", "vsd.h")).read()
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[\w\s\*]+?\b(vsd_\w+)\s*\(", src, re.M)))


# Tests that pass fake device pointers rely on the host-side checks returning
# before anything is enqueued.  They run only where no GPU is present, so that
# a regression that let a call through could never launch a kernel on bogus
# addresses on a shared GPU.
def _no_gpu():
    try:
        import torch
        return not torch.cuda.is_available()
    except Exception:
        return True


host_only = pytest.mark.skipif(not _no_gpu(), reason="fake device pointers: host-only checks")


def test_header_symbols_exported(vsd):
    names = declared_symbols()
    assert len(names) >= 8, names
    lib = vsd.load()
    for n in names:
        assert hasattr(lib, n), "missing export %s" % n
    assert set(vsd.SYMBOLS) <= set(names)


def test_version_and_status_strings(vsd):
    lib = vsd.load()
    assert lib.vsd_version().decode().count(".") == 2
    for code in range(7):
        assert len(lib.vsd_status_string(code)) > 0
    assert lib.vsd_status_string(99) == b"unknown status"


def test_workspace_bytes(vsd):
    lay = vsd.layout(32, 16, 8, 128256)
    n = vsd.workspace_bytes(lay)
    R = 32 * 16 * 8
    # per row: records (~160 B) and the fused kernel's chunk table (16 B per
    # 512 logits)
    assert R * 64 < n < R * (400 + 16 * ((128256 + 511) // 512))
    small = vsd.workspace_bytes(vsd.layout(2, 4, 4, 1024))
    assert 0 < small < n
    lib = vsd.load()
    for bad in (vsd.layout(0, 1, 1, 8), vsd.layout(1, 0, 1, 8), vsd.layout(1, 1, 65, 8),
                vsd.layout(1, 257, 1, 8), vsd.layout(1, 1, 1, (1 << 20) + 1),
                vsd.layout(1, 1, 1, 0)):
        assert lib.vsd_workspace_bytes(bad) == 0


@host_only
def test_argument_checks_before_any_launch(vsd):
    lib = vsd.load()
    lay = vsd.layout(2, 4, 4, 1024)
    fake = C.c_void_p(0x1000)  # never dereferenced: every call below fails its checks
    big = 1 << 30
    outs = vsd.LinearOutputs()
    # null pointers
    assert lib.vsd_sample_paths(None, 0, lay, 1.0, fake, fake, fake, None, fake, big, None) == 1
    # temperature 0 is unsupported, negative / nan invalid
    assert lib.vsd_sample_paths(fake, 0, lay, 0.0, fake, fake, fake, None, fake, big, None) == 2
    assert lib.vsd_sample_paths(fake, 0, lay, -1.0, fake, fake, fake, None, fake, big, None) == 1
    assert lib.vsd_sample_paths(fake, 0, lay, float("nan"), fake, fake, fake, None, fake, big,
                                None) == 1
    # bad dtype
    assert lib.vsd_sample_paths(fake, 7, lay, 1.0, fake, fake, fake, None, fake, big, None) == 1
    # workspace too small / missing / misaligned
    assert lib.vsd_sample_paths(fake, 0, lay, 1.0, fake, fake, fake, None, fake, 16, None) == 5
    assert lib.vsd_sample_paths(fake, 0, lay, 1.0, fake, fake, fake, None, None, big, None) == 5
    assert lib.vsd_sample_paths(fake, 0, lay, 1.0, fake, fake, fake, None, C.c_void_p(0x1004),
                                big, None) == 5
    # fused: required outputs missing
    assert lib.vsd_estep_mstep(fake, fake, 1, lay, 1.0, fake, fake, fake, None, None,
                               C.byref(outs), fake, big, None) == 1
    # bad M-step parameters
    o = vsd.LinearOutputs(*([0x1000] * len(vsd.LINEAR_FIELDS)))
    for prm in (vsd.params(w_base=0.0), vsd.params(tau_car=0.0), vsd.params(zeta_mode=3),
                vsd.params(grad_dtype=5)):
        assert lib.vsd_estep_mstep(fake, fake, 1, lay, 1.0, fake, fake, fake, None, C.byref(prm),
                                   C.byref(o), fake, big, None) == 1
    # tree layout: reference log-kappa is not accepted, outputs required
    tlay = vsd.Layout(2, 1, 1, 1024, 60, 0x1000)
    to = vsd.TreeOutputs()
    assert lib.vsd_verify_paths(fake, fake, 1, tlay, 1.0, fake, fake, fake, None, None,
                                C.byref(to), fake, big, None) == 1
    # linear-only entry points reject a tree layout
    assert lib.vsd_sample_paths(fake, 1, tlay, 1.0, fake, fake, fake, None, fake, big, None) == 1


def test_binding_refuses_cpu_tensors(vsd):
    torch = pytest.importorskip("torch")
    x = torch.zeros(4, 8)
    u = torch.zeros(4)
    with pytest.raises(ValueError):
        vsd.sample_paths(x, u, 1, 4, 1.0)


@host_only
def test_lmhead_argument_checks_before_any_launch(vsd):
    lib = vsd.load()
    fake = C.c_void_p(0x1000)  # never dereferenced: every call below fails its checks
    ws = C.c_void_p(0x100000)
    # N and K must be multiples of 8, M >= 1, pointers 16-byte aligned
    assert lib.vsd_lmhead_logits(fake, fake, 128, 260, 64, fake, ws, 256, None) == 1
    assert lib.vsd_lmhead_logits(fake, fake, 128, 256, 60, fake, ws, 256, None) == 1
    assert lib.vsd_lmhead_logits(fake, fake, 0, 256, 64, fake, ws, 256, None) == 1
    assert lib.vsd_lmhead_logits(C.c_void_p(0x1008), fake, 128, 256, 64, fake, ws, 256,
                                 None) == 1
    assert lib.vsd_lmhead_logits(None, fake, 128, 256, 64, fake, ws, 256, None) == 1
    # workspace: present, 256 bytes, 256-byte aligned
    assert lib.vsd_lmhead_logits(fake, fake, 128, 256, 64, fake, None, 256, None) == 5
    assert lib.vsd_lmhead_logits(fake, fake, 128, 256, 64, fake, ws, 16, None) == 5
    # the fused variant: linear layouts only, H a multiple of 8
    lay = vsd.layout(2, 4, 4, 1024)
    o = vsd.LinearOutputs(*([0x1000] * len(vsd.LINEAR_FIELDS)))
    assert lib.vsd_lmhead_estep_mstep(fake, fake, 100, fake, lay, 1.0, fake, fake, fake, None,
                                      None, fake, C.byref(o), ws, 1 << 30, None) == 1
    tlay = vsd.Layout(2, 1, 1, 1024, 60, 0x1000)
    assert lib.vsd_lmhead_estep_mstep(fake, fake, 128, fake, tlay, 1.0, fake, fake, fake, None,
                                      None, fake, C.byref(o), ws, 1 << 30, None) == 1
    assert lib.vsd_lmhead_estep_mstep(fake, fake, 128, fake, lay, -1.0, fake, fake, fake, None,
                                      None, fake, C.byref(o), ws, 1 << 30, None) == 1


@host_only
def test_lmhead_backward_argument_checks_before_any_launch(vsd):
    lib = vsd.load()
    fake = C.c_void_p(0x1000)  # never dereferenced: every call below returns before a launch
    lay = vsd.layout(2, 4, 4, 1024)
    big = 1 << 30
    # H a multiple of 8, linear layouts only, outputs 16-byte aligned, T >= 0
    assert lib.vsd_lmhead_backward(fake, fake, 100, fake, lay, 1.0, None, fake, fake, fake, big,
                                   None) == 1
    tlay = vsd.Layout(2, 1, 1, 1024, 60, 0x1000)
    assert lib.vsd_lmhead_backward(fake, fake, 128, fake, tlay, 1.0, None, fake, fake, fake, big,
                                   None) == 1
    assert lib.vsd_lmhead_backward(fake, fake, 128, fake, lay, 1.0, None, C.c_void_p(0x1004),
                                   fake, fake, big, None) == 1
    assert lib.vsd_lmhead_backward(fake, fake, 128, fake, lay, -1.0, None, fake, fake, fake, big,
                                   None) == 1
    assert lib.vsd_lmhead_backward(None, fake, 128, fake, lay, 1.0, None, fake, fake, fake, big,
                                   None) == 1
    # the workspace of the preceding call's layout
    assert lib.vsd_lmhead_backward(fake, fake, 128, fake, lay, 1.0, None, fake, fake, fake, 256,
                                   None) == 5
    # nothing asked for: nothing launched
    assert lib.vsd_lmhead_backward(fake, fake, 128, fake, lay, 1.0, None, None, None, fake, big,
                                   None) == 0


@host_only
def test_kl_greedy_and_reference_argument_checks(vsd):
    lib = vsd.load()
    fake = C.c_void_p(0x1000)  # never dereferenced: every call below fails its checks
    big = 1 << 30
    lay = vsd.layout(2, 4, 4, 1024)
    o = vsd.LinearOutputs(*([0x1000] * len(vsd.LINEAR_FIELDS)))
    # the top-K term: a weight >= 0 and 1 <= K <= 16
    for prm in (vsd.params(kl_weight=-1.0), vsd.params(kl_weight=1.0, kl_topk=0),
                vsd.params(kl_weight=1.0, kl_topk=17), vsd.params(kl_weight=float("inf"))):
        assert lib.vsd_estep_mstep(fake, fake, 1, lay, 1.0, fake, fake, fake, None, C.byref(prm),
                                   C.byref(o), fake, big, None) == 1
    # the separate M-step does not serve it, nor T = 0
    prm = vsd.params(kl_weight=0.5)
    assert lib.vsd_weighted_loss_fwd_bwd(fake, 1, lay, 1.0, C.byref(o), C.byref(prm), fake,
                                         fake, None, fake, big, None) == 2
    assert lib.vsd_weighted_loss_fwd_bwd(fake, 1, lay, 0.0, C.byref(o), None, fake, fake, None,
                                         fake, big, None) == 2
    # the reference from supplied rows: pointers, temperature, workspace
    ref = lib.vsd_reference_logkappa
    assert ref(None, fake, 1, 2, 4, 1024, 1.0, fake, fake, big, None) == 1
    assert ref(fake, fake, 1, 2, 4, 1024, 1.0, None, fake, big, None) == 1
    assert ref(fake, fake, 1, 2, 4, 1024, -0.5, fake, fake, big, None) == 1
    assert ref(fake, fake, 1, 0, 4, 1024, 1.0, fake, fake, big, None) == 1
    assert ref(fake, fake, 1, 2, 65, 1024, 1.0, fake, fake, big, None) == 1
    assert ref(fake, fake, 1, 2, 4, 1024, 1.0, fake, None, big, None) == 5
    assert ref(fake, fake, 1, 2, 4, 1024, 1.0, fake, fake, 16, None) == 5
