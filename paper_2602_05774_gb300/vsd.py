"""Python binding of libvsd (include/vsd.h): argument marshalling only.

Every step of the E-step / M-step runs in the library's CUDA kernels; this
module checks tensor shapes and dtypes, allocates output tensors when the
caller gives none, passes raw device pointers and the current CUDA stream, and
turns status codes into exceptions.  PyTorch provides device memory and
streams.  There is no CPU fallback: if libvsd.so is missing or fails to load,
every call raises.
"""
import ctypes as C
import os

import torch

from . import build as _build

VSD_F32, VSD_BF16 = 0, 1
STATUS_BAD_ROW, STATUS_TIMEOUT, STATUS_BAD_TREE, STATUS_BAD_TOKEN = 1, 2, 4, 8
_STATUS_NAMES = {0: "VSD_OK", 1: "VSD_ERR_INVALID_ARG", 2: "VSD_ERR_UNSUPPORTED",
                 3: "VSD_ERR_CUDA", 4: "VSD_ERR_TIMEOUT", 5: "VSD_ERR_WORKSPACE",
                 6: "VSD_ERR_DEVICE_DATA", 7: "VSD_ERR_TOO_LARGE"}

SYMBOLS = ("vsd_workspace_bytes", "vsd_sample_paths", "vsd_verify_paths",
           "vsd_weighted_loss_fwd_bwd", "vsd_estep_mstep", "vsd_device_status",
           "vsd_status_string", "vsd_version", "vsd_estep_mstep_noalloc",
           "vsd_noalloc_device_status", "vsd_lmhead_logits", "vsd_lmhead_estep_mstep",
           "vsd_reference_logkappa", "vsd_tree_estep_mstep", "vsd_lmhead_backward")
NOALLOC_SCRATCH_BYTES = 32 << 20


class VsdError(RuntimeError):
    def __init__(self, code, where):
        self.code = code
        msg = _lib().vsd_status_string(code).decode() if _LIB is not None else "?"
        super().__init__("%s: %s (%s)" % (where, _STATUS_NAMES.get(code, code), msg))


class Layout(C.Structure):
    _fields_ = [("B", C.c_int32), ("K", C.c_int32), ("D", C.c_int32), ("V", C.c_int32),
                ("N", C.c_int32), ("parent", C.c_void_p), ("tree_rule", C.c_int32)]


TREE_INDEPENDENT, TREE_SEQUENTIAL = 0, 1


class Params(C.Structure):
    _fields_ = [("w_base", C.c_double), ("tau_car", C.c_double), ("zeta_mode", C.c_int32),
                ("grad_dtype", C.c_int32), ("wait_timeout_ns", C.c_uint64),
                ("test_never_publish", C.c_int32), ("kl_weight", C.c_double),
                ("kl_topk", C.c_int32)]


LINEAR_FIELDS = ("tokens", "logq_tok", "alpha", "accept", "accept_len", "corr_tokens",
                 "logq_corr", "alpha_corr", "logkappa", "logkappa_corr", "logkappa_ref",
                 "ref_tokens", "expected_len", "row_stats", "weights", "loss", "grad",
                 "kl_loss")
TREE_FIELDS = ("alpha", "accept", "path_accept", "logkappa", "corr_tokens", "deepest",
               "accept_len", "bonus", "row_stats")
TREE_EM_FIELDS = ("corr_tokens", "logq_tok", "logq_corr", "logkappa", "logkappa_corr",
                  "logkappa_ref", "weights", "loss", "grad")


class LinearOutputs(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in LINEAR_FIELDS]


class TreeOutputs(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in TREE_FIELDS]


class TreeEmOutputs(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in TREE_EM_FIELDS]


_LIB = None


def library_path():
    return _build.LIB


def _lib():
    global _LIB
    if _LIB is None:
        path = library_path()
        if not os.path.exists(path):
            raise RuntimeError("libvsd.so is not built (%s); run __graft_entry__.build()" % path)
        lib = C.CDLL(path)
        vp = C.c_void_p
        lib.vsd_workspace_bytes.argtypes = [Layout]
        lib.vsd_workspace_bytes.restype = C.c_size_t
        lib.vsd_sample_paths.argtypes = [vp, C.c_int, Layout, C.c_float, vp, vp, vp, vp, vp,
                                         C.c_size_t, vp]
        lib.vsd_verify_paths.argtypes = [vp, vp, C.c_int, Layout, C.c_float, vp, vp, vp, vp,
                                         C.POINTER(LinearOutputs), C.POINTER(TreeOutputs), vp,
                                         C.c_size_t, vp]
        lib.vsd_weighted_loss_fwd_bwd.argtypes = [vp, C.c_int, Layout, C.c_float,
                                                  C.POINTER(LinearOutputs), C.POINTER(Params),
                                                  vp, vp, vp, vp, C.c_size_t, vp]
        lib.vsd_estep_mstep.argtypes = [vp, vp, C.c_int, Layout, C.c_float, vp, vp, vp, vp,
                                        C.POINTER(Params), C.POINTER(LinearOutputs), vp,
                                        C.c_size_t, vp]
        lib.vsd_estep_mstep_noalloc.argtypes = [vp, vp, C.c_int, Layout, C.c_float, vp, vp, vp,
                                                vp, C.POINTER(Params), C.POINTER(LinearOutputs),
                                                vp]
        lib.vsd_lmhead_logits.argtypes = [vp, vp, C.c_int32, C.c_int32, C.c_int32, vp, vp,
                                          C.c_size_t, vp]
        lib.vsd_lmhead_estep_mstep.argtypes = [vp, vp, C.c_int32, vp, Layout, C.c_float, vp, vp,
                                               vp, vp, C.POINTER(Params), vp,
                                               C.POINTER(LinearOutputs), vp, C.c_size_t, vp]
        lib.vsd_lmhead_backward.argtypes = [vp, vp, C.c_int32, vp, Layout, C.c_float,
                                            C.POINTER(Params), vp, vp, vp, C.c_size_t, vp]
        lib.vsd_device_status.argtypes = [vp, vp, C.POINTER(C.c_int32)]
        lib.vsd_noalloc_device_status.argtypes = [vp, C.POINTER(C.c_int32)]
        lib.vsd_reference_logkappa.argtypes = [vp, vp, C.c_int, C.c_int32, C.c_int32, C.c_int32,
                                               C.c_float, vp, vp, C.c_size_t, vp]
        lib.vsd_tree_estep_mstep.argtypes = [vp, vp, C.c_int, Layout, C.c_float, vp, vp, vp,
                                             C.POINTER(Params), C.POINTER(TreeEmOutputs), vp,
                                             C.c_size_t, vp]
        lib.vsd_status_string.argtypes = [C.c_int]
        lib.vsd_status_string.restype = C.c_char_p
        lib.vsd_version.restype = C.c_char_p
        for name in ("vsd_sample_paths", "vsd_verify_paths", "vsd_weighted_loss_fwd_bwd",
                     "vsd_estep_mstep", "vsd_device_status", "vsd_estep_mstep_noalloc",
                     "vsd_noalloc_device_status", "vsd_reference_logkappa",
                     "vsd_tree_estep_mstep",
                     "vsd_lmhead_logits", "vsd_lmhead_estep_mstep", "vsd_lmhead_backward"):
            getattr(lib, name).restype = C.c_int
        _LIB = lib
    return _LIB


def load():
    """Load libvsd.so (raises if it is missing); returns the ctypes handle."""
    return _lib()


def _check(code, where):
    if code != 0:
        raise VsdError(code, where)


def _dtype_code(t):
    if t.dtype == torch.float32:
        return VSD_F32
    if t.dtype == torch.bfloat16:
        return VSD_BF16
    raise TypeError("logits must be float32 or bfloat16, got %s" % t.dtype)


def _ptr(t):
    return None if t is None else C.c_void_p(t.data_ptr())


def _stream(device):
    return C.c_void_p(torch.cuda.current_stream(device).cuda_stream)


def _need_cuda(*ts):
    for t in ts:
        if t is not None:
            if not t.is_cuda:
                raise ValueError("tensors must live on a CUDA device")
            if not t.is_contiguous():
                raise ValueError("tensors must be contiguous")


def layout(B, K=1, D=1, V=1, N=0, parent=None, tree_rule=TREE_INDEPENDENT):
    return Layout(int(B), int(K), int(D), int(V), int(N),
                  None if parent is None else parent.data_ptr(), int(tree_rule))


def workspace_bytes(lay):
    n = _lib().vsd_workspace_bytes(lay)
    if n == 0:
        raise ValueError("invalid layout")
    return n


def new_workspace(lay, device):
    return torch.empty(workspace_bytes(lay), dtype=torch.uint8, device=device)


def params(w_base=1.05, tau_car=0.2, zeta_mode=0, grad_dtype=None, wait_timeout_ns=0,
           test_never_publish=0, like=None, kl_weight=0.0, kl_topk=10):
    if grad_dtype is None:
        grad_dtype = VSD_BF16 if (like is not None and like.dtype == torch.bfloat16) else VSD_F32
    elif isinstance(grad_dtype, torch.dtype):
        grad_dtype = VSD_BF16 if grad_dtype == torch.bfloat16 else VSD_F32
    return Params(float(w_base), float(tau_car), int(zeta_mode), int(grad_dtype),
                  int(wait_timeout_ns), int(test_never_publish), float(kl_weight), int(kl_topk))


def _ws(ws, lay, device):
    if ws is None:
        ws = new_workspace(lay, device)
    elif ws.numel() < workspace_bytes(lay):
        raise ValueError("workspace too small")
    return ws


def _rows(x, V):
    if x.numel() % V:
        raise ValueError("logit tensor size is not a multiple of V")
    return x.numel() // V


def linear_outputs(B, K, D, V, device, grad_dtype=torch.bfloat16, grad=True, full=True, kl=False):
    """Allocate the output tensors of the linear E-step / M-step (kl: the
    per-row top-K terms of VSD (KL) too)."""
    R = B * K * D
    f = dict(device=device)
    o = dict(tokens=torch.empty(R, dtype=torch.int32, **f),
             accept_len=torch.empty(B * K, dtype=torch.int32, **f),
             corr_tokens=torch.empty(R, dtype=torch.int32, **f),
             logkappa=torch.empty(R, dtype=torch.float32, **f),
             loss=torch.empty(B + 1, dtype=torch.float32, **f))
    if full:
        o.update(logq_tok=torch.empty(R, dtype=torch.float32, **f),
                 alpha=torch.empty(R, dtype=torch.float32, **f),
                 accept=torch.empty(R, dtype=torch.uint8, **f),
                 logq_corr=torch.empty(R, dtype=torch.float32, **f),
                 alpha_corr=torch.empty(R, dtype=torch.float32, **f),
                 logkappa_corr=torch.empty(R, dtype=torch.float32, **f),
                 logkappa_ref=torch.empty(R, dtype=torch.float32, **f),
                 ref_tokens=torch.empty(R, dtype=torch.int32, **f),
                 expected_len=torch.empty(B * K, dtype=torch.float32, **f),
                 row_stats=torch.empty(R, 4, dtype=torch.float32, **f),
                 weights=torch.empty(B, D, K, 4, dtype=torch.float32, **f))
    if kl:
        o["kl_loss"] = torch.empty(R, dtype=torch.float32, **f)
    if grad:
        o["grad"] = torch.empty(R, V, dtype=grad_dtype, **f)
    return o


def _linear_struct(o):
    return LinearOutputs(*[(o[n].data_ptr() if o.get(n) is not None else None)
                           for n in LINEAR_FIELDS])


def sample_paths(draft, u_draft, K, D, T, workspace=None):
    """z~ ~ q for every row (Algorithm 1): tokens, log q(z~), row statistics."""
    _need_cuda(draft, u_draft)
    V = draft.shape[-1]
    R = _rows(draft, V)
    B = R // (K * D)
    lay = layout(B, K, D, V)
    dev = draft.device
    ws = _ws(workspace, lay, dev)
    out = dict(tokens=torch.empty(R, dtype=torch.int32, device=dev),
               logq_tok=torch.empty(R, dtype=torch.float32, device=dev),
               row_stats=torch.empty(R, 4, dtype=torch.float32, device=dev))
    _check(_lib().vsd_sample_paths(_ptr(draft), _dtype_code(draft), lay, float(T), _ptr(u_draft),
                                   _ptr(out["tokens"]), _ptr(out["logq_tok"]),
                                   _ptr(out["row_stats"]), _ptr(ws), ws.numel(), _stream(dev)),
           "vsd_sample_paths")
    return out


def verify_paths(draft, target, tokens, u_accept, u_correct, K, D, T, ref_logkappa=None,
                 workspace=None):
    """Eq. 1 per token, accepted lengths, residual correction, log-kappas."""
    _need_cuda(draft, target, tokens, u_accept, u_correct, ref_logkappa)
    V = draft.shape[-1]
    R = _rows(draft, V)
    B = R // (K * D)
    lay = layout(B, K, D, V)
    dev = draft.device
    ws = _ws(workspace, lay, dev)
    o = linear_outputs(B, K, D, V, dev, grad=False)
    del o["loss"], o["weights"]
    o["tokens"] = torch.empty(R, dtype=torch.int32, device=dev)
    st = _linear_struct(o)
    _check(_lib().vsd_verify_paths(_ptr(draft), _ptr(target), _dtype_code(draft), lay, float(T),
                                   _ptr(tokens), _ptr(u_accept), _ptr(u_correct),
                                   _ptr(ref_logkappa), C.byref(st), None, _ptr(ws), ws.numel(),
                                   _stream(dev)), "vsd_verify_paths")
    return o


def tree_outputs(B, N, device, row_stats=True):
    """Output tensors of verify_tree, to pass as out= and reuse across calls.
    Without row_stats the kernel reads no leaf row but the one a bonus token
    may need."""
    f = dict(device=device)
    o = dict(alpha=torch.empty(B, N, dtype=torch.float32, **f),
             accept=torch.empty(B, N, dtype=torch.uint8, **f),
             path_accept=torch.empty(B, N, dtype=torch.uint8, **f),
             logkappa=torch.empty(B, N, dtype=torch.float32, **f),
             corr_tokens=torch.empty(B, N, dtype=torch.int32, **f),
             deepest=torch.empty(B, dtype=torch.int32, **f),
             accept_len=torch.empty(B, dtype=torch.int32, **f),
             bonus=torch.empty(B, dtype=torch.int32, **f))
    if row_stats:
        o["row_stats"] = torch.empty(B * N, 4, dtype=torch.float32, **f)
    return o


def verify_tree(draft, target, parent, tokens, u_accept, u_correct, T, workspace=None, out=None,
                rule=TREE_INDEPENDENT):
    """Tree verification (App. E tree, Eq. 1 per node, Sec. 3 residual); rule
    TREE_SEQUENTIAL tries siblings in turn (lossless multi-draft)."""
    _need_cuda(draft, target, parent, tokens, u_accept, u_correct)
    V = draft.shape[-1]
    B, N = parent.shape
    lay = layout(B, V=V, N=N, parent=parent, tree_rule=rule)
    dev = draft.device
    ws = _ws(workspace, lay, dev)
    o = out if out is not None else tree_outputs(B, N, dev)
    st = TreeOutputs(*[o[n].data_ptr() if o.get(n) is not None else None for n in TREE_FIELDS])
    _check(_lib().vsd_verify_paths(_ptr(draft), _ptr(target), _dtype_code(draft), lay, float(T),
                                   _ptr(tokens), _ptr(u_accept), _ptr(u_correct), None, None,
                                   C.byref(st), _ptr(ws), ws.numel(), _stream(dev)),
           "vsd_verify_paths(tree)")
    return o


def tree_estep_mstep(draft, target, parent, tokens, u_accept, u_correct, T, prm=None,
                     workspace=None, full=True):
    """The E-step + M-step over draft trees, every node a latent proposal
    (vsd_tree_estep_mstep).  Returns the outputs by name."""
    _need_cuda(draft, target, parent, tokens, u_accept, u_correct)
    V = draft.shape[-1]
    B, N = parent.shape
    lay = layout(B, V=V, N=N, parent=parent)
    dev = draft.device
    ws = _ws(workspace, lay, dev)
    prm = prm or params(like=draft)
    gdt = torch.bfloat16 if prm.grad_dtype == VSD_BF16 else torch.float32
    f = dict(device=dev)
    o = dict(loss=torch.empty(B + 1, dtype=torch.float32, **f),
             grad=torch.empty(B * N, V, dtype=gdt, **f))
    if full:
        o.update(corr_tokens=torch.empty(B, N, dtype=torch.int32, **f),
                 logq_tok=torch.empty(B, N, dtype=torch.float32, **f),
                 logq_corr=torch.empty(B, N, dtype=torch.float32, **f),
                 logkappa=torch.empty(B, N, dtype=torch.float32, **f),
                 logkappa_corr=torch.empty(B, N, dtype=torch.float32, **f),
                 logkappa_ref=torch.empty(B, N, dtype=torch.float32, **f),
                 weights=torch.empty(B, N, 4, dtype=torch.float32, **f))
    st = TreeEmOutputs(*[o[n].data_ptr() if o.get(n) is not None else None
                         for n in TREE_EM_FIELDS])
    _check(_lib().vsd_tree_estep_mstep(_ptr(draft), _ptr(target), _dtype_code(draft), lay,
                                       float(T), _ptr(tokens), _ptr(u_accept), _ptr(u_correct),
                                       C.byref(prm), C.byref(st), _ptr(ws), ws.numel(),
                                       _stream(dev)), "vsd_tree_estep_mstep")
    return o


def weighted_loss_fwd_bwd(draft, estep, K, D, T, prm=None, workspace=None, grad=None,
                          weights=True):
    """M-step: o~, o', beta, zeta, loss and gradient from E-step results."""
    _need_cuda(draft)
    V = draft.shape[-1]
    R = _rows(draft, V)
    B = R // (K * D)
    lay = layout(B, K, D, V)
    dev = draft.device
    ws = _ws(workspace, lay, dev)
    prm = prm or params(like=draft)
    if grad is None:
        grad = torch.empty(R, V, dtype=torch.bfloat16 if prm.grad_dtype == VSD_BF16
                           else torch.float32, device=dev)
    loss = torch.empty(B + 1, dtype=torch.float32, device=dev)
    w = torch.empty(B, D, K, 4, dtype=torch.float32, device=dev) if weights else None
    st = _linear_struct(estep)
    _check(_lib().vsd_weighted_loss_fwd_bwd(_ptr(draft), _dtype_code(draft), lay, float(T),
                                            C.byref(st), C.byref(prm), _ptr(loss), _ptr(grad),
                                            _ptr(w), _ptr(ws), ws.numel(), _stream(dev)),
           "vsd_weighted_loss_fwd_bwd")
    return dict(loss=loss, grad=grad, weights=w)


def estep_mstep(draft, target, u_draft, u_accept, u_correct, K, D, T, ref_logkappa=None,
                prm=None, workspace=None, out=None, full=True, grad=True):
    """The fused E-step + M-step (one persistent kernel).  Returns the outputs
    (grad=False: no dense gradient, for lmhead_backward on the same workspace)."""
    _need_cuda(draft, target, u_draft, u_accept, u_correct, ref_logkappa)
    V = draft.shape[-1]
    R = _rows(draft, V)
    B = R // (K * D)
    lay = layout(B, K, D, V)
    dev = draft.device
    ws = _ws(workspace, lay, dev)
    prm = prm or params(like=draft)
    if out is None:
        gdt = torch.bfloat16 if prm.grad_dtype == VSD_BF16 else torch.float32
        out = linear_outputs(B, K, D, V, dev, grad_dtype=gdt, grad=grad, full=full,
                             kl=prm.kl_weight != 0)
    st = _linear_struct(out)
    _check(_lib().vsd_estep_mstep(_ptr(draft), _ptr(target), _dtype_code(draft), lay, float(T),
                                  _ptr(u_draft), _ptr(u_accept), _ptr(u_correct),
                                  _ptr(ref_logkappa), C.byref(prm), C.byref(st), _ptr(ws),
                                  ws.numel(), _stream(dev)), "vsd_estep_mstep")
    return out


def reference_logkappa(ref_draft, ref_target, B, D, T, workspace=None):
    """log kappa of supplied greedy reference paths (Algorithm 2's z-bar with
    its own rows [B*D, V]): [B, D] float32, to pass as ref_logkappa."""
    _need_cuda(ref_draft, ref_target)
    V = ref_draft.shape[-1]
    if _rows(ref_draft, V) != B * D or ref_target.shape != ref_draft.shape:
        raise ValueError("reference rows must be [B*D, V] for both tensors")
    lay = layout(B, 1, D, V)
    dev = ref_draft.device
    ws = _ws(workspace, lay, dev)
    out = torch.empty(B, D, dtype=torch.float32, device=dev)
    _check(_lib().vsd_reference_logkappa(_ptr(ref_draft), _ptr(ref_target),
                                         _dtype_code(ref_draft), int(B), int(D), int(V), float(T),
                                         _ptr(out), _ptr(ws), ws.numel(), _stream(dev)),
           "vsd_reference_logkappa")
    return out


def lmhead_logits(hidden, weight, out=None, workspace=None):
    """Draft logits [M][N] = hidden [M][K] . weight [N][K]^T on the tensor cores
    (bf16 in, fp32 accumulation, bf16 out)."""
    _need_cuda(hidden, weight)
    if hidden.dtype != torch.bfloat16 or weight.dtype != torch.bfloat16:
        raise ValueError("the LM head takes bf16 hidden states and weights")
    M, K = hidden.shape
    N = weight.shape[0]
    if weight.shape[1] != K:
        raise ValueError("hidden and weight disagree on the hidden size")
    dev = hidden.device
    if out is None:
        out = torch.empty(M, N, dtype=torch.bfloat16, device=dev)
    ws = workspace if workspace is not None else torch.empty(256, dtype=torch.uint8, device=dev)
    _check(_lib().vsd_lmhead_logits(_ptr(hidden), _ptr(weight), M, N, K, _ptr(out), _ptr(ws),
                                    ws.numel(), _stream(dev)), "vsd_lmhead_logits")
    return out


def lmhead_estep_mstep(hidden, weight, target, u_draft, u_accept, u_correct, K, D, T,
                       ref_logkappa=None, prm=None, workspace=None, out=None, draft_logits=None,
                       full=True, grad=True):
    """The LM head, then the fused E-step + M-step on its logits.  Returns the
    outputs of estep_mstep() plus "draft_logits"."""
    _need_cuda(hidden, weight, target, u_draft, u_accept, u_correct, ref_logkappa)
    V = weight.shape[0]
    H = hidden.shape[-1]
    R = hidden.numel() // H
    B = R // (K * D)
    lay = layout(B, K, D, V)
    dev = hidden.device
    ws = _ws(workspace, lay, dev)
    prm = prm or params(like=target)
    if draft_logits is None:
        draft_logits = torch.empty(R, V, dtype=torch.bfloat16, device=dev)
    if out is None:
        gdt = torch.bfloat16 if prm.grad_dtype == VSD_BF16 else torch.float32
        out = linear_outputs(B, K, D, V, dev, grad_dtype=gdt, grad=grad, full=full,
                             kl=prm.kl_weight != 0)
    st = _linear_struct(out)
    _check(_lib().vsd_lmhead_estep_mstep(_ptr(hidden), _ptr(weight), H, _ptr(target), lay,
                                         float(T), _ptr(u_draft), _ptr(u_accept),
                                         _ptr(u_correct), _ptr(ref_logkappa), C.byref(prm),
                                         _ptr(draft_logits), C.byref(st), _ptr(ws), ws.numel(),
                                         _stream(dev)), "vsd_lmhead_estep_mstep")
    out["draft_logits"] = draft_logits
    return out


def lmhead_backward(hidden, weight, draft_logits, K, D, T, workspace, prm=None,
                    d_hidden=True, d_weight=True):
    """The draft LM head's backward after lmhead_estep_mstep() (or estep_mstep()
    on bf16 draft logits) on the same workspace: returns {"d_hidden": [R][H],
    "d_weight": [V][H]} (float32), the M-step gradient of the draft logits
    carried through logits = hidden . weight^T.  Pass False to skip one, or a
    float32 tensor to write into."""
    _need_cuda(hidden, weight, draft_logits)
    V, H = weight.shape
    R = hidden.numel() // H
    lay = layout(R // (K * D), K, D, V)
    dev = hidden.device
    prm = prm or params(like=draft_logits)
    res = {}
    for name, shape, want in (("d_hidden", (R, H), d_hidden), ("d_weight", (V, H), d_weight)):
        if want is True:
            res[name] = torch.empty(*shape, dtype=torch.float32, device=dev)
        elif want is not False and want is not None:
            res[name] = want
    _check(_lib().vsd_lmhead_backward(_ptr(hidden), _ptr(weight), H, _ptr(draft_logits), lay,
                                      float(T), C.byref(prm), _ptr(res.get("d_hidden")),
                                      _ptr(res.get("d_weight")), _ptr(workspace),
                                      workspace.numel(), _stream(dev)), "vsd_lmhead_backward")
    return res


def estep_mstep_noalloc(draft, target, u_draft, u_accept, u_correct, K, D, T,
                        ref_logkappa=None, prm=None, out=None, full=True):
    """The fused E-step + M-step without a workspace argument, for callers that
    cannot allocate device scratch: the library uses its own fixed array in
    device memory (limit: layouts whose workspace fits NOALLOC_SCRATCH_BYTES).
    Calls on one device share that array, so they must not overlap on the GPU.
    Outputs are allocated here when `out` is None, as in estep_mstep()."""
    _need_cuda(draft, target, u_draft, u_accept, u_correct, ref_logkappa)
    V = draft.shape[-1]
    R = _rows(draft, V)
    B = R // (K * D)
    lay = layout(B, K, D, V)
    dev = draft.device
    prm = prm or params(like=draft)
    if out is None:
        gdt = torch.bfloat16 if prm.grad_dtype == VSD_BF16 else torch.float32
        out = linear_outputs(B, K, D, V, dev, grad_dtype=gdt, full=full, kl=prm.kl_weight != 0)
    st = _linear_struct(out)
    _check(_lib().vsd_estep_mstep_noalloc(_ptr(draft), _ptr(target), _dtype_code(draft), lay,
                                          float(T), _ptr(u_draft), _ptr(u_accept),
                                          _ptr(u_correct), _ptr(ref_logkappa), C.byref(prm),
                                          C.byref(st), _stream(dev)), "vsd_estep_mstep_noalloc")
    return out


def noalloc_device_status(device=None):
    """(status code, status bits) of the vsd_estep_mstep_noalloc calls on the
    current device; synchronises the current stream."""
    bits = C.c_int32(0)
    dev = torch.device("cuda", torch.cuda.current_device()) if device is None else device
    code = _lib().vsd_noalloc_device_status(_stream(dev), C.byref(bits))
    return code, bits.value


def device_status(workspace):
    """(status code, status bits) of the last call on this workspace; synchronises."""
    bits = C.c_int32(0)
    code = _lib().vsd_device_status(_ptr(workspace), _stream(workspace.device), C.byref(bits))
    return code, bits.value


class _Feeder:
    """Two device copies of a step's inputs.  Each step queues the
    host-to-device copies of its inputs on a copy stream, into the copy the
    step before last used (after that step's kernels were queued), and the
    caller's stream waits for them; so the copies of one step run while the
    kernels of the step before it do."""

    def __init__(self, shapes, device):
        self.dev = torch.device(device)
        self.stream = torch.cuda.Stream(device=self.dev)
        self.bufs = []
        for _ in range(2):
            b = {k: torch.empty(sh, dtype=dt, device=self.dev) for k, (sh, dt) in shapes.items()}
            for t in b.values():
                t.record_stream(self.stream)
            self.bufs.append(b)
        self.copied = [torch.cuda.Event() for _ in range(2)]
        self.released = [None, None]
        self.n = 0

    def nbytes(self):
        return sum(t.numel() * t.element_size() for t in self.bufs[0].values())

    def feed(self, host):
        """Queue the copies of host (pinned tensors by name); returns the slot
        and its device tensors, ready on the caller's stream."""
        s = self.n % 2
        self.n += 1
        with torch.cuda.stream(self.stream):
            if self.released[s] is not None:
                self.stream.wait_event(self.released[s])
            for k, h in host.items():
                self.bufs[s][k].copy_(h, non_blocking=True)
            self.copied[s].record(self.stream)
        torch.cuda.current_stream(self.dev).wait_event(self.copied[s])
        return s, self.bufs[s]

    def release(self, s):
        """The kernels reading slot s have been queued on the caller's stream."""
        ev = torch.cuda.Event()
        ev.record(torch.cuda.current_stream(self.dev))
        self.released[s] = ev


class HostStep:
    """End-to-end E-step + M-step from pinned host tensors: each call copies
    its inputs to the device (double-buffered, overlapping the previous call's
    kernel), runs the fused kernel and queues the read-back of the loss.  The
    returned pinned loss tensor is valid after a synchronise and until the
    call after next."""

    def __init__(self, B, K, D, V, dtype, device, prm=None, full=False):
        self.B, self.K, self.D, self.V = B, K, D, V
        R = B * K * D
        self.dev = torch.device(device)
        self.feed = _Feeder(dict(draft=((R, V), dtype), target=((R, V), dtype),
                                 u=((3, R), torch.float32)), self.dev)
        self.prm = prm or params(like=self.feed.bufs[0]["draft"])
        gdt = torch.bfloat16 if self.prm.grad_dtype == VSD_BF16 else torch.float32
        self.out = linear_outputs(B, K, D, V, self.dev, grad_dtype=gdt, full=full)
        self.ws = new_workspace(layout(B, K, D, V), self.dev)
        self.loss_host = [torch.empty(B + 1, dtype=torch.float32).pin_memory() for _ in range(2)]

    def h2d_bytes(self):
        return self.feed.nbytes()

    def d2h_bytes(self):
        return self.loss_host[0].numel() * 4

    def __call__(self, h_draft, h_target, h_u, T):
        s, d = self.feed.feed(dict(draft=h_draft, target=h_target, u=h_u))
        estep_mstep(d["draft"], d["target"], d["u"][0], d["u"][1], d["u"][2], self.K, self.D, T,
                    prm=self.prm, workspace=self.ws, out=self.out)
        self.feed.release(s)
        self.loss_host[s].copy_(self.out["loss"], non_blocking=True)
        return self.loss_host[s]


class HostLMHeadStep:
    """HostStep for the LM head fused with the E-step + M-step: per call the
    hidden states, target logits and uniforms come from pinned host tensors
    (double-buffered); the LM-head weight stays on the device.  train=True:
    the draft head's training step, no dense gradient and the LM head's
    backward (d_hidden, d_weight left on the device)."""

    def __init__(self, weight, B, K, D, V, prm=None, full=True, train=False):
        self.B, self.K, self.D, self.V = B, K, D, V
        R, H = B * K * D, weight.shape[1]
        self.dev = weight.device
        self.weight = weight
        self.feed = _Feeder(dict(hidden=((R, H), torch.bfloat16), target=((R, V), torch.bfloat16),
                                 u=((3, R), torch.float32)), self.dev)
        self.prm = prm or params(grad_dtype=torch.bfloat16)
        gdt = torch.bfloat16 if self.prm.grad_dtype == VSD_BF16 else torch.float32
        self.train = train
        self.out = linear_outputs(B, K, D, V, self.dev, grad_dtype=gdt, full=full, grad=not train)
        self.ws = new_workspace(layout(B, K, D, V), self.dev)
        self.logits = torch.empty(R, V, dtype=torch.bfloat16, device=self.dev)
        if train:
            self.d_hidden = torch.empty(R, H, dtype=torch.float32, device=self.dev)
            self.d_weight = torch.empty(V, H, dtype=torch.float32, device=self.dev)
        self.loss_host = [torch.empty(B + 1, dtype=torch.float32).pin_memory() for _ in range(2)]

    def h2d_bytes(self):
        return self.feed.nbytes()

    def d2h_bytes(self):
        return self.loss_host[0].numel() * 4

    def __call__(self, h_hidden, h_target, h_u, T):
        s, d = self.feed.feed(dict(hidden=h_hidden, target=h_target, u=h_u))
        lmhead_estep_mstep(d["hidden"], self.weight, d["target"], d["u"][0], d["u"][1],
                           d["u"][2], self.K, self.D, T, prm=self.prm, workspace=self.ws,
                           out=self.out, draft_logits=self.logits)
        if self.train:
            lmhead_backward(d["hidden"], self.weight, self.logits, self.K, self.D, T, self.ws,
                            prm=self.prm, d_hidden=self.d_hidden, d_weight=self.d_weight)
        self.feed.release(s)
        self.loss_host[s].copy_(self.out["loss"], non_blocking=True)
        return self.loss_host[s]


class HostTreeStep:
    """HostStep for tree verification: per call the logits, the tree and the
    uniforms come from pinned host tensors (double-buffered); the accepted
    lengths are read back."""

    def __init__(self, B, N, V, dtype, device):
        self.B, self.N, self.V = B, N, V
        self.dev = torch.device(device)
        i32, f32 = torch.int32, torch.float32
        self.feed = _Feeder(dict(draft=((B * N, V), dtype), target=((B * N, V), dtype),
                                 parent=((B, N), i32), tokens=((B, N), i32),
                                 u_accept=((B, N), f32), u_correct=((B, N), f32)), self.dev)
        self.ws = new_workspace(layout(B, V=V, N=N, parent=self.feed.bufs[0]["parent"]), self.dev)
        self.out = tree_outputs(B, N, self.dev, row_stats=False)
        self.len_host = [torch.empty(B, dtype=i32).pin_memory() for _ in range(2)]

    def h2d_bytes(self):
        return self.feed.nbytes()

    def d2h_bytes(self):
        return self.len_host[0].numel() * 4

    def __call__(self, host, T):
        """host: pinned tensors draft, target, parent, tokens, u_accept, u_correct."""
        s, d = self.feed.feed(host)
        verify_tree(d["draft"], d["target"], d["parent"], d["tokens"], d["u_accept"],
                    d["u_correct"], T, workspace=self.ws, out=self.out)
        self.feed.release(s)
        self.len_host[s].copy_(self.out["accept_len"], non_blocking=True)
        return self.len_host[s]

