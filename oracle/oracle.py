"""ctypes front end of the C oracle (oracle/vsd_oracle.c).

TEST INFRASTRUCTURE ONLY: the tests, the smoke check and the benchmark's
CPU-baseline leg call this module; the library under test never does.  It
takes numpy arrays, widens logits to float32 (bf16 values are exact in f32)
and returns float64/int results.  Each function cites the passage of the paper
(arxiv 2602.05774) it restates; see vsd_oracle.c for the readings R1..R10.
"""
import ctypes as C
import numpy as np

from .build import build_oracle

_lib = None


class _LinearIn(C.Structure):
    _fields_ = [
        ("draft", C.c_void_p), ("target", C.c_void_p),
        ("B", C.c_int32), ("K", C.c_int32), ("D", C.c_int32),
        ("V", C.c_int64), ("T", C.c_double),
        ("u_draft", C.c_void_p), ("u_accept", C.c_void_p), ("u_correct", C.c_void_p),
        ("ref_logkappa", C.c_void_p),
        ("w_base", C.c_double), ("tau_car", C.c_double), ("zeta_mode", C.c_int32),
        ("kl_weight", C.c_double), ("kl_topk", C.c_int32),
    ]


class _LinearOut(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in (
        "tokens", "logq_tok", "alpha", "accept", "accept_len", "corr_tokens",
        "logq_corr", "alpha_corr", "logkappa", "logkappa_corr", "logkappa_ref",
        "ref_tokens", "expected_len", "row_lse", "weights", "loss", "grad", "margins",
        "kl_loss")]


class _TreeIn(C.Structure):
    _fields_ = [
        ("draft", C.c_void_p), ("target", C.c_void_p),
        ("B", C.c_int32), ("N", C.c_int32), ("V", C.c_int64), ("T", C.c_double),
        ("parent", C.c_void_p), ("tokens", C.c_void_p),
        ("u_accept", C.c_void_p), ("u_correct", C.c_void_p), ("rule", C.c_int32),
    ]


class _TreeEmIn(C.Structure):
    _fields_ = [
        ("draft", C.c_void_p), ("target", C.c_void_p),
        ("B", C.c_int32), ("N", C.c_int32), ("V", C.c_int64), ("T", C.c_double),
        ("parent", C.c_void_p), ("tokens", C.c_void_p),
        ("u_accept", C.c_void_p), ("u_correct", C.c_void_p),
        ("w_base", C.c_double), ("tau_car", C.c_double), ("zeta_mode", C.c_int32),
    ]


class _TreeEmOut(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in (
        "corr_tokens", "logq_tok", "logq_corr", "logkappa", "logkappa_corr", "logkappa_ref",
        "weights", "loss", "grad", "margins")]


class _TreeOut(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in (
        "alpha", "accept", "path_accept", "logkappa", "corr_tokens", "deepest",
        "accept_len", "bonus", "margins")]


def _bind(path):
    """Load an oracle shared library and declare its entry points."""
    lib_ = C.CDLL(path)
    lib_.vso_linear.argtypes = [C.POINTER(_LinearIn), C.POINTER(_LinearOut)]
    lib_.vso_linear.restype = C.c_int
    lib_.vso_tree.argtypes = [C.POINTER(_TreeIn), C.POINTER(_TreeOut)]
    lib_.vso_tree.restype = C.c_int
    lib_.vso_log_softmax.argtypes = [C.c_void_p, C.c_int64, C.c_double, C.c_void_p]
    lib_.vso_log_softmax.restype = C.c_double
    lib_.vso_sample.argtypes = [C.c_void_p, C.c_int64, C.c_double, C.c_void_p]
    lib_.vso_sample.restype = C.c_int64
    lib_.vso_prefix_weights.argtypes = [
        C.c_int, C.c_int, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p,
        C.c_double, C.c_double, C.c_int, C.c_void_p]
    lib_.vso_prefix_weights.restype = C.c_double
    lib_.vso_prefix_objective.argtypes = [
        C.c_void_p, C.c_int, C.c_int, C.c_int64, C.c_double, C.c_void_p, C.c_void_p,
        C.c_void_p, C.c_double, C.c_int, C.c_void_p]
    lib_.vso_prefix_objective.restype = C.c_double
    lib_.vso_decision_margin.argtypes = [C.c_double, C.c_double, C.c_int, C.c_void_p,
                                         C.c_void_p, C.c_void_p, C.c_void_p]
    lib_.vso_decision_margin.restype = C.c_double
    lib_.vso_topk_ce.argtypes = [C.c_void_p, C.c_void_p, C.c_int64, C.c_double, C.c_int,
                                 C.c_void_p, C.c_void_p]
    lib_.vso_topk_ce.restype = C.c_double
    lib_.vso_reference_logkappa.argtypes = [C.c_void_p, C.c_void_p, C.c_int32, C.c_int32,
                                            C.c_int64, C.c_double, C.c_void_p]
    lib_.vso_reference_logkappa.restype = C.c_int
    lib_.vso_tree_em.argtypes = [C.POINTER(_TreeEmIn), C.POINTER(_TreeEmOut)]
    lib_.vso_tree_em.restype = C.c_int
    return lib_


def lib():
    global _lib
    if _lib is None:
        _lib = _bind(build_oracle())
    return _lib


class using_library:
    """Context manager that routes this module's functions to another build of
    the oracle (the mutation test compiles deliberately broken copies of
    vsd_oracle.c and checks that the pins reject each of them)."""

    def __init__(self, path):
        self.path = path

    def __enter__(self):
        global _lib
        self.saved = lib()
        _lib = _bind(self.path)
        return self

    def __exit__(self, *exc):
        global _lib
        _lib = self.saved


def _f32(a):
    return np.ascontiguousarray(np.asarray(a, dtype=np.float32))


def _i32(a):
    return np.ascontiguousarray(np.asarray(a, dtype=np.int32))


def _ptr(a):
    return None if a is None else a.ctypes.data


def log_softmax(x, T=1.0):
    """Eq. 1's distributions: log softmax(x / T) of one row, float64."""
    x = _f32(x).reshape(-1)
    out = np.empty(x.size, dtype=np.float64)
    lib().vso_log_softmax(_ptr(x), x.size, float(T), _ptr(out))
    return out


def sample(prob, u):
    """Inverse-CDF draw (smallest v with u < F(v)); returns (v, margin)."""
    prob = np.ascontiguousarray(np.asarray(prob, dtype=np.float64)).reshape(-1)
    m = np.zeros(1, dtype=np.float64)
    v = lib().vso_sample(_ptr(prob), prob.size, float(u), _ptr(m))
    return int(v), float(m[0])


def linear(draft, target, T, u_draft, u_accept, u_correct, K, D, ref_logkappa=None,
           w_base=1.05, tau_car=0.2, zeta_mode=0, want_grad=True, kl_weight=0.0, kl_topk=10):
    """E-step + M-step over linear paths (Algorithm 1, Algorithm 2, Eqs. 1, 2, 11,
    beta, zeta, advance); with kl_weight != 0 the VSD (KL) variant adds
    kl_weight times the prefix's top-kl_topk term of Eq. klv (reading R11).
    T = 0 is greedy decoding (reading R12).

    draft, target: [B*K*D, V] (any float dtype; widened to f32 exactly).
    Returns a dict of numpy arrays named as the C-ABI outputs.
    """
    draft = _f32(draft)
    target = _f32(target)
    V = draft.shape[-1]
    R = draft.size // V
    B = R // (K * D)
    assert B * K * D == R and target.shape == draft.shape
    ud, ua, uc = _f32(u_draft).reshape(-1), _f32(u_accept).reshape(-1), _f32(u_correct).reshape(-1)
    assert ud.size == R and ua.size == R and uc.size == R
    ref = None if ref_logkappa is None else _f32(ref_logkappa).reshape(-1)
    if ref is not None:
        assert ref.size == B * D
    o = dict(
        tokens=np.zeros(R, np.int32), logq_tok=np.zeros(R), alpha=np.zeros(R),
        accept=np.zeros(R, np.uint8), accept_len=np.zeros(B * K, np.int32),
        corr_tokens=np.zeros(R, np.int32), logq_corr=np.zeros(R), alpha_corr=np.zeros(R),
        logkappa=np.zeros(R), logkappa_corr=np.zeros(R), logkappa_ref=np.zeros(R),
        ref_tokens=np.zeros(R, np.int32), expected_len=np.zeros(B * K),
        row_lse=np.zeros((R, 2)), weights=np.zeros((B, D, K, 4)), loss=np.zeros(B + 1),
        grad=np.zeros((R, V)) if want_grad else None, margins=np.zeros((R, 6)),
        kl_loss=np.zeros(R))
    li = _LinearIn(_ptr(draft), _ptr(target), B, K, D, V, float(T), _ptr(ud), _ptr(ua),
                   _ptr(uc), _ptr(ref), float(w_base), float(tau_car), int(zeta_mode),
                   float(kl_weight), int(kl_topk))
    lo = _LinearOut(*[_ptr(o[n]) for n, _ in _LinearOut._fields_])
    rc = lib().vso_linear(C.byref(li), C.byref(lo))
    if rc != 0:
        raise ValueError("oracle rejected the arguments (code %d)" % rc)
    return o


def tree(draft, target, T, parent, tokens, u_accept, u_correct, rule=0):
    """Verification of a draft tree with parent pointers (App. E tree, Eq. 1 per
    node, Sec. 3 residual).  draft/target [B*N, V]; parent, tokens, uniforms [B, N].
    rule 0: every branch verified alone; 1: sequential siblings (reading R14)."""
    draft = _f32(draft)
    target = _f32(target)
    parent = _i32(parent)
    B, N = parent.shape
    V = draft.shape[-1]
    assert draft.size == B * N * V and target.shape == draft.shape
    tokens = _i32(tokens).reshape(B, N)
    ua, uc = _f32(u_accept).reshape(B, N), _f32(u_correct).reshape(B, N)
    o = dict(alpha=np.zeros((B, N)), accept=np.zeros((B, N), np.uint8),
             path_accept=np.zeros((B, N), np.uint8), logkappa=np.zeros((B, N)),
             corr_tokens=np.zeros((B, N), np.int32), deepest=np.zeros(B, np.int32),
             accept_len=np.zeros(B, np.int32), bonus=np.zeros(B, np.int32),
             margins=np.zeros((B, N, 2)))
    ti = _TreeIn(_ptr(draft), _ptr(target), B, N, V, float(T), _ptr(parent), _ptr(tokens),
                 _ptr(ua), _ptr(uc), int(rule))
    to = _TreeOut(*[_ptr(o[n]) for n, _ in _TreeOut._fields_])
    rc = lib().vso_tree(C.byref(ti), C.byref(to))
    if rc != 0:
        raise ValueError("oracle rejected the tree (code %d)" % rc)
    return o


def tree_em(draft, target, T, parent, tokens, u_accept, u_correct, w_base=1.05, tau_car=0.2,
            zeta_mode=0, want_grad=True):
    """E-step + M-step over draft trees, every node a latent proposal (reading
    R15; Algorithm 1 and 2, Eqs. 1, 2, beta, zeta, advance on the tree's root
    paths).  draft/target [B*N, V]; parent, tokens, uniforms [B, N]."""
    draft = _f32(draft)
    target = _f32(target)
    parent = _i32(parent)
    B, N = parent.shape
    V = draft.shape[-1]
    assert draft.size == B * N * V and target.shape == draft.shape
    tokens = _i32(tokens).reshape(B, N)
    ua, uc = _f32(u_accept).reshape(B, N), _f32(u_correct).reshape(B, N)
    o = dict(corr_tokens=np.zeros((B, N), np.int32), logq_tok=np.zeros((B, N)),
             logq_corr=np.zeros((B, N)), logkappa=np.zeros((B, N)),
             logkappa_corr=np.zeros((B, N)), logkappa_ref=np.zeros((B, N)),
             weights=np.zeros((B, N, 4)), loss=np.zeros(B + 1),
             grad=np.zeros((B * N, V)) if want_grad else None, margins=np.zeros((B, N, 3)))
    ti = _TreeEmIn(_ptr(draft), _ptr(target), B, N, V, float(T), _ptr(parent), _ptr(tokens),
                   _ptr(ua), _ptr(uc), float(w_base), float(tau_car), int(zeta_mode))
    to = _TreeEmOut(*[_ptr(o[n]) for n, _ in _TreeEmOut._fields_])
    rc = lib().vso_tree_em(C.byref(ti), C.byref(to))
    if rc != 0:
        raise ValueError("oracle rejected the tree (code %d)" % rc)
    return o


def reference_logkappa(ref_draft, ref_target, T, B, D):
    """log kappa of supplied greedy reference paths (Algorithm 2, reading R13):
    rows [B*D, V] along z-bar; returns [B, D] prefix sums of log min(1, p/q)
    at each row's target argmax (T = 0: the greedy limits)."""
    xq = _f32(ref_draft)
    xp = _f32(ref_target)
    V = xq.shape[-1]
    assert xq.size == B * D * V and xp.shape == xq.shape
    out = np.zeros((B, D))
    rc = lib().vso_reference_logkappa(_ptr(xq), _ptr(xp), B, D, V, float(T), _ptr(out))
    if rc != 0:
        raise ValueError("oracle rejected the arguments (code %d)" % rc)
    return out


def topk_ce(draft_row, target_row, T=1.0, k=10):
    """Eq. klv for one row: (L, Omega [k] in selection order, dL/dx at Omega)."""
    xq = _f32(draft_row).reshape(-1)
    xp = _f32(target_row).reshape(-1)
    kk = min(k, xq.size)
    tok = np.zeros(max(kk, 1), np.int32)
    dl = np.zeros(max(kk, 1))
    L = lib().vso_topk_ce(_ptr(xq), _ptr(xp), xq.size, float(T), int(k), _ptr(tok), _ptr(dl))
    return L, tok[:kk], dl[:kk]


def decision_margin(a, b, ra, ta, rb=None, tb=None):
    """Margin of the comparison log k(z_a) >= log k(z_b) of Algorithm 2, as the
    parity protocol uses it: |a - b| for unequal sums; for equal sums the
    smallest log-ratio log(p/q) at the positions where the two paths hold
    different tokens if every one of them is >= 0 (so min(0, .) clips it and
    the equality is exact), else 0; 0 for an equality with an input reference
    other than 0 (rb = None).  ra, rb: log(p/q) per position."""
    ra = np.ascontiguousarray(ra, dtype=np.float64).reshape(-1)
    ta = _i32(ta).reshape(-1)
    n = ra.size
    if rb is not None:
        rb = np.ascontiguousarray(rb, dtype=np.float64).reshape(-1)
        tb = _i32(tb).reshape(-1)
        assert rb.size == n and tb.size == n
    return lib().vso_decision_margin(float(a), float(b), n, _ptr(ra), _ptr(ta), _ptr(rb),
                                     _ptr(tb))


def prefix_weights(logkappa, logkappa_corr, logkappa_ref, logq_path, w_base=1.05,
                   tau_car=0.2, zeta_mode=0):
    """o~, o', beta, zeta of one prefix (Algorithm 1 M-step lines, Eqs. beta and
    zeta).  Inputs are [K, D] tables; returns ([D, K, 4] weights, N_b)."""
    lk = np.ascontiguousarray(logkappa, dtype=np.float64)
    K, D = lk.shape
    args = [np.ascontiguousarray(a, dtype=np.float64).reshape(K, D)
            for a in (logkappa_corr, logkappa_ref, logq_path)]
    w = np.zeros((D, K, 4))
    N = lib().vso_prefix_weights(K, D, _ptr(lk), _ptr(args[0]), _ptr(args[1]), _ptr(args[2]),
                                 float(w_base), float(tau_car), int(zeta_mode), _ptr(w))
    return w, N


def prefix_objective(draft, T, tokens, corr_tokens, weights, N, B_total, want_grad=True):
    """J_b of Eq. advance for one prefix with fixed weights, and the gradient of
    -(1/B) J_b / N_b with respect to the draft logits.  draft [K, D, V]."""
    draft = _f32(draft)
    K, D, V = draft.shape
    tok = _i32(tokens).reshape(K, D)
    ctok = _i32(corr_tokens).reshape(K, D)
    w = np.ascontiguousarray(weights, dtype=np.float64).reshape(D, K, 4)
    g = np.zeros((K, D, V)) if want_grad else None
    J = lib().vso_prefix_objective(_ptr(draft), K, D, V, float(T), _ptr(tok), _ptr(ctok),
                                   _ptr(w), float(N), int(B_total), _ptr(g))
    return J, g


def lmhead_logits(hidden, weight):
    """The draft LM head (paper Sec. 5, the draft head's output layer): logits =
    hidden . weight^T from the exact input values, in float64 (a library
    matmul: one product per (row, vocabulary entry), no blocking of our own)."""
    h = np.asarray(hidden, dtype=np.float64)
    w = np.asarray(weight, dtype=np.float64)
    return h @ w.T


def lmhead_backward(grad, hidden, weight):
    """The LM head's backward (Algorithm 1's M-step carried into the draft
    head): with logits = hidden . weight^T and G = d loss / d logits,
    d loss / d hidden = G . weight and d loss / d weight = G^T . hidden, in
    float64 library matmuls of the exact inputs (no blocking of our own).
    grad [R, V], hidden [R, H], weight [V, H]; returns (d_hidden, d_weight),
    with None for the one whose other factor (weight, hidden) is None."""
    G = np.asarray(grad, dtype=np.float64)
    d_hidden = None if weight is None else G @ np.asarray(weight, dtype=np.float64)
    d_weight = None if hidden is None else G.T @ np.asarray(hidden, dtype=np.float64)
    return d_hidden, d_weight


def round_bf16(x):
    """Round float64 values to the nearest bfloat16 (8 significant bits), ties
    to even, returned as float32 holding the bfloat16 value exactly.  Finite
    values in the normal range of bfloat16."""
    x = np.asarray(x, dtype=np.float64)
    m, e = np.frexp(x)                     # x = m 2^e, 0.5 <= |m| < 1
    r = np.rint(m * 256.0) / 256.0         # 8 significant bits; rint rounds ties to even
    return np.ldexp(r, e).astype(np.float32)
