"""Python binding of the fp64 CPU oracle (oracle/luna_oracle.c).

TEST INFRASTRUCTURE ONLY: imported by the tests, by the graft smoke check and
by the CPU-baseline leg of the benchmark, never by the library path.  It shares
no code with the CUDA path; both sides only share the seeded input generator
in `synth`.

Parity pins (tests/test_oracle_pins.py): hand-computed feature maps
(tests/golden/phi_hand.json), brute-force quadratic form of Eq. (kernel-attn),
constant-channel closed form, Gram matrix PSD (Prop. 1), permutation/padding/
linearity invariances, normalised weights summing to 1, causal = masked
quadratic form, and central finite differences of every gradient.  The
attention weights of the conversion stage (tests/test_oracle_weights.py): their
product with V is the linear form's output, rows sum to den/(den+eps), constant
channels give uniform weights, the softmax teacher against a closed form.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "luna_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD_DIR, "libluna_oracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle shared library with gcc (OpenMP when available)."""
    os.makedirs(_BUILD_DIR, exist_ok=True)
    if not force and os.path.exists(_SO) and os.path.getmtime(_SO) >= os.path.getmtime(_SRC):
        return _SO
    base = ["gcc", "-O2", "-std=c99", "-fPIC", "-shared", "-ffp-contract=off", _SRC, "-lm"]
    tmp = _SO + f".tmp{os.getpid()}"
    try:
        subprocess.run(base[:-1] + ["-fopenmp", "-o", tmp, "-lm"], check=True, capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base + ["-o", tmp], check=True)
    os.replace(tmp, _SO)
    return _SO


class _Phi(ctypes.Structure):
    _fields_ = [("d", ctypes.c_int), ("M", ctypes.c_int), ("L", ctypes.c_int), ("hid", ctypes.c_int)] + [
        (k, ctypes.c_void_p) for k in ("W", "b", "w1", "b1", "w2", "b2")
    ] + [("shared", ctypes.c_int), ("ch_rms_target", ctypes.c_double), ("chs", ctypes.c_void_p), ("heads", ctypes.c_int),
         ("signed_out", ctypes.c_int), ("act", ctypes.c_int), ("We", ctypes.c_void_p), ("be", ctypes.c_void_p),
         ("coef", ctypes.c_void_p)]

# hidden-unit activations of the channel MLPs, by name (the code the C oracle takes)
ACTS = {"relu": 0, "gelu": 1, "silu": 2, "tanh": 3}


_P = ctypes.c_void_p
_I = ctypes.c_int
_D = ctypes.c_double
_I64 = ctypes.c_int64


def lib():
    global _lib
    with _lock:
        if _lib is None:
            so = build()
            L = ctypes.CDLL(so)
            phi = ctypes.POINTER(_Phi)
            L.oracle_featmap.argtypes = [phi, _P, _I64, _P]
            L.oracle_kink_margin.argtypes = [phi, _P, _I64, _P]
            L.oracle_psi.argtypes = [phi, _I, _D]
            L.oracle_psi.restype = _D
            L.oracle_attn_fwd.argtypes = [phi, _I, _I, _I, _I, _I, _D, _P, _P, _P, _P, _P]
            L.oracle_attn_quadratic.argtypes = [phi, _I, _I, _I, _I, _I, _D, _P, _P, _P, _P, _P]
            L.oracle_attn_bwd.argtypes = [phi, _I, _I, _I, _I, _I, _D, _P, _P, _P, _P, _P, _P, _P, _P] + [_P] * 6
            L.oracle_attn_bwd_var.argtypes = [phi, _I, _I, _I, _I, _I, _D, _P, _P, _P, _P, _P, _P, _P, _P] + [_P] * 9
            L.oracle_ch_rms.argtypes = [phi, _P, _I, _I, _I, _P, _P, _P]
            L.oracle_attn_weights.argtypes = [phi, _I, _I, _I, _I, _D, _P, _P, _P, _I, _I, _I, _P]
            L.oracle_max_threads.restype = _I
            L.oracle_set_threads.argtypes = [_I]
            L.oracle_set_abs_terms.argtypes = [_I]
            L.oracle_phi_size.restype = ctypes.c_size_t
            L.oracle_phi_offset.restype = ctypes.c_size_t
            L.oracle_phi_offset.argtypes = [_I]
            # the mirror of the C struct must have its layout
            assert L.oracle_phi_size() == ctypes.sizeof(_Phi)
            for i, f in enumerate(("W", "shared", "ch_rms_target", "chs", "heads", "signed_out", "act", "We", "coef")):
                assert L.oracle_phi_offset(i) == getattr(_Phi, f).offset, f
            _lib = L
    return _lib


def max_threads() -> int:
    return lib().oracle_max_threads()


def set_threads(t: int) -> None:
    lib().oracle_set_threads(int(t))


def _f64(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float64)


class PhiParams:
    """fp64 copies of the feature-map parameters (W, b, w1, b1, w2, b2).  One MLP per
    channel: w1, b1, w2 of shape (L, hidden); the shared-channel MLP: w1, b1 of shape
    (hidden,) and w2 of shape (L, hidden).  Per-head parameters carry a leading head axis
    on every array (W of shape (H, M, d), ...): head h of every sequence then uses slice h,
    and the gradients keep that axis.  nonneg=False is the listing's option of that name:
    the channel outputs without the outer ReLU.  ch_rms_target > 0 turns on the channel RMS
    normalisation: every channel's MLP outputs are scaled by
    s_l = min(target / (rms_l + 1e-6), 1) with rms_l over the valid rows of the input
    the feature map is applied to (the queries and the keys separately).

    The ablation variants of the feature map (Sec. 5.4, Table 5) and the listing's activation:
    act in ACTS (the hidden-unit activation of the channel MLPs; "relu" is the default);
    params["We"] (L, d) and params["be"] (L,) add the envelope gate
    h_l(x) = sigmoid(We_l . x + be_l) multiplying channel l of every projection;
    params["coef"] (L,) adds the Bank+Coef coefficient c_l multiplying channel l.  These
    combine with each other, not with per-head parameters or ch_rms."""

    def __init__(self, params: dict, ch_rms_target: float = 0.0, nonneg: bool = True, act: str = "relu"):
        self.arrays = {k: _f64(params[k]) for k in ("W", "b", "w1", "b1", "w2", "b2")}
        self.extra = {k: _f64(params[k]) for k in ("We", "be", "coef") if params.get(k) is not None}
        W = self.arrays["W"]
        self.heads = W.shape[0] if W.ndim == 3 else 0
        lead = (self.heads,) if self.heads else ()
        self.M, self.d = W.shape[-2:]
        core = {k: v.shape[len(lead):] for k, v in self.arrays.items()}
        self.shared = len(core["w1"]) == 1
        self.L, self.hid = core["w2"]
        assert all(v.shape[:len(lead)] == lead for v in self.arrays.values())
        assert core["b"] == (self.M,)
        assert core["w1"] == core["b1"] == ((self.hid,) if self.shared else (self.L, self.hid))
        assert core["b2"] == (self.L,)
        if self.heads and ch_rms_target > 0:
            raise ValueError("channel normalisation with per-head parameters is not defined here")
        self.act = act
        self.variant = act != "relu" or bool(self.extra)
        if self.variant and (self.heads or ch_rms_target > 0):
            raise ValueError("the feature-map variants combine with neither per-head parameters nor ch_rms")
        assert ("We" in self.extra) == ("be" in self.extra)
        if "We" in self.extra:
            assert self.extra["We"].shape == (self.L, self.d) and self.extra["be"].shape == (self.L,)
        if "coef" in self.extra:
            assert self.extra["coef"].shape == (self.L,)
        ex = [self.extra[k].ctypes.data if k in self.extra else None for k in ("We", "be", "coef")]
        self.struct = _Phi(self.d, self.M, self.L, self.hid,
                           *[self.arrays[k].ctypes.data for k in ("W", "b", "w1", "b1", "w2", "b2")],
                           int(self.shared), float(ch_rms_target), None, int(self.heads), int(not nonneg),
                           ACTS[act], *ex)
        self.ch_rms_target = float(ch_rms_target)
        self.nonneg = bool(nonneg)

    @property
    def D(self) -> int:
        return self.M * self.L

    def head(self, h: int) -> "PhiParams":
        """The parameters of head h (per-head parameters only)."""
        assert self.heads
        return PhiParams({k: v[h] for k, v in self.arrays.items()}, nonneg=self.nonneg, act=self.act)

    def ref(self):
        return ctypes.byref(self.struct)


def _as_params(params) -> PhiParams:
    return params if isinstance(params, PhiParams) else PhiParams(params)


def ch_rms(params, X, lengths=None):
    """Channel RMS statistics of the MLP outputs over the valid rows of X (B,H,n,d):
    (s, rms), each of shape (L,), s = min(target / (rms + 1e-6), 1)."""
    p = _as_params(params)
    assert not p.heads
    X = _f64(X)
    B, H, n, d = X.shape
    la, lp = _lens(lengths, B)
    s = np.empty(p.L)
    rms = np.empty(p.L)
    lib().oracle_ch_rms(p.ref(), X.ctypes.data, B, H, n, lp, s.ctypes.data, rms.ctypes.data)
    return s, rms


def featmap(params, X) -> np.ndarray:
    """phi(X) for rows of X (..., d) -> (..., M*L), feature index i*L + l.  With channel
    RMS normalisation the statistics are those of all rows of X.  With per-head parameters
    X is (..., H, n, d) and head h's rows use head h's parameters."""
    p = _as_params(params)
    X = _f64(X)
    if p.heads:
        assert X.ndim >= 3 and X.shape[-3] == p.heads
        return np.stack([featmap(p.head(h), X[..., h, :, :]) for h in range(p.heads)], axis=-3)
    rows = X.size // p.d
    out = np.empty(X.shape[:-1] + (p.D,), dtype=np.float64)
    lib().oracle_featmap(p.ref(), X.ctypes.data, rows, out.ctypes.data)
    return out


def kink_margin(params, X) -> np.ndarray:
    p = _as_params(params)
    X = _f64(X)
    if p.heads:
        assert X.ndim >= 3 and X.shape[-3] == p.heads
        return np.stack([kink_margin(p.head(h), X[..., h, :, :]) for h in range(p.heads)], axis=-2)
    out = np.empty(X.shape[:-1], dtype=np.float64)
    lib().oracle_kink_margin(p.ref(), X.ctypes.data, X.size // p.d, out.ctypes.data)
    return out


def psi(params, l: int, u: float) -> float:
    p = _as_params(params)
    assert not p.heads
    return lib().oracle_psi(p.ref(), int(l), float(u))


def _lens(lengths, B):
    if lengths is None:
        return None, 0
    a = np.ascontiguousarray(lengths, dtype=np.int32)
    assert a.shape == (B,)
    return a, a.ctypes.data


def attn_fwd(params, Q, K, V, lengths=None, causal=False, eps=1e-6) -> np.ndarray:
    """Linear (sufficient statistics) form; Q, K (B,H,n,d), V (B,H,n,dv)."""
    p = _as_params(params)
    Q, K, V = _f64(Q), _f64(K), _f64(V)
    B, H, n, d = Q.shape
    dv = V.shape[-1]
    assert d == p.d and K.shape == Q.shape and V.shape[:3] == Q.shape[:3]
    assert p.heads in (0, H)
    la, lp = _lens(lengths, B)
    O = np.empty(V.shape, dtype=np.float64)
    lib().oracle_attn_fwd(p.ref(), B, H, n, dv, int(bool(causal)), float(eps),
                          Q.ctypes.data, K.ctypes.data, V.ctypes.data, lp, O.ctypes.data)
    return O


def attn_quadratic(params, Q, K, V, lengths=None, causal=False, eps=1e-6) -> np.ndarray:
    """Brute force: O_i = sum_j k(q_i,k_j) v_j / (sum_j k(q_i,k_j) + eps)."""
    p = _as_params(params)
    Q, K, V = _f64(Q), _f64(K), _f64(V)
    B, H, n, d = Q.shape
    dv = V.shape[-1]
    assert p.heads in (0, H)
    la, lp = _lens(lengths, B)
    O = np.empty(V.shape, dtype=np.float64)
    lib().oracle_attn_quadratic(p.ref(), B, H, n, dv, int(bool(causal)), float(eps),
                                Q.ctypes.data, K.ctypes.data, V.ctypes.data, lp, O.ctypes.data)
    return O


def attn_weights(params, Q, K, lengths=None, causal=False, eps=1e-6, row0=0, rows=None, teacher=False) -> np.ndarray:
    """Attention weights of query rows [row0, row0 + rows) of every (b, h): (B, H, rows, n).
    teacher=False: the LUNA weights a_ij = k(q_i,k_j) / (sum_j k + eps) (O = A V);
    teacher=True: the softmax weights exp(q_i.k_j/sqrt(d)) / sum_j exp(...) over the same keys."""
    p = _as_params(params)
    Q, K = _f64(Q), _f64(K)
    B, H, n, d = Q.shape
    rows = n - row0 if rows is None else rows
    assert p.heads in (0, H) and K.shape == Q.shape
    la, lp = _lens(lengths, B)
    A = np.empty((B, H, rows, n), dtype=np.float64)
    lib().oracle_attn_weights(p.ref(), B, H, n, int(bool(causal)), float(eps), Q.ctypes.data, K.ctypes.data, lp,
                              int(row0), int(rows), int(bool(teacher)), A.ctypes.data)
    return A


def attn_bwd_abs_terms(params, Q, K, V, dO, lengths=None, causal=False, eps=1e-6) -> dict:
    """For every feature-map parameter gradient, the sum of the absolute values
    of its per-sample contributions (same chain rule as attn_bwd, with |term|
    accumulated): the scale of the rounding error of a finite-precision
    evaluation of that gradient sum."""
    lib().oracle_set_abs_terms(1)
    try:
        g = attn_bwd(params, Q, K, V, dO, lengths, causal, eps)
    finally:
        lib().oracle_set_abs_terms(0)
    return {k: v for k, v in g.items() if k not in ("dQ", "dK", "dV")}


def attn_bwd(params, Q, K, V, dO, lengths=None, causal=False, eps=1e-6) -> dict:
    """Gradients of sum(O * dO) w.r.t. Q, K, V and every feature-map parameter."""
    p = _as_params(params)
    Q, K, V, dO = _f64(Q), _f64(K), _f64(V), _f64(dO)
    B, H, n, d = Q.shape
    dv = V.shape[-1]
    assert p.heads in (0, H)
    la, lp = _lens(lengths, B)
    out = {"dQ": np.empty(Q.shape), "dK": np.empty(K.shape), "dV": np.empty(V.shape)}
    out.update({"d" + k: np.empty(p.arrays[k].shape) for k in ("W", "b", "w1", "b1", "w2", "b2")})
    out.update({"d" + k: np.empty(v.shape) for k, v in p.extra.items()})
    lib().oracle_attn_bwd_var(p.ref(), B, H, n, dv, int(bool(causal)), float(eps),
                              Q.ctypes.data, K.ctypes.data, V.ctypes.data, dO.ctypes.data, lp,
                              out["dQ"].ctypes.data, out["dK"].ctypes.data, out["dV"].ctypes.data,
                              *[out[k].ctypes.data for k in ("dW", "db", "dw1", "db1", "dw2", "db2")],
                              *[out["d" + k].ctypes.data if k in p.extra else None for k in ("We", "be", "coef")])
    return out
