"""Thin Python binding of the C ABI in include/luna.h (argument marshalling only).

Every function here has the name of the C entry point it calls and does no
arithmetic of its own: tensors are passed as device pointers, the stream as
torch's current CUDA stream.  PyTorch provides device memory and streams.
If the compiled library is missing this module raises at import time; there
is no fallback implementation.
"""
from __future__ import annotations

import ctypes
import os

import torch

from . import build as _build

LUNA_OK = 0
STATUS_NAMES = {0: "LUNA_OK", 1: "LUNA_ERR_INVALID_ARG", 2: "LUNA_ERR_UNSUPPORTED", 3: "LUNA_ERR_WORKSPACE",
                4: "LUNA_ERR_CUDA", 5: "LUNA_ERR_DEVICE_TIMEOUT"}
LUNA_F32, LUNA_BF16 = 0, 1
_DTYPES = {torch.float32: LUNA_F32, torch.bfloat16: LUNA_BF16}
# names of the tensor-core kernels accepted by luna_profile_start
TC_KERNELS: list[str] = ["tile_split", "tc_keys", "tc_query", "tc_bwd_query", "tc_bwd_key", "tc_causal", "seg_scan",
                         "tcc_query", "tcc_dstats", "seg_rscan", "tcc_key", "tc_phi_bwd"]


class LunaError(RuntimeError):
    def __init__(self, status: int, where: str):
        super().__init__(f"{where}: {STATUS_NAMES.get(status, status)}")
        self.status = status


class PhiDesc(ctypes.Structure):
    _fields_ = [("M", ctypes.c_int), ("L", ctypes.c_int), ("hidden", ctypes.c_int), ("shared_channels", ctypes.c_int),
                ("ch_rms_target", ctypes.c_float), ("signed_outputs", ctypes.c_int),
                ("param_head_stride", ctypes.c_int64), ("act", ctypes.c_int), ("envelope", ctypes.c_int),
                ("bank_coef", ctypes.c_int)]


PARAM_KEYS = ("W", "b", "w1", "b1", "w2", "b2", "We", "be", "coef")
GRAD_KEYS = tuple("d" + k for k in PARAM_KEYS)
ACTS = {"relu": 0, "gelu": 1, "silu": 2, "tanh": 3}  # luna_act


class PhiParams(ctypes.Structure):
    _fields_ = [(k, ctypes.c_void_p) for k in PARAM_KEYS]


class PhiGrads(ctypes.Structure):
    _fields_ = [(k, ctypes.c_void_p) for k in GRAD_KEYS]


class AttnDesc(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int), ("H", ctypes.c_int), ("n", ctypes.c_int), ("d", ctypes.c_int),
                ("dv", ctypes.c_int), ("causal", ctypes.c_int), ("chunk", ctypes.c_int), ("eps", ctypes.c_float),
                ("io", ctypes.c_int)]


def library_path() -> str:
    return _build.LIB


def _load():
    path = library_path()
    if not os.path.exists(path):
        raise ImportError(f"LUNA CUDA library not built ({path}); run paper_2512_08061_gb300.build.build()")
    lib = ctypes.CDLL(path)
    P, S, I, I64 = ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int, ctypes.c_int64
    pd, ad = ctypes.POINTER(PhiDesc), ctypes.POINTER(AttnDesc)
    sig = {
        "luna_status_string": ([I], ctypes.c_char_p),
        "luna_version": ([], I),
        "luna_phi_table_size": ([pd, I, ctypes.POINTER(S)], I),
        "luna_phi_prepare": ([pd, I, ctypes.POINTER(PhiParams), P, S, P], I),
        "luna_featmap": ([pd, I, P, P, I, I64, P, P], I),
        "luna_workspace_size": ([ad, pd, I, ctypes.POINTER(S)], I),
        "luna_state_size": ([ad, pd, ctypes.POINTER(S)], I),
        "luna_attn_fwd": ([ad, pd, P, P, P, P, P, P, P, P, S, P], I),
        "luna_attn_bwd": ([ad, pd, P, P, P, P, P, P, P, P, P, P, ctypes.POINTER(PhiGrads), P, S, P], I),
        "luna_device_status": ([P, P], I),
        "luna_profile_start": ([ctypes.c_char_p], I),
        "luna_profile_stop": ([ctypes.POINTER(ctypes.c_double), ctypes.POINTER(I)], I),
        "luna_launch_count": ([], ctypes.c_uint64),
        "luna_attn_fwd_noalloc": ([ad, pd, P, P, P, P, P, P, P], I),
        "luna_state_final": ([ad, pd, P, ctypes.POINTER(P), ctypes.POINTER(I64), ctypes.POINTER(P),
                              ctypes.POINTER(I64)], I),
        "luna_attn_decode": ([ad, pd, P, P, P, P, P, P, I64, P, I64, P], I),
        "luna_selftest_wait": ([P, I64, P], I),
        "luna_noalloc_scratch": ([ctypes.POINTER(P), ctypes.POINTER(S)], I),
        "luna_attn_weights": ([ad, pd, P, P, P, P, I, I, I, P, P], I),
    }
    for name, (args, res) in sig.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = res
    return lib


_lib = _load()
EXPORTED = ("luna_status_string", "luna_version", "luna_phi_table_size", "luna_phi_prepare", "luna_featmap",
            "luna_workspace_size", "luna_state_size", "luna_attn_fwd", "luna_attn_bwd", "luna_device_status",
            "luna_profile_start", "luna_profile_stop", "luna_launch_count", "luna_attn_fwd_noalloc",
            "luna_state_final", "luna_attn_decode", "luna_selftest_wait", "luna_noalloc_scratch",
            "luna_attn_weights")


def _ptr(t):
    """Device address of a tensor, or a raw address given as an int."""
    if t is None:
        return None
    if isinstance(t, int):
        return ctypes.c_void_p(t)
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _check(st: int, where: str) -> None:
    if st != LUNA_OK:
        raise LunaError(st, where)


def _io_code(t: torch.Tensor) -> int:
    if t.dtype not in _DTYPES:
        raise TypeError(f"unsupported dtype {t.dtype}")
    return _DTYPES[t.dtype]


def phi_desc(M: int, L: int, hidden: int, shared: bool = False, ch_rms_target: float = 0.0,
             signed: bool = False, param_head_stride: int = 0, act: str = "relu", envelope: bool = False,
             bank_coef: bool = False) -> PhiDesc:
    return PhiDesc(M, L, hidden, int(bool(shared)), float(ch_rms_target), int(bool(signed)), int(param_head_stride),
                   ACTS[act], int(bool(envelope)), int(bool(bank_coef)))


def attn_desc(B, H, n, d, dv, causal=False, chunk=0, eps=1e-6, io=LUNA_BF16) -> AttnDesc:
    return AttnDesc(B, H, n, d, dv, int(bool(causal)), chunk, eps, io)


def luna_status_string(status: int) -> str:
    return _lib.luna_status_string(status).decode()


def luna_version() -> int:
    return _lib.luna_version()


def luna_phi_table_size(pd: PhiDesc, d: int) -> int:
    out = ctypes.c_size_t(0)
    _check(_lib.luna_phi_table_size(ctypes.byref(pd), d, ctypes.byref(out)), "luna_phi_table_size")
    return out.value


def luna_phi_prepare(pd: PhiDesc, d: int, params: dict, table: torch.Tensor, stream=None) -> None:
    pp = PhiParams(*[_ptr(params.get(k)) for k in PARAM_KEYS])
    _check(_lib.luna_phi_prepare(ctypes.byref(pd), d, ctypes.byref(pp), _ptr(table), table.numel() * table.element_size(),
                                 _stream(stream)), "luna_phi_prepare")


def luna_featmap(pd: PhiDesc, d: int, table: torch.Tensor, X: torch.Tensor, Phi: torch.Tensor, stream=None) -> None:
    rows = X.numel() // d if d else 0
    _check(_lib.luna_featmap(ctypes.byref(pd), d, _ptr(table), _ptr(X), _io_code(X), rows, _ptr(Phi), _stream(stream)),
           "luna_featmap")


def luna_workspace_size(ad: AttnDesc, pd: PhiDesc, backward: bool) -> int:
    out = ctypes.c_size_t(0)
    _check(_lib.luna_workspace_size(ctypes.byref(ad), ctypes.byref(pd), int(bool(backward)), ctypes.byref(out)),
           "luna_workspace_size")
    return out.value


def luna_state_size(ad: AttnDesc, pd: PhiDesc) -> int:
    out = ctypes.c_size_t(0)
    _check(_lib.luna_state_size(ctypes.byref(ad), ctypes.byref(pd), ctypes.byref(out)), "luna_state_size")
    return out.value


def luna_attn_fwd(ad, pd, table, Q, K, V, lengths, O, state, workspace, stream=None) -> None:
    _check(_lib.luna_attn_fwd(ctypes.byref(ad), ctypes.byref(pd), _ptr(table), _ptr(Q), _ptr(K), _ptr(V),
                              _ptr(lengths), _ptr(O), _ptr(state), _ptr(workspace),
                              workspace.numel() * workspace.element_size(), _stream(stream)), "luna_attn_fwd")


def luna_attn_bwd(ad, pd, table, Q, K, V, dO, lengths, state, dQ, dK, dV, grads: dict, workspace, stream=None) -> None:
    pg = PhiGrads(*[_ptr(grads.get(k)) for k in GRAD_KEYS])
    _check(_lib.luna_attn_bwd(ctypes.byref(ad), ctypes.byref(pd), _ptr(table), _ptr(Q), _ptr(K), _ptr(V), _ptr(dO),
                              _ptr(lengths), _ptr(state), _ptr(dQ), _ptr(dK), _ptr(dV), ctypes.byref(pg),
                              _ptr(workspace), workspace.numel() * workspace.element_size(), _stream(stream)),
           "luna_attn_bwd")


def luna_attn_fwd_noalloc(ad, pd, table, Q, K, V, lengths, O, stream=None) -> None:
    _check(_lib.luna_attn_fwd_noalloc(ctypes.byref(ad), ctypes.byref(pd), _ptr(table), _ptr(Q), _ptr(K), _ptr(V),
                                      _ptr(lengths), _ptr(O), _stream(stream)), "luna_attn_fwd_noalloc")


NOALLOC_SCRATCH_BYTES = 16 << 20


def luna_attn_weights(ad, pd, table, Q, K, lengths, row0: int, rows: int, teacher: bool, A: torch.Tensor,
                      stream=None) -> None:
    _check(_lib.luna_attn_weights(ctypes.byref(ad), ctypes.byref(pd), _ptr(table), _ptr(Q), _ptr(K), _ptr(lengths),
                                  int(row0), int(rows), int(bool(teacher)), _ptr(A), _stream(stream)),
           "luna_attn_weights")


def luna_state_final(ad, pd, state) -> tuple[int, int, int, int]:
    """(S address, S stride, z address, z stride) of the final causal state inside `state` (floats)."""
    S, Ss, z, zs = ctypes.c_void_p(), ctypes.c_int64(), ctypes.c_void_p(), ctypes.c_int64()
    _check(_lib.luna_state_final(ctypes.byref(ad), ctypes.byref(pd), _ptr(state), ctypes.byref(S), ctypes.byref(Ss),
                                 ctypes.byref(z), ctypes.byref(zs)), "luna_state_final")
    return S.value, Ss.value, z.value, zs.value


def luna_attn_decode(ad, pd, table, q, k, v, o, S, S_stride, z, z_stride, stream=None) -> None:
    """S, z: tensors (their data pointers are used) or raw device addresses."""
    sp = _ptr(S) if isinstance(S, torch.Tensor) else ctypes.c_void_p(S)
    zp = _ptr(z) if isinstance(z, torch.Tensor) else ctypes.c_void_p(z)
    _check(_lib.luna_attn_decode(ctypes.byref(ad), ctypes.byref(pd), _ptr(table), _ptr(q), _ptr(k), _ptr(v), _ptr(o),
                                 sp, S_stride, zp, z_stride, _stream(stream)), "luna_attn_decode")


def luna_device_status(workspace: torch.Tensor, stream=None) -> int:
    return _lib.luna_device_status(_ptr(workspace), _stream(stream))


def luna_noalloc_scratch() -> tuple[int, int]:
    """(device address, bytes) of the no-allocation entry point's scratch array on the current device."""
    p, n = ctypes.c_void_p(), ctypes.c_size_t(0)
    _check(_lib.luna_noalloc_scratch(ctypes.byref(p), ctypes.byref(n)), "luna_noalloc_scratch")
    return p.value, n.value


def luna_selftest_wait(workspace: torch.Tensor, limit_ns: int, stream=None) -> None:
    _check(_lib.luna_selftest_wait(_ptr(workspace), int(limit_ns), _stream(stream)), "luna_selftest_wait")


def luna_profile_start(kernel: str) -> None:
    _check(_lib.luna_profile_start(kernel.encode()), "luna_profile_start")


def luna_profile_stop() -> tuple[float, int]:
    ms, n = ctypes.c_double(0.0), ctypes.c_int(0)
    _check(_lib.luna_profile_stop(ctypes.byref(ms), ctypes.byref(n)), "luna_profile_stop")
    return ms.value, n.value


def luna_launch_count() -> int:
    return int(_lib.luna_launch_count())


# ---------------------------------------------------------------------------
# convenience: buffers sized by the library, allocated with torch

def alloc_bytes(nbytes: int, device) -> torch.Tensor:
    """A 256-byte aligned uint8 device buffer (torch's caching allocator aligns to 512)."""
    return torch.empty(max(int(nbytes), 256), dtype=torch.uint8, device=device)


class Luna:
    """Owns the table, workspace and state buffers of one problem shape."""

    def __init__(self, B, H, n, d, dv, M, L, hidden=64, causal=False, eps=1e-6, io=torch.bfloat16, chunk=0,
                 device="cuda", shared=False, ch_rms_target=0.0, signed=False, per_head=False, act="relu",
                 envelope=False, bank_coef=False):
        self.pd = phi_desc(M, L, hidden, shared, ch_rms_target, signed, 0, act, envelope, bank_coef)
        self.ad = attn_desc(B, H, n, d, dv, causal, chunk, eps, _DTYPES[io])
        self.d = d
        self.device = torch.device(device)
        tb = luna_phi_table_size(self.pd, d)
        self.heads = H if per_head else 0  # per-head parameters: one table per head, tb bytes apart
        if per_head:
            self.pd.param_head_stride = tb
        self.table = alloc_bytes(tb * max(1, self.heads), self.device)
        self.ws = alloc_bytes(max(luna_workspace_size(self.ad, self.pd, False),
                                  luna_workspace_size(self.ad, self.pd, True)), self.device)
        self.state = alloc_bytes(luna_state_size(self.ad, self.pd), self.device)

    def prepare(self, params: dict, stream=None):
        """params: W, b, w1, b1, w2, b2 device tensors (with a leading head axis for per-head parameters),
        and We, be (envelope) or coef (Bank+Coef) with those variants."""
        if not self.heads:
            luna_phi_prepare(self.pd, self.d, params, self.table, stream)
            return
        tb = self.pd.param_head_stride
        for h in range(self.heads):
            luna_phi_prepare(self.pd, self.d, {k: v[h] for k, v in params.items()}, self.table[h * tb:(h + 1) * tb],
                             stream)

    def forward(self, Q, K, V, lengths=None, O=None, save_state=True, stream=None):
        if O is None:
            O = torch.empty(Q.shape[:-1] + (self.ad.dv,), dtype=Q.dtype, device=Q.device)
        luna_attn_fwd(self.ad, self.pd, self.table, Q, K, V, lengths, O, self.state if save_state else None,
                      self.ws, stream)
        return O

    def backward(self, Q, K, V, dO, lengths=None, use_state=True, out=None, stream=None):
        if out is None:
            M, L, hid = self.pd.M, self.pd.L, self.pd.hidden
            f32 = dict(dtype=torch.float32, device=Q.device)
            fc1 = (hid,) if self.pd.shared_channels else (L, hid)
            g = (self.heads,) if self.heads else ()
            out = {"dQ": torch.empty_like(Q), "dK": torch.empty_like(K), "dV": torch.empty_like(V),
                   "dW": torch.empty(g + (M, self.d), **f32), "db": torch.empty(g + (M,), **f32),
                   "dw1": torch.empty(g + fc1, **f32), "db1": torch.empty(g + fc1, **f32),
                   "dw2": torch.empty(g + (L, hid), **f32), "db2": torch.empty(g + (L,), **f32)}
            if self.pd.envelope:
                out.update(dWe=torch.empty((L, self.d), **f32), dbe=torch.empty((L,), **f32))
            if self.pd.bank_coef:
                out["dcoef"] = torch.empty((L,), **f32)
        luna_attn_bwd(self.ad, self.pd, self.table, Q, K, V, dO, lengths, self.state if use_state else None,
                      out["dQ"], out["dK"], out["dV"], out, self.ws, stream)
        return out

    def decode(self, q, k, v, o=None, stream=None):
        """One streaming-form step per (b, h) from the final state of the last causal forward
        (saved with save_state=True), which it advances in place.  q, k: (B, H, d); v: (B, H, dv)."""
        if o is None:
            o = torch.empty(q.shape[:-1] + (self.ad.dv,), dtype=q.dtype, device=q.device)
        S, Ss, z, zs = luna_state_final(self.ad, self.pd, self.state)
        luna_attn_decode(self.ad, self.pd, self.table, q, k, v, o, S, Ss, z, zs, stream)
        return o
