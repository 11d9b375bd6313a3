"""Helpers for the GPU parity tests: seeded cases, device transfer, error metric."""
from __future__ import annotations

import math

import numpy as np

import oracle
import synth

TOL = {"f32": 1e-4, "bf16": 2e-2}
KINK_MARGIN = 1e-5


def relerr(got, ref) -> float:
    """max_i |g_i - r_i| / max(|r_i|, rms(r)): the element-wise relative error,
    floored at the tensor's rms so that near-zero entries are judged on the
    scale of the tensor."""
    g = np.asarray(got, dtype=np.float64)
    r = np.asarray(ref, dtype=np.float64)
    if r.size == 0:
        return 0.0
    rms = float(np.sqrt(np.mean(r * r)))
    if rms == 0.0:
        return float(np.max(np.abs(g)))
    return float(np.max(np.abs(g - r) / np.maximum(np.abs(r), rms)))


def relerr_rows(got, ref) -> float:
    """max_i |g_i - r_i| / max(|r_i|, rms of r_i's row): the element-wise
    relative error floored at the rms of its row (last axis).  Used for outputs
    of the streaming form, where every row is its own normalised average of the
    values and the first rows of a sequence are an order of magnitude larger
    than the last."""
    g = np.asarray(got, dtype=np.float64)
    r = np.asarray(ref, dtype=np.float64)
    if r.size == 0:
        return 0.0
    rms = np.sqrt(np.mean(r * r, axis=-1, keepdims=True))
    floor = np.maximum(np.abs(r), rms)
    err = np.abs(g - r)
    zero = floor == 0.0
    return float(max(np.max(np.where(zero, 0.0, err / np.where(zero, 1.0, floor))), np.max(np.where(zero, err, 0.0))))


# ---------------------------------------------------------------------------
# guard bands (the sanitizer's out-of-bounds checks are not available): every
# buffer the library writes in the parity tests sits between two bands of a
# known byte pattern that must still be intact after each call

GUARD_BYTES = 4096  # keeps the 256-byte alignment the library asks for
GUARD_PATTERN = 0x5A


def guarded_bytes(nbytes: int, device, registry: list):
    """A uint8 device buffer of nbytes between two guard bands; the band is recorded in `registry`."""
    import torch
    base = torch.full((int(nbytes) + 2 * GUARD_BYTES,), GUARD_PATTERN, dtype=torch.uint8, device=device)
    registry.append((base, int(nbytes)))
    return base[GUARD_BYTES:GUARD_BYTES + int(nbytes)]


def guarded_empty(shape, dtype, device, registry: list):
    """An uninitialised-looking tensor (filled with the guard pattern) of `shape` and `dtype` between guard bands."""
    import torch
    n = int(np.prod(shape)) * torch.empty((), dtype=dtype).element_size()
    return guarded_bytes(n, device, registry).view(dtype).view(tuple(shape))


def check_guards(registry: list) -> None:
    """Asserts that no guard band of `registry` was written."""
    import torch
    torch.cuda.synchronize()
    for base, n in registry:
        for band in (base[:GUARD_BYTES], base[GUARD_BYTES + n:]):
            bad = torch.nonzero(band != GUARD_PATTERN)
            assert bad.numel() == 0, f"guard band of a {n}-byte buffer written at byte {int(bad[0, 0])}"


def run_in_child(module: str, func: str, args=(), env=None, timeout=1200) -> None:
    """Runs tests/<module>.<func>(*args) in a fresh Python process with extra environment variables, for
    settings the library reads once, when it is loaded; fails with the child's output if the child fails."""
    import os
    import subprocess
    import sys
    tests = os.path.dirname(os.path.abspath(__file__))
    root = os.path.dirname(tests)
    code = f"import sys; sys.path[:0] = [{root!r}, {tests!r}]; import {module} as m; m.{func}(*{tuple(args)!r})"
    e = dict(os.environ)
    e.update(env or {})
    r = subprocess.run([sys.executable, "-c", code], env=e, capture_output=True, text=True, timeout=timeout)
    assert r.returncode == 0, (r.stdout[-3000:] + "\n" + r.stderr[-6000:])


def to_device(t: "synth.IOTensor"):
    import torch
    if t.io == "f32":
        return torch.from_numpy(np.ascontiguousarray(t.raw)).cuda()
    return torch.from_numpy(np.ascontiguousarray(t.raw).view(np.int16)).cuda().view(torch.bfloat16)


def to_host(x) -> np.ndarray:
    import torch
    return x.detach().to(torch.float64).cpu().numpy()


class Case:
    def __init__(self, B, H, n, d, M, L, io, causal=False, seed=0, qkv_scale=1.0, len_range=None, hidden=64,
                 eps=1e-6, dv=None, with_grad=False, lengths=None, shared=False, ch_rms_target=0.0, signed=False,
                 params=None, per_head=False, act="relu", envelope=False, bank_coef=False):
        self.B, self.H, self.n, self.d, self.M, self.L = B, H, n, d, M, L
        self.act, self.envelope, self.bank_coef = act, envelope, bank_coef
        self.ch_rms_target = ch_rms_target
        self.signed = signed
        self.per_head = per_head
        self.dv = dv or d
        self.io, self.causal, self.eps, self.hidden, self.shared = io, causal, eps, hidden, shared
        if params is None and per_head:  # one parameter set per head, each from its own seed
            sets = [synth.phi_params(seed * 1000 + h, d, M, L, hidden, shared) for h in range(H)]
            params = {k: np.stack([s[k] for s in sets]) for k in sets[0]}
        self.params = params if params is not None else synth.phi_params(seed, d, M, L, hidden, shared)
        if envelope and "We" not in self.params:  # gate pre-activations We_l . x of standard deviation 2
            w_scale = 2.0 / (qkv_scale * math.sqrt(d))
            self.params = {**self.params,
                           "We": (synth.normal(seed, "case.We", (L, d)) * w_scale).astype(np.float32),
                           "be": synth.normal(seed, "case.be", (L,)).astype(np.float32)}
        if bank_coef and "coef" not in self.params:  # coefficients in [0.25, ~3): kernel values stay positive
            self.params = {**self.params,
                           "coef": (0.25 + np.abs(synth.normal(seed, "case.coef", (L,)))).astype(np.float32)}
        self.inp = synth.attn_inputs(seed, B, H, n, d, self.dv, io, qkv_scale, len_range, with_grad)
        if lengths is not None:
            self.inp["lengths"] = np.asarray(lengths, dtype=np.int32)
        self.lengths = self.inp["lengths"]

    # ---- device side
    def luna(self, chunk=0):
        """The library object for this case, its table, workspace and state buffers between guard bands."""
        import torch
        import paper_2512_08061_gb300.luna as L
        lu = L.Luna(self.B, self.H, self.n, self.d, self.dv, self.M, self.L, self.hidden, self.causal, self.eps,
                    torch.float32 if self.io == "f32" else torch.bfloat16, chunk, shared=self.shared,
                    ch_rms_target=self.ch_rms_target, signed=self.signed, per_head=self.per_head, act=self.act,
                    envelope=self.envelope, bank_coef=self.bank_coef)
        self.guards = []
        for name in ("table", "ws", "state"):
            setattr(lu, name, guarded_bytes(getattr(lu, name).numel(), lu.device, self.guards))
        params = {k: torch.from_numpy(v).cuda() for k, v in self.params.items()}
        lu.prepare(params)
        self.dev = {k: to_device(self.inp[k]) for k in ("Q", "K", "V", "dO") if k in self.inp}
        self.dev["lengths"] = None if self.lengths is None else torch.from_numpy(self.lengths).cuda()
        check_guards(self.guards)
        return lu

    def run_fwd(self, lu, save_state=True):
        d = self.dev
        O = guarded_empty(tuple(d["V"].shape), d["V"].dtype, d["V"].device, self.guards)
        out = lu.forward(d["Q"], d["K"], d["V"], d["lengths"], O=O, save_state=save_state)
        check_guards(self.guards)
        return out

    def run_bwd(self, lu, use_state=True):
        import torch
        d = self.dev
        dev = d["Q"].device
        fc1 = (self.hidden,) if self.shared else (self.L, self.hidden)
        g = (self.H,) if self.per_head else ()
        shapes = {"dQ": (tuple(d["Q"].shape), d["Q"].dtype), "dK": (tuple(d["K"].shape), d["K"].dtype),
                  "dV": (tuple(d["V"].shape), d["V"].dtype), "dW": (g + (self.M, self.d), torch.float32),
                  "db": (g + (self.M,), torch.float32), "dw1": (g + fc1, torch.float32),
                  "db1": (g + fc1, torch.float32), "dw2": (g + (self.L, self.hidden), torch.float32),
                  "db2": (g + (self.L,), torch.float32)}
        if self.envelope:
            shapes.update(dWe=((self.L, self.d), torch.float32), dbe=((self.L,), torch.float32))
        if self.bank_coef:
            shapes["dcoef"] = ((self.L,), torch.float32)
        out = {k: guarded_empty(shp, dt, dev, self.guards) for k, (shp, dt) in shapes.items()}
        g = lu.backward(d["Q"], d["K"], d["V"], d["dO"], d["lengths"], use_state=use_state, out=out)
        check_guards(self.guards)
        return g

    # ---- oracle side
    @property
    def phi(self):
        """The oracle's feature map: the parameters, with the channel normalisation and the signed
        channel outputs when they are on."""
        if self.ch_rms_target or self.signed or self.per_head or self.variant:
            return oracle.PhiParams(self.params, self.ch_rms_target, nonneg=not self.signed, act=self.act)
        return self.params

    @property
    def variant(self) -> bool:
        return self.act != "relu" or self.envelope or self.bank_coef

    def oracle_fwd(self):
        i = self.inp
        return oracle.attn_fwd(self.phi, i["Q"].value, i["K"].value, i["V"].value, self.lengths, self.causal,
                               self.eps)

    def oracle_bwd(self):
        i = self.inp
        return oracle.attn_bwd(self.phi, i["Q"].value, i["K"].value, i["V"].value, i["dO"].value, self.lengths,
                               self.causal, self.eps)

    def smooth_rows(self, which: str) -> np.ndarray:
        """Rows whose feature map has no ReLU argument within rounding distance of
        its kink: there the gradient is unique at fp32 resolution."""
        return oracle.kink_margin(self.phi, self.inp[which].value) > KINK_MARGIN
