"""GPU parity at the full sizes of the benchmark workloads, in the launch
configuration bench.py times: the same descriptor, the same seeded inputs,
the forward pass saving its state and the backward pass reusing it.

The oracle checks every head of lra, bert, vit and tiny_f32 (a few seconds on
the host cores).  At causal_long (4.2 M rows of d = 128) it checks O, dQ, dK
and dV on two heads (the first and the last; about 12 s each) and the
feature-map parameter gradients, which sum over every head, against the
oracle run over all heads in chunks.  The decode workload checks every head's
output after the causal prefill against the oracle's causal row at that
position.
"""
import math
import os
import sys

import numpy as np
import pytest

import oracle
import synth
from cases import TOL, relerr, relerr_rows, to_host

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

pytestmark = pytest.mark.gpu

KINK_MARGIN = 1e-5


@pytest.fixture(scope="module", autouse=True)
def _lib():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2512_08061_gb300 import build
    build.build()


def _device(t):
    import torch
    if t.io == "f32":
        return torch.from_numpy(np.ascontiguousarray(t.raw)).cuda()
    return torch.from_numpy(np.ascontiguousarray(t.raw).view(np.int16)).cuda().view(torch.bfloat16)


def _run_like_bench(w):
    """The bench's step on the workload: prepare, forward (state saved), backward (state reused)."""
    import torch
    import bench
    import paper_2512_08061_gb300.luna as L
    inp, params = bench.host_inputs(w)
    io = torch.float32 if w.io == "f32" else torch.bfloat16
    dev = {k: _device(inp[k]) for k in ("Q", "K", "V", "dO") if k in inp}
    lengths = None if inp["lengths"] is None else torch.from_numpy(inp["lengths"]).cuda()
    lu = L.Luna(w.B, w.H, w.n, w.d, w.dv, w.M, w.L, w.hidden, w.causal, w.eps, io, w.chunk)
    lu.prepare({k: torch.from_numpy(v).cuda() for k, v in params.items()})
    O = lu.forward(dev["Q"], dev["K"], dev["V"], lengths, save_state=True)
    g = None
    if w.backward:
        g = lu.backward(dev["Q"], dev["K"], dev["V"], dev["dO"], lengths, use_state=True)
    torch.cuda.synchronize()
    return inp, params, O, g


def _head_slice(inp, b, h):
    """The (1, 1, n, .) fp64 inputs of head (b, h) and its length."""
    sl = {k: inp[k].value[b:b + 1, h:h + 1] for k in ("Q", "K", "V", "dO") if k in inp}
    ln = None if inp["lengths"] is None else np.asarray(inp["lengths"][b:b + 1], dtype=np.int32)
    return sl, ln


@pytest.mark.parametrize("name", ["tiny_f32", "lra", "bert", "vit"])
def test_full_size_every_head(name):
    from synth.workloads import WORKLOADS
    w = WORKLOADS[name]
    inp, params, O, g = _run_like_bench(w)
    tol = TOL[w.io]
    q, k, v = inp["Q"].value, inp["K"].value, inp["V"].value
    ref_O = oracle.attn_fwd(params, q, k, v, inp["lengths"], w.causal, w.eps)
    assert relerr(to_host(O), ref_O) < tol
    if w.backward:
        ref = oracle.attn_bwd(params, q, k, v, inp["dO"].value, inp["lengths"], w.causal, w.eps)
        got = {key: to_host(val) for key, val in g.items()}
        okq = oracle.kink_margin(params, q) > KINK_MARGIN
        okk = oracle.kink_margin(params, k) > KINK_MARGIN
        assert okq.mean() > 0.9 and okk.mean() > 0.9
        assert relerr(got["dQ"][okq], ref["dQ"][okq]) < tol
        assert relerr(got["dK"][okk], ref["dK"][okk]) < tol
        assert relerr(got["dV"], ref["dV"]) < tol
        for key in ("dW", "db", "dw1", "db1", "dw2", "db2"):
            assert relerr(got[key], ref[key]) < tol, key


def test_full_size_causal_long():
    from synth.workloads import WORKLOADS
    w = WORKLOADS["causal_long"]
    inp, params, O, g = _run_like_bench(w)
    p = oracle.PhiParams(params)
    tol = TOL[w.io]
    got = {key: to_host(g[key]) for key in ("dW", "db", "dw1", "db1", "dw2", "db2")}
    # every output and input gradient of two heads, by the oracle head by head (the GPU's
    # tensors are sliced on the device: the full ones would need 17 GB as fp64 on the host)
    for b, h in ((0, 0), (w.B - 1, w.H - 1)):
        sl, ln = _head_slice(inp, b, h)
        ref_O = oracle.attn_fwd(p, sl["Q"], sl["K"], sl["V"], ln, True, w.eps)
        assert relerr_rows(to_host(O[b:b + 1, h:h + 1]), ref_O) < tol, (b, h)
        ref = oracle.attn_bwd(p, sl["Q"], sl["K"], sl["V"], sl["dO"], ln, True, w.eps)
        okq = oracle.kink_margin(p, sl["Q"]) > KINK_MARGIN
        okk = oracle.kink_margin(p, sl["K"]) > KINK_MARGIN
        assert relerr(to_host(g["dQ"][b:b + 1, h:h + 1])[okq], ref["dQ"][okq]) < tol, (b, h)
        assert relerr(to_host(g["dK"][b:b + 1, h:h + 1])[okk], ref["dK"][okk]) < tol, (b, h)
        assert relerr(to_host(g["dV"][b:b + 1, h:h + 1]), ref["dV"]) < tol, (b, h)
    # parameter gradients: sums over every head, the oracle over chunks of heads
    acc = None
    BH = w.B * w.H
    q4 = inp["Q"].value.reshape(BH, 1, w.n, w.d)
    k4 = inp["K"].value.reshape(BH, 1, w.n, w.d)
    v4 = inp["V"].value.reshape(BH, 1, w.n, w.dv)
    d4 = inp["dO"].value.reshape(BH, 1, w.n, w.dv)
    for c0 in range(0, BH, 16):
        c1 = min(BH, c0 + 16)
        r = oracle.attn_bwd(p, q4[c0:c1], k4[c0:c1], v4[c0:c1], d4[c0:c1], None, True, w.eps)
        part = {key: r[key] for key in ("dW", "db", "dw1", "db1", "dw2", "db2")}
        acc = part if acc is None else {key: acc[key] + part[key] for key in acc}
    for key in ("dW", "db", "dw1", "db1", "dw2", "db2"):
        assert relerr(got[key], acc[key]) < tol, key


def test_full_size_decode():
    """Every head of the decode workload: one step after the 1024-token causal
    prefill equals the oracle's causal output at position 1024."""
    import torch
    import bench
    import paper_2512_08061_gb300.luna as L
    from synth.workloads import WORKLOADS
    w = WORKLOADS["decode"]
    inp, params = bench.host_inputs(w)
    dev = {k: _device(inp[k]) for k in ("Q", "K", "V")}
    lu = L.Luna(w.B, w.H, w.n, w.d, w.dv, w.M, w.L, w.hidden, True, w.eps, torch.bfloat16, w.chunk)
    lu.prepare({k: torch.from_numpy(v).cuda() for k, v in params.items()})
    lu.forward(dev["Q"], dev["K"], dev["V"], None, save_state=True)
    tok = {k: synth.IOTensor(synth.normal(w.seed, f"decode.{k}", (w.B, w.H, n)) * w.qkv_scale, w.io)
           for k, n in (("q", w.d), ("k", w.d), ("v", w.dv))}
    o = to_host(lu.decode(_device(tok["q"]), _device(tok["k"]), _device(tok["v"])))
    # the oracle on the prefill plus the token, every head; only its last row is compared
    full = {k: np.concatenate([inp[K].value, tok[k].value[:, :, None, :]], axis=2)
            for k, K in (("q", "Q"), ("k", "K"), ("v", "V"))}
    ref = oracle.attn_fwd(params, full["q"], full["k"], full["v"], None, True, w.eps)[:, :, -1]
    assert relerr_rows(o, ref) < TOL["bf16"]
