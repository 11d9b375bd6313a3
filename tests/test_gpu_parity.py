"""GPU parity: the CUDA path through the C ABI against the fp64 oracle on the
same seeded inputs, at sizes that span several tiles and a ragged tail.

Tolerances (max element-wise relative error, floored at the tensor's rms):
1e-4 for fp32 I/O (fp32 arithmetic throughout) and 2e-2 for bf16 I/O (bf16
tensor-core operands, fp32 accumulation).
"""
import math

import numpy as np
import pytest

import oracle
import synth
from cases import (TOL, Case, check_guards, guarded_bytes, guarded_empty, relerr, relerr_rows, run_in_child, to_device,
                   to_host)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2512_08061_gb300 import build
    build.build()


# --------------------------------------------------------------------------
# feature map

@pytest.mark.parametrize("io,d,M", [("f32", 32, 8), ("bf16", 64, 8), ("f32", 128, 16), ("bf16", 128, 16)])
def test_featmap(io, d, M):
    import torch
    import paper_2512_08061_gb300.luna as L
    params = synth.phi_params(3, d, M, 8, 64)
    X = synth.IOTensor(synth.normal(3, "fm.X", (1037, d)), io)
    pd = L.phi_desc(M, 8, 64)
    table = L.alloc_bytes(L.luna_phi_table_size(pd, d), "cuda")
    L.luna_phi_prepare(pd, d, {k: torch.from_numpy(v).cuda() for k, v in params.items()}, table)
    Phi = torch.empty(1037, M * 8, dtype=torch.float32, device="cuda")
    L.luna_featmap(pd, d, table, to_device(X), Phi)
    ref = oracle.featmap(params, X.value)
    assert relerr(to_host(Phi), ref) < 1e-4
    assert torch.all(Phi >= 0)


def test_featmap_exact_at_kinks():
    """Inputs placed exactly on (and one ulp around) the hidden-unit kinks: the
    piecewise-linear table is continuous there and matches direct evaluation."""
    import torch
    import paper_2512_08061_gb300.luna as L
    d = M = 4
    Lc, hid = 8, 64
    params = synth.phi_params(5, d, M, Lc, hid)
    params["W"] = np.eye(d, dtype=np.float32)
    params["b"] = np.zeros(d, dtype=np.float32)
    t = (-params["b1"] / params["w1"]).astype(np.float32).ravel()
    t = t[np.isfinite(t) & (np.abs(t) < 50)]
    vals = np.concatenate([t, np.nextafter(t, np.float32(np.inf)), np.nextafter(t, np.float32(-np.inf))])
    vals = np.resize(vals, (len(vals) + 3) // 4 * 4).astype(np.float32)
    X = vals.reshape(-1, d)
    pd = L.phi_desc(M, Lc, hid)
    table = L.alloc_bytes(L.luna_phi_table_size(pd, d), "cuda")
    L.luna_phi_prepare(pd, d, {k: torch.from_numpy(np.ascontiguousarray(v)).cuda() for k, v in params.items()}, table)
    Phi = torch.empty(X.shape[0], M * Lc, dtype=torch.float32, device="cuda")
    L.luna_featmap(pd, d, table, torch.from_numpy(X).cuda(), Phi)
    ref = oracle.featmap(params, X.astype(np.float64))
    assert relerr(to_host(Phi), ref) < 1e-5


# --------------------------------------------------------------------------
# forward

FWD_CASES = [
    # B, H, n, d, M, io, causal, len_range / lengths
    dict(B=1, H=1, n=256, d=64, M=8, io="f32", causal=False),                  # the 256-token fp32 workload
    dict(B=2, H=3, n=300, d=32, M=8, io="bf16", causal=False, lengths=[300, 177]),
    dict(B=3, H=2, n=197, d=64, M=8, io="bf16", causal=False),                 # ViT-like ragged length
    dict(B=1, H=2, n=333, d=128, M=16, io="bf16", causal=False, lengths=[260]),
    dict(B=2, H=1, n=129, d=32, M=8, io="f32", causal=False, lengths=[1, 0]),
    dict(B=1, H=2, n=300, d=32, M=8, io="f32", causal=True),
    dict(B=2, H=2, n=270, d=64, M=8, io="bf16", causal=True, lengths=[270, 100]),
    dict(B=1, H=1, n=400, d=128, M=16, io="bf16", causal=True),
    dict(B=1, H=1, n=200, d=128, M=16, io="f32", causal=True),
]


def _case_id(c):
    return f"{c['io']}-{'causal' if c['causal'] else 'full'}-B{c['B']}H{c['H']}n{c['n']}d{c['d']}M{c['M']}"


@pytest.mark.parametrize("c", FWD_CASES, ids=_case_id)
def test_forward(c):
    case = Case(c["B"], c["H"], c["n"], c["d"], c["M"], 8, c["io"], c["causal"], seed=7,
                qkv_scale=1.0 / math.sqrt(c["d"]), lengths=c.get("lengths"))
    lu = case.luna()
    O = to_host(case.run_fwd(lu))
    ref = case.oracle_fwd()
    err = relerr_rows(O, ref) if c["causal"] else relerr(O, ref)  # causal rows differ in scale
    assert err < TOL[c["io"]]
    if case.lengths is not None:
        for b, ln in enumerate(case.lengths):
            assert np.all(O[b, :, ln:] == 0)


@pytest.mark.parametrize("tiles", ["1", "5", "9"])
@pytest.mark.parametrize("d,M", [(32, 8), (64, 8), (128, 16)])
def test_forward_tensor_core_tile_loops(d, M, tiles, monkeypatch):
    """bf16 forward through the tensor-core kernels with 1, 5 and 9 tiles of
    128 rows per block: covers the staging ring wrapping around, ragged last
    tiles, splits with no valid row, and several splits per head."""
    monkeypatch.setenv("LUNA_TC_TILES_PER_SPLIT", tiles)
    case = Case(2, 2, 1500, d, M, 8, "bf16", False, seed=41, qkv_scale=1.0 / math.sqrt(d),
                lengths=[1500, 333])
    lu = case.luna()
    O = to_host(case.run_fwd(lu))
    ref = case.oracle_fwd()
    assert relerr(O, ref) < TOL["bf16"]
    assert np.all(O[1, :, 333:] == 0)


@pytest.mark.parametrize("seg_rows", ["128", "384", "1280"])
def test_forward_tensor_core_causal(seg_rows):
    """Streaming form through the tensor-core kernels (d = 128, M = 16): state
    segments of 1, 3 and 9 tiles (the running state carried across tiles in
    TMEM), a ragged last tile, a sequence with padding and segments that hold
    no valid row.  The library reads the segment length once, when it is
    loaded, so each length runs in a process of its own."""
    run_in_child("test_gpu_parity", "check_forward_tensor_core_causal", env={"LUNA_CAUSAL_SEG_ROWS": seg_rows})


def check_forward_tensor_core_causal():
    case = Case(2, 2, 1100, 128, 16, 8, "bf16", True, seed=59, qkv_scale=1.0 / math.sqrt(128),
                lengths=[1100, 333])
    lu = case.luna()
    O = to_host(case.run_fwd(lu))
    ref = case.oracle_fwd()
    assert relerr_rows(O, ref) < TOL["bf16"]
    assert np.all(O[1, :, 333:] == 0)


# --------------------------------------------------------------------------
# backward

BWD_CASES = [
    dict(B=1, H=1, n=256, d=64, M=8, io="f32", causal=False),
    dict(B=2, H=3, n=300, d=32, M=8, io="bf16", causal=False, lengths=[300, 177]),
    dict(B=1, H=2, n=197, d=64, M=8, io="bf16", causal=False),
    dict(B=1, H=2, n=160, d=128, M=16, io="bf16", causal=False),
    dict(B=1, H=2, n=300, d=32, M=8, io="f32", causal=True),
    dict(B=2, H=1, n=270, d=64, M=8, io="bf16", causal=True, lengths=[270, 100]),
    dict(B=1, H=1, n=200, d=128, M=16, io="bf16", causal=True),
]


@pytest.mark.parametrize("c", BWD_CASES, ids=_case_id)
def test_backward(c):
    case = Case(c["B"], c["H"], c["n"], c["d"], c["M"], 8, c["io"], c["causal"], seed=11,
                qkv_scale=1.0 / math.sqrt(c["d"]), lengths=c.get("lengths"), with_grad=True)
    lu = case.luna()
    case.run_fwd(lu)
    g = {k: to_host(v) for k, v in case.run_bwd(lu).items()}
    ref = case.oracle_bwd()
    tol = TOL[c["io"]]
    okq, okk = case.smooth_rows("Q"), case.smooth_rows("K")
    assert okq.mean() > 0.9 and okk.mean() > 0.9
    assert relerr(g["dQ"][okq], ref["dQ"][okq]) < tol
    assert relerr(g["dK"][okk], ref["dK"][okk]) < tol
    assert relerr(g["dV"], ref["dV"]) < tol
    for k in ("dQ", "dK", "dV"):
        assert np.all(np.isfinite(g[k]))
    for k in ("dW", "db", "dw1", "db1", "dw2", "db2"):
        assert relerr(g[k], ref[k]) < tol, k
    if case.lengths is not None:
        for b, ln in enumerate(case.lengths):
            for k in ("dQ", "dK", "dV"):
                assert np.all(g[k][b, :, ln:] == 0)


@pytest.mark.parametrize("seed", [21, 22, 23, 24])
@pytest.mark.parametrize("causal,d,lengths", [(False, 64, None), (False, 32, [300, 123]), (True, 32, [300, 201])])
def test_backward_fp32_parameter_gradients(seed, causal, d, lengths):
    """fp32 I/O: every parameter gradient within the plain 1e-4 gate on several
    seeds.  These gradients are sums over every row, projection and channel
    whose terms cancel to a few hundredths of a percent of their absolute sum
    (the loss barely changes under a common scale of the features)."""
    case = Case(len(lengths) if lengths else 1, 2, 300, d, 8, 8, "f32", causal, seed=seed,
                qkv_scale=1.0 / math.sqrt(d), lengths=lengths, with_grad=True)
    lu = case.luna()
    case.run_fwd(lu)
    g = {k: to_host(v) for k, v in case.run_bwd(lu).items()}
    ref = case.oracle_bwd()
    for k in ("dW", "db", "dw1", "db1", "dw2", "db2"):
        assert relerr(g[k], ref[k]) < TOL["f32"], k


def _check_bwd(case, g, ref, tol):
    okq, okk = case.smooth_rows("Q"), case.smooth_rows("K")
    assert okq.mean() > 0.9 and okk.mean() > 0.9
    assert relerr(g["dQ"][okq], ref["dQ"][okq]) < tol
    assert relerr(g["dK"][okk], ref["dK"][okk]) < tol
    assert relerr(g["dV"], ref["dV"]) < tol
    for k in ("dW", "db", "dw1", "db1", "dw2", "db2"):
        assert relerr(g[k], ref[k]) < tol, k


@pytest.mark.parametrize("tiles", ["1", "3", "5"])
@pytest.mark.parametrize("d", [32, 64])
def test_backward_tensor_core_tile_loops(d, tiles, monkeypatch):
    """bf16 backward through the tensor-core kernels (d = 32 and d = 64, M = 8)
    with 1, 3 and 5 tiles of 128 rows per work item: per-head runs that span
    several blocks and blocks that span several heads, the staging rings
    wrapping around, ragged last tiles and items with no valid row."""
    monkeypatch.setenv("LUNA_TC_TILES_PER_SPLIT", tiles)
    case = Case(2, 3, 1100, d, 8, 8, "bf16", False, seed=43, qkv_scale=1.0 / math.sqrt(d),
                lengths=[1100, 290], with_grad=True)
    lu = case.luna()
    case.run_fwd(lu)
    g = {k: to_host(v) for k, v in case.run_bwd(lu).items()}
    _check_bwd(case, g, case.oracle_bwd(), TOL["bf16"])
    for k in ("dQ", "dK", "dV"):
        assert np.all(g[k][1, :, 290:] == 0)


def test_backward_tensor_core_hidden_32():
    """Tensor-core backward with a shorter kink list (hidden = 32: 256 kinks,
    257 intervals), so the histogram is smaller than its maximum size."""
    case = Case(1, 2, 400, 32, 8, 8, "bf16", False, seed=47, qkv_scale=1.0 / math.sqrt(32),
                with_grad=True, hidden=32)
    lu = case.luna()
    case.run_fwd(lu)
    g = {k: to_host(v) for k, v in case.run_bwd(lu).items()}
    _check_bwd(case, g, case.oracle_bwd(), TOL["bf16"])


@pytest.mark.parametrize("d,lengths", [(32, None), (64, None), (32, [700, 333])])
def test_backward_tensor_core_repeat_bitwise(d, lengths):
    """dQ, dK and dV of the tensor-core backward do not depend on the order of
    floating-point atomics, so repeated runs agree bit for bit (d = 32 and 64,
    and with padded sequences, whose work items are split by valid tiles)."""
    case = Case(2, 2, 700, d, 8, 8, "bf16", False, seed=53, with_grad=True, lengths=lengths)
    lu = case.luna()
    case.run_fwd(lu)
    g1 = {k: to_host(v) for k, v in case.run_bwd(lu).items()}
    g2 = {k: to_host(v) for k, v in case.run_bwd(lu).items()}
    for k in ("dQ", "dK", "dV"):
        assert np.array_equal(g1[k], g2[k]), k


@pytest.mark.parametrize("d,tiles", [(32, "1"), (32, "4"), (64, "2")])
def test_backward_tensor_core_balanced_split(d, tiles, monkeypatch):
    """Work items split over the persistent grid by valid tiles: sequences of
    length 0, 1, a tile minus one, one, plus one, half and full in one batch,
    so that whole runs of items hold no tile, every block must still get an
    item, and one head's items spread over several blocks (partial slots and
    the last-block reduction of each head).  The output rows past each length
    are zeroed by the split launch."""
    monkeypatch.setenv("LUNA_TC_TILES_PER_SPLIT", tiles)
    lengths = [1500, 0, 1, 127, 128, 129, 750, 1499]
    case = Case(len(lengths), 2, 1500, d, 8, 8, "bf16", False, seed=89, qkv_scale=1.0 / math.sqrt(d),
                lengths=lengths, with_grad=True)
    lu = case.luna()
    O = to_host(case.run_fwd(lu))
    ref_O = case.oracle_fwd()
    assert relerr(O, ref_O) < TOL["bf16"]
    g = {k: to_host(v) for k, v in case.run_bwd(lu).items()}
    ref = case.oracle_bwd()
    okq, okk = case.smooth_rows("Q"), case.smooth_rows("K")
    for k, ok in (("dQ", okq), ("dK", okk), ("dV", None)):
        got, want = (g[k], ref[k]) if ok is None else (g[k][ok], ref[k][ok])
        assert relerr(got, want) < TOL["bf16"], k
    for k in ("dW", "db", "dw1", "db1", "dw2", "db2"):
        assert relerr(g[k], ref[k]) < TOL["bf16"], k
    for b, ln in enumerate(lengths):
        assert np.all(O[b, :, ln:] == 0)
        for k in ("dQ", "dK", "dV"):
            assert np.all(g[k][b, :, ln:] == 0), (k, b)


@pytest.mark.parametrize("d,M,causal", [(32, 8, False), (64, 8, False), (128, 16, True)])
def test_backward_tensor_core_histogram_ranges(d, M, causal):
    """The fixed-point interval histogram of the channel-MLP gradient
    statistics when the output gradient is zero on the first 300 rows of every
    sequence (no scale until a later tile) and then grows by four orders of
    magnitude along the sequence, so that every group of tiles outgrows the
    scales taken from the group before it and its large values go to the
    unscaled fallback.  One work item per head (18 tiles of 128 rows), so that
    a block walks more than one group (16 tiles of 128 rows x 8 projections,
    8 tiles of 128 x 16).  Runs in a process of its own with the segment length
    set (the library reads it once, when it is loaded)."""
    run_in_child("test_gpu_parity", "check_backward_histogram_ranges", (d, M, causal),
                 env={"LUNA_TC_TILES_PER_SPLIT": "18", "LUNA_CAUSAL_SEG_ROWS": "2304"})


def check_backward_histogram_ranges(d, M, causal):
    n = 2200
    case = Case(2, 2, n, d, M, 8, "bf16", causal, seed=83, qkv_scale=1.0 / math.sqrt(d), with_grad=True)
    ramp = 10.0 ** (4.0 * np.arange(n) / n)
    ramp[:300] = 0.0
    case.inp["dO"] = synth.IOTensor(case.inp["dO"].value * ramp[None, None, :, None], "bf16")
    lu = case.luna()
    case.run_fwd(lu)
    g = {k: to_host(v) for k, v in case.run_bwd(lu).items()}
    _check_bwd(case, g, case.oracle_bwd(), TOL["bf16"])


@pytest.mark.parametrize("seg_rows", ["128", "384", "1280"])
def test_backward_tensor_core_causal(seg_rows):
    """Streaming-form backward through the tensor-core kernels (d = 128, M = 16):
    state segments of 2, 6 and 20 tiles of 64 rows (the running S and dS carried
    across tiles in TMEM, the reverse scan of the segment sums), ragged last
    tiles, a sequence with padding and segments that hold no valid row.  One
    process per segment length (read once, when the library is loaded)."""
    run_in_child("test_gpu_parity", "check_backward_tensor_core_causal", env={"LUNA_CAUSAL_SEG_ROWS": seg_rows})


def check_backward_tensor_core_causal():
    case = Case(2, 2, 1100, 128, 16, 8, "bf16", True, seed=61, qkv_scale=1.0 / math.sqrt(128),
                lengths=[1100, 333], with_grad=True)
    lu = case.luna()
    case.run_fwd(lu)
    g = {k: to_host(v) for k, v in case.run_bwd(lu).items()}
    _check_bwd(case, g, case.oracle_bwd(), TOL["bf16"])
    for k in ("dQ", "dK", "dV"):
        assert np.all(np.isfinite(g[k]))
        assert np.all(g[k][1, :, 333:] == 0)


@pytest.mark.parametrize("n,lengths", [(2, None), (63, None), (65, [65, 1]), (130, [0, 129])])
def test_backward_tensor_core_causal_edges(n, lengths):
    """Streaming-form tensor-core backward on the edges of its 64-row tiles: a
    two-row sequence, one row short of and one past a tile, and sequences of
    length 0 and 1 in a batch (no valid row in a segment).  (The first row of a
    sequence attends to itself alone: O_0 = v_0 up to eps, and its dphi(q) and
    dphi(k) are eps-level remainders of an exact cancellation, below fp32
    resolution of the cancelling parts; with one row per sequence the whole
    dQ and dK would be such remainders, so the shortest case here has two.)"""
    B = 1 if lengths is None else len(lengths)
    case = Case(B, 2, n, 128, 16, 8, "bf16", True, seed=73, qkv_scale=1.0 / math.sqrt(128), lengths=lengths,
                with_grad=True)
    lu = case.luna()
    case.run_fwd(lu)
    g = {k: to_host(v) for k, v in case.run_bwd(lu).items()}
    ref = case.oracle_bwd()
    okq, okk = case.smooth_rows("Q"), case.smooth_rows("K")
    for k, ok in (("dQ", okq), ("dK", okk), ("dV", None)):
        assert np.all(np.isfinite(g[k]))
        got, want = (g[k], ref[k]) if ok is None else (g[k][ok], ref[k][ok])
        assert relerr(got, want) < TOL["bf16"], k
    for k in ("dW", "db", "dw1", "db1", "dw2", "db2"):
        assert relerr(g[k], ref[k]) < TOL["bf16"], k
    if lengths is not None:
        for b, ln in enumerate(lengths):
            for k in ("dQ", "dK", "dV"):
                assert np.all(g[k][b, :, ln:] == 0)


def test_backward_tensor_core_causal_state_and_repeat():
    """The tensor-core streaming-form backward gives the same bits with the
    forward's saved segment prefixes as without them, and on a repeated run."""
    case = Case(1, 2, 700, 128, 16, 8, "bf16", True, seed=67, qkv_scale=1.0 / math.sqrt(128),
                with_grad=True)
    lu = case.luna()
    case.run_fwd(lu)
    a = {k: to_host(v) for k, v in case.run_bwd(lu, use_state=True).items()}
    b = {k: to_host(v) for k, v in case.run_bwd(lu, use_state=False).items()}
    c = {k: to_host(v) for k, v in case.run_bwd(lu, use_state=False).items()}
    for k in ("dQ", "dK", "dV"):
        assert np.array_equal(a[k], b[k]), k
        assert np.array_equal(b[k], c[k]), k


@pytest.mark.parametrize("causal", [False, True])
def test_backward_with_and_without_saved_state(causal):
    case = Case(2, 2, 200, 32, 8, 8, "f32", causal, seed=13, with_grad=True, lengths=[200, 150])
    lu = case.luna()
    case.run_fwd(lu)
    a = {k: to_host(v) for k, v in case.run_bwd(lu, use_state=True).items()}
    b = {k: to_host(v) for k, v in case.run_bwd(lu, use_state=False).items()}
    for k in a:
        assert relerr(a[k], b[k]) < 1e-5, k


@pytest.mark.parametrize("causal", [False, True])
def test_repeat_runs_are_bitwise_identical(causal):
    case = Case(2, 2, 300, 64, 8, 8, "bf16", causal, seed=17, with_grad=True)
    lu = case.luna()
    O1 = to_host(case.run_fwd(lu))
    g1 = {k: to_host(v) for k, v in case.run_bwd(lu).items()}
    O2 = to_host(case.run_fwd(lu))
    g2 = {k: to_host(v) for k, v in case.run_bwd(lu).items()}
    assert np.array_equal(O1, O2)
    for k in ("dQ", "dK", "dV"):
        assert np.array_equal(g1[k], g2[k]), k


def test_all_padded_and_empty():
    import torch
    case = Case(2, 1, 64, 32, 8, 8, "f32", False, seed=19, with_grad=True, lengths=[0, 0])
    lu = case.luna()
    O = to_host(case.run_fwd(lu))
    assert np.all(O == 0)
    g = case.run_bwd(lu)
    for k, v in g.items():
        assert torch.all(v == 0), k
    # B = 0: a successful no-op that still defines the parameter gradients
    empty = Case(0, 1, 64, 32, 8, 8, "f32", False, seed=19, with_grad=True)
    lu = empty.luna()
    g = empty.run_bwd(lu)
    for k in ("dW", "db", "dw1", "db1", "dw2", "db2"):
        assert torch.all(g[k] == 0)


def test_unit_values_give_unit_outputs():
    """V = 1 and eps = 0: every row with a positive normaliser outputs exactly 1
    up to rounding (row-wise normalisation of Eq. kernel-attn)."""
    import torch
    case = Case(1, 2, 300, 32, 8, 8, "f32", False, seed=23, eps=0.0)
    lu = case.luna()
    case.dev["V"] = torch.ones_like(case.dev["V"])
    O = to_host(case.run_fwd(lu))
    nz = np.any(O != 0, axis=-1)
    assert nz.mean() > 0.9
    assert np.max(np.abs(O[nz] - 1.0)) < 1e-5


@pytest.mark.parametrize("io,d,dv,M", [("bf16", 128, 128, 16), ("f32", 64, 64, 8), ("f32", 64, 32, 8)])
def test_decode_continues_the_streaming_form(io, d, dv, M):
    """Recurrent decode (luna_attn_decode): a causal forward over the first
    tokens of each (padded) sequence saves its state; three decode steps then
    feed the tokens that follow each sequence's last valid one.  Each step's
    output equals the oracle's causal output at that position of the extended
    sequence (streaming form, Sec. 3.2)."""
    import torch
    import paper_2512_08061_gb300.luna as L
    B, H, n0, T = 3, 2, 300, 3
    lens = [300, 177, 0]  # the last sequence starts from an empty state
    case = Case(B, H, n0 + T, d, M, 8, io, True, seed=71, qkv_scale=1.0 / math.sqrt(d), dv=dv,
                lengths=[ln + T for ln in lens])
    dt = torch.float32 if io == "f32" else torch.bfloat16
    lu = L.Luna(B, H, n0, d, dv, M, 8, 64, True, case.eps, dt)
    lu.prepare({k: torch.from_numpy(v).cuda() for k, v in case.params.items()})
    full = {k: to_device(case.inp[k]) for k in ("Q", "K", "V")}
    pre = {k: v[:, :, :n0].contiguous() for k, v in full.items()}
    lu.forward(pre["Q"], pre["K"], pre["V"], torch.tensor(lens, dtype=torch.int32, device="cuda"), save_state=True)
    outs = []
    for t in range(T):
        tok = {k: torch.stack([v[b, :, lens[b] + t] for b in range(B)]).contiguous() for k, v in full.items()}
        outs.append(to_host(lu.decode(tok["Q"], tok["K"], tok["V"])))
    ref = case.oracle_fwd()
    tol = TOL[io]
    for t in range(T):
        want = np.stack([ref[b, :, lens[b] + t] for b in range(B)])
        assert relerr_rows(outs[t], want) < tol, t


def test_bounded_wait_reports_timeout_and_context_stays_usable():
    """Failure path of the bounded device waits: a wait on a barrier phase that
    nothing completes gives up after 10 ms and sets the workspace's status word;
    luna_device_status reports LUNA_ERR_DEVICE_TIMEOUT once and clears it, and
    the same context then computes the same results as before."""
    import paper_2512_08061_gb300.luna as L
    case = Case(1, 2, 256, 64, 8, 8, "f32", False, seed=3)
    lu = case.luna()
    O1 = to_host(case.run_fwd(lu))
    assert L.luna_device_status(lu.ws) == 0
    L.luna_selftest_wait(lu.ws, 10_000_000)
    assert L.luna_device_status(lu.ws) == 5  # LUNA_ERR_DEVICE_TIMEOUT
    assert L.luna_device_status(lu.ws) == 0  # read once, then cleared
    O2 = to_host(case.run_fwd(lu))
    assert np.array_equal(O1, O2)
    assert L.luna_device_status(lu.ws) == 0


@pytest.mark.parametrize("io,d,M,causal", [("bf16", 32, 8, False), ("f32", 64, 8, True), ("bf16", 128, 16, True),
                                           ("bf16", 64, 8, False)])
def test_shared_channel_mlp(io, d, M, causal):
    """The listing's shared_channels option (one MLP with L outputs): forward and
    backward through the tensor-core path (bf16 non-causal d = 32 and 64, the
    streaming form at d = 128) and the generic path (fp32), every gradient
    including dw1, db1 of the one shared fc1 (summed over the channels)."""
    case = Case(2, 2, 300, d, M, 8, io, causal, seed=79, qkv_scale=1.0 / math.sqrt(d), lengths=[300, 177],
                with_grad=True, shared=True)
    lu = case.luna()
    O = to_host(case.run_fwd(lu))
    ref = case.oracle_fwd()
    assert (relerr_rows(O, ref) if causal else relerr(O, ref)) < TOL[io]
    g = {k: to_host(v) for k, v in case.run_bwd(lu).items()}
    rb = case.oracle_bwd()
    okq, okk = case.smooth_rows("Q"), case.smooth_rows("K")
    assert relerr(g["dQ"][okq], rb["dQ"][okq]) < TOL[io]
    assert relerr(g["dK"][okk], rb["dK"][okk]) < TOL[io]
    assert relerr(g["dV"], rb["dV"]) < TOL[io]
    assert g["dw1"].shape == (64,) and g["db1"].shape == (64,)
    for k in ("dW", "db", "dw1", "db1", "dw2", "db2"):
        assert relerr(g[k], rb[k]) < TOL[io], k


def test_shared_channel_featmap():
    """luna_featmap of the shared-channel MLP against the oracle, with the
    kinks of the one fc1 (64 kinks, 65 intervals)."""
    import torch
    import paper_2512_08061_gb300.luna as L
    d, M = 64, 8
    params = synth.phi_params(83, d, M, 8, 64, shared=True)
    X = synth.IOTensor(synth.normal(83, "fms.X", (777, d)), "f32")
    pd = L.phi_desc(M, 8, 64, shared=True)
    table = L.alloc_bytes(L.luna_phi_table_size(pd, d), "cuda")
    L.luna_phi_prepare(pd, d, {k: torch.from_numpy(v).cuda() for k, v in params.items()}, table)
    Phi = torch.empty(777, M * 8, dtype=torch.float32, device="cuda")
    L.luna_featmap(pd, d, table, to_device(X), Phi)
    assert relerr(to_host(Phi), oracle.featmap(params, X.value)) < 1e-4


def _median_channel_rms(case):
    """A target between the channels' RMS values: some channels clamped, some not."""
    p = oracle.PhiParams(case.params, 1.0)
    rq = oracle.ch_rms(p, case.inp["Q"].value, case.lengths)[1]
    rk = oracle.ch_rms(p, case.inp["K"].value, case.lengths)[1]
    return float(np.median(np.concatenate([rq, rk])))


@pytest.mark.parametrize("io,d,M,lengths,causal", [("bf16", 32, 8, [300, 177], False), ("bf16", 64, 8, None, False),
                                                   ("bf16", 128, 16, [300, 1], False), ("f32", 16, 4, [300, 41], False),
                                                   ("bf16", 128, 16, [300, 250], True), ("f32", 16, 4, [300, 41], True),
                                                   ("bf16", 64, 8, None, True)])
def test_channel_rms_normalisation(io, d, M, lengths, causal):
    """The listing's ch_rms option: statistics over all valid query rows and all
    valid key rows, forward and backward (with the dependence of the scales on
    every sample).  Non-causal: the tensor-core path (bf16 d = 32 and 64), the
    generic backward on tensor-core statistics (bf16 d = 128) and the generic
    path (fp32).  Streaming form: the tensor-core kernels (bf16 d = 128) and the
    generic ones (fp32; bf16 d = 64), on the table scaled by sqrt(s^q s^k).  The
    backward with the forward's saved state and with the statistics
    recomputed."""
    case = Case(2, 2, 300, d, M, 8, io, causal, seed=91, qkv_scale=1.0 / math.sqrt(d), lengths=lengths,
                with_grad=True)
    case.ch_rms_target = _median_channel_rms(case)
    lu = case.luna()
    O = to_host(case.run_fwd(lu))
    ref = case.oracle_fwd()
    assert (relerr_rows(O, ref) if causal else relerr(O, ref)) < TOL[io]
    okq, okk = case.smooth_rows("Q"), case.smooth_rows("K")
    assert okq.mean() > 0.9 and okk.mean() > 0.9
    rb = case.oracle_bwd()
    for use_state in (True, False):
        g = {k: to_host(v) for k, v in case.run_bwd(lu, use_state=use_state).items()}
        assert relerr(g["dQ"][okq], rb["dQ"][okq]) < TOL[io], use_state
        assert relerr(g["dK"][okk], rb["dK"][okk]) < TOL[io], use_state
        assert relerr(g["dV"], rb["dV"]) < TOL[io], use_state
        for k in ("dW", "db", "dw1", "db1", "dw2", "db2"):
            assert relerr(g[k], rb[k]) < TOL[io], (k, use_state)
        if case.lengths is not None:
            for b, ln in enumerate(case.lengths):
                for k in ("dQ", "dK", "dV"):
                    assert np.all(g[k][b, :, ln:] == 0)


@pytest.mark.parametrize("d", [32, 64])
def test_channel_rms_normalisation_many_tiles(d):
    """The non-causal channel normalisation on the tensor-core statistics and scale-term passes with
    more tiles than blocks (each block of a side takes several, some none), ragged lengths that end
    inside a tile and an empty sequence; the scale term adds into dQ and dK, whose padded rows must
    stay zero."""
    case = Case(4, 4, 1400, d, 8, 8, "bf16", False, seed=93, qkv_scale=1.0 / math.sqrt(d),
                lengths=[1400, 1029, 0, 130], with_grad=True)
    case.ch_rms_target = _median_channel_rms(case)
    lu = case.luna()
    O = to_host(case.run_fwd(lu))
    assert relerr(O, case.oracle_fwd()) < TOL["bf16"]
    okq, okk = case.smooth_rows("Q"), case.smooth_rows("K")
    rb = case.oracle_bwd()
    g = {k: to_host(v) for k, v in case.run_bwd(lu).items()}
    assert relerr(g["dQ"][okq], rb["dQ"][okq]) < TOL["bf16"]
    assert relerr(g["dK"][okk], rb["dK"][okk]) < TOL["bf16"]
    assert relerr(g["dV"], rb["dV"]) < TOL["bf16"]
    for k in ("dW", "db", "dw1", "db1", "dw2", "db2"):
        assert relerr(g[k], rb[k]) < TOL["bf16"], k
    for b, ln in enumerate(case.lengths):
        for k in ("dQ", "dK", "dV"):
            assert np.all(g[k][b, :, ln:] == 0)


# --------------------------------------------------------------------------
# attention weights of a block of query rows (conversion, stage 1)

@pytest.mark.parametrize("teacher", [False, True])
@pytest.mark.parametrize("io,d,M,causal,lengths,row0,rows", [
    ("f32", 64, 8, False, [300, 177], 0, 300),
    ("bf16", 32, 8, False, [300, 1], 37, 70),
    ("f32", 128, 16, True, [300, 250], 100, 131),
    ("bf16", 64, 8, True, None, 250, 50),
])
def test_attention_weights(io, d, M, causal, lengths, row0, rows, teacher):
    """luna_attn_weights against the oracle's weights: LUNA's normalised kernel
    weights (whose product with V is the attention output) and the softmax
    teacher's, for a window of query rows with ragged 32-row blocks, padded
    sequences (including a one-token one), causal and not; masked entries and
    padded rows exactly zero, every row a distribution."""
    import torch
    import paper_2512_08061_gb300.luna as L
    case = Case(2, 2, 300, d, M, 8, io, causal, seed=97, qkv_scale=1.0 / math.sqrt(d), lengths=lengths)
    lu = case.luna()
    A = torch.full((2, 2, rows, 300), float("nan"), dtype=torch.float32, device="cuda")
    L.luna_attn_weights(lu.ad, lu.pd, lu.table, case.dev["Q"], case.dev["K"], case.dev["lengths"], row0, rows,
                        teacher, A)
    got = to_host(A)
    i = case.inp
    ref = oracle.attn_weights(case.params, i["Q"].value, i["K"].value, case.lengths, causal, case.eps, row0, rows,
                              teacher)
    assert np.all(np.isfinite(got))
    assert np.array_equal(got == 0, ref == 0)  # the same masked keys and padded rows
    assert relerr(got, ref) < TOL[io]
    s = got.sum(-1)
    live = ref.sum(-1) > 0
    assert np.allclose(s[live], 1.0, atol=1e-4)


def test_attention_weights_times_values_is_the_forward():
    """The weights of every row times V equals luna_attn_fwd's output (fp32)."""
    import torch
    import paper_2512_08061_gb300.luna as L
    case = Case(1, 2, 200, 32, 8, 8, "f32", False, seed=101, qkv_scale=1.0 / math.sqrt(32), lengths=[150])
    lu = case.luna()
    O = to_host(case.run_fwd(lu))
    A = torch.empty((1, 2, 200, 200), dtype=torch.float32, device="cuda")
    L.luna_attn_weights(lu.ad, lu.pd, lu.table, case.dev["Q"], case.dev["K"], case.dev["lengths"], 0, 200, False, A)
    AV = to_host(A) @ case.inp["V"].value
    assert relerr(AV, O) < 1e-4


# --------------------------------------------------------------------------
# signed channel outputs (the listing's nonneg = False)

def _signed_params(seed, d, M, L=8, hidden=64, shift=0.5):
    """Random-init parameters with fc2's bias raised by `shift`: most channel outputs positive, some
    negative, so the kernel's row sums stay away from zero while the signed path is exercised."""
    p = synth.phi_params(seed, d, M, L, hidden)
    p["b2"] = (p["b2"] + np.float32(shift)).astype(np.float32)
    return p


@pytest.mark.parametrize("io,d,M,causal,lengths", [("bf16", 32, 8, False, [300, 177]), ("bf16", 64, 8, False, None),
                                                   ("bf16", 128, 16, True, [300, 250]), ("f32", 32, 8, False, [300, 9]),
                                                   ("f32", 32, 8, True, None)])
def test_signed_channel_outputs(io, d, M, causal, lengths):
    """Signed channel outputs (no outer ReLU) through the tensor-core kernels
    (bf16 non-causal d = 32 and 64, the streaming form at d = 128) and the
    generic ones (fp32, causal and not), forward and backward, against the
    oracle's nonneg = False; some features must be negative for the case to
    mean anything."""
    params = _signed_params(103, d, M)
    case = Case(2, 2, 300, d, M, 8, io, causal, seed=103, qkv_scale=1.0 / math.sqrt(d), lengths=lengths,
                with_grad=True, signed=True, params=params)
    phiq = oracle.featmap(case.phi, case.inp["Q"].value)
    assert 0.01 < np.mean(phiq < 0) < 0.5
    lu = case.luna()
    O = to_host(case.run_fwd(lu))
    ref = case.oracle_fwd()
    assert (relerr_rows(O, ref) if causal else relerr(O, ref)) < TOL[io]
    g = {k: to_host(v) for k, v in case.run_bwd(lu).items()}
    rb = case.oracle_bwd()
    okq, okk = case.smooth_rows("Q"), case.smooth_rows("K")
    assert okq.mean() > 0.9 and okk.mean() > 0.9
    assert relerr(g["dQ"][okq], rb["dQ"][okq]) < TOL[io]
    assert relerr(g["dK"][okk], rb["dK"][okk]) < TOL[io]
    assert relerr(g["dV"], rb["dV"]) < TOL[io]
    for k in ("dW", "db", "dw1", "db1", "dw2", "db2"):
        assert relerr(g[k], rb[k]) < TOL[io], k


def test_signed_channel_featmap_and_decode():
    """luna_featmap and the decode step with signed channel outputs."""
    import torch
    import paper_2512_08061_gb300.luna as L
    d, M = 64, 8
    params = _signed_params(107, d, M)
    X = synth.IOTensor(synth.normal(107, "sg.X", (777, d)), "f32")
    pd = L.phi_desc(M, 8, 64, signed=True)
    table = L.alloc_bytes(L.luna_phi_table_size(pd, d), "cuda")
    L.luna_phi_prepare(pd, d, {k: torch.from_numpy(v).cuda() for k, v in params.items()}, table)
    Phi = torch.empty(777, M * 8, dtype=torch.float32, device="cuda")
    L.luna_featmap(pd, d, table, to_device(X), Phi)
    ref = oracle.featmap(oracle.PhiParams(params, nonneg=False), X.value)
    assert np.mean(ref < 0) > 0.01
    assert relerr(to_host(Phi), ref) < 1e-4
    # one decode step after a causal prefill of 40 tokens equals the causal output of token 41
    n = 41
    case = Case(2, 2, n, d, M, 8, "f32", True, seed=109, qkv_scale=1.0 / math.sqrt(d), signed=True, params=params)
    full = case.oracle_fwd()
    pre = Case(2, 2, n - 1, d, M, 8, "f32", True, seed=109, qkv_scale=1.0 / math.sqrt(d), signed=True,
               params=params)
    for k in ("Q", "K", "V"):
        pre.inp[k] = synth.IOTensor(case.inp[k].value[:, :, :n - 1], "f32")
    lu = pre.luna()
    pre.run_fwd(lu, save_state=True)
    tok = {k: torch.from_numpy(np.ascontiguousarray(case.inp[k].value[:, :, n - 1]).astype(np.float32)).cuda()
           for k in ("Q", "K", "V")}
    o = to_host(lu.decode(tok["Q"], tok["K"], tok["V"]))
    assert relerr(o, full[:, :, n - 1]) < 1e-4


# --------------------------------------------------------------------------
# per-head feature-map parameters (the conversion's per-layer, per-head instantiation)

@pytest.mark.parametrize("io,d,M,causal,lengths,H", [
    ("bf16", 32, 8, False, [300, 177, 1], 3),   # tensor-core non-causal, d = 32 (LRA shape)
    ("bf16", 64, 8, False, None, 4),            # tensor-core non-causal, d = 64 (BERT / ViT shape)
    ("bf16", 128, 16, True, [300, 250], 2),     # tensor-core streaming form, d = 128
    ("f32", 32, 8, False, [300, 41], 3),        # generic kernels
    ("f32", 32, 8, True, [300, 200], 2),
])
def test_per_head_parameters(io, d, M, causal, lengths, H):
    """Head h of every sequence uses its own W, b and channel MLPs: forward and
    backward against the oracle's per-head mode, each head's parameter
    gradients summed over the batch only, with the state saved by the forward
    (the library runs one sub-problem per head index over strided views of the
    caller's tensors, state and gradients)."""
    B = len(lengths) if lengths else 2
    case = Case(B, H, 300, d, M, 8, io, causal, seed=113, qkv_scale=1.0 / math.sqrt(d), lengths=lengths,
                with_grad=True, per_head=True)
    assert case.params["W"].shape == (H, M, d)
    lu = case.luna()
    O = to_host(case.run_fwd(lu))
    ref = case.oracle_fwd()
    assert (relerr_rows(O, ref) if causal else relerr(O, ref)) < TOL[io]
    g = {k: to_host(v) for k, v in case.run_bwd(lu).items()}
    rb = case.oracle_bwd()
    okq, okk = case.smooth_rows("Q"), case.smooth_rows("K")
    assert okq.mean() > 0.9 and okk.mean() > 0.9
    assert relerr(g["dQ"][okq], rb["dQ"][okq]) < TOL[io]
    assert relerr(g["dK"][okk], rb["dK"][okk]) < TOL[io]
    assert relerr(g["dV"], rb["dV"]) < TOL[io]
    for k in ("dW", "db", "dw1", "db1", "dw2", "db2"):
        assert g[k].shape[0] == H
        for h in range(H):
            assert relerr(g[k][h], rb[k][h]) < TOL[io], (k, h)
    if lengths is not None:
        for b, ln in enumerate(lengths):
            for k in ("dQ", "dK", "dV"):
                assert np.all(g[k][b, :, ln:] == 0)


def test_per_head_parameters_decode_and_weights():
    """The decode step and the attention weights read the table of their own head."""
    import torch
    import paper_2512_08061_gb300.luna as L
    d, M, H, n = 64, 8, 3, 41
    case = Case(2, H, n, d, M, 8, "f32", True, seed=127, qkv_scale=1.0 / math.sqrt(d), per_head=True)
    full = case.oracle_fwd()
    pre = Case(2, H, n - 1, d, M, 8, "f32", True, seed=127, qkv_scale=1.0 / math.sqrt(d), per_head=True,
               params=case.params)
    for k in ("Q", "K", "V"):
        pre.inp[k] = synth.IOTensor(case.inp[k].value[:, :, :n - 1], "f32")
    lu = pre.luna()
    pre.run_fwd(lu, save_state=True)
    tok = {k: torch.from_numpy(np.ascontiguousarray(case.inp[k].value[:, :, n - 1]).astype(np.float32)).cuda()
           for k in ("Q", "K", "V")}
    o = to_host(lu.decode(tok["Q"], tok["K"], tok["V"]))
    assert relerr(o, full[:, :, n - 1]) < 1e-4
    lu2 = case.luna()
    A = torch.empty((2, H, n, n), dtype=torch.float32, device="cuda")
    L.luna_attn_weights(lu2.ad, lu2.pd, lu2.table, case.dev["Q"], case.dev["K"], None, 0, n, False, A)
    ref = oracle.attn_weights(case.phi, case.inp["Q"].value, case.inp["K"].value, None, True, case.eps)
    assert relerr(to_host(A), ref) < 1e-4


# the feature-map variants: (activation, envelope gate, Bank+Coef, shared-channel MLP)
VARIANTS = {
    "gelu": ("gelu", False, False, False),
    "silu": ("silu", False, False, False),
    "tanh": ("tanh", False, False, False),
    "tanh-shared": ("tanh", False, False, True),
    "envelope": ("relu", True, False, False),
    "coef": ("relu", False, True, False),
    "gelu+envelope+coef": ("gelu", True, True, False),
}


@pytest.mark.parametrize("io,causal", [("f32", False), ("f32", True), ("bf16", False), ("bf16", True)])
@pytest.mark.parametrize("name", sorted(VARIANTS))
def test_feature_map_variants(name, io, causal):
    """The kernel ablation's feature maps (Sec. 5.4, Table 5) and the channel MLPs' activation on the
    generic kernels, forward and backward (every parameter gradient, the gate's and the coefficients'
    included), against the oracle: direct evaluation of GELU / SiLU / tanh MLPs, the envelope gate
    sigmoid(We x + be) and the Bank+Coef coefficients; ragged lengths over several 16- and 32-row
    tiles."""
    act, env, coef, shared = VARIANTS[name]
    d, M = 32, 8
    seed = 300 + sorted(VARIANTS).index(name)
    case = Case(2, 2, 150, d, M, 8, io, causal, seed=seed, qkv_scale=1.0 / math.sqrt(d), lengths=[150, 71],
                with_grad=True, shared=shared, act=act, envelope=env, bank_coef=coef)
    phiq = oracle.featmap(case.phi, case.inp["Q"].value)
    assert np.mean(phiq > 0) > 0.1  # the map is not dead
    lu = case.luna()
    O = to_host(case.run_fwd(lu))
    ref = case.oracle_fwd()
    assert (relerr_rows(O, ref) if causal else relerr(O, ref)) < TOL[io]
    g = {k: to_host(v) for k, v in case.run_bwd(lu).items()}
    rb = case.oracle_bwd()
    okq, okk = case.smooth_rows("Q"), case.smooth_rows("K")
    assert okq.mean() > 0.9 and okk.mean() > 0.9
    assert relerr(g["dQ"][okq], rb["dQ"][okq]) < TOL[io]
    assert relerr(g["dK"][okk], rb["dK"][okk]) < TOL[io]
    assert relerr(g["dV"], rb["dV"]) < TOL[io]
    keys = ["dW", "db", "dw1", "db1", "dw2", "db2"] + (["dWe", "dbe"] if env else []) + (["dcoef"] if coef else [])
    for k in keys:
        assert relerr(g[k], rb[k]) < TOL[io], k


@pytest.mark.parametrize("name", sorted(VARIANTS))
def test_feature_map_variants_featmap(name):
    """luna_featmap of every variant, fp32 and bf16 rows, against the oracle's feature map."""
    import torch
    import paper_2512_08061_gb300.luna as L
    act, env, coef, shared = VARIANTS[name]
    d, M = 64, 8
    seed = 320 + sorted(VARIANTS).index(name)
    case = Case(1, 1, 8, d, M, 8, "f32", seed=seed, qkv_scale=1.0 / math.sqrt(d), shared=shared, act=act,
                envelope=env, bank_coef=coef)
    pd = L.phi_desc(M, 8, 64, shared, act=act, envelope=env, bank_coef=coef)
    guards = []
    table = guarded_bytes(L.luna_phi_table_size(pd, d), "cuda", guards)
    L.luna_phi_prepare(pd, d, {k: torch.from_numpy(v).cuda() for k, v in case.params.items()}, table)
    for io in ("f32", "bf16"):
        X = synth.IOTensor(synth.normal(seed, "var.X", (333, d)) / math.sqrt(d), io)
        Phi = guarded_empty((333, M * 8), torch.float32, "cuda", guards)
        L.luna_featmap(pd, d, table, to_device(X), Phi)
        check_guards(guards)
        ref = oracle.featmap(case.phi, X.value)
        assert relerr(to_host(Phi), ref) < 1e-4, io


@pytest.mark.parametrize("causal", [False, True])
def test_feature_map_variants_many_blocks(causal):
    """Every variant at once on a longer ragged problem: many work splits per head, so the
    gate's, the coefficients' and the directly summed MLP gradients are reduced over many
    block partials (fp32 I/O, the plain 1e-4 gate)."""
    d, M = 32, 8
    case = Case(2, 3, 1100, d, M, 8, "f32", causal, seed=340, qkv_scale=1.0 / math.sqrt(d), lengths=[1100, 613],
                with_grad=True, act="silu", envelope=True, bank_coef=True)
    lu = case.luna()
    O = to_host(case.run_fwd(lu))
    ref = case.oracle_fwd()
    assert (relerr_rows(O, ref) if causal else relerr(O, ref)) < TOL["f32"]
    g = {k: to_host(v) for k, v in case.run_bwd(lu).items()}
    rb = case.oracle_bwd()
    okq, okk = case.smooth_rows("Q"), case.smooth_rows("K")
    assert relerr(g["dQ"][okq], rb["dQ"][okq]) < TOL["f32"]
    assert relerr(g["dK"][okk], rb["dK"][okk]) < TOL["f32"]
    assert relerr(g["dV"], rb["dV"]) < TOL["f32"]
    for k in ("dW", "db", "dw1", "db1", "dw2", "db2", "dWe", "dbe", "dcoef"):
        assert relerr(g[k], rb[k]) < TOL["f32"], k
