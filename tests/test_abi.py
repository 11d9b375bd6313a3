"""The C-ABI library loads and exports every entry point that include/luna.h
declares; size queries and argument checks work without a GPU (no compute
call is made here)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    from paper_2512_08061_gb300 import build
    build.build()
    import paper_2512_08061_gb300.luna as L
    return L


def declared_entry_points():
    src = open(os.path.join(ROOT, "include", "luna.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(luna_[a-z_0-9]+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = declared_entry_points()
    for required in ("luna_phi_prepare", "luna_featmap", "luna_attn_fwd", "luna_attn_bwd", "luna_workspace_size",
                     "luna_status_string"):
        assert required in names


def test_every_declared_symbol_is_exported(L):
    lib = ctypes.CDLL(L.library_path())
    for name in declared_entry_points():
        assert hasattr(lib, name), f"{name} declared in include/luna.h but not exported"
    assert set(L.EXPORTED) <= set(declared_entry_points())


def test_status_strings(L):
    assert L.luna_status_string(0) == "LUNA_OK"
    assert L.luna_status_string(5) == "LUNA_ERR_DEVICE_TIMEOUT"
    assert L.luna_version() >= 100


def test_size_queries(L):
    pd = L.phi_desc(8, 8, 64)
    t = L.luna_phi_table_size(pd, 32)
    assert t % 256 == 0 and t > 4 * (512 + 513 * 16)
    ad = L.attn_desc(32, 4, 4096, 32, 32, False, 0, 1e-6, L.LUNA_BF16)
    fwd, bwd = L.luna_workspace_size(ad, pd, False), L.luna_workspace_size(ad, pd, True)
    assert 0 < fwd <= bwd
    assert L.luna_state_size(ad, pd) >= 32 * 4 * (64 * 32 + 64) * 4
    # empty problems need no real workspace
    ad0 = L.attn_desc(0, 4, 4096, 32, 32)
    assert L.luna_workspace_size(ad0, pd, True) == 256


def test_argument_errors_return_before_launch(L):
    pd = L.phi_desc(8, 8, 64)
    with pytest.raises(L.LunaError) as e:
        L.luna_phi_table_size(L.phi_desc(0, 8, 64), 32)
    assert e.value.status == 1
    with pytest.raises(L.LunaError) as e:
        L.luna_phi_table_size(L.phi_desc(8, 8, 128), 32)  # L*hidden > 512
    assert e.value.status == 2
    with pytest.raises(L.LunaError) as e:
        L.luna_workspace_size(L.attn_desc(1, 1, 16, 256, 32), pd, False)  # d > 128
    assert e.value.status == 2
    with pytest.raises(L.LunaError) as e:
        L.luna_workspace_size(L.attn_desc(1, 1, 16, 32, 32, eps=-1.0), pd, False)
    assert e.value.status == 1
    with pytest.raises(L.LunaError) as e:
        L.luna_workspace_size(L.attn_desc(1, 1, 16, 32, 32, chunk=17), pd, False)
    assert e.value.status == 1
    # NULL pointers are rejected before any CUDA call
    lib = L._lib
    ad = L.attn_desc(1, 1, 16, 32, 32)
    st = lib.luna_attn_fwd(ctypes.byref(ad), ctypes.byref(pd), None, None, None, None, None, None, None, None, 0, None)
    assert st == 1
    st = lib.luna_phi_prepare(ctypes.byref(pd), 32, None, None, 0, None)
    assert st == 1
    # an empty problem is a successful no-op
    ad0 = L.attn_desc(1, 1, 0, 32, 32)
    st = lib.luna_attn_fwd(ctypes.byref(ad0), ctypes.byref(pd), None, None, None, None, None, None, None, None, 0,
                           None)
    assert st == 0


def test_decode_arguments_and_state_layout(L):
    """luna_attn_decode and luna_state_final check their arguments before any
    launch; the final causal state sits at segment nseg of each head's block of
    nseg + 1 segment prefixes (S first for all heads, then z)."""
    lib = L._lib
    pd = L.phi_desc(16, 8, 64)
    ad = L.attn_desc(2, 3, 1000, 128, 128, causal=True)
    P, I64 = ctypes.c_void_p, ctypes.c_int64
    # NULL tensors, a too-small stride and a bad eps are rejected
    st = lib.luna_attn_decode(ctypes.byref(ad), ctypes.byref(pd), None, None, None, None, None, None, 0, None, 0, None)
    assert st == 1
    st = lib.luna_attn_decode(ctypes.byref(ad), ctypes.byref(pd), P(256), P(256), P(256), P(256), P(256), P(256),
                              128 * 128 - 1, P(256), 0, None)
    assert st == 1
    bad = L.attn_desc(2, 3, 1000, 128, 128, causal=True, eps=-1.0)
    st = lib.luna_attn_decode(ctypes.byref(bad), ctypes.byref(pd), P(256), P(256), P(256), P(256), P(256), P(256),
                              0, P(256), 0, None)
    assert st == 1
    # B*H = 0 is a no-op
    ad0 = L.attn_desc(0, 3, 1, 128, 128)
    assert lib.luna_attn_decode(ctypes.byref(ad0), ctypes.byref(pd), None, None, None, None, None, None, 0, None, 0,
                                None) == 0
    # state layout: nseg from the state size, S and z offsets of the last segment
    SD, D, BH = 128 * 128, 128, 6
    size = L.luna_state_size(ad, pd)
    nseg1 = size // (4 * BH * (SD + D))
    assert size == 4 * BH * nseg1 * (SD + D)
    base = 1 << 20
    S, Ss, z, zs = (ctypes.c_void_p(), I64(), ctypes.c_void_p(), I64())
    assert lib.luna_state_final(ctypes.byref(ad), ctypes.byref(pd), P(base), ctypes.byref(S), ctypes.byref(Ss),
                                ctypes.byref(z), ctypes.byref(zs)) == 0
    assert Ss.value == nseg1 * SD and zs.value == nseg1 * D
    assert S.value == base + 4 * (nseg1 - 1) * SD
    assert z.value == base + 4 * (BH * nseg1 * SD + (nseg1 - 1) * D)
    nc = L.attn_desc(2, 3, 1000, 128, 128, causal=False)
    assert lib.luna_state_final(ctypes.byref(nc), ctypes.byref(pd), P(base), ctypes.byref(S), ctypes.byref(Ss),
                                ctypes.byref(z), ctypes.byref(zs)) == 1


def test_selftest_wait_arguments(L):
    lib = L._lib
    assert lib.luna_selftest_wait(None, 10_000_000, None) == 1
    assert lib.luna_selftest_wait(ctypes.c_void_p(256), 0, None) == 1
    assert lib.luna_selftest_wait(ctypes.c_void_p(256), 2_000_000_000, None) == 1


def test_shared_channel_descriptor(L):
    """shared_channels must be 0 or 1; the shared-channel table holds the kinks of
    the one fc1 (hidden of them), so it is smaller than the per-channel table."""
    with pytest.raises(L.LunaError) as e:
        pd = L.PhiDesc(8, 8, 64, 2)
        L.luna_phi_table_size(pd, 32)
    assert e.value.status == 1
    per = L.luna_phi_table_size(L.phi_desc(8, 8, 64), 32)
    shared = L.luna_phi_table_size(L.phi_desc(8, 8, 64, shared=True), 32)
    assert 0 < shared < per


def test_channel_rms_descriptor(L):
    """ch_rms_target: 0 is off, a positive value turns the channel normalisation on
    (more workspace: the statistics and the partials of the scale term; the
    streaming form also holds the scaled table), negative, NaN or infinite targets
    are rejected; luna_featmap and luna_attn_decode do not support it (all checked
    before any device call)."""
    lib = L._lib
    for bad in (-0.1, float("nan"), float("inf")):
        with pytest.raises(L.LunaError) as e:
            L.luna_phi_table_size(L.phi_desc(8, 8, 64, ch_rms_target=bad), 32)
        assert e.value.status == 1
    pd0, pd1 = L.phi_desc(8, 8, 64), L.phi_desc(8, 8, 64, ch_rms_target=0.1)
    assert L.luna_phi_table_size(pd0, 32) == L.luna_phi_table_size(pd1, 32)
    ad = L.attn_desc(32, 4, 4096, 32, 32, False, 0, 1e-6, L.LUNA_BF16)
    for bwd in (False, True):
        assert L.luna_workspace_size(ad, pd1, bwd) > L.luna_workspace_size(ad, pd0, bwd)
    assert L.luna_state_size(ad, pd1) == L.luna_state_size(ad, pd0)
    pdc0, pdc1 = L.phi_desc(16, 8, 64), L.phi_desc(16, 8, 64, ch_rms_target=0.1)
    adc = L.attn_desc(2, 4, 1024, 128, 128, True)
    for bwd in (False, True):
        assert L.luna_workspace_size(adc, pdc1, bwd) > L.luna_workspace_size(adc, pdc0, bwd)
    assert lib.luna_featmap(ctypes.byref(pd1), 32, None, None, L.LUNA_F32, 1, None, None) == 2
    dec = L.attn_desc(2, 4, 1, 32, 32, True)
    assert lib.luna_attn_decode(ctypes.byref(dec), ctypes.byref(pd1), None, None, None, None, None, None, 0, None, 0,
                                None) == 2


def test_attention_weights_arguments(L):
    """luna_attn_weights checks its row window, flags and descriptors before any launch; an
    empty window is a no-op."""
    lib = L._lib
    P = ctypes.c_void_p
    pd = L.phi_desc(8, 8, 64)
    ad = L.attn_desc(2, 2, 100, 32, 32)
    args = (P(256), P(256), P(256), None)
    assert lib.luna_attn_weights(ctypes.byref(ad), ctypes.byref(pd), *args, 90, 11, 0, P(256), None) == 1
    assert lib.luna_attn_weights(ctypes.byref(ad), ctypes.byref(pd), *args, -1, 5, 0, P(256), None) == 1
    assert lib.luna_attn_weights(ctypes.byref(ad), ctypes.byref(pd), *args, 0, 5, 2, P(256), None) == 1
    assert lib.luna_attn_weights(ctypes.byref(ad), ctypes.byref(pd), *args, 0, 5, 0, None, None) == 1
    assert lib.luna_attn_weights(ctypes.byref(ad), ctypes.byref(pd), None, P(256), P(256), None, 0, 5, 0, P(256),
                                 None) == 1  # the LUNA weights need the table
    rms = L.phi_desc(8, 8, 64, ch_rms_target=0.1)
    assert lib.luna_attn_weights(ctypes.byref(ad), ctypes.byref(rms), *args, 0, 5, 0, P(256), None) == 2
    assert lib.luna_attn_weights(ctypes.byref(ad), ctypes.byref(pd), None, None, None, None, 100, 0, 0, None,
                                 None) == 0


def test_variant_descriptors(L):
    """The feature-map variants: act in 0..3 and the envelope / bank_coef flags in {0, 1}
    (else LUNA_ERR_INVALID_ARG); the gate's and the coefficients' parameters enlarge the
    table; the variants do not combine with ch_rms or per-head parameters, and
    luna_attn_weights / luna_attn_decode do not support them (all before any launch);
    luna_phi_prepare and luna_attn_bwd require the variants' parameter and gradient
    pointers."""
    lib = L._lib
    P = ctypes.c_void_p
    for kw in ({"act": 4}, {"act": -1}, {"envelope": 2}, {"bank_coef": 3}):
        pd = L.phi_desc(8, 8, 64)
        for k, v in kw.items():
            setattr(pd, k, v)
        with pytest.raises(L.LunaError) as e:
            L.luna_phi_table_size(pd, 32)
        assert e.value.status == 1, kw
    base = L.luna_phi_table_size(L.phi_desc(8, 8, 64), 32)
    assert L.luna_phi_table_size(L.phi_desc(8, 8, 64, act="gelu"), 32) == base
    assert L.luna_phi_table_size(L.phi_desc(8, 8, 64, envelope=True), 32) >= base + 4 * 8 * 32
    assert L.luna_phi_table_size(L.phi_desc(8, 8, 64, bank_coef=True), 32) >= base  # 8 floats: may fit the padding
    for kw in ({"act": "tanh"}, {"envelope": True}, {"bank_coef": True}):
        with pytest.raises(L.LunaError) as e:
            L.luna_phi_table_size(L.phi_desc(8, 8, 64, ch_rms_target=0.1, **kw), 32)
        assert e.value.status == 2, kw
        with pytest.raises(L.LunaError) as e:
            L.luna_phi_table_size(L.phi_desc(8, 8, 64, param_head_stride=1 << 20, **kw), 32)
        assert e.value.status == 2, kw
        pd = L.phi_desc(8, 8, 64, **kw)
        ad = L.attn_desc(2, 2, 100, 32, 32)
        assert lib.luna_attn_weights(ctypes.byref(ad), ctypes.byref(pd), P(256), P(256), P(256), None, 0, 5, 0,
                                     P(256), None) == 2
        dec = L.attn_desc(2, 4, 1, 32, 32, True)
        assert lib.luna_attn_decode(ctypes.byref(dec), ctypes.byref(pd), None, None, None, None, None, None, 0, None,
                                    0, None) == 2
        assert L.luna_workspace_size(ad, pd, True) >= L.luna_workspace_size(ad, pd, False) > 0
    # prepare without the gate's parameters, backward without its gradients: argument errors
    pd = L.phi_desc(8, 8, 64, envelope=True)
    pp = L.PhiParams(*([P(256)] * 6 + [None, None, None]))
    assert lib.luna_phi_prepare(ctypes.byref(pd), 32, ctypes.byref(pp), P(256), 1 << 20, None) == 1
    ad = L.attn_desc(2, 2, 64, 32, 32)
    pg = L.PhiGrads(*([P(256)] * 6 + [None, None, None]))
    assert lib.luna_attn_bwd(ctypes.byref(ad), ctypes.byref(pd), P(256), P(256), P(256), P(256), P(256), None, None,
                             P(256), P(256), P(256), ctypes.byref(pg), P(256), 1 << 30, None) == 1
