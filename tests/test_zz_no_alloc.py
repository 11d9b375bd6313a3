"""luna_attn_fwd_noalloc: the forward pass for callers that cannot allocate
device memory.

Such a caller is handed only its input and output tensors (for example an
operator inside an inference engine whose device memory is planned before it
runs), so it cannot supply the workspace that luna_attn_fwd needs.  The
no-allocation entry point keeps its scratch in a library-owned static device
array instead.  Through the C ABI, its outputs must match luna_attn_fwd's on
two calls in a row (the second call must not see the first call's scratch),
and problems larger than the array must be rejected before any launch.
"""
import math

import numpy as np
import pytest

from cases import TOL, Case, relerr, to_host

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2512_08061_gb300 import build
    build.build()


def _noalloc_forward(case, lu):
    import torch
    import paper_2512_08061_gb300.luna as L
    d = case.dev
    O = torch.full_like(d["V"], float("nan"))
    L.luna_attn_fwd_noalloc(lu.ad, lu.pd, lu.table, d["Q"], d["K"], d["V"], d["lengths"], O)
    return to_host(O)


def test_noalloc_forward_matches_workspace_forward_on_two_calls():
    first = Case(4, 2, 1000, 32, 8, 8, "bf16", False, seed=31, qkv_scale=1 / math.sqrt(32),
                 lengths=[1000, 640, 999, 1])
    second = Case(2, 3, 300, 64, 8, 8, "f32", False, seed=37, qkv_scale=1 / math.sqrt(64), lengths=[300, 123])
    for case in (first, second):
        lu = case.luna()
        ref = to_host(case.run_fwd(lu, save_state=False))
        got = _noalloc_forward(case, lu)
        assert np.all(np.isfinite(got))
        assert relerr(got, ref) < TOL[case.io]
        assert relerr(got, case.oracle_fwd()) < TOL[case.io]
        for b, ln in enumerate(case.lengths):
            assert np.all(got[b, :, ln:] == 0)


def test_noalloc_rejects_problems_beyond_the_scratch_array():
    import torch
    import paper_2512_08061_gb300.luna as L
    ad = L.attn_desc(64, 16, 65536, 128, 128, False, 0, 1e-6, L.LUNA_BF16)
    pd = L.phi_desc(16, 8, 64)
    assert L.luna_workspace_size(ad, pd, False) > L.NOALLOC_SCRATCH_BYTES
    dummy = torch.empty(256, dtype=torch.uint8, device="cuda")
    with pytest.raises(L.LunaError) as e:
        L.luna_attn_fwd_noalloc(ad, pd, dummy, dummy, dummy, dummy, None, dummy)
    assert e.value.status == 3  # LUNA_ERR_WORKSPACE, returned before any launch


def test_noalloc_status_word_reports_a_timed_out_wait():
    """The status word at the start of the scratch array is read through
    luna_noalloc_scratch + luna_device_status: a bounded wait that ran out in
    that array (the self-test) is reported once, and the next no-allocation
    call clears the word and computes as before."""
    import paper_2512_08061_gb300.luna as L
    case = Case(2, 2, 300, 32, 8, 8, "bf16", False, seed=43, qkv_scale=1 / math.sqrt(32), lengths=[300, 77])
    lu = case.luna()
    first = _noalloc_forward(case, lu)
    scratch, nbytes = L.luna_noalloc_scratch()
    assert scratch != 0 and nbytes == L.NOALLOC_SCRATCH_BYTES
    assert L.luna_device_status(scratch) == 0
    L.luna_selftest_wait(scratch, 10_000_000)
    assert L.luna_device_status(scratch) == 5  # LUNA_ERR_DEVICE_TIMEOUT
    assert L.luna_device_status(scratch) == 0  # read once, then cleared
    again = _noalloc_forward(case, lu)
    assert np.array_equal(first, again)
    assert L.luna_device_status(scratch) == 0
