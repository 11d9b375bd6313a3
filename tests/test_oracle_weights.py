"""Pins of the oracle's attention weights (conversion stage 1: the student's
attention distribution, matched to the softmax teacher's; appendix,
"Stage 1: attention distillation").  The LUNA weights are Eq. (kernel-attn)
read as a weighted average of the values, a_ij = k(q_i,k_j) / (sum_j k + eps),
so their product with V must equal the linear (sufficient-statistics) form,
a different computation in the oracle.  The teacher is checked against the
textbook softmax written out in numpy."""
import math

import numpy as np
import pytest

import oracle
import synth


def _inputs(seed, B, H, n, d, dv, lengths=None):
    inp = synth.attn_inputs(seed, B, H, n, d, dv, "f32", 1.0 / math.sqrt(d), None, False)
    ln = None if lengths is None else np.asarray(lengths, dtype=np.int32)
    return inp["Q"].value, inp["K"].value, inp["V"].value, ln


@pytest.mark.parametrize("causal", [False, True])
@pytest.mark.parametrize("eps", [0.0, 1e-6, 0.3])
def test_weights_times_values_is_the_linear_form(causal, eps):
    p = synth.phi_params(5, 8, 3, 4, 6)
    Q, K, V, ln = _inputs(5, 2, 2, 23, 8, 5, [23, 11])
    A = oracle.attn_weights(p, Q, K, ln, causal, eps)
    O = oracle.attn_fwd(p, Q, K, V, ln, causal, eps)
    assert np.allclose(A @ V, O, rtol=1e-12, atol=1e-14)


def test_weights_are_a_distribution_over_the_valid_keys():
    p = synth.phi_params(7, 8, 3, 4, 6)
    Q, K, V, ln = _inputs(7, 2, 2, 17, 8, 4, [17, 6])
    for causal in (False, True):
        A = oracle.attn_weights(p, Q, K, ln, causal, 0.0)
        assert np.all(A >= 0.0)
        for b, L in enumerate(ln):
            rows = A[b, :, :L]
            s = rows.sum(-1)
            nz = s > 0  # rows whose features are all zero give a zero row
            assert np.allclose(s[nz], 1.0, rtol=1e-13) and nz.mean() > 0.9
            assert np.all(A[b, :, L:] == 0.0) and np.all(A[b, :, :, L:] == 0.0)
            if causal:
                assert np.all(np.triu(A[b, :, :L, :L], 1) == 0.0)


def test_constant_channels_give_uniform_weights():
    """w1 = 0, b1 = 1: every hidden unit outputs 1, so phi is the same for every token and each valid
    query spreads its weight evenly: 1/len (non-causal), 1/(i+1) (causal)."""
    p = synth.phi_params(9, 6, 2, 3, 5)
    p["w1"][:] = 0.0
    p["b1"][:] = 1.0
    p["w2"][:] = 0.25
    Q, K, V, ln = _inputs(9, 1, 1, 12, 6, 3, [10])
    A = oracle.attn_weights(p, Q, K, ln, False, 0.0)[0, 0]
    assert np.allclose(A[:10, :10], 0.1, rtol=1e-14) and np.all(A[10:] == 0) and np.all(A[:, 10:] == 0)
    C = oracle.attn_weights(p, Q, K, ln, True, 0.0)[0, 0]
    for i in range(10):
        assert np.allclose(C[i, :i + 1], 1.0 / (i + 1), rtol=1e-14) and np.all(C[i, i + 1:] == 0)


def test_row_window_is_a_slice_of_the_full_matrix():
    p = synth.phi_params(11, 8, 2, 4, 5)
    Q, K, V, ln = _inputs(11, 2, 1, 30, 8, 4, [30, 19])
    for causal in (False, True):
        for teacher in (False, True):
            full = oracle.attn_weights(p, Q, K, ln, causal, 1e-6, teacher=teacher)
            win = oracle.attn_weights(p, Q, K, ln, causal, 1e-6, row0=7, rows=15, teacher=teacher)
            assert np.array_equal(win, full[:, :, 7:22])
            assert np.all(oracle.attn_weights(p, Q, K, ln, causal, 1e-6, row0=30, rows=3, teacher=teacher) == 0)


@pytest.mark.parametrize("causal", [False, True])
def test_teacher_is_the_scaled_dot_product_softmax(causal):
    p = synth.phi_params(13, 8, 2, 4, 5)
    Q, K, V, ln = _inputs(13, 2, 2, 14, 8, 4, [14, 9])
    T = oracle.attn_weights(p, Q, K, ln, causal, 0.0, teacher=True)
    for b in range(2):
        L = ln[b]
        for h in range(2):
            s = Q[b, h, :L] @ K[b, h, :L].T / math.sqrt(8)
            if causal:
                s = np.where(np.tril(np.ones((L, L), bool)), s, -np.inf)
            e = np.exp(s - s.max(-1, keepdims=True))
            ref = e / e.sum(-1, keepdims=True)
            assert np.allclose(T[b, h, :L, :L], ref, rtol=1e-12, atol=1e-15)
            assert np.all(T[b, h, L:] == 0) and np.all(T[b, h, :, L:] == 0)
    # equal scores: the teacher is uniform over the keys a query sees
    Z = np.zeros_like(Q)
    U = oracle.attn_weights(p, Z, K, None, False, 0.0, teacher=True)
    assert np.allclose(U, 1.0 / 14, rtol=1e-14)
