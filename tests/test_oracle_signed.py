"""Pins of the oracle's signed channel outputs (the listing's ScalarMLP with
nonneg = False: no outer ReLU, so features and kernel values can be negative).

Checked by a closed-form special case, by the reduction to the default map
where every channel output is positive anyway, by the brute-force quadratic
form of Eq. (kernel-attn), by the Gram matrix (still positive semi-definite:
an inner product of real feature vectors, now of either sign), and by
central finite differences of every gradient.
"""
import math

import numpy as np
import pytest

import oracle
import synth


def _params(seed, d, M, L, hid, shared=False):
    return {k: v.astype(np.float64) for k, v in synth.phi_params(seed, d, M, L, hid, shared).items()}


def _inputs(seed, B, H, n, d, dv, scale=1.0):
    Q = synth.normal(seed, "s.Q", (B, H, n, d)) * scale
    K = synth.normal(seed, "s.K", (B, H, n, d)) * scale
    V = synth.normal(seed, "s.V", (B, H, n, dv))
    dO = synth.normal(seed, "s.dO", (B, H, n, dv))
    return Q, K, V, dO


def test_signed_special_case():
    """hidden = 1, w1 = 1, b1 = 0, w2 = 1, b2 = -1/2, W = I, b = 0: psi(u) = relu(u) - 1/2,
    so phi(x) = (relu(x) - 1/2) / sqrt(d) without the outer ReLU and relu(relu(x) - 1/2) / sqrt(d)
    with it."""
    d = 5
    p = {"W": np.eye(d), "b": np.zeros(d), "w1": np.ones((1, 1)), "b1": np.zeros((1, 1)),
         "w2": np.ones((1, 1)), "b2": np.full(1, -0.5)}
    X = synth.normal(17, "s.X", (13, d))
    y = np.maximum(X, 0) - 0.5
    np.testing.assert_allclose(oracle.featmap(oracle.PhiParams(p, nonneg=False), X), y / math.sqrt(d), rtol=0,
                               atol=1e-15)
    np.testing.assert_allclose(oracle.featmap(p, X), np.maximum(y, 0) / math.sqrt(d), rtol=0, atol=1e-15)


@pytest.mark.parametrize("causal", [False, True])
def test_positive_outputs_reduce_to_the_default_map(causal):
    """With every channel output positive (fc2 bias raised well above the MLP's range) the
    outer ReLU never acts: outputs and gradients equal the default map's exactly."""
    d, M, L, hid = 8, 4, 8, 16
    p = _params(18, d, M, L, hid)
    p["b2"] = p["b2"] + 10.0
    Q, K, V, dO = _inputs(18, 2, 2, 20, d, 3)
    lengths = np.array([20, 9], dtype=np.int32)
    ps = oracle.PhiParams(p, nonneg=False)
    assert oracle.featmap(ps, Q).min() > 0
    assert np.array_equal(oracle.attn_fwd(ps, Q, K, V, lengths, causal), oracle.attn_fwd(p, Q, K, V, lengths, causal))
    g1, g0 = oracle.attn_bwd(ps, Q, K, V, dO, lengths, causal), oracle.attn_bwd(p, Q, K, V, dO, lengths, causal)
    for k in g0:
        assert np.array_equal(g1[k], g0[k]), k


@pytest.mark.parametrize("causal", [False, True])
def test_signed_linear_form_equals_quadratic_form(causal):
    p = oracle.PhiParams(_params(19, 8, 4, 8, 16), nonneg=False)
    Q, K, V, _ = _inputs(19, 2, 2, 30, 8, 4)
    lengths = np.array([30, 12], dtype=np.int32)
    a = oracle.attn_fwd(p, Q, K, V, lengths, causal, 0.3)
    b = oracle.attn_quadratic(p, Q, K, V, lengths, causal, 0.3)
    assert np.max(np.abs(a - b)) < 1e-9 * max(1.0, np.max(np.abs(b)))


def test_signed_gram_matrix_is_psd():
    p = oracle.PhiParams(_params(20, 8, 4, 8, 16), nonneg=False)
    X = synth.normal(20, "s.G", (40, 8))
    phi = oracle.featmap(p, X)
    G = phi @ phi.T
    assert phi.min() < 0  # negative features: the outer ReLU is off
    assert np.linalg.eigvalsh(G).min() > -1e-10 * np.abs(G).max()


@pytest.mark.parametrize("causal", [False, True])
def test_signed_gradients_match_finite_differences(causal):
    d, M, L, hid, n = 3, 2, 2, 3, 6
    seed = 21 + (1 if causal else 0)
    p = _params(seed, d, M, L, hid)
    Q, K, V, dO = _inputs(seed, 2, 1, n, d, 2, scale=1.5)
    lengths = np.array([n, 4], dtype=np.int32)
    eps = 1.0  # signed kernel values: keep every normaliser away from zero
    ps = oracle.PhiParams(p, nonneg=False)
    g = oracle.attn_bwd(ps, Q, K, V, dO, lengths, causal, eps)
    mq, mk = oracle.kink_margin(ps, Q), oracle.kink_margin(ps, K)
    h = 1e-6
    checked = 0

    def loss():
        return float(np.sum(oracle.attn_fwd(oracle.PhiParams(p, nonneg=False), Q, K, V, lengths, causal, eps) * dO))

    def fd(base):
        nonlocal checked
        flat = base.reshape(-1)
        out = np.empty_like(flat)
        for e in range(flat.size):
            x0 = flat[e]
            flat[e] = x0 + h
            lp = loss()
            flat[e] = x0 - h
            lm = loss()
            flat[e] = x0
            out[e] = (lp - lm) / (2 * h)
            checked += 1
        return out.reshape(base.shape)

    for name, arr, margin in (("dQ", Q, mq), ("dK", K, mk), ("dV", V, None)):
        num, ana = fd(arr), g[name]
        if margin is not None:
            ok = margin > 1e-3
            num, ana = num[ok], ana[ok]
        np.testing.assert_allclose(ana, num, rtol=2e-5, atol=2e-7 * max(1.0, np.abs(num).max()), err_msg=name)
    if min(mq.min(), mk.min()) > 1e-4:
        for name, key in (("dW", "W"), ("db", "b"), ("dw1", "w1"), ("db1", "b1"), ("dw2", "w2"), ("db2", "b2")):
            num = fd(p[key])
            np.testing.assert_allclose(g[name], num, rtol=2e-5, atol=2e-7 * max(1.0, np.abs(num).max()),
                                       err_msg=name)
    assert checked > 50
