"""Pins of the oracle's per-head feature-map parameters (the conversion
experiments instantiate the feature map per layer and head): head h of every
sequence uses its own W, b and channel MLPs, and each head's parameter
gradients are summed over the batch only.

Checked against the shared-parameter oracle (already pinned by its own
tests): identical heads reduce to it, and every head equals it run on that
head's slice alone; and by central finite differences of the per-head
gradients.
"""
import numpy as np
import pytest

import oracle
import synth


def _params(seed, d, M, L, hid, shared=False):
    return {k: v.astype(np.float64) for k, v in synth.phi_params(seed, d, M, L, hid, shared).items()}


def _stack(ps):
    return {k: np.stack([p[k] for p in ps]) for k in ps[0]}


def _inputs(seed, B, H, n, d, dv, scale=1.0):
    Q = synth.normal(seed, "h.Q", (B, H, n, d)) * scale
    K = synth.normal(seed, "h.K", (B, H, n, d)) * scale
    V = synth.normal(seed, "h.V", (B, H, n, dv))
    dO = synth.normal(seed, "h.dO", (B, H, n, dv))
    return Q, K, V, dO


@pytest.mark.parametrize("causal", [False, True])
def test_identical_heads_are_the_shared_parameters(causal):
    B, H, n, d = 3, 2, 20, 8
    p = _params(60, d, 4, 8, 16)
    Q, K, V, dO = _inputs(60, B, H, n, d, 3)
    lengths = np.array([20, 7, 13], dtype=np.int32)
    ph = _stack([p, p])
    assert np.array_equal(oracle.attn_fwd(ph, Q, K, V, lengths, causal), oracle.attn_fwd(p, Q, K, V, lengths, causal))
    g1, g0 = oracle.attn_bwd(ph, Q, K, V, dO, lengths, causal), oracle.attn_bwd(p, Q, K, V, dO, lengths, causal)
    for k in ("dQ", "dK", "dV"):
        assert np.array_equal(g1[k], g0[k]), k
    for k in ("dW", "db", "dw1", "db1", "dw2", "db2"):
        assert g1[k].shape == (H,) + g0[k].shape
        np.testing.assert_allclose(g1[k].sum(axis=0), g0[k], rtol=1e-12, atol=1e-14 * np.abs(g0[k]).max())


@pytest.mark.parametrize("shared", [False, True])
@pytest.mark.parametrize("causal", [False, True])
def test_every_head_is_the_shared_oracle_on_its_slice(causal, shared):
    """B != H, so a head index taken from the batch position would fail."""
    B, H, n, d = 3, 2, 18, 8
    ps = [_params(61 + h, d, 4, 8, 16, shared) for h in range(H)]
    ph = _stack(ps)
    Q, K, V, dO = _inputs(61, B, H, n, d, 3)
    lengths = np.array([18, 5, 11], dtype=np.int32)
    O = oracle.attn_fwd(ph, Q, K, V, lengths, causal)
    g = oracle.attn_bwd(ph, Q, K, V, dO, lengths, causal)
    for h in range(H):
        sl = (slice(None), slice(h, h + 1))
        assert np.array_equal(O[sl], oracle.attn_fwd(ps[h], Q[sl], K[sl], V[sl], lengths, causal))
        gh = oracle.attn_bwd(ps[h], Q[sl], K[sl], V[sl], dO[sl], lengths, causal)
        for k in ("dQ", "dK", "dV"):
            assert np.array_equal(g[k][sl], gh[k]), (h, k)
        for k in ("dW", "db", "dw1", "db1", "dw2", "db2"):
            assert np.array_equal(g[k][h], gh[k]), (h, k)
    # the per-head feature map and kink margin take head h's rows with head h's parameters
    phi = oracle.featmap(ph, Q)
    for h in range(H):
        assert np.array_equal(phi[:, h], oracle.featmap(ps[h], Q[:, h]))
    assert np.array_equal(oracle.kink_margin(ph, Q)[:, 1], oracle.kink_margin(ps[1], Q[:, 1]))


@pytest.mark.parametrize("causal", [False, True])
def test_per_head_gradients_match_finite_differences(causal):
    B, H, n, d, M, L, hid = 2, 2, 5, 3, 2, 2, 3
    ph = _stack([_params(70 + h + (5 if causal else 0), d, M, L, hid) for h in range(H)])
    Q, K, V, dO = _inputs(70, B, H, n, d, 2, scale=1.5)
    lengths = np.array([5, 3], dtype=np.int32)
    eps = 1e-3
    g = oracle.attn_bwd(ph, Q, K, V, dO, lengths, causal, eps)
    mq, mk = oracle.kink_margin(ph, Q), oracle.kink_margin(ph, K)
    assert min(mq.min(), mk.min()) > 1e-4
    h = 1e-6

    def loss():
        return float(np.sum(oracle.attn_fwd(ph, Q, K, V, lengths, causal, eps) * dO))

    for name, key in (("dW", "W"), ("db", "b"), ("dw1", "w1"), ("db1", "b1"), ("dw2", "w2"), ("db2", "b2")):
        flat = ph[key].reshape(-1)
        num = np.empty_like(flat)
        for e in range(flat.size):
            x0 = flat[e]
            flat[e] = x0 + h
            lp = loss()
            flat[e] = x0 - h
            lm = loss()
            flat[e] = x0
            num[e] = (lp - lm) / (2 * h)
        num = num.reshape(ph[key].shape)
        np.testing.assert_allclose(g[name], num, rtol=2e-5, atol=2e-7 * max(1.0, np.abs(num).max()), err_msg=name)


def test_normalisation_with_per_head_parameters_is_rejected():
    ph = _stack([_params(80, 8, 4, 8, 16), _params(81, 8, 4, 8, 16)])
    with pytest.raises(ValueError):
        oracle.PhiParams(ph, 0.1)
