"""Pins of the fp64 CPU oracle against what the paper and the mathematics fix.

None of these compares the oracle with itself: each check is a hand-computed
value, a closed form, an invariant of Eq. (kernel-attn), the positive
semi-definiteness of Prop. 1, a brute-force evaluation of a different formula,
or a finite-difference derivative.
"""
import json
import math
import os

import numpy as np
import pytest

import oracle
import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _hand_params():
    g = json.load(open(os.path.join(GOLDEN, "phi_hand.json")))
    p = {k: np.array(g[k], dtype=np.float64) for k in ("W", "b", "w1", "b1", "w2", "b2")}
    return g, p


def _rand_params(seed, d, M, L, hid, shared=False):
    return {k: v.astype(np.float64) for k, v in synth.phi_params(seed, d, M, L, hid, shared).items()}


def _rand_inputs(seed, B, H, n, d, dv, scale=1.0):
    Q = synth.normal(seed, "t.Q", (B, H, n, d)) * scale
    K = synth.normal(seed, "t.K", (B, H, n, d)) * scale
    V = synth.normal(seed, "t.V", (B, H, n, dv))
    return Q, K, V


def _relerr(a, b):
    return float(np.max(np.abs(a - b)) / max(np.max(np.abs(b)), 1e-300))


# --------------------------------------------------------------------------
# feature map

def test_phi_hand_example():
    """Eq. (phi-def-scalarenv) / listing: values worked out by hand."""
    g, p = _hand_params()
    X = np.array(g["X"])
    phi = oracle.featmap(p, X)
    expect = np.array(g["psi_unscaled"]) / math.sqrt(2.0)
    np.testing.assert_allclose(phi, expect, rtol=0, atol=1e-15)


def test_phi_relu_special_case():
    """hidden=1, w1=1, b1=0, w2=1, b2=0, W=I, b=0 gives phi(x) = relu(x)/sqrt(d)."""
    d = 5
    p = {"W": np.eye(d), "b": np.zeros(d), "w1": np.ones((1, 1)), "b1": np.zeros((1, 1)),
         "w2": np.ones((1, 1)), "b2": np.zeros(1)}
    X = synth.normal(7, "relu.X", (11, d))
    np.testing.assert_allclose(oracle.featmap(p, X), np.maximum(X, 0) / math.sqrt(d), rtol=0, atol=1e-15)


def test_shared_mlp_with_one_channel_is_the_per_channel_mlp():
    """Listing: ScalarMLP(L=1) is the same module whether it serves as the one
    shared MLP or as the per-channel MLP of a single channel."""
    d, M, hid = 4, 3, 5
    ps = _rand_params(41, d, M, 1, hid, shared=True)
    pc = dict(ps, w1=ps["w1"].reshape(1, hid), b1=ps["b1"].reshape(1, hid))
    Q, K, V = _rand_inputs(41, 1, 2, 7, d, 3, scale=1.5)
    dO = synth.normal(41, "shared1.dO", V.shape)
    np.testing.assert_array_equal(oracle.featmap(ps, Q), oracle.featmap(pc, Q))
    gs = oracle.attn_bwd(ps, Q, K, V, dO, causal=True)
    gc = oracle.attn_bwd(pc, Q, K, V, dO, causal=True)
    for k in gs:
        np.testing.assert_allclose(gs[k].reshape(-1), gc[k].reshape(-1), rtol=1e-14, atol=0)


def test_shared_mlp_by_hand():
    """Shared-channel MLP (listing: one ScalarMLP with L outputs): fc1 units
    relu(u), relu(-u) and fc2 rows selecting one unit each give
    phi(x) = [relu(u), relu(-u)] / sqrt(M) for u = w^T x + b."""
    p = {"W": np.array([[1.0, -2.0]]), "b": np.array([0.5]), "w1": np.array([1.0, -1.0]),
         "b1": np.array([0.0, 0.0]), "w2": np.array([[1.0, 0.0], [0.0, 1.0]]), "b2": np.array([0.0, 0.0])}
    X = np.array([[1.0, 0.0], [0.0, 1.0], [3.0, 1.0], [-1.0, 0.25]])
    u = X @ p["W"][0] + p["b"][0]  # 1.5, -1.5, 1.5, -1.0
    np.testing.assert_allclose(oracle.featmap(p, X), np.stack([np.maximum(u, 0), np.maximum(-u, 0)], axis=1),
                               rtol=0, atol=1e-15)


def test_shared_fc1_gradient_sums_over_channels():
    """In the shared-channel MLP every channel reads every hidden unit, so the
    fc1 gradients collect the chain rule through all channels: central finite
    differences of sum(O * dO) in fp64 (both channels active on both units)."""
    p = {"W": np.array([[0.8, -0.6]]), "b": np.array([0.1]), "w1": np.array([1.0, -1.0]),
         "b1": np.array([0.1, 0.2]), "w2": np.array([[1.0, 0.5], [0.5, 1.0]]), "b2": np.array([0.05, 0.05])}
    Q, K, V = _rand_inputs(43, 1, 1, 6, 2, 2, scale=1.5)
    dO = synth.normal(43, "sharedfd.dO", V.shape)
    for causal in (False, True):
        g = oracle.attn_bwd(p, Q, K, V, dO, causal=causal, eps=1e-3)
        h = 1e-6
        for name, key in (("dw1", "w1"), ("db1", "b1"), ("dw2", "w2")):
            arr = p[key].reshape(-1)
            num = np.empty_like(arr)
            for e in range(arr.size):
                x0 = arr[e]
                arr[e] = x0 + h
                lp = _loss(p, Q, K, V, dO, None, causal, 1e-3)
                arr[e] = x0 - h
                lm = _loss(p, Q, K, V, dO, None, causal, 1e-3)
                arr[e] = x0
                num[e] = (lp - lm) / (2 * h)
            np.testing.assert_allclose(g[name].reshape(-1), num, rtol=2e-5, atol=2e-7 * max(1.0, np.abs(num).max()))


def test_phi_nonnegative_and_scale():
    """nonneg=True in the listing: every feature is >= 0; doubling M with the
    same projections duplicated scales phi by 1/sqrt(2)."""
    p = _rand_params(3, 6, 4, 3, 8)
    X = synth.normal(3, "nn.X", (50, 6))
    phi = oracle.featmap(p, X)
    assert np.all(phi >= 0)
    p2 = dict(p)
    p2["W"] = np.concatenate([p["W"], p["W"]])
    p2["b"] = np.concatenate([p["b"], p["b"]])
    phi2 = oracle.featmap(p2, X)
    np.testing.assert_allclose(phi2[:, :12], phi / math.sqrt(2.0), rtol=1e-14, atol=0)
    np.testing.assert_allclose(phi2[:, 12:], phi / math.sqrt(2.0), rtol=1e-14, atol=0)


def test_gram_psd_and_symmetric():
    """Prop. 1: k(x,y) = phi(x)^T phi(y) is a positive-definite kernel, so its
    Gram matrix on any point set is symmetric positive semi-definite."""
    p = _rand_params(5, 8, 4, 8, 64)
    X = synth.normal(5, "psd.X", (48, 8))
    phi = oracle.featmap(p, X)
    G = np.array([[float(np.dot(phi[i], phi[j])) for j in range(48)] for i in range(48)])
    assert np.array_equal(G, G.T)
    ev = np.linalg.eigvalsh(G)
    assert ev.min() >= -1e-12 * np.trace(G)
    # rank is bounded by the feature dimension D = 32 < 48 points
    assert np.sum(ev > 1e-10 * ev.max()) <= 32


# --------------------------------------------------------------------------
# attention forward

def test_attention_hand_example():
    g, p = _hand_params()
    X = np.array(g["X"])[None, None]
    V = np.array(g["attention"]["V"])[None, None]
    O = oracle.attn_fwd(p, X, X, V, eps=0.0)
    np.testing.assert_allclose(O[0, 0], np.array(g["attention"]["O_noncausal"]), rtol=1e-14, atol=1e-15)
    Oc = oracle.attn_fwd(p, X, X, V, causal=True, eps=0.0)
    np.testing.assert_allclose(Oc[0, 0], np.array(g["attention"]["O_causal"]), rtol=1e-14, atol=1e-15)


@pytest.mark.parametrize("causal", [False, True])
@pytest.mark.parametrize("eps", [0.0, 1e-6, 0.3])
def test_linear_form_equals_quadratic_form(causal, eps):
    """Eq. (kernel-attn): the sufficient-statistics form equals the brute-force
    sum_j k(q_i,k_j) v_j / (sum_j k(q_i,k_j) + eps), causal = masked j <= i."""
    p = _rand_params(11, 16, 4, 8, 64)
    Q, K, V = _rand_inputs(11, 2, 3, 70, 16, 5)
    lengths = np.array([70, 41], dtype=np.int32)
    O_lin = oracle.attn_fwd(p, Q, K, V, lengths, causal=causal, eps=eps)
    O_quad = oracle.attn_quadratic(p, Q, K, V, lengths, causal=causal, eps=eps)
    assert _relerr(O_lin, O_quad) < 1e-12


@pytest.mark.parametrize("causal", [False, True])
def test_constant_channels_give_mean(causal):
    """With w1 = 0, b1 = 1, w2 = c every feature is the same constant, so all
    kernel values are equal and O_i is the plain (prefix) mean of valid v_j."""
    d, M, L, hid = 6, 3, 2, 4
    p = {"W": synth.normal(1, "c.W", (M, d)), "b": np.zeros(M), "w1": np.zeros((L, hid)),
         "b1": np.ones((L, hid)), "w2": np.full((L, hid), 0.25), "b2": np.zeros(L)}
    Q, K, V = _rand_inputs(2, 2, 2, 33, d, 4)
    lengths = np.array([33, 20], dtype=np.int32)
    O = oracle.attn_fwd(p, Q, K, V, lengths, causal=causal, eps=0.0)
    for b in range(2):
        ln = lengths[b]
        for h in range(2):
            v = V[b, h, :ln]
            if causal:
                expect = np.cumsum(v, axis=0) / np.arange(1, ln + 1)[:, None]
            else:
                expect = np.broadcast_to(v.mean(axis=0), v.shape)
            np.testing.assert_allclose(O[b, h, :ln], expect, rtol=1e-13, atol=1e-14)
            assert np.all(O[b, h, ln:] == 0)


@pytest.mark.parametrize("causal", [False, True])
def test_unit_values_give_unit_outputs(causal):
    """V = 1 gives O = 1 on every row with a non-zero denominator (eps = 0):
    the normalisation of Eq. (kernel-attn) is row-wise."""
    p = _rand_params(4, 8, 4, 8, 64)
    Q, K, _ = _rand_inputs(4, 1, 2, 40, 8, 3)
    V = np.ones((1, 2, 40, 3))
    O = oracle.attn_fwd(p, Q, K, V, causal=causal, eps=0.0)
    phq, phk = oracle.featmap(p, Q), oracle.featmap(p, K)
    for h in range(2):
        for i in range(40):
            jmax = i + 1 if causal else 40
            den = float(phq[0, h, i] @ phk[0, h, :jmax].sum(axis=0))
            if den > 0:
                np.testing.assert_allclose(O[0, h, i], 1.0, rtol=1e-13)
            else:
                assert np.all(O[0, h, i] == 0)


def test_weights_nonnegative_and_sum_to_one():
    """Identity values (dv = n) expose the normalised weights a_ij = k_ij/sum_j k_ij:
    non-negative (nonneg=True) and summing to 1 per row."""
    n = 24
    p = _rand_params(6, 8, 4, 8, 64)
    Q, K, _ = _rand_inputs(6, 1, 1, n, 8, 1)
    V = np.eye(n)[None, None]
    for causal in (False, True):
        A = oracle.attn_fwd(p, Q, K, V, causal=causal, eps=0.0)[0, 0]
        assert np.all(A >= 0)
        rows = A.sum(axis=1)
        nz = rows > 0
        np.testing.assert_allclose(rows[nz], 1.0, rtol=1e-13)
        if causal:
            assert np.all(np.triu(A, 1) == 0)


def test_noncausal_permutation_invariance():
    p = _rand_params(8, 8, 4, 8, 64)
    Q, K, V = _rand_inputs(8, 1, 2, 50, 8, 6)
    perm = np.random.default_rng(0).permutation(50)
    O1 = oracle.attn_fwd(p, Q, K, V)
    O2 = oracle.attn_fwd(p, Q, K[:, :, perm], V[:, :, perm])
    assert _relerr(O1, O2) < 1e-13


@pytest.mark.parametrize("causal", [False, True])
def test_padding_is_ignored(causal):
    """Keys at or beyond the valid length do not affect O; padded query rows are 0."""
    p = _rand_params(9, 8, 4, 8, 64)
    Q, K, V = _rand_inputs(9, 2, 2, 40, 8, 3)
    lengths = np.array([25, 40], dtype=np.int32)
    O1 = oracle.attn_fwd(p, Q, K, V, lengths, causal=causal)
    K2, V2, Q2 = K.copy(), V.copy(), Q.copy()
    K2[0, :, 25:] = 100.0
    V2[0, :, 25:] = -7.0
    Q2[0, :, 25:] = 3.0
    O2 = oracle.attn_fwd(p, Q2, K2, V2, lengths, causal=causal)
    assert np.array_equal(O1, O2)
    assert np.all(O1[0, :, 25:] == 0)
    # and a length-25 sequence equals the truncated computation
    O3 = oracle.attn_fwd(p, Q[:1, :, :25], K[:1, :, :25], V[:1, :, :25], causal=causal)
    assert _relerr(O1[:1, :, :25], O3) < 1e-14


def test_linearity_in_values():
    p = _rand_params(10, 8, 4, 8, 64)
    Q, K, V = _rand_inputs(10, 1, 1, 30, 8, 4)
    V2 = synth.normal(10, "lin.V2", V.shape)
    for causal in (False, True):
        a = oracle.attn_fwd(p, Q, K, 2.0 * V - 3.0 * V2, causal=causal)
        b = 2.0 * oracle.attn_fwd(p, Q, K, V, causal=causal) - 3.0 * oracle.attn_fwd(p, Q, K, V2, causal=causal)
        assert _relerr(a, b) < 1e-12


def test_causal_first_row():
    """O_0 = v_0 * kappa / (kappa + eps) with kappa = phi(q_0)^T phi(k_0)."""
    p = _rand_params(12, 8, 4, 8, 64)
    Q, K, V = _rand_inputs(12, 1, 1, 5, 8, 3)
    eps = 0.05
    O = oracle.attn_fwd(p, Q, K, V, causal=True, eps=eps)
    kappa = float(oracle.featmap(p, Q[0, 0, 0]) @ oracle.featmap(p, K[0, 0, 0]))
    np.testing.assert_allclose(O[0, 0, 0], V[0, 0, 0] * kappa / (kappa + eps), rtol=1e-14)


# --------------------------------------------------------------------------
# backward: central finite differences in fp64

def _loss(p, Q, K, V, dO, lengths, causal, eps):
    return float(np.sum(oracle.attn_fwd(p, Q, K, V, lengths, causal=causal, eps=eps) * dO))


@pytest.mark.parametrize("shared", [False, True])
@pytest.mark.parametrize("causal", [False, True])
def test_gradients_match_finite_differences(causal, shared):
    d, M, L, hid, n = 3, 2, 2, 3, 6
    rng_seed = (21 if causal else 20) + (10 if shared else 0)
    p = _rand_params(rng_seed, d, M, L, hid, shared)
    # push projections away from zero so that the hidden-unit pattern is rich
    Q, K, V = _rand_inputs(rng_seed, 2, 1, n, d, 2, scale=1.5)
    dO = synth.normal(rng_seed, "fd.dO", V.shape)
    lengths = np.array([n, 4], dtype=np.int32)
    eps = 1e-3
    g = oracle.attn_bwd(p, Q, K, V, dO, lengths, causal=causal, eps=eps)
    h = 1e-6
    # rows near a ReLU kink have no unique derivative: skip those entries
    mq = oracle.kink_margin(p, Q)
    mk = oracle.kink_margin(p, K)
    checked = 0

    def fd(setter, base):
        nonlocal checked
        flat = base.reshape(-1)
        out = np.empty_like(flat)
        for e in range(flat.size):
            x0 = flat[e]
            flat[e] = x0 + h
            lp = setter()
            flat[e] = x0 - h
            lm = setter()
            flat[e] = x0
            out[e] = (lp - lm) / (2 * h)
            checked += 1
        return out.reshape(base.shape)

    f = lambda: _loss(p, Q, K, V, dO, lengths, causal, eps)
    for name, arr, margin in (("dQ", Q, mq), ("dK", K, mk), ("dV", V, None)):
        num = fd(f, arr)
        ana = g[name]
        if margin is not None:
            ok = margin > 1e-3
            num, ana = num[ok], ana[ok]
        np.testing.assert_allclose(ana, num, rtol=2e-5, atol=2e-7 * max(1.0, np.abs(num).max()))
    # parameters: skip only if any row's margin is tiny
    if min(mq.min(), mk.min()) > 1e-4:
        for name, key in (("dW", "W"), ("db", "b"), ("dw1", "w1"), ("db1", "b1"), ("dw2", "w2"), ("db2", "b2")):
            num = fd(f, p[key])
            np.testing.assert_allclose(g[name], num, rtol=2e-5, atol=2e-7 * max(1.0, np.abs(num).max()))
    assert checked > 50


def test_gradients_zero_on_padding():
    p = _rand_params(13, 8, 4, 8, 64)
    Q, K, V = _rand_inputs(13, 2, 1, 20, 8, 3)
    dO = synth.normal(13, "pad.dO", V.shape)
    lengths = np.array([12, 20], dtype=np.int32)
    for causal in (False, True):
        g = oracle.attn_bwd(p, Q, K, V, dO, lengths, causal=causal)
        for k in ("dQ", "dK", "dV"):
            assert np.all(g[k][0, :, 12:] == 0)


def test_abs_terms_bound_the_gradients():
    """The absolute-contribution mode sums |term| over the same per-sample terms
    as the gradients: it bounds every gradient element (triangle inequality) and
    equals it when every term of a sum has the same sign (one row, one unit:
    the query and key paths of that row give same-signed terms here)."""
    d, M, L, hid = 3, 2, 2, 3
    p = _rand_params(31, d, M, L, hid)
    Q, K, V = _rand_inputs(31, 1, 2, 5, d, 2, scale=1.5)
    dO = synth.normal(31, "abs.dO", V.shape)
    for causal in (False, True):
        g = oracle.attn_bwd(p, Q, K, V, dO, None, causal=causal, eps=1e-3)
        a = oracle.attn_bwd_abs_terms(p, Q, K, V, dO, None, causal=causal, eps=1e-3)
        for k in ("dW", "db", "dw1", "db1", "dw2", "db2"):
            assert np.all(a[k] >= np.abs(g[k]) * (1 - 1e-12) - 1e-300), k
        # the mode is switched off again afterwards
        g2 = oracle.attn_bwd(p, Q, K, V, dO, None, causal=causal, eps=1e-3)
        for k in g:
            np.testing.assert_array_equal(g[k], g2[k])
    # one row, one projection, one channel, one hidden unit: two same-signed terms per sum
    p1 = {"W": np.array([[1.0]]), "b": np.array([0.0]), "w1": np.array([[1.0]]), "b1": np.array([[0.5]]),
          "w2": np.array([[2.0]]), "b2": np.array([0.1])}
    X = np.array([[[[0.7]]]])
    V1 = np.array([[[[1.3]]]])
    dO1 = np.array([[[[-0.4]]]])
    g = oracle.attn_bwd(p1, X, X, V1, dO1, None, causal=False, eps=0.25)
    a = oracle.attn_bwd_abs_terms(p1, X, X, V1, dO1, None, causal=False, eps=0.25)
    for k in ("dW", "db", "dw1", "db1", "dw2", "db2"):
        np.testing.assert_allclose(a[k], np.abs(g[k]), rtol=1e-14, atol=0)
