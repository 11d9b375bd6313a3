"""Pins of the oracle's feature-map variants: the channel MLPs' hidden-unit
activation other than ReLU (GELU, SiLU, tanh: the listing's ScalarMLP `act`),
the envelope-gated map (channel l of every projection multiplied by the
tokenwise gate h_l(x) = sigmoid(We_l . x + be_l), Sec. 5.4 / Table 5) and
Bank+Coef (channel l multiplied by a learned global coefficient c_l, Table 5).

Checked by closed-form special cases (tabulated values of the normal
distribution function, tanh and the logistic function, and scipy's special
functions, which share no code with the oracle), by invariances of Eq.
(kernel-attn) under a common scale of the features, by the brute-force
quadratic form, and by central finite differences of every gradient.
"""
import math

import numpy as np
import pytest

import oracle
import synth

special = pytest.importorskip("scipy.special")


def _params(seed, d, M, L, hid, shared=False):
    return {k: v.astype(np.float64) for k, v in synth.phi_params(seed, d, M, L, hid, shared).items()}


def _gate(seed, d, L, scale=1.0):
    return {"We": synth.normal(seed, "v.We", (L, d)) * scale / math.sqrt(d),
            "be": synth.normal(seed, "v.be", (L,)) * 0.5}


def _coef(seed, L):
    return {"coef": 0.5 + np.abs(synth.normal(seed, "v.coef", (L,)))}


def _inputs(seed, B, H, n, d, dv, scale=1.0):
    Q = synth.normal(seed, "v.Q", (B, H, n, d)) * scale
    K = synth.normal(seed, "v.K", (B, H, n, d)) * scale
    V = synth.normal(seed, "v.V", (B, H, n, dv))
    dO = synth.normal(seed, "v.dO", (B, H, n, dv))
    return Q, K, V, dO


def _identity_map(d, b2=0.0):
    """hidden = 1, w1 = 1, b1 = 0, w2 = 1, W = I, b = 0, one channel: psi(u) = act(u) + b2."""
    return {"W": np.eye(d), "b": np.zeros(d), "w1": np.ones((1, 1)), "b1": np.zeros((1, 1)),
            "w2": np.ones((1, 1)), "b2": np.full(1, b2)}


def test_activation_tabulated_values():
    """psi(u) = act(u) without the outer ReLU at points whose values are tabulated:
    GELU(1) = Phi(1), GELU(-1) = -Phi(-1) (standard normal distribution function),
    tanh(1/2), SiLU(2) = 2 / (1 + e^-2)."""
    d = 2
    cases = {"gelu": [(1.0, 0.8413447460685429), (-1.0, -0.15865525393145705)],
             "tanh": [(0.5, 0.46211715726000974), (-0.5, -0.46211715726000974)],
             "silu": [(2.0, 1.7615941559557646), (-2.0, -0.23840584404423537)]}
    for act, pts in cases.items():
        p = oracle.PhiParams(_identity_map(d), nonneg=False, act=act)
        X = np.array([[pts[0][0], pts[1][0]]])
        want = np.array([[pts[0][1], pts[1][1]]]) / math.sqrt(d)
        np.testing.assert_allclose(oracle.featmap(p, X), want, rtol=1e-14, atol=0, err_msg=act)


@pytest.mark.parametrize("act", ["gelu", "silu", "tanh"])
def test_activation_against_special_functions(act):
    """psi(u) = relu(act(u) - 1/4) on a dense grid, against scipy.special: GELU(u) = u ndtr(u),
    SiLU(u) = u expit(u)."""
    d = 4
    X = np.linspace(-6.0, 6.0, 4 * 301).reshape(-1, d)
    ref = {"gelu": lambda u: u * special.ndtr(u), "silu": lambda u: u * special.expit(u), "tanh": np.tanh}[act](X)
    p = oracle.PhiParams(_identity_map(d, -0.25), act=act)
    np.testing.assert_allclose(oracle.featmap(p, X), np.maximum(ref - 0.25, 0) / math.sqrt(d), rtol=1e-13,
                               atol=1e-15)


def test_envelope_gate_by_hand():
    """One channel, W = I, psi = relu: phi_i(x) = sigmoid(We . x + be) relu(x_i) / sqrt(d)."""
    d = 3
    p0 = _identity_map(d)
    We, be = np.array([[1.0, -2.0, 0.5]]), np.array([0.25])
    X = synth.normal(31, "v.Xg", (11, d))
    h = special.expit(X @ We[0] + be[0])
    p = oracle.PhiParams({**p0, "We": We, "be": be})
    np.testing.assert_allclose(oracle.featmap(p, X), h[:, None] * np.maximum(X, 0) / math.sqrt(d), rtol=1e-14,
                               atol=0)


def test_constant_gate_and_coefficients_scale_the_channels():
    """We = 0: h_l = sigmoid(be_l) for every row; with coefficients c_l the feature i*L + l is
    the default map's times sigmoid(be_l) c_l."""
    d, M, L, hid = 6, 3, 4, 8
    p = _params(32, d, M, L, hid)
    be = np.array([-1.0, 0.0, 0.5, 3.0])
    c = np.array([0.5, 2.0, 1.5, 0.25])
    X = synth.normal(32, "v.Xc", (9, d))
    got = oracle.featmap(oracle.PhiParams({**p, "We": np.zeros((L, d)), "be": be, "coef": c}), X)
    want = oracle.featmap(p, X) * np.tile(special.expit(be) * c, M)
    np.testing.assert_allclose(got, want, rtol=1e-14, atol=0)


@pytest.mark.parametrize("causal", [False, True])
def test_common_feature_scale_leaves_the_outputs(causal):
    """Eq. (kernel-attn) with eps = 0 is a ratio of two sums linear in phi(q_i): a gate that is
    the same for every row and channel (We = 0, equal be) or equal coefficients leave O unchanged."""
    d, M, L, hid = 6, 3, 4, 8
    p = _params(33, d, M, L, hid)
    Q, K, V, _ = _inputs(33, 2, 2, 17, d, 3)
    lengths = np.array([17, 6], dtype=np.int32)
    O = oracle.attn_fwd(p, Q, K, V, lengths, causal, 0.0)
    for extra in ({"We": np.zeros((L, d)), "be": np.full(L, 0.7)}, {"coef": np.full(L, 3.0)}):
        Ov = oracle.attn_fwd(oracle.PhiParams({**p, **extra}), Q, K, V, lengths, causal, 0.0)
        np.testing.assert_allclose(Ov, O, rtol=1e-12, atol=1e-14)


@pytest.mark.parametrize("causal", [False, True])
def test_variant_linear_form_equals_quadratic_form(causal):
    d, M, L, hid = 6, 3, 4, 8
    p = oracle.PhiParams({**_params(34, d, M, L, hid), **_gate(34, d, L), **_coef(34, L)}, act="gelu")
    Q, K, V, _ = _inputs(34, 2, 2, 25, d, 4)
    lengths = np.array([25, 10], dtype=np.int32)
    a = oracle.attn_fwd(p, Q, K, V, lengths, causal, 0.3)
    b = oracle.attn_quadratic(p, Q, K, V, lengths, causal, 0.3)
    assert np.max(np.abs(a - b)) < 1e-10 * max(1.0, np.max(np.abs(b)))


VARIANTS = {
    "gelu": ("gelu", False, False, False),
    "silu": ("silu", False, False, False),
    "tanh": ("tanh", False, False, False),
    "tanh-shared": ("tanh", False, False, True),
    "envelope": ("relu", True, False, False),
    "coef": ("relu", False, True, False),
    "gelu+envelope+coef": ("gelu", True, True, False),
}


@pytest.mark.parametrize("causal", [False, True])
@pytest.mark.parametrize("name", sorted(VARIANTS))
def test_variant_gradients_match_finite_differences(name, causal):
    act, env, coef, shared = VARIANTS[name]
    d, M, L, hid, n = 3, 2, 2, 3, 6
    seed = 40 + sorted(VARIANTS).index(name) * 2 + (1 if causal else 0)
    p = _params(seed, d, M, L, hid, shared)
    if env:
        p.update(_gate(seed, d, L, scale=2.0))
    if coef:
        p.update(_coef(seed, L))
    Q, K, V, dO = _inputs(seed, 2, 1, n, d, 2, scale=1.5)
    lengths = np.array([n, 4], dtype=np.int32)
    eps = 1e-3
    mk = lambda: oracle.PhiParams(p, act=act)
    g = oracle.attn_bwd(mk(), Q, K, V, dO, lengths, causal, eps)
    assert set(g) >= {"dWe", "dbe"} if env else "dWe" not in g
    mq, mkk = oracle.kink_margin(mk(), Q), oracle.kink_margin(mk(), K)
    h = 1e-6
    checked = 0

    def loss():
        return float(np.sum(oracle.attn_fwd(mk(), Q, K, V, lengths, causal, eps) * dO))

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

    for gname, arr, margin in (("dQ", Q, mq), ("dK", K, mkk), ("dV", V, None)):
        num, ana = fd(arr), g[gname]
        if margin is not None:
            ok = margin > 1e-3
            num, ana = num[ok], ana[ok]
        np.testing.assert_allclose(ana, num, rtol=2e-5, atol=2e-7 * max(1.0, np.abs(num).max()), err_msg=gname)
    keys = ["W", "b", "w1", "b1", "w2", "b2"] + (["We", "be"] if env else []) + (["coef"] if coef else [])
    assert min(mq.min(), mkk.min()) > 1e-4, "inputs too close to a kink for the parameter check"
    for key in keys:
        num = fd(p[key])
        np.testing.assert_allclose(g["d" + key], num, rtol=2e-5, atol=2e-7 * max(1.0, np.abs(num).max()),
                                   err_msg="d" + key)
    assert checked > 60
