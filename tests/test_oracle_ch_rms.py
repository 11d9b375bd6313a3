"""Pins of the oracle's channel RMS normalisation of the feature map (the
listing's MLPLearnableFeatureMap with ch_rms on): every channel's MLP outputs
y_l are scaled by s_l = min(target / (rms_l + 1e-6), 1), rms_l the root mean
square of y_l over every valid row and projection of the input the map is
applied to (the queries and the keys separately).

Each check rests on something other than the oracle's own formula: a target
above every channel's RMS reduces to the plain map bit for bit; the scaled
outputs have RMS equal to the target; constant channels give hand-computable
features; the attention output recomputed in numpy from the feature map of
all rows; the invariance of a clamped channel to the scale of its MLP
(forward and gradient); padding invariance; central finite differences.
"""
import math

import numpy as np
import pytest

import oracle
import synth


def _rand_params(seed, d, M, L, hid, shared=False):
    return {k: v.astype(np.float64) for k, v in synth.phi_params(seed, d, M, L, hid, shared).items()}


def _rand_inputs(seed, B, H, n, d, dv, scale=1.0):
    Q = synth.normal(seed, "r.Q", (B, H, n, d)) * scale
    K = synth.normal(seed, "r.K", (B, H, n, d)) * scale
    V = synth.normal(seed, "r.V", (B, H, n, dv))
    return Q, K, V


def _relerr(a, b):
    return float(np.max(np.abs(a - b)) / max(np.max(np.abs(b)), 1e-300))


def _rms_all(p, X, lengths=None):
    """Per-channel RMS of both sides' inputs (for choosing targets)."""
    return oracle.ch_rms(oracle.PhiParams(p, 1.0), X, lengths)[1]


@pytest.mark.parametrize("causal", [False, True])
def test_target_above_every_rms_is_the_plain_map(causal):
    """s_l = 1 on every channel: forward and backward equal the unnormalised oracle exactly."""
    p = _rand_params(40, 8, 4, 8, 16)
    Q, K, V = _rand_inputs(40, 2, 2, 30, 8, 3)
    dO = synth.normal(40, "r.dO", V.shape)
    lengths = np.array([30, 17], dtype=np.int32)
    big = 10.0 * max(_rms_all(p, Q, lengths).max(), _rms_all(p, K, lengths).max())
    pn = oracle.PhiParams(p, big)
    assert np.all(oracle.ch_rms(pn, Q, lengths)[0] == 1.0)
    assert np.array_equal(oracle.attn_fwd(pn, Q, K, V, lengths, causal),
                          oracle.attn_fwd(p, Q, K, V, lengths, causal))
    g0 = oracle.attn_bwd(p, Q, K, V, dO, lengths, causal)
    g1 = oracle.attn_bwd(pn, Q, K, V, dO, lengths, causal)
    for k in g0:
        assert np.array_equal(g0[k], g1[k]), k


def test_normalised_channels_have_the_target_rms():
    """Where a channel is clamped, the RMS of its scaled outputs sqrt(M) * phi over all
    rows and projections is the target, up to the 1e-6 regularisers; where it is not,
    the outputs are the unscaled MLP outputs."""
    d, M, L = 8, 6, 8
    p = _rand_params(41, d, M, L, 16)
    X = synth.normal(41, "r.X", (3, 2, 25, d))
    rms = _rms_all(p, X)
    target = float(np.median(rms))
    pn = oracle.PhiParams(p, target)
    phi = oracle.featmap(pn, X).reshape(-1, M, L) * math.sqrt(M)
    plain = oracle.featmap(p, X).reshape(-1, M, L) * math.sqrt(M)
    got = np.sqrt(np.mean(phi ** 2, axis=(0, 1)))
    raw = np.sqrt(np.mean(plain ** 2, axis=(0, 1)))
    clamped = raw > target * 1.01
    unclamped = raw < target * 0.99
    assert clamped.any() and unclamped.any()
    # the 1e-6 inside and outside the square root pull the RMS below the target by at
    # most 1e-6 / (2 rms^2) + 1e-6 / rms, relative
    bound = 1e-6 / (2 * raw[clamped] ** 2) + 1e-6 / raw[clamped]
    rel = 1.0 - got[clamped] / target
    assert np.all(rel >= -1e-14) and np.all(rel <= bound), (rel, bound)
    np.testing.assert_array_equal(phi[:, :, unclamped], plain[:, :, unclamped])


def test_constant_channels_by_hand():
    """w1 = 0, b1 = 1, w2 = c_l, b2 = 0: y_l = hid * c_l on every sample, so
    rms_l = sqrt(y_l^2 + 1e-6) and the features are known in closed form."""
    d, M, L, hid = 4, 3, 3, 2
    c = np.array([0.05, 0.5, 2.0])
    p = {"W": synth.normal(42, "r.W", (M, d)), "b": np.zeros(M), "w1": np.zeros((L, hid)),
         "b1": np.ones((L, hid)), "w2": np.repeat(c[:, None], hid, axis=1), "b2": np.zeros(L)}
    X = synth.normal(42, "r.X", (5, d))
    target = 0.3
    y = hid * c                                     # 0.1, 1, 4
    rms = np.sqrt(y * y + 1e-6)
    s = np.minimum(target / (rms + 1e-6), 1.0)      # 1 (0.3 > 0.1), ~0.3, ~0.075
    expect = np.tile(s * y / math.sqrt(M), M)
    got = oracle.featmap(oracle.PhiParams(p, target), X)
    np.testing.assert_allclose(got, np.broadcast_to(expect, got.shape), rtol=1e-14, atol=0)


@pytest.mark.parametrize("causal", [False, True])
def test_attention_from_the_feature_map_of_all_rows(causal):
    """The attention output is Eq. (kernel-attn) evaluated in numpy on the feature
    maps of the queries and of the keys, each normalised by the statistics of all
    of its own rows (every head of the batch)."""
    d, M, L, n = 8, 4, 8, 20
    p = _rand_params(43, d, M, L, 16)
    Q, K, V = _rand_inputs(43, 2, 3, n, d, 5)
    target = float(np.median(np.concatenate([_rms_all(p, Q), _rms_all(p, K)])))
    pn = oracle.PhiParams(p, target)
    sq, sk = oracle.ch_rms(pn, Q)[0], oracle.ch_rms(pn, K)[0]
    assert np.any(sq < 1) and np.any(sq == 1) and not np.array_equal(sq, sk)
    eps = 1e-3
    pq, pk = oracle.featmap(pn, Q), oracle.featmap(pn, K)
    A = np.einsum("bhif,bhjf->bhij", pq, pk)
    if causal:
        A = A * np.tril(np.ones((n, n)))
    expect = np.einsum("bhij,bhjc->bhic", A, V) / (A.sum(-1, keepdims=True) + eps)
    assert _relerr(oracle.attn_fwd(pn, Q, K, V, None, causal, eps), expect) < 1e-12
    assert _relerr(oracle.attn_quadratic(pn, Q, K, V, None, causal, eps), expect) < 1e-12


@pytest.mark.parametrize("causal", [False, True])
def test_padding_is_ignored(causal):
    """Rows at or past a sequence's length enter neither the attention nor the
    channel statistics; a batch of one sequence equals its truncation."""
    p = _rand_params(44, 8, 4, 8, 16)
    Q, K, V = _rand_inputs(44, 2, 2, 30, 8, 3)
    dO = synth.normal(44, "r.dO", V.shape)
    lengths = np.array([19, 30], dtype=np.int32)
    target = float(np.median(_rms_all(p, Q, lengths)))
    pn = oracle.PhiParams(p, target)
    Q2, K2, V2 = Q.copy(), K.copy(), V.copy()
    Q2[0, :, 19:] = 5.0
    K2[0, :, 19:] = -9.0
    V2[0, :, 19:] = 2.0
    assert np.array_equal(oracle.attn_fwd(pn, Q, K, V, lengths, causal), oracle.attn_fwd(pn, Q2, K2, V2, lengths, causal))
    g1 = oracle.attn_bwd(pn, Q, K, V, dO, lengths, causal)
    g2 = oracle.attn_bwd(pn, Q2, K2, V2, dO, lengths, causal)
    for k in g1:
        assert np.array_equal(g1[k], g2[k]), k
        if k in ("dQ", "dK", "dV"):
            assert np.all(g1[k][0, :, 19:] == 0)
    one = np.array([19], dtype=np.int32)
    a = oracle.attn_fwd(pn, Q[:1], K[:1], V[:1], one, causal)
    b = oracle.attn_fwd(pn, Q[:1, :, :19], K[:1, :, :19], V[:1, :, :19], None, causal)
    assert _relerr(a[:, :, :19], b) < 1e-14


@pytest.mark.parametrize("causal", [False, True])
def test_clamped_channel_is_invariant_to_its_mlp_scale(causal):
    """A channel whose scale is clamped outputs target * y_l / rms_l, invariant (up to
    the 1e-6 terms) to multiplying its fc2 weights and bias by a > 0.  So the output is
    unchanged, and the gradient is orthogonal to that direction:
    sum_k w2_lk dw2_lk + b2_l db2_l = 0, which holds only with the term that carries the
    dependence of s_l on the channel's outputs."""
    d, M, L, hid = 8, 4, 4, 16
    p = _rand_params(47, d, M, L, hid)
    Q, K, V = _rand_inputs(47, 2, 2, 24, d, 3)
    dO = synth.normal(47, "r.dO", V.shape)
    rmin = np.minimum(_rms_all(p, Q), _rms_all(p, K))
    alive = rmin > 0.01                             # channels that are not zero everywhere
    assert alive.sum() >= 3
    target = 0.5 * float(rmin[alive].min())         # every live channel clamped, on both sides
    pn = oracle.PhiParams(p, target)
    O = oracle.attn_fwd(pn, Q, K, V, None, causal)
    g = oracle.attn_bwd(pn, Q, K, V, dO, None, causal)
    g_plain = oracle.attn_bwd(p, Q, K, V, dO, None, causal)
    for l in np.flatnonzero(alive):
        # relative size of the 1e-6 regularisers against the channel's RMS
        tol = 10 * (1e-6 / (2 * rmin[l] ** 2) + 1e-6 / rmin[l])
        p2 = {k: v.copy() for k, v in p.items()}
        p2["w2"][l] *= 1.7
        p2["b2"][l] *= 1.7
        O2 = oracle.attn_fwd(oracle.PhiParams(p2, target), Q, K, V, None, causal)
        assert _relerr(O2, O) < tol, l
        along = float(p["w2"][l] @ g["dw2"][l] + p["b2"][l] * g["db2"][l])
        scale = float(np.abs(p["w2"][l] * g["dw2"][l]).sum() + abs(p["b2"][l] * g["db2"][l]))
        assert abs(along) < tol * scale, (l, along, scale)
        # without normalisation the same directional derivative is far from zero
        plain = float(p["w2"][l] @ g_plain["dw2"][l] + p["b2"][l] * g_plain["db2"][l])
        assert abs(plain) > 100 * tol * scale, (l, plain, scale)


def _loss(p, target, Q, K, V, dO, lengths, causal, eps):
    return float(np.sum(oracle.attn_fwd(oracle.PhiParams(p, target), Q, K, V, lengths, causal, eps) * dO))


@pytest.mark.parametrize("mix", ["clamped", "mixed", "shared"])
@pytest.mark.parametrize("causal", [False, True])
def test_gradients_match_finite_differences(causal, mix):
    """Every gradient with the normalisation on (every live channel clamped, a mix
    of clamped and unclamped channels, and the shared-channel MLP with every live
    channel clamped) against central differences of the forward pass."""
    d, M, L, hid, n = 3, 2, 3, 3, 6
    seed = 46 + (1 if causal else 0) + {"clamped": 0, "mixed": 2, "shared": 4}[mix]
    p = _rand_params(seed, d, M, L, hid, shared=(mix == "shared"))
    Q, K, V = _rand_inputs(seed, 2, 1, n, d, 2, scale=1.5)
    dO = synth.normal(seed, "r.dO", V.shape)
    lengths = np.array([n, 4], dtype=np.int32)
    eps = 1e-3
    rms = np.concatenate([_rms_all(p, Q, lengths), _rms_all(p, K, lengths)])
    if mix in ("clamped", "shared"):
        target = 0.5 * float(rms[rms > 0.01].min())
    else:  # between the channels' RMS values, away from every one of them
        srt = np.sort(rms)
        gaps = srt[1:] / srt[:-1]
        k = int(np.argmax(gaps))
        assert gaps[k] > 1.2
        target = float(math.sqrt(srt[k] * srt[k + 1]))
    g = oracle.attn_bwd(oracle.PhiParams(p, target), Q, K, V, dO, lengths, causal, eps)
    h = 1e-6
    mq = oracle.kink_margin(p, Q)
    mk = oracle.kink_margin(p, K)
    checked = 0

    def fd(base):
        nonlocal checked
        flat = base.reshape(-1)
        out = np.empty_like(flat)
        for e in range(flat.size):
            x0 = flat[e]
            flat[e] = x0 + h
            lp = _loss(p, target, Q, K, V, dO, lengths, causal, eps)
            flat[e] = x0 - h
            lm = _loss(p, target, Q, K, V, dO, lengths, causal, eps)
            flat[e] = x0
            out[e] = (lp - lm) / (2 * h)
            checked += 1
        return out.reshape(base.shape)

    for name, arr, margin in (("dQ", Q, mq), ("dK", K, mk), ("dV", V, None)):
        num = fd(arr)
        ana = g[name]
        if margin is not None:
            ok = margin > 1e-3
            num, ana = num[ok], ana[ok]
        np.testing.assert_allclose(ana, num, rtol=2e-5, atol=2e-7 * max(1.0, np.abs(num).max()))
    if min(mq.min(), mk.min()) > 1e-4:
        for name, key in (("dW", "W"), ("db", "b"), ("dw1", "w1"), ("db1", "b1"), ("dw2", "w2"), ("db2", "b2")):
            num = fd(p[key])
            np.testing.assert_allclose(g[name], num, rtol=2e-5, atol=2e-7 * max(1.0, np.abs(num).max()))
    assert checked > 50
