"""The seeded input generator shared by the oracle side and the CUDA side.

Pinned against its published definition (SplitMix64: Steele, Lea & Flood,
"Fast splittable pseudorandom number generators", OOPSLA 2014), against
PyTorch's float32 -> bfloat16 conversion (round to nearest even), and by the
distributions and ranges the input recipes promise.
"""
import math

import numpy as np
import pytest

import synth


def test_splitmix64_reference_sequence():
    """A stream is the SplitMix64 output sequence from state `key`: element k is
    mix(key + k * 0x9E3779B97F4A7C15), k = 1, 2, ...  From state 1234567 the
    reference generator's first five outputs are the values below."""
    expect = [6457827717110365317, 3203168211198807973, 9817491932198370423, 4593380528125082431,
              16408922859458223821]
    with np.errstate(over="ignore"):
        got = synth._mix(np.uint64(1234567) + np.arange(1, 6, dtype=np.uint64) * synth.GOLDEN)
    assert [int(x) for x in got] == expect


def test_streams_are_deterministic_and_keyed_by_name():
    a = synth.raw_u64(3, "t.a", 1000)
    assert np.array_equal(a, synth.raw_u64(3, "t.a", 1000))
    assert np.array_equal(a[:10], synth.raw_u64(3, "t.a", 10))  # a prefix does not depend on the count
    assert not np.array_equal(a, synth.raw_u64(3, "t.b", 1000))
    assert not np.array_equal(a, synth.raw_u64(4, "t.a", 1000))


def test_uniform_and_normal_moments():
    n = 1 << 20
    u = synth.uniform01(5, "t.u", n)
    assert u.min() >= 0.0 and u.max() < 1.0
    assert abs(u.mean() - 0.5) < 5 * math.sqrt(1 / 12 / n)
    assert abs(u.var() - 1 / 12) < 1e-3
    z = synth.normal(5, "t.z", (n,))
    assert abs(z.mean()) < 5 / math.sqrt(n)
    assert abs(z.var() - 1.0) < 5 * math.sqrt(2 / n)
    assert abs(np.mean(z ** 4) - 3.0) < 0.05
    # Box-Muller pairs: the radius of a pair is Rayleigh, P(r^2 > t) = exp(-t / 2)
    r2 = z[0::2] ** 2 + z[1::2] ** 2
    assert abs(np.mean(r2 > 2.0) - math.exp(-1.0)) < 5 * math.sqrt(0.25 / (n // 2))


def test_randint_range():
    v = synth.randint(9, "t.i", (100000,), 2048, 4096)
    assert v.min() >= 2048 and v.max() <= 4096 and v.dtype == np.int64
    assert v.min() < 2100 and v.max() > 4040


def test_bf16_rounding_matches_torch():
    torch = pytest.importorskip("torch")
    x = synth.normal(11, "t.bf", (100000,)).astype(np.float32) * np.float32(3.0)
    # exact ties between two bf16 values, with even and odd lower neighbours, both signs
    ties = (np.arange(1, 257, dtype=np.uint32) << np.uint32(16)) | np.uint32(0x8000)
    ties = np.concatenate([ties | np.uint32(0x3F000000), ties | np.uint32(0xBF000000)]).view(np.float32)
    x = np.concatenate([x, ties, np.array([0.0, -0.0, 1e-40, 3.0e38], dtype=np.float32)])
    got = synth.f32_to_bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(got, ref)
    t = synth.IOTensor(x.astype(np.float64), "bf16")
    assert np.array_equal(t.value, torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy())


def test_phi_params_follow_the_listing_initialisation():
    d, M, L, hid = 32, 8, 8, 64
    p = synth.phi_params(1, d, M, L, hid)
    assert all(v.dtype == np.float32 for v in p.values())
    assert p["W"].shape == (M, d) and np.all(p["b"] == 0)
    assert abs(p["W"].std() * math.sqrt(d) - 1.0) < 0.15
    for k in ("w1", "b1"):
        assert p[k].shape == (L, hid) and np.abs(p[k]).max() <= 1.0
    bound = 1 / math.sqrt(hid)
    assert np.abs(p["w2"]).max() <= bound and np.abs(p["b2"]).max() <= bound
    s = synth.phi_params(1, d, M, L, hid, shared=True)
    assert s["w1"].shape == (hid,) and s["w2"].shape == (L, hid)


def test_attn_inputs_shapes_and_lengths():
    inp = synth.attn_inputs(2, 3, 2, 50, 16, 8, "bf16", 0.5, (10, 40), with_grad=True)
    assert inp["Q"].shape == (3, 2, 50, 16) and inp["V"].shape == (3, 2, 50, 8) and inp["dO"].shape == (3, 2, 50, 8)
    assert inp["lengths"].dtype == np.int32 and np.all((inp["lengths"] >= 10) & (inp["lengths"] <= 40))
    # bf16 values: the fp64 value of every element has at most 8 significant bits
    v = inp["Q"].value
    assert np.array_equal(v, synth.bf16_bits_to_f64(synth.f32_to_bf16_bits(v.astype(np.float32))))


def test_normal_at_equals_the_full_draw():
    """Drawing chosen elements of a normal stream gives the same values, bit for bit, as drawing the
    whole tensor and indexing it (odd and even positions, both ends)."""
    full = synth.normal(9, "na.X", (7, 13, 5)).ravel()
    idx = np.array([0, 1, 2, 3, 64, 65, 299, 453, 454, full.size - 1])
    assert np.array_equal(synth.normal_at(9, "na.X", idx), full[idx])
    rows = (np.arange(3)[:, None] * 65 + np.arange(5)[None, :]).ravel()
    assert np.array_equal(synth.normal_at(9, "na.X", rows), full[rows])
