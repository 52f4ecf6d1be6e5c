"""Pins of the oracle's layer primitives against closed forms and independent
library routines (the C oracle calls none of these libraries)."""
import json
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import oracle as orc

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_rmsnorm_closed_form():
    # x = (3, 4), g = 1, eps = 0: mean(x^2) = 12.5, so out = x / sqrt(12.5).
    out = orc.rmsnorm([3.0, 4.0], [1.0, 1.0], 0.0)
    assert out == pytest.approx([3 / math.sqrt(12.5), 4 / math.sqrt(12.5)], abs=1e-15)
    # gain scales elementwise; eps enters under the root
    out = orc.rmsnorm([1.0, 1.0], [2.0, -1.0], 1.0)
    assert out == pytest.approx([2 / math.sqrt(2.0), -1 / math.sqrt(2.0)], abs=1e-15)


def test_rmsnorm_vs_torch_library():
    rng = np.random.default_rng(0)
    x = rng.normal(size=256)
    g = rng.normal(size=256)
    ref = F.rms_norm(torch.tensor(x), (256,), weight=torch.tensor(g), eps=1e-6).numpy()
    np.testing.assert_allclose(orc.rmsnorm(x, g, 1e-6), ref, rtol=1e-13, atol=1e-13)


def test_rope_closed_form():
    # head_dim 4, pos 1, theta 1e4.  Pair (0, 2) turns by 1 * 1e4^0 = 1 rad,
    # pair (1, 3) by 1 * 1e4^(-2/4) = 0.01 rad; (a, b) -> (a cos - b sin, b cos + a sin).
    c1, s1, c2, s2 = math.cos(1.0), math.sin(1.0), math.cos(0.01), math.sin(0.01)
    out = orc.rope([1.0, 2.0, 3.0, 4.0], 1, 1e4)
    assert out == pytest.approx([1 * c1 - 3 * s1, 2 * c2 - 4 * s2, 3 * c1 + 1 * s1, 4 * c2 + 2 * s2],
                                abs=1e-15)
    # position 0 is the identity
    assert orc.rope([1.0, 2.0, 3.0, 4.0], 0, 1e4) == pytest.approx([1, 2, 3, 4], abs=0)


def test_rope_as_complex_rotation_and_relative_position():
    # Rotate-half RoPE is multiplication of z_i = v_i + j v_{i+hd/2} by
    # exp(j pos theta^(-2i/hd)); compare with torch's complex arithmetic.
    rng = np.random.default_rng(1)
    hd, theta = 128, 1e4
    v = rng.normal(size=hd)
    for pos in (0, 1, 7, 1000, 4095):
        z = torch.complex(torch.tensor(v[: hd // 2]), torch.tensor(v[hd // 2:]))
        freqs = theta ** (-2.0 * torch.arange(hd // 2, dtype=torch.float64) / hd)
        zr = z * torch.polar(torch.ones(hd // 2, dtype=torch.float64), pos * freqs)
        ref = np.concatenate([zr.real.numpy(), zr.imag.numpy()])
        np.testing.assert_allclose(orc.rope(v, pos, theta), ref, rtol=1e-12, atol=1e-12)
    # norm preserved; q.k depends only on the position difference
    q, k = rng.normal(size=hd), rng.normal(size=hd)
    assert np.linalg.norm(orc.rope(q, 37, theta)) == pytest.approx(np.linalg.norm(q), rel=1e-13)
    d1 = orc.rope(q, 50, theta) @ orc.rope(k, 20, theta)
    d2 = orc.rope(q, 530, theta) @ orc.rope(k, 500, theta)
    assert d1 == pytest.approx(d2, rel=1e-9)


def test_silu_closed_form_and_library():
    assert orc.silu(0.0) == 0.0
    assert orc.silu(1.0) == pytest.approx(1 / (1 + math.exp(-1)), abs=1e-16)
    assert orc.silu(-1.0) == pytest.approx(-1 / (1 + math.e), abs=1e-16)
    zs = np.linspace(-20, 20, 81)
    ref = F.silu(torch.tensor(zs)).numpy()
    np.testing.assert_allclose([orc.silu(z) for z in zs], ref, rtol=1e-14, atol=1e-15)


def test_attend_closed_form():
    # scores (q.k0, q.k1)/sqrt(4) = (1, 0): weights (e, 1)/(1 + e)
    out = orc.attend([2.0, 0, 0, 0], [[1.0, 0, 0, 0], [0, 0, 0, 0]], [[1.0, 0, 0, 0], [0, 1.0, 0, 0]])
    e = math.e
    assert out == pytest.approx([e / (1 + e), 1 / (1 + e), 0, 0], abs=1e-15)
    # a single key returns its value exactly; equal scores give the mean
    rng = np.random.default_rng(2)
    v = rng.normal(size=(1, 8))
    np.testing.assert_array_equal(orc.attend(rng.normal(size=8), rng.normal(size=(1, 8)), v), v[0])
    vv = rng.normal(size=(5, 8))
    np.testing.assert_allclose(orc.attend(np.zeros(8), rng.normal(size=(5, 8)), vv), vv.mean(0), atol=1e-15)


def test_attend_vs_torch_sdpa():
    rng = np.random.default_rng(3)
    hd, n = 64, 37
    q, k, v = rng.normal(size=hd), rng.normal(size=(n, hd)), rng.normal(size=(n, hd))
    ref = F.scaled_dot_product_attention(torch.tensor(q)[None, None, None],
                                         torch.tensor(k)[None, None], torch.tensor(v)[None, None])
    np.testing.assert_allclose(orc.attend(q, k, v), ref[0, 0, 0].numpy(), rtol=1e-12, atol=1e-13)


def test_argmax_top2_ties_and_gap():
    assert orc.argmax_top2(np.array([0.5, 2.0, 1.0, 2.0])) == (1, 0.0)  # lowest index, gap 0
    tok, gap = orc.argmax_top2(np.array([0.5, 3.0, 1.0, 2.5]))
    assert tok == 1 and gap == pytest.approx(0.5)


def test_splitmix64_published_vector():
    fx = json.load(open(os.path.join(GOLDEN, "splitmix64_seed1234567.json")))
    got = [orc.splitmix64_output(fx["seed"], i) for i in range(1, 6)]
    assert got == [int(s) for s in fx["outputs"]]


def test_guess_token_ranges():
    V = 32000
    toks = [orc.guess_token(7, b, s, k, V) for b in range(3) for s in range(5) for k in range(16)]
    assert all(0 <= t < V for t in toks)
    assert len(set(toks)) > 200  # 240 draws, essentially all distinct
    prompt = [11, 22, 33]
    picks = {orc.guess_token(7, 0, s, k, V, prompt) for s in range(10) for k in range(10)}
    assert picks == set(prompt)
    # the map from the top 32 bits is the multiply-high: r * V >> 32
    r = orc.splitmix64_output(7, orc.guess_counter(1, 2, 3) + 1) >> 32
    assert orc.guess_token(7, 1, 2, 3, V) == (r * V) >> 32


def test_guess_token_golden_from_published_vector():
    """Stored tokens derived from the published splitmix64 outputs: slot s of
    sequence 0 at iteration 0 uses output s + 1."""
    fx = json.load(open(os.path.join(GOLDEN, "guess_tokens_seed1234567.json")))
    for V, want in fx["tokens"].items():
        got = [orc.guess_token(fx["seed"], fx["b"], fx["step"], s, int(V)) for s in fx["slots"]]
        assert got == want, V
    picks = [orc.guess_token(fx["seed"], 0, 0, s, 32000, fx["prompt"]) for s in fx["slots"]]
    assert picks == fx["prompt_picks"]


def _splitmix64_sequential(seed, count):
    """The generator as published: a 64-bit state advanced by the golden-ratio
    increment before each output, then the three-step mix.  Yields `count`
    outputs in order."""
    m = (1 << 64) - 1
    state = seed & m
    for _ in range(count):
        state = (state + 0x9E3779B97F4A7C15) & m
        z = state
        z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & m
        z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & m
        yield z ^ (z >> 31)


def test_guess_token_counter_layout_by_sequential_generator():
    """The counter-based draw for (iteration j, slot s) of sequence 0 is the
    (j * 2^16 + s + 1)-th output of the sequential generator."""
    V, seed = 32000, 1234567
    outs = list(_splitmix64_sequential(seed, (1 << 16) + 8))
    fx = json.load(open(os.path.join(GOLDEN, "splitmix64_seed1234567.json")))
    assert outs[:5] == [int(s) for s in fx["outputs"]]
    for step, slot in ((0, 0), (0, 7), (1, 0), (1, 3)):
        i = (step << 16) + slot  # 0-based index of the output
        assert orc.guess_token(seed, 0, step, slot, V) == ((outs[i] >> 32) * V) >> 32, (step, slot)
