"""The seeded input generators both sides are fed from (CPU): deterministic
per seed, within range, shaped as the workloads state, and free of the
method's arithmetic."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from paper_2403_00835_gb300 import synthetic as syn


def test_prompts_are_seeded_and_in_vocab():
    a = syn.make_prompts(2048, [5, 17, 1], seed=3)
    b = syn.make_prompts(2048, [5, 17, 1], seed=3)
    c = syn.make_prompts(2048, [5, 17, 1], seed=4)
    assert a == b and a != c
    assert [len(p) for p in a] == [5, 17, 1]
    assert all(0 <= t < 2048 for p in a for t in p)


def test_prompts_are_uniform_over_the_vocabulary():
    (p,) = syn.make_prompts(16, [160000], seed=1)
    counts = np.bincount(p, minlength=16)
    # chi-square with 15 degrees of freedom: 99.9th percentile is 37.7
    chi2 = ((counts - 10000.0) ** 2 / 10000.0).sum()
    assert chi2 < 37.7


def test_ragged_lengths_span_the_stated_range():
    lens = syn.ragged_lens(4096, 256, 1024, seed=1)
    assert lens == syn.ragged_lens(4096, 256, 1024, seed=1)
    assert min(lens) >= 256 and max(lens) <= 1024
    assert min(lens) < 300 and max(lens) > 980  # both ends are reached


def test_guesses_shape_and_range():
    g = syn.make_guesses(32000, 3, 16, seed=2)
    assert len(g) == 3 and all(len(r) == 16 for r in g)
    assert all(0 <= t < 32000 for r in g for t in r)
    assert g == syn.make_guesses(32000, 3, 16, seed=2)


def test_weights_follow_the_recipe():
    cfg = syn.TINY
    w = syn.make_weights(cfg, seed=0, device="cpu")
    w2 = syn.make_weights(cfg, seed=0, device="cpu")
    assert torch.equal(w["wq"][0], w2["wq"][0]) and torch.equal(w["lm_head"], w2["lm_head"])
    # N(0, 0.02^2) matrices, unit RMSNorm gains, untied LM head
    big = torch.cat([w["wq"][0].flatten(), w["w_down"][1].flatten(), w["tok_emb"].flatten()])
    assert abs(float(big.mean())) < 1e-3
    assert abs(float(big.std()) - 0.02) < 5e-4
    assert torch.all(w["attn_norm"][0] == 1) and torch.all(w["final_norm"] == 1)
    assert not torch.equal(w["lm_head"], w["tok_emb"])
    assert tuple(w["wq"][0].shape) == (cfg.n_heads * cfg.head_dim, cfg.d_model)
    assert tuple(w["w_gate"][0].shape) == (cfg.ffn, cfg.d_model)
    assert tuple(w["w_down"][0].shape) == (cfg.d_model, cfg.ffn)
    assert len(w["wq"]) == cfg.n_layers


def test_seven_b_shapes():
    for cfg in (syn.LLAMA7B, syn.CODER7B):
        assert (cfg.n_layers, cfg.d_model, cfg.n_heads, cfg.head_dim, cfg.ffn) == (32, 4096, 32, 128, 11008)
    assert syn.LLAMA7B.vocab == 32000 and syn.CODER7B.vocab == 32256
    assert syn.LLAMA7B.rope_theta == 1e4 and syn.CODER7B.rope_theta == 1e5
    # about 6.7 B parameters
    assert 6.5e9 < syn.LLAMA7B.n_params < 6.9e9
