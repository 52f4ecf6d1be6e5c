"""Pins of the oracle's decoder forward pass.

* against a composition of torch library routines in fp64 (F.rms_norm,
  F.scaled_dot_product_attention with a causal mask, complex-number RoPE,
  F.silu); the C oracle uses none of them;
* a special case with a closed form (zeroed output projections make every layer
  the identity);
* KV-cache consistency: a block forward over a cached prefix equals the same
  rows computed in one pass, and equals one-token-at-a-time forwards (the
  premise of Jacobi decoding with KV cache, Sec. 3.1);
* causality: a row does not depend on later tokens (Eq. 3's causal mask).
"""
import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import oracle as orc
from paper_2403_00835_gb300 import synthetic as syn


def oracle_model(cfg, w):
    wd = orc.ORC_F32 if cfg.dtype == "f32" else orc.ORC_BF16
    return orc.OracleModel(orc.OracleArch(**syn.oracle_arch_kwargs(cfg)), w, wd)


def torch_reference_logits(cfg, w, tokens):
    """Independent fp64 forward from library routines (all rows, from position 0)."""
    d64 = lambda t: t.detach().to(torch.float64)
    H, Hkv, hd = cfg.n_heads, cfg.n_kv_heads, cfg.head_dim
    T = len(tokens)
    x = d64(w["tok_emb"])[torch.tensor(tokens)]
    pos = torch.arange(T, dtype=torch.float64)
    freqs = cfg.rope_theta ** (-2.0 * torch.arange(hd // 2, dtype=torch.float64) / hd)
    rot = torch.polar(torch.ones(T, hd // 2, dtype=torch.float64), pos[:, None] * freqs[None])

    def rope(t):  # [T, heads, hd], rotate-half pairs as complex numbers
        z = torch.complex(t[..., : hd // 2], t[..., hd // 2:]) * rot[:, None, :]
        return torch.cat([z.real, z.imag], dim=-1)

    for l in range(cfg.n_layers):
        h = F.rms_norm(x, (cfg.d_model,), weight=d64(w["attn_norm"][l]), eps=cfg.rms_eps)
        q = rope((h @ d64(w["wq"][l]).T).view(T, H, hd))
        k = rope((h @ d64(w["wk"][l]).T).view(T, Hkv, hd))
        v = (h @ d64(w["wv"][l]).T).view(T, Hkv, hd)
        k = k.repeat_interleave(H // Hkv, dim=1)
        v = v.repeat_interleave(H // Hkv, dim=1)
        a = F.scaled_dot_product_attention(q.transpose(0, 1)[None], k.transpose(0, 1)[None],
                                           v.transpose(0, 1)[None], is_causal=True)
        a = a[0].transpose(0, 1).reshape(T, H * hd)
        x = x + a @ d64(w["wo"][l]).T
        h = F.rms_norm(x, (cfg.d_model,), weight=d64(w["mlp_norm"][l]), eps=cfg.rms_eps)
        x = x + (F.silu(h @ d64(w["w_gate"][l]).T) * (h @ d64(w["w_up"][l]).T)) @ d64(w["w_down"][l]).T
    h = F.rms_norm(x, (cfg.d_model,), weight=d64(w["final_norm"]), eps=cfg.rms_eps)
    return (h @ d64(w["lm_head"]).T).numpy()


@pytest.fixture(scope="module")
def tiny():
    cfg = syn.TINY
    w = syn.make_weights(cfg, seed=0)
    return cfg, w, oracle_model(cfg, w)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_forward_matches_library_composition(dtype):
    cfg = syn.TINY if dtype == "f32" else syn.TINY_BF16
    w = syn.make_weights(cfg, seed=0)
    m = oracle_model(cfg, w)
    toks = syn.make_prompts(cfg.vocab, [24], seed=5)[0]
    got = m.session(64).forward(toks, 0)
    ref = torch_reference_logits(cfg, w, toks)
    np.testing.assert_allclose(got, ref, rtol=0, atol=1e-11 * np.abs(ref).max())


def test_forward_gqa_matches_library_composition():
    from dataclasses import replace
    cfg = replace(syn.TINY, n_heads=4, n_kv_heads=2, name="tiny-gqa")
    w = syn.make_weights(cfg, seed=3)
    m = oracle_model(cfg, w)
    toks = syn.make_prompts(cfg.vocab, [19], seed=6)[0]
    np.testing.assert_allclose(m.session(32).forward(toks, 0), torch_reference_logits(cfg, w, toks),
                               rtol=0, atol=1e-12)


def test_identity_layers_closed_form(tiny):
    cfg, w, _ = tiny
    w = dict(w)
    w["wo"] = [torch.zeros_like(t) for t in w["wo"]]
    w["w_down"] = [torch.zeros_like(t) for t in w["w_down"]]
    m = oracle_model(cfg, w)
    toks = [5, 17, 2047, 0, 5]
    got = m.session(8).forward(toks, 0)
    e = w["tok_emb"].double().numpy()[toks]
    h = e / np.sqrt((e ** 2).mean(axis=1, keepdims=True) + cfg.rms_eps) * w["final_norm"].double().numpy()
    ref = h @ w["lm_head"].double().numpy().T
    np.testing.assert_allclose(got, ref, rtol=0, atol=1e-12)
    np.testing.assert_array_equal(got[0], got[4])  # same token, position-independent here


def test_kv_cache_block_equals_one_pass_and_sequential(tiny):
    cfg, w, m = tiny
    toks = syn.make_prompts(cfg.vocab, [40], seed=7)[0]
    full = m.session(64).forward(toks, 0)
    # prefix of 31 then a block of 9 over the cache
    s = m.session(64)
    s.forward(toks[:31], 0, rows=[])
    blk = s.forward(toks[31:], 31)
    np.testing.assert_allclose(blk, full[31:], rtol=0, atol=1e-12)
    # one token at a time
    s2 = m.session(64)
    s2.forward(toks[:31], 0, rows=[])
    seq = np.stack([s2.forward([toks[31 + i]], 31 + i)[0] for i in range(9)])
    np.testing.assert_allclose(seq, full[31:], rtol=0, atol=1e-12)


def test_stale_cache_positions_are_overwritten(tiny):
    # Alg. 3 "removes the KV cache of false tokens": rewriting a block at the
    # same start position must not see the earlier (false) block.
    cfg, w, m = tiny
    toks = syn.make_prompts(cfg.vocab, [20], seed=8)[0]
    s = m.session(64)
    s.forward(toks, 0, rows=[])
    s.forward([1, 2, 3, 4, 5, 6], 20, rows=[])  # a false block
    blk = [9, 8, 7, 6]
    got = s.forward(blk, 20)
    ref = m.session(64).forward(toks + blk, 0, rows=range(20, 24))
    np.testing.assert_allclose(got, ref, rtol=0, atol=1e-12)


def test_causality(tiny):
    cfg, w, m = tiny
    a = syn.make_prompts(cfg.vocab, [16], seed=9)[0]
    b = list(a)
    b[12:] = [(t + 1) % cfg.vocab for t in b[12:]]
    la = m.session(32).forward(a, 0)
    lb = m.session(32).forward(b, 0)
    np.testing.assert_array_equal(la[:12], lb[:12])
    assert np.abs(la[12:] - lb[12:]).max() > 1e-6


def test_bad_arguments_rejected(tiny):
    cfg, w, m = tiny
    s = m.session(8)
    with pytest.raises(ValueError):
        s.forward([cfg.vocab], 0)
    with pytest.raises(ValueError):
        s.forward([1, 2, 3], 6)
