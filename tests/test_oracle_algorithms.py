"""Pins of the oracle's decoding algorithms against what Sec. 3.1 fixes.

* the Jacobi fixed point is the greedy AR output (Sec. 3.1, citing Song et al.);
* every iteration with KV cache fixes at least one token (Sec. 3.1, "Jacobi
  decoding with KV cache"), so an n-token window converges in k <= n
  iterations; vanilla Jacobi (Eq. 3 without cache) needs at most n + 1 passes
  to observe y^(k) = y^(k-1);
* a guess that already equals the AR continuation is accepted whole in one step;
* n = 1 Jacobi is AR, step for step;
* brute force over every initial block of a micro model: each cached step's
  accepted count equals the count obtained by evaluating Eq. 3 row by row
  without any cache.
"""
from dataclasses import replace

import numpy as np
import pytest

from oracle import oracle as orc
from paper_2403_00835_gb300 import synthetic as syn

MICRO = replace(syn.TINY, name="micro", n_layers=1, d_model=16, n_heads=2, n_kv_heads=2,
                head_dim=8, ffn=24, vocab=8)


def oracle_model(cfg, w):
    wd = orc.ORC_F32 if cfg.dtype == "f32" else orc.ORC_BF16
    return orc.OracleModel(orc.OracleArch(**syn.oracle_arch_kwargs(cfg)), w, wd)


@pytest.fixture(scope="module")
def tiny():
    cfg = syn.TINY
    return cfg, oracle_model(cfg, syn.make_weights(cfg, seed=0))


@pytest.fixture(scope="module")
def micro():
    # large init scale so the micro model's argmax is far from uniform
    return oracle_model(MICRO, syn.make_weights(MICRO, seed=11, std=0.7))


@pytest.mark.parametrize("mode", ["refill", "shrink"])
@pytest.mark.parametrize("n,seed", [(8, 2), (5, 3), (16, 4)])
def test_jacobi_fixed_point_equals_ar(tiny, mode, n, seed):
    cfg, m = tiny
    prompt = syn.make_prompts(cfg.vocab, [32], seed=1)[0]
    ar = orc.ar_decode(m, prompt, 40)
    jr = orc.jacobi_decode(m, prompt, n, 40, seed=seed, mode=mode)
    assert jr.tokens == ar.tokens
    assert all(a >= 1 for a in jr.accepted)
    assert sum(jr.accepted) == 40
    assert jr.iterations == len(jr.accepted) <= 40


def test_jacobi_prompt_guesses_fixed_point(tiny):
    cfg, m = tiny
    prompt = syn.make_prompts(cfg.vocab, [32], seed=1)[0]
    ar = orc.ar_decode(m, prompt, 24)
    jr = orc.jacobi_decode(m, prompt, 8, 24, seed=9, guess_init="prompt", record=True)
    assert jr.tokens == ar.tokens
    # every initial guess slot is a prompt token
    assert set(jr.trajectory[0][1:]) <= set(prompt)


def test_shrink_window_converges_within_n(tiny):
    cfg, m = tiny
    prompt = syn.make_prompts(cfg.vocab, [32], seed=1)[0]
    n = 8
    jr = orc.jacobi_decode(m, prompt, n, 48, seed=5, mode="shrink", record=True)
    # windows are delimited by the block width returning to n
    widths = [len(b) for b in jr.trajectory]
    windows, cur = [], 0
    for i, wdt in enumerate(widths):
        if wdt == n and i > 0:
            windows.append(cur)
            cur = 0
        cur += 1
    windows.append(cur)
    assert all(k <= n for k in windows)
    assert sum(jr.accepted) == 48


def test_ar_guess_converges_in_one_step(tiny):
    cfg, m = tiny
    prompt = syn.make_prompts(cfg.vocab, [32], seed=1)[0]
    n = 8
    ar = orc.ar_decode(m, prompt, n + 1)
    s = m.session(64)
    head, _, _ = orc.prefill(s, prompt)
    assert head == ar.tokens[0]
    st = orc.jacobi_step(s, ar.tokens[:n], len(prompt))
    assert st.accepted == n
    assert st.pred[n - 1] == ar.tokens[n]  # the next head is the (n+1)-th AR token


def test_n1_jacobi_is_ar(tiny):
    cfg, m = tiny
    prompt = syn.make_prompts(cfg.vocab, [32], seed=1)[0]
    ar = orc.ar_decode(m, prompt, 20)
    jr = orc.jacobi_decode(m, prompt, 1, 20, seed=0)
    assert jr.tokens == ar.tokens
    assert jr.accepted == [1] * 20 and jr.iterations == 20


def test_eos_stops_decoding(tiny):
    cfg, m = tiny
    prompt = syn.make_prompts(cfg.vocab, [32], seed=1)[0]
    ar = orc.ar_decode(m, prompt, 30)
    eos = ar.tokens[11]
    first = ar.tokens.index(eos)
    jr = orc.jacobi_decode(m, prompt, 8, 30, seed=2, eos_id=eos)
    assert jr.tokens == ar.tokens[: first + 1]
    assert orc.ar_decode(m, prompt, 30, eos_id=eos).tokens == ar.tokens[: first + 1]


def test_vanilla_jacobi_fixed_point(tiny):
    cfg, m = tiny
    prompt = syn.make_prompts(cfg.vocab, [12], seed=4)[0]
    n = 6
    ar = orc.ar_decode(m, prompt, n)
    for seed in range(3):
        y0 = syn.make_guesses(cfg.vocab, 1, n, seed=seed)[0]
        ystar, k = orc.jacobi_vanilla(m, prompt, y0)
        assert ystar == ar.tokens
        assert 1 <= k <= n + 1


def _definitional_accept(model, prompt, block):
    """Longest prefix of the block that Eq. 3's rows reproduce, each row
    evaluated by a fresh full forward of [x; block_<i] (no cache reuse)."""
    a = 1
    while a < len(block):
        seq = list(prompt) + list(block[:a])
        row = model.session(len(seq)).forward(seq, 0, rows=[len(seq) - 1])[0]
        if int(np.argmax(row)) != block[a]:
            break
        a += 1
    return a


def test_brute_force_micro_model(micro):
    m = micro
    V, n = MICRO.vocab, 3
    prompt = [3, 1, 4, 1, 5]
    ar = orc.ar_decode(m, prompt, n + 2)
    s0 = m.session(16)
    head, _, _ = orc.prefill(s0, prompt)
    assert head == ar.tokens[0]
    seen_a = set()
    for g1 in range(V):
        for g2 in range(V):
            block = [head, g1, g2]
            s = m.session(16)
            s.forward(prompt, 0, rows=[])
            st = orc.jacobi_step(s, block, len(prompt))
            assert st.accepted == _definitional_accept(m, prompt, block)
            seen_a.add(st.accepted)
    assert seen_a == {1, 2, 3}
    # vanilla Jacobi from every one of the V^n initial blocks reaches the AR output
    for idx in range(V ** n):
        y0 = [(idx // V ** i) % V for i in range(n)]
        ystar, k = orc.jacobi_vanilla(m, prompt, y0)
        assert ystar == ar.tokens[:n] and k <= n + 1
    # full decodes from several guess streams, both block policies
    for seed in range(8):
        for mode in ("refill", "shrink"):
            assert orc.jacobi_decode(m, prompt, n, 12, seed=seed, mode=mode).tokens == \
                orc.ar_decode(m, prompt, 12).tokens


# ---- the lookahead combination (Sec. 3.3): n-gram pool feeding the refill block

def test_ngram_pool_step_worked_example():
    """Hand-worked step of the pool rule: predictions [5, 6, 7, 8, 9], two
    tokens accepted, trigrams (two-token values).  The head 6 has the pool
    continuation [1, 2], which replaces refill slots 1-2; the iteration's
    trigrams keyed 5, 6, 7 then enter the pool (6's value replaced)."""
    pool = {6: [1, 2]}
    out = orc.ngram_pool_step(pool, [5, 6, 7, 8, 9], 2, [6, 7, 8, 9, 42], 3)
    assert out == [6, 1, 2, 9, 42]
    assert pool == {5: [6, 7], 6: [7, 8], 7: [8, 9]}


def test_ngram_pool_step_edges():
    # no entry for the head: the refill block unchanged
    pool = {}
    assert orc.ngram_pool_step(pool, [3, 3, 4, 3, 5], 1, [3, 3, 4, 3, 5], 2) == [3, 3, 4, 3, 5]
    # the same key several times in one iteration: the last n-gram wins
    assert pool == {3: [5], 4: [3]}
    # a candidate longer than the block is cut at the block's end; a block
    # shorter than the n-gram adds nothing to the pool
    pool = {7: [1, 2, 3, 4, 5]}
    assert orc.ngram_pool_step(pool, [7, 0, 0], 1, [7, 9, 9], 6) == [7, 1, 2]
    assert pool == {7: [1, 2, 3, 4, 5]}


@pytest.mark.parametrize("n,ngram,seed", [(8, 3, 2), (8, 5, 3), (16, 4, 4), (4, 2, 5)])
def test_lookahead_decode_equals_ar(tiny, n, ngram, seed):
    """Whatever the pool proposes, a token is committed only when the step
    verifies it, so the decode is the greedy AR output (Sec. 3.1)."""
    cfg, m = tiny
    for pl in (32, 9):
        prompt = syn.make_prompts(cfg.vocab, [pl], seed=seed)[0]
        ar = orc.ar_decode(m, prompt, 40)
        jr = orc.jacobi_decode(m, prompt, n, 40, seed=seed, mode="lookahead", ngram=ngram)
        assert jr.tokens == ar.tokens
        assert all(a >= 1 for a in jr.accepted)
        assert sum(jr.accepted) == 40


# ---- the same combination with a verification branch of several n-grams

def test_ngram_pool_push_worked_example():
    """Hand-worked pool updates with trigrams and at most two values a key:
    a key keeps its distinct values most recent first, an n-gram entered again
    moves to the front, and a third distinct value drops the oldest."""
    pool = {}
    orc.ngram_pool_push(pool, [5, 6, 7, 6, 7, 8], 3, 2)
    assert pool == {5: [(6, 7)], 6: [(7, 8), (7, 6)], 7: [(6, 7)]}
    orc.ngram_pool_push(pool, [6, 7, 6, 9], 3, 2)
    assert pool[6] == [(7, 6), (7, 8)] and pool[7] == [(6, 9), (6, 7)]
    orc.ngram_pool_push(pool, [6, 1, 1], 3, 2)
    assert pool[6] == [(1, 1), (7, 6)]
    # fewer predictions than the n-gram: nothing enters
    orc.ngram_pool_push(pool, [2, 3], 3, 2)
    assert 2 not in pool


def test_verify_candidates_brute_force_micro_model(micro):
    """Every two-token candidate after the head of a micro model, verified in
    one call: each accepted count equals the count from Eq. 3's rows evaluated
    by fresh full forwards, so no candidate sees another's K/V."""
    m = micro
    V = MICRO.vocab
    prompt = [3, 1, 4, 1, 5]
    ar = orc.ar_decode(m, prompt, 4)
    head = ar.tokens[0]
    cands = [[g1, g2] for g1 in range(V) for g2 in range(V)]
    s = m.session(16)
    s.forward(prompt, 0, rows=[])
    res = orc.verify_candidates(s, head, cands, len(prompt))
    seen = set()
    for c, (a, q, gaps) in zip(cands, res):
        assert a == _definitional_accept(m, prompt, [head] + c)
        assert q[0] == ar.tokens[1] and len(q) == len(gaps) == 3
        seen.add(a)
    assert seen == {1, 2, 3}
    # the AR continuation is accepted whole, and predicts the token after it
    (a, q, _), = orc.verify_candidates(s, head, [ar.tokens[1:3]], len(prompt))
    assert a == 3 and q == ar.tokens[1:4]


@pytest.mark.parametrize("n,ngram,ncand,seed", [(8, 3, 4, 2), (8, 5, 2, 3), (16, 4, 4, 4), (4, 2, 1, 5)])
def test_verify_decode_equals_ar(tiny, n, ngram, ncand, seed):
    """A candidate's tokens are committed only as far as the model verifies
    them, with their own K/V, so the decode is the greedy AR output
    (Sec. 3.1); on this model's repeating continuations some iterations
    commit a candidate, and then more tokens than the block would have."""
    cfg, m = tiny
    won = 0
    for pl in (32, 17, 9):
        prompt = syn.make_prompts(cfg.vocab, [pl], seed=seed)[0]
        ar = orc.ar_decode(m, prompt, 48)
        jr = orc.jacobi_decode(m, prompt, n, 48, seed=seed, mode="verify", ngram=ngram, ncand=ncand,
                               record=True)
        assert jr.tokens == ar.tokens
        assert all(a >= 1 for a in jr.accepted) and sum(jr.accepted) == 48
        assert len(jr.branch) == len(jr.candidates) == jr.iterations
        for br, cands in zip(jr.branch, jr.candidates):
            assert len(cands) <= ncand and all(len(c) == ngram - 1 for c in cands)
            assert -1 <= br < len(cands)
        won += sum(1 for br in jr.branch if br >= 0)
    assert won >= 1


def test_verify_without_pool_entries_is_refill(tiny):
    """With n-grams longer than the block nothing enters the pool, no
    candidate is verified, and the decode is the refill decode iteration for
    iteration."""
    cfg, m = tiny
    prompt = syn.make_prompts(cfg.vocab, [17], seed=2)[0]
    rf = orc.jacobi_decode(m, prompt, 8, 40, seed=3, mode="refill", record=True)
    vr = orc.jacobi_decode(m, prompt, 8, 40, seed=3, mode="verify", ngram=9, ncand=4, record=True)
    assert vr.trajectory == rf.trajectory and vr.accepted == rf.accepted
    assert vr.branch == [-1] * vr.iterations and all(c == [] for c in vr.candidates)


def test_verify_eos_inside_a_candidate(tiny):
    """An EOS inside a committed candidate ends the decode at the EOS, as for
    the block (Alg. 1's stop rule)."""
    cfg, m = tiny
    prompt = syn.make_prompts(cfg.vocab, [17], seed=2)[0]
    jr = orc.jacobi_decode(m, prompt, 8, 48, seed=3, mode="verify", ngram=3, ncand=4)
    ar_full = orc.ar_decode(m, prompt, 48).tokens
    # the first token that a candidate committed beyond the head
    pos, k = 0, None
    for a, br in zip(jr.accepted, jr.branch):
        if br >= 0 and a >= 2:
            k = pos + 1
            break
        pos += a
    assert k is not None
    eos = ar_full[k]
    first = ar_full.index(eos)
    got = orc.jacobi_decode(m, prompt, 8, 48, seed=3, mode="verify", ngram=3, ncand=4, eos_id=eos)
    assert got.tokens == ar_full[:first + 1]
    assert got.tokens == orc.ar_decode(m, prompt, 48, eos_id=eos).tokens


def test_verify_candidates_come_from_earlier_iterations(tiny):
    """Sec. 3.3: candidates are n-grams generated in previous iterations.
    Every n-gram verified at iteration i follows its head in the predictions
    of some iteration before i, and the first iteration verifies none."""
    cfg, m = tiny
    ngram = 3
    for pl, seed in ((17, 2), (9, 3)):
        prompt = syn.make_prompts(cfg.vocab, [pl], seed=seed)[0]
        jr = orc.jacobi_decode(m, prompt, 8, 48, seed=seed, mode="verify", ngram=ngram, ncand=4,
                               record=True, keep_steps=True)
        assert jr.candidates[0] == []
        checked = 0
        for i, (block, cands) in enumerate(zip(jr.trajectory, jr.candidates)):
            earlier = {tuple(st.pred[k:k + ngram]) for st in jr.steps[:i]
                       for k in range(len(st.pred) - ngram + 1)}
            for c in cands:
                assert (block[0], *c) in earlier, f"iteration {i}"
                checked += 1
        assert checked >= 1
