"""Pins of the trajectory profiling (Sec. 3.3, Table 3): hand-built
trajectories with known accepted and stationary counts, and the accepted
counts of the oracle's own decode (Alg. 3's i*) recovered from its recorded
blocks."""
import numpy as np
import pytest

from paper_2403_00835_gb300 import trajectory as tj

FINAL = [10, 11, 12, 13, 14, 15, 16, 17, 18, 19]


def test_hand_trajectory_refill():
    # n = 4, refill: the block always covers the next 4 positions
    blocks = [
        [10, 99, 12, 98],  # slot 2 final while slot 1 is wrong -> candidate
        [11, 12, 97, 96],  # positions 1..4: 11 and 12 accepted; position 2 committed
        [13, 14, 15, 16],  # all four accepted
        [17, 18, 19, 95],
    ]
    st = tj.analyse(blocks, FINAL, 4, 4)
    assert st.accepted == [1, 2, 4, 3]
    # windows: [0,4) and [4,8) and [8,12); position 2 is the only stationary token
    assert st.window_stationary[0] == 1
    assert sum(st.window_stationary) == 1


def test_token_that_changes_is_not_stationary():
    blocks = [
        [10, 99, 12, 98],  # position 2 final early ...
        [11, 97, 96, 95],  # ... but replaced here (position 2 holds 97)
        [12, 13, 14, 15],
        [16, 17, 18, 19],
    ]
    st = tj.analyse(blocks, FINAL, 4, 4)
    assert st.accepted == [1, 1, 4, 4]
    assert sum(st.window_stationary) == 0


def test_shrink_windows():
    # shrink: widths 4, 3 (after 1 accepted), then a fresh window of 4
    blocks = [
        [10, 99, 12, 13],        # a = 1; positions 2 and 3 final behind a wrong slot
        [11, 12, 13, -1],        # a = 3: window [0, 4) fixed; 2 and 3 stationary
        [14, 15, 98, 17],        # fresh window [4, 8): a = 2, position 7 candidate
        [16, 17, -1, -1],        # a = 2: position 7 committed -> stationary
    ]
    st = tj.analyse(blocks, FINAL, 4, 4)
    assert st.accepted == [1, 3, 2, 2]
    assert st.window_stationary == [2, 1]
    assert st.window_iterations == [2, 2]


@pytest.mark.parametrize("mode", ["refill", "shrink"])
def test_accepted_counts_match_oracle_decode(mode):
    pytest.importorskip("torch")
    from oracle import oracle as orc
    from paper_2403_00835_gb300 import synthetic as syn
    from tests.parity_util import oracle_for
    cfg = syn.TINY
    om = oracle_for(cfg, syn.make_weights(cfg, seed=0, device="cpu"))
    prompt = syn.make_prompts(cfg.vocab, [24], seed=1)[0]
    n, max_new = 8, 32
    jr = orc.jacobi_decode(om, prompt, n, max_new, seed=2, mode=mode, record=True)
    blocks = [list(b) + [-1] * (n - len(b)) for b in jr.trajectory]
    st = tj.analyse(blocks, jr.tokens, jr.iterations, n)
    assert st.accepted == jr.accepted
    assert sum(st.accepted) == len(jr.tokens)
