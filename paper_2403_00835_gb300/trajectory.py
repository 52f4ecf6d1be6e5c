"""Profiling of recorded Jacobi trajectories (Sec. 3.3, Table 3): accepted
(fast-forwarded) tokens per iteration and stationary tokens per n-token window.

Input: the blocks y^(0), y^(1), ... of one sequence as recorded by
``cllm_decode_read_trajectory`` (slots beyond a shrunken window are -1) and the
sequence's final committed tokens.  Host-side bookkeeping only: the blocks
themselves come from the CUDA decode.

Readings (the paper defines both phenomena in words only):
  * accepted count of iteration j: the length of the block's longest prefix
    that equals the final tokens at those positions.  The block's first token
    is the head, always correct, so the count is >= 1; it "includes the one
    token that will be predicted right even without fast-forwarding" (Table 3
    caption).  Under greedy decoding a token whose prefix is correct is
    accepted exactly when it equals the final token, so this is Alg. 3's i*.
  * a window (an "n-token sequence") is the run of positions covered by the
    first block that starts at or after the end of the previous window; it
    lasts until all of its positions are committed.  Under the shrink policy
    that is exactly one fresh n-wide block and its shrinking successors;
    under the refill policy, consecutive runs of n positions.
  * a position of a window is stationary when, at some iteration before it is
    committed, it already holds its final token while an earlier position of
    the window does not, and it keeps that token in every later block until
    it is committed.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import List, Sequence

import numpy as np


@dataclass
class TrajectoryStats:
    accepted: List[int] = field(default_factory=list)      # per iteration
    window_stationary: List[int] = field(default_factory=list)  # per window
    window_iterations: List[int] = field(default_factory=list)  # per window

    @property
    def mean_accepted(self) -> float:
        return float(np.mean(self.accepted)) if self.accepted else 0.0

    @property
    def mean_stationary(self) -> float:
        return float(np.mean(self.window_stationary)) if self.window_stationary else 0.0


def _block(row: Sequence[int]) -> List[int]:
    out = []
    for t in row:
        if t < 0:
            break
        out.append(int(t))
    return out


def analyse(blocks: Sequence[Sequence[int]], tokens: Sequence[int], iterations: int,
            n: int) -> TrajectoryStats:
    """Statistics of one sequence's trajectory.  ``blocks[j]`` is y^(j) (-1
    padded), ``tokens`` the committed tokens (-1 padded), ``iterations`` the
    number of iterations the sequence ran."""
    final = [int(t) for t in tokens if t >= 0]
    st = TrajectoryStats()
    c = 0              # tokens committed before iteration j
    windows = []       # [first position, end position, iterations]
    candidate = set()  # positions holding their final token since a wrong slot preceded them
    stationary = set()
    for j in range(iterations):
        blk = _block(blocks[j])
        if not blk:
            break
        if not windows or c >= windows[-1][1]:
            windows.append([c, c + len(blk), 0])
        windows[-1][2] += 1
        a = 0  # accepted: the longest prefix equal to the final tokens
        while a < len(blk) and c + a < len(final) and blk[a] == final[c + a]:
            a += 1
        a = max(a, 1)
        st.accepted.append(a)
        for k in range(len(blk)):
            p = c + k
            if not (p < len(final) and blk[k] == final[p]):
                candidate.discard(p)    # a stationary token may not change
            elif k > a:
                candidate.add(p)        # final while slot a (before it) is wrong
        for p in [q for q in candidate if q < c + a]:
            stationary.add(p)           # kept its token until committed
            candidate.discard(p)
        c += a
    for w0, w1, its in windows:
        st.window_stationary.append(sum(1 for p in stationary if w0 <= p < w1))
        st.window_iterations.append(its)
    return st


def analyse_batch(traj: np.ndarray, tokens: np.ndarray, iters: np.ndarray, n: int) -> TrajectoryStats:
    """All sequences of a recorded decode: traj[it][b][k], tokens[b][max_new],
    iters[b].  Iterations and windows of every sequence are pooled."""
    out = TrajectoryStats()
    for b in range(traj.shape[1]):
        s = analyse(traj[:, b, :], tokens[b], int(min(iters[b], traj.shape[0])), n)
        out.accepted += s.accepted
        out.window_stationary += s.window_stationary
        out.window_iterations += s.window_iterations
    return out
