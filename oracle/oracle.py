"""Oracle for Jacobi decoding of a LLaMA-style decoder (CLLMs, arXiv 2403.00835).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this module.  The product path (the
CUDA library behind ``include/cllm.h`` and its binding in
``paper_2403_00835_gb300``) never imports it, and the two share no code.

Layout
  * ``cllm_oracle.c``  -- fp64 forward pass of the decoder with a KV cache
                          (the map p(. | y_<i, x) of Eq. 1 and Eq. 3).
  * this module        -- ctypes binding, argmax/top-2, the guess generator and
                          the decoding algorithms, each written in the paper's
                          order:
        ``ar_decode``       greedy AR decoding, Eq. 1 (Sec. 3.1).
        ``jacobi_decode``   Jacobi decoding with KV cache (Sec. 3.1 "Jacobi
                            Decoding with KV Cache", App. C Alg. 3) in two block
                            policies: ``refill`` keeps the block at width n by
                            appending fresh guesses after each commit; ``shrink``
                            follows Alg. 3 (the state shrinks by the accepted
                            count until the n-token window is fixed, then the next
                            window starts as in Alg. 1's x <- cat(x, y*)); and
                            ``lookahead``, the refill policy with an n-gram pool
                            (Sec. 3.3's combination with lookahead decoding,
                            see ``ngram_pool_step``); ``verify``, the refill
                            policy with a verification branch of several
                            pooled n-grams (``ngram_pool_push``,
                            ``verify_candidates``).
        ``jacobi_step``     one iteration of the above from an explicit block.
        ``jacobi_vanilla``  Eq. 3 iterated without any cache until
                            y^(k) = y^(k-1) (Sec. 3.1), used only as a pin.

Readings of the paper this oracle takes:
  * The first block token is the head: the prediction from the committed
    context, correct by construction (Alg. 3's y_0 from the prefill).  The
    accepted count of a step is a = 1 + the number of leading positions k >= 1
    with block[k] == P[k-1], where P[k] is the argmax of row k.  Alg. 3's i*
    is this quantity; its printed index range is garbled.
  * The next head is P[a-1]; refill keeps P[a-1:] and appends a-1 fresh guesses.
  * Argmax ties go to the lowest token id; gap = top1 - top2 of the raw logits
    (duplicates allowed, so gap may be 0).
  * Lookahead combination (Sec. 3.3 gives one sentence: n-grams generated
    in previous Jacobi iterations are collected as candidates and verified in
    the next iteration).  Reading: each iteration's predictions P are an
    n-gram source -- for every k with k + N - 1 < n, key P[k] and value
    P[k+1..k+N-1] (N = n-gram size), later k replacing earlier ones under the
    same key.  Before the iteration's n-grams enter the pool, the next block
    (the refill block) takes the pool's value for its head P[a-1], if there is
    one, in slots 1..N-1; the next iteration's acceptance verifies it.  One
    candidate per iteration, inside the Jacobi block: no separate lookahead
    window and no parallel verification branch.
  * The same combination with a verification branch (``verify``): the same
    n-gram source, but a key keeps up to G distinct values, most recent first.
    Each iteration verifies, beside the Jacobi block, every pooled value c of
    the block's head h, each as its own causal sequence [h, c] over the
    committed cache (in one batched pass this is a mask under which a
    candidate's rows see the cache, h and their own earlier rows only).  The
    longest accepted run is committed (the block wins ties, then the most
    recent n-gram) with its own K/V; the next head is that run's prediction
    after its last accepted row, followed by the block's predictions for the
    positions after it and fresh guesses (the refill block when the block
    won).  The iteration's n-grams enter the pool after the verification.
  * Guesses ("random tokens", Alg. 3) are drawn from a counter-based
    splitmix64 stream (Vigna), keyed by (seed, sequence b, iteration, slot):
    uniform over the vocabulary, or uniform over the prompt's tokens.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from dataclasses import dataclass, field
from typing import Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "cllm_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

ORC_F32 = 0
ORC_BF16 = 1


def build(force: bool = False) -> str:
    """Compile cllm_oracle.c into liboracle.so (gcc, OpenMP).  Returns its path."""
    with _lock:
        stale = (not os.path.exists(_LIB)) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC)
        if force or stale:
            tmp = _LIB + f".tmp{os.getpid()}"
            cmd = ["gcc", "-O3", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-Wall",
                   _SRC, "-o", tmp, "-lm"]
            subprocess.run(cmd, check=True)
            os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        dp = ctypes.POINTER(ctypes.c_double)
        ip = ctypes.POINTER(ctypes.c_int32)
        lib.orc_create.restype = ctypes.c_void_p
        lib.orc_create.argtypes = [ip, dp, ctypes.c_int, ctypes.POINTER(ctypes.c_void_p), ctypes.c_int]
        lib.orc_destroy.argtypes = [ctypes.c_void_p]
        lib.orc_forward.restype = ctypes.c_int
        lib.orc_forward.argtypes = [ctypes.c_void_p, ip, ctypes.c_int, ctypes.c_int, ip, ctypes.c_int, dp]
        lib.orc_rmsnorm.argtypes = [dp, dp, ctypes.c_int, ctypes.c_double, dp]
        lib.orc_rope.argtypes = [dp, ctypes.c_int, ctypes.c_int, ctypes.c_double]
        lib.orc_silu.restype = ctypes.c_double
        lib.orc_silu.argtypes = [ctypes.c_double]
        lib.orc_attend.argtypes = [dp, dp, dp, ctypes.c_int, ctypes.c_int, ctypes.c_int, dp]
        lib.orc_num_threads.restype = ctypes.c_int
        lib.orc_set_num_threads.argtypes = [ctypes.c_int]
        _lib = lib
    return _lib


def _dptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_double))


def _iptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_int32))


# ---- layer primitives (thin wrappers, used by the pin tests) ----------------

def rmsnorm(x, g, eps):
    x = np.ascontiguousarray(x, dtype=np.float64)
    g = np.ascontiguousarray(g, dtype=np.float64)
    out = np.empty_like(x)
    _load().orc_rmsnorm(_dptr(x), _dptr(g), x.shape[0], float(eps), _dptr(out))
    return out


def rope(v, pos, theta):
    v = np.array(v, dtype=np.float64)
    _load().orc_rope(_dptr(v), v.shape[0], int(pos), float(theta))
    return v


def silu(z: float) -> float:
    return _load().orc_silu(float(z))


def attend(q, k, v):
    """q [hd], k/v [n, hd] -> softmax(q k^T / sqrt(hd)) v."""
    q = np.ascontiguousarray(q, dtype=np.float64)
    k = np.ascontiguousarray(k, dtype=np.float64)
    v = np.ascontiguousarray(v, dtype=np.float64)
    out = np.empty(q.shape[0], dtype=np.float64)
    _load().orc_attend(_dptr(q), _dptr(k), _dptr(v), k.shape[0], q.shape[0], q.shape[0], _dptr(out))
    return out


def num_threads() -> int:
    return _load().orc_num_threads()


def set_num_threads(n: int) -> None:
    _load().orc_set_num_threads(int(n))


# ---- argmax / top-2 (Eq. 1 and Eq. 3's argmax) ------------------------------

def argmax_top2(row: np.ndarray):
    """Return (token, gap): the lowest index attaining the maximum logit, and
    top1 - top2 where top2 is the largest logit of the remaining entries."""
    row = np.asarray(row, dtype=np.float64)
    tok = int(np.argmax(row))  # first occurrence = lowest index on ties
    top1 = row[tok]
    rest = np.delete(row, tok)
    top2 = rest.max() if rest.size else -np.inf
    return tok, float(top1 - top2)


# ---- guess generator: counter-based splitmix64 (Vigna) -----------------------

_M64 = (1 << 64) - 1
_GAMMA = 0x9E3779B97F4A7C15


def splitmix64_output(seed: int, i: int) -> int:
    """The i-th output (i >= 1) of splitmix64 started from state ``seed``:
    state_i = seed + i * 0x9E3779B97F4A7C15 (mod 2^64), then the published
    mixing function (xor-shift 30, * 0xBF58476D1CE4E5B9, xor-shift 27,
    * 0x94D049BB133111EB, xor-shift 31)."""
    z = (seed + i * _GAMMA) & _M64
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _M64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _M64
    return z ^ (z >> 31)


def guess_counter(b: int, step: int, slot: int) -> int:
    """Counter of the guess for sequence b, iteration ``step``, block slot."""
    assert 0 <= b < (1 << 24) and 0 <= step < (1 << 24) and 0 <= slot < (1 << 16)
    return (b << 40) | (step << 16) | slot


def guess_token(seed: int, b: int, step: int, slot: int, vocab: int,
                prompt: Sequence[int] | None = None) -> int:
    """A random initial/refill token.  Uniform over [0, vocab) by the
    multiply-high of the output's top 32 bits, or (``prompt`` given) a uniform
    pick among the prompt's tokens ("random tokens from x", Alg. 3)."""
    r = splitmix64_output(seed & _M64, guess_counter(b, step, slot) + 1) >> 32
    if prompt is None:
        return (r * vocab) >> 32
    return int(prompt[(r * len(prompt)) >> 32])


# ---- model ------------------------------------------------------------------

@dataclass
class OracleArch:
    n_layers: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    ffn: int
    vocab: int
    rms_eps: float
    rope_theta: float


def _as_host(a, wdtype):
    """numpy view of a weight: float32 for fp32 weights, uint16 bit patterns
    for bf16 weights.  Accepts numpy arrays or CPU torch tensors."""
    if hasattr(a, "detach"):  # torch tensor
        t = a.detach().contiguous()
        if wdtype == ORC_BF16:
            import torch
            return t.view(torch.int16).numpy().view(np.uint16)
        return t.float().numpy()
    a = np.ascontiguousarray(a)
    if wdtype == ORC_BF16:
        assert a.dtype == np.uint16
    else:
        a = a.astype(np.float32, copy=False)
    return a


class OracleModel:
    """Weights of one decoder, borrowed by the C forward pass.

    ``weights`` maps 'tok_emb', 'final_norm', 'lm_head' to arrays and
    'attn_norm', 'wq', 'wk', 'wv', 'wo', 'mlp_norm', 'w_gate', 'w_up', 'w_down'
    to per-layer lists.  Matrices are [out, in] row-major."""

    LAYER_KEYS = ("attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "w_gate", "w_up", "w_down")

    def __init__(self, arch: OracleArch, weights: dict, wdtype: int):
        self.arch = arch
        self.wdtype = wdtype
        self._keep = []
        ptrs = []
        for key in ("tok_emb", "final_norm", "lm_head"):
            a = _as_host(weights[key], wdtype)
            self._keep.append(a)
            ptrs.append(a.ctypes.data)
        for l in range(arch.n_layers):
            for key in self.LAYER_KEYS:
                a = _as_host(weights[key][l], wdtype)
                self._keep.append(a)
                ptrs.append(a.ctypes.data)
        self._ptrs = (ctypes.c_void_p * len(ptrs))(*ptrs)
        self._iarch = np.array([arch.n_layers, arch.d_model, arch.n_heads, arch.n_kv_heads,
                                arch.head_dim, arch.ffn, arch.vocab], dtype=np.int32)
        self._farch = np.array([arch.rms_eps, arch.rope_theta], dtype=np.float64)

    def session(self, max_pos: int) -> "OracleSession":
        return OracleSession(self, max_pos)


class OracleSession:
    """One sequence's KV cache over ``max_pos`` positions."""

    def __init__(self, model: OracleModel, max_pos: int):
        self.model = model
        lib = _load()
        self._h = lib.orc_create(_iptr(model._iarch), _dptr(model._farch), model.wdtype,
                                 model._ptrs, int(max_pos))
        if not self._h:
            raise MemoryError("oracle cache allocation failed")
        self.max_pos = max_pos

    def close(self):
        if self._h:
            _load().orc_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def forward(self, tokens: Sequence[int], start_pos: int, rows: Sequence[int] | None = None):
        """Logits [len(rows), vocab] (fp64) of the given rows of a forward over
        ``tokens`` at positions start_pos..; writes their K/V into the cache."""
        toks = np.ascontiguousarray(np.asarray(tokens, dtype=np.int32))
        if rows is None:
            rows = range(len(toks))
        rows = np.ascontiguousarray(np.asarray(list(rows), dtype=np.int32))
        out = np.empty((len(rows), self.model.arch.vocab), dtype=np.float64)
        rc = _load().orc_forward(self._h, _iptr(toks), len(toks), int(start_pos), _iptr(rows),
                                 len(rows), _dptr(out))
        if rc != 0:
            raise ValueError("oracle forward: bad arguments")
        return out


# ---- decoding algorithms ----------------------------------------------------

@dataclass
class StepResult:
    pred: list            # P[k] = argmax of row k (the new y^(j+1) values)
    gap: list             # top1 - top2 of row k
    accepted: int         # a
    logits: np.ndarray | None = None


def jacobi_step(sess: OracleSession, block: Sequence[int], L: int, keep_logits: bool = False) -> StepResult:
    """One Jacobi iteration with KV cache from committed length L: one forward
    over the block (Eq. 3: all rows in one causal pass), then the accepted
    count a (Alg. 3's fast-forwarded count, with the head counted)."""
    logits = sess.forward(block, L)
    pred, gap = [], []
    for r in logits:
        t, g = argmax_top2(r)
        pred.append(t)
        gap.append(g)
    a = 1
    while a < len(block) and block[a] == pred[a - 1]:
        a += 1
    return StepResult(pred, gap, a, logits if keep_logits else None)


def prefill(sess: OracleSession, prompt: Sequence[int]):
    """Prefill (Alg. 3, first forward): cache of the prompt and the head
    y_1 = argmax p(. | x).  Returns (head, gap, logits_row)."""
    logits = sess.forward(prompt, 0, rows=[len(prompt) - 1])
    tok, gap = argmax_top2(logits[0])
    return tok, gap, logits[0]


@dataclass
class DecodeResult:
    tokens: list
    iterations: int
    accepted: list = field(default_factory=list)   # a per iteration
    min_gap: list = field(default_factory=list)    # per iteration: min gap over the committed rows' predictions
    min_gap_all: list = field(default_factory=list)  # per iteration: min gap over every row of the block
    trajectory: list = field(default_factory=list)  # blocks fed to each iteration
    steps: list = field(default_factory=list)  # StepResult of each iteration (keep_steps)
    branch: list = field(default_factory=list)  # verify: per iteration -1 (the block) or the candidate committed
    candidates: list = field(default_factory=list)  # verify (record): the n-grams verified per iteration


def ar_decode(model: OracleModel, prompt: Sequence[int], max_new: int, eos_id: int = -1) -> DecodeResult:
    """Greedy AR decoding, Eq. 1: y_i = argmax p(y | y_<i, x), one pass per token."""
    sess = model.session(len(prompt) + max_new + 1)
    head, gap, _ = prefill(sess, prompt)
    out, gaps = [], [gap]
    L = len(prompt)
    passes = 0
    while True:
        out.append(head)
        if head == eos_id or len(out) >= max_new:
            break
        logits = sess.forward([head], L)
        L += 1
        passes += 1
        head, g = argmax_top2(logits[0])
        gaps.append(g)
    sess.close()
    return DecodeResult(out, passes, [1] * len(out), gaps[:len(out)])


def ngram_pool_step(pool: dict, pred: Sequence[int], a: int, block: Sequence[int], ngram: int) -> list:
    """The lookahead policy's step (reading of Sec. 3.3 in the module header):
    the refill ``block`` takes the pool's (ngram - 1)-token continuation of
    its head pred[a-1] in slots 1.., then this iteration's n-grams of ``pred``
    enter ``pool`` (key pred[k], value pred[k+1 .. k+ngram-1], k ascending).
    Returns the next block; ``pool`` is updated in place."""
    W = ngram - 1
    out = list(block)
    cand = pool.get(pred[a - 1])
    if cand is not None:
        w = min(W, len(out) - 1)
        out[1:1 + w] = cand[:w]
    for k in range(len(pred) - W):
        pool[pred[k]] = list(pred[k + 1:k + 1 + W])
    return out


def ngram_pool_push(pool: dict, pred: Sequence[int], ngram: int, ncand: int) -> None:
    """The verification branch's pool (reading of Sec. 3.3 in the module
    header): this iteration's n-grams of ``pred`` (key pred[k], value
    pred[k+1 .. k+ngram-1], k ascending) enter ``pool``, where a key keeps at
    most ``ncand`` distinct values, the most recently entered first (an
    n-gram already held moves to the front)."""
    W = ngram - 1
    for k in range(len(pred) - W):
        v = tuple(pred[k + 1:k + 1 + W])
        held = pool.setdefault(pred[k], [])
        if v in held:
            held.remove(v)
        held.insert(0, v)
        del held[ncand:]


def verify_candidates(sess: OracleSession, head: int, cands: Sequence[Sequence[int]], L: int) -> list:
    """The verification branch of one iteration: candidate c is checked by
    the causal forward of [head, c] over the committed cache of length L,
    alone (no row of another candidate or of the Jacobi block is visible to
    it).  Its accepted count is defined as the Jacobi block's: 1 + the number
    of leading j with c[j] equal to the prediction of the row before it.
    Returns (accepted, predictions, gaps) per candidate; the cache past L
    holds the last candidate's K/V afterwards."""
    out = []
    for c in cands:
        toks = [head] + list(c)
        q, gaps = [], []
        for r in sess.forward(toks, L):
            t, gp = argmax_top2(r)
            q.append(t)
            gaps.append(gp)
        a = 1
        while a < len(toks) and toks[a] == q[a - 1]:
            a += 1
        out.append((a, q, gaps))
    return out


def jacobi_decode(model: OracleModel, prompt: Sequence[int], n: int, max_new: int, seed: int,
                  b: int = 0, mode: str = "refill", guess_init: str = "uniform",
                  eos_id: int = -1, record: bool = False, keep_steps: bool = False,
                  ngram: int = 4, ncand: int = 4) -> DecodeResult:
    """Jacobi decoding with KV cache (Alg. 3) of one sequence ``b``.

    Each iteration forwards the current block over the committed cache,
    accepts a tokens (a >= 1), commits them (their K/V stay in the cache), and
    forms the next block from the remaining predictions (Alg. 3's
    z_next <- z_next[>= i*]); ``refill`` tops the block up to n with fresh
    guesses, ``shrink`` lets it shrink until the window is fixed.
    ``verify`` adds the verification branch (module header): up to ``ncand``
    pooled n-grams following the head are verified beside the block, and the
    longest accepted run is committed (the block wins ties, then the most
    recent n-gram).
    ``record`` keeps the block of every iteration (and, for ``verify``, the
    candidates verified) and ``keep_steps`` every iteration's StepResult with
    its logits (recorded only, never used)."""
    assert mode in ("refill", "shrink", "lookahead", "verify") and n >= 1 and max_new >= 1
    assert mode not in ("lookahead", "verify") or ngram >= 2
    assert mode != "verify" or ncand >= 1
    pool: dict = {}
    V = model.arch.vocab
    src = list(prompt) if guess_init == "prompt" else None

    def g(step, slot):
        return guess_token(seed, b, step, slot, V, src)

    sess = model.session(len(prompt) + max_new + n + 1)
    head, _, _ = prefill(sess, prompt)
    L = len(prompt)
    block = [head] + [g(0, i) for i in range(1, n)]
    res = DecodeResult([], 0)
    while len(res.tokens) < max_new:
        if record:
            res.trajectory.append(list(block))
        st = jacobi_step(sess, block, L, keep_logits=keep_steps)
        if keep_steps:
            res.steps.append(st)
        m = len(block)
        a = st.accepted
        # the committed run: the block's, or a verified candidate's
        toks, pred, gaps, gaps_all = block, st.pred, st.gap, list(st.gap)
        if mode == "verify":
            cands = list(pool.get(block[0], []))  # from earlier iterations only
            if record:
                res.candidates.append([list(c) for c in cands])
            best = -1
            for i, (ac, q, gq) in enumerate(verify_candidates(sess, block[0], cands, L)):
                gaps_all += gq
                if ac > a:
                    a, toks, pred, gaps, best = ac, [block[0]] + list(cands[i]), q, gq, i
            res.branch.append(best)
        stop = False
        if eos_id >= 0 and eos_id in toks[:a]:
            a = toks.index(eos_id) + 1
            stop = True
        a = min(a, max_new - len(res.tokens))
        res.tokens += toks[:a]
        res.accepted.append(a)
        res.min_gap.append(min(gaps[:a]))
        res.min_gap_all.append(min(gaps_all))
        if mode == "verify" and cands:
            # the cache past L holds the last forward's K/V: commit the
            # accepted tokens' own
            sess.forward(toks[:a], L, rows=[])
        L += a
        res.iterations += 1
        if stop or len(res.tokens) >= max_new:
            break
        it = res.iterations
        if mode in ("refill", "lookahead"):
            block = st.pred[a - 1:] + [g(it, i) for i in range(m - a + 1, m)]
            if mode == "lookahead":
                block = ngram_pool_step(pool, st.pred, a, block, ngram)
        elif mode == "verify":
            # the committed run's next head, then the block's own predictions
            # for the positions after it (refill when the block won)
            block = [pred[a - 1]] + st.pred[a:m] + [g(it, i) for i in range(max(1, m - a + 1), m)]
            ngram_pool_push(pool, st.pred, ngram, ncand)
        elif a == m:
            block = [st.pred[m - 1]] + [g(it, i) for i in range(1, n)]
        else:
            block = st.pred[a - 1:m - 1]
    sess.close()
    return res


def jacobi_vanilla(model: OracleModel, prompt: Sequence[int], y0: Sequence[int]):
    """Eq. 3 without a cache: every iteration recomputes [x; y^(j)] from scratch;
    exits at the first k with y^(k) = y^(k-1) (Sec. 3.1).  Returns (y*, k)."""
    y = list(y0)
    n = len(y)
    nx = len(prompt)
    k = 0
    while True:
        seq = list(prompt) + y[:n - 1]
        sess = model.session(len(seq))
        logits = sess.forward(seq, 0, rows=range(nx - 1, nx - 1 + n))
        sess.close()
        y_new = [argmax_top2(r)[0] for r in logits]
        k += 1
        if y_new == y:
            return y, k
        y = y_new
