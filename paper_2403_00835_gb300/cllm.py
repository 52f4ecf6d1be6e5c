"""Python binding of the C ABI in include/cllm.h (argument marshalling only).

Every step of the decode runs in the CUDA library ``_build/libcllm.so``; this
module only converts Python/numpy/torch arguments to the ABI's plain pointers
and sizes.  There is no fallback: if the library is missing or fails to load,
``load()`` raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Sequence

import numpy as np

from . import build as _build

CLLM_OK = 0
STATUS = {0: "CLLM_OK", -1: "CLLM_EINVAL", -2: "CLLM_ENOMEM", -3: "CLLM_ECUDA", -4: "CLLM_ECAPACITY",
          -5: "CLLM_ETIMEOUT", -6: "CLLM_EDEVICE", -7: "CLLM_ESTATE", -8: "CLLM_EUNSUPPORTED"}
CLLM_F32, CLLM_BF16 = 0, 1
CLLM_GUESS_UNIFORM, CLLM_GUESS_FROM_PROMPT = 0, 1
CLLM_BLOCK_REFILL = 0
CLLM_BLOCK_SHRINK = 1
CLLM_BLOCK_LOOKAHEAD = 2

# Every function declared in include/cllm.h.
EXPORTS = ("cllm_create", "cllm_destroy", "cllm_prefill", "cllm_jacobi_step", "cllm_jacobi_decode",
           "cllm_ar_decode", "cllm_status_string", "cllm_decode_begin", "cllm_decode_run",
           "cllm_decode_read", "cllm_set_profiling", "cllm_profile_read",
           "cllm_kernels_per_iteration", "cllm_committed_lengths", "cllm_gemm_bf16_noalloc",
           "cllm_set_option", "cllm_uses_persistent", "cllm_last_cuda_error",
           "cllm_decode_read_trajectory", "cllm_decode_read_stats")
CLLM_OPT_PERSISTENT = 1
CLLM_OPT_PARK_SLOTS = 3
CLLM_OPT_L2_PAIRS = 2
CLLM_OPT_DATAFLOW = 4


class CllmError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {STATUS.get(status, status)} ({_status_string(status)})")


class Arch(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int), ("d_model", ctypes.c_int), ("n_heads", ctypes.c_int),
                ("n_kv_heads", ctypes.c_int), ("head_dim", ctypes.c_int), ("ffn", ctypes.c_int),
                ("vocab", ctypes.c_int), ("rms_eps", ctypes.c_float), ("rope_theta", ctypes.c_float),
                ("dtype", ctypes.c_int), ("max_batch", ctypes.c_int), ("max_seq", ctypes.c_int),
                ("max_block", ctypes.c_int)]


_PP = ctypes.POINTER(ctypes.c_void_p)


class Weights(ctypes.Structure):
    _fields_ = [("tok_emb", ctypes.c_void_p), ("final_norm", ctypes.c_void_p),
                ("lm_head", ctypes.c_void_p), ("attn_norm", _PP), ("wq", _PP), ("wk", _PP),
                ("wv", _PP), ("wo", _PP), ("mlp_norm", _PP), ("w_gate", _PP), ("w_up", _PP),
                ("w_down", _PP)]


class DecodeOpts(ctypes.Structure):
    _fields_ = [("seed", ctypes.c_uint64), ("eos_id", ctypes.c_int), ("guess_init", ctypes.c_int),
                ("block_mode", ctypes.c_int), ("record_cap", ctypes.c_int), ("stats", ctypes.c_int),
                ("ngram", ctypes.c_int)]


class AcceptStats(ctypes.Structure):
    _fields_ = [("iterations", ctypes.c_int64), ("accepted", ctypes.c_int64),
                ("windows", ctypes.c_int64), ("stationary", ctypes.c_int64)]


_lib = None


def library_path() -> str:
    return _build.LIB


def load(build_if_missing: bool = True):
    """Load libcllm.so (building it first if asked and absent).  Raises on failure."""
    global _lib
    if _lib is not None:
        return _lib
    path = _build.LIB
    if not os.path.exists(path):
        if not build_if_missing:
            raise RuntimeError(f"CUDA library not built: {path}")
        path = _build.build()
    lib = ctypes.CDLL(path)
    i32p = ctypes.POINTER(ctypes.c_int32)
    f32p = ctypes.POINTER(ctypes.c_float)
    vp = ctypes.c_void_p
    lib.cllm_create.argtypes = [ctypes.POINTER(Arch), ctypes.POINTER(Weights), vp, ctypes.POINTER(vp)]
    lib.cllm_create.restype = ctypes.c_int
    lib.cllm_destroy.argtypes = [vp]
    lib.cllm_destroy.restype = None
    lib.cllm_prefill.argtypes = [vp, ctypes.c_int, i32p, i32p, i32p]
    lib.cllm_jacobi_step.argtypes = [vp, i32p, ctypes.c_int, i32p, i32p, f32p, f32p]
    lib.cllm_jacobi_decode.argtypes = [vp, ctypes.c_int, i32p, i32p, ctypes.c_int, ctypes.c_int,
                                       ctypes.POINTER(DecodeOpts), i32p, i32p]
    lib.cllm_ar_decode.argtypes = [vp, ctypes.c_int, i32p, i32p, ctypes.c_int, ctypes.c_int, i32p]
    lib.cllm_status_string.argtypes = [ctypes.c_int]
    lib.cllm_status_string.restype = ctypes.c_char_p
    lib.cllm_decode_begin.argtypes = [vp, ctypes.c_int, ctypes.c_int, ctypes.POINTER(DecodeOpts)]
    lib.cllm_decode_run.argtypes = [vp, ctypes.c_int, ctypes.POINTER(ctypes.c_int),
                                    ctypes.POINTER(ctypes.c_int64)]
    lib.cllm_decode_read.argtypes = [vp, i32p, i32p]
    lib.cllm_set_profiling.argtypes = [vp, ctypes.c_int]
    lib.cllm_profile_read.argtypes = [vp, ctypes.POINTER(ctypes.c_char_p), f32p,
                                      ctypes.POINTER(ctypes.c_int), ctypes.c_int]
    lib.cllm_kernels_per_iteration.argtypes = [vp, ctypes.c_int]
    lib.cllm_committed_lengths.argtypes = [vp, i32p]
    lib.cllm_gemm_bf16_noalloc.argtypes = [vp, vp, vp, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                           ctypes.c_int, vp]
    lib.cllm_gemm_bf16_noalloc.restype = ctypes.c_int
    lib.cllm_set_option.argtypes = [vp, ctypes.c_int, ctypes.c_int]
    lib.cllm_set_option.restype = ctypes.c_int
    lib.cllm_uses_persistent.argtypes = [vp, ctypes.c_int]
    lib.cllm_uses_persistent.restype = ctypes.c_int
    lib.cllm_decode_read_trajectory.argtypes = [vp, i32p]
    i64p = ctypes.POINTER(ctypes.c_int64)
    lib.cllm_decode_read_stats.argtypes = [vp, ctypes.POINTER(AcceptStats), i64p, i64p]
    lib.cllm_decode_read_stats.restype = ctypes.c_int
    lib.cllm_last_cuda_error.argtypes = []
    lib.cllm_last_cuda_error.restype = ctypes.c_char_p
    for name in ("cllm_prefill", "cllm_jacobi_step", "cllm_jacobi_decode", "cllm_ar_decode",
                 "cllm_decode_begin", "cllm_decode_run", "cllm_decode_read", "cllm_set_profiling",
                 "cllm_profile_read", "cllm_kernels_per_iteration", "cllm_committed_lengths"):
        getattr(lib, name).restype = ctypes.c_int
    _lib = lib
    return lib


def _status_string(s: int) -> str:
    try:
        return load(build_if_missing=False).cllm_status_string(int(s)).decode()
    except Exception:
        return STATUS.get(s, "unknown")


def _check(rc: int, where: str):
    if rc != CLLM_OK:
        if rc == -3:
            try:
                where += " [" + load(build_if_missing=False).cllm_last_cuda_error().decode() + "]"
            except Exception:
                pass
        raise CllmError(rc, where)


def _i32(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.int32))


def _ip(a: np.ndarray):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_int32))


def _fp(a: np.ndarray):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_float))


def _flatten_prompts(prompts: Sequence[Sequence[int]]):
    lens = _i32([len(p) for p in prompts])
    toks = _i32([t for p in prompts for t in p])
    return toks, lens


class Engine:
    """One cllm context: a decoder's borrowed device weights plus the KV cache,
    scratch and CUDA graphs the library owns."""

    def __init__(self, cfg, weights: dict, max_batch: int, max_seq: int, max_block: int,
                 stream=None):
        import torch
        lib = load()
        self.cfg = cfg
        self.vocab = cfg.vocab
        self._weights = weights  # keep the device tensors alive
        a = Arch(cfg.n_layers, cfg.d_model, cfg.n_heads, cfg.n_kv_heads, cfg.head_dim, cfg.ffn,
                 cfg.vocab, cfg.rms_eps, cfg.rope_theta,
                 CLLM_F32 if cfg.dtype == "f32" else CLLM_BF16, max_batch, max_seq, max_block)
        want = torch.float32 if cfg.dtype == "f32" else torch.bfloat16
        for k, v in weights.items():
            for t in (v if isinstance(v, list) else [v]):
                if not (t.is_cuda and t.dtype == want and t.is_contiguous()):
                    raise ValueError(f"weight {k}: need contiguous {want} CUDA tensors")
        self._lists = {}
        for k in ("attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "w_gate", "w_up", "w_down"):
            arr = (ctypes.c_void_p * cfg.n_layers)(*[t.data_ptr() for t in weights[k]])
            self._lists[k] = arr
        wl = self._lists
        w = Weights(weights["tok_emb"].data_ptr(), weights["final_norm"].data_ptr(),
                    weights["lm_head"].data_ptr(),
                    *[ctypes.cast(wl[k], _PP) for k in ("attn_norm", "wq", "wk", "wv", "wo", "mlp_norm",
                                                         "w_gate", "w_up", "w_down")])
        self._stream = stream
        sp = ctypes.c_void_p(stream.cuda_stream if stream is not None else None)
        h = ctypes.c_void_p()
        _check(lib.cllm_create(ctypes.byref(a), ctypes.byref(w), sp, ctypes.byref(h)), "cllm_create")
        self._h = h
        self._lib = lib
        self.max_batch, self.max_seq, self.max_block = max_batch, max_seq, max_block
        self.B = 0

    def close(self):
        if getattr(self, "_h", None) is not None and self._h.value:
            self._lib.cllm_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # ---- calls -------------------------------------------------------------
    def prefill(self, prompts: Sequence[Sequence[int]]) -> np.ndarray:
        toks, lens = _flatten_prompts(prompts)
        heads = np.zeros(len(prompts), dtype=np.int32)
        _check(self._lib.cllm_prefill(self._h, len(prompts), _ip(toks), _ip(lens), _ip(heads)),
               "cllm_prefill")
        self.B = len(prompts)
        return heads

    def jacobi_step(self, guess, want_gap: bool = True, want_logits: bool = False) -> dict:
        g = _i32(guess)
        B, n = g.shape
        nxt = np.zeros((B, n), dtype=np.int32)
        acc = np.zeros(B, dtype=np.int32)
        gap = np.zeros((B, n), dtype=np.float32) if want_gap else None
        lg = np.zeros((B, n, self.vocab), dtype=np.float32) if want_logits else None
        _check(self._lib.cllm_jacobi_step(self._h, _ip(g), n, _ip(nxt), _ip(acc),
                                          _fp(gap) if gap is not None else None,
                                          _fp(lg) if lg is not None else None), "cllm_jacobi_step")
        return {"next": nxt, "accepted": acc, "gap": gap, "logits": lg}

    def jacobi_decode(self, prompts, n: int, max_new: int, seed: int = 0, eos_id: int = -1,
                      guess_init: int = CLLM_GUESS_UNIFORM, block_mode: int = CLLM_BLOCK_REFILL,
                      record_cap: int = 0, stats: bool = False, ngram: int = 4):
        """Tokens [B][max_new] and iterations [B]; with record_cap > 0 also the
        trajectory [record_cap][B][n] (-1 outside the window).  With stats the
        device keeps the acceptance statistics (read with decode_read_stats)."""
        toks, lens = _flatten_prompts(prompts)
        B = len(prompts)
        out = np.zeros((B, max_new), dtype=np.int32)
        its = np.zeros(B, dtype=np.int32)
        o = DecodeOpts(seed, eos_id, guess_init, block_mode, record_cap, 1 if stats else 0, ngram)
        _check(self._lib.cllm_jacobi_decode(self._h, B, _ip(toks), _ip(lens), n, max_new,
                                            ctypes.byref(o), _ip(out), _ip(its)), "cllm_jacobi_decode")
        self.B = B
        self._dec_n = n
        if record_cap > 0:
            traj = np.zeros((record_cap, B, n), dtype=np.int32)
            _check(self._lib.cllm_decode_read_trajectory(self._h, _ip(traj)),
                   "cllm_decode_read_trajectory")
            return out, its, traj
        return out, its

    def ar_decode(self, prompts, max_new: int, eos_id: int = -1):
        toks, lens = _flatten_prompts(prompts)
        B = len(prompts)
        out = np.zeros((B, max_new), dtype=np.int32)
        _check(self._lib.cllm_ar_decode(self._h, B, _ip(toks), _ip(lens), max_new, eos_id, _ip(out)),
               "cllm_ar_decode")
        self.B = B
        return out

    def decode_begin(self, n: int, max_new: int, seed: int = 0, eos_id: int = -1,
                     guess_init: int = CLLM_GUESS_UNIFORM, block_mode: int = CLLM_BLOCK_REFILL,
                     stats: bool = False, ngram: int = 4):
        o = DecodeOpts(seed, eos_id, guess_init, block_mode, 0, 1 if stats else 0, ngram)
        _check(self._lib.cllm_decode_begin(self._h, n, max_new, ctypes.byref(o)), "cllm_decode_begin")
        self._dec_max_new = max_new
        self._dec_n = n

    def decode_read_stats(self):
        """The device's acceptance statistics of the current decode: totals
        (iterations, accepted, windows, stationary) and the histograms
        acc_hist[a] (iterations accepting a tokens) and win_hist[s] (windows
        with s stationary tokens), both [n + 1]."""
        n = self._dec_n
        st = AcceptStats()
        ah = np.zeros(n + 1, dtype=np.int64)
        wh = np.zeros(n + 1, dtype=np.int64)
        _check(self._lib.cllm_decode_read_stats(self._h, ctypes.byref(st),
                                                ah.ctypes.data_as(ctypes.POINTER(ctypes.c_int64)),
                                                wh.ctypes.data_as(ctypes.POINTER(ctypes.c_int64))),
               "cllm_decode_read_stats")
        return {"iterations": st.iterations, "accepted": st.accepted, "windows": st.windows,
                "stationary": st.stationary, "acc_hist": ah, "win_hist": wh}

    def decode_run(self, max_iters: int):
        it = ctypes.c_int(0)
        com = ctypes.c_int64(0)
        _check(self._lib.cllm_decode_run(self._h, max_iters, ctypes.byref(it), ctypes.byref(com)),
               "cllm_decode_run")
        return it.value, com.value

    def decode_read(self):
        out = np.zeros((self.B, self._dec_max_new), dtype=np.int32)
        its = np.zeros(self.B, dtype=np.int32)
        _check(self._lib.cllm_decode_read(self._h, _ip(out), _ip(its)), "cllm_decode_read")
        return out, its

    def set_persistent(self, on: bool):
        _check(self._lib.cllm_set_option(self._h, CLLM_OPT_PERSISTENT, 1 if on else 0), "cllm_set_option")

    def set_l2_pairs(self, pairs: int):
        _check(self._lib.cllm_set_option(self._h, CLLM_OPT_L2_PAIRS, int(pairs)), "cllm_set_option")

    def set_park_slots(self, tiles: int):
        _check(self._lib.cllm_set_option(self._h, CLLM_OPT_PARK_SLOTS, int(tiles)), "cllm_set_option")

    def set_dataflow(self, on: bool):
        _check(self._lib.cllm_set_option(self._h, CLLM_OPT_DATAFLOW, 1 if on else 0), "cllm_set_option")

    def uses_persistent(self, n: int) -> bool:
        r = self._lib.cllm_uses_persistent(self._h, n)
        if r < 0:
            raise CllmError(r, "cllm_uses_persistent")
        return bool(r)

    def set_profiling(self, on: bool):
        _check(self._lib.cllm_set_profiling(self._h, 1 if on else 0), "cllm_set_profiling")

    def profile_read(self) -> dict:
        cap = 64
        names = (ctypes.c_char_p * cap)()
        ms = np.zeros(cap, dtype=np.float32)
        cnt = (ctypes.c_int * cap)()
        k = self._lib.cllm_profile_read(self._h, names, _fp(ms), cnt, cap)
        return {names[i].decode(): (float(ms[i]), int(cnt[i])) for i in range(min(k, cap))}

    def kernels_per_iteration(self, n: int) -> int:
        r = self._lib.cllm_kernels_per_iteration(self._h, n)
        if r < 0:
            raise CllmError(r, "cllm_kernels_per_iteration")
        return r

    def committed_lengths(self) -> np.ndarray:
        out = np.zeros(self.B, dtype=np.int32)
        _check(self._lib.cllm_committed_lengths(self._h, _ip(out)), "cllm_committed_lengths")
        return out
