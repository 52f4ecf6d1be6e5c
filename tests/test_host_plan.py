"""Host logic of the weight-GEMM work split (no GPU): the properties the CUDA
path's bit-identity rests on.  A token column's result must not depend on how
many columns a launch carries (so that a Jacobi step over n rows computes each
row exactly as an AR step does, and the fixed point equals greedy decoding bit
for bit, Sec. 3.1): for T <= 256 the split-K partition of the (tile, chunk)
space depends on the weight shape and the SM count only.  The ranges cover
every chunk once, and a tile shared by several CTAs is reduced by the CTA for
which it is the last segment of its range."""
import ctypes

import pytest

from paper_2403_00835_gb300.cllm import load

SMS = 152
# 7B-shaped launches: (weight tiles, K) of QKV, O, gate/up (64-row halves), down, LM head
SHAPES_7B = {
    "qkv": (3 * 4096 // 128, 4096),
    "o": (4096 // 128, 4096),
    "gateup": ((11008 + 63) // 64, 4096),
    "down": (4096 // 128, 11008),
    "lmhead": ((32000 + 127) // 128, 4096),
}
FIELDS = ("mtiles", "ntiles", "kchunks", "cpc", "bn", "bn_max", "maxc", "grid")


@pytest.fixture(scope="module")
def plan():
    lib = load()
    f = lib.cllm_test_plan_gemm
    f.argtypes = [ctypes.c_int] * 4 + [ctypes.POINTER(ctypes.c_int)]
    f.restype = ctypes.c_int

    def run(mtiles, K, T, sms=SMS):
        out = (ctypes.c_int * 8)()
        assert f(mtiles, K, T, sms, out) == 0
        return dict(zip(FIELDS, list(out)))
    return run


@pytest.mark.parametrize("name", sorted(SHAPES_7B))
def test_split_is_independent_of_token_count(plan, name):
    mtiles, K = SHAPES_7B[name]
    ref = plan(mtiles, K, 1)
    for T in (2, 15, 16, 17, 32, 48, 64, 100, 128, 129, 200, 256):
        p = plan(mtiles, K, T)
        for k in ("ntiles", "kchunks", "cpc", "maxc", "grid"):
            assert p[k] == ref[k], (name, T, k)
        assert p["bn"] == -(-T // 16) * 16
        assert p["bn_max"] == min(b for b in (32, 64, 128, 256) if b >= p["bn"])


@pytest.mark.parametrize("name", sorted(SHAPES_7B))
@pytest.mark.parametrize("sms", [1, 7, 148, 152])
def test_ranges_cover_chunks_and_owners_end_ranges(plan, name, sms):
    mtiles, K = SHAPES_7B[name]
    p = plan(mtiles, K, 16, sms)
    kc, cpc, grid = p["kchunks"], p["cpc"], p["grid"]
    total = mtiles * kc
    # even chunk counts: every tile and every range starts on a pair of chunks
    assert kc == -(-(-(-K // 64)) // 2) * 2
    assert kc % 2 == 0 and cpc % 2 == 0
    assert grid <= sms
    ranges = [(c * cpc, min(total, (c + 1) * cpc)) for c in range(grid)]
    assert ranges[0][0] == 0 and ranges[-1][1] == total
    assert all(a < b for a, b in ranges)
    assert all(ranges[i][1] == ranges[i + 1][0] for i in range(grid - 1))
    maxc = 1
    for u in range(mtiles):
        lo, hi = u * kc, (u + 1) * kc
        sharing = [c for c, (a, b) in enumerate(ranges) if a < hi and b > lo]
        first, last = sharing[0], sharing[-1]
        assert sharing == list(range(first, last + 1))
        assert first == lo // cpc and last == (hi - 1) // cpc
        maxc = max(maxc, len(sharing))
        if len(sharing) > 1:
            # the owner's range ends inside this tile: it is its last segment
            assert lo < ranges[first][1] < hi
            # every other contributor starts its range inside this tile
            assert all(lo < ranges[c][0] < hi for c in sharing[1:])
    assert maxc == p["maxc"]


def test_wide_launches_take_whole_tiles(plan):
    mtiles, K = SHAPES_7B["qkv"]
    for T in (257, 512, 2048):
        p = plan(mtiles, K, T)
        assert p["bn"] == p["bn_max"] == 256
        assert p["ntiles"] == -(-T // 256)
        assert p["maxc"] == 1
        assert p["cpc"] % p["kchunks"] == 0
        units = mtiles * p["ntiles"]
        assert p["grid"] * (p["cpc"] // p["kchunks"]) >= units


def test_bad_arguments_are_rejected():
    lib = load()
    f = lib.cllm_test_plan_gemm
    f.argtypes = [ctypes.c_int] * 4 + [ctypes.POINTER(ctypes.c_int)]
    f.restype = ctypes.c_int
    out = (ctypes.c_int * 8)()
    assert f(0, 64, 16, 152, out) == -1
    assert f(4, 64, 0, 152, out) == -1
    assert f(4, 64, 16, 0, out) == -1
    assert f(4, 64, 16, 152, None) == -1
