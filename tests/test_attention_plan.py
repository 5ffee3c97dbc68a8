"""The attention tile plan (host logic, no GPU).

dopr_debug_attention_plan returns the tiles dopr_score launches for one
document's run of pairs (the prefix-plus-causal attention of Sec. 3.4).  The
rule: tiles take consecutive packed tokens, at most rows_per_tile of them and
at most 16 pairs; a tile's key columns are the prefix (rounded up to 64)
followed by one 16-aligned segment per pair it touches, each running from the
pair's first token to the tile's last; a tensor-core tile keeps within 256
key columns and ends only where the next token would break a limit; a long
tile (no key limit) is made only when the first token alone needs more than
256 columns.  Checked on cases worked by hand, on invariants, and against an
independent greedy restatement on random runs.
"""
import numpy as np
import pytest

from paper_2609_03311_gb300 import build as libbuild
from paper_2609_03311_gb300 import dopr

MAX_KEYS, MAX_SEGS = 256, 16


@pytest.fixture(scope="module")
def lib():
    libbuild.build()
    return dopr.load()


def c16(x):
    return (x + 15) // 16 * 16


def c64(x):
    return (x + 63) // 64 * 64


def decode(plan):
    out = []
    for row in plan:
        kind, tb, n, keys, nseg = (int(x) for x in row[:5])
        segs = [((int(v) >> 16) & 0xFFFF, int(np.int16(np.uint16(int(v) & 0xFFFF)))) for v in row[8:8 + nseg]]
        out.append((kind, tb, n, keys, segs))
    return out


def reference_plan(m, tt, lens):
    """The same rule, restated token by token from the pairs' extents."""
    starts = np.concatenate([[0], np.cumsum(lens)])
    total = int(starts[-1])

    def touched(lo, hi):  # pairs with a token in [lo, hi]
        return [p for p in range(len(lens)) if starts[p] <= hi and starts[p + 1] > lo]

    def keys_of(lo, t):
        return c64(m) + sum(c16(min(starts[p + 1], t + 1) - starts[p]) for p in touched(lo, t))

    tiles, tok = [], 0
    while tok < total:
        def grow(limit):
            n = 0
            while n < tt and tok + n < total:
                t = tok + n
                if len(touched(tok, t)) > MAX_SEGS or (limit and keys_of(tok, t) > MAX_KEYS):
                    break
                n += 1
            return n

        n, kind = grow(True), 0
        if n == 0:
            n, kind = grow(False), 1
        last = tok + n - 1
        segs = [(min(starts[p + 1], last + 1) - starts[p], starts[p] - tok) for p in touched(tok, last)]
        tiles.append((kind, tok, n, keys_of(tok, last), segs))
        tok += n
    return tiles


def test_long_query_splits_into_tensor_core_then_long_tiles(lib):
    # m = 128, 32 tokens per tile, one pair of 200 tokens: own keys grow by 32 per tile
    tiles = decode(dopr.attention_plan(128, 32, [200]))
    assert [(k, tb, n, keys) for k, tb, n, keys, _ in tiles] == [
        (0, 0, 32, 160), (0, 32, 32, 192), (0, 64, 32, 224), (0, 96, 32, 256),
        (1, 128, 32, 288), (1, 160, 32, 320), (1, 192, 8, 336)]
    assert all(segs == [(tb + n, -tb)] for _, tb, n, _, segs in tiles)


def test_full_prefix_makes_every_tile_long(lib):
    # a 256-key prefix leaves no room for even one own key
    tiles = decode(dopr.attention_plan(256, 32, [10, 40]))
    assert all(k == 1 for k, *_ in tiles)
    assert [(tb, n) for _, tb, n, _, _ in tiles] == [(0, 32), (32, 18)]


def test_short_pairs_share_a_tile_up_to_the_key_budget(lib):
    # m = 0, 64 tokens per tile, pairs of 5 tokens (16 columns each): 13 pairs touch a
    # full 64-token tile, 208 key columns
    tiles = decode(dopr.attention_plan(0, 64, [5] * 20))
    kind, tb, n, keys, segs = tiles[0]
    assert (kind, tb, n, keys) == (0, 0, 64, 208) and len(segs) == 13
    assert segs[-1] == (4, 60)  # the 13th pair: 4 of its 5 tokens fall in the tile
    assert decode(dopr.attention_plan(0, 64, [5] * 20))[1][4][0] == (5, -4)


def test_segment_limit_cuts_a_tile(lib):
    # 20 one-token pairs, 128 tokens per tile: 16 pairs at most
    tiles = decode(dopr.attention_plan(0, 128, [1] * 20))
    assert [(k, n, len(s)) for k, _, n, _, s in tiles] == [(0, 16, 16), (0, 4, 4)]


@pytest.mark.parametrize("seed", range(40))
def test_random_runs_match_the_restated_rule(lib, seed):
    rng = np.random.default_rng(seed)
    m = int(rng.choice([0, 1, 33, 64, 100, 128, 192, 255, 256, 300]))
    tt = int(rng.choice([16, 32, 64, 128]))
    lens = rng.integers(1, 400 if seed % 3 else 40, size=int(rng.integers(1, 13))).astype(np.int32)
    got = decode(dopr.attention_plan(m, tt, lens))
    assert got == reference_plan(m, tt, lens)
    # invariants: token coverage in order, limits, key count from the segments
    tok = 0
    for kind, tb, n, keys, segs in got:
        assert tb == tok and 1 <= n <= tt and 1 <= len(segs) <= MAX_SEGS
        assert keys == c64(m) + sum(c16(v) for v, _ in segs)
        assert kind == 1 or keys <= MAX_KEYS
        if kind == 1:  # its first token alone is over budget: prefix + its pair's keys up to it
            assert c64(m) + c16(1 - segs[0][1]) > MAX_KEYS
        tok += n
    assert tok == int(lens.sum())


def test_bad_arguments_rejected(lib):
    with pytest.raises(dopr.DoprError):
        dopr.attention_plan(-1, 32, [3])
    with pytest.raises(dopr.DoprError):
        dopr.attention_plan(64, 0, [3])
    with pytest.raises(dopr.DoprError):
        dopr.attention_plan(64, 32, [3, 0])
