"""The packed stream format on the CPU: the numpy packer the GPU tests compare
loip_k_pack with (tests/packfmt.py) is checked here against a decoder written
separately from the format's definition (the layout documented with
loip_k_pack), word by word in plain Python, and against superblocks built to
sit exactly at and just past each of the format's limits.  So the packer's
expected bytes are pinned by something other than themselves: a dropped
field, a shifted offset, a wrong rank order or a wrong limit fails here."""
import os
import re

import numpy as np
import pytest

from packfmt import PACKED, SB, awkward_words, pack_ref
from paper_2512_21835_gb300 import inputs

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def decode_superblock(p):
    """One packed superblock (1440 bytes) -> (1024 words, None), or (None,
    largest exponent) if it is flagged as carried raw.  Follows the layout
    field by field; also checks the record's counts and ranks against the
    codes it decodes."""
    rec = [int(x) for x in p[1408:1440].view("<u4")]
    emax, flag = rec[0] & 0xFF, (rec[0] >> 8) & 0xFF
    if flag == 0xFF:
        assert rec[0] >> 16 == 0 and not any(rec[1:]) and not p[:1408].any()
        return None, emax
    assert flag == 0
    rank = [(rec[0] >> 16) & 0xFF, (rec[0] >> 24) & 0xFF] + [(rec[1] >> (8 * i)) & 0xFF for i in range(4)]
    n1, n2, n3 = rec[2] & 0xFFFF, (rec[2] >> 16) & 0xFF, rec[2] >> 24
    assert len(set(rank)) == 6 and max(rank) <= 14 and n3 <= 5
    exc = {rec[3 + m] & 0xFFFF: rec[3 + m] >> 16 for m in range(n3)}
    words, e1, e2, e3 = [], 0, 0, 0
    for i in range(SB):
        c = (int(p[1024 + i // 4]) >> (2 * (i % 4))) & 3
        if c < 3:
            ex = emax - rank[c]
        else:
            d = (int(p[1280 + e1 // 4]) >> (2 * (e1 % 4))) & 3
            e1 += 1
            if d < 3:
                ex = emax - rank[3 + d]
            else:
                v = (int(p[1368 + e2 // 2]) >> (4 * (e2 % 2))) & 15
                e2 += 1
                if v < 15:
                    ex = emax - v
                else:
                    ex = exc[i]
                    e3 += 1
        b = int(p[i])
        words.append(((b & 0x80) << 8) | (ex << 7) | (b & 0x7F))
    assert (e1, e2, e3) == (n1, n2, n3)
    return np.array(words, np.uint16), emax


def check_ranks(words, packed_sb):
    """rank[] must be the six most frequent k in 0..14, most frequent first,
    ties to the smaller k: counted here directly."""
    e = [(int(w) >> 7) & 0xFF for w in words]
    emax = max(e)
    cnt = [0] * 15
    for x in e:
        if emax - x <= 14:
            cnt[emax - x] += 1
    want = sorted(range(15), key=lambda k: (-cnt[k], k))[:6]
    rec = packed_sb[1408:1416].view("<u4")
    got = [(int(rec[0]) >> 16) & 0xFF, (int(rec[0]) >> 24) & 0xFF] + [(int(rec[1]) >> (8 * i)) & 0xFF for i in range(4)]
    assert got == want


def round_trip(words, packer=pack_ref):
    packed, raw = packer(words)
    P = packed.reshape(-1, PACKED)
    W = words.reshape(-1, SB)
    seen_raw = []
    for s in range(P.shape[0]):
        got, emax = decode_superblock(P[s])
        assert emax == max((int(w) >> 7) & 0xFF for w in W[s])
        if got is None:
            seen_raw.append(s)
        else:
            assert np.array_equal(got, W[s]), s
            check_ranks(W[s], P[s])
    assert seen_raw == raw
    return raw


def test_awkward_superblocks_round_trip_through_an_independent_decoder():
    words = awkward_words(23, 16)
    raw = round_trip(words)
    # raw: a run of 300 zeros (300 exceptions), an infinity (largest exponent 255:
    # every other word is more than 14 binades down), random bit patterns, six
    # exceptions; packed: a lone subnormal, five exceptions, gains near 1
    assert raw == [5, 8, 12, 14]


def test_weight_like_words_pack_to_seventy_percent_and_use_every_level():
    words = inputs.bf16_bits(5, (48 * SB,), 0.02).astype(np.uint16)
    assert round_trip(words) == []
    rec = pack_ref(words)[0].reshape(-1, PACKED)[:, 1408:1440].copy().view("<u4")
    n1, n2 = rec[:, 2] & 0xFFFF, (rec[:, 2] >> 16) & 0xFF
    assert n1.min() > 0 and n2.max() > 0  # level-2 and level-3 codes occur
    assert PACKED / (2 * SB) < 0.71


def _from_k(ks, seed):
    """A superblock whose words have the given k (largest exponent 120 at k = 0;
    k >= 120 gives exponent 0, a zero or subnormal), random signs and mantissas."""
    rng = np.random.default_rng(seed)
    ks = np.asarray(ks)
    assert ks.size == SB
    ex = np.maximum(120 - ks, 0).astype(np.uint32)
    w = (rng.integers(0, 2, SB).astype(np.uint32) << 15) | (ex << 7) | rng.integers(0, 128, SB).astype(np.uint32)
    return rng.permutation(w).astype(np.uint16)


def _counts(c):
    return np.repeat(np.arange(len(c)), c)


def level1_case(extra):
    """352 + extra level-1 escapes: top three k hold 300 + 200 + (172 - extra)
    words; the others 120, 110, 100 at k 3..5 and 22 + extra at k 6..8 (within
    the level-2 limit)."""
    rest = np.array_split(np.arange(22 + extra), 3)
    ks = np.concatenate([_counts([300, 200, 172 - extra, 120, 110, 100]),
                         np.concatenate([np.full(len(r), 6 + j) for j, r in enumerate(rest)])])
    return _from_k(ks, 31 + extra)


def level2_case(extra):
    """80 + extra level-2 escapes at k 6..14 (at most 9 each); ranks 0..5 hold
    the other words."""
    tail = np.array_split(np.arange(80 + extra), 9)
    ks = np.concatenate([_counts([400, 250, 120, 90, 60, 24 - extra]),
                         np.concatenate([np.full(len(r), 6 + j) for j, r in enumerate(tail)])])
    return _from_k(ks, 41 + extra)


def exception_case(n_exc):
    """n_exc words more than 14 binades below the largest."""
    ks = np.concatenate([_counts([600, 300, 100]), np.full(24 - n_exc, 4), np.full(n_exc, 30)])
    return _from_k(ks, 51 + n_exc)


def limit_cases():
    """(words, the superblocks expected raw): each limit met exactly, then
    passed by one."""
    return [(level1_case(0), []), (level1_case(1), [0]), (level2_case(0), []), (level2_case(1), [0]),
            (exception_case(5), []), (exception_case(6), [0])]


@pytest.mark.parametrize("i", range(6))
def test_limits_at_and_past_each_bound(i):
    words, want_raw = limit_cases()[i]
    assert round_trip(words) == want_raw


# plausible mistakes in the packer, each of which a test above must catch
MUTANTS = {
    "ties to the larger k": ("(15 - np.arange(15))[None, :]", "np.arange(15)[None, :]"),
    "level-1 limit off by one": ("(n1 > 352)", "(n1 > 353)"),
    "level-2 limit off by one": ("(n2 > 80)", "(n2 > 81)"),
    "exception limit off by one": ("(n3 > 5)", "(n3 > 6)"),
    "level-3 nibbles swapped": ("L3[:, 0::2] | (L3[:, 1::2] << 4)", "(L3[:, 0::2] << 4) | L3[:, 1::2]"),
    "level-2 codes out of order": ("L2[:, 0::4] | (L2[:, 1::4] << 2)", "L2[:, 1::4] | (L2[:, 0::4] << 2)"),
    "sign bit dropped": ("((W >> 8) & 0x80) | (W & 0x7F)", "(W & 0x7F)"),
    "exception count misplaced": ("(n3 << 24)", "(n3 << 20)"),
    "raw record without its exponent": ("(emax[raw].astype(np.uint32) | (0xFF << 8))", "(np.zeros_like(emax[raw], np.uint32) | (0xFF << 8))"),
    "escape positions from 1": ("pos1 = np.cumsum(esc1, 1) - 1", "pos1 = np.cumsum(esc1, 1)"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_a_planted_mistake_in_the_packer_is_caught(name):
    import packfmt
    src = open(packfmt.__file__).read()
    a, b = MUTANTS[name]
    assert src.count(a) == 1
    ns = {}
    exec(compile(src.replace(a, b), "packfmt_mutant", "exec"), ns)
    cases = [(awkward_words(23, 16), [5, 8, 12, 14]), (inputs.bf16_bits(5, (8 * SB,), 0.02).astype(np.uint16), [])]
    caught = 0
    for words, want_raw in cases + limit_cases():
        try:
            caught += round_trip(words, ns["pack_ref"]) != want_raw
        except (AssertionError, KeyError, IndexError):
            caught += 1
    assert caught > 0, name


def test_header_states_the_packed_size():
    with open(os.path.join(ROOT, "include", "loip.h")) as f:
        m = re.search(r"#define LOIP_PACKED_SB (\d+)", f.read())
    assert m and int(m.group(1)) == PACKED
