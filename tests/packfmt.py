"""The packed stream format (loip_k_pack / loip_k_unpack) written out in numpy
from its definition, for the tests: a packer and the awkward inputs that
exercise every branch of the format.  No code of the CUDA path is used."""
import numpy as np

from paper_2512_21835_gb300 import inputs

SB, PACKED = 1024, 1440


def pack_ref(words):
    """The packed format, from its definition.  Per 1024-word superblock, with
    k = (largest exponent) - (exponent of the word): the sign-and-mantissa bytes;
    2-bit codes naming the three most frequent k in 0..14 (ties to the smaller k;
    3 = escape); for the escapes, in word order, 2-bit codes naming the next three
    (3 = escape); for those, in word order, 4-bit k (0..14) or 15 (an exception);
    a 32-byte record (largest exponent, flag, the six ranked k, the three counts,
    up to 5 exceptions as index | exponent << 16).  Over a limit (352, 80, 5):
    flag 0xff and every other byte zero."""
    W = words.reshape(-1, SB).astype(np.uint32)
    n_sb = W.shape[0]
    rows = np.arange(n_sb)[:, None]
    E = ((W >> 7) & 0xFF).astype(np.int64)
    emax = E.max(axis=1)
    K = emax[:, None] - E
    hist = np.zeros((n_sb, 16), np.int64)
    np.add.at(hist, (np.broadcast_to(rows, K.shape), np.minimum(K, 15)), 1)
    key = hist[:, :15] * 16 + (15 - np.arange(15))[None, :]  # most frequent first, then the smaller k
    order = np.argsort(-key, axis=1, kind="stable")[:, :6]
    table = np.full((n_sb, 256), 6, np.int64)
    table[rows, order] = np.arange(6)[None, :]
    R = table[rows, K]
    esc1, esc2 = R >= 3, R >= 6
    exc = esc2 & (K > 14)
    n1, n2, n3 = esc1.sum(1), esc2.sum(1), exc.sum(1)
    raw = (n1 > 352) | (n2 > 80) | (n3 > 5)
    out = np.zeros((n_sb, PACKED), np.uint8)
    out[:, :1024] = ((W >> 8) & 0x80) | (W & 0x7F)
    C = np.minimum(R, 3).astype(np.uint8)
    out[:, 1024:1280] = C[:, 0::4] | (C[:, 1::4] << 2) | (C[:, 2::4] << 4) | (C[:, 3::4] << 6)
    L2 = np.zeros((n_sb, 352 + 1024), np.uint8)  # room for any count; only rows within the limit are kept
    pos1 = np.cumsum(esc1, 1) - 1
    r_, c_ = np.nonzero(esc1)
    L2[r_, pos1[r_, c_]] = np.where(R[r_, c_] < 6, R[r_, c_] - 3, 3)
    L2 = L2[:, :352]
    out[:, 1280:1368] = L2[:, 0::4] | (L2[:, 1::4] << 2) | (L2[:, 2::4] << 4) | (L2[:, 3::4] << 6)
    L3 = np.zeros((n_sb, 80 + 1024), np.uint8)
    pos2 = np.cumsum(esc2, 1) - 1
    r_, c_ = np.nonzero(esc2)
    L3[r_, pos2[r_, c_]] = np.where(K[r_, c_] <= 14, K[r_, c_], 15)
    L3 = L3[:, :80]
    out[:, 1368:1408] = L3[:, 0::2] | (L3[:, 1::2] << 4)
    rec = np.zeros((n_sb, 8), np.uint32)
    o = order.astype(np.uint32)
    rec[:, 0] = emax | (o[:, 0] << 16) | (o[:, 1] << 24)
    rec[:, 1] = o[:, 2] | (o[:, 3] << 8) | (o[:, 4] << 16) | (o[:, 5] << 24)
    rec[:, 2] = n1 | (n2 << 16) | (n3 << 24)
    pos3 = np.cumsum(exc, 1) - 1
    r_, c_ = np.nonzero(exc)
    keep = pos3[r_, c_] < 5
    rec[r_[keep], 3 + pos3[r_[keep], c_[keep]]] = c_[keep].astype(np.uint32) | (E[r_[keep], c_[keep]] << 16).astype(np.uint32)
    out[:, 1408:] = rec.view(np.uint8)
    out[raw] = 0
    out[raw, 1408:1412] = (emax[raw].astype(np.uint32) | (0xFF << 8)).view(np.uint8).reshape(-1, 4)
    return out.reshape(-1), sorted(np.nonzero(raw)[0].tolist())


def awkward_words(seed, n_sb):
    w = inputs.bf16_bits(seed, (n_sb * SB,), 0.02).astype(np.uint16)
    rng = np.random.default_rng(seed)
    w[5 * SB:5 * SB + 300] = 0                                  # a zero run (padding)
    w[7 * SB + 3] = 0x0001                                      # a subnormal
    w[8 * SB + 9] = 0x7F80                                      # +inf
    w[8 * SB + 10] = 0xFFC1                                     # a NaN
    w[9 * SB + rng.integers(0, SB, 5)] = 0x0300                 # 5 tiny values: exceptions
    w[10 * SB:11 * SB] = inputs.bf16_bits(seed + 1, (SB,), 1.0)  # gains-like values near 1
    w[10 * SB:11 * SB] = ((w[10 * SB:11 * SB] & 0x807F) | (127 << 7)).astype(np.uint16)
    w[12 * SB:13 * SB] = rng.integers(0, 1 << 16, SB).astype(np.uint16)  # random patterns: raw
    w[14 * SB:14 * SB + 6] = 0x0200                             # 6 exceptions: one too many, raw
    w[15 * SB:15 * SB + 3] = 0x0200                             # 3 (+ any natural ones): packed
    return w
