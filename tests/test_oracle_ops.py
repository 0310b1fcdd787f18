"""Pins for the oracle's layer operations: closed forms, invariants, library routines."""
import math

import numpy as np

from paper_2512_21835_gb300 import inputs

ONE_BF16 = 0x3F80


def test_rmsnorm_unit_rms_and_scale_invariance(orc):
    x = inputs.normal_f32(1, 4096, 3.0).astype(np.float64)
    g1 = np.full(4096, ONE_BF16, dtype=np.uint16)
    eps = 1e-5
    y = orc.rmsnorm(x, g1, eps)
    ms = np.mean(x * x)
    assert abs(math.sqrt(np.mean(y * y)) - math.sqrt(ms / (ms + eps))) < 1e-12
    y2 = orc.rmsnorm(x * 7.5, g1, 0.0)
    y3 = orc.rmsnorm(x, g1, 0.0)
    assert np.max(np.abs(y2 - y3)) < 1e-12
    # the gain multiplies elementwise
    g = inputs.bf16_bits(2, 4096, 1.0)
    yg = orc.rmsnorm(x, g, eps)
    assert np.max(np.abs(yg - y * orc.bf16_bits_to_f64(g))) < 1e-12


def test_gemv_matches_numpy_and_generated_rows(orc):
    W = inputs.bf16_bits(3, (300, 520))
    x = inputs.normal_f32(4, 520).astype(np.float64)
    y = orc.gemv(W, 520, x)
    ref = orc.bf16_bits_to_f64(W) @ x
    assert np.max(np.abs(y - ref)) < 1e-12
    # generated tensor: sampled rows equal rows of the materialised tensor
    tid = orc.tensor_id(1, 4)
    full = orc.gen_tensor(5, tid, 64 * 520, 0).reshape(64, 520)
    rows = np.array([0, 7, 63, 31])
    ys = orc.gemv((5, tid, 0), 520, x, rows=rows)
    assert np.max(np.abs(ys - orc.bf16_bits_to_f64(full[rows]) @ x)) < 1e-12


def test_rope_invariants(orc):
    d, theta = 128, 500000.0
    q = inputs.normal_f32(5, d).astype(np.float64)
    k = inputs.normal_f32(6, d).astype(np.float64)
    assert np.array_equal(orc.rope(q, 0, theta), q)                       # p = 0: identity
    for p in (1, 17, 1000, 123456):
        assert abs(np.linalg.norm(orc.rope(q, p, theta)) - np.linalg.norm(q)) < 1e-10
    # scores depend only on the relative position
    a = orc.rope(q, 40, theta) @ orc.rope(k, 25, theta)
    b = orc.rope(q, 57, theta) @ orc.rope(k, 42, theta)
    c = orc.rope(q, 41, theta) @ orc.rope(k, 25, theta)
    assert abs(a - b) < 1e-10 and abs(a - c) > 1e-6
    # d = 2: a plain 2-D rotation by p radians (frequency theta^0 = 1), counter-clockwise
    v = orc.rope(np.array([1.0, 0.0]), 3, theta)
    assert np.allclose(v, [math.cos(3), math.sin(3)], atol=1e-15)
    # half-split pairing: component i pairs with i + d/2, pair i rotates at theta^(-2i/d)
    e = np.zeros(8)
    e[1] = 1.0
    r = orc.rope(e, 5, 10000.0)
    ang = 5 * 10000.0 ** (-2 / 8)
    assert np.allclose(r, [0, math.cos(ang), 0, 0, 0, math.sin(ang), 0, 0], atol=1e-15)


def test_silu_identities(orc):
    assert orc.silu(0.0) == 0.0
    for z in (0.3, 1.7, 5.0, 12.0):
        assert abs(orc.silu(z) - orc.silu(-z) - z) < 1e-12                 # z*s(z) + z*s(-z) = z
    assert abs(orc.silu(40.0) - 40.0) < 1e-12 and abs(orc.silu(-40.0)) < 1e-12
    assert abs(orc.silu(1.0) - 1.0 / (1.0 + math.exp(-1.0))) < 1e-15


def test_attention_invariants(orc):
    Hq, Hkv, d, T = 8, 2, 16, 13
    q = inputs.normal_f32(7, (Hq, d)).astype(np.float64)
    K = inputs.normal_f32(8, (T, Hkv, d)).astype(np.float64)
    V = inputs.normal_f32(9, (T, Hkv, d)).astype(np.float64)
    o, p = orc.attention(q, K, V, Hkv, return_probs=True)
    assert np.allclose(p.sum(axis=1), 1.0, atol=1e-14)
    # one cached token: output is that token's value of the group's kv head
    o1 = orc.attention(q, K[:1], V[:1], Hkv)
    for h in range(Hq):
        assert np.allclose(o1[h], V[0, h // (Hq // Hkv)], atol=1e-15)
    # identical keys: output is the mean of the values
    Ke = np.repeat(K[:1], T, axis=0)
    oe = orc.attention(q, Ke, V, Hkv)
    for h in range(Hq):
        assert np.allclose(oe[h], V[:, h // 4].mean(axis=0), atol=1e-13)
    # group mapping: kv head j holds constant value j -> head h sees h // G
    Vc = np.zeros((T, Hkv, d))
    for j in range(Hkv):
        Vc[:, j, :] = j
    og = orc.attention(q, K, Vc, Hkv)
    assert np.allclose(og[:, 0], [h // 4 for h in range(Hq)], atol=1e-13)
    # G = 1 (plain multi-head) equals a per-head softmax computed with numpy
    Km = inputs.normal_f32(10, (T, Hq, d)).astype(np.float64)
    Vm = inputs.normal_f32(11, (T, Hq, d)).astype(np.float64)
    om = orc.attention(q, Km, Vm, Hq)
    for h in range(Hq):
        s = Km[:, h, :] @ q[h] / math.sqrt(d)
        w = np.exp(s - s.max())
        w /= w.sum()
        assert np.allclose(om[h], w @ Vm[:, h, :], atol=1e-13)
