"""The C ABI library loads, exports every declared symbol, validates arguments,
and its host-only planner matches the planner oracle."""
import re

import numpy as np
import pytest

from oracle import planner as OP
from paper_2512_21835_gb300 import configs, loip

HEADER = __import__("os").path.join(__import__("os").path.dirname(__file__), "..", "include", "loip.h")


@pytest.fixture(scope="module")
def L():
    from paper_2512_21835_gb300 import build
    build.build()
    return loip.lib()


def test_exports_every_declared_symbol(L):
    text = open(HEADER).read()
    declared = set(re.findall(r"^\s*(?:int|int32_t|void|const char\*|uint64_t|void\*)\s+(loip_\w+)\s*\(", text, re.M))
    assert len(declared) >= 30
    for name in declared:
        assert hasattr(L, name), name
    assert declared == set(loip.exported_names())


def test_layer_layout_sizes(L):
    for name in ("tiny", "llama3-8b", "llama3-70b"):
        m = configs.MODELS[name]
        lay = loip.loip_layer_layout(m)
        params = configs.layer_params(m)
        assert params * 2 <= lay["l_size"] <= params * 2 + 8 * 256
        assert lay["mha_bytes"] + lay["mlp_bytes"] == lay["l_size"]
        for k in ("off_wqkv", "off_wo", "off_g_mlp", "off_wg", "off_wu", "off_wd"):
            assert lay[k] % 256 == 0
    lay70 = loip.loip_layer_layout(configs.MODELS["llama3-70b"])
    # p_A of the 70B shape: (10240 + 8192) x 8192 + 8192 of 855,654,400 parameters
    assert abs(lay70["mha_bytes"] / lay70["l_size"] - 0.17647) < 1e-4


def test_invalid_arguments_rejected_without_gpu(L):
    bad = dict(configs.MODELS["tiny"], head_dim=48)
    with pytest.raises(loip.LoipError) as e:
        loip.loip_layer_layout(bad)
    assert e.value.code == loip.ERR_INVALID
    with pytest.raises(loip.LoipError):
        loip.loip_plan_residency(configs.MODELS["tiny"], [100, 100], 1000, 0, 0, 4, 1.0, 1.0)  # 4 slots
    # create rejects a null arena before touching the device
    import ctypes as C
    h = C.c_void_p()
    cfg = loip.config(budget=1 << 20)
    rc = L.loip_create(C.byref(loip.model_desc(configs.MODELS["tiny"])), C.byref(cfg), None, 1 << 20, C.byref(h))
    assert rc == loip.ERR_INVALID and not h.value


@pytest.mark.parametrize("L_layers,budget_layers,K", [(80, 30, 2), (80, 12, 3), (32, 40, 2), (10, 4, 1), (16, 9, 2)])
def test_plan_matches_planner_oracle(L, L_layers, budget_layers, K):
    l_size = 1_711_308_800
    fixed, kv = 4_200_000_000, 360_000_000
    budget = fixed + kv + budget_layers * l_size + l_size // 3
    m = dict(configs.MODELS["llama3-70b"], n_layers=L_layers)
    got = loip.loip_plan_residency(m, [l_size] * L_layers, budget, kv, fixed, K, 6.7e12, 2.1e11)
    want = OP.plan(L_layers, l_size, budget, fixed, kv, K, 6.7e12, 2.1e11)
    assert got["n_resident"] == want["R"]
    assert list(~got["resident"]) == want["offloaded"]
    assert got["pred_step_s"] == pytest.approx(want["pred_step_s"], rel=1e-12)
    comp, load = [l_size / 6.7e12] * L_layers, [l_size / 2.1e11] * L_layers
    assert got["eq1_step_s"] == pytest.approx(OP.eq1_single_device(comp, load, want["offloaded"]), rel=1e-12)
    left = budget - fixed - kv - want["R"] * l_size - (K * l_size if want["R"] < L_layers else 0)
    assert got["left_bytes"] == left
    # tokens beyond the current KV the left-over memory holds (Eq. 6 reading)
    assert loip.loip_kv_threshold(left, 327_680) == OP.kv_threshold_tokens(budget, fixed + kv, l_size, want["R"],
                                                                          K if want["R"] < L_layers else 0, 327_680)


def test_plan_infeasible(L):
    with pytest.raises(loip.LoipError) as e:
        loip.loip_plan_residency(configs.MODELS["tiny"], [100, 100], 349, 50, 100, 2, 1.0, 1.0)
    assert e.value.code == loip.ERR_INFEASIBLE


def test_demotion_rule_oracle_properties():
    # demoting one layer at a time from the even spacing keeps the runs within 1 of each other
    for L_layers in (10, 32, 80):
        mask = [False] * L_layers
        for step in range(L_layers):
            mask, v = OP.demote_one(mask)
            assert v is not None and sum(mask) == step + 1
            idx = [i for i, o in enumerate(mask) if o]
            runs = [((idx[(j + 1) % len(idx)] - idx[j] - 1) % L_layers) for j in range(len(idx))]
            if len(idx) < L_layers:
                assert max(runs) <= 2 * min(runs) + 2
        assert OP.demote_one(mask)[1] is None


def test_fixed_bytes(L):
    m = configs.MODELS["llama3-70b"]
    fb = loip.loip_fixed_bytes(m, loip.config(budget=60 * 10 ** 9, max_batch=1, max_ctx=1088,
                                              max_prefill_tokens=1024))
    # embedding + LM head dominate: 2 x 128256 x 8192 x 2 bytes
    assert 2 * 128256 * 8192 * 2 < fb < 2 * 128256 * 8192 * 2 + 400 * 2 ** 20


@pytest.mark.parametrize("model", ["tiny", "llama3-70b"])
@pytest.mark.parametrize("mp, ring", [(256, 6), (512, 6), (1536, 6), (1792, 7), (2048, 8), (4096, 8)])
def test_fixed_part_embedding_placement_and_staging_ring(L, model, mp, ring):
    """The memory term the plan starts from: keeping the embedding table in host
    memory takes exactly its V x H x 2 bytes out of the device's fixed part; the
    packed stream adds a staging ring of R = max(6, min(8, prefill rows / 256))
    chunks of min(32768, superblocks of the larger block) packed superblocks of
    1440 bytes, plus the raw-superblock list (257 uint32), each part rounded up
    to 256 bytes; with direct access or an SSD tier nothing is packed."""
    m = configs.MODELS[model]
    al = lambda b: (b + 255) // 256 * 256
    base = dict(budget=60 * 10 ** 9, max_batch=1, max_ctx=1088, max_prefill_tokens=mp)
    f0 = loip.loip_fixed_bytes(m, loip.config(**base))
    assert f0 - loip.loip_fixed_bytes(m, loip.config(**base, embed_on_host=1)) == al(m["vocab"] * m["hidden"] * 2)
    lay = loip.loip_layer_layout(m)
    chunk = max(1, min(32768, max(lay["mha_bytes"], lay["mlp_bytes"]) // 2048))
    fp = loip.loip_fixed_bytes(m, loip.config(**base, pack_stream=1))
    assert fp - f0 == al(ring * chunk * 1440) + al(4 * 257)
    assert loip.loip_fixed_bytes(m, loip.config(**base, pack_stream=1, mode=loip.MODE_DIRECT)) == f0
    assert loip.loip_fixed_bytes(m, loip.config(**base, pack_stream=1, host_budget_bytes=10 ** 9)) == f0
    if model == "llama3-70b" and mp == 512:  # the decode benchmark's ring: 6 x 47.2 MB
        assert fp - f0 == 6 * 32768 * 1440 + 1280


@pytest.mark.parametrize("model", ["tiny", "llama3-8b", "llama3-70b"])
def test_block_refinement_and_eq7_match_planner_oracle(L, model):
    """loip_refine_blocks / loip_eq7_choice (C) against the planner oracle, on the
    model's real block sizes."""
    import random
    m = configs.MODELS[model]
    lay = loip.loip_layer_layout(m)
    A, M = lay["mha_bytes"], lay["mlp_bytes"]
    rng = random.Random(7)
    for _ in range(50):
        Lm = m["n_layers"]
        off = [rng.random() < 0.6 for _ in range(Lm)]
        left = rng.randint(0, 3 * M)
        masks, rest = loip.loip_refine_blocks(m, left, off)
        want, want_rest = OP.refine_blocks(left, off, A, M)
        assert list(masks) == want and rest == want_rest
        na, nm = rng.randint(0, Lm), rng.randint(0, Lm)
        need = rng.randint(0, 2 * M)
        assert loip.loip_eq7_choice(m, need, na, nm) == OP.eq7_choice(need, na, nm, A, M)


def test_ssd_tier_roundtrip(L, tmp_path):
    """The SSD tier's O_DIRECT file and raw io_uring reads return what was written
    (96 MB: three 32 MB requests in flight; and a single 4 KB block)."""
    assert loip.loip_ssd_roundtrip(str(tmp_path), 96 << 20)
    assert loip.loip_ssd_roundtrip(str(tmp_path), 4096)
    with pytest.raises(RuntimeError):
        loip.loip_ssd_roundtrip(str(tmp_path), 1000)  # not a multiple of the 4 KB block


def _no_device():
    try:
        import torch
        return not torch.cuda.is_available()
    except ImportError:
        return True


def test_noalloc_attention_refusals_without_gpu(L):
    """The allocation-free attention's argument checks, on a machine without a
    GPU: every call here must be refused before the library touches CUDA (the
    pointers are aligned dummies that nothing may read).  The size limit is
    checked at the boundary for many shapes: refused exactly when the scratch
    the shape needs exceeds the fixed array."""
    if not _no_device():
        pytest.skip("dummy pointers: run only where no CUDA device exists")
    LIM = loip.NOALLOC_SCRATCH_FLOATS
    q, kv, pt, cl, o = 1 << 20, 2 << 20, 3 << 20, 4 << 20, 5 << 20  # 16-byte aligned, never dereferenced

    def call(B, Hq, Hkv, d, max_ctx, q=q, kv=kv, pt=pt, cl=cl, o=o):
        pages = (max_ctx + 63) // 64
        return L.loip_k_attention_noalloc(q, kv, pt, pages, cl, B, Hq, Hkv, d, 64, 0, 2 * Hkv * 64 * d * 2,
                                          max_ctx, o, None)

    n_edge = 0
    for B in (1, 3, 8, 16):
        for Hq, Hkv in ((8, 8), (16, 8), (32, 8), (64, 8), (40, 5)):
            for d in (64, 128):
                need = [loip.loip_k_attention_scratch_floats(B, Hq, d, c, 64) for c in range(64, 16385, 64)]
                assert need == sorted(need)
                # the smallest context that no longer fits, and one page below it
                over = next((c for c, n in zip(range(64, 16385, 64), need) if n > LIM), None)
                if over is None or over - 64 < 1:
                    continue
                assert loip.loip_k_attention_scratch_floats(B, Hq, d, over - 64, 64) <= LIM
                for c in (over - 63, over):  # first position of the page that crosses the limit, and its last
                    assert loip.loip_k_attention_scratch_floats(B, Hq, d, c, 64) > LIM
                    assert call(B, Hq, Hkv, d, c) == loip.ERR_INVALID
                n_edge += 1
    assert n_edge >= 15
    # misaligned pointers and unsupported head ratios, in shapes that fit the array
    ok = dict(B=2, Hq=8, Hkv=2, d=64, max_ctx=100)
    assert loip.loip_k_attention_scratch_floats(2, 8, 64, 100, 64) <= LIM
    for bad in (dict(q=q + 4), dict(q=q + 8), dict(kv=kv + 2), dict(pt=pt + 4), dict(cl=cl + 2), dict(o=o + 1)):
        assert call(**ok, **bad) == loip.ERR_INVALID, bad
    assert call(B=2, Hq=24, Hkv=8, d=64, max_ctx=100) == loip.ERR_INVALID  # 3 query heads per kv head
    assert call(B=2, Hq=48, Hkv=3, d=64, max_ctx=100) == loip.ERR_INVALID  # 16
    assert call(B=2, Hq=8, Hkv=2, d=96, max_ctx=100) == loip.ERR_INVALID   # head size


def test_host_deadline_loop_without_gpu(L):
    """The deadline loop of every host wait, against a fake device: done after
    some polls well inside the limit, or never done and given up once the limit
    has passed (not long after it)."""
    rc, w = loip.loip_poll_deadline_check(5000, 0)
    assert rc == loip.OK and w < 100
    rc, w = loip.loip_poll_deadline_check(5000, 2000)
    assert rc == loip.OK and w < 2000
    rc, w = loip.loip_poll_deadline_check(60, -1)
    assert rc == loip.ERR_TIMEOUT and 60 <= w < 2000
    rc, w = loip.loip_poll_deadline_check(0, -1)
    assert rc == loip.ERR_TIMEOUT and w < 1000
