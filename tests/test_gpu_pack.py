"""Lossless packing of the streamed weights (loip_config.pack_stream).

* Kernel level: loip_k_pack against a numpy packer written from the format's
  definition (byte for byte, raw list as a set), and loip_k_unpack restoring
  every packed superblock bit for bit while leaving the unpacked ones alone.
  Inputs: weight-like bf16 words plus the awkward cases -- zeros and zero runs,
  subnormals, infinities and NaNs, values far below their superblock's largest
  (exceptions), norm gains near 1, and superblocks whose exponents are spread
  so widely that they must travel raw.
* Runtime: a context that streams packed layers gives bit-identical results to
  one that streams raw blobs (several slot counts, naive mode, block-level
  residency), moves fewer bytes over the link, and handles a layer with a few
  raw superblocks and a layer that cannot be packed at all (loaded through
  loip_load_layer)."""
import numpy as np
import pytest

from gpu_util import need_gpu
from packfmt import PACKED, SB, awkward_words, pack_ref
from paper_2512_21835_gb300 import configs, inputs

pytestmark = pytest.mark.gpu
TINY6 = dict(configs.MODELS["tiny"], n_layers=6)


@pytest.fixture(scope="module")
def torch():
    return need_gpu()


@pytest.fixture(scope="module")
def L(torch):
    from paper_2512_21835_gb300 import loip
    return loip


@pytest.mark.parametrize("n_sb", [16, 70001])
def test_pack_matches_format_and_round_trips(torch, L, n_sb):
    words = awkward_words(7 + n_sb, n_sb)
    want, want_raw = pack_ref(words)
    dw = torch.from_numpy(words.view(np.int16)).cuda()
    packed = torch.zeros(n_sb * PACKED, dtype=torch.uint8, device="cuda")
    raw_list = torch.zeros(1 + 64, dtype=torch.int32, device="cuda")
    L.loip_k_pack(dw, packed, raw_list, first_sb=1000, raw_cap=64)
    torch.cuda.synchronize()
    got = packed.cpu().numpy()
    assert np.array_equal(got, want)
    rl = raw_list.cpu().numpy().view(np.uint32)
    assert rl[0] == len(want_raw) and sorted((rl[1:1 + rl[0]] - 1000).tolist()) == want_raw
    assert 12 in want_raw and 14 in want_raw
    nexc = (want.reshape(-1, PACKED)[:, 1408 + 11]).astype(int)
    flag = want.reshape(-1, PACKED)[:, 1408 + 1]
    assert np.any((nexc >= 3) & (flag == 0))  # packed superblocks with exceptions are exercised
    assert np.any((want.reshape(-1, PACKED)[:, 1408 + 10] > 0) & (flag == 0))  # level-3 codes too
    out = torch.full((n_sb * SB,), 0x5555, dtype=torch.int16, device="cuda")
    L.loip_k_unpack(packed, out)
    torch.cuda.synchronize()
    back = out.cpu().numpy().view(np.uint16).reshape(-1, SB)
    ref = words.reshape(-1, SB)
    for sb in range(n_sb):
        if sb in want_raw:
            assert np.all(back[sb] == 0x5555)  # left for the raw copy
        else:
            assert np.array_equal(back[sb], ref[sb]), sb
    # weight-like words pack to ~70 % of their bytes
    assert PACKED / (2 * SB) < 0.71


def _budget(L, m, kw, resident):
    lay = L.loip_layer_layout(m)
    fixed = L.loip_fixed_bytes(m, L.config(budget=1 << 40, **kw))
    group = ((2 * m["n_kv_heads"] * 64 * m["head_dim"] * 2 * m["n_layers"]) + 255) // 256 * 256
    blk = (lay["l_size"] + 255) // 256 * 256
    pages = kw["max_batch"] * ((kw["max_ctx"] + 63) // 64)
    slots = 0 if resident >= m["n_layers"] else kw.get("n_slots", 2)
    return fixed + pages * group + 256 + (resident + slots) * blk + blk // 2


PROMPTS = [inputs.token_ids(601, 21, 1024), inputs.token_ids(602, 9, 1024)]
CONT = [[int(a), int(b)] for a, b in zip(inputs.token_ids(603, 5, 1024), inputs.token_ids(604, 5, 1024))]


def _run(L, torch, kw, resident, blobs=None, budget=None):
    m = TINY6
    budget = budget or _budget(L, m, kw, resident)
    ctx = L.Context(m, L.config(budget=budget, **kw))
    ctx.load_weights_generated(configs.WEIGHT_SEED)
    for l, blob in (blobs or {}).items():
        ctx.load_layer(l, blob)
    hid = torch.empty(2, m["hidden"], dtype=torch.float32, device="cuda")
    toks = [ctx.prefill(PROMPTS, out_hidden=hid)]
    hids = [hid.cpu().numpy().copy()]
    ctx.synchronize()
    b0 = ctx.stats()["h2d_weight_bytes"]
    for step in CONT:
        toks.append(ctx.decode_step(step, out_hidden=hid))
        hids.append(hid.cpu().numpy().copy())
    ctx.synchronize()
    st = ctx.stats()
    plan = ctx.plan()
    ctx.close()
    return np.array(toks), np.array(hids), plan, (st["h2d_weight_bytes"] - b0) / len(CONT)


@pytest.mark.parametrize("resident,K,mode", [(2, 2, 0), (0, 1, 0), (2, 3, 0), (2, 1, 1)])
def test_packed_streaming_is_bitwise_lossless(torch, L, resident, K, mode):
    kw = dict(max_batch=2, max_ctx=64, n_slots=K, mode=mode)
    raw = _run(L, torch, kw, resident)
    pk = _run(L, torch, dict(kw, pack_stream=1), resident)  # its budget counts the staging ring
    assert pk[2]["n_resident"] == resident
    assert np.array_equal(raw[0], pk[0])
    assert np.array_equal(raw[1].view(np.uint32), pk[1].view(np.uint32))
    assert 0.65 < pk[3] / raw[3] < 0.75, (pk[3], raw[3])  # bytes over the link per step


def test_packed_streaming_with_block_residency(torch, L):
    """One streamed layer keeps its MLP block resident (Algorithm 1's block step):
    only its MHA unit streams, packed."""
    m = TINY6
    lay = L.loip_layer_layout(m)
    kw = dict(max_batch=2, max_ctx=64, n_slots=2)
    def budget(k):  # no slack beyond the whole blocks but one MLP block
        return _budget(L, m, k, 2) - (lay["l_size"] + 255) // 256 * 256 // 2 + lay["mlp_bytes"] + 256
    kp = dict(kw, pack_stream=1)
    raw = _run(L, torch, kw, 2, budget=budget(kw))
    pk = _run(L, torch, kp, 2, budget=budget(kp))
    assert np.array_equal(raw[0], pk[0])
    assert np.array_equal(raw[1].view(np.uint32), pk[1].view(np.uint32))


def _layer_blob(L, orc, l, seed):
    """Layer l's blob as loip_load_weights_generated fills it (zero padding)."""
    m = TINY6
    lay = L.loip_layer_layout(m)
    H, F = m["hidden"], m["ffn"]
    qd, kvd = m["n_heads"] * m["head_dim"], m["n_kv_heads"] * m["head_dim"]
    blob = np.zeros(lay["l_size"] // 2, dtype=np.uint16)
    parts = [("off_g_attn", H, 0, 1), ("off_wqkv", qd * H, 1, 0), ("off_wqkv", kvd * H, 2, 0),
             ("off_wqkv", kvd * H, 3, 0), ("off_wo", H * qd, 4, 0), ("off_g_mlp", H, 5, 1),
             ("off_wg", F * H, 6, 0), ("off_wu", F * H, 7, 0), ("off_wd", H * F, 8, 0)]
    extra = {2: qd * H, 3: (qd + kvd) * H}
    for key, n, which, kind in parts:
        o = lay[key] // 2 + extra.get(which, 0)
        blob[o:o + n] = orc.gen_tensor(seed, 16 + 16 * l + which, n, kind)
    return blob


def test_packed_streaming_with_raw_superblocks_and_an_unpackable_layer(torch, L, orc):
    """Streamed layer 1 gets three superblocks of random bit patterns in its MLP
    block (carried raw beside the packed stream); streamed layer 2's MLP block is
    random patterns throughout (more raw superblocks than a layer may carry: the
    layer streams as a raw blob).  Both contexts load the same blobs; results are
    bit-identical."""
    rng = np.random.default_rng(11)
    lay = L.loip_layer_layout(TINY6)
    blobs = {}
    for l, n_bad in ((1, 3), (2, None)):  # offloaded at 2 of 6 resident: layers 1, 2, 4, 5
        b = _layer_blob(L, orc, l, configs.WEIGHT_SEED)
        o = lay["off_wd"] // 2
        if n_bad is None:
            span = b[lay["mha_bytes"] // 2:]
        else:
            span = b[o:o + n_bad * SB]
        # random signs and mantissas, exponents spread over [100, 126]: finite, small
        r = rng.integers(0, 1 << 16, span.size).astype(np.uint16)
        span[:] = (r & 0x807F) | (rng.integers(100, 127, span.size).astype(np.uint16) << 7)
        blobs[l] = b
    kw = dict(max_batch=2, max_ctx=64, n_slots=2)
    raw = _run(L, torch, kw, 2, blobs=blobs)
    pk = _run(L, torch, dict(kw, pack_stream=1), 2, blobs=blobs)
    assert np.array_equal(raw[0], pk[0])
    assert np.array_equal(raw[1].view(np.uint32), pk[1].view(np.uint32))


LLAMA8B = configs.MODELS["llama3-8b"]


def _passes(L, torch, m, cfg, prompts_a, conts_a, prompts_b, conts_b):
    """prefill -> decode steps -> prefill of new prompts -> decode steps; tokens
    and final hidden rows of every call."""
    ctx = L.Context(m, cfg)
    ctx.load_weights_generated(configs.WEIGHT_SEED)
    hid = torch.empty(len(prompts_a), m["hidden"], dtype=torch.float32, device="cuda")
    toks, hids = [], []
    for prompts, conts in ((prompts_a, conts_a), (prompts_b, conts_b)):
        toks.append(ctx.prefill(prompts, out_hidden=hid))
        hids.append(hid.cpu().numpy().copy())
        for step in conts:
            toks.append(ctx.decode_step(step, out_hidden=hid))
            hids.append(hid.cpu().numpy().copy())
    plan, st = ctx.plan(), ctx.stats()
    ctx.close()
    torch.cuda.empty_cache()
    return np.array(toks), np.array(hids), plan, st


@pytest.mark.parametrize("max_prefill,batch", [(512, 1), (512, 2), (2048, 1)])
def test_packed_streaming_8b_layers_many_chunks(torch, L, max_prefill, batch):
    """8B-shaped layers (each streamed layer is 8 staging chunks: 2 of its MHA
    block, 6 of its MLP block) with staging rings of 6 and 8 chunks: batch-1
    decode steps unpack on the compute stream, two chunks per launch; batch-2
    decode steps and prefill passes unpack on the unpack stream; and the passes
    alternate (decode -> prefill -> decode hands pending unpacks over).
    Embedding table in mapped host memory, as in the offloaded benchmarks.
    Bit-identical to the same calls with every layer resident."""
    m = LLAMA8B
    V = m["vocab"]
    pa = [inputs.token_ids(701, 70, V), inputs.token_ids(702, 33, V)][:batch]
    pb = [inputs.token_ids(703, 41, V), inputs.token_ids(704, 90, V)][:batch]
    ca = [[int(a), int(b)][:batch] for a, b in zip(inputs.token_ids(705, 3, V), inputs.token_ids(706, 3, V))]
    cb = [[int(a), int(b)][:batch] for a, b in zip(inputs.token_ids(707, 2, V), inputs.token_ids(708, 2, V))]
    kw = dict(max_batch=batch, max_ctx=160, n_slots=2, max_prefill_tokens=max_prefill)
    ref = _passes(L, torch, m, L.config(budget=40_000_000_000, **kw), pa, ca, pb, cb)
    assert ref[2]["n_offloaded"] == 0
    kp = dict(kw, pack_stream=1, embed_on_host=1)
    got = _passes(L, torch, m, L.config(budget=_budget(L, m, kp, 12), **kp), pa, ca, pb, cb)
    assert 16 <= got[2]["n_offloaded"] <= 20, got[2]
    assert got[3]["unpack_launches"] > 0
    assert np.array_equal(ref[0], got[0])
    assert np.array_equal(ref[1].view(np.uint32), got[1].view(np.uint32))
