"""The layer-level C ABI (loip_stream_layer + loip_layer_forward) and
user-supplied weights (loip_load_layer + loip_load_globals) give the same bits
as loip_decode_step on generated weights."""
import numpy as np
import pytest

from gpu_util import dev_bits, need_gpu
from paper_2512_21835_gb300 import configs, inputs

pytestmark = pytest.mark.gpu
TINY6 = dict(configs.MODELS["tiny"], n_layers=6)


def _cfg(L, m, resident, K=2, max_ctx=64):
    lay = L.loip_layer_layout(m)
    cfg = L.config(budget=1 << 40, n_slots=K, max_batch=1, max_ctx=max_ctx)
    fixed = L.loip_fixed_bytes(m, cfg)
    group = ((2 * m["n_kv_heads"] * 64 * m["head_dim"] * 2 * m["n_layers"]) + 255) // 256 * 256
    blk = (lay["l_size"] + 255) // 256 * 256
    kv_groups = (max_ctx + 63) // 64
    budget = fixed + kv_groups * group + 256 + (resident + K) * blk + blk // 2
    return L.config(budget=budget, n_slots=K, max_batch=1, max_ctx=max_ctx)


def test_layer_level_api_matches_decode_step(orc):
    torch = need_gpu()
    from paper_2512_21835_gb300 import loip as L
    m = TINY6
    prompt = inputs.token_ids(51, 12, m["vocab"])
    nxt = int(inputs.token_ids(52, 1, m["vocab"])[0])
    ctxs = []
    for _ in range(2):
        c = L.Context(m, _cfg(L, m, resident=3))
        c.load_weights_generated(configs.WEIGHT_SEED)
        c.prefill([prompt])
        ctxs.append(c)
    a, b = ctxs
    plan = b.plan()
    assert plan["n_offloaded"] == 3
    hid_a = torch.empty(1, m["hidden"], dtype=torch.float32, device="cuda")
    tok_a = a.decode_step([nxt], out_hidden=hid_a)
    # the same step through the layer-level calls
    cs, ps = b.compute_stream(), b.copy_stream()
    E = orc.gen_tensor(configs.WEIGHT_SEED, 1, m["vocab"] * m["hidden"], 0).reshape(m["vocab"], m["hidden"])
    x = torch.empty(1, m["hidden"], dtype=torch.float32, device="cuda")
    tokd = torch.tensor([nxt], dtype=torch.int32, device="cuda")
    pos = torch.tensor([len(prompt)], dtype=torch.int32, device="cuda")
    Ed = dev_bits(E)
    torch.cuda.synchronize()
    L.loip_k_embed(Ed, tokd, x, stream=cs)
    b.synchronize()  # the ring's prefetches into the slots have landed
    slot = 0
    for layer in range(m["n_layers"]):
        if plan["resident"][layer]:
            b.layer_forward(layer, -1, x, pos, compute_stream=cs)
        else:
            b.stream_layer(layer, slot, copy_stream=ps)
            b.layer_forward(layer, slot, x, pos, compute_stream=cs)
            slot ^= 1
    b.synchronize()
    g = dev_bits(orc.gen_tensor(configs.WEIGHT_SEED, 3, m["hidden"], 1))
    W = dev_bits(orc.gen_tensor(configs.WEIGHT_SEED, 2, m["vocab"] * m["hidden"], 0).reshape(m["vocab"], m["hidden"]))
    z = torch.empty(1, m["hidden"], dtype=torch.float32, device="cuda")
    lg = torch.empty(1, m["vocab"], dtype=torch.float32, device="cuda")
    tk = torch.empty(1, dtype=torch.int32, device="cuda")
    sc = torch.empty(L.loip_k_lm_head_scratch_bytes(1, m["vocab"]), dtype=torch.uint8, device="cuda")
    L.loip_k_lm_head(x, g, W, m["rms_eps"], z, lg, tk, sc, stream=cs)
    b.synchronize()
    assert np.array_equal(z.cpu().numpy().view(np.uint32), hid_a.cpu().numpy().view(np.uint32))
    assert int(tk.cpu()[0]) == int(tok_a[0])
    a.close()
    b.close()


def _blob(orc, m, layer, lay):
    H, F = m["hidden"], m["ffn"]
    qd, kvd = m["n_heads"] * m["head_dim"], m["n_kv_heads"] * m["head_dim"]
    blob = np.zeros(lay["l_size"] // 2, dtype=np.uint16)
    tid = lambda w: 16 + 16 * layer + w
    parts = [("off_g_attn", [(0, H, 1)]), ("off_wqkv", [(1, qd * H, 0), (2, kvd * H, 0), (3, kvd * H, 0)]),
             ("off_wo", [(4, H * qd, 0)]), ("off_g_mlp", [(5, H, 1)]), ("off_wg", [(6, F * H, 0)]),
             ("off_wu", [(7, F * H, 0)]), ("off_wd", [(8, H * F, 0)])]
    for key, tensors in parts:
        off = lay[key] // 2
        for w, n, kind in tensors:
            blob[off:off + n] = orc.gen_tensor(configs.WEIGHT_SEED, tid(w), n, kind)
            off += n
    return blob


def test_user_weights_match_generated(orc):
    torch = need_gpu()
    from paper_2512_21835_gb300 import loip as L
    m = TINY6
    lay = L.loip_layer_layout(m)
    prompt = inputs.token_ids(61, 10, m["vocab"])
    steps = [int(t) for t in inputs.token_ids(62, 4, m["vocab"])]
    outs = []
    for user in (False, True):
        c = L.Context(m, _cfg(L, m, resident=2))
        if user:
            V, H = m["vocab"], m["hidden"]
            c.load_globals(orc.gen_tensor(configs.WEIGHT_SEED, 1, V * H, 0), orc.gen_tensor(configs.WEIGHT_SEED, 2, V * H, 0),
                           orc.gen_tensor(configs.WEIGHT_SEED, 3, H, 1))
            for layer in range(m["n_layers"]):
                c.load_layer(layer, _blob(orc, m, layer, lay))
        else:
            c.load_weights_generated(configs.WEIGHT_SEED)
        hid = torch.empty(1, m["hidden"], dtype=torch.float32, device="cuda")
        toks = [int(c.prefill([prompt], out_hidden=hid)[0])]
        hs = [hid.cpu().numpy().copy()]
        for t in steps:
            toks.append(int(c.decode_step([t], out_hidden=hid)[0]))
            hs.append(hid.cpu().numpy().copy())
        c.close()
        outs.append((toks, np.array(hs)))
    assert outs[0][0] == outs[1][0]
    assert np.array_equal(outs[0][1].view(np.uint32), outs[1][1].view(np.uint32))
