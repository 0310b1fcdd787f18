"""Failure handling on the GPU, in the forms that fault nothing: each fault is
armed through loip_inject_fault and made on the host (a wait whose event
reads as pending, a copy call that reports an error, a pinned allocation that
fails) or as a device wait with a short bound (a layer-run block that misses a
grid barrier, so every barrier wait gives up after 10 ms).  Each test checks
the status the call returns, that a failed context refuses further work, and
that the GPU stays usable: a fresh context afterwards gives the same results as
a context that never saw a fault."""
import numpy as np
import pytest

from gpu_util import need_gpu
from paper_2512_21835_gb300 import configs, inputs

pytestmark = pytest.mark.gpu
M6 = dict(configs.MODELS["tiny"], n_layers=6)


@pytest.fixture(scope="module")
def torch():
    return need_gpu()


@pytest.fixture(scope="module")
def L(torch):
    from paper_2512_21835_gb300 import loip
    return loip


def _budget(L, m, kw, resident):
    lay = L.loip_layer_layout(m)
    fixed = L.loip_fixed_bytes(m, L.config(budget=1 << 40, **kw))
    group = ((2 * m["n_kv_heads"] * 64 * m["head_dim"] * 2 * m["n_layers"]) + 255) // 256 * 256
    blk = (lay["l_size"] + 255) // 256 * 256
    pages = kw["max_batch"] * ((kw["max_ctx"] + 63) // 64)
    slots = 0 if resident >= m["n_layers"] else kw.get("n_slots", 2)
    return fixed + pages * group + 256 + (resident + slots) * blk + blk // 2


def _context(L, kw, resident):
    ctx = L.Context(M6, L.config(budget=_budget(L, M6, kw, resident), **kw))
    return ctx


PROMPT = inputs.token_ids(501, 40, M6["vocab"])
FEED = [int(t) for t in inputs.token_ids(502, 4, M6["vocab"])]


def _clean_run(L, torch, kw, resident):
    """Prefill and four decode steps on a context that sees no fault."""
    ctx = _context(L, kw, resident)
    ctx.load_weights_generated(configs.WEIGHT_SEED)
    hid = torch.empty(1, M6["hidden"], dtype=torch.float32, device="cuda")
    toks = [int(ctx.prefill([PROMPT])[0])]
    for t in FEED:
        toks.append(int(ctx.decode_step([t], out_hidden=hid)[0]))
    out = hid.cpu().numpy().copy()
    ctx.close()
    return toks, out


def _expect(L, code, fn, *a):
    with pytest.raises(L.LoipError) as e:
        fn(*a)
    assert e.value.code == code, e.value
    return e.value


def test_wait_deadline_times_out_and_fails_the_context(torch, L):
    kw = dict(max_batch=1, max_ctx=64, n_slots=2, timeout_ms=300)
    want = _clean_run(L, torch, kw, 3)
    ctx = _context(L, kw, 3)
    ctx.load_weights_generated(configs.WEIGHT_SEED)
    ctx.prefill([PROMPT])
    ctx.inject_fault(L.FAULT_WAIT)
    _expect(L, L.ERR_TIMEOUT, ctx.decode_step, [FEED[0]])
    err = _expect(L, L.ERR_STATE, ctx.decode_step, [FEED[1]])
    assert "timed out" in str(err)
    _expect(L, L.ERR_STATE, ctx.prefill, [PROMPT])
    ctx.close()
    assert _clean_run(L, torch, kw, 3)[0] == want[0]


def test_failed_weight_copy_fails_the_context(torch, L):
    kw = dict(max_batch=1, max_ctx=64, n_slots=2)
    want = _clean_run(L, torch, kw, 2)
    ctx = _context(L, kw, 2)
    assert ctx.plan()["n_offloaded"] == 4
    ctx.load_weights_generated(configs.WEIGHT_SEED)
    ctx.prefill([PROMPT])
    ctx.inject_fault(L.FAULT_COPY)
    _expect(L, L.ERR_CUDA, ctx.decode_step, [FEED[0]])
    _expect(L, L.ERR_STATE, ctx.decode_step, [FEED[1]])
    ctx.close()
    got = _clean_run(L, torch, kw, 2)
    assert got[0] == want[0] and np.array_equal(got[1].view(np.uint32), want[1].view(np.uint32))


def test_failed_host_pool_allocation_is_recoverable(torch, L):
    kw = dict(max_batch=1, max_ctx=64, n_slots=1)
    want = _clean_run(L, torch, kw, 3)
    ctx = _context(L, kw, 3)
    ctx.inject_fault(L.FAULT_HOST_ALLOC)
    _expect(L, L.ERR_OOM, ctx.load_weights_generated, configs.WEIGHT_SEED)
    ctx.load_weights_generated(configs.WEIGHT_SEED)  # the fault fired once; the retry succeeds
    hid = torch.empty(1, M6["hidden"], dtype=torch.float32, device="cuda")
    toks = [int(ctx.prefill([PROMPT])[0])]
    for t in FEED:
        toks.append(int(ctx.decode_step([t], out_hidden=hid)[0]))
    got = hid.cpu().numpy()
    ctx.close()
    assert toks == want[0] and np.array_equal(got.view(np.uint32), want[1].view(np.uint32))


@pytest.mark.parametrize("block", [0, 151])
def test_layer_run_barrier_gives_up_and_reports_timeout(torch, L, block):
    kw = dict(max_batch=1, max_ctx=64, n_slots=2, layer_run_kernel=1)
    want = _clean_run(L, torch, kw, 6)
    ctx = _context(L, kw, 6)
    ctx.load_weights_generated(configs.WEIGHT_SEED)
    ctx.prefill([PROMPT])
    ctx.decode_step([FEED[0]])  # the layer-run kernel works before the fault
    ctx.inject_fault(L.FAULT_BARRIER, block)
    err = _expect(L, L.ERR_TIMEOUT, ctx.decode_step, [FEED[1]])
    assert "grid barrier" in str(err)
    _expect(L, L.ERR_STATE, ctx.decode_step, [FEED[2]])
    ctx.close()
    torch.cuda.synchronize()
    # the GPU is fine: a new context (fresh barrier words) runs the same kernel
    assert _clean_run(L, torch, kw, 6)[0] == want[0]
