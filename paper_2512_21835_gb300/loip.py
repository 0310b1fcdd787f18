"""Python binding of libloip (include/loip.h): argument marshalling only.

Every step of the decoder runs in the library's CUDA kernels; this module
turns torch tensors / numpy arrays into pointers and status codes into
exceptions.  It refuses to load without the compiled library -- there is no
fallback path.
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libloip.so")

OK, ERR_INVALID, ERR_OOM, ERR_INFEASIBLE, ERR_CUDA, ERR_TIMEOUT, ERR_STATE = range(7)
MODE_OVERLAP, MODE_NAIVE, MODE_DIRECT = 0, 1, 2
FAULT_NONE, FAULT_WAIT, FAULT_COPY, FAULT_HOST_ALLOC, FAULT_BARRIER = range(5)
_NAMES = {1: "INVALID", 2: "OOM", 3: "INFEASIBLE", 4: "CUDA", 5: "TIMEOUT", 6: "STATE"}


class LoipError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"LOIP_ERR_{_NAMES.get(code, code)}: {msg}")
        self.code = code


class ModelDesc(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("hidden", C.c_int32), ("n_heads", C.c_int32), ("n_kv_heads", C.c_int32),
                ("head_dim", C.c_int32), ("ffn", C.c_int32), ("vocab", C.c_int32), ("rms_eps", C.c_float),
                ("rope_theta", C.c_float), ("qk_norm", C.c_int32)]


class Config(C.Structure):
    _fields_ = [("device_budget_bytes", C.c_uint64), ("n_slots", C.c_int32), ("page_tokens", C.c_int32),
                ("max_batch", C.c_int32), ("max_ctx", C.c_int32), ("layer_run_kernel", C.c_int32), ("mode", C.c_int32),
                ("timeout_ms", C.c_uint32), ("hbm_Bps", C.c_double), ("link_Bps", C.c_double),
                ("kv_reserve_bytes", C.c_uint64), ("max_prefill_tokens", C.c_int32), ("whole_layers", C.c_int32),
                ("host_budget_bytes", C.c_uint64), ("ssd_dir", C.c_char_p), ("pack_stream", C.c_int32),
                ("embed_on_host", C.c_int32)]


class LayerLayout(C.Structure):
    _fields_ = [(n, C.c_uint64) for n in ("off_g_attn", "off_wqkv", "off_wo", "off_g_mlp", "off_wg", "off_wu",
                                          "off_wd", "l_size", "mha_bytes", "mlp_bytes", "off_g_q", "off_g_k")]


class Plan(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("n_resident", C.c_int32), ("n_offloaded", C.c_int32),
                ("resident", C.POINTER(C.c_uint8)), ("pred_step_s", C.c_double), ("pred_copy_s", C.c_double),
                ("pred_compute_s", C.c_double), ("eq1_step_s", C.c_double), ("left_bytes", C.c_uint64)]


class Stats(C.Structure):
    _fields_ = [("steps", C.c_uint64), ("tokens", C.c_uint64), ("h2d_weight_bytes", C.c_uint64),
                ("last_step_ms", C.c_double), ("copy_busy_ms", C.c_double), ("compute_ms", C.c_double),
                ("n_resident", C.c_int32), ("n_offloaded", C.c_int32), ("n_replans", C.c_int32),
                ("kv_tokens", C.c_uint64), ("kv_bytes", C.c_uint64), ("arena_used", C.c_uint64),
                ("kernel_ms", C.c_double * 16), ("kernel_launches", C.c_uint64 * 16),
                ("copy_ms_total", C.c_double), ("copies_total", C.c_uint64),
                ("pool_min_GBps", C.c_double), ("pool_median_GBps", C.c_double), ("pool_replaced", C.c_uint64),
                ("n_ssd_layers", C.c_int32), ("ssd_read_bytes", C.c_uint64), ("ssd_wait_ms", C.c_double),
                ("ssd_stage_wait_ms", C.c_double), ("ssd_copy_ms", C.c_double), ("pool_numa_node", C.c_int32),
                ("pool_blobs", C.c_int32), ("pool_blobs_on_node", C.c_int32), ("pool_huge_min", C.c_double),
                ("unpack_launches", C.c_uint64), ("unpack_bytes", C.c_uint64)]


P, U64, I32, U32, F32, F64, VP = C.c_void_p, C.c_uint64, C.c_int32, C.c_uint32, C.c_float, C.c_double, C.c_void_p
_SIGS = {
    "loip_layer_layout": (C.c_int, [C.POINTER(ModelDesc), C.POINTER(LayerLayout)]),
    "loip_plan_residency": (C.c_int, [C.POINTER(ModelDesc), P, U64, U64, U64, I32, F64, F64, C.POINTER(Plan)]),
    "loip_kv_threshold": (C.c_int, [U64, U64, C.POINTER(C.c_uint64)]),
    "loip_refine_blocks": (C.c_int, [C.POINTER(ModelDesc), U64, P, P, C.POINTER(C.c_uint64)]),
    "loip_eq7_choice": (C.c_int, [C.POINTER(ModelDesc), U64, I32, I32, C.POINTER(C.c_int32), C.POINTER(C.c_int32)]),
    "loip_fixed_bytes": (C.c_int, [C.POINTER(ModelDesc), C.POINTER(Config), C.POINTER(C.c_uint64)]),
    "loip_create": (C.c_int, [C.POINTER(ModelDesc), C.POINTER(Config), P, U64, C.POINTER(C.c_void_p)]),
    "loip_destroy": (None, [P]),
    "loip_last_error": (C.c_char_p, [P]),
    "loip_load_weights_generated": (C.c_int, [P, U64]),
    "loip_load_layer": (C.c_int, [P, I32, P, U64]),
    "loip_load_globals": (C.c_int, [P, P, P, P]),
    "loip_get_plan": (C.c_int, [P, C.POINTER(Plan)]),
    "loip_get_block_plan": (C.c_int, [P, P, C.POINTER(C.c_uint64)]),
    "loip_stream_layer": (C.c_int, [P, I32, I32, P]),
    "loip_layer_forward": (C.c_int, [P, I32, I32, P, P, I32, P]),
    "loip_set_batch": (C.c_int, [P, I32, P]),
    "loip_decode_step": (C.c_int, [P, P, I32, P, P]),
    "loip_decode_step_device": (C.c_int, [P, P, I32, P, P]),
    "loip_prefill": (C.c_int, [P, P, P, I32, P, P]),
    "loip_replan": (C.c_int, [P, I32]),
    "loip_inject_fault": (C.c_int, [P, I32, I32]),
    "loip_get_copy_log": (I32, [P, P, P, I32]),
    "loip_get_pool_nodes": (C.c_int, [P, P]),
    "loip_poll_deadline_check": (C.c_int, [C.c_uint32, I32, C.POINTER(C.c_double)]),
    "loip_get_stats": (C.c_int, [P, C.POINTER(Stats)]),
    "loip_synchronize": (C.c_int, [P]),
    "loip_set_kernel_timing": (C.c_int, [P, I32]),
    "loip_measure_h2d": (C.c_int, [U64, I32, C.POINTER(C.c_double)]),
    "loip_measure_direct_read": (C.c_int, [U64, I32, C.POINTER(C.c_double)]),
    "loip_ssd_roundtrip": (C.c_int, [C.c_char_p, U64, C.POINTER(C.c_int32)]),
    "loip_compute_stream": (C.c_void_p, [P]),
    "loip_copy_stream": (C.c_void_p, [P]),
    "loip_k_generate": (C.c_int, [P, U64, U64, U64, U32, I32, P]),
    "loip_k_embed": (C.c_int, [P, P, I32, I32, P, P]),
    "loip_k_qkv_rope": (C.c_int, [P, P, P, I32, I32, I32, I32, I32, F32, F32, P, P, P, P, I32, I32, I32, U64, P]),
    "loip_k_attention": (C.c_int, [P, P, P, I32, P, I32, I32, I32, I32, I32, I32, U64, I32, P, P, P]),
    "loip_k_attention_scratch_floats": (C.c_uint64, [I32, I32, I32, I32, I32]),
    "loip_k_attention_noalloc": (C.c_int, [P, P, P, I32, P, I32, I32, I32, I32, I32, I32, U64, I32, P, P]),
    "loip_k_oproj": (C.c_int, [P, P, I32, I32, I32, P, P]),
    "loip_k_gate_up": (C.c_int, [P, P, P, P, I32, I32, I32, F32, P, P]),
    "loip_k_down": (C.c_int, [P, P, I32, I32, I32, P, P]),
    "loip_k_lm_head": (C.c_int, [P, P, P, I32, I32, I32, F32, P, P, P, P, P]),
    "loip_k_lm_head_scratch_bytes": (C.c_uint64, [I32, I32]),
    "loip_k_gemm_bf16": (C.c_int, [P, P, I32, I32, I32, P, P]),
    "loip_k_gemm_split": (C.c_int, [P, P, I32, I32, I32, P, P]),
    "loip_k_prefill_attention": (C.c_int, [P, P, P, I32, P, P, I32, I32, I32, I32, I32, I32, U64, P, P, P]),
    "loip_k_attention_tc_status": (C.c_int, []),
    "loip_k_pack": (C.c_int, [P, U64, P, P, C.c_uint32, C.c_uint32, P]),
    "loip_k_unpack": (C.c_int, [P, U64, P, P]),
    "loip_k_tc_status": (C.c_int, []),
}

_lib = None


def lib():
    """The loaded library.  Raises if it has not been built: there is no other path."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"{LIB_PATH} is missing: build it with `python -c 'import __graft_entry__ as g; "
                              "g.build()'` (nvcc, sm_103a)")
        L = C.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def exported_names():
    return list(_SIGS)


def _ptr(x):
    """Pointer of a torch tensor, numpy array, int or None."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if isinstance(x, np.ndarray):
        assert x.flags["C_CONTIGUOUS"]
        return x.ctypes.data
    return x.data_ptr()


def _check(rc, ctx=None):
    if rc != OK:
        msg = lib().loip_last_error(ctx)
        raise LoipError(rc, msg.decode() if msg else "")


def model_desc(m: dict) -> ModelDesc:
    return ModelDesc(m["n_layers"], m["hidden"], m["n_heads"], m["n_kv_heads"], m["head_dim"], m["ffn"], m["vocab"],
                     m.get("rms_eps", 1e-5), m.get("rope_theta", 500000.0), int(m.get("qk_norm", 0)))


def config(budget: int, n_slots: int = 2, max_batch: int = 1, max_ctx: int = 2048, mode: int = MODE_OVERLAP,
           timeout_ms: int = 0, hbm_Bps: float = 6.7e12, link_Bps: float = 2.1e11, kv_reserve_bytes: int = 0,
           max_prefill_tokens: int = 512, page_tokens: int = 64, layer_run_kernel: int = 0,
           whole_layers: int = 0, host_budget_bytes: int = 0, ssd_dir: str | None = None,
           embed_on_host: int = 0, pack_stream: int = 0) -> Config:
    return Config(budget, n_slots, page_tokens, max_batch, max_ctx, layer_run_kernel, mode, timeout_ms, hbm_Bps,
                  link_Bps, kv_reserve_bytes, max_prefill_tokens, whole_layers, host_budget_bytes,
                  ssd_dir.encode() if ssd_dir else None, pack_stream, embed_on_host)


# ----------------------------------------------------------------------------
# host-only planning
# ----------------------------------------------------------------------------
def loip_layer_layout(m: dict) -> dict:
    out = LayerLayout()
    _check(lib().loip_layer_layout(C.byref(model_desc(m)), C.byref(out)))
    return {n: getattr(out, n) for n, _ in LayerLayout._fields_}


def loip_plan_residency(m: dict, layer_bytes, budget: int, kv_bytes: int, fixed_bytes: int, n_slots: int,
                        hbm_Bps: float, link_Bps: float) -> dict:
    lb = np.ascontiguousarray(layer_bytes, dtype=np.uint64)
    res = np.zeros(m["n_layers"], dtype=np.uint8)
    plan = Plan()
    plan.resident = res.ctypes.data_as(C.POINTER(C.c_uint8))
    _check(lib().loip_plan_residency(C.byref(model_desc(m)), lb.ctypes.data, budget, kv_bytes, fixed_bytes, n_slots,
                                     hbm_Bps, link_Bps, C.byref(plan)))
    return {"n_resident": plan.n_resident, "n_offloaded": plan.n_offloaded, "resident": res.astype(bool),
            "pred_step_s": plan.pred_step_s, "pred_copy_s": plan.pred_copy_s, "pred_compute_s": plan.pred_compute_s,
            "eq1_step_s": plan.eq1_step_s, "left_bytes": plan.left_bytes}


def loip_refine_blocks(m: dict, left_bytes: int, offloaded) -> tuple:
    """Algorithm 1's block-level refinement: (per-layer resident-block masks, bytes left)."""
    off = np.ascontiguousarray(offloaded, dtype=np.uint8)
    masks = np.zeros(off.size, dtype=np.uint8)
    left = C.c_uint64()
    _check(lib().loip_refine_blocks(C.byref(model_desc(m)), left_bytes, off.ctypes.data, masks.ctypes.data,
                                    C.byref(left)))
    return masks, left.value


def loip_eq7_choice(m: dict, need_bytes: int, n_mha: int, n_mlp: int):
    """Eq. 7: (alpha, beta) resident MHA / MLP blocks to offload, or None."""
    a, b = C.c_int32(), C.c_int32()
    rc = lib().loip_eq7_choice(C.byref(model_desc(m)), need_bytes, n_mha, n_mlp, C.byref(a), C.byref(b))
    if rc == 3:  # LOIP_ERR_INFEASIBLE
        return None
    _check(rc)
    return a.value, b.value


def loip_kv_threshold(left_bytes: int, kv_bytes_per_token: int) -> int:
    out = C.c_uint64()
    _check(lib().loip_kv_threshold(left_bytes, kv_bytes_per_token, C.byref(out)))
    return out.value


def loip_measure_h2d(nbytes: int = 1 << 30, reps: int = 5) -> float:
    """Host-to-device copy throughput (bytes/s) from the pool's kind of pinned memory."""
    out = C.c_double()
    _check(lib().loip_measure_h2d(nbytes, reps, C.byref(out)))
    return out.value


def loip_measure_direct_read(nbytes: int = 1 << 30, reps: int = 5) -> float:
    """Throughput (bytes/s) of a kernel streaming mapped pinned host memory."""
    out = C.c_double()
    _check(lib().loip_measure_direct_read(nbytes, reps, C.byref(out)))
    return out.value


def loip_ssd_roundtrip(directory: str | None = None, nbytes: int = 64 << 20) -> bool:
    """Writes and reads back `nbytes` through the SSD tier's io_uring path; True if they match."""
    ok = C.c_int32()
    _check(lib().loip_ssd_roundtrip(directory.encode() if directory else None, nbytes, C.byref(ok)))
    return bool(ok.value)


def loip_fixed_bytes(m: dict, cfg: Config) -> int:
    out = C.c_uint64()
    _check(lib().loip_fixed_bytes(C.byref(model_desc(m)), C.byref(cfg), C.byref(out)))
    return out.value


# ----------------------------------------------------------------------------
# context
# ----------------------------------------------------------------------------
class Context:
    """A loip_ctx plus the device arena (a torch uint8 tensor) it lives in."""

    def __init__(self, m: dict, cfg: Config, arena=None):
        import torch
        self.model = dict(m)
        self.cfg = cfg
        if arena is None:
            arena = torch.empty(cfg.device_budget_bytes, dtype=torch.uint8, device="cuda")
        self.arena = arena
        h = C.c_void_p()
        rc = lib().loip_create(C.byref(model_desc(m)), C.byref(cfg), _ptr(arena), arena.numel(), C.byref(h))
        _check(rc, None)
        self.h = h

    def close(self):
        if getattr(self, "h", None):
            lib().loip_destroy(self.h)
            self.h = None
        self.arena = None  # the device arena goes back to the allocator now, not at collection

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _c(self, rc):
        _check(rc, self.h)

    def load_weights_generated(self, seed: int):
        self._c(lib().loip_load_weights_generated(self.h, seed))

    def load_layer(self, layer: int, blob: np.ndarray):
        self._c(lib().loip_load_layer(self.h, layer, _ptr(blob), blob.nbytes))

    def load_globals(self, embed: np.ndarray, lm_head: np.ndarray, g_final: np.ndarray):
        self._c(lib().loip_load_globals(self.h, _ptr(embed), _ptr(lm_head), _ptr(g_final)))

    def plan(self) -> dict:
        res = np.zeros(self.model["n_layers"], dtype=np.uint8)
        p = Plan()
        p.resident = res.ctypes.data_as(C.POINTER(C.c_uint8))
        self._c(lib().loip_get_plan(self.h, C.byref(p)))
        return {"n_resident": p.n_resident, "n_offloaded": p.n_offloaded, "resident": res.astype(bool),
                "pred_step_s": p.pred_step_s, "eq1_step_s": p.eq1_step_s, "left_bytes": p.left_bytes}

    def block_plan(self) -> dict:
        """Resident blocks per layer (bit 0 MHA, bit 1 MLP) and bytes streamed per pass."""
        masks = np.zeros(self.model["n_layers"], dtype=np.uint8)
        b = C.c_uint64()
        self._c(lib().loip_get_block_plan(self.h, masks.ctypes.data, C.byref(b)))
        return {"masks": masks, "stream_bytes": b.value}

    def set_batch(self, ctx_lens):
        cl = np.ascontiguousarray(ctx_lens, dtype=np.int32)
        self._c(lib().loip_set_batch(self.h, cl.size, cl.ctypes.data))

    def decode_step(self, tokens, out_hidden=None) -> np.ndarray:
        t = np.ascontiguousarray(tokens, dtype=np.int32)
        out = np.empty_like(t)
        self._c(lib().loip_decode_step(self.h, t.ctypes.data, t.size, out.ctypes.data, _ptr(out_hidden)))
        return out

    def decode_step_device(self, tokens_dev, out_tokens_dev, out_hidden=None):
        self._c(lib().loip_decode_step_device(self.h, _ptr(tokens_dev), tokens_dev.numel(), _ptr(out_tokens_dev),
                                              _ptr(out_hidden)))

    def prefill(self, prompts, out_hidden=None) -> np.ndarray:
        """prompts: list of 1-D int arrays.  Returns the argmax after each prompt."""
        lens = np.array([len(p) for p in prompts], dtype=np.int32)
        toks = np.ascontiguousarray(np.concatenate([np.asarray(p, dtype=np.int32) for p in prompts]))
        out = np.empty(len(prompts), dtype=np.int32)
        self._c(lib().loip_prefill(self.h, toks.ctypes.data, lens.ctypes.data, len(prompts), out.ctypes.data,
                                   _ptr(out_hidden)))
        return out

    def stream_layer(self, layer: int, slot: int, copy_stream=None):
        self._c(lib().loip_stream_layer(self.h, layer, slot, copy_stream))

    def layer_forward(self, layer: int, slot: int, hidden, positions, compute_stream=None):
        self._c(lib().loip_layer_forward(self.h, layer, slot, _ptr(hidden), _ptr(positions), hidden.shape[0],
                                         compute_stream))

    def replan(self, lookahead_tokens: int = 0):
        self._c(lib().loip_replan(self.h, lookahead_tokens))

    def copy_log(self, max_n: int = 8192):
        """(ms, bytes) arrays of the most recent completed layer copies, oldest first."""
        ms, by = np.zeros(max_n, dtype=np.float64), np.zeros(max_n, dtype=np.uint64)
        n = lib().loip_get_copy_log(self.h, _ptr(ms), _ptr(by), max_n)
        if n < 0:
            raise LoipError(ERR_INVALID, "copy log")
        return ms[:n], by[:n]

    def pool_nodes(self):
        nodes = np.zeros(self.model["n_layers"], dtype=np.int32)
        self._c(lib().loip_get_pool_nodes(self.h, _ptr(nodes)))
        return nodes

    def inject_fault(self, kind: int, arg: int = 0):
        """Arms one host-side (or bounded device-wait) fault for a test."""
        self._c(lib().loip_inject_fault(self.h, kind, arg))

    def stats(self) -> dict:
        s = Stats()
        self._c(lib().loip_get_stats(self.h, C.byref(s)))
        out = {n: getattr(s, n) for n, _ in Stats._fields_}
        out["kernel_ms"] = list(s.kernel_ms)
        out["kernel_launches"] = list(s.kernel_launches)
        return out

    def set_kernel_timing(self, on: bool):
        self._c(lib().loip_set_kernel_timing(self.h, 1 if on else 0))

    def synchronize(self):
        self._c(lib().loip_synchronize(self.h))

    def compute_stream(self) -> int:
        return lib().loip_compute_stream(self.h)

    def copy_stream(self) -> int:
        return lib().loip_copy_stream(self.h)


def loip_create(m: dict, cfg: Config, arena=None) -> Context:
    return Context(m, cfg, arena)


# ----------------------------------------------------------------------------
# kernel-level entry points (torch tensors in, async on `stream`)
# ----------------------------------------------------------------------------
def _s(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return stream


def loip_k_generate(out, first: int, seed: int, tensor_id: int, kind: int, stream=None):
    _check(lib().loip_k_generate(_ptr(out), out.numel(), first, seed, tensor_id, kind, _s(stream)))


def loip_k_embed(embed, tokens, x, stream=None):
    _check(lib().loip_k_embed(_ptr(embed), _ptr(tokens), tokens.numel(), embed.shape[1], _ptr(x), _s(stream)))


def loip_k_qkv_rope(x, g, wqkv, Hq, Hkv, d, eps, theta, positions, q_out, kv_base, page_offsets, max_pages,
                    page_tokens, layer, layer_page_bytes, stream=None):
    B, H = x.shape
    _check(lib().loip_k_qkv_rope(_ptr(x), _ptr(g), _ptr(wqkv), B, H, Hq, Hkv, d, eps, theta, _ptr(positions),
                                 _ptr(q_out), _ptr(kv_base), _ptr(page_offsets), max_pages, page_tokens, layer,
                                 layer_page_bytes, _s(stream)))


def loip_poll_deadline_check(timeout_ms: int, pending_polls: int):
    """(status, waited_ms) of the library's host deadline loop against a fake
    device that stays pending for `pending_polls` polls (< 0: forever)."""
    w = C.c_double(0.0)
    rc = lib().loip_poll_deadline_check(timeout_ms, pending_polls, C.byref(w))
    return rc, w.value


def loip_k_attention_scratch_floats(B, Hq, d, max_ctx, page_tokens) -> int:
    return int(lib().loip_k_attention_scratch_floats(B, Hq, d, max_ctx, page_tokens))


def loip_k_attention(q, kv_base, page_offsets, max_pages, ctx_lens, Hq, Hkv, d, page_tokens, layer,
                     layer_page_bytes, max_ctx, scratch, o, stream=None):
    B = q.shape[0]
    _check(lib().loip_k_attention(_ptr(q), _ptr(kv_base), _ptr(page_offsets), max_pages, _ptr(ctx_lens), B, Hq, Hkv, d,
                                  page_tokens, layer, layer_page_bytes, max_ctx, _ptr(scratch), _ptr(o), _s(stream)))


NOALLOC_SCRATCH_FLOATS = 4 << 20


def loip_k_attention_noalloc(q, kv_base, page_offsets, max_pages, ctx_lens, Hq, Hkv, d, page_tokens, layer,
                             layer_page_bytes, max_ctx, o, stream=None):
    """loip_k_attention for callers that cannot allocate device memory: the
    partial-state scratch is the library's own 16 MiB device array per GPU."""
    B = q.shape[0]
    _check(lib().loip_k_attention_noalloc(_ptr(q), _ptr(kv_base), _ptr(page_offsets), max_pages, _ptr(ctx_lens), B, Hq,
                                          Hkv, d, page_tokens, layer, layer_page_bytes, max_ctx, _ptr(o), _s(stream)))


def loip_k_prefill_attention(q, kv_base, page_offsets, max_pages, prompt_lens, first_pos, Hq, Hkv, d, page_tokens,
                             layer, layer_page_bytes, tiles, o2, stream=None):
    """Causal prefill attention on the tensor cores; o2: [2, M, Hq*d] int16 (bf16 hi, lo)."""
    lens = np.ascontiguousarray(prompt_lens, dtype=np.int32)
    fp = None if first_pos is None else np.ascontiguousarray(first_pos, dtype=np.int32)
    _check(lib().loip_k_prefill_attention(_ptr(q), _ptr(kv_base), _ptr(page_offsets), max_pages, _ptr(lens), _ptr(fp),
                                          len(lens), Hq, Hkv, d, page_tokens, layer, layer_page_bytes, _ptr(tiles),
                                          _ptr(o2), _s(stream)))


def loip_k_attention_tc_status() -> int:
    return int(lib().loip_k_attention_tc_status())


def loip_k_oproj(o, wo, x, stream=None):
    B, K = o.shape
    _check(lib().loip_k_oproj(_ptr(o), _ptr(wo), B, x.shape[1], K, _ptr(x), _s(stream)))


def loip_k_gate_up(x, g, wg, wu, eps, a, stream=None):
    B, H = x.shape
    _check(lib().loip_k_gate_up(_ptr(x), _ptr(g), _ptr(wg), _ptr(wu), B, H, wg.shape[0], eps, _ptr(a), _s(stream)))


def loip_k_down(a, wd, x, stream=None):
    B, F = a.shape
    _check(lib().loip_k_down(_ptr(a), _ptr(wd), B, x.shape[1], F, _ptr(x), _s(stream)))


def loip_k_gemm_bf16(A, W, x, stream=None):
    """x += A W^T on the tensor cores (A [M, K], W [N, K] bf16 as int16 tensors)."""
    M, K = A.shape
    _check(lib().loip_k_gemm_bf16(_ptr(A), _ptr(W), M, W.shape[0], K, _ptr(x), _s(stream)))


def loip_k_gemm_split(A2, W, x, stream=None):
    """x += (A2[0] + A2[1]) W^T on the tensor cores (A2 [2, M, K], W [N, K] bf16
    as int16 tensors): the split-pair operand at fp32 activation precision."""
    _, M, K = A2.shape
    _check(lib().loip_k_gemm_split(_ptr(A2), _ptr(W), M, W.shape[0], K, _ptr(x), _s(stream)))


PACKED_SB = 1440


def loip_k_pack(words, packed, raw_list=None, first_sb=0, raw_cap=0, stream=None):
    """Pack words (int16 [n_sb * 1024]) into packed (uint8 [n_sb * 1440])."""
    n_sb = words.numel() // 1024
    _check(lib().loip_k_pack(_ptr(words), n_sb, _ptr(packed), _ptr(raw_list), first_sb, raw_cap, _s(stream)))


def loip_k_unpack(packed, words, stream=None):
    n_sb = packed.numel() // PACKED_SB
    _check(lib().loip_k_unpack(_ptr(packed), n_sb, _ptr(words), _s(stream)))


def loip_k_tc_status() -> int:
    return int(lib().loip_k_tc_status())


def loip_k_lm_head_scratch_bytes(B, V) -> int:
    return int(lib().loip_k_lm_head_scratch_bytes(B, V))


def loip_k_lm_head(x, g_final, lm_head, eps, z, logits, tokens, scratch, stream=None):
    B, H = x.shape
    _check(lib().loip_k_lm_head(_ptr(x), _ptr(g_final), _ptr(lm_head), B, H, lm_head.shape[0], eps, _ptr(z),
                                _ptr(logits), _ptr(tokens), _ptr(scratch), _s(stream)))
