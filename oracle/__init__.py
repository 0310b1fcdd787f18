"""Oracle for the LOIP decoder hot path -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The product (``paper_2512_21835_gb300``)
never imports it, and it imports nothing from the product.

Contents
  * ``oracle.c`` (compiled to ``liboracle.so``): the fp64 decoder definition and
    the seeded weight generator, wrapped here with numpy.
  * ``planner.py``: the single-device residency planner and its discrete-event
    step model (Eq. 1, Eq. 2, Algorithm 1's memory-first fill, Eq. 6).

Parity status: every function here is pinned by ``tests/test_oracle_*.py``
(closed forms, invariants, brute force, published generator outputs).
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess

import numpy as np

_DIR = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_DIR, "oracle.c")
_LIB_PATH = os.path.join(_DIR, "liboracle.so")

KV_BF16 = 1  # keys and values rounded to bf16 as they enter the cache (the device's cache type)
PREFILL_FLAGS = KV_BF16
DECODE_FLAGS = KV_BF16

# tensor order inside a model (mirrors oracle.c)
T_EMBED, T_LMHEAD, T_GFINAL, T_LAYER0, T_PER_LAYER = 0, 1, 2, 3, 9
(L_GATTN, L_WQ, L_WK, L_WV, L_WO, L_GMLP, L_WG, L_WU, L_WD) = range(9)


def build(force: bool = False) -> str:
    """Compile oracle.c with gcc (OpenMP if available).  Returns the .so path."""
    if not force and os.path.exists(_LIB_PATH) and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC):
        return _LIB_PATH
    base = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off", "-fno-fast-math", _SRC, "-o",
            _LIB_PATH + ".tmp", "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True, capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(_LIB_PATH + ".tmp", _LIB_PATH)
    return _LIB_PATH


class _Tensor(C.Structure):
    _fields_ = [("data", C.c_void_p), ("seed", C.c_uint64), ("tensor_id", C.c_uint32), ("kind", C.c_int32)]


class _Desc(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("hidden", C.c_int32), ("n_heads", C.c_int32),
                ("n_kv_heads", C.c_int32), ("head_dim", C.c_int32), ("ffn", C.c_int32),
                ("vocab", C.c_int32), ("rms_eps", C.c_double), ("rope_theta", C.c_double), ("qk_norm", C.c_int32)]


_lib = None


def _bind(L):
    """Declares the C signatures on a loaded oracle library."""
    L.orc_splitmix64.restype = C.c_uint64
    L.orc_splitmix64.argtypes = [C.c_uint64, C.c_uint64]
    L.orc_gen_elem.restype = C.c_uint16
    L.orc_gen_elem.argtypes = [C.c_uint64, C.c_uint32, C.c_uint64, C.c_int]
    L.orc_gen_tensor.restype = None
    L.orc_gen_tensor.argtypes = [C.c_uint64, C.c_uint32, C.c_uint64, C.c_uint64, C.c_int, C.c_void_p]
    L.orc_f32_to_bf16.restype = C.c_uint16
    L.orc_f32_to_bf16.argtypes = [C.c_float]
    L.orc_bf16_to_f32.restype = C.c_float
    L.orc_bf16_to_f32.argtypes = [C.c_uint16]
    L.orc_round_bf16.restype = C.c_double
    L.orc_round_bf16.argtypes = [C.c_double]
    L.orc_rmsnorm.restype = None
    L.orc_rmsnorm.argtypes = [C.c_void_p, C.POINTER(_Tensor), C.c_int, C.c_double, C.c_void_p]
    L.orc_gemv.restype = None
    L.orc_gemv.argtypes = [C.POINTER(_Tensor), C.c_int64, C.c_void_p, C.c_int64, C.c_void_p, C.c_void_p]
    L.orc_rope.restype = None
    L.orc_rope.argtypes = [C.c_void_p, C.c_int, C.c_int64, C.c_double]
    L.orc_silu.restype = C.c_double
    L.orc_silu.argtypes = [C.c_double]
    L.orc_attention.restype = None
    L.orc_attention.argtypes = [C.c_void_p, C.c_void_p, C.c_void_p, C.c_int64, C.c_int, C.c_int, C.c_int,
                                C.c_void_p, C.c_void_p]
    L.orc_tensor_id.restype = C.c_uint32
    L.orc_tensor_id.argtypes = [C.c_int, C.c_int]
    L.orc_generated_tensors.restype = None
    L.orc_generated_tensors.argtypes = [C.POINTER(_Desc), C.c_uint64, C.POINTER(_Tensor)]
    L.orc_forward.restype = C.c_int
    L.orc_forward.argtypes = [C.POINTER(_Desc), C.POINTER(_Tensor), C.c_void_p, C.c_int64, C.c_int64, C.c_int,
                              C.c_int, C.c_void_p, C.c_void_p, C.c_void_p]
    L.orc_num_threads.restype = C.c_int
    return L


def lib():
    global _lib
    if _lib is None:
        _lib = _bind(C.CDLL(build()))
    return _lib


class use_library:
    """Context manager: route every oracle call through another build of
    oracle.c (the pin tests use it to check that planted mistakes are caught)."""

    def __init__(self, path: str):
        self.path = path

    def __enter__(self):
        global _lib
        self.saved = lib()
        _lib = _bind(C.CDLL(self.path))
        return _lib

    def __exit__(self, *exc):
        global _lib
        _lib = self.saved
        return False


def _ptr(a: np.ndarray) -> int:
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data


def num_threads() -> int:
    return int(lib().orc_num_threads())


# ----------------------------------------------------------------------------
# generator and bf16 helpers
# ----------------------------------------------------------------------------
def splitmix64(seed: int, k: int) -> int:
    return int(lib().orc_splitmix64(seed, k))


def tensor_id(layer: int, which: int) -> int:
    """Generator id of a tensor: layer -1 -> embed (0), lm_head (1), g_final (2)."""
    return int(lib().orc_tensor_id(layer, which))


def gen_tensor(seed: int, tid: int, n: int, kind: int = 0, first: int = 0) -> np.ndarray:
    """Generated bf16 bits (uint16) of elements first..first+n-1 of tensor `tid`."""
    out = np.empty(n, dtype=np.uint16)
    lib().orc_gen_tensor(seed, tid, first, n, kind, _ptr(out))
    return out


def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def round_bf16(x: np.ndarray) -> np.ndarray:
    f = np.vectorize(lambda v: lib().orc_round_bf16(float(v)), otypes=[np.float64])
    return f(np.asarray(x, dtype=np.float64))


# ----------------------------------------------------------------------------
# model description and tensors
# ----------------------------------------------------------------------------
class ModelDesc:
    def __init__(self, n_layers, hidden, n_heads, n_kv_heads, head_dim, ffn, vocab, rms_eps=1e-5,
                 rope_theta=500000.0, qk_norm=0):
        self.n_layers, self.hidden, self.n_heads, self.n_kv_heads = n_layers, hidden, n_heads, n_kv_heads
        self.head_dim, self.ffn, self.vocab, self.rms_eps, self.rope_theta = head_dim, ffn, vocab, rms_eps, rope_theta
        self.qk_norm = int(qk_norm)

    def c(self) -> _Desc:
        return _Desc(self.n_layers, self.hidden, self.n_heads, self.n_kv_heads, self.head_dim, self.ffn, self.vocab,
                     self.rms_eps, self.rope_theta, self.qk_norm)

    def n_tensors(self) -> int:
        return 3 + 9 * self.n_layers + (2 * self.n_layers if self.qk_norm else 0)

    def shapes(self):
        """Per-tensor shapes in oracle order."""
        H, F, V = self.hidden, self.ffn, self.vocab
        qd, kvd = self.n_heads * self.head_dim, self.n_kv_heads * self.head_dim
        s = [(V, H), (V, H), (H,)]
        for _ in range(self.n_layers):
            s += [(H,), (qd, H), (kvd, H), (kvd, H), (H, qd), (H,), (F, H), (F, H), (H, F)]
        if self.qk_norm:  # g_q, g_k per layer, after every layer's main tensors
            s += [(self.head_dim,)] * (2 * self.n_layers)
        return s

    def kinds(self):
        k = [0, 0, 1]
        for _ in range(self.n_layers):
            k += [1, 0, 0, 0, 0, 1, 0, 0, 0]
        if self.qk_norm:
            k += [1] * (2 * self.n_layers)
        return k

    def ids(self):
        ids = [tensor_id(-1, w) for w in range(3)]
        for l in range(self.n_layers):
            ids += [tensor_id(l, w) for w in range(9)]
        if self.qk_norm:
            for l in range(self.n_layers):
                ids += [tensor_id(l, 9), tensor_id(l, 10)]
        return ids


class Weights:
    """A model's tensors for the oracle: each entry is a bf16-bits array or None
    (generated from `seed` on the fly)."""

    def __init__(self, desc: ModelDesc, seed: int, arrays=None):
        self.desc, self.seed = desc, seed
        n = desc.n_tensors()
        self.arrays = list(arrays) if arrays is not None else [None] * n
        assert len(self.arrays) == n

    @staticmethod
    def materialize(desc: ModelDesc, seed: int) -> "Weights":
        arrs = []
        for shp, kind, tid in zip(desc.shapes(), desc.kinds(), desc.ids()):
            arrs.append(gen_tensor(seed, tid, int(np.prod(shp)), kind).reshape(shp))
        return Weights(desc, seed, arrs)

    def c_tensors(self):
        n = len(self.arrays)
        ts = (_Tensor * n)()
        lib().orc_generated_tensors(C.byref(self.desc.c()), self.seed, ts)
        keep = []
        for i, a in enumerate(self.arrays):
            if a is not None:
                a = np.ascontiguousarray(a, dtype=np.uint16)
                keep.append(a)
                ts[i].data = _ptr(a)
        return ts, keep

    def f64(self, i: int) -> np.ndarray:
        """Tensor i widened to fp64 (materialises generated tensors)."""
        a = self.arrays[i]
        shp = self.desc.shapes()[i]
        if a is None:
            a = gen_tensor(self.seed, self.desc.ids()[i], int(np.prod(shp)), self.desc.kinds()[i]).reshape(shp)
        return bf16_bits_to_f64(np.asarray(a))


def tensor_struct(seed: int, tid: int, kind: int, data: np.ndarray | None = None):
    t = _Tensor(0, seed, tid, kind)
    keep = None
    if data is not None:
        keep = np.ascontiguousarray(data, dtype=np.uint16)
        t.data = _ptr(keep)
    return t, keep


# ----------------------------------------------------------------------------
# operations
# ----------------------------------------------------------------------------
def rmsnorm(x: np.ndarray, g_bits: np.ndarray, eps: float) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float64)
    t, keep = tensor_struct(0, 0, 0, g_bits)
    y = np.empty_like(x)
    lib().orc_rmsnorm(_ptr(x), C.byref(t), x.size, eps, _ptr(y))
    return y


def gemv(W: np.ndarray | tuple, ncols: int, x: np.ndarray, rows=None, nrows: int | None = None) -> np.ndarray:
    """y[r] = sum_k W[r,k] x[k].  W is bf16 bits [rows, ncols] or a generated
    tensor given as (seed, tensor_id, kind)."""
    x = np.ascontiguousarray(x, dtype=np.float64)
    assert x.size == ncols
    if isinstance(W, tuple):
        t, keep = tensor_struct(W[0], W[1], W[2])
        assert rows is not None or nrows is not None
    else:
        t, keep = tensor_struct(0, 0, 0, W)
        if nrows is None and rows is None:
            nrows = W.shape[0]
    if rows is not None:
        rows = np.ascontiguousarray(rows, dtype=np.int64)
        y = np.empty(rows.size)
        lib().orc_gemv(C.byref(t), ncols, _ptr(rows), rows.size, _ptr(x), _ptr(y))
    else:
        y = np.empty(nrows)
        lib().orc_gemv(C.byref(t), ncols, None, nrows, _ptr(x), _ptr(y))
    return y


def rope(v: np.ndarray, pos: int, theta: float) -> np.ndarray:
    v = np.array(v, dtype=np.float64)
    lib().orc_rope(_ptr(v), v.size, pos, theta)
    return v


def silu(z: float) -> float:
    return float(lib().orc_silu(z))


def attention(q: np.ndarray, K: np.ndarray, V: np.ndarray, n_kv_heads: int, return_probs: bool = False):
    """q [Hq, d]; K, V [T, Hkv, d] -> o [Hq, d] (and probs [Hq, T])."""
    q = np.ascontiguousarray(q, dtype=np.float64)
    K = np.ascontiguousarray(K, dtype=np.float64)
    V = np.ascontiguousarray(V, dtype=np.float64)
    Hq, d = q.shape
    T = K.shape[0]
    o = np.empty((Hq, d))
    probs = np.empty((Hq, max(T, 1))) if return_probs else None
    lib().orc_attention(_ptr(q), _ptr(K), _ptr(V), T, Hq, n_kv_heads, d, _ptr(o),
                        _ptr(probs) if return_probs else None)
    return (o, probs[:, :T]) if return_probs else o


def forward(desc: ModelDesc, weights: Weights, tokens, n_prefill: int = 0, prefill_flags: int = PREFILL_FLAGS,
            decode_flags: int = DECODE_FLAGS, want_logits: bool = False):
    """Causal forward over `tokens` (one sequence).  Returns dict with
    'hidden' [n, H] (final-norm output), 'argmax' [n] and optionally 'logits'."""
    toks = np.ascontiguousarray(tokens, dtype=np.int32)
    n = toks.size
    hid = np.empty((n, desc.hidden))
    am = np.empty(n, dtype=np.int32)
    lg = np.empty((n, desc.vocab)) if want_logits else None
    ts, keep = weights.c_tensors()
    rc = lib().orc_forward(C.byref(desc.c()), ts, _ptr(toks), n, n_prefill, prefill_flags, decode_flags, _ptr(hid),
                           _ptr(lg) if want_logits else None, _ptr(am))
    if rc != 0:
        raise ValueError("oracle forward rejected its arguments")
    out = {"hidden": hid, "argmax": am}
    if want_logits:
        out["logits"] = lg
    return out
