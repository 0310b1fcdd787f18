"""Kernel microbenchmarks through the kernel-level C ABI.

    python -m paper_2512_21835_gb300.kbench [--only NAME] [--shape 8b|70b|all|none] [--B N] [--iters K]

Prints, per kernel and model shape, the average duration of back-to-back
launches (CUDA events on the current stream, after 3 warm-up launches) and the
resulting bandwidth over the kernel's algorithmic bytes (weights streamed once),
or TFLOP/s for the tensor-core GEMM.  Weight matrices rotate among several
copies so that no launch finds its weights in L2.  Used to produce the ncu
captures in profiles/.
"""
from __future__ import annotations

import argparse

import torch

from . import build, loip as L

SHAPES = {"8b": (4096, 14336, 32, 8), "70b": (8192, 28672, 64, 8)}


def _gen(n, tid):
    t = torch.empty(n, dtype=torch.int16, device="cuda")
    L.loip_k_generate(t, 0, 7, tid, 0)
    return t


def _time(fn, iters):
    for i in range(3):
        fn(i)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for i in range(iters):
        fn(i)
    e1.record()
    e1.synchronize()
    return e0.elapsed_time(e1) / iters / 1e3


def run_shape(name, only, B, iters):
    H, F, Hq, Hkv = SHAPES[name]
    d = 128
    qd, N = Hq * d, (Hq + 2 * Hkv) * d
    ncopy = 2 if name == "70b" else 4
    x = torch.randn(B, max(H, F), device="cuda")
    xh = x[:, :H].contiguous()
    g = _gen(H, 3)
    g.fill_(0x3F80)
    res = {}
    if only in ("", "gate_up"):
        wg = [_gen(F * H, 10 + i).view(F, H) for i in range(ncopy)]
        wu = [_gen(F * H, 20 + i).view(F, H) for i in range(ncopy)]
        out = torch.empty(B, F, device="cuda")
        res["gate_up"] = (2 * F * H * 2, _time(lambda i: L.loip_k_gate_up(xh, g, wg[i % ncopy], wu[i % ncopy], 1e-5,
                                                                         out), iters))
        del wg, wu
    if only in ("", "down"):
        wd = [_gen(H * F, 30 + i).view(H, F) for i in range(ncopy)]
        xx, aa = torch.zeros(B, H, device="cuda"), torch.randn(B, F, device="cuda")
        res["down"] = (H * F * 2, _time(lambda i: L.loip_k_down(aa, wd[i % ncopy], xx), iters))
        del wd
    if only in ("", "oproj"):
        wo = [_gen(H * qd, 40 + i).view(H, qd) for i in range(2 * ncopy)]
        xx, oo = torch.zeros(B, H, device="cuda"), torch.randn(B, qd, device="cuda")
        res["oproj"] = (H * qd * 2, _time(lambda i: L.loip_k_oproj(oo, wo[i % (2 * ncopy)], xx), iters))
        del wo
    if only in ("", "qkv"):
        wq = [_gen(N * H, 50 + i).view(N, H) for i in range(2 * ncopy)]
        P, max_pages = 64, 4
        lpb = 2 * Hkv * P * d * 2
        kv = torch.zeros(B * max_pages * lpb, dtype=torch.uint8, device="cuda")
        pt = (torch.arange(B * max_pages, device="cuda", dtype=torch.int64) * lpb).view(B, max_pages)
        pos = torch.full((B,), 100, dtype=torch.int32, device="cuda")
        q = torch.empty(B, qd, device="cuda")
        res["qkv"] = (N * H * 2, _time(lambda i: L.loip_k_qkv_rope(xh, g, wq[i % (2 * ncopy)], Hq, Hkv, d, 1e-5,
                                                                  500000.0, pos, q, kv, pt, max_pages, P, 0, lpb),
                                       iters))
        del wq
    if only in ("", "attn"):
        P, ctx = 64, 1088
        max_pages = (ctx + P - 1) // P
        lpb = 2 * Hkv * P * d * 2
        kv = (torch.randn(B * max_pages * lpb // 4, device="cuda") * 0.1).view(torch.uint8)
        pt = (torch.arange(B * max_pages, device="cuda", dtype=torch.int64) * lpb).view(B, max_pages)
        cl = torch.full((B,), ctx, dtype=torch.int32, device="cuda")
        qq, oo = torch.randn(B, qd, device="cuda") * 0.01, torch.empty(B, qd, device="cuda")
        sc = torch.empty(L.loip_k_attention_scratch_floats(B, Hq, d, ctx, P), device="cuda")
        res["attn"] = (B * ctx * Hkv * d * 4, _time(lambda i: L.loip_k_attention(qq, kv, pt, max_pages, cl, Hq, Hkv, d,
                                                                                 P, 0, lpb, ctx, sc, oo), iters))
    if only in ("", "lm_head"):
        V = 128256
        wl = [_gen(V * H, 60 + i).view(V, H) for i in range(2)]
        z, lg = torch.empty(B, H, device="cuda"), torch.empty(B, V, device="cuda")
        tk = torch.empty(B, dtype=torch.int32, device="cuda")
        sc = torch.empty(L.loip_k_lm_head_scratch_bytes(B, V), dtype=torch.uint8, device="cuda")
        res["lm_head"] = (V * H * 2, _time(lambda i: L.loip_k_lm_head(xh, g, wl[i % 2], 1e-5, z, lg, tk, sc), iters))
        del wl
    for k, (by, t) in res.items():
        print(f"{name} B={B} {k:8s} {by / 1e6:9.1f} MB  {t * 1e6:9.1f} us  {by / t / 1e9:8.1f} GB/s")
    torch.cuda.empty_cache()


def run_tc(iters):
    """The prefill GEMM shapes (4 x 512 tokens of the 70B layer): one bf16 plane,
    and the split pair (two MMAs per K step).  TFLOP/s counts 2 M N K (the
    product's algorithmic flops) for both."""
    for (M, N, K) in [(2048, 8192, 8192), (2048, 57344, 8192), (2048, 8192, 28672), (2048, 10240, 8192)]:
        A2, W = _gen(2 * M * K, 70).view(2, M, K), _gen(N * K, 71).view(N, K)
        x = torch.zeros(M, N, device="cuda")
        t = _time(lambda i: L.loip_k_gemm_bf16(A2[0], W, x), iters)
        ts = _time(lambda i: L.loip_k_gemm_split(A2, W, x), iters)
        print(f"tc gemm M={M} N={N} K={K}: bf16 {t * 1e6:9.1f} us {2 * M * N * K / t / 1e12:7.1f} TFLOP/s | "
              f"split {ts * 1e6:9.1f} us {2 * M * N * K / ts / 1e12:7.1f} TFLOP/s "
              f"({4 * M * N * K / ts / 1e12:7.1f} issued)  status {L.loip_k_tc_status()}")
        del A2, W, x
        torch.cuda.empty_cache()


def run_pack(iters):
    """Lossless pack / unpack of one 70B layer's worth of weight-like words
    (855.6 M words); GB/s over the bytes each kernel reads plus writes."""
    n_sb = 855654400 // 1024
    w = _gen(n_sb * 1024, 80)
    packed = torch.empty(n_sb * L.PACKED_SB, dtype=torch.uint8, device="cuda")
    out = torch.empty_like(w)
    tp = _time(lambda i: L.loip_k_pack(w, packed), iters)
    tu = _time(lambda i: L.loip_k_unpack(packed, out), iters)
    rw = n_sb * (2048 + L.PACKED_SB)
    print(f"pack   {n_sb} superblocks: {tp * 1e6:9.1f} us  {rw / tp / 1e9:8.1f} GB/s (read + write)")
    print(f"unpack {n_sb} superblocks: {tu * 1e6:9.1f} us  {rw / tu / 1e9:8.1f} GB/s (read + write)")
    del w, packed, out
    torch.cuda.empty_cache()


def run_attn_tc(iters):
    """Tensor-core causal prefill attention, 70B heads (64 query, 8 kv, d 128), 4
    prompts x 512 tokens; TFLOP/s over 4 B_r L_q L_k d / 2 (causal half of QK^T and PV)."""
    Hq, Hkv, d, P, B, n = 64, 8, 128, 64, 4, 512
    pages = n // P
    lpb = 2 * Hkv * P * d * 2
    kv = (torch.randn(B * pages * lpb // 4, device="cuda") * 0.1).view(torch.uint8)
    pt = (torch.arange(B * pages, device="cuda", dtype=torch.int64) * lpb).view(B, pages)
    q = torch.randn(B * n, Hq * d, device="cuda") * 0.3
    tiles = torch.empty((B * n + B) * 4, dtype=torch.int32, device="cuda")
    o2 = torch.empty(2, B * n, Hq * d, dtype=torch.int16, device="cuda")
    t = _time(lambda i: L.loip_k_prefill_attention(q, kv, pt, pages, [n] * B, None, Hq, Hkv, d, P, 0, lpb, tiles,
                                                   o2), iters)
    flops = 2 * 2 * B * Hq * d * (n * (n + 1) / 2)
    print(f"prefill attention 4 x 512, 70B heads: {t * 1e6:9.1f} us  {flops / t / 1e12:7.1f} TFLOP/s "
          f"(x80 layers: {80 * t * 1e3:.1f} ms)  status {L.loip_k_attention_tc_status()}")


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--only", default="")
    ap.add_argument("--iters", type=int, default=20)
    ap.add_argument("--shape", default="all", choices=["all", "8b", "70b", "none"])
    ap.add_argument("--B", type=int, default=1)
    a = ap.parse_args()
    build.build()
    for name in SHAPES:
        if a.shape in ("all", name):
            run_shape(name, a.only, a.B, a.iters)
    if a.only in ("", "tc"):
        run_tc(max(3, min(a.iters, 10)))
    if a.only in ("", "pack"):
        run_pack(max(3, min(a.iters, 10)))
    if a.only in ("", "attn_tc"):
        run_attn_tc(max(3, min(a.iters, 10)))


if __name__ == "__main__":
    main()
