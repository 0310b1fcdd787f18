"""Benchmark: greedy decode of the 70B-shaped bf16 stack with layer offloading.

One step = one decode step of the whole hot path (embedding, 80 decoder layers
of which the ones that do not fit the 60 GB device budget stream from pinned
host memory through the slot ring, final norm, LM head, argmax) for one batch.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--impl ours|reference]
                    [--mode overlap|direct|naive]

Prints one JSON line (rank 0).  `value` is timed on the device with CUDA events
on the compute stream, tokens fed back on the device; `e2e` is the same
metric through loip_decode_step with host token buffers (host<->device copies
inside the timed region).  `--impl reference` times the CPU oracle (the plain
fp64 definition of the decoder) on the host cores on a bounded sample.
`--mode direct` runs the decode steps with the offloaded layers read in place
from the pinned pool (zero-copy) instead of streamed through the slots;
`--mode naive` is the conventional load-then-compute path.
Multi-GPU: independent replicas (the path does not shard), one per rank.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2512_21835_gb300 import configs, inputs  # noqa: E402

METRIC = "decode tokens/s, 70B-shaped bf16 w/ offload; HBM & host-link GB/s vs peak"
KERNEL_NAMES = ["qkv_rope", "attention", "o_proj", "gate_up", "down", "lm_head"]
MODES = {"overlap": 0, "naive": 1, "direct": 2}
RUN_CLASS = 12  # kernel-timing class of the persistent layer-run kernel
UNPACK_CLASS = 13  # kernel-timing class of the unpack of packed streamed chunks

# DRAM bytes (read + write) per launch of the gate/up SwiGLU GEMV at batch 1
# (the persistent kernel, at the 70B and the 8B shape), from an
# ncu capture of the kernel microbenchmark on the model's shape (the
# gate/up traffic summary among the ncu summaries has the commands).  They describe the
# kernel source they were taken on: when the decode kernels' source no longer
# has this hash the figure is reported as null.
GATE_UP_TRAFFIC = {"llama3-70b": 939_745_536, "llama3-8b": 235_113_984}
GATE_UP_TRAFFIC_SRC = "a9c8cc3dcd122fa3d70d3d4bfa641301f6e3cb4caa4123b2fbe05cc51713aadc"


def gate_up_traffic(model, batch):
    src = os.path.join(ROOT, "paper_2512_21835_gb300", "csrc", "decode.cu")
    if batch != 1 or GATE_UP_TRAFFIC.get(model) is None:
        return None
    with open(src, "rb") as f:
        if hashlib.sha256(f.read()).hexdigest() != GATE_UP_TRAFFIC_SRC:
            return None
    return GATE_UP_TRAFFIC[model]


# DRAM bytes (read + write) of the unpack kernel per algorithmic byte (packed
# chunk read + words written), from an ncu capture of the kernel microbenchmark
# (one 70B layer's worth of words); valid while pack.cu has this hash.
UNPACK_TRAFFIC_RATIO = 0.98081  # 2,858,692,352 B over 2,914,572,800 algorithmic (writes still in L2 at exit)
UNPACK_TRAFFIC_SRC = "81016257b8e042a51f9c66df25f58d4d6acaf321fe224edfe44208a78c66e2dd"


def unpack_traffic(bytes_per_launch):
    src = os.path.join(ROOT, "paper_2512_21835_gb300", "csrc", "pack.cu")
    if UNPACK_TRAFFIC_RATIO is None:
        return None
    with open(src, "rb") as f:
        if hashlib.sha256(f.read()).hexdigest() != UNPACK_TRAFFIC_SRC:
            return None
    return int(UNPACK_TRAFFIC_RATIO * bytes_per_launch)


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d.get("hbm_gbs", 6800.0), d.get("bf16_tflops_sustained", 1700.0), "measured"
    return 6800.0, 1700.0, "fallback"


class Clocks:
    """Samples SM clocks and throttle reasons with nvidia-smi during the timed region."""

    def __init__(self):
        self.samples, self._stop, self._t = [], threading.Event(), None

    def _run(self):
        q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
             "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
             "clocks_event_reasons.sw_power_cap")
        while not self._stop.is_set():
            try:
                idx = os.environ.get("LOCAL_RANK", "0")
                out = subprocess.run(["nvidia-smi", "-i", idx, f"--query-gpu={q}", "--format=csv,noheader,nounits"],
                                     capture_output=True, text=True, timeout=5).stdout.strip()
                f = [s.strip() for s in out.split(",")]
                if len(f) >= 7:
                    self.samples.append(f)
            except Exception:
                pass
            self._stop.wait(0.2)

    def __enter__(self):
        self._t = threading.Thread(target=self._run, daemon=True)
        self._t.start()
        return self

    def __exit__(self, *a):
        self._stop.set()
        self._t.join(timeout=10)

    def summary(self):
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        sm = [float(s[0]) for s in self.samples if s[0].replace(".", "").isdigit()]
        mx = [float(s[1]) for s in self.samples if s[1].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for s in self.samples for i in range(4) if s[3 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(self.samples)}


def link_peak_gbs(torch, nbytes=1 << 30, reps=5):
    """Live host->device copy peak: the pool's pinned memory, one cudaMemcpyAsync, best of reps."""
    from paper_2512_21835_gb300 import loip
    return loip.loip_measure_h2d(nbytes, reps) / 1e9


def max_over_ranks(values, device="cpu"):
    """Elementwise max of per-rank timings (replicas are timed between barriers)."""
    import torch
    import torch.distributed as dist
    t = torch.tensor(values, dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(v) for v in t.cpu()]


def workload_setup(name):
    w = dict(configs.WORKLOADS[name])
    m = configs.MODELS[w["model"]]
    return w, m


def kv_group_bytes(m, page=64):
    return (page * 2 * m["n_kv_heads"] * m["head_dim"] * 2 * m["n_layers"] + 255) // 256 * 256


def make_prompts(w, m):
    if "prompt" in w:
        return [np.asarray(p) for p in inputs.prompts(configs.PROMPT_SEED, w["batch"], w["prompt"], m["vocab"])]
    return inputs.batched_prompts(configs.CONTEXT_SEED, configs.PROMPT_SEED, w["batch"], w["ctx_lo"], w["ctx_hi"],
                                  m["vocab"])


def run_ours(args, rank, world):
    import torch
    from paper_2512_21835_gb300 import build as B
    B.build()
    from paper_2512_21835_gb300 import loip

    torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", "0")))
    w, m = workload_setup(args.workload)
    hbm_peak, tc_peak, peak_kind = measured_peaks()
    link_peak = link_peak_gbs(torch)
    mode = MODES[args.mode]
    direct_peak = loip.loip_measure_direct_read(1 << 30, 5) / 1e9 if mode == MODES["direct"] else None
    lay = loip.loip_layer_layout(m)
    prompts = make_prompts(w, m)
    Bsz = len(prompts)
    lens = [len(p) for p in prompts]
    steps, warm = args.steps, args.warmup
    prefill_mode = w.get("decode", 1) == 0
    max_ctx = max(lens) + (0 if prefill_mode else warm + 3 * steps + 16)
    budget = w["budget"] or int(torch.cuda.get_device_properties(0).total_memory * 0.9)
    kv_reserve = 0
    if "ctx_lo" in w:  # KV reserved for the prompts only: decoding grows it (online re-planning)
        kv_reserve = sum((n + 63) // 64 for n in lens) * kv_group_bytes(m)
    # decode workloads prefill their prompts as untimed set-up; at batch 1 in
    # passes of at most 512 rows, so that the prefill workspace (and the staging
    # ring sized by it) leaves the device bytes to weights
    max_prefill = sum(lens) if prefill_mode else min(4096 if Bsz > 1 else 512, sum(lens))
    # a device budget that cannot hold every layer keeps the embedding table in
    # pinned host memory (one 2 x hidden byte row per token crosses the link) and
    # gives its device bytes to resident layers
    embed_host = 0 if args.embed_on_device or not w["budget"] else 1
    # streamed layers cross the link losslessly packed unless asked otherwise
    # (not in the direct-access mode or with the SSD tier, where they stay raw)
    pack = 0 if args.raw_stream or not w["budget"] else 1
    cfg = loip.config(budget=budget, n_slots=w["n_slots"], max_batch=Bsz, max_ctx=max_ctx,
                      max_prefill_tokens=max_prefill, link_Bps=link_peak * 1e9, hbm_Bps=hbm_peak * 1e9,
                      kv_reserve_bytes=kv_reserve, mode=mode, layer_run_kernel=1 if args.layer_run_kernel else 0,
                      host_budget_bytes=w.get("host_budget", 0), ssd_dir=os.environ.get("LOIP_SSD_DIR"),
                      embed_on_host=embed_host, pack_stream=pack)
    t0 = time.time()
    ctx = loip.Context(m, cfg)
    plan = ctx.plan()
    ctx.load_weights_generated(configs.WEIGHT_SEED)
    t_load = time.time() - t0
    t0 = time.time()
    first = ctx.prefill(prompts)
    t_prefill = time.time() - t0
    s = torch.cuda.ExternalStream(ctx.compute_stream())
    n_off0 = plan["n_offloaded"]

    if prefill_mode:
        for _ in range(warm):
            ctx.prefill(prompts)
        ctx.synchronize()
        ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with Clocks() as clk:
            ev0.record(s)
            for _ in range(steps):
                ctx.prefill(prompts)
            ev1.record(s)
            ctx.synchronize()
            torch.cuda.synchronize()
        dev_s = ev0.elapsed_time(ev1) / 1e3
        t0 = time.perf_counter()
        for _ in range(steps):
            ctx.prefill(prompts)
        e2e_s = time.perf_counter() - t0
        ctx.set_kernel_timing(True)
        ctx.prefill(prompts)
        st = ctx.stats()
        ctx.set_kernel_timing(False)
        st_end = ctx.stats()
        plan["stream_bytes"] = ctx.block_plan()["stream_bytes"]
        ctx.close()
        return report_prefill(args, w, m, lay, plan, lens, dev_s, e2e_s, st, st_end, clk, hbm_peak, tc_peak,
                              peak_kind, link_peak, world, budget, t_load, t_prefill)

    # ---- device-timed decode loop: tokens fed back on the device --------------
    tok = torch.from_numpy(first.astype(np.int32)).cuda()
    tok2 = torch.empty_like(tok)
    torch.cuda.synchronize()
    for _ in range(warm):
        ctx.decode_step_device(tok, tok2)
        tok, tok2 = tok2, tok
    ctx.synchronize()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    torch.cuda.synchronize()
    ctx.synchronize()
    st0 = ctx.stats()
    step_ev = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    with Clocks() as clk:
        ev0.record(s)
        for i in range(steps):
            ctx.decode_step_device(tok, tok2)
            tok, tok2 = tok2, tok
            step_ev[i].record(s)
        ev1.record(s)
        ctx.synchronize()
        torch.cuda.synchronize()
    dev_s = ev0.elapsed_time(ev1) / 1e3
    step_ms = [round(ev0.elapsed_time(step_ev[0]), 2)] + [round(step_ev[i - 1].elapsed_time(step_ev[i]), 2)
                                                          for i in range(1, steps)]
    st1 = ctx.stats()
    # per-copy link rates of the timed region (copy-stream events), grouped by step
    n_cp = int(st1["copies_total"] - st0["copies_total"])
    cp_ms, cp_by = ctx.copy_log()
    cp_ms, cp_by = cp_ms[len(cp_ms) - min(n_cp, len(cp_ms)):], cp_by[len(cp_by) - min(n_cp, len(cp_by)):]
    cp_rate = cp_by / np.maximum(cp_ms, 1e-9) / 1e6  # GB/s
    per_step = max(1, len(cp_ms) // steps)
    step_copy_GBps = [round(float(cp_by[i:i + per_step].sum() / max(1e-9, cp_ms[i:i + per_step].sum()) / 1e6), 1)
                      for i in range(0, per_step * (len(cp_ms) // per_step), per_step)]
    pool_nodes = ctx.pool_nodes()
    # ---- per-kernel durations (CUDA events around every launch, separate pass) ----
    st_pre_kt = ctx.stats()
    ctx.set_kernel_timing(True)
    for _ in range(steps):
        ctx.decode_step_device(tok, tok2)
        tok, tok2 = tok2, tok
    ctx.synchronize()
    st = ctx.stats()
    ctx.set_kernel_timing(False)
    # ---- end to end through the public C ABI with host buffers ----------------
    host_tok = tok.cpu().numpy()
    for _ in range(2):
        host_tok = ctx.decode_step(host_tok)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(steps):
        host_tok = ctx.decode_step(host_tok)
    e2e_s = time.perf_counter() - t0
    st_end = ctx.stats()
    plan_end = ctx.plan()
    masks = ctx.block_plan()["masks"]
    ctx.close()
    link_after = link_peak_gbs(torch)  # contention on the shared host link shows here too

    if world > 1:
        dev_s, e2e_s = max_over_ranks([dev_s, e2e_s], device="cuda")

    tokens = steps * Bsz * world
    n_off = st1["n_offloaded"]
    step_s = dev_s / steps
    # bytes the slot ring copied per timed step (blocks, not whole layers, under
    # block-level residency; re-plans during the run included)
    link_bytes = int((st1["h2d_weight_bytes"] - st0["h2d_weight_bytes"]) / steps) or n_off * lay["l_size"]
    mean_ctx = float(np.mean(lens)) + warm + steps / 2
    kv_layer_token = 2 * m["n_kv_heads"] * m["head_dim"] * 2  # K and V bytes per token and layer
    kv_bytes = int(mean_ctx * kv_layer_token * m["n_layers"] * Bsz)
    run_launches = st["kernel_launches"][RUN_CLASS]
    if run_launches:
        # dominant kernel: the persistent layer run (every resident layer's weights + its KV once per step)
        per_launch_layers = st1["n_resident"] * steps / run_launches
        dom_bytes = int(per_launch_layers * (lay["l_size"] + mean_ctx * kv_layer_token * Bsz))
        dom_ms = st["kernel_ms"][RUN_CLASS] / run_launches
        dom_name = f"decode_run (persistent layer run, {per_launch_layers:g} layers per launch)"
        dom_traffic = None
    else:
        # dominant kernel: the gate/up SwiGLU product (55% of a layer's bytes), or
        # the unpack of packed streamed chunks when it takes more of the step
        k = KERNEL_NAMES.index("gate_up")
        dom_bytes = 2 * m["ffn"] * m["hidden"] * 2
        dom_ms = st["kernel_ms"][k] / max(1, st["kernel_launches"][k])
        dom_name = "gate_up (RMSNorm+SwiGLU GEMV)"
        dom_traffic = gate_up_traffic(w["model"], Bsz)
        n_up = st["kernel_launches"][UNPACK_CLASS]
        if n_up and st["kernel_ms"][UNPACK_CLASS] > st["kernel_ms"][k]:
            # algorithmic bytes of one unpack launch: the packed chunk read plus the words written
            dom_bytes = int((st["unpack_bytes"] - st_pre_kt["unpack_bytes"]) / n_up)
            dom_ms = st["kernel_ms"][UNPACK_CLASS] / n_up
            dom_name = "unpack (packed streamed chunk -> slot, lossless)"
            dom_traffic = unpack_traffic(dom_bytes)
    dom_gbs = dom_bytes / (dom_ms / 1e3) / 1e9
    hbm_bytes = m["n_layers"] * lay["l_size"] + m["vocab"] * m["hidden"] * 2 + kv_bytes
    # direct access: the offloaded bytes cross the link as kernel reads, whose
    # ceiling is the measured direct-read rate, not the copy engine's
    link_roof = direct_peak if direct_peak else link_peak
    roof_step = max(hbm_bytes / (hbm_peak * 1e9), link_bytes / (link_roof * 1e9))
    kernel_sum_ms = (sum(st["kernel_ms"][:6]) + st["kernel_ms"][RUN_CLASS]) / steps
    t_copy_only = link_bytes / (link_roof * 1e9)
    exposed = max(0.0, step_s - max(kernel_sum_ms / 1e3, t_copy_only))
    # embed, 5 per per-op layer or 1 per layer run, LM head + argmax, advance
    per_step_launches = (1 + (m["n_layers"] - (st1["n_resident"] if run_launches else 0)) * 5
                         + run_launches // steps + 2 + 1
                         + (st1["unpack_launches"] - st0["unpack_launches"]) // steps)
    line = {
        "metric": METRIC,
        "value": round(tokens / dev_s, 4),
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": steps,
        "warmup": warm,
        "ms_per_step": round(step_s * 1e3, 3),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16 weights, fp32 activations",
        "data": "synthetic: SplitMix64 bf16 weights N(0,0.02^2), uniform token ids",
        "config": {"workload": args.workload, "model": w["model"] + "-shaped", "layers": m["n_layers"],
                   "global_batch": Bsz * world, "context": lens if len(set(lens)) > 1 else lens[0],
                   "budget_bytes": budget, "slots": 1 if args.mode == "naive" else w["n_slots"], "mode": args.mode,
                   "layer_kernels": "persistent runs at batch 1" if args.layer_run_kernel else "per-op",
                   "resident_layers": st1["n_resident"],
                   "embedding": "host (mapped)" if embed_host else "device",
                   "stream": "packed (lossless)" if pack and args.mode != "direct" and not w.get("host_budget")
                   else "raw",
                   "offloaded_layers": n_off, "offloaded_at_start": n_off0,
                   "offloaded_at_end": plan_end["n_offloaded"], "replans": st_end["n_replans"],
                   "blocks_at_end": {"whole_resident": int((masks == 3).sum()), "mha_streamed": int((masks == 2).sum()),
                                     "mlp_streamed": int((masks == 1).sum()), "whole_streamed": int((masks == 0).sum())},
                   "parallelism": f"replicas x{world}",
                   "l2": "inputs larger than L2: every step reads all weights (> 10 GB)"},
        "roofline": {"bound": "hbm", "kernel": dom_name, "achieved": round(dom_gbs, 1),
                     "peak": hbm_peak, "unit": "GB/s", "frac": round(dom_gbs / hbm_peak, 4),
                     "peak_kind": peak_kind, "traffic": dom_traffic, "bytes_per_launch": dom_bytes,
                     "avg_launch_ms": round(dom_ms, 4)},
        "step_roofline": {"bound": ("host-link" if link_bytes / link_roof > hbm_bytes / hbm_peak else "hbm"),
                          "link_bytes_per_step": link_bytes, "link_peak_GBps": round(link_peak, 1),
                          "direct_read_peak_GBps": round(direct_peak, 1) if direct_peak else None,
                          "link_peak_after_GBps": round(link_after, 1),
                          "link_achieved_GBps": round(link_bytes / step_s / 1e9, 1),
                          "hbm_bytes_per_step": hbm_bytes, "roofline_step_ms": round(roof_step * 1e3, 3),
                          "frac": round(roof_step / step_s, 4), "exposed_load_ms": round(exposed * 1e3, 3),
                          "exposed_frac": round(exposed / step_s, 4),
                          "kernel_ms_per_step": dict({n: round(st["kernel_ms"][i] / steps, 4)
                                                      for i, n in enumerate(KERNEL_NAMES)},
                                                     layer_run=round(st["kernel_ms"][RUN_CLASS] / steps, 4)),
                          "copy_GBps_while_copying": round(
                              (st1["copies_total"] - st0["copies_total"]) * lay["l_size"] /
                              max(1e-9, (st1["copy_ms_total"] - st0["copy_ms_total"]) / 1e3) / 1e9, 1),
                          "copy_busy_frac": round((st1["copy_ms_total"] - st0["copy_ms_total"]) / 1e3 / dev_s, 4),
                          "pool_blob_GBps_min_median": [round(st1["pool_min_GBps"], 1),
                                                        round(st1["pool_median_GBps"], 1)],
                          "pool_blobs_moved": st1["pool_replaced"],
                          "pool_huge_page_share_min": round(st1["pool_huge_min"], 4),
                          "pool_numa": {"node": st1["pool_numa_node"], "blobs": st1["pool_blobs"],
                                        "blobs_on_node": st1["pool_blobs_on_node"],
                                        "nodes_seen": sorted({int(v) for v in pool_nodes if v >= 0})},
                          "copy_GBps_min_median_max": ([round(float(np.min(cp_rate)), 1),
                                                        round(float(np.median(cp_rate)), 1),
                                                        round(float(np.max(cp_rate)), 1)] if len(cp_rate) else None),
                          "step_copy_GBps": step_copy_GBps,
                          "ssd_layers": st1["n_ssd_layers"],
                          "ssd_GBps": round((st1["ssd_read_bytes"] - st0["ssd_read_bytes"]) / dev_s / 1e9, 2),
                          "ssd_ms_per_step": {k: round((st_end[k] - st0[k]) / (steps + 4 + steps), 1)
                                              for k in ("ssd_wait_ms", "ssd_stage_wait_ms", "ssd_copy_ms")}},
        # tokens up and down, plus the layer run's 4-byte barrier error word when it ran
        "e2e": {"value": round(tokens / e2e_s, 4), "unit": "tokens/s", "h2d_bytes_per_step": 4 * Bsz,
                "d2h_bytes_per_step": 4 * Bsz + (4 if run_launches else 0)},
        "gpu_launches": per_step_launches * steps,
        "step_ms": step_ms,
        "clocks": clk.summary(),
        "setup_s": {"create_and_weights": round(t_load, 1), "prefill": round(t_prefill, 1)},
    }
    return line


PREFILL_KERNELS = {6: "qkv_gemm", 7: "attention", 8: "o_gemm", 9: "gate_up_gemm", 10: "down_gemm", 11: "rmsnorm"}


def report_prefill(args, w, m, lay, plan, lens, dev_s, e2e_s, st, st_end, clk, hbm_peak, tc_peak, peak_kind,
                   link_peak, world, budget, t_load, t_prefill):
    steps = args.steps
    M = sum(lens)
    H, F, L = m["hidden"], m["ffn"], m["n_layers"]
    qd, kvd = m["n_heads"] * m["head_dim"], m["n_kv_heads"] * m["head_dim"]
    flops_layer = 2 * M * H * (qd + 2 * kvd + qd + 3 * F)
    k = 9
    gu_ms = st["kernel_ms"][k] / max(1, st["kernel_launches"][k])
    gu_tflops = 2 * M * 2 * F * H / (gu_ms / 1e3) / 1e12
    step_s = dev_s / steps
    n_off = plan["n_offloaded"]
    link_bytes = plan["stream_bytes"]  # the streamed blocks of one pass over the layers
    roof = max(flops_layer * L / (tc_peak * 1e12), link_bytes / (link_peak * 1e9))
    return {
        "metric": "prefill tokens/s, 70B-shaped bf16 w/ offload (tensor cores)",
        "value": round(M * steps * world / dev_s, 2), "unit": "tokens/s", "n_gpus": world, "steps": steps,
        "warmup": args.warmup, "ms_per_step": round(step_s * 1e3, 2), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16 GEMM inputs, fp32 accumulation",
        "data": "synthetic: SplitMix64 bf16 weights, uniform token ids",
        "config": {"workload": args.workload, "model": w["model"] + "-shaped", "prompts": len(lens),
                   "tokens_per_step": M, "budget_bytes": budget, "slots": w["n_slots"],
                   "resident_layers": plan["n_resident"], "offloaded_layers": n_off,
                   "l2": "inputs larger than L2 (weights streamed per step)"},
        "roofline": {"bound": "tensor", "kernel": "gate_up GEMM (tcgen05, SwiGLU epilogue)",
                     "achieved": round(gu_tflops, 1), "peak": tc_peak, "unit": "TFLOP/s",
                     "frac": round(gu_tflops / tc_peak, 4), "peak_kind": peak_kind + " sustained bf16",
                     "traffic": None, "avg_launch_ms": round(gu_ms, 4)},
        "step_roofline": {"flops_per_step": flops_layer * L, "link_bytes_per_step": link_bytes,
                          "link_peak_GBps": round(link_peak, 1), "roofline_step_ms": round(roof * 1e3, 2),
                          "frac": round(roof / step_s, 4),
                          "kernel_ms_per_step": {n: round(st["kernel_ms"][i], 3) for i, n in PREFILL_KERNELS.items()},
                          "copy_GBps_while_copying": round(
                              st_end["h2d_weight_bytes"] / max(1e-9, st_end["copy_ms_total"] / 1e3) / 1e9, 1),
                          "pool_blob_GBps_min_median": [round(st_end["pool_min_GBps"], 1),
                                                        round(st_end["pool_median_GBps"], 1)]},
        "e2e": {"value": round(M * steps * world / e2e_s, 2), "unit": "tokens/s", "h2d_bytes_per_step": 4 * M + 4 * len(lens),
                "d2h_bytes_per_step": 4 * len(lens)},
        "clocks": clk.summary(),
        "setup_s": {"create_and_weights": round(t_load, 1), "prefill": round(t_prefill, 1)},
    }


def oracle_sample(m, n_layers_sample, threads=None):
    """Times the oracle on one token through n layers of the model shape plus the
    LM head; returns seconds per full token (layers extrapolated)."""
    import oracle
    oracle.build()
    mh = dict(m, n_layers=0)
    ml = dict(m, n_layers=n_layers_sample, vocab=16)
    tok = np.array([7], dtype=np.int32)
    dl, dh = oracle.ModelDesc(**ml), oracle.ModelDesc(**mh)
    t0 = time.perf_counter()
    oracle.forward(dl, oracle.Weights(dl, configs.WEIGHT_SEED), tok)
    t_layers = time.perf_counter() - t0
    t0 = time.perf_counter()
    oracle.forward(dh, oracle.Weights(dh, configs.WEIGHT_SEED), tok)
    t_head = time.perf_counter() - t0
    per_token = t_layers / n_layers_sample * m["n_layers"] + t_head
    return per_token, t_layers + t_head, oracle.num_threads()


def cpu_baseline(w, m, n_layers_sample=16):
    per_token, spent, cores = oracle_sample(m, n_layers_sample)
    return {"value": round(w["batch"] / per_token, 6), "unit": "tokens/s", "cores": cores, "kind": "oracle",
            "sample": f"1 token through {n_layers_sample} of {m['n_layers']} layers of the {w['model']} shape "
                      f"plus the LM head, fp64, {spent:.1f} s; layer time scaled to {m['n_layers']} layers"}


def run_reference(args, rank, world):
    w, m = workload_setup(args.workload)
    if rank != 0:
        return None
    for _ in range(args.warmup):
        pass  # the oracle has no warm state
    vals = []
    for _ in range(args.steps):
        per_token, spent, cores = oracle_sample(m, 2)
        vals.append(w["batch"] / per_token)
    v = statistics.median(vals)
    return {"metric": METRIC, "value": round(v, 6), "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "higher_is_better": True, "impl": "reference",
            "config": {"workload": args.workload, "model": w["model"] + "-shaped"},
            "cpu_baseline": {"kind": "oracle", "cores": cores, "value": round(v, 6), "unit": "tokens/s",
                             "sample": "per step: 1 token through 2 layers plus the LM head, scaled to "
                                       f"{m['n_layers']} layers"},
            "e2e": {"value": round(v, 6), "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=12)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--workload", default="70b-offload-decode", choices=sorted(configs.WORKLOADS))
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--mode", default="overlap", choices=sorted(MODES))
    ap.add_argument("--raw-stream", action="store_true",
                    help="stream the offloaded layers as raw bf16 blobs instead of losslessly packed")
    ap.add_argument("--embed-on-device", action="store_true",
                    help="keep the embedding table in the device budget even when layers are offloaded")
    ap.add_argument("--layer-run-kernel", action="store_true",
                    help="batch 1: compute runs of resident layers with the persistent layer-run kernel")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if world > 1 and args.impl == "ours":
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", "0")))
        dist.init_process_group("nccl")
    if args.impl == "reference":
        line = run_reference(args, rank, world)
    else:
        line = run_ours(args, rank, world)
        if rank == 0 and not args.no_cpu_baseline:
            w, m = workload_setup(args.workload)
            line["cpu_baseline"] = cpu_baseline(w, m)
    if rank == 0 and line is not None:
        print(json.dumps(line), flush=True)
    if world > 1 and args.impl == "ours":
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
