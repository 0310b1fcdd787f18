"""Model shapes and workloads (plain data, no arithmetic of the method).

The shapes are those of the paper's models (Sec. IV-A, "Models": LLaMA3.3-70B;
the 8B shape is the same family at the size that fits one GPU resident), and
of a tiny model for exhaustive parity checks.
"""

MODELS = {
    # 2 layers, hidden 256, 4 query heads x 64, 2 kv heads, SwiGLU 688, vocab 1024
    "tiny": dict(n_layers=2, hidden=256, n_heads=4, n_kv_heads=2, head_dim=64, ffn=688, vocab=1024,
                 rms_eps=1e-5, rope_theta=500000.0),
    # plain multi-head attention (one kv head per query head)
    "tiny-mha": dict(n_layers=3, hidden=256, n_heads=4, n_kv_heads=4, head_dim=64, ffn=688, vocab=1024,
                     rms_eps=1e-5, rope_theta=10000.0),
    # the paper's 13B model shape (LLaMA2-13B: MHA, vocabulary 32000, rotary base 10000)
    "llama2-13b": dict(n_layers=40, hidden=5120, n_heads=40, n_kv_heads=40, head_dim=128, ffn=13824, vocab=32000,
                       rms_eps=1e-5, rope_theta=10000.0),
    "llama3-8b": dict(n_layers=32, hidden=4096, n_heads=32, n_kv_heads=8, head_dim=128, ffn=14336, vocab=128256,
                      rms_eps=1e-5, rope_theta=500000.0),
    "llama3-70b": dict(n_layers=80, hidden=8192, n_heads=64, n_kv_heads=8, head_dim=128, ffn=28672, vocab=128256,
                       rms_eps=1e-5, rope_theta=500000.0),
    # Qwen3-style layers (per-head RMSNorm of queries and keys before the rotation;
    # query width Hq x d larger than the hidden size)
    "tiny-qk": dict(n_layers=2, hidden=256, n_heads=8, n_kv_heads=2, head_dim=64, ffn=688, vocab=1024,
                    rms_eps=1e-6, rope_theta=1000000.0, qk_norm=1),
    # the paper's Qwen3-32B model shape
    "qwen3-32b": dict(n_layers=64, hidden=5120, n_heads=64, n_kv_heads=8, head_dim=128, ffn=25600, vocab=151936,
                      rms_eps=1e-6, rope_theta=1000000.0, qk_norm=1),
}

WEIGHT_SEED = 0x10A1B
PROMPT_SEED = 1
CONTEXT_SEED = 2

# Workloads: decode/prefill runs on synthetic uniform token ids.
WORKLOADS = {
    "tiny-decode": dict(model="tiny", batch=1, prompt=32, decode=16, budget=None, n_slots=2),
    "8b-decode": dict(model="llama3-8b", batch=1, prompt=512, decode=128, budget=None, n_slots=2),
    "13b-decode": dict(model="llama2-13b", batch=1, prompt=512, decode=128, budget=None, n_slots=2),
    "32b-decode": dict(model="qwen3-32b", batch=1, prompt=512, decode=128, budget=None, n_slots=2),
    "70b-offload-decode": dict(model="llama3-70b", batch=1, prompt=1024, decode=64, budget=60_000_000_000,
                               n_slots=2),
    "70b-offload-prefill": dict(model="llama3-70b", batch=4, prompt=512, decode=0, budget=60_000_000_000,
                                n_slots=2),
    # SSD tier: the host pool holds 26 of the 50 streamed layers (+ 4 staging buffers), the rest
    # are read back from a scratch file every step
    "70b-ssd-decode": dict(model="llama3-70b", batch=1, prompt=1024, decode=16, budget=60_000_000_000,
                           n_slots=2, host_budget=30 * 1_711_308_800),
    "70b-offload-batched": dict(model="llama3-70b", batch=8, ctx_lo=128, ctx_hi=4096, decode=256,
                                budget=96_000_000_000, n_slots=2),
}


def layer_params(m: dict) -> int:
    H, F = m["hidden"], m["ffn"]
    qd, kvd = m["n_heads"] * m["head_dim"], m["n_kv_heads"] * m["head_dim"]
    return 2 * H + (qd + 2 * kvd) * H + H * qd + 2 * F * H + H * F + (2 * m["head_dim"] if m.get("qk_norm") else 0)
