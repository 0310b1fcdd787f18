"""The oracle's pins catch plausible mistakes.  Each mutant is oracle.c with one
planted error (a dropped term, a wrong sign or index, a transposed operand, ...),
compiled on the CPU into a separate library; running the pin tests against it
must fail at least one of them.  oracle.c itself is not modified."""
import os
import subprocess
import tempfile

import pytest

import oracle
import test_oracle_generator as T_GEN
import test_oracle_model as T_MODEL
import test_oracle_ops as T_OPS

SRC = os.path.join(os.path.dirname(oracle.__file__), "oracle.c")

MUTANTS = {
    "rmsnorm drops eps": ("double inv = 1.0 / sqrt(ss / n + eps);", "double inv = 1.0 / sqrt(ss / n);"),
    "rope rotation sign": ("v[i] = u * c - w * s;", "v[i] = u * c + w * s;"),
    "rope adjacent pairing": ("double u = v[i], w = v[i + half];\n        v[i] = u * c - w * s;\n        v[i + half] = w * c + u * s;",
                              "double u = v[2 * i], w = v[2 * i + 1];\n        v[2 * i] = u * c - w * s;\n        v[2 * i + 1] = w * c + u * s;"),
    "attention drops 1/sqrt(d)": ("double scale = 1.0 / sqrt((double)d);", "double scale = 1.0;"),
    "gqa head mapping": ("int kh = h / G;", "int kh = h % Hkv;"),
    "silu becomes sigmoid": ("double orc_silu(double z) { return z / (1.0 + exp(-z)); }",
                             "double orc_silu(double z) { return 1.0 / (1.0 + exp(-z)); }"),
    "mlp residual dropped": ("orc_gemv(&lt[L_WD], F, NULL, H, a, r);\n            for (int i = 0; i < H; ++i) x[i] += r[i];",
                             "orc_gemv(&lt[L_WD], F, NULL, H, a, r);\n            for (int i = 0; i < H; ++i) x[i] = r[i];"),
    "gemv transposed": ("acc += tensor_at(W, (uint64_t)r * (uint64_t)ncols + (uint64_t)k) * x[k];",
                        "acc += tensor_at(W, (uint64_t)k * (uint64_t)nrows + (uint64_t)r) * x[k];"),
    "attention excludes current token": ("orc_attention(q, Kl, Vl, t + 1, Hq, Hkv, hd, o, NULL);",
                                         "orc_attention(q, Kl, Vl, t > 0 ? t : 1, Hq, Hkv, hd, o, NULL);"),
    "argmax highest index on ties": ("if (fv > bv) { bv = fv; best = i; }", "if (fv >= bv) { bv = fv; best = i; }"),
    "final norm uses the wrong gain": ("orc_rmsnorm(x, &ts[T_GFINAL], H, d->rms_eps, z);",
                                       "orc_rmsnorm(x, &ts[T_LAYER0 + T_PER_LAYER * (L - 1) + L_GMLP], H, d->rms_eps, z);"),
    "generator drops a field": ("+\n                (int32_t)(r >> 48);", "+\n                32767;"),
    "rope frequency exponent": ("double freq = pow(theta, -2.0 * (double)i / (double)d);",
                                "double freq = pow(theta, -1.0 * (double)i / (double)d);"),
    "attention values read from K": ("const double* vt = V + ((size_t)t * Hkv + kh) * d;",
                                     "const double* vt = K + ((size_t)t * Hkv + kh) * d;"),
    "keys not rotated": ("for (int h = 0; h < Hkv; ++h) orc_rope(k + (size_t)h * hd, hd, t, d->rope_theta);",
                         "for (int h = 0; h < Hkv; ++h) (void)0;"),
    "keys and values swapped": ("orc_gemv(&lt[L_WK], H, NULL, kvd, y, k);\n            orc_gemv(&lt[L_WV], H, NULL, kvd, y, v);",
                                "orc_gemv(&lt[L_WK], H, NULL, kvd, y, v);\n            orc_gemv(&lt[L_WV], H, NULL, kvd, y, k);"),
    "softmax not normalised": ("double p = s[t] / l;", "double p = s[t];"),
    "keys and queries rotated before the qk-norm too": ("            if (d->qk_norm) { /* per-head RMSNorm with the layer's g_q / g_k, before the rotation */",
                                   "            for (int h = 0; h < Hq; ++h) orc_rope(q + (size_t)h * hd, hd, t, d->rope_theta);\n            for (int h = 0; h < Hkv; ++h) orc_rope(k + (size_t)h * hd, hd, t, d->rope_theta);\n            if (d->qk_norm) {"),
    "qk-norm uses the query gain for keys": ("orc_rmsnorm(k + (size_t)h * hd, &qk[1], hd,", "orc_rmsnorm(k + (size_t)h * hd, &qk[0], hd,"),
    "kv rounding skipped": ("Kl[(size_t)t * kvd + i] = maybe_bf16(k[i], kvb);", "Kl[(size_t)t * kvd + i] = k[i];"),
    "value rounding skipped": ("Vl[(size_t)t * kvd + i] = maybe_bf16(v[i], kvb);", "Vl[(size_t)t * kvd + i] = v[i];"),
    # the one storage rounding, moved: keys rounded before their rotation instead of after
    "keys rounded before the rotation": (
        "            for (int h = 0; h < Hkv; ++h) orc_rope(k + (size_t)h * hd, hd, t, d->rope_theta);\n"
        "            for (int i = 0; i < kvd; ++i) {\n                Kl[(size_t)t * kvd + i] = maybe_bf16(k[i], kvb);",
        "            for (int i = 0; i < kvd; ++i) k[i] = maybe_bf16(k[i], kvb);\n"
        "            for (int h = 0; h < Hkv; ++h) orc_rope(k + (size_t)h * hd, hd, t, d->rope_theta);\n"
        "            for (int i = 0; i < kvd; ++i) {\n                Kl[(size_t)t * kvd + i] = k[i];"),
    # ... or spread to a value the device keeps in fp32: the rotated queries
    "queries rounded like the cache": (
        "            orc_attention(q, Kl, Vl, t + 1, Hq, Hkv, hd, o, NULL);",
        "            for (int i = 0; i < qd; ++i) q[i] = maybe_bf16(q[i], kvb);\n"
        "            orc_attention(q, Kl, Vl, t + 1, Hq, Hkv, hd, o, NULL);"),
    # ... or to the attention output (the input of the output projection)
    "attention output rounded like the cache": (
        "            orc_gemv(&lt[L_WO], qd, NULL, H, o, r);",
        "            for (int i = 0; i < qd; ++i) o[i] = maybe_bf16(o[i], kvb);\n"
        "            orc_gemv(&lt[L_WO], qd, NULL, H, o, r);"),
}


def _pins():
    """Every pin test function with the fixtures it needs (the oracle module)."""
    fns = []
    for mod in (T_GEN, T_OPS, T_MODEL):
        for name in dir(mod):
            if name.startswith("test_"):
                fns.append((f"{mod.__name__}.{name}", getattr(mod, name)))
    return fns


def _build_mutant(old, new, tmp):
    src = open(SRC).read()
    assert src.count(old) == 1, "mutation site not found once: " + old
    path = os.path.join(tmp, "oracle_mutant.c")
    with open(path, "w") as f:
        f.write(src.replace(old, new))
    so = os.path.join(tmp, "liboracle_mutant.so")
    subprocess.run(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off", "-fno-fast-math", path, "-o",
                    so, "-lm"], check=True, capture_output=True)
    return so


def _fails(fn):
    try:
        fn(oracle)
        return False
    except (AssertionError, ValueError):
        return True


def test_pins_pass_on_the_oracle():
    for name, fn in _pins():
        assert not _fails(fn), name


@pytest.mark.parametrize("mutant", sorted(MUTANTS))
def test_each_planted_mistake_fails_a_pin(mutant):
    old, new = MUTANTS[mutant]
    with tempfile.TemporaryDirectory() as tmp:
        so = _build_mutant(old, new, tmp)
        with oracle.use_library(so):
            caught = [name for name, fn in _pins() if _fails(fn)]
    assert caught, f"no pin catches the mutant '{mutant}'"


PLANNER_MUTANTS = {
    "fill ignores the slots": ("avail = free - n_slots * l_size", "avail = free"),
    "fill ignores the kv cache": ("free = budget - fixed - kv", "free = budget - fixed"),
    "fill rounds up": ("return min(n_layers, avail // l_size), True", "return min(n_layers, -(-avail // l_size)), True"),
    "spacing compares with >=": ("((l + 1) * m) // n_layers > (l * m) // n_layers", "((l + 1) * m) // n_layers >= (l * m) // n_layers"),
    "spacing bunches the offloaded layers": ("return [((l + 1) * m) // n_layers > (l * m) // n_layers for l in range(n_layers)]",
                                             "return [l >= n_layers - m for l in range(n_layers)]"),
    "eq1 idle window counts offloaded compute": ("t_idle = sum(c for c, o in zip(comp, offloaded) if not o)",
                                                 "t_idle = sum(c for c, o in zip(comp, offloaded))"),
    "simulation ignores slot reuse": ("if next_copy - n_slots >= 0:", "if False:"),
    "simulation reuses a slot one copy early": ("ps, pl = order[next_copy - n_slots]",
                                                "ps, pl = order[max(next_copy - n_slots - 1, 0)]"),
    "threshold ignores the slots": ("left = budget - fixed - (R + n_slots_used) * l_size",
                                    "left = budget - fixed - R * l_size"),
    "demotion takes the upper middle": ("victim = (best_start + (best_len - 1) // 2) % L",
                                        "victim = (best_start + best_len // 2) % L"),
    "demotion takes the shortest run": ("if run > best_len:", "if best_len < 0 or run < best_len:"),
    "refinement keeps the MHA block first": ("        if left >= mlp_bytes:\n            masks[l] = 2\n            left -= mlp_bytes\n        elif left >= mha_bytes:\n            masks[l] = 1\n            left -= mha_bytes",
                                             "        if left >= mha_bytes:\n            masks[l] = 1\n            left -= mha_bytes\n        elif left >= mlp_bytes:\n            masks[l] = 2\n            left -= mlp_bytes"),
    "eq7 minimises the block count": ("key = (a * mha_bytes + b * mlp_bytes, a + b)", "key = (a + b, a * mha_bytes + b * mlp_bytes)"),
    "eq7 rounds the MLP count down": ("b = 0 if rest <= 0 else -(-rest // mlp_bytes)", "b = 0 if rest <= 0 else rest // mlp_bytes"),
}


def _planner_pins():
    import test_oracle_planner as T_PLAN
    return T_PLAN, [(n, getattr(T_PLAN, n)) for n in dir(T_PLAN) if n.startswith("test_")]


@pytest.mark.parametrize("mutant", sorted(PLANNER_MUTANTS))
def test_each_planted_planner_mistake_fails_a_pin(mutant):
    import types
    from oracle import planner
    old, new = PLANNER_MUTANTS[mutant]
    src = open(planner.__file__).read()
    assert src.count(old) == 1, "mutation site not found once: " + old
    mod = types.ModuleType("planner_mutant")
    exec(compile(src.replace(old, new), "planner_mutant.py", "exec"), mod.__dict__)
    T_PLAN, pins = _planner_pins()
    saved = T_PLAN.P
    T_PLAN.P = mod
    try:
        caught = []
        for name, fn in pins:
            try:
                fn()
            except Exception:
                caught.append(name)
    finally:
        T_PLAN.P = saved
    assert caught, f"no pin catches the planner mutant '{mutant}'"


def test_planner_pins_pass_on_the_oracle():
    for name, fn in _planner_pins()[1]:
        fn()
