/*
 * oracle.c -- plain, slow, fp64 CPU reference for the LOIP decoder hot path.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product (the CUDA library and its
 * Python binding) may call, link or include this file.  Only tests/, the
 * smoke check in __graft_entry__.py and the CPU-baseline leg of bench.py use it.
 * It shares no code, header, table or constant generator with the CUDA path.
 *
 * What it computes.  LOIP (arXiv 2512.21835) is lossless: the offloaded run
 * must give exactly what the unmodified model gives (Sec. IV-A, "Evaluation
 * Metrics": accuracy identical to the original model).  The paper never writes
 * the decoder maths; it runs LLaMA-family checkpoints (Sec. IV-A, "Models").
 * So this oracle is the plain definition of a LLaMA-3 style decoder forward:
 * pre-norm RMSNorm, rotary position embedding (half-split pairing, no frequency
 * scaling), grouped-query attention with a softmax over all cached positions,
 * SwiGLU MLP, untied LM head, greedy argmax (lowest index on ties).
 * Arithmetic is fp64, sequential sums, no blocking or reordering.
 *
 * Storage precision.  The one value the method stores in a narrower type than
 * it computes is the KV cache: the device keeps keys (after rotation) and values
 * in bf16.  Flag ORC_KV_BF16 rounds them to bf16 as they enter the cache, so that
 * the oracle attends over the same stored values.  Every other quantity stays
 * fp64 here (the device computes activations in fp32, and its prefill feeds the
 * tensor cores each activation as a pair of bf16 terms whose sum carries ~16
 * significant bits, so no activation rounding is mirrored).
 * The argmax is decided on logits rounded to fp32, the precision in which the
 * device decides it.
 *
 * Weights.  Each tensor is either a caller-supplied bf16 array or generated on
 * the fly from the counter-based generator below, so that full-size shapes need
 * no storage.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORC_KV_BF16 1

/* ------------------------------------------------------------------------- */
/* Seeded synthetic weights: SplitMix64 (Steele, Lea & Flood, "Fast splittable
 * pseudorandom number generators", OOPSLA 2014) used as a counter-based
 * generator: output k of the stream seeded with s is mix(s + (k+1)*gamma).    */
/* ------------------------------------------------------------------------- */
uint64_t orc_splitmix64(uint64_t seed, uint64_t k) {
    uint64_t z = seed + (k + 1u) * 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

/* fp32 -> bf16, round to nearest even (finite inputs). */
uint16_t orc_f32_to_bf16(float f) {
    uint32_t u;
    memcpy(&u, &f, 4);
    if ((u & 0x7f800000u) == 0x7f800000u) return (uint16_t)((u >> 16) | ((u & 0xffffu) ? 0x40u : 0u));
    u += 0x7fffu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

float orc_bf16_to_f32(uint16_t h) {
    uint32_t u = (uint32_t)h << 16;
    float f;
    memcpy(&f, &u, 4);
    return f;
}

/* fp64 -> bf16 round to nearest even, directly from the double (one rounding). */
static double round_bf16(double v) {
    if (v == 0.0 || !isfinite(v)) return v;
    int e;
    frexp(v, &e);                    /* |v| in [2^(e-1), 2^e) */
    double ulp = ldexp(1.0, e - 8);  /* bf16 keeps 8 significant bits */
    double q = v / ulp;              /* exact: power-of-two scaling */
    double r = nearbyint(q);         /* default rounding mode: to nearest even */
    return r * ulp;
}

double orc_round_bf16(double v) { return round_bf16(v); }

/* Element `index` of generated tensor `tensor_id`: the four 16-bit fields of
 * one SplitMix64 output are summed (Irwin-Hall, n = 4), centred and scaled to
 * unit variance times 0.02 in fp32, then rounded to bf16.  kind 0: weight
 * w = bf16(0.02*z); kind 1: norm gain g = bf16(1 + 0.02*z).  All fp32 steps are
 * single IEEE operations, so the value is reproducible bit for bit. */
uint16_t orc_gen_elem(uint64_t seed, uint32_t tensor_id, uint64_t index, int kind) {
    uint64_t r = orc_splitmix64(seed, ((uint64_t)tensor_id << 40) | index);
    int32_t s = (int32_t)(r & 0xffff) + (int32_t)((r >> 16) & 0xffff) + (int32_t)((r >> 32) & 0xffff) +
                (int32_t)(r >> 48);
    volatile float z = (float)(s - 131070) * 0x1p-16f;
    volatile float w = z * 0x1.1bc77ap-5f; /* 0.02*sqrt(3) in fp32: Var(z) = 1/3 */
    if (kind == 1) {
        volatile float g = 1.0f + w;
        return orc_f32_to_bf16(g);
    }
    return orc_f32_to_bf16(w);
}

void orc_gen_tensor(uint64_t seed, uint32_t tensor_id, uint64_t first, uint64_t n, int kind, uint16_t* out) {
    /* each element depends on its index only: the order of evaluation is free */
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < (int64_t)n; ++i) out[i] = orc_gen_elem(seed, tensor_id, first + (uint64_t)i, kind);
}

/* ------------------------------------------------------------------------- */
/* Tensors: stored bf16 or generated.                                         */
/* ------------------------------------------------------------------------- */
typedef struct {
    const uint16_t* data; /* row-major bf16, or NULL: generate */
    uint64_t seed;
    uint32_t tensor_id;
    int32_t kind;
} orc_tensor;

static double tensor_at(const orc_tensor* t, uint64_t idx) {
    uint16_t h = t->data ? t->data[idx] : orc_gen_elem(t->seed, t->tensor_id, idx, t->kind);
    return (double)orc_bf16_to_f32(h);
}

/* ------------------------------------------------------------------------- */
/* The layer operations (plain definitions).                                  */
/* ------------------------------------------------------------------------- */

/* RMSNorm: y = x / sqrt(mean(x^2) + eps) * g. */
void orc_rmsnorm(const double* x, const orc_tensor* g, int n, double eps, double* y) {
    double ss = 0.0;
    for (int i = 0; i < n; ++i) ss += x[i] * x[i];
    double inv = 1.0 / sqrt(ss / n + eps);
    for (int i = 0; i < n; ++i) y[i] = x[i] * inv * tensor_at(g, (uint64_t)i);
}

/* Matrix-vector product y[r] = sum_k W[r,k] x[k] for the listed rows r of a
 * row-major [rows, ncols] weight (rows == NULL: rows 0..nrows-1). */
void orc_gemv(const orc_tensor* W, int64_t ncols, const int64_t* rows, int64_t nrows, const double* x,
              double* y) {
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < nrows; ++i) {
        int64_t r = rows ? rows[i] : i;
        double acc = 0.0;
        for (int64_t k = 0; k < ncols; ++k) acc += tensor_at(W, (uint64_t)r * (uint64_t)ncols + (uint64_t)k) * x[k];
        y[i] = acc;
    }
}

/* Rotary position embedding of one head vector v[d] at integer position p:
 * pairs (v_i, v_{i+d/2}), angle p * theta^(-2i/d), rotated counter-clockwise. */
void orc_rope(double* v, int d, int64_t p, double theta) {
    int half = d / 2;
    for (int i = 0; i < half; ++i) {
        double freq = pow(theta, -2.0 * (double)i / (double)d);
        double a = (double)p * freq;
        double c = cos(a), s = sin(a);
        double u = v[i], w = v[i + half];
        v[i] = u * c - w * s;
        v[i + half] = w * c + u * s;
    }
}

double orc_silu(double z) { return z / (1.0 + exp(-z)); }

/* Grouped-query attention for one token.  q [Hq, d]; K, V [T, Hkv, d] (cached
 * positions 0..T-1); query head h reads kv head h / (Hq/Hkv).  Scores scaled by
 * 1/sqrt(d), softmax with max subtraction; o [Hq, d].  If probs != NULL the
 * softmax rows [Hq, T] are returned too. */
void orc_attention(const double* q, const double* K, const double* V, int64_t T, int Hq, int Hkv, int d, double* o,
                   double* probs) {
    int G = Hq / Hkv;
    double scale = 1.0 / sqrt((double)d);
    double* s = (double*)malloc(sizeof(double) * (size_t)(T > 0 ? T : 1));
    for (int h = 0; h < Hq; ++h) {
        int kh = h / G;
        const double* qh = q + (size_t)h * d;
        double m = -INFINITY;
        for (int64_t t = 0; t < T; ++t) {
            const double* kt = K + ((size_t)t * Hkv + kh) * d;
            double dot = 0.0;
            for (int j = 0; j < d; ++j) dot += qh[j] * kt[j];
            s[t] = dot * scale;
            if (s[t] > m) m = s[t];
        }
        double l = 0.0;
        for (int64_t t = 0; t < T; ++t) {
            s[t] = exp(s[t] - m);
            l += s[t];
        }
        double* oh = o + (size_t)h * d;
        for (int j = 0; j < d; ++j) oh[j] = 0.0;
        for (int64_t t = 0; t < T; ++t) {
            double p = s[t] / l;
            if (probs) probs[(size_t)h * T + t] = p;
            const double* vt = V + ((size_t)t * Hkv + kh) * d;
            for (int j = 0; j < d; ++j) oh[j] += p * vt[j];
        }
    }
    free(s);
}

/* ------------------------------------------------------------------------- */
/* The model.                                                                 */
/* ------------------------------------------------------------------------- */
typedef struct {
    int32_t n_layers, hidden, n_heads, n_kv_heads, head_dim, ffn, vocab;
    double rms_eps, rope_theta;
    int32_t qk_norm; /* Qwen3: per-head RMSNorm of q and k (gains g_q, g_k [d]) before RoPE */
} orc_desc;

/* Tensor order: embed [V,H], lm_head [V,H], g_final [H], then per layer:
 * g_attn [H], wq [Hq*d,H], wk [Hkv*d,H], wv [Hkv*d,H], wo [H,Hq*d], g_mlp [H],
 * wg [F,H], wu [F,H], wd [H,F]; with qk_norm, then per layer g_q [d], g_k [d]. */
enum { T_EMBED = 0, T_LMHEAD = 1, T_GFINAL = 2, T_LAYER0 = 3, T_PER_LAYER = 9 };
enum { L_GATTN = 0, L_WQ, L_WK, L_WV, L_WO, L_GMLP, L_WG, L_WU, L_WD, L_GQ, L_GK };

/* Tensor ids used by the generator (the device library uses the same ids). */
uint32_t orc_tensor_id(int layer, int which) {
    if (layer < 0) return (uint32_t)(1 + which); /* embed 1, lm_head 2, g_final 3 */
    return (uint32_t)(16 + 16 * layer + which);
}

/* Fill tensor descriptors for a generated model. */
void orc_generated_tensors(const orc_desc* d, uint64_t seed, orc_tensor* ts) {
    for (int w = 0; w < 3; ++w) {
        ts[w].data = NULL;
        ts[w].seed = seed;
        ts[w].tensor_id = orc_tensor_id(-1, w);
        ts[w].kind = (w == T_GFINAL) ? 1 : 0;
    }
    for (int l = 0; l < d->n_layers; ++l)
        for (int w = 0; w < T_PER_LAYER; ++w) {
            orc_tensor* t = &ts[T_LAYER0 + T_PER_LAYER * l + w];
            t->data = NULL;
            t->seed = seed;
            t->tensor_id = orc_tensor_id(l, w);
            t->kind = (w == L_GATTN || w == L_GMLP) ? 1 : 0;
        }
    if (d->qk_norm)
        for (int l = 0; l < d->n_layers; ++l)
            for (int w = 0; w < 2; ++w) {
                orc_tensor* t = &ts[T_LAYER0 + T_PER_LAYER * d->n_layers + 2 * l + w];
                t->data = NULL;
                t->seed = seed;
                t->tensor_id = orc_tensor_id(l, L_GQ + w);
                t->kind = 1;
            }
}

static double maybe_bf16(double v, int on) { return on ? round_bf16(v) : v; }

/* Causal forward of one token sequence, one position at a time with a KV cache
 * (identical to a causal prefill of the whole sequence).  Positions
 * t < n_prefill use `prefill_flags`, later ones `decode_flags`.
 * Outputs per position (each may be NULL): final hidden z = RMSNorm(x)*g_final
 * [n, H]; logits [n, V]; argmax [n] (fp32 logits, lowest index on ties).
 * Returns 0, or -1 on bad arguments / allocation failure. */
int orc_forward(const orc_desc* d, const orc_tensor* ts, const int32_t* tokens, int64_t n, int64_t n_prefill,
                int prefill_flags, int decode_flags, double* out_hidden, double* out_logits, int32_t* out_argmax) {
    const int H = d->hidden, Hq = d->n_heads, Hkv = d->n_kv_heads, hd = d->head_dim, F = d->ffn, V = d->vocab;
    const int L = d->n_layers;
    if (H <= 0 || Hq <= 0 || Hkv <= 0 || hd <= 0 || (hd & 1) || Hq % Hkv || F <= 0 || V <= 0 || L < 0) return -1;
    const int qd = Hq * hd, kvd = Hkv * hd;
    for (int64_t t = 0; t < n; ++t)
        if (tokens[t] < 0 || tokens[t] >= V) return -1;

    double* Kc = (double*)malloc(sizeof(double) * (size_t)L * (size_t)(n > 0 ? n : 1) * kvd);
    double* Vc = (double*)malloc(sizeof(double) * (size_t)L * (size_t)(n > 0 ? n : 1) * kvd);
    double* x = (double*)malloc(sizeof(double) * H);
    double* y = (double*)malloc(sizeof(double) * H);
    double* q = (double*)malloc(sizeof(double) * qd);
    double* k = (double*)malloc(sizeof(double) * kvd);
    double* v = (double*)malloc(sizeof(double) * kvd);
    double* o = (double*)malloc(sizeof(double) * qd);
    double* r = (double*)malloc(sizeof(double) * (H > F ? H : F));
    double* gt = (double*)malloc(sizeof(double) * F);
    double* ut = (double*)malloc(sizeof(double) * F);
    double* a = (double*)malloc(sizeof(double) * F);
    double* z = (double*)malloc(sizeof(double) * H);
    double* lg = (double*)malloc(sizeof(double) * V);
    if (!Kc || !Vc || !x || !y || !q || !k || !v || !o || !r || !gt || !ut || !a || !z || !lg) {
        free(Kc); free(Vc); free(x); free(y); free(q); free(k); free(v); free(o); free(r);
        free(gt); free(ut); free(a); free(z); free(lg);
        return -1;
    }

    for (int64_t t = 0; t < n; ++t) {
        const int flags = t < n_prefill ? prefill_flags : decode_flags;
        const int kvb = flags & ORC_KV_BF16;
        /* embedding row */
        for (int i = 0; i < H; ++i) x[i] = tensor_at(&ts[T_EMBED], (uint64_t)tokens[t] * H + i);
        for (int l = 0; l < L; ++l) {
            const orc_tensor* lt = &ts[T_LAYER0 + T_PER_LAYER * l];
            double* Kl = Kc + (size_t)l * (size_t)n * kvd;
            double* Vl = Vc + (size_t)l * (size_t)n * kvd;
            /* attention block */
            orc_rmsnorm(x, &lt[L_GATTN], H, d->rms_eps, y);
            orc_gemv(&lt[L_WQ], H, NULL, qd, y, q);
            orc_gemv(&lt[L_WK], H, NULL, kvd, y, k);
            orc_gemv(&lt[L_WV], H, NULL, kvd, y, v);
            if (d->qk_norm) { /* per-head RMSNorm with the layer's g_q / g_k, before the rotation */
                const orc_tensor* qk = &ts[T_LAYER0 + T_PER_LAYER * L + 2 * l];
                for (int h = 0; h < Hq; ++h) orc_rmsnorm(q + (size_t)h * hd, &qk[0], hd, d->rms_eps, q + (size_t)h * hd);
                for (int h = 0; h < Hkv; ++h) orc_rmsnorm(k + (size_t)h * hd, &qk[1], hd, d->rms_eps, k + (size_t)h * hd);
            }
            for (int h = 0; h < Hq; ++h) orc_rope(q + (size_t)h * hd, hd, t, d->rope_theta);
            for (int h = 0; h < Hkv; ++h) orc_rope(k + (size_t)h * hd, hd, t, d->rope_theta);
            for (int i = 0; i < kvd; ++i) {
                Kl[(size_t)t * kvd + i] = maybe_bf16(k[i], kvb);
                Vl[(size_t)t * kvd + i] = maybe_bf16(v[i], kvb);
            }
            orc_attention(q, Kl, Vl, t + 1, Hq, Hkv, hd, o, NULL);
            orc_gemv(&lt[L_WO], qd, NULL, H, o, r);
            for (int i = 0; i < H; ++i) x[i] += r[i];
            /* MLP block */
            orc_rmsnorm(x, &lt[L_GMLP], H, d->rms_eps, y);
            orc_gemv(&lt[L_WG], H, NULL, F, y, gt);
            orc_gemv(&lt[L_WU], H, NULL, F, y, ut);
            for (int i = 0; i < F; ++i) a[i] = orc_silu(gt[i]) * ut[i];
            orc_gemv(&lt[L_WD], F, NULL, H, a, r);
            for (int i = 0; i < H; ++i) x[i] += r[i];
        }
        orc_rmsnorm(x, &ts[T_GFINAL], H, d->rms_eps, z);
        if (out_hidden) memcpy(out_hidden + (size_t)t * H, z, sizeof(double) * H);
        if (out_logits || out_argmax) {
            orc_gemv(&ts[T_LMHEAD], H, NULL, V, z, lg);
            if (out_logits) memcpy(out_logits + (size_t)t * V, lg, sizeof(double) * V);
            if (out_argmax) {
                int best = 0;
                float bv = (float)lg[0];
                for (int i = 1; i < V; ++i) {
                    float fv = (float)lg[i];
                    if (fv > bv) { bv = fv; best = i; }
                }
                out_argmax[t] = best;
            }
        }
    }
    free(Kc); free(Vc); free(x); free(y); free(q); free(k); free(v); free(o); free(r);
    free(gt); free(ut); free(a); free(z); free(lg);
    return 0;
}

int orc_num_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
