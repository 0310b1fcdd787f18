/*
 * loip.h -- C ABI of libloip: single-GPU lossless LLaMA-style decoding with
 * layer weights offloaded to pinned host memory and streamed into device slots
 * while earlier layers compute (LOIP, arXiv 2512.21835, reduced to one GPU).
 *
 * Conventions
 *   - Every call returns an int status (LOIP_OK = 0 or a LOIP_ERR_* code); no
 *     C++ exception crosses this boundary.  loip_last_error() gives a message.
 *   - "dev" pointers are CUDA device pointers, "host" pointers are ordinary
 *     host memory.  The caller owns every pointer it passes in; the library
 *     never frees them.  Streams are passed as `void*` holding a cudaStream_t
 *     (NULL = the context's own stream).
 *   - bf16 values are passed as uint16_t bit patterns; activations are fp32.
 *   - Weight matrices are row-major [out, in] (out rows of `in` contiguous
 *     elements).
 *   - Calls on one context are not thread-safe.
 *
 * Layer blob (one decoder layer, the unit that is offloaded and streamed):
 *   g_attn [H] | wqkv [(Hq+2Hkv)*d, H] (q rows, then k rows, then v rows) |
 *   wo [H, Hq*d] | g_mlp [H] | wg [F, H] | wu [F, H] | wd [H, F]
 *   all bf16, each part starting at a 256-byte boundary of the blob;
 *   loip_layer_layout() returns the offsets and the blob size (l_size).
 *   The MHA block is g_attn..wo and the MLP block g_mlp..wd (the paper's
 *   decomposition of a layer into MHA and MLP blocks, Sec. III-D).
 */
#ifndef LOIP_H
#define LOIP_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum {
    LOIP_OK = 0,
    LOIP_ERR_INVALID = 1,    /* bad argument (null pointer, size, range, alignment) */
    LOIP_ERR_OOM = 2,        /* device arena or pinned host memory exhausted */
    LOIP_ERR_INFEASIBLE = 3, /* budget cannot hold the fixed part, KV cache and slots */
    LOIP_ERR_CUDA = 4,       /* a CUDA runtime call failed (message has the CUDA error) */
    LOIP_ERR_TIMEOUT = 5,    /* a host wait on the device passed its deadline */
    LOIP_ERR_STATE = 6       /* call not valid in the context's current state */
};

/* OVERLAP: offloaded layers stream into the device slots on the copy stream
 *   while earlier layers compute (Sec. III-C).
 * NAIVE: the conventional path the paper measures against (Sec. II-B): one
 *   slot, each load issued when its layer is reached, compute waits for it.
 * DIRECT: decode steps read the offloaded layers' weights in place from the
 *   pinned host pool through its device mapping (zero-copy over the host link;
 *   the counterpart of the paper's UMA-aware loading, Sec. III-C, on a
 *   discrete-memory GPU).  Prefill, loip_stream_layer and loip_layer_forward
 *   keep using the slots, so the plan still reserves them.  At batch 1 the
 *   projections of host-resident weights run on the persistent GEMV (the
 *   resident path uses the block-tile one for row-poor matrices), so decode
 *   hidden states equal an all-resident run's to rounding (tokens equal in
 *   the tests) rather than bit for bit; at larger batches both paths agree bit for bit. */
enum { LOIP_MODE_OVERLAP = 0, LOIP_MODE_NAIVE = 1, LOIP_MODE_DIRECT = 2 };

typedef struct loip_model_desc {
    int32_t n_layers, hidden, n_heads, n_kv_heads, head_dim, ffn, vocab;
    float rms_eps;    /* RMSNorm epsilon */
    float rope_theta; /* rotary base */
    int32_t qk_norm;  /* 1: Qwen3-style layer, a per-head RMSNorm of the queries and keys
                       * (gains g_q, g_k [head_dim], epsilon rms_eps) before the rotation */
} loip_model_desc;

typedef struct loip_config {
    uint64_t device_budget_bytes; /* size of the device arena the context may use */
    int32_t n_slots;              /* device slots for streamed layers, 1..3 */
    int32_t page_tokens;          /* KV page size in tokens (64) */
    int32_t max_batch;            /* largest decode batch (<= 8) */
    int32_t max_ctx;              /* largest context per request, tokens */
    int32_t layer_run_kernel;     /* 0: one kernel launch per operation (default, fastest as
                                   * measured); 1: at batch 1, each run of consecutive resident
                                   * layers is computed by one persistent cooperative kernel
                                   * (grid barriers between the phases of a layer) */
    int32_t mode;                 /* LOIP_MODE_OVERLAP, LOIP_MODE_NAIVE or LOIP_MODE_DIRECT */
    uint32_t timeout_ms;          /* deadline of every host wait (0 = 600000) */
    double hbm_Bps;               /* bandwidths used by the planner's step model */
    double link_Bps;
    uint64_t kv_reserve_bytes;    /* KV bytes to reserve at create (0 = max_batch*max_ctx) */
    int32_t max_prefill_tokens;   /* tokens per prefill pass (workspace size; 0 = 512) */
    int32_t whole_layers;         /* 0: block granularity (Sec. III-D/E): memory left after the
                                   * whole-layer plan keeps MHA/MLP blocks of offloaded layers
                                   * resident (loip_refine_blocks), and KV growth offloads single
                                   * blocks chosen by Eq. 7 (loip_eq7_choice); 1: whole layers
                                   * only (one more layer offloaded per threshold) */
    uint64_t host_budget_bytes;   /* pinned host memory for streamed layers (0 = unlimited); layers
                                   * beyond it live in the SSD tier (ssd_dir), read back through four
                                   * staging buffers taken out of this budget */
    const char* ssd_dir;          /* directory of the SSD tier's scratch file (caller-owned string,
                                   * read at create; NULL = /tmp) */
    int32_t pack_stream;          /* 1: streamed layers cross the host link losslessly packed
                                   * (sign-and-mantissa bytes + exponents coded in three levels
                                   * per 1024-word superblock, 1440 of 2048 bytes; unpacked into
                                   * the slot on the device, bit for bit) -- see loip_k_pack.  Ignored in
                                   * LOIP_MODE_DIRECT and with the SSD tier (host_budget_bytes > 0).
                                   * 0: raw blobs (default) */
    int32_t embed_on_host;        /* 1: the embedding table [vocab, hidden] stays in pinned host
                                   * memory, mapped for the device, and the embedding gather reads
                                   * each token's row over the host link (16 KB per token at the 70B
                                   * shape); its vocab * hidden * 2 bytes of device budget go to
                                   * resident weights instead.  0: in the device arena (default) */
} loip_config;

typedef struct loip_layer_layout_t {
    uint64_t off_g_attn, off_wqkv, off_wo, off_g_mlp, off_wg, off_wu, off_wd;
    uint64_t l_size;   /* blob bytes */
    uint64_t mha_bytes, mlp_bytes;
    uint64_t off_g_q, off_g_k;  /* QK-norm gains (qk_norm models; inside the MHA block, after Wo) */
} loip_layer_layout_t;

typedef struct loip_plan {
    int32_t n_layers;
    int32_t n_resident, n_offloaded;
    uint8_t* resident;     /* [n_layers], caller-owned; 1 = resident in HBM, 0 = streamed */
    double pred_step_s;    /* discrete-event step time with n_slots slots */
    double pred_copy_s;    /* offloaded bytes / link bandwidth */
    double pred_compute_s; /* all weight bytes / HBM bandwidth */
    double eq1_step_s;     /* Eq. 1 with one device (single-slot bound) */
    uint64_t left_bytes;   /* budget left after fixed, KV, resident layers and slots */
} loip_plan;

typedef struct loip_stats {
    uint64_t steps, tokens;
    uint64_t h2d_weight_bytes; /* bytes streamed host -> slots */
    double last_step_ms;       /* host wall time of the last decode/prefill call */
    double copy_busy_ms;       /* copy-stream busy time, last step (events) */
    double compute_ms;         /* compute-stream time, last step (events) */
    int32_t n_resident, n_offloaded, n_replans;
    uint64_t kv_tokens;        /* tokens held in the KV cache (all requests) */
    uint64_t kv_bytes;         /* bytes of KV pages allocated */
    uint64_t arena_used;       /* device arena bytes in use */
    /* per kernel class, accumulated while kernel timing is on (loip_set_kernel_timing):
     * decode: 0 qkv+rope, 1 attention (+combine), 2 o-proj, 3 gate/up, 4 down, 5 lm head (+argmax);
     * prefill: 6 qkv GEMM, 7 attention, 8 o-proj GEMM, 9 gate/up GEMM, 10 down GEMM, 11 RMSNorm;
     * 12 persistent layer run (decode at batch 1, a run of resident layers in one launch);
     * 13 unpack of packed streamed chunks (on the unpack stream); 14-15 unused */
    double kernel_ms[16];
    uint64_t kernel_launches[16];
    double copy_ms_total;      /* summed duration of every completed layer copy (events) */
    uint64_t copies_total;     /* number of completed layer copies */
    double pool_min_GBps;      /* slowest host-pool blob copy when the pool was qualified */
    double pool_median_GBps;   /* median blob copy rate at qualification */
    uint64_t pool_replaced;    /* blobs moved to fresh host memory because they copied slowly */
    int32_t n_ssd_layers;      /* streamed layers whose blob lives in the SSD tier */
    uint64_t ssd_read_bytes;   /* bytes read from the SSD tier since create */
    double ssd_wait_ms;        /* host time spent waiting for SSD-tier reads to land */
    double ssd_stage_wait_ms;  /* host time spent waiting for a staging buffer's copy to a slot */
    double ssd_copy_ms;        /* summed duration of the copies out of staging buffers (events) */
    int32_t pool_numa_node;    /* host NUMA node the pool's pages were asked for (the GPU's, -1: none) */
    int32_t pool_blobs;        /* streamed layers with a blob in the host pool */
    int32_t pool_blobs_on_node;/* of those, blobs whose sampled pages are mostly on pool_numa_node */
    double pool_huge_min;      /* smallest share of a host-pool region in huge pages (1 = all) */
    uint64_t unpack_launches;  /* unpack kernels enqueued (packed streaming) */
    uint64_t unpack_bytes;     /* packed bytes they read plus raw bytes they write */
} loip_stats;

typedef struct loip_ctx loip_ctx;

/* ---------------------------------------------------------------------------
 * Host-only planning (no GPU needed)
 * ------------------------------------------------------------------------- */

/* Blob layout of one layer of `desc`.  LOIP_ERR_INVALID on bad shapes
 * (hidden and ffn multiples of 8, head_dim even, n_heads % n_kv_heads == 0). */
int loip_layer_layout(const loip_model_desc* desc, loip_layer_layout_t* out);

/* Residency plan (Algorithm 1's memory-first fill, Sec. III-D; Eq. 1 and Eq. 2,
 * Sec. III-B/III-D, with a single device and no network term).
 *   layer_bytes [n_layers]: bytes of each layer (slots are sized by the largest).
 *   R = the largest count with fixed + kv + R*l + n_slots*l <= budget (no slot
 *   if all layers fit); the n_layers-R offloaded layers are spread evenly
 *   (layer i offloaded iff floor((i+1)m/L) > floor(i m/L)), the single-device
 *   form of the interleaved placement of Sec. III-A.
 *   out->resident must point to n_layers bytes.
 * LOIP_ERR_INFEASIBLE if the budget cannot hold fixed + kv + the slots. */
int loip_plan_residency(const loip_model_desc* desc, const uint64_t* layer_bytes, uint64_t device_budget,
                        uint64_t kv_bytes, uint64_t fixed_bytes, int32_t n_slots, double hbm_Bps, double link_Bps,
                        loip_plan* out);

/* Eq. 6 (online memory-aware planner, Sec. III-E), read as a token count:
 * the number of KV tokens the memory left after a plan can still hold. */
int loip_kv_threshold(uint64_t left_bytes, uint64_t kv_bytes_per_token, uint64_t* out_tokens);

/* Algorithm 1's fine-grained step (Sec. III-D) on one device: a decoder layer
 * is an MHA block (g_attn, Wqkv, Wo: loip_layer_layout's mha_bytes) and an MLP
 * block (g_mlp, Wg, Wu, Wd: mlp_bytes).  While `left_bytes` (device memory left
 * after the whole-layer plan) can hold a block of a still fully offloaded
 * layer, that layer (in layer order) keeps its MLP block resident if it fits,
 * else its MHA block.  offloaded[l] != 0 marks the plan's offloaded layers
 * (n_layers bytes); masks[l] (n_layers bytes, caller-owned) receives the
 * resident blocks: bit 0 MHA, bit 1 MLP (3 = whole layer).  *left_out = memory
 * still left.  Host only. */
int loip_refine_blocks(const loip_model_desc* desc, uint64_t left_bytes, const uint8_t* offloaded, uint8_t* masks,
                       uint64_t* left_out);

/* Eq. 7 (online memory-aware planner, Sec. III-E) on one device: the numbers
 * of resident MHA blocks (*alpha <= n_mha) and MLP blocks (*beta <= n_mlp) to
 * offload so that their memory covers need_bytes, with the fewest bytes
 * offloaded (each is streamed once per step afterwards), then the fewest
 * blocks.  LOIP_ERR_INFEASIBLE when all of them together do not cover it. */
int loip_eq7_choice(const loip_model_desc* desc, uint64_t need_bytes, int32_t n_mha, int32_t n_mlp, int32_t* alpha,
                    int32_t* beta);

/* Bytes of the fixed device part of a context (embedding, LM head, final
 * gain, page table, workspaces) for `desc` and `cfg`. */
int loip_fixed_bytes(const loip_model_desc* desc, const loip_config* cfg, uint64_t* out);

/* ---------------------------------------------------------------------------
 * Context
 * ------------------------------------------------------------------------- */

/* Creates a context on the current CUDA device.  `device_arena` (dev, at least
 * cfg->device_budget_bytes, 256-byte aligned) holds every device byte the
 * context uses: fixed part, resident layers, slots, KV pages.  The library
 * allocates pinned host memory for offloaded layers (it owns it) and its own
 * streams and events.  The plan is made here (loip_plan_residency with the KV
 * reserve).  *out is NULL on failure. */
int loip_create(const loip_model_desc* desc, const loip_config* cfg, void* device_arena, uint64_t arena_bytes,
                loip_ctx** out);

void loip_destroy(loip_ctx* ctx);

/* Message of the last failed call on ctx (or, when ctx is NULL, of the last
 * failed create or kernel-level loip_k_* launch on this thread).  Valid until
 * the next call. */
const char* loip_last_error(const loip_ctx* ctx);

/* Fills every weight with the seeded SplitMix64 generator (bf16 N(0, 0.02^2)
 * approximations; norm gains 1 + 0.02 z): resident layers are written in place,
 * offloaded layers are generated on the device and copied to the pinned host
 * pool.  Then the first slots are filled.  Synchronous. */
int loip_load_weights_generated(loip_ctx* ctx, uint64_t seed);

/* Loads one layer from a caller blob (host, l_size bytes, layout above) into
 * its resident block or host-pool entry.  Synchronous. */
int loip_load_layer(loip_ctx* ctx, int32_t layer, const void* host_blob, uint64_t bytes);

/* Loads embedding / LM head [vocab, hidden] and final gain [hidden] (host bf16). */
int loip_load_globals(loip_ctx* ctx, const uint16_t* embed, const uint16_t* lm_head, const uint16_t* g_final);

/* Current plan (resident[] must hold n_layers bytes). */
int loip_get_plan(const loip_ctx* ctx, loip_plan* out);

/* The context's block-level residency: masks[l] (n_layers bytes, caller-owned)
 * = resident blocks of layer l (bit 0 MHA, bit 1 MLP; 3 = whole layer, 0 =
 * fully streamed); *stream_bytes_per_step = bytes the slot ring copies per
 * pass over the layers (every non-resident block once). */
int loip_get_block_plan(const loip_ctx* ctx, uint8_t* masks, uint64_t* stream_bytes_per_step);

/* Enqueues the copy of offloaded `layer` from the pinned host pool into device
 * slot `slot` on `copy_stream` (the "stream layer" step, Sec. III-C: the slot
 * is rewritten only after the compute that used it has signalled, through a
 * CUDA event, that it is done).  Records the slot-full event.  Async. */
int loip_stream_layer(loip_ctx* ctx, int32_t layer, int32_t slot, void* copy_stream);

/* Enqueues one decoder layer on `compute_stream` for `batch` requests:
 *   hidden (dev, fp32 [batch, H]) is updated in place (residual stream);
 *   positions (dev, int32 [batch]) are the token positions; the new k/v are
 *   appended to each request's KV pages at that position (request b = row b).
 *   The layer's weights are its resident block, or slot `slot` if offloaded
 *   (the call waits on that slot's full event and records its free event).
 * Async.  Requires that the requests' contexts were set by loip_set_batch. */
int loip_layer_forward(loip_ctx* ctx, int32_t layer, int32_t slot, float* hidden, const int32_t* positions,
                       int32_t batch, void* compute_stream);

/* Declares the active requests for the following decode steps: request b has
 * ctx_lens[b] tokens already in its cache (host, int32 [batch]).  Allocates KV
 * pages as needed. */
int loip_set_batch(loip_ctx* ctx, int32_t batch, const int32_t* ctx_lens);

/* One greedy decode step for the active batch: tokens (host, int32 [batch]) are
 * the current tokens; out_tokens (host, int32 [batch]) receive the argmax of
 * the logits (lowest index on ties); out_hidden (dev fp32 [batch, H] or NULL)
 * receives the final-norm hidden state.  Streams offloaded layers through the
 * slots with the copy of slot k starting once its previous layer is computed,
 * continuing into the next step's first layers.  Synchronous. */
int loip_decode_step(loip_ctx* ctx, const int32_t* tokens, int32_t batch, int32_t* out_tokens, float* out_hidden);

/* Same step, with tokens, out_tokens (int32 [batch]) and out_hidden in device
 * memory; enqueued on the context's compute stream without a host wait. */
int loip_decode_step_device(loip_ctx* ctx, const int32_t* tokens_dev, int32_t batch, int32_t* out_tokens_dev,
                            float* out_hidden);

/* Prefill of n_prompts prompts (tokens host int32, concatenated; prompt_lens
 * host int32 [n_prompts]) into requests 0..n_prompts-1, each starting at
 * position 0.  Writes the argmax after each prompt's last token (host int32
 * [n_prompts]) and optionally the final hidden of those tokens (dev fp32
 * [n_prompts, H]).  Weights stream exactly as in decode.  Synchronous. */
int loip_prefill(loip_ctx* ctx, const int32_t* tokens, const int32_t* prompt_lens, int32_t n_prompts,
                 int32_t* out_tokens, float* out_hidden);

/* The most recent completed layer copies into the slots (up to 8192 kept):
 * writes min(max_n, kept) entries, oldest first, of their duration (ms, CUDA
 * events on the copy stream) and size (bytes) to ms / bytes (host arrays of
 * max_n) and returns the count, or -1 on bad arguments.  Per-copy rates show
 * which steps the host link slowed (Sec. III-C's loading path). */
int32_t loip_get_copy_log(loip_ctx* ctx, double* ms, uint64_t* bytes, int32_t max_n);

/* Host NUMA node holding most of each layer's pool blob (host int32
 * [n_layers]; -1 for layers without a blob, or when the kernel cannot tell),
 * read with move_pages queries of 32 pages per blob when the pool was filled.
 * The pool asks for the GPU's host node (loip_stats.pool_numa_node). */
int loip_get_pool_nodes(loip_ctx* ctx, int32_t* nodes);

/* Fault injection, for tests of the failure handling (the paper has no
 * counterpart: it reports only out-of-memory and out-of-time outcomes, Sec.
 * IV-A).  Arms one fault on the context; it fires once, at the next place
 * named below, and is made on the host or as a bounded device wait -- never as
 * a GPU fault, trap or hang:
 *   LOIP_FAULT_WAIT        the next host wait on the device treats its event
 *                          as still pending: the call returns LOIP_ERR_TIMEOUT
 *                          after loip_config.timeout_ms (the device work itself
 *                          completes) and the context then refuses every call
 *                          with LOIP_ERR_STATE;
 *   LOIP_FAULT_COPY        the next weight copy into a slot reports a CUDA error
 *                          before anything is enqueued: LOIP_ERR_CUDA, context
 *                          failed;
 *   LOIP_FAULT_HOST_ALLOC  the next pinned host-pool allocation fails:
 *                          LOIP_ERR_OOM (the context stays usable);
 *   LOIP_FAULT_BARRIER     the next layer-run kernel launch (batch-1 decode with
 *                          loip_config.layer_run_kernel = 1): block `arg` does
 *                          not arrive at the first grid barrier and every
 *                          barrier wait of that launch gives up after 10 ms; the
 *                          kernel sets its error word and returns, and the step
 *                          returns LOIP_ERR_TIMEOUT (context failed; the GPU and
 *                          other contexts stay usable);
 *   LOIP_FAULT_NONE        disarms.
 * LOIP_ERR_INVALID for an unknown kind or a negative block. */
#define LOIP_FAULT_NONE 0
#define LOIP_FAULT_WAIT 1
#define LOIP_FAULT_COPY 2
#define LOIP_FAULT_HOST_ALLOC 3
#define LOIP_FAULT_BARRIER 4
int loip_inject_fault(loip_ctx* ctx, int32_t kind, int32_t arg);

/* The deadline loop every host wait of the library runs, driven by a fake
 * device that reports "pending" for `pending_polls` polls (< 0: forever):
 * LOIP_OK once it reports done, LOIP_ERR_TIMEOUT once timeout_ms of wall time
 * have passed; *waited_ms (may be NULL) gets the time spent.  Makes no CUDA
 * call, so it checks the deadline logic on a machine without a GPU. */
int loip_poll_deadline_check(uint32_t timeout_ms, int32_t pending_polls, double* waited_ms);

/* Re-plans for the current KV size (Eq. 6 thresholds): while the KV pages the
 * next `lookahead_tokens` tokens of every request need do not fit, device
 * weights are given up for KV memory.  With block granularity (the default,
 * loip_config.whole_layers = 0) Eq. 7 chooses how many MHA and MLP blocks to
 * give up for the shortfall (the fewest streamed bytes that cover it); with
 * whole_layers = 1 one more resident layer is demoted at a time, evenly
 * spaced.  Demoted weights keep a host copy and stream from then on.
 * Synchronous. */
int loip_replan(loip_ctx* ctx, int32_t lookahead_tokens);

int loip_get_stats(const loip_ctx* ctx, loip_stats* out);

/* Kernel timing: when enable != 0, every decode-layer kernel is bracketed by
 * CUDA events on its stream and the durations are summed per kernel class into
 * loip_stats.kernel_ms / kernel_launches (reset on every enable call). */
int loip_set_kernel_timing(loip_ctx* ctx, int32_t enable);

/* Waits (with the context deadline) until all work of the context is done. */
int loip_synchronize(loip_ctx* ctx);

/* Host-link throughput as the layer copies see it: best of `reps` timed
 * cudaMemcpyAsync of `bytes` (>= 1 MiB) from pinned, huge-page-backed host
 * memory (the pool's allocator) to device memory on the current device.
 * Allocates and frees its own buffers.  *out_Bps in bytes per second. */
int loip_measure_h2d(uint64_t bytes, int32_t reps, double* out_Bps);

/* SSD tier check (Sec. III-C's storage tier; loip_config.ssd_dir): writes
 * `bytes` (a multiple of 4096) of a pattern to an unlinked O_DIRECT scratch file
 * in `dir` (NULL: /tmp) and reads it back through io_uring; *ok = 1 when the
 * bytes match.  Host only.  LOIP_ERR_STATE when the file or the ring cannot be
 * set up on this machine. */
int loip_ssd_roundtrip(const char* dir, uint64_t bytes, int32_t* ok);

/* Host-link throughput as direct-access kernels see it: best of `reps` timed
 * launches of a kernel that streams `bytes` (>= 1 MiB, a multiple of 16) with
 * 128-bit loads from a pinned, mapped host buffer (the pool's allocator), one
 * block per SM x 4.  Allocates and frees its own buffers.  *out_Bps in bytes
 * per second.  The paper has no counterpart; it is the roofline of
 * LOIP_MODE_DIRECT decode. */
int loip_measure_direct_read(uint64_t bytes, int32_t reps, double* out_Bps);

/* Device pointer of the compute / copy stream (cudaStream_t). */
void* loip_compute_stream(loip_ctx* ctx);
void* loip_copy_stream(loip_ctx* ctx);

/* ---------------------------------------------------------------------------
 * Kernel-level entry points (the fused kernels of one decoder layer, for tests
 * and for callers that compose their own loop).  All are async on `stream`,
 * take device pointers, and return LOIP_ERR_INVALID on bad sizes or
 * misaligned pointers (weights and vectors 16-byte aligned).  B <= 8.
 * ------------------------------------------------------------------------- */

/* Seeded generator: out (dev bf16 [n]) = element first..first+n-1 of tensor
 * `tensor_id`; kind 0 = weight 0.02 z, kind 1 = gain 1 + 0.02 z. */
int loip_k_generate(uint16_t* out, uint64_t n, uint64_t first, uint64_t seed, uint32_t tensor_id, int32_t kind,
                    void* stream);

/* x[b, :] = embed[tokens[b], :] (bf16 -> fp32). */
int loip_k_embed(const uint16_t* embed, const int32_t* tokens, int32_t B, int32_t H, float* x, void* stream);

/* RMSNorm (LLaMA pre-norm) fused into a matrix-vector product with query/key
 * rotation: y = x / sqrt(mean(x^2) + eps) * g; qkv = wqkv y; q and k heads
 * rotated at positions[b] (pairs (i, i + d/2), angle pos * theta^(-2i/d),
 * computed in fp64); q -> q_out (fp32 [B, Hq*d]); k and v are rounded to bf16
 * and written into request b's paged cache at positions[b] (page table row b,
 * page layout as for loip_k_attention). */
int loip_k_qkv_rope(const float* x, const uint16_t* g, const uint16_t* wqkv, int32_t B, int32_t H, int32_t Hq,
                    int32_t Hkv, int32_t d, float eps, float theta, const int32_t* positions, float* q_out,
                    const void* kv_base, const int64_t* page_offsets, int32_t max_pages, int32_t page_tokens,
                    int32_t layer, uint64_t layer_page_bytes, void* stream);

/* Split-K grouped-query decode attention over a paged cache:
 *   q (fp32 [B, Hq*d]); request b attends over its first ctx_lens[b] cached
 *   positions; page_offsets (dev int64 [B, max_pages]) gives each page's byte
 *   offset from kv_base; a page holds, for layer `layer`, K then V as
 *   [Hkv][page_tokens][d] bf16 at layer * layer_page_bytes inside the page
 *   (page_tokens = 64; q, kv_base 16-byte aligned; max_ctx <= 16384).
 *   Writes o (fp32 [B, Hq*d]).  `scratch` (dev, at least
 *   loip_k_attention_scratch_floats(...) floats) holds the per-page partial
 *   softmax states and per-(request, head) completion counters; it needs no
 *   initialisation (the call zeroes the counters on `stream`). */
int loip_k_attention(const float* q, const void* kv_base, const int64_t* page_offsets, int32_t max_pages,
                     const int32_t* ctx_lens, int32_t B, int32_t Hq, int32_t Hkv, int32_t d, int32_t page_tokens,
                     int32_t layer, uint64_t layer_page_bytes, int32_t max_ctx, float* scratch, float* o,
                     void* stream);
uint64_t loip_k_attention_scratch_floats(int32_t B, int32_t Hq, int32_t d, int32_t max_ctx, int32_t page_tokens);

/* Scratch of loip_k_attention_noalloc: 4 Mi floats (16 MiB) per GPU. */
#define LOIP_NOALLOC_SCRATCH_FLOATS (4ull << 20)

/* loip_k_attention for callers that cannot allocate device memory: a process
 * whose HBM is fully reserved by another allocator (a fixed arena, a caching
 * allocator), where cudaMalloc would fail or break the memory budget, or a
 * latency-critical path that must not pay the device-wide synchronisation of
 * cudaMalloc/cudaFree.  The paper has no counterpart; this is a library
 * convenience.  Same arguments and result as loip_k_attention without
 * `scratch`: the partial softmax states and completion counters go to a
 * file-scope device array of LOIP_NOALLOC_SCRATCH_FLOATS floats that every GPU
 * loading the library holds until the process exits.  LOIP_ERR_INVALID when
 * loip_k_attention_scratch_floats(B, Hq, d, max_ctx, page_tokens) exceeds that
 * size, when Hq / Hkv is not 1, 2, 4 or 8, or when a pointer is misaligned (q
 * and kv_base need 16 bytes, page_offsets 8, ctx_lens and o 4); every refusal
 * happens before anything is enqueued.  It allocates nothing (no cudaMalloc, cudaFree or allocating library
 * call).  The first call on a device, with that device current, looks up the
 * array's device address (cudaGetSymbolAddress); make that first call before
 * any stream capture.  All calls on a device share the array and it keeps the
 * last call's contents; each call clears the counters it needs on `stream`
 * (cudaMemsetAsync) before its kernel: calls that overlap on the GPU race. */
int loip_k_attention_noalloc(const float* q, const void* kv_base, const int64_t* page_offsets, int32_t max_pages,
                             const int32_t* ctx_lens, int32_t B, int32_t Hq, int32_t Hkv, int32_t d,
                             int32_t page_tokens, int32_t layer, uint64_t layer_page_bytes, int32_t max_ctx, float* o,
                             void* stream);

/* Causal prefill attention on the tensor cores (the attention of a prefill
 * pass, Sec. III-A's decoder layer on a prompt): n_prompts prompts of
 * prompt_lens[i] tokens (host int32) whose rows are concatenated in q (fp32
 * [M, Hq*d], M = sum of the lengths, 16-byte aligned); prompt i's rows sit at
 * positions first_pos[i] .. first_pos[i] + len - 1 (host int32, NULL = 0) of
 * request i, and each row attends over that request's cached positions 0 ..
 * its own (keys and values already in the pages, layout as in
 * loip_k_attention; request i's pages are row i of page_offsets).  Query and
 * probability operands go to the tensor cores as split bf16 pairs (fp32
 * accuracy).  Writes o2 (bf16 [2][M][Hq*d]: hi = bf16(o) then lo = bf16(o -
 * hi), the next projection's split operand).  `tiles` is device scratch of at
 * least (M + n_prompts) * 16 bytes (the query-tile list, uploaded on `stream`).
 * d = 64 or 128, Hq / Hkv = 1, 2, 4 or 8, page_tokens = 64. */
int loip_k_prefill_attention(const float* q, const void* kv_base, const int64_t* page_offsets, int32_t max_pages,
                             const int32_t* prompt_lens, const int32_t* first_pos, int32_t n_prompts, int32_t Hq,
                             int32_t Hkv, int32_t d, int32_t page_tokens, int32_t layer, uint64_t layer_page_bytes,
                             void* tiles, uint16_t* o2, void* stream);

/* 0 if no tensor-core attention launch has recorded a failure (a bounded wait
 * that ran out); otherwise the first failure code.  -1 if unreadable. */
int loip_k_attention_tc_status(void);

/* x += wo o  (output projection with the residual add); o fp32 [B, Hq*d].  As in
 * decode, at batch 1 the blocks of the first wave also pull the later blocks'
 * weight tiles into L2 (a cache hint: results equal loip_k_down's bit for bit). */
int loip_k_oproj(const float* o, const uint16_t* wo, int32_t B, int32_t H, int32_t K, float* x, void* stream);

/* a = silu(wg y) * (wu y) with y = RMSNorm(x) * g (SwiGLU MLP input half);
 * a fp32 [B, F]. */
int loip_k_gate_up(const float* x, const uint16_t* g, const uint16_t* wg, const uint16_t* wu, int32_t B, int32_t H,
                   int32_t F, float eps, float* a, void* stream);

/* x += wd a  (down projection with the residual add); a fp32 [B, F]. */
int loip_k_down(const float* a, const uint16_t* wd, int32_t B, int32_t H, int32_t F, float* x, void* stream);

/* Prefill projection on the tensor cores: x[M, N] += A[M, K] * W[N, K]^T with
 * A and W bf16 row-major (K-contiguous, K % 8 == 0, 16-byte aligned), x fp32
 * (N % 4 == 0), fp32 accumulation (tcgen05, TMA; the product the prefill runs
 * for the output and down projections). */
int loip_k_gemm_bf16(const uint16_t* A, const uint16_t* W, int32_t M, int32_t N, int32_t K, float* x, void* stream);

/* The prefill's projection at fp32 activation precision: x[M, N] += A W^T
 * where A (fp32 [M, K]) is given as a split pair of bf16 planes A2 = [2][M][K]:
 * A2[0] = bf16(A) and A2[1] = bf16(A - A2[0]), so A2[0] + A2[1] carries A to
 * ~2^-17 relative.  Every K step issues two tensor-core MMAs into the same
 * fp32 accumulator (A2[0] W^T + A2[1] W^T); W stays the unmodified bf16 weight
 * (the losslessness of Sec. IV-A: no weight is changed).  Same layout, sizes
 * and alignment rules as loip_k_gemm_bf16; M * K elements per plane. */
int loip_k_gemm_split(const uint16_t* A2, const uint16_t* W, int32_t M, int32_t N, int32_t K, float* x, void* stream);

/* Lossless packing of bf16 weights for the host link (the streamed layers'
 * transport under loip_config.pack_stream): n_sb superblocks of 1024 words
 * (in: bf16 [n_sb * 1024], dev, 16-byte aligned) become n_sb packed
 * superblocks of LOIP_PACKED_SB bytes (out, dev, 16-byte aligned):
 *   bytes 0..1023     the sign-and-mantissa byte of every word;
 *   bytes 1024..1279  2 bits per word: with k = (the superblock's largest
 *                     exponent) - (the word's exponent), codes 0..2 name the
 *                     three most frequent k of the superblock, 3 escapes;
 *   bytes 1280..1367  2 bits per level-1 escape, in word order: codes 0..2 name
 *                     the next three most frequent k, 3 escapes (at most 352);
 *   bytes 1368..1407  4 bits per level-2 escape, in word order: k itself (0..14)
 *                     or 15, an exception (at most 80);
 *   bytes 1408..1439  a record of 8 uint32: [0] largest exponent | flag << 8 |
 *                     rank[0] << 16 | rank[1] << 24, [1] rank[2..5], [2] the
 *                     escape counts n1 | n2 << 16 | the exception count << 24,
 *                     [3..7] up to 5 exceptions as index | exponent << 16.
 * rank[] lists the six most frequent k in 0..14, most frequent first, ties to
 * the smaller k.  A superblock over one of the limits is not packed: its
 * record's first word is its largest exponent | 0xff << 8, every other byte of
 * the superblock is 0, and its index (first_sb + i) is appended
 * to raw_list (dev uint32 [1 + raw_cap]: raw_list[0] counts every such
 * superblock, the first raw_cap indices follow, in no particular order;
 * raw_list may be NULL).  loip_k_unpack restores every packed superblock bit
 * for bit and leaves the words of the others untouched.  Lossless: no weight
 * changes (Sec. IV-A). */
#define LOIP_PACKED_SB 1440
int loip_k_pack(const uint16_t* in, uint64_t n_sb, uint8_t* out, uint32_t* raw_list, uint32_t first_sb,
                uint32_t raw_cap, void* stream);
int loip_k_unpack(const uint8_t* in, uint64_t n_sb, uint16_t* out, void* stream);

/* 0 if no tensor-core GEMM launch has recorded a failure (a bounded pipeline
 * wait that ran out); otherwise the first failure code.  -1 if unreadable. */
int loip_k_tc_status(void);

/* Final RMSNorm and LM head: z = RMSNorm(x) * g_final (fp32 [B, H], may be
 * NULL), logits = lm_head z (fp32 [B, V], may be NULL) and the greedy token
 * (int32 [B], lowest index on ties).  `scratch` (dev, at least
 * loip_k_lm_head_scratch_bytes(B, V) bytes) holds per-block partial maxima. */
int loip_k_lm_head(const float* x, const uint16_t* g_final, const uint16_t* lm_head, int32_t B, int32_t H,
                   int32_t V, float eps, float* z, float* logits, int32_t* tokens, void* scratch, void* stream);
uint64_t loip_k_lm_head_scratch_bytes(int32_t B, int32_t V);

#ifdef __cplusplus
}
#endif
#endif /* LOIP_H */
