// internal.h -- launchers shared between the translation units of libloip.
// Host-side declarations only; kernels live in decode.cu / prefill.cu.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

namespace loip {

// Paged KV cache view for one layer.  A page (one per page_tokens positions of
// one request) is a contiguous group holding every layer's keys and values:
// at byte offset layer * layer_page_bytes sit K [Hkv][page_tokens][d] and then
// V [Hkv][page_tokens][d], bf16.  page_offsets[row * max_pages + i] is the
// byte offset of page i of page-table row `row` from `base`.
// Rotary inverse frequencies theta^(-2i/d), i < d/2, computed in fp64 on the host.
struct RopeFreqs {
    double inv_freq[64];
};
RopeFreqs rope_freqs(float theta, int d);

// cos/sin of pos * inv_freq: the angle is formed and reduced modulo 2*pi in fp64
// (two-term Cody-Waite reduction), then sincosf on the reduced angle.
__device__ __forceinline__ void rope_cos_sin(int pos, double inv_freq, float* c, float* s) {
    const double a = (double)pos * inv_freq;
    const double k = rint(a * 0.15915494309189535);  // 1 / (2 pi)
    double r = fma(-k, 6.283185307179586, a);          // 2 pi, high part
    r = fma(-k, 2.4492935982947064e-16, r);            // 2 pi - high part
    sincosf((float)r, s, c);
}

struct KvView {
    char* base;
    const int64_t* page_offsets;
    int32_t max_pages;
    int32_t page_tokens;
    int32_t layer;
    uint64_t layer_page_bytes;
};

// Weight-stationary matrix-vector family (decode).  B = batch rows of the fp32
// activation; every kernel streams its weight matrix exactly once.  w_host: the
// weight pointer is the device address of mapped host memory (direct access
// over the host link); the kernels then skip their L2 prefetch of it.
cudaError_t launch_qkv_rope(const float* x, const uint16_t* g, const uint16_t* wqkv, int B, int H, int Hq, int Hkv,
                            int d, float eps, float theta, const int32_t* positions, float* q_out, KvView kv,
                            const int32_t* row_req, cudaStream_t st, bool pdl = false, bool w_host = false,
                            float* qk_raw = nullptr);
// QK-norm layers (Qwen3): with qk_raw set, launch_qkv_rope leaves the query and
// key rows unrotated in qk_raw ([B][(Hq + 2 Hkv) d] fp32; values still go to the
// cache), and launch_qk_norm_rope then applies the per-head RMSNorm (gains g_q,
// g_k [d]) and the rotation and makes the usual stores.  with_v: the value rows
// of `raw` are copied to the cache as well (prefill, where raw holds all rows).
cudaError_t launch_qk_norm_rope(const float* raw, int rows, int Hq, int Hkv, int d, bool with_v, const uint16_t* g_q,
                                const uint16_t* g_k, float eps, float theta, const int32_t* positions,
                                const int32_t* row_req, float* q_out, KvView kv, cudaStream_t st, bool pdl = false);
// x += W in (W [N, K] bf16).  prefetch_waves: batch-1 tiles beyond the first
// wave are pulled into L2 by the first-wave blocks while they wait on the
// previous kernel (for the O-projection, whose predecessor, attention, leaves
// HBM idle; behind a bandwidth-bound kernel the prefetch only competes).
cudaError_t launch_resid_gemv(const float* in, const uint16_t* w, int B, int N, int K, float* x, cudaStream_t st,
                              bool pdl = false, bool w_host = false, bool prefetch_waves = false);
cudaError_t launch_gate_up(const float* x, const uint16_t* g, const uint16_t* wg, const uint16_t* wu, int B, int H,
                           int F, float eps, float* a, cudaStream_t st, bool pdl = false, bool w_host = false);
// Streams `bytes` (a multiple of 16) from `src` with 128-bit loads over `blocks`
// blocks and writes one xor-fold per block to sink[blocks] (so no load is
// dropped).  Used to measure how fast kernels read mapped host memory.
cudaError_t launch_read_stream(const void* src, uint64_t bytes, int blocks, uint32_t* sink, cudaStream_t st);
cudaError_t launch_lm_head(const float* x, const uint16_t* g, const uint16_t* w, int B, int H, int V, float eps,
                           float* z, float* logits, int32_t* tokens, void* scratch, cudaStream_t st,
                           bool pdl = false);
size_t lm_head_scratch_bytes(int B, int V);

// Grouped-query attention over the paged cache.  Rows b = 0..B-1 attend over
// their first ctx_lens[b] positions with query q[b] (ctx_lens NULL: over
// positions[b] + 1 positions, the causal window of the token at positions[b]).  row_req maps a row to its
// page-table row (NULL = identity).  split: one block per page writes its
// partial state to scratch and the last block of each (row, kv head) combines
// them into o (max_ctx <= 16384); otherwise one block per (row, kv head) loops
// over all pages.  o_split: write o as a pair of bf16 planes [2][B][Hq d],
// hi = bf16(v) and lo = bf16(v - hi) (the prefill's tensor-core operand),
// instead of fp32.
// scratch_rows: the batch the scratch was sized for (attention_scratch_floats);
// the completion counters sit after that many rows of partial states, so the
// same scratch serves every batch up to it (0 = B).  wide: split mode with a
// 256-thread block per page (same scratch layout and counters).
cudaError_t launch_attention(const float* q, KvView kv, const int32_t* ctx_lens, const int32_t* positions,
                             const int32_t* row_req, int B, int Hq, int Hkv, int d, int max_ctx, bool split,
                             float* scratch, void* o, bool o_split, cudaStream_t st, bool pdl = false,
                             int scratch_rows = 0, bool wide = false);
size_t attention_scratch_floats(int B, int Hq, int d, int max_ctx, int page_tokens);
// Split attention keeps one int completion counter per (row, head) after the
// partial states; they must be zero before a launch and every launch leaves
// them zero.
int* attention_counters(float* scratch, int B, int Hq, int d, int max_ctx, int page_tokens);

// Persistent layer run (batch 1).  One cooperative launch computes decoder
// layers layer0 .. layer0 + n_layers - 1 (all resident in device memory) for
// the single row of x: for each layer, the QKV + RoPE + KV-append tiles, the
// split attention, the O-projection, the gate/up SwiGLU and the down tiles,
// separated by grid-wide barriers.  Blocks stay resident for the whole run,
// stage each phase's input row in shared memory, take tiles from per-phase
// counters and prefetch the next phase's first weight tiles into L2 before each
// barrier.  Same arithmetic per output as the batch-1 kernels above.  sync[0]
// is the barrier counter and sync[2 ..] the tile counters (zeroed by the
// launcher on the stream); sync[1] is an error word set to 1 when a barrier
// wait passes its 1 s bound (every block then leaves).
constexpr int kMaxRunLayers = 128;
struct DecodeRunArgs {
    const char* base[kMaxRunLayers];  // device address of each layer's blob
    int n_layers, layer0;
    uint64_t off_g_attn, off_wqkv, off_wo, off_g_mlp, off_wg, off_wu, off_wd;  // blob byte offsets
    int H, Hq, Hkv, d, F;
    float eps, theta;
    float *x, *q, *o, *a;            // [H], [Hq d], [Hq d], [F] fp32
    const int32_t* positions;        // [1]: position of the token
    KvView kv;                       // layer field ignored
    float* attn_scratch;             // attention_scratch_floats(scratch_rows, Hq, d, max_ctx, page_tokens)
    int scratch_rows, max_ctx;
    unsigned* sync;                  // [2 + 4 * kMaxRunLayers]: barrier, error word, tile counters
    int skip_block;                  // fault injection: block that skips its first barrier arrival (-1: none)
    uint32_t barrier_limit_us;       // bound of each barrier wait (0: 1 s)
};
bool decode_run_supported(int Hq, int Hkv, int d);
cudaError_t launch_decode_run(const DecodeRunArgs& a, cudaStream_t st);

cudaError_t launch_embed(const uint16_t* embed, const int32_t* tokens, int B, int H, int V, float* x,
                         cudaStream_t st, bool pdl = false);
cudaError_t launch_advance(int32_t* positions, int B, cudaStream_t st, bool pdl = false);
cudaError_t launch_generate(uint16_t* out, uint64_t n, uint64_t first, uint64_t seed, uint32_t tensor_id, int kind,
                            cudaStream_t st);

// Prefill (M tokens at once).  y = RMSNorm(x) * g as a split pair of bf16
// planes [2][M][H]: hi = bf16(y), lo = bf16(y - hi).
cudaError_t launch_rmsnorm_split(const float* x, const uint16_t* g, int M, int H, float eps, uint16_t* y,
                                 cudaStream_t st);
// Prefill projections on the tensor cores (tcgen05, TMA), fused epilogues.
// The activation operand (y, a) is a split pair of bf16 planes [2][M][K] when
// `split` is set (two MMAs per K step), else one bf16 plane [M][K].  The
// SwiGLU output `a` is always written as a split pair [2][M][F].
cudaError_t launch_tc_gemm_qkv_rope(const uint16_t* y, bool split, const uint16_t* wqkv, int M, int H, int Hq,
                                    int Hkv, int d, float theta, const int32_t* positions, const int32_t* row_req,
                                    float* q, KvView kv, cudaStream_t st);
cudaError_t launch_tc_gemm_resid(const uint16_t* a, bool split, const uint16_t* w, int M, int N, int K, float* x,
                                 cudaStream_t st);
cudaError_t launch_tc_gemm_swiglu(const uint16_t* y, bool split, const uint16_t* wg, const uint16_t* wu, int M, int H,
                                  int F, uint16_t* a, cudaStream_t st);
// Lossless packing of bf16 weights for the host link (pack.cu): superblocks of
// kPackWords words become kPackedSb bytes (sign-and-mantissa bytes, exponents
// as codes of one, two or three levels relative to the superblock's largest
// exponent, a record with up to kPackMaxExc exceptions).  A superblock over
// one of the limits (kPackEsc1 level-1 escapes, kPackEsc2 level-2 escapes,
// kPackMaxExc exceptions) is marked unpacked (record byte 1 = 0xff): unpack
// leaves its words untouched and they travel raw.  in / out 16-byte aligned.
constexpr int kPackWords = 1024;
constexpr int kPackedSb = 1440;
constexpr int kPackEsc1 = 352;
constexpr int kPackEsc2 = 80;
constexpr int kPackMaxExc = 5;
// raw_list (may be null): [0] counts the superblocks left unpacked, then their
// indices (first_sb + i), at most raw_cap of them.
cudaError_t launch_pack(const uint16_t* in, uint64_t n_sb, uint8_t* out, uint32_t* raw_list, uint32_t first_sb,
                        uint32_t raw_cap, cudaStream_t st);
cudaError_t launch_unpack(const uint8_t* in, uint64_t n_sb, uint16_t* out, cudaStream_t st);
// two segments in one launch (either may be empty)
cudaError_t launch_unpack2(const uint8_t* in0, uint64_t n0, uint16_t* out0, const uint8_t* in1, uint64_t n1,
                           uint16_t* out1, cudaStream_t st);

// First failure code recorded by a tensor-core GEMM launch (0 = none).
cudaError_t tc_error(int* code);
// Causal prefill attention on the tensor cores (attn_tc.cu).  tiles[i] =
// {first row, rows, request, position of the first row}: a run of at most
// attention_tc_tile_positions(Hq, Hkv) = 128 / (Hq / Hkv) consecutive positions
// of one request, rows of q (fp32 [M, Hq d]); each row attends over its
// request's cached positions 0 .. its own.  o: split pair [2][M][Hq d].
// d = 64 or 128, Hq / Hkv = 1, 2, 4 or 8, page_tokens = 64.
int attention_tc_tile_positions(int Hq, int Hkv);
cudaError_t launch_attention_tc(const float* q, KvView kv, const int4* tiles, int n_tiles, int M, int Hq, int Hkv,
                                int d, uint16_t* o, cudaStream_t st);
cudaError_t attention_tc_error(int* code);
cudaError_t launch_gather_rows(const float* x, const int32_t* rows, int n, int H, float* out, cudaStream_t st);

}  // namespace loip
