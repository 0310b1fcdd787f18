// runtime.cu -- the LOIP runtime on one GPU: device arena and block allocator,
// pinned host weight pool, slot ring on a dedicated copy stream chained to the
// compute stream by CUDA events, paged KV cache, decode step, prefill and
// online re-planning; and the C ABI (include/loip.h).
//
// Loading path (Sec. III-C).  The paper replaces copy-then-compute with one
// reusable loading slot that the runtime refills as soon as the GPU signals,
// through a CUDA event, that it finished the weights in it.  Here the slot is
// a ring of K device slots: the copy of offloaded layer j+K into slot
// (j mod K) waits on slot_free[j mod K] (recorded on the compute stream after
// layer j's kernels) and records slot_full, which layer j+K's kernels wait
// for.  The ring runs across step boundaries, so the first offloaded layers of
// the next step load during the tail of the current one (Fig. 2b, F_N').
// Layer descriptors are computed once (the paper's proxy modules): a slot
// rebinding is a pointer change.
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdio.h>
#include <string.h>
#include <time.h>

#include <algorithm>
#include <chrono>
#include <deque>
#include <string>
#include <thread>
#include <vector>

#include "../../include/loip.h"
#include "disktier.h"
#include "hostpool.h"
#include "internal.h"
#include "plan.h"

using namespace loip;

namespace {

thread_local std::string g_create_error;

// The deadline loop of every host wait: polls query() (cudaSuccess: done,
// cudaErrorNotReady: pending, anything else: failed) until it is not pending
// or timeout_ms of wall time have passed (*timed_out set, returns
// cudaErrorNotReady).  Host code only; the poll is the only device contact.
template <class Q>
cudaError_t poll_until(Q query, uint32_t timeout_ms, bool* timed_out, double* waited_ms) {
    const auto t0 = std::chrono::steady_clock::now();
    auto ms = [&] { return std::chrono::duration<double, std::milli>(std::chrono::steady_clock::now() - t0).count(); };
    *timed_out = false;
    for (;;) {
        const cudaError_t r = query();
        if (r != cudaErrorNotReady) {
            if (waited_ms) *waited_ms = ms();
            return r;
        }
        const double w = ms();
        if (w > (double)timeout_ms) {
            *timed_out = true;
            if (waited_ms) *waited_ms = w;
            return cudaErrorNotReady;
        }
        std::this_thread::yield();
    }
}

constexpr uint64_t kAlign = 256;
inline uint64_t align_up(uint64_t v, uint64_t a = kAlign) { return (v + a - 1) / a * a; }

enum BlockKind { B_FREE = 0, B_LAYER = 1, B_SLOT = 2, B_KV = 3 };

struct Request {
    std::vector<int64_t> pages;  // byte offsets of page groups from the arena base
    int32_t len = 0;             // tokens in the cache
};

struct Fixed {  // offsets inside the fixed region
    uint64_t embed, lm_head, g_final, x, q, o, a, z, logits, attn_scratch, lm_scratch;
    uint64_t tokens, out_tokens, positions, ctx_lens, row_req, page_table, last_rows, dec_pos, run_sync, qk_raw;
    uint64_t px, py, pq, po, pa, ptiles, pack_stage, pack_list;
    uint64_t total;
};

int validate_desc(const loip_model_desc* d) {
    if (!d) return LOIP_ERR_INVALID;
    if (d->n_layers <= 0 || d->hidden <= 0 || d->n_heads <= 0 || d->n_kv_heads <= 0 || d->head_dim <= 0 ||
        d->ffn <= 0 || d->vocab <= 0)
        return LOIP_ERR_INVALID;
    if (d->hidden % 8 || d->ffn % 8 || (d->head_dim != 64 && d->head_dim != 128) || d->n_heads % d->n_kv_heads)
        return LOIP_ERR_INVALID;
    int G = d->n_heads / d->n_kv_heads;
    if (G != 1 && G != 2 && G != 4 && G != 8) return LOIP_ERR_INVALID;
    if (!(d->rms_eps > 0) || !(d->rope_theta > 1) || (d->qk_norm != 0 && d->qk_norm != 1)) return LOIP_ERR_INVALID;
    return LOIP_OK;
}

void layout_of(const loip_model_desc* d, loip_layer_layout_t* o) {
    const uint64_t H = d->hidden, F = d->ffn, qd = (uint64_t)d->n_heads * d->head_dim,
                   kvd = (uint64_t)d->n_kv_heads * d->head_dim;
    uint64_t off = 0;
    o->off_g_attn = off;
    off = align_up(off + H * 2);
    o->off_wqkv = off;
    off = align_up(off + (qd + 2 * kvd) * H * 2);
    o->off_wo = off;
    off = align_up(off + H * qd * 2);
    o->off_g_q = o->off_g_k = off;
    if (d->qk_norm) {
        o->off_g_q = off;
        off = align_up(off + (uint64_t)d->head_dim * 2);
        o->off_g_k = off;
        off = align_up(off + (uint64_t)d->head_dim * 2);
    }
    o->mha_bytes = off;
    o->off_g_mlp = off;
    off = align_up(off + H * 2);
    o->off_wg = off;
    off = align_up(off + F * H * 2);
    o->off_wu = off;
    off = align_up(off + F * H * 2);
    o->off_wd = off;
    off = align_up(off + H * F * 2);
    o->l_size = off;
    o->mlp_bytes = off - o->mha_bytes;
}

loip_config normalized(const loip_config* c) {
    loip_config r = *c;
    if (r.page_tokens <= 0) r.page_tokens = 64;
    if (r.timeout_ms == 0) r.timeout_ms = 600000;
    if (r.max_prefill_tokens <= 0) r.max_prefill_tokens = 512;
    if (!(r.hbm_Bps > 0)) r.hbm_Bps = 6.7e12;
    if (!(r.link_Bps > 0)) r.link_Bps = 2.0e11;
    return r;
}

// Packed streaming (loip_config.pack_stream): not with direct access (kernels
// read the host blobs in place) nor with the SSD tier (its blobs stay raw).
constexpr uint64_t kPackChunkSb = 32768;  // superblocks per staging chunk (47 MB packed)
constexpr uint32_t kPackRawCap = 256;     // superblocks per layer that may travel unpacked
bool packing_enabled(const loip_config* c) {
    return c->pack_stream && c->mode != LOIP_MODE_DIRECT && c->host_budget_bytes == 0;
}
// Chunks in the device staging ring.  In decode the compute stream unpacks
// two landed chunks per launch while the copy engine fills two more, and a
// layer's compute (up to ~0.9 ms for a streamed layer and its resident
// neighbour at the 70B shape, about four chunks' worth of link time) must not
// stall the copies: six chunks.  In a
// prefill pass a chunk is unpacked by a kernel on its own stream, which only
// gets SMs when a compute kernel ends, and the tensor-core GEMMs hold every SM
// for up to a few ms (the gate/up GEMM of 2048 rows at the 70B shape: ~2.1 ms,
// nine chunks' worth of link time): one chunk per 256 prefill rows, at most
// kPackRingMax.
constexpr int kPackRingMax = 8;
int pack_ring_chunks(const loip_config* c) {
    return std::max(6, std::min(kPackRingMax, c->max_prefill_tokens / 256));
}
// superblocks per staging chunk: kPackChunkSb, or the larger block of a small layer
uint64_t pack_chunk_sb(const loip_model_desc* d) {
    loip_layer_layout_t y{};
    layout_of(d, &y);
    const uint64_t big = std::max(y.mha_bytes, y.mlp_bytes) / (2 * kPackWords);
    return std::max<uint64_t>(1, std::min(kPackChunkSb, big));
}

Fixed fixed_layout(const loip_model_desc* d, const loip_config* c) {
    Fixed f{};
    const uint64_t H = d->hidden, V = d->vocab, F = d->ffn, qd = (uint64_t)d->n_heads * d->head_dim;
    const uint64_t B = c->max_batch, Mp = c->max_prefill_tokens;
    const uint64_t rows = std::max<uint64_t>(B, Mp);
    const uint64_t max_pages = (c->max_ctx + c->page_tokens - 1) / c->page_tokens;
    uint64_t off = 0;
    auto take = [&](uint64_t bytes) {
        uint64_t o = off;
        off = align_up(off + bytes);
        return o;
    };
    f.embed = c->embed_on_host ? UINT64_MAX : take(V * H * 2);  // on the host: no device bytes
    f.lm_head = take(V * H * 2);
    f.g_final = take(H * 2);
    f.x = take(B * H * 4);
    f.q = take(B * qd * 4);
    f.o = take(B * qd * 4);
    f.a = take(B * F * 4);
    f.z = take(B * H * 4);
    f.logits = take(B * V * 4);
    f.attn_scratch = take(attention_scratch_floats((int)B, d->n_heads, d->head_dim, c->max_ctx, c->page_tokens) * 4);
    f.lm_scratch = take(lm_head_scratch_bytes((int)B, (int)V));
    f.tokens = take(rows * 4);
    f.out_tokens = take(rows * 4);
    f.positions = take(rows * 4);
    f.ctx_lens = take(rows * 4);
    f.row_req = take(rows * 4);
    f.last_rows = take(B * 4);
    f.dec_pos = take(B * 4);
    f.page_table = take(B * max_pages * 8);
    f.run_sync = take(4 * (2 + 4 * kMaxRunLayers));
    f.qk_raw = d->qk_norm ? take(rows * (uint64_t)(d->n_heads + 2 * d->n_kv_heads) * d->head_dim * 4) : 0;
    // prefill: residual rows fp32; GEMM operands as split pairs of bf16 planes
    f.px = take(Mp * H * 4);
    f.py = take(2 * Mp * H * 2);
    f.pq = take(Mp * qd * 4);
    f.po = take(2 * Mp * qd * 2);
    f.pa = take(2 * Mp * F * 2);
    f.ptiles = take((Mp + (uint64_t)B + 16) * 16);  // tensor-core attention's query tiles (int4 each)
    if (packing_enabled(c)) {  // the staging ring of packed superblocks, the raw-superblock list
        f.pack_stage = take((uint64_t)pack_ring_chunks(c) * pack_chunk_sb(d) * (uint64_t)kPackedSb);
        f.pack_list = take(4 * (kPackRawCap + 1));
    }
    f.total = off;
    return f;
}

}  // namespace

struct loip_ctx {
    loip_model_desc desc{};
    loip_config cfg{};
    loip_layer_layout_t lay{};
    int L = 0, H = 0, Hq = 0, Hkv = 0, d = 0, F = 0, V = 0, qd = 0, kvd = 0;
    char* arena = nullptr;
    uint64_t budget = 0;
    Fixed fx{};
    // blocks (layer-sized)
    uint64_t block_bytes = 0, blocks_off = 0;
    int n_blocks = 0;
    std::vector<int> block_kind, block_owner;
    std::vector<int> layer_block;   // block of each layer holding one or both of its blocks, -1 if none
    std::vector<uint8_t> offloaded;  // 1: the layer streams at least one of its blocks through the slots
    // block granularity: resident blocks of each layer (bit 0 MHA, bit 1 MLP;
    // 3 = whole layer) and their device addresses (nullptr: streamed)
    std::vector<uint8_t> res_mask;
    std::vector<char*> mha_at, mlp_at;
    uint64_t tail_off = 0, tail_used = 0;  // memory after the whole blocks: refined resident blocks
    std::vector<int> slot_block;
    std::vector<int> off_order;     // offloaded layers in order
    // KV
    uint64_t kv_tok_bytes = 0, layer_page_bytes = 0, group_bytes = 0, kv_region_off = 0, kv_region_bytes = 0;
    std::vector<int64_t> free_groups;
    uint64_t kv_groups_total = 0;
    std::vector<Request> reqs;
    int max_pages = 0;
    bool pt_dirty = true;
    // embedding table in mapped pinned host memory (loip_config.embed_on_host)
    HostBuf embed_host;
    // the table the embedding gather reads: the arena's copy, or the device
    // address of the mapped host copy (nullptr until it is allocated)
    const uint16_t* embed_table() {
        if (!cfg.embed_on_host) return fixed_ptr<uint16_t>(fx.embed);
        return static_cast<const uint16_t*>(embed_host.dev);
    }
    int ensure_embed_host() {
        if (!cfg.embed_on_host || embed_host.ptr) return LOIP_OK;
        cudaError_t e = host_buf_alloc((size_t)V * H * 2, &embed_host);
        if (e != cudaSuccess) return fail(LOIP_ERR_OOM, "pinned allocation of the embedding table failed");
        if (!embed_host.dev) {
            host_buf_free(&embed_host);
            return fail(LOIP_ERR_CUDA, "the host embedding table cannot be mapped for the device");
        }
        return LOIP_OK;
    }
    // host pool: blobs of offloaded layers inside pinned huge-page regions
    std::vector<void*> host_layer;
    std::vector<HostBuf> host_regions;
    // SSD tier: streamed layers beyond the host budget live in a file (disk_off[l]
    // >= 0); io_uring reads them one layer ahead, in ring order, into two pinned
    // staging buffers that the copy stream then moves into the slots
    static constexpr int kStages = 4;  // staging buffers: reads run up to three layers ahead
    DiskTier disk;
    std::vector<int64_t> disk_off;
    uint64_t disk_stride = 0;
    HostBuf stage[kStages];
    int stage_layer[kStages] = {-1, -1, -1, -1};  // layer whose read was queued into the buffer
    cudaEvent_t stage_done[kStages] = {};         // last copy out of the buffer
    int32_t* h_stage = nullptr;  // pinned staging for small transfers (last word: layer-run error)
    bool run_launched = false;   // a layer-run kernel has been enqueued (its error word is checked)
    size_t h_stage_ints = 0;
    int64_t* h_pt = nullptr;     // pinned page-table staging
    // streams and events
    cudaStream_t compute = nullptr, copy = nullptr;
    std::vector<cudaEvent_t> slot_full, slot_free;
    cudaEvent_t ev_done = nullptr, ev_step0 = nullptr, ev_step1 = nullptr, ev_reach = nullptr;
    cudaEvent_t ev_stage = nullptr;  // last transfer that read the pinned staging buffers
    bool pos_dirty = true;
    struct CopyEv {
        cudaEvent_t a, b;
        bool ssd;  // out of an SSD-tier staging buffer
        uint64_t bytes;
    };
    std::deque<CopyEv> copy_events;
    // duration and size of the most recent completed layer copies (loip_get_copy_log)
    static constexpr size_t kCopyLog = 8192;
    std::vector<std::pair<float, uint64_t>> copy_log;
    size_t copy_log_next = 0;
    // where the host pool's pages landed: majority NUMA node of each pooled blob (-1: none)
    std::vector<int> pool_node;
    std::vector<cudaEvent_t> event_pool;
    uint64_t copy_seq = 0, compute_seq = 0;
    bool ktiming = false;
    // true when the last operation enqueued on the compute stream is a kernel
    // of the decode chain, so the next kernel may use programmatic launch
    bool chain = false;
    bool pdl() const { return chain && !ktiming; }
    struct KEv {
        int cls;
        cudaEvent_t a, b;
    };
    std::deque<KEv> kernel_events;
    bool weights_loaded = false;
    bool failed = false;
    int prefill_tiles = 0;  // query tiles of the current prefill chunk (tensor-core attention)
    // ---- packed streaming: each streamed layer's two blocks (units) in the host
    // pool as packed superblocks; the copy stream moves them chunk by chunk into
    // a device staging ring (pack_ring_chunks) and the unpack stream expands each chunk
    // into the slot.  Host area of a layer: [unit 0 packed | unit 0 tail | unit 1
    // packed | unit 1 tail | up to kPackRawCap raw superblocks of 2048 bytes].
    struct PackUnit {
        uint64_t off = 0, n_sb = 0, tail = 0;  // blob offset; packed superblocks; raw tail bytes after them
        uint64_t host_off = 0;                  // offset of the unit inside the layer's host area
    };
    struct PackLayer {
        bool on = false;
        std::vector<std::pair<int, uint32_t>> raw;  // (unit, superblock) carried raw, in raw-area order
    };
    bool packing = false;
    uint64_t chunk_sb = 1;  // superblocks per staging chunk
    int ring = 2;           // chunks in the staging ring
    PackUnit pu[2];
    uint64_t pack_area = 0;  // host bytes per packed layer
    std::vector<PackLayer> pk;
    cudaStream_t unpack_st = nullptr;
    cudaEvent_t chunk_ready[kPackRingMax] = {}, chunk_free[kPackRingMax] = {};
    // The pieces of packed layer copies wait in pack_fifo, in ring order, until
    // pump() enqueues them.  A packed chunk takes staging entry seq % ring; the
    // pump hands out sequence number seq only once the unpack of seq - ring, the
    // entry's previous chunk, has been enqueued (so that every wait on
    // chunk_free / chunk_ready refers to the right record).  A layer's pieces are
    // its chunks, then one end job: the raw tails and raw superblocks, copied
    // straight into the slot after the slot is free.
    //
    // Where a chunk is unpacked is fixed when its layer's copy is issued: by a
    // kernel on the unpack stream (prefill passes, explicit stream_layer calls,
    // naive mode; slot_full is recorded there), or inline, on the compute stream
    // right before the layer computes (decode passes: the step waits on the link
    // anyway, and an unpack on its own stream would queue behind the decode
    // GEMVs, whose persistent blocks hold every SM).
    struct PackJob {
        int layer, slot, unit;  // unit 0 / 1: a chunk of that block; 2: the end job
        uint64_t c0, n;         // chunk: first superblock and count
        bool inl;               // unpacked inline by the compute stream
        bool first;             // the layer's first piece (copy timing starts)
        cudaStream_t cs;        // copy stream
    };
    struct InlineChunk {
        uint64_t seq;
        int unit;
        uint64_t c0, n;
    };
    std::deque<PackJob> pack_fifo;
    uint64_t ring_next = 0, ring_done = 0;  // sequence numbers handed out; below ring_done: unpack enqueued
    std::deque<bool> ring_unpacked;         // seq in [ring_done, ring_next): unpack enqueued
    bool inline_unpack = false;             // copies issued now unpack inline (decode passes)
    // per slot: the layer it is being filled with unpacks inline; its pumped
    // chunks awaiting their unpack; chunks not yet unpack-enqueued; end job pumped
    std::vector<uint8_t> slot_inline, raw_pumped;
    std::vector<std::deque<InlineChunk>> inl_chunks;
    std::vector<int> inl_left;
    std::vector<cudaEvent_t> raw_done;      // per slot: the end job's copies landed (copy stream)
    cudaEvent_t pump_e0 = nullptr;          // copy timing of the layer being pumped
    uint64_t pump_bytes = 0;
    bool packed(int l) const { return packing && l < (int)pk.size() && pk[l].on; }
    uint64_t host_bytes(int l) const { return packed(l) ? pack_area : lay.l_size; }
    void init_packing() {
        packing = packing_enabled(&cfg);
        pk.assign(L, PackLayer{});
        if (!packing) return;
        chunk_sb = pack_chunk_sb(&desc);
        ring = pack_ring_chunks(&cfg);
        const uint64_t offs[2] = {0, lay.mha_bytes}, sizes[2] = {lay.mha_bytes, lay.mlp_bytes};
        uint64_t at = 0;
        for (int u = 0; u < 2; ++u) {
            pu[u].off = offs[u];
            pu[u].n_sb = sizes[u] / (2 * kPackWords);
            pu[u].tail = sizes[u] - pu[u].n_sb * 2 * kPackWords;
            at = (at + 4095) / 4096 * 4096;  // each unit's packed data on a 4 KB boundary
            pu[u].host_off = at;
            at += pu[u].n_sb * kPackedSb + pu[u].tail;
        }
        pack_area = at + (uint64_t)kPackRawCap * 2 * kPackWords;
    }
    // Packs layer l's blob (device, blob layout at dev) into its host area.
    // Returns LOIP_OK with pk[l].on set, or LOIP_OK with it cleared when more
    // than kPackRawCap superblocks would travel raw (the layer then streams raw).
    int pack_layer(int l, const char* dev) {
        char* host = static_cast<char*>(host_layer[l]);
        uint8_t* stage = fixed_ptr<uint8_t>(fx.pack_stage);
        uint32_t* list = fixed_ptr<uint32_t>(fx.pack_list);
        cudaStream_t s = compute;
        std::vector<std::pair<int, uint32_t>> raw;
        for (int u = 0; u < 2; ++u) {
            const PackUnit& U = pu[u];
            cudaError_t e = cudaMemsetAsync(list, 0, 4, s);
            for (uint64_t c0 = 0; c0 < U.n_sb && e == cudaSuccess; c0 += chunk_sb) {
                const uint64_t n = std::min<uint64_t>(chunk_sb, U.n_sb - c0);
                uint8_t* st_c = stage + ((c0 / chunk_sb) & 1) * chunk_sb * kPackedSb;
                e = launch_pack(reinterpret_cast<const uint16_t*>(dev + U.off) + c0 * kPackWords, n, st_c, list,
                                (uint32_t)c0, kPackRawCap, s);
                if (e == cudaSuccess)
                    e = cudaMemcpyAsync(host + U.host_off + c0 * kPackedSb, st_c, n * kPackedSb,
                                        cudaMemcpyDeviceToHost, s);
            }
            if (e == cudaSuccess && U.tail)
                e = cudaMemcpyAsync(host + U.host_off + U.n_sb * kPackedSb, dev + U.off + U.n_sb * 2 * kPackWords,
                                    U.tail, cudaMemcpyDeviceToHost, s);
            uint32_t h_list[1 + kPackRawCap];
            if (e == cudaSuccess) e = cudaMemcpyAsync(h_list, list, sizeof h_list, cudaMemcpyDeviceToHost, s);
            if (e == cudaSuccess) e = cudaStreamSynchronize(s);
            if (e != cudaSuccess) return cuda_fail(e, "weight packing");
            if (h_list[0] > kPackRawCap || raw.size() + h_list[0] > kPackRawCap) {
                pk[l].on = false;
                return LOIP_OK;
            }
            std::vector<uint32_t> idx(h_list + 1, h_list + 1 + h_list[0]);
            std::sort(idx.begin(), idx.end());
            for (uint32_t i : idx) raw.push_back({u, i});
        }
        // the raw superblocks' own bytes, after the units
        char* raw_area = host + pu[1].host_off + pu[1].n_sb * kPackedSb + pu[1].tail;
        for (size_t j = 0; j < raw.size(); ++j) {
            cudaError_t e = cudaMemcpy(raw_area + j * 2 * kPackWords,
                                       dev + pu[raw[j].first].off + (uint64_t)raw[j].second * 2 * kPackWords,
                                       2 * kPackWords, cudaMemcpyDeviceToHost);
            if (e != cudaSuccess) return cuda_fail(e, "weight packing");
        }
        pk[l].raw = std::move(raw);
        pk[l].on = true;
        return LOIP_OK;
    }
    // Stores layer l (device blob at dev) in the host pool packed; when it cannot
    // be packed (too many raw superblocks) it gets a raw region of its own.
    int store_packed(int l, const char* dev) {
        int rc = pack_layer(l, dev);
        if (rc || pk[l].on) return rc;
        HostBuf hb;
        if (host_buf_alloc(lay.l_size, &hb) != cudaSuccess) return fail(LOIP_ERR_OOM, "pinned host allocation failed");
        host_regions.push_back(hb);
        host_layer[l] = hb.ptr;
        cudaError_t e = cudaMemcpy(hb.ptr, dev, lay.l_size, cudaMemcpyDeviceToHost);
        return e == cudaSuccess ? LOIP_OK : cuda_fail(e, "layer copy to the host pool");
    }
    // Queues the pieces of packed layer l (streamed units only) for slot `slot`
    // and pumps what the ring allows.
    int queue_packed(int l, int slot, cudaStream_t cs, bool inl) {
        bool first = true;
        int chunks = 0;
        uint64_t bytes = 0;  // what the layer's copies will move over the link
        for (int u = 0; u < 2; ++u) {
            if (res_mask[l] & (1 << u)) continue;  // this block is resident
            bytes += pu[u].n_sb * kPackedSb + pu[u].tail;
            for (const auto& r : pk[l].raw) bytes += r.first == u ? 2 * kPackWords : 0;
            // chunks of about equal size, at most chunk_sb superblocks (no short
            // last chunk), a multiple of 128 superblocks so that each copy starts
            // on a 4 KB boundary of the host area (the copy engine read
            // 32-byte-aligned chunks ~4% slower)
            const uint64_t nc = (pu[u].n_sb + chunk_sb - 1) / chunk_sb;
            const uint64_t per = nc ? std::min(chunk_sb, ((pu[u].n_sb + nc - 1) / nc + 127) / 128 * 128) : 1;
            for (uint64_t c0 = 0; c0 < pu[u].n_sb; c0 += per) {
                pack_fifo.push_back({l, slot, u, c0, std::min<uint64_t>(per, pu[u].n_sb - c0), inl, first, cs});
                first = false;
                ++chunks;
            }
        }
        pack_fifo.push_back({l, slot, 2, 0, 0, inl, first, cs});
        slot_inline[slot] = inl;
        inl_left[slot] = inl ? chunks : 0;
        raw_pumped[slot] = 0;
        st.h2d_weight_bytes += bytes;  // counted when issued, like raw layer copies
        return pump();
    }
    void mark_unpacked(uint64_t seq) {
        ring_unpacked[seq - ring_done] = true;
        while (!ring_unpacked.empty() && ring_unpacked.front()) {
            ring_unpacked.pop_front();
            ++ring_done;
        }
    }
    // Unpack of one staged chunk (or two: b != nullptr, one launch) into the
    // slot, on stream s, after their copies landed.
    cudaError_t enqueue_unpack(int slot, const InlineChunk& a, const InlineChunk* b, cudaStream_t s) {
        const InlineChunk* c[2] = {&a, b};
        const uint8_t* in[2] = {nullptr, nullptr};
        uint16_t* out[2] = {nullptr, nullptr};
        uint64_t n[2] = {0, 0};
        cudaError_t e = cudaSuccess;
        for (int i = 0; i < 2 && c[i] && e == cudaSuccess; ++i) {
            const int g = (int)(c[i]->seq % (uint64_t)ring);
            in[i] = fixed_ptr<uint8_t>(fx.pack_stage) + (uint64_t)g * chunk_sb * kPackedSb;
            out[i] = reinterpret_cast<uint16_t*>(slot_ptr(slot) + pu[c[i]->unit].off) + c[i]->c0 * kPackWords;
            n[i] = c[i]->n;
            e = cudaStreamWaitEvent(s, chunk_ready[g], 0);
        }
        if (e == cudaSuccess)
            e = timed(13, s, [&] { return launch_unpack2(in[0], n[0], out[0], in[1], n[1], out[1], s); });
        for (int i = 0; i < 2 && c[i]; ++i) {
            if (e == cudaSuccess) e = cudaEventRecord(chunk_free[c[i]->seq % (uint64_t)ring], s);
            mark_unpacked(c[i]->seq);
        }
        st.unpack_launches += 1;
        st.unpack_bytes += (n[0] + n[1]) * (uint64_t)(kPackedSb + 2 * kPackWords);
        return e;
    }
    // Enqueues queued pieces in order while the staging ring has room.
    int pump() {
        cudaError_t e = cudaSuccess;
        while (!pack_fifo.empty() && e == cudaSuccess) {
            const PackJob j = pack_fifo.front();
            const char* host = static_cast<const char*>(host_layer[j.layer]);
            char* dst = slot_ptr(j.slot);
            if (j.unit < 2 && ring_next >= ring_done + (uint64_t)ring) break;  // entry still in use
            if (j.first) {
                pump_e0 = take_event();
                pump_bytes = 0;
                e = cudaEventRecord(pump_e0, j.cs);
                if (e != cudaSuccess) break;
                if (!j.inl) e = cudaStreamWaitEvent(unpack_st, slot_free[j.slot], 0);  // unpacks write the slot
                if (e != cudaSuccess) break;
            }
            if (j.unit < 2) {
                const PackUnit& U = pu[j.unit];
                const uint64_t seq = ring_next++;
                ring_unpacked.push_back(false);
                const int g = (int)(seq % (uint64_t)ring);
                uint8_t* st_c = fixed_ptr<uint8_t>(fx.pack_stage) + (uint64_t)g * chunk_sb * kPackedSb;
                e = cudaStreamWaitEvent(j.cs, chunk_free[g], 0);  // the entry's previous chunk has been unpacked
                if (e == cudaSuccess)
                    e = cudaMemcpyAsync(st_c, host + U.host_off + j.c0 * kPackedSb, j.n * kPackedSb,
                                        cudaMemcpyHostToDevice, j.cs);
                if (e == cudaSuccess) e = cudaEventRecord(chunk_ready[g], j.cs);
                pump_bytes += j.n * kPackedSb;
                if (e == cudaSuccess) {
                    const InlineChunk c{seq, j.unit, j.c0, j.n};
                    if (j.inl)
                        inl_chunks[j.slot].push_back(c);
                    else
                        e = enqueue_unpack(j.slot, c, nullptr, unpack_st);
                }
            } else {  // end job: raw tails and raw superblocks into the slot once it is free
                const char* raw_area = host + pu[1].host_off + pu[1].n_sb * kPackedSb + pu[1].tail;
                e = cudaStreamWaitEvent(j.cs, slot_free[j.slot], 0);
                for (int u = 0; u < 2 && e == cudaSuccess; ++u) {
                    if (res_mask[j.layer] & (1 << u)) continue;
                    const PackUnit& U = pu[u];
                    if (U.tail) {
                        e = cudaMemcpyAsync(dst + U.off + U.n_sb * 2 * kPackWords,
                                            host + U.host_off + U.n_sb * kPackedSb, U.tail, cudaMemcpyHostToDevice,
                                            j.cs);
                        pump_bytes += U.tail;
                    }
                    for (size_t r = 0; r < pk[j.layer].raw.size() && e == cudaSuccess; ++r) {
                        if (pk[j.layer].raw[r].first != u) continue;
                        e = cudaMemcpyAsync(dst + U.off + (uint64_t)pk[j.layer].raw[r].second * 2 * kPackWords,
                                            raw_area + r * 2 * kPackWords, 2 * kPackWords, cudaMemcpyHostToDevice,
                                            j.cs);
                        pump_bytes += 2 * kPackWords;
                    }
                }
                cudaEvent_t e1 = take_event();
                if (e == cudaSuccess) e = cudaEventRecord(e1, j.cs);
                if (e == cudaSuccess) {
                    copy_events.push_back({pump_e0, e1, false, pump_bytes});
                    if (j.inl) {
                        e = cudaEventRecord(raw_done[j.slot], j.cs);
                    } else {  // the slot is full once every chunk is unpacked and the raw copies landed
                        e = cudaStreamWaitEvent(unpack_st, e1, 0);
                        if (e == cudaSuccess) e = cudaEventRecord(slot_full[j.slot], unpack_st);
                    }
                }
                raw_pumped[j.slot] = 1;
            }
            pack_fifo.pop_front();
        }
        if (e != cudaSuccess) return cuda_fail(e, "packed layer copy");
        return LOIP_OK;
    }
    // Before a packed layer in `slot` computes on stream s: its inline unpacks
    // (after their chunks landed; two chunks per launch when the ring leaves the
    // copy engine four more meanwhile) and the wait for its raw pieces, or the
    // wait for slot_full.
    int wait_packed_slot(int slot, cudaStream_t s) {
        cudaError_t e = cudaSuccess;
        const size_t per_launch = ring >= 6 ? 2 : 1;
        while (inl_left[slot] > 0) {
            const size_t want = std::min<size_t>(per_launch, (size_t)inl_left[slot]);
            while (inl_chunks[slot].size() < want) {
                const size_t have = inl_chunks[slot].size();
                int rc = pump();
                if (rc) return rc;
                if (inl_chunks[slot].size() == have) return fail(LOIP_ERR_STATE, "packed copy queue out of order");
            }
            const InlineChunk c = inl_chunks[slot].front();
            inl_chunks[slot].pop_front();
            InlineChunk c2{};
            const bool two = want == 2;
            if (two) {
                c2 = inl_chunks[slot].front();
                inl_chunks[slot].pop_front();
            }
            inl_left[slot] -= two ? 2 : 1;
            e = enqueue_unpack(slot, c, two ? &c2 : nullptr, s);
            if (e != cudaSuccess) return cuda_fail(e, "unpack kernel");
            chain = false;
            int rc = pump();  // the freed entries let the next chunks' copies go
            if (rc) return rc;
        }
        while (!raw_pumped[slot]) {
            const size_t before = pack_fifo.size();
            int rc = pump();
            if (rc) return rc;
            if (pack_fifo.size() == before) return fail(LOIP_ERR_STATE, "packed copy queue stalled");
        }
        e = cudaStreamWaitEvent(s, slot_inline[slot] ? raw_done[slot] : slot_full[slot], 0);
        if (e != cudaSuccess) return cuda_fail(e, "compute wait");
        return LOIP_OK;
    }
    // Hands every inline unpack still pending to the unpack stream (before a
    // prefill pass or an explicit stream_layer call), so that those layers'
    // slots get slot_full without the compute stream's help.
    int flush_inline() {
        if (!packing) return LOIP_OK;
        for (auto& j : pack_fifo) j.inl = false;
        for (int s = 0; s < cfg.n_slots; ++s) {
            if (!slot_inline[s]) continue;
            cudaError_t e = cudaStreamWaitEvent(unpack_st, slot_free[s], 0);
            while (e == cudaSuccess && !inl_chunks[s].empty()) {
                const InlineChunk c = inl_chunks[s].front();
                inl_chunks[s].pop_front();
                e = enqueue_unpack(s, c, nullptr, unpack_st);
            }
            if (e == cudaSuccess && raw_pumped[s]) {  // end job already enqueued: slot_full after it
                e = cudaStreamWaitEvent(unpack_st, raw_done[s], 0);
                if (e == cudaSuccess) e = cudaEventRecord(slot_full[s], unpack_st);
            }
            if (e != cudaSuccess) return cuda_fail(e, "unpack kernel");
            slot_inline[s] = 0;
            inl_left[s] = 0;
        }
        return pump();
    }
    // Forgets queued and staged pieces (the streams are idle: after sync_all).
    void reset_pack_queue() {
        pack_fifo.clear();
        ring_done = ring_next;
        ring_unpacked.clear();
        for (int s = 0; s < (int)slot_inline.size(); ++s) {
            slot_inline[s] = 0;
            raw_pumped[s] = 1;
            inl_left[s] = 0;
            inl_chunks[s].clear();
        }
    }
    // fault injection (loip_inject_fault): one armed fault, fired once
    int fault_kind = 0, fault_arg = 0;
    bool take_fault(int kind) {
        if (fault_kind != kind) return false;
        fault_kind = 0;
        return true;
    }
    int active_batch = 0;
    loip_stats st{};
    std::string err;

    // ---------------------------------------------------------------------
    int fail(int code, const std::string& m) {
        err = m;
        return code;
    }
    int cuda_fail(cudaError_t e, const char* what) {
        err = std::string(what) + ": " + cudaGetErrorString(e);
        if (e != cudaErrorNotReady) failed = true;
        cudaGetLastError();  // a non-sticky error must not surface again in a later, unrelated launch
        return LOIP_ERR_CUDA;
    }
    template <class T>
    T* fixed_ptr(uint64_t off) {
        return reinterpret_cast<T*>(arena + off);
    }
    char* block_ptr(int b) { return arena + blocks_off + (uint64_t)b * block_bytes; }
    char* slot_ptr(int k) { return block_ptr(slot_block[k]); }
    int n_slots_used() const { return off_order.empty() ? 0 : cfg.n_slots; }

    cudaEvent_t take_event() {
        if (!event_pool.empty()) {
            cudaEvent_t e = event_pool.back();
            event_pool.pop_back();
            return e;
        }
        cudaEvent_t e = nullptr;
        cudaEventCreate(&e);
        return e;
    }

    int wait_event(cudaEvent_t e) {
        // an injected wait fault reports the event as pending until the deadline
        const bool stuck = take_fault(LOIP_FAULT_WAIT);
        bool timed_out = false;
        cudaError_t r = poll_until([&] { return stuck ? cudaErrorNotReady : cudaEventQuery(e); }, cfg.timeout_ms,
                                   &timed_out, nullptr);
        if (timed_out) {
            failed = true;
            return fail(LOIP_ERR_TIMEOUT, "timed out waiting for the device");
        }
        if (r != cudaSuccess) return cuda_fail(r, "device work failed");
        return LOIP_OK;
    }

    // After a host sync point: a layer-run kernel whose grid barrier timed out
    // left its error word set; the context cannot continue.
    int check_run_error() {
        if (!run_launched) return LOIP_OK;
        if (h_stage[h_stage_ints - 1] != 0) {
            failed = true;
            return fail(LOIP_ERR_TIMEOUT, "a grid barrier of the persistent layer-run kernel timed out");
        }
        return LOIP_OK;
    }

    int sync_all() {
        cudaError_t e = cudaEventRecord(ev_done, copy);
        if (e != cudaSuccess) return cuda_fail(e, "event record");
        int r = wait_event(ev_done);
        if (r) return r;
        if (unpack_st) {
            e = cudaEventRecord(ev_done, unpack_st);
            if (e != cudaSuccess) return cuda_fail(e, "event record");
            r = wait_event(ev_done);
            if (r) return r;
        }
        e = cudaEventRecord(ev_done, compute);
        if (e != cudaSuccess) return cuda_fail(e, "event record");
        return wait_event(ev_done);
    }

    // Blob-relative bases of layer l's MHA and MLP blocks: base + lay.off_x is
    // part x, whether the block is resident (at its own address) or streamed
    // into `slot` (the slot holds the blob layout).
    const uint16_t* mha_base(int l, int slot) {
        return reinterpret_cast<const uint16_t*>(mha_at[l] ? mha_at[l] : slot_ptr(slot));
    }
    const uint16_t* mlp_base(int l, int slot) {
        return reinterpret_cast<const uint16_t*>(mlp_at[l] ? mlp_at[l] - lay.mha_bytes : slot_ptr(slot));
    }
    // bytes layer l streams per pass
    uint64_t stream_bytes(int l) const {  // bytes a step moves over the link for layer l
        if (packed(l)) {
            uint64_t b = 0;
            for (int u = 0; u < 2; ++u)
                if (!(res_mask[l] & (1 << u))) b += pu[u].n_sb * kPackedSb + pu[u].tail;
            for (const auto& r : pk[l].raw)
                if (!(res_mask[l] & (1 << r.first))) b += 2 * kPackWords;
            return b;
        }
        return ((res_mask[l] & 1) ? 0 : lay.mha_bytes) + ((res_mask[l] & 2) ? 0 : lay.mlp_bytes);
    }
    void set_resident_block(int l, int b) {  // whole layer in block b
        layer_block[l] = b;
        res_mask[l] = 3;
        mha_at[l] = block_ptr(b);
        mlp_at[l] = block_ptr(b) + lay.mha_bytes;
        offloaded[l] = 0;
    }

    KvView kv_view(int layer, const int64_t* pt) {
        KvView v;
        v.base = arena;
        v.page_offsets = pt;
        v.max_pages = max_pages;
        v.page_tokens = cfg.page_tokens;
        v.layer = layer;
        v.layer_page_bytes = layer_page_bytes;
        return v;
    }

    // ---- block and KV allocation -----------------------------------------
    int take_free_block() {
        for (int b = 0; b < n_blocks; ++b)
            if (block_kind[b] == B_FREE) return b;
        return -1;
    }

    // page groups from a freed range [ptr, ptr + bytes) of the arena (256-aligned)
    void carve_kv(const char* ptr, uint64_t bytes) {
        const uint64_t off = (uint64_t)(ptr - arena);
        const uint64_t n = bytes / group_bytes;
        for (uint64_t i = 0; i < n; ++i) free_groups.push_back((int64_t)(off + i * group_bytes));
        kv_groups_total += n;
    }

    int grow_kv() {  // converts one free block into page groups
        int b = take_free_block();
        if (b < 0) return -1;
        block_kind[b] = B_KV;
        uint64_t n = block_bytes / group_bytes;
        for (uint64_t i = 0; i < n; ++i)
            free_groups.push_back((int64_t)(blocks_off + (uint64_t)b * block_bytes + i * group_bytes));
        kv_groups_total += n;
        return b;
    }

    int ensure_pages(int req, int tokens) {
        Request& r = reqs[req];
        int need = (tokens + cfg.page_tokens - 1) / cfg.page_tokens;
        if (need > max_pages) return fail(LOIP_ERR_INVALID, "context longer than max_ctx");
        while ((int)r.pages.size() < need) {
            if (free_groups.empty()) {
                if (grow_kv() < 0) {
                    int rc = demote_for_kv();  // frees a block, or carves groups from offloaded blocks
                    if (rc) return rc;
                    if (free_groups.empty() && grow_kv() < 0) return fail(LOIP_ERR_OOM, "no block for the KV cache");
                }
            }
            r.pages.push_back(free_groups.back());
            free_groups.pop_back();
            pt_dirty = true;
        }
        return LOIP_OK;
    }

    void release_pages(int req) {
        for (int64_t g : reqs[req].pages) free_groups.push_back(g);
        reqs[req].pages.clear();
        reqs[req].len = 0;
        pt_dirty = true;
    }

    int upload_page_table(cudaStream_t s) {
        if (!pt_dirty) return LOIP_OK;
        int rc = wait_event(ev_stage);  // a previous upload may still read the staging buffer
        if (rc) return rc;
        for (int b = 0; b < cfg.max_batch; ++b)
            for (int i = 0; i < max_pages; ++i)
                h_pt[(size_t)b * max_pages + i] = i < (int)reqs[b].pages.size() ? reqs[b].pages[i] : 0;
        cudaError_t e = cudaMemcpyAsync(arena + fx.page_table, h_pt, (size_t)cfg.max_batch * max_pages * 8,
                                        cudaMemcpyHostToDevice, s);
        if (e != cudaSuccess) return cuda_fail(e, "page table upload");
        cudaEventRecord(ev_stage, s);
        pt_dirty = false;
        return LOIP_OK;
    }

    int upload_positions(int B, cudaStream_t s) {
        if (!pos_dirty) return LOIP_OK;
        int rc = wait_event(ev_stage);
        if (rc) return rc;
        int32_t* hp = h_stage + 2 * (h_stage_ints / 4);
        for (int b = 0; b < B; ++b) hp[b] = reqs[b].len;
        cudaError_t e = cudaMemcpyAsync(arena + fx.dec_pos, hp, (size_t)B * 4, cudaMemcpyHostToDevice, s);
        if (e != cudaSuccess) return cuda_fail(e, "positions upload");
        cudaEventRecord(ev_stage, s);
        pos_dirty = false;
        return LOIP_OK;
    }

    // ---- SSD tier -------------------------------------------------------------
    // Queues the read of disk layer l into staging buffer b once the buffer's
    // previous copy to a slot has finished (bounded wait).
    // a failed SSD-tier wait: out of time, or an I/O error
    int disk_fail(const std::string& err) { return fail(disk.timed_out() ? LOIP_ERR_TIMEOUT : LOIP_ERR_STATE, err); }

    int queue_read(int l, int b) {
        const auto t0 = std::chrono::steady_clock::now();
        int rc = wait_event(stage_done[b]);
        if (rc) return rc;
        st.ssd_stage_wait_ms += std::chrono::duration<double, std::milli>(std::chrono::steady_clock::now() - t0).count();
        std::string err;
        if (!disk.submit_read((uint64_t)disk_off[l], stage[b].ptr, disk_stride, b, &err))
            return fail(LOIP_ERR_STATE, err);
        stage_layer[b] = l;
        st.ssd_read_bytes += disk_stride;
        return LOIP_OK;
    }
    // The staging buffer holding disk layer l, its read complete.
    int staged_blob(int l, int* b_out) {
        int b = -1;
        for (int i = 0; i < kStages && b < 0; ++i)
            if (stage_layer[i] == l) b = i;
        if (b < 0) {  // not read ahead (ring restart): read it now, into a free buffer if there is one
            for (int i = 0; i < kStages && b < 0; ++i)
                if (stage_layer[i] < 0) b = i;
            if (b < 0) {
                b = kStages - 1;
                std::string err;
                if (!disk.wait(b, cfg.timeout_ms, &err)) return disk_fail(err);
            }
            int rc = queue_read(l, b);
            if (rc) return rc;
        }
        std::string err;
        const auto t0 = std::chrono::steady_clock::now();
        if (!disk.wait(b, cfg.timeout_ms, &err)) return disk_fail(err);
        st.ssd_wait_ms += std::chrono::duration<double, std::milli>(std::chrono::steady_clock::now() - t0).count();
        *b_out = b;
        return LOIP_OK;
    }
    // After the copy of disk layer l: queue the reads of the next disk layers in
    // ring order into the free staging buffers (they overlap the copies and
    // compute in between).
    int read_ahead(int l) {
        const int m = (int)off_order.size();
        int pos = 0;
        while (pos < m && off_order[pos] != l) ++pos;
        for (int k = 1; k < m; ++k) {
            const int nl = off_order[(pos + k) % m];
            if (disk_off[nl] < 0) continue;
            bool queued = false;
            int b = -1;
            for (int i = 0; i < kStages; ++i) {
                queued |= stage_layer[i] == nl;
                if (b < 0 && stage_layer[i] < 0) b = i;
            }
            if (queued) continue;
            if (b < 0) return LOIP_OK;  // every buffer holds a pending read
            int rc = queue_read(nl, b);
            if (rc) return rc;
        }
        return LOIP_OK;
    }
    // Writes layer l's blob (in device memory at src) to the SSD tier through
    // staging buffer 0.
    int write_disk_blob(int l, const char* src, cudaMemcpyKind kind) {
        int rc = wait_event(stage_done[0]);
        if (rc) return rc;
        if (stage_layer[0] >= 0) {
            std::string err;
            if (!disk.wait(0, cfg.timeout_ms, &err)) return disk_fail(err);
            stage_layer[0] = -1;
        }
        cudaError_t e = cudaMemcpy(stage[0].ptr, src, lay.l_size, kind);
        if (e != cudaSuccess) return cuda_fail(e, "SSD-tier staging copy");
        std::string err;
        if (!disk.write((uint64_t)disk_off[l], stage[0].ptr, disk_stride, &err)) return fail(LOIP_ERR_STATE, err);
        return LOIP_OK;
    }

    // ---- streaming ------------------------------------------------------------
    int enqueue_copy(int layer, int slot, cudaStream_t cs, bool inl = false) {
        if (take_fault(LOIP_FAULT_COPY))  // as if the copy call had failed; nothing is enqueued
            return cuda_fail(cudaErrorInvalidValue, "layer copy (injected fault)");
        if (packed(layer)) return queue_packed(layer, slot, cs, inl);
        cudaError_t e = cudaStreamWaitEvent(cs, slot_free[slot], 0);
        if (e != cudaSuccess) return cuda_fail(e, "copy wait");
        const char* src = static_cast<const char*>(host_layer[layer]);
        int sb = -1;
        if (disk_off[layer] >= 0) {  // SSD tier: the staged copy of the blob
            int rc = staged_blob(layer, &sb);
            if (rc) return rc;
            src = static_cast<const char*>(stage[sb].ptr);
        }
        cudaEvent_t e0 = take_event(), e1 = take_event();
        cudaEventRecord(e0, cs);
        // the blocks the layer streams, at their blob offsets
        const uint64_t off0 = (res_mask[layer] & 1) ? lay.mha_bytes : 0;
        const uint64_t off1 = (res_mask[layer] & 2) ? lay.mha_bytes : lay.l_size;
        e = cudaMemcpyAsync(slot_ptr(slot) + off0, src + off0, off1 - off0, cudaMemcpyHostToDevice, cs);
        if (e != cudaSuccess) return cuda_fail(e, "layer copy");
        if (sb >= 0) {
            cudaEventRecord(stage_done[sb], cs);
            stage_layer[sb] = -1;
            int rc = read_ahead(layer);
            if (rc) return rc;
        }
        cudaEventRecord(e1, cs);
        copy_events.push_back({e0, e1, sb >= 0, off1 - off0});
        e = cudaEventRecord(slot_full[slot], cs);
        if (e != cudaSuccess) return cuda_fail(e, "slot event");
        st.h2d_weight_bytes += stream_bytes(layer);
        return LOIP_OK;
    }

    int issue_next_copy() {  // ring order over offloaded layers, across steps
        const int m = (int)off_order.size();
        int rc = enqueue_copy(off_order[copy_seq % m], (int)(copy_seq % cfg.n_slots), copy, inline_unpack);
        if (rc) return rc;
        ++copy_seq;
        return LOIP_OK;
    }

    int prime_slots() {  // the streams are idle (callers synchronise first)
        copy_seq = compute_seq = 0;
        if (packing) reset_pack_queue();
        if (off_order.empty() || cfg.mode == LOIP_MODE_NAIVE) return LOIP_OK;
        for (int k = 0; k < cfg.n_slots; ++k) {
            int rc = issue_next_copy();
            if (rc) return rc;
        }
        return LOIP_OK;
    }

    void rebuild_order() {
        off_order.clear();
        for (int l = 0; l < L; ++l)
            if (offloaded[l]) off_order.push_back(l);
    }

    // ---- kernel timing ------------------------------------------------------
    template <class Fn>
    cudaError_t timed(int cls, cudaStream_t s, Fn&& fn) {
        if (!ktiming) return fn();
        cudaEvent_t a = take_event(), b = take_event();
        cudaEventRecord(a, s);
        chain = false;
        cudaError_t e = fn();
        cudaEventRecord(b, s);
        chain = false;
        kernel_events.push_back({cls, a, b});
        return e;
    }
    void collect_kernel_times() {
        while (!kernel_events.empty()) {
            KEv k = kernel_events.front();
            if (cudaEventQuery(k.b) != cudaSuccess) break;
            float ms = 0;
            cudaEventElapsedTime(&ms, k.a, k.b);
            st.kernel_ms[k.cls] += ms;
            st.kernel_launches[k.cls] += 1;
            event_pool.push_back(k.a);
            event_pool.push_back(k.b);
            kernel_events.pop_front();
        }
    }

    // ---- one decoder layer ---------------------------------------------------
    // Decode-time layer on rows 0..B-1 of the fixed activations.
    int decode_layer(int l, int B, const int32_t* pos_dev, cudaStream_t s, int slot) {
        return decode_layer_w(l, B, pos_dev, s, mha_base(l, slot), mlp_base(l, slot), false, false);
    }

    // Device address of offloaded layer l's host blob (mapped pinned memory).
    const uint16_t* host_direct(int l) {
        const char* h = static_cast<const char*>(host_layer[l]);
        if (!h) return nullptr;
        for (const HostBuf& r : host_regions) {
            const char* p = static_cast<const char*>(r.ptr);
            if (r.dev && h >= p && h + lay.l_size <= p + r.bytes)
                return reinterpret_cast<const uint16_t*>(static_cast<const char*>(r.dev) + (h - p));
        }
        return nullptr;
    }

    // Decode over every layer with the offloaded ones read in place from host
    // memory: no slots, no copy stream.
    int run_layers_direct(int B, const int32_t* pos_dev, cudaStream_t s) {
        for (int l = 0; l < L; ++l) {
            if (res_mask[l] == 3 && fuse_runs(B)) {
                int e = l;
                while (e < L && res_mask[e] == 3) ++e;
                int rc = decode_run(l, e, pos_dev, s);
                if (rc) return rc;
                l = e - 1;
                continue;
            }
            const bool ha = !(res_mask[l] & 1), hm = !(res_mask[l] & 2);
            const uint16_t* hw = (ha || hm) ? host_direct(l) : nullptr;
            if ((ha || hm) && !hw) return fail(LOIP_ERR_STATE, "offloaded layer has no device-mapped host copy");
            const uint16_t* wa = ha ? hw : mha_base(l, -1);
            const uint16_t* wm = hm ? hw : mlp_base(l, -1);
            int rc = decode_layer_w(l, B, pos_dev, s, wa, wm, ha, hm);
            if (rc) return rc;
        }
        return LOIP_OK;
    }

    // wa, wm: blob-relative bases of the MHA and MLP blocks (mha_base, mlp_base);
    // host_a, host_m: that block is read in place from mapped host memory
    int decode_layer_w(int l, int B, const int32_t* pos_dev, cudaStream_t s, const uint16_t* wa, const uint16_t* wm,
                       bool host_a, bool host_m) {
        const uint16_t* g_attn = wa + lay.off_g_attn / 2;
        const uint16_t* wqkv = wa + lay.off_wqkv / 2;
        const uint16_t* wo = wa + lay.off_wo / 2;
        const uint16_t* g_mlp = wm + lay.off_g_mlp / 2;
        const uint16_t* wg = wm + lay.off_wg / 2;
        const uint16_t* wu = wm + lay.off_wu / 2;
        const uint16_t* wd = wm + lay.off_wd / 2;
        float* x = fixed_ptr<float>(fx.x);
        float* q = fixed_ptr<float>(fx.q);
        float* o = fixed_ptr<float>(fx.o);
        float* a = fixed_ptr<float>(fx.a);
        const int64_t* pt = fixed_ptr<int64_t>(fx.page_table);
        KvView kv = kv_view(l, pt);
        cudaError_t e;
        float* qk_raw = desc.qk_norm ? fixed_ptr<float>(fx.qk_raw) : nullptr;
        e = timed(0, s, [&] {
            cudaError_t r = launch_qkv_rope(x, g_attn, wqkv, B, H, Hq, Hkv, d, desc.rms_eps, desc.rope_theta, pos_dev,
                                            q, kv, nullptr, s, pdl(), host_a, qk_raw);
            if (r == cudaSuccess && qk_raw)
                r = launch_qk_norm_rope(qk_raw, B, Hq, Hkv, d, false, wa + lay.off_g_q / 2, wa + lay.off_g_k / 2,
                                        desc.rms_eps, desc.rope_theta, pos_dev, nullptr, q, kv, s, pdl());
            return r;
        });
        if (e != cudaSuccess) return cuda_fail(e, "qkv kernel");
        chain = true;
        e = timed(1, s, [&] {
            return launch_attention(q, kv, nullptr, pos_dev, nullptr, B, Hq, Hkv, d, cfg.max_ctx, true,
                                    fixed_ptr<float>(fx.attn_scratch), o, false, s, pdl(), cfg.max_batch, true);
        });
        if (e != cudaSuccess) return cuda_fail(e, "attention kernel");
        e = timed(2, s, [&] { return launch_resid_gemv(o, wo, B, H, qd, x, s, pdl(), host_a, true); });
        if (e != cudaSuccess) return cuda_fail(e, "o-proj kernel");
        e = timed(3, s, [&] {
            return launch_gate_up(x, g_mlp, wg, wu, B, H, F, desc.rms_eps, a, s, pdl(), host_m);
        });
        if (e != cudaSuccess) return cuda_fail(e, "gate/up kernel");
        e = timed(4, s, [&] { return launch_resid_gemv(a, wd, B, H, F, x, s, pdl(), host_m); });
        if (e != cudaSuccess) return cuda_fail(e, "down kernel");
        return LOIP_OK;
    }

    // Prefill layer on Mc token rows held in the prefill workspace.
    int prefill_layer(int l, int Mc, cudaStream_t s, int slot) {
        const uint16_t* wa = mha_base(l, slot);
        const uint16_t* wm = mlp_base(l, slot);
        float* px = fixed_ptr<float>(fx.px);
        uint16_t* py = fixed_ptr<uint16_t>(fx.py);
        float* pq = fixed_ptr<float>(fx.pq);
        uint16_t* po = fixed_ptr<uint16_t>(fx.po);
        uint16_t* pa = fixed_ptr<uint16_t>(fx.pa);
        const int32_t* pos = fixed_ptr<int32_t>(fx.positions);
        const int32_t* req = fixed_ptr<int32_t>(fx.row_req);
        const int64_t* pt = fixed_ptr<int64_t>(fx.page_table);
        KvView kv = kv_view(l, pt);
        cudaError_t e;
        e = timed(11, s, [&] { return launch_rmsnorm_split(px, wa + lay.off_g_attn / 2, Mc, H, desc.rms_eps, py, s); });
        if (e == cudaSuccess && !desc.qk_norm)
            e = timed(6, s, [&] {
                return launch_tc_gemm_qkv_rope(py, true, wa + lay.off_wqkv / 2, Mc, H, Hq, Hkv, d, desc.rope_theta, pos,
                                               req, pq, kv, s);
            });
        if (e == cudaSuccess && desc.qk_norm)  // raw projections (GEMM into zeros), then norm + rotation + stores
            e = timed(6, s, [&] {
                const int nqkv = (Hq + 2 * Hkv) * d;
                float* raw = fixed_ptr<float>(fx.qk_raw);
                cudaError_t r = cudaMemsetAsync(raw, 0, (size_t)Mc * nqkv * 4, s);
                if (r == cudaSuccess) r = launch_tc_gemm_resid(py, true, wa + lay.off_wqkv / 2, Mc, nqkv, H, raw, s);
                if (r == cudaSuccess)
                    r = launch_qk_norm_rope(raw, Mc, Hq, Hkv, d, true, wa + lay.off_g_q / 2, wa + lay.off_g_k / 2,
                                            desc.rms_eps, desc.rope_theta, pos, req, pq, kv, s);
                return r;
            });
        if (e == cudaSuccess)
            e = timed(7, s, [&] {
                return launch_attention_tc(pq, kv, fixed_ptr<int4>(fx.ptiles), prefill_tiles, Mc, Hq, Hkv, d, po, s);
            });
        if (e == cudaSuccess)
            e = timed(8, s, [&] { return launch_tc_gemm_resid(po, true, wa + lay.off_wo / 2, Mc, H, qd, px, s); });
        if (e == cudaSuccess)
            e = timed(11, s, [&] { return launch_rmsnorm_split(px, wm + lay.off_g_mlp / 2, Mc, H, desc.rms_eps, py, s); });
        if (e == cudaSuccess)
            e = timed(9, s, [&] {
                return launch_tc_gemm_swiglu(py, true, wm + lay.off_wg / 2, wm + lay.off_wu / 2, Mc, H, F, pa, s);
            });
        if (e == cudaSuccess)
            e = timed(10, s, [&] { return launch_tc_gemm_resid(pa, true, wm + lay.off_wd / 2, Mc, H, F, px, s); });
        if (e != cudaSuccess) return cuda_fail(e, "prefill kernel");
        return LOIP_OK;
    }

    // Layers l0 .. l1-1 (resident) of a batch-1 decode step in one persistent
    // launch.
    int decode_run(int l0, int l1, const int32_t* pos_dev, cudaStream_t s) {
        for (int b0 = l0; b0 < l1; b0 += kMaxRunLayers) {
            const int b1 = std::min(l1, b0 + kMaxRunLayers);
            DecodeRunArgs a{};
            for (int l = b0; l < b1; ++l) a.base[l - b0] = mha_at[l];  // whole layers: the blob base
            a.n_layers = b1 - b0;
            a.layer0 = b0;
            a.off_g_attn = lay.off_g_attn;
            a.off_wqkv = lay.off_wqkv;
            a.off_wo = lay.off_wo;
            a.off_g_mlp = lay.off_g_mlp;
            a.off_wg = lay.off_wg;
            a.off_wu = lay.off_wu;
            a.off_wd = lay.off_wd;
            a.H = H;
            a.Hq = Hq;
            a.Hkv = Hkv;
            a.d = d;
            a.F = F;
            a.eps = desc.rms_eps;
            a.theta = desc.rope_theta;
            a.x = fixed_ptr<float>(fx.x);
            a.q = fixed_ptr<float>(fx.q);
            a.o = fixed_ptr<float>(fx.o);
            a.a = fixed_ptr<float>(fx.a);
            a.positions = pos_dev;
            a.kv = kv_view(0, fixed_ptr<int64_t>(fx.page_table));
            a.attn_scratch = fixed_ptr<float>(fx.attn_scratch);
            a.scratch_rows = cfg.max_batch;
            a.max_ctx = cfg.max_ctx;
            a.sync = fixed_ptr<unsigned>(fx.run_sync);
            a.skip_block = -1;
            a.barrier_limit_us = 0;
            if (take_fault(LOIP_FAULT_BARRIER)) {  // one block misses the first barrier; waits give up after 10 ms
                a.skip_block = fault_arg;
                a.barrier_limit_us = 10000;
            }
            chain = false;
            cudaError_t e = timed(12, s, [&] { return launch_decode_run(a, s); });
            chain = false;
            if (e != cudaSuccess) return cuda_fail(e, "layer-run kernel");
            run_launched = true;
        }
        return LOIP_OK;
    }

    // Whether a batch-B decode step computes its runs of resident layers with
    // the persistent layer-run kernel.
    bool fuse_runs(int B) const {
        return B == 1 && cfg.layer_run_kernel && !desc.qk_norm && decode_run_supported(Hq, Hkv, d) &&
               cfg.max_ctx <= 64 * 256;
    }

    // Runs all layers once (decode or prefill pass) with the streaming ring.
    // run_pos != nullptr: batch-1 decode; runs of resident layers go to the
    // persistent layer-run kernel.
    template <class LayerFn>
    int run_layers(LayerFn&& fn, const int32_t* run_pos = nullptr) {
        const bool naive = cfg.mode == LOIP_MODE_NAIVE;
        for (int l = 0; l < L; ++l) {
            if (run_pos && !offloaded[l]) {
                int e = l;
                while (e < L && !offloaded[e]) ++e;
                int rc = decode_run(l, e, run_pos, compute);
                if (rc) return rc;
                l = e - 1;
                continue;
            }
            int slot = -1;
            if (offloaded[l]) {
                if (naive) {
                    // conventional path: load when needed, compute waits
                    slot = 0;
                    cudaEventRecord(ev_reach, compute);
                    chain = false;
                    cudaStreamWaitEvent(copy, ev_reach, 0);
                    int rc = enqueue_copy(l, 0, copy);
                    if (rc) return rc;
                } else {
                    slot = (int)(compute_seq % cfg.n_slots);
                    if (off_order[compute_seq % off_order.size()] != l)
                        return fail(LOIP_ERR_STATE, "slot ring out of order");
                }
                if (packed(l)) {
                    int rc = wait_packed_slot(slot, compute);
                    if (rc) return rc;
                } else {
                    cudaError_t e = cudaStreamWaitEvent(compute, slot_full[slot], 0);
                    if (e != cudaSuccess) return cuda_fail(e, "compute wait");
                }
                chain = false;
            }
            int rc = fn(l, slot);
            if (rc) return rc;
            if (offloaded[l]) {
                cudaError_t e = cudaEventRecord(slot_free[slot], compute);
                if (e != cudaSuccess) return cuda_fail(e, "slot free event");
                chain = false;
                if (!naive) {
                    ++compute_seq;
                    rc = issue_next_copy();
                    if (rc) return rc;
                }
            }
        }
        return LOIP_OK;
    }

    void collect_copy_time() {
        double busy = 0;
        while (!copy_events.empty()) {
            const CopyEv ce = copy_events.front();
            if (cudaEventQuery(ce.b) != cudaSuccess) break;
            float ms = 0;
            cudaEventElapsedTime(&ms, ce.a, ce.b);
            busy += ms;
            st.copy_ms_total += ms;
            st.copies_total += 1;
            if (copy_log.size() < kCopyLog) copy_log.resize(kCopyLog);
            copy_log[copy_log_next % kCopyLog] = {ms, ce.bytes};
            ++copy_log_next;
            if (ce.ssd) st.ssd_copy_ms += ms;
            event_pool.push_back(ce.a);
            event_pool.push_back(ce.b);
            copy_events.pop_front();
        }
        st.copy_busy_ms = busy;
    }

    // ---- online re-planning (Eq. 6) -------------------------------------------
    // Eq. 7 on one device: the resident blocks to offload for one more page
    // group, the fewest bytes first (an MHA block while any is resident); the
    // victim layer is the middle of the longest run of whole resident layers
    // (keeping the streamed layers evenly spaced), else the first layer still
    // holding a block of that kind.  The freed range becomes page groups.
    int demote_block_for_kv(uint64_t need_groups) {
        int n_mha = 0, n_mlp = 0;
        for (int l = 0; l < L; ++l) {
            n_mha += (res_mask[l] & 1) ? 1 : 0;
            n_mlp += (res_mask[l] & 2) ? 1 : 0;
        }
        if (lay.mha_bytes < group_bytes) n_mha = 0;  // a block that cannot hold a page group frees nothing
        if (lay.mlp_bytes < group_bytes) n_mlp = 0;
        int alpha = 0, beta = 0;
        if (!eq7_choice(need_groups * group_bytes, n_mha, n_mlp, lay.mha_bytes, lay.mlp_bytes, &alpha, &beta) &&
            !eq7_choice(group_bytes, n_mha, n_mlp, lay.mha_bytes, lay.mlp_bytes, &alpha, &beta))
            return fail(LOIP_ERR_OOM, "KV cache does not fit even with every block offloaded");
        int rc = sync_all();
        if (rc) return rc;
        rc = ensure_slots();
        if (rc) return rc;
        for (int which = 0; which < 2; ++which) {
            const int count = which == 0 ? alpha : beta;
            const uint8_t bit = which == 0 ? 1 : 2;
            for (int c = 0; c < count; ++c) {
                std::vector<uint8_t> mask = offloaded;
                int victim = -1;
                bool any_whole = false;
                for (int l = 0; l < L; ++l) any_whole |= res_mask[l] == 3;
                if (any_whole) victim = demote_one(L, mask.data());
                if (victim < 0 || !(res_mask[victim] & bit))
                    for (int l = 0; l < L && victim < 0; ++l)
                        if (res_mask[l] & bit) victim = l;
                if (victim < 0 || !(res_mask[victim] & bit)) return fail(LOIP_ERR_STATE, "no resident block to offload");
                rc = ensure_host_copy(victim);
                if (rc) return rc;
                if (bit == 1) {
                    carve_kv(mha_at[victim], lay.mha_bytes);
                    mha_at[victim] = nullptr;
                } else {
                    carve_kv(mlp_at[victim], lay.mlp_bytes);
                    mlp_at[victim] = nullptr;
                }
                res_mask[victim] &= (uint8_t)~bit;
                offloaded[victim] = 1;
                if (res_mask[victim] == 0 && layer_block[victim] >= 0) {  // its whole block now serves the KV cache
                    block_kind[layer_block[victim]] = B_KV;
                    block_owner[layer_block[victim]] = -1;
                    layer_block[victim] = -1;
                }
            }
        }
        rebuild_order();
        st.n_replans++;
        return prime_slots();
    }

    // The slot ring needs its blocks once a first layer streams: free blocks, or
    // the blocks of whole layers taken for it.
    int ensure_slots() {
        if (!off_order.empty()) return LOIP_OK;
        std::vector<uint8_t> mask = offloaded;
        for (int k = 0; k < cfg.n_slots; ++k) {
            int b = take_free_block();
            if (b < 0) {
                int v2 = demote_one(L, mask.data());
                if (v2 < 0 || res_mask[v2] != 3) return fail(LOIP_ERR_OOM, "no room for slots");
                int rc2 = demote_layer(v2);
                if (rc2) return rc2;
                b = take_free_block();
            }
            block_kind[b] = B_SLOT;
            block_owner[b] = k;
            slot_block[k] = b;
        }
        return LOIP_OK;
    }

    // a host copy of layer l's whole blob (gathered from its resident blocks)
    int ensure_host_copy(int l) {
        if (host_layer[l]) return LOIP_OK;
        HostBuf hb;
        cudaError_t e = host_buf_alloc(lay.l_size, &hb);
        if (e != cudaSuccess) return fail(LOIP_ERR_OOM, "pinned allocation for a demoted layer failed");
        host_regions.push_back(hb);
        host_layer[l] = hb.ptr;
        char* h = static_cast<char*>(hb.ptr);
        if (mha_at[l]) e = cudaMemcpy(h, mha_at[l], lay.mha_bytes, cudaMemcpyDeviceToHost);
        if (e == cudaSuccess && mlp_at[l]) e = cudaMemcpy(h + lay.mha_bytes, mlp_at[l], lay.mlp_bytes, cudaMemcpyDeviceToHost);
        if (e != cudaSuccess) return cuda_fail(e, "demote copy");
        return LOIP_OK;
    }

    // KV growth past the memory left (Eq. 6): make room for need_groups more page
    // groups (at least one) by offloading blocks (Eq. 7) or one whole layer
    int demote_for_kv(uint64_t need_groups = 1) {
        if (!cfg.whole_layers) return demote_block_for_kv(need_groups < 1 ? 1 : need_groups);
        // offload one more resident layer; its block becomes free
        std::vector<uint8_t> mask = offloaded;
        int victim = demote_one(L, mask.data());
        if (victim < 0) return fail(LOIP_ERR_OOM, "KV cache does not fit even with every layer offloaded");
        int rc = sync_all();
        if (rc) return rc;
        if (off_order.empty()) {
            // the first offloaded layer also needs the slots
            for (int k = 0; k < cfg.n_slots; ++k) {
                int b = take_free_block();
                if (b < 0) {
                    // take resident layers until the slots fit
                    std::vector<uint8_t> m2 = mask;
                    int v2 = demote_one(L, m2.data());
                    if (v2 < 0) return fail(LOIP_ERR_OOM, "no room for slots");
                    int rc2 = demote_layer(v2);
                    if (rc2) return rc2;
                    mask = m2;
                    b = take_free_block();
                }
                block_kind[b] = B_SLOT;
                block_owner[b] = k;
                slot_block[k] = b;
            }
        }
        rc = demote_layer(victim);
        if (rc) return rc;
        rebuild_order();
        st.n_replans++;
        return prime_slots();
    }

    int demote_layer(int l) {  // a whole resident layer: its block becomes free
        int rc = ensure_host_copy(l);
        if (rc) return rc;
        int b = layer_block[l];
        block_kind[b] = B_FREE;
        block_owner[b] = -1;
        layer_block[l] = -1;
        res_mask[l] = 0;
        mha_at[l] = mlp_at[l] = nullptr;
        offloaded[l] = 1;
        return LOIP_OK;
    }

    // Times one copy of every offloaded layer's host blob into slot 0 and moves
    // blobs that copy clearly slower than the pool's median (pages the host
    // could not back with huge pages copy at a fraction of the link rate) to a
    // fresh buffer, keeping the slow memory reserved while retrying so it is not
    // handed back.  At most 3 attempts per blob; the fastest buffer wins.
    int qualify_host_pool() {
        std::vector<int> pooled;  // streamed layers with a blob in the host pool (not in the SSD tier)
        for (int l : off_order)
            if (host_layer[l]) pooled.push_back(l);
        if (pooled.empty()) return LOIP_OK;
        cudaEvent_t a = take_event(), b = take_event();
        auto rate = [&](const void* src, double* gbps, uint64_t bytes) -> int {
            cudaEventRecord(a, compute);
            cudaError_t e = cudaMemcpyAsync(slot_ptr(0), src, bytes, cudaMemcpyHostToDevice, compute);
            cudaEventRecord(b, compute);
            if (e == cudaSuccess) e = cudaEventSynchronize(b);
            float ms = 0;
            if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, a, b);
            if (e != cudaSuccess) return cuda_fail(e, "pool qualification copy");
            *gbps = ms > 0 ? (double)bytes / (ms * 1e-3) / 1e9 : 0.0;
            return LOIP_OK;
        };
        std::vector<double> r(L, 0.0);
        for (int l : pooled) {
            int rc = rate(host_layer[l], &r[l], host_bytes(l));
            if (rc) return rc;
        }
        std::vector<double> sorted;
        for (int l : pooled) sorted.push_back(r[l]);
        std::sort(sorted.begin(), sorted.end());
        const double median = sorted[sorted.size() / 2];
        std::vector<HostBuf> spare;  // rejected buffers, released after the search
        for (int l : pooled) {
            for (int attempt = 0; attempt < 3 && r[l] < 0.9 * median; ++attempt) {
                HostBuf hb;
                if (host_buf_alloc(host_bytes(l), &hb) != cudaSuccess) break;
                double g = 0;
                int rc = rate(hb.ptr, &g, host_bytes(l));
                if (rc) return rc;
                if (g > r[l]) {
                    // (the pool is filled after qualification: nothing to move)
                    host_regions.push_back(hb);
                    host_layer[l] = hb.ptr;
                    r[l] = g;
                    st.pool_replaced += 1;
                } else {
                    spare.push_back(hb);
                }
            }
        }
        for (auto& hb : spare) host_buf_free(&hb);
        double mn = 1e30;
        for (int l : pooled) mn = std::min(mn, r[l]);
        st.pool_min_GBps = mn;
        st.pool_median_GBps = median;
        record_pool_placement(pooled);
        event_pool.push_back(a);
        event_pool.push_back(b);
        return LOIP_OK;
    }

    // Where the pooled blobs' pages landed (32 sampled pages per blob) against
    // the node the pool asked for (the GPU's host node).
    void record_pool_placement(const std::vector<int>& pooled) {
        pool_node.assign(L, -1);
        int want = -1;
        for (const HostBuf& hb : host_regions)
            if (hb.node >= 0) want = hb.node;
        int on = 0;
        for (int l : pooled) {
            double frac = 0;
            pool_node[l] = host_range_node(host_layer[l], host_bytes(l), 32, &frac);
            on += (want >= 0 && pool_node[l] == want) ? 1 : 0;
        }
        st.pool_numa_node = want;
        st.pool_blobs = (int32_t)pooled.size();
        st.pool_blobs_on_node = on;
    }

    // One pinned region for every offloaded layer that has no host copy yet.
    int ensure_host_pool() {
        std::vector<int> need;
        for (int l = 0; l < L; ++l)
            if (offloaded[l] && !host_layer[l] && disk_off[l] < 0) need.push_back(l);
        if (need.empty()) return LOIP_OK;
        // packed layers take their packed area; the layer is marked packed now
        // and cleared by pack_layer if it has to travel raw after all
        const uint64_t per = packing ? pack_area : lay.l_size;
        if (take_fault(LOIP_FAULT_HOST_ALLOC)) return fail(LOIP_ERR_OOM, "pinned host pool allocation failed");
        // regions of about 8 GB, each entirely in huge pages: a region that comes
        // back partly in base pages is held (so the next try gets other memory)
        // and allocated again, up to three more times; the best one is kept
        const size_t group = std::max<size_t>(1, (size_t)((8ull << 30) / per));
        std::vector<HostBuf> spare;
        double huge_min = 1.0;
        for (size_t g0 = 0; g0 < need.size(); g0 += group) {
            const size_t n = std::min(group, need.size() - g0);
            HostBuf best;
            for (int attempt = 0; attempt < 4; ++attempt) {
                HostBuf b;
                if (host_buf_alloc(n * per, &b) != cudaSuccess) break;
                if (!best.ptr || b.huge > best.huge) {
                    if (best.ptr) spare.push_back(best);
                    best = b;
                } else {
                    spare.push_back(b);
                }
                if (best.huge >= 0.999) break;
            }
            if (!best.ptr) {
                for (auto& hb : spare) host_buf_free(&hb);
                return fail(LOIP_ERR_OOM, "pinned host pool allocation failed");
            }
            huge_min = std::min(huge_min, best.huge);
            host_regions.push_back(best);
            for (size_t i = 0; i < n; ++i) {
                host_layer[need[g0 + i]] = static_cast<char*>(best.ptr) + i * per;
                if (packing) pk[need[g0 + i]].on = true;
            }
        }
        for (auto& hb : spare) host_buf_free(&hb);
        st.pool_huge_min = huge_min;
        return qualify_host_pool();
    }

    uint64_t arena_used() const {
        uint64_t used = fx.total + kv_region_bytes + tail_used;
        for (int b = 0; b < n_blocks; ++b)
            if (block_kind[b] != B_FREE) used += block_bytes;
        return used;
    }
};

// ============================================================================
// C ABI
// ============================================================================
#define CTX_GUARD(ctx)                                                             \
    do {                                                                           \
        if (!(ctx)) return LOIP_ERR_INVALID;                                       \
        if ((ctx)->failed) return (ctx)->fail(LOIP_ERR_STATE, "context failed earlier: " + (ctx)->err); \
    } while (0)

extern "C" int loip_layer_layout(const loip_model_desc* desc, loip_layer_layout_t* out) {
    if (!out || validate_desc(desc)) return LOIP_ERR_INVALID;
    layout_of(desc, out);
    return LOIP_OK;
}

extern "C" int loip_fixed_bytes(const loip_model_desc* desc, const loip_config* cfg, uint64_t* out) {
    if (!out || !cfg || validate_desc(desc) || cfg->max_batch < 1 || cfg->max_batch > 8 || cfg->max_ctx < 1)
        return LOIP_ERR_INVALID;
    loip_config c = normalized(cfg);
    *out = fixed_layout(desc, &c).total;
    return LOIP_OK;
}

extern "C" const char* loip_last_error(const loip_ctx* ctx) {
    return ctx ? ctx->err.c_str() : g_create_error.c_str();
}

extern "C" void loip_destroy(loip_ctx* ctx) {
    if (!ctx) return;
    if (ctx->compute) cudaStreamSynchronize(ctx->compute);
    if (ctx->copy) cudaStreamSynchronize(ctx->copy);
    if (ctx->unpack_st) cudaStreamSynchronize(ctx->unpack_st);
    for (auto& hb : ctx->host_regions) host_buf_free(&hb);
    host_buf_free(&ctx->embed_host);
    for (int b = 0; b < loip_ctx::kStages; ++b) {
        host_buf_free(&ctx->stage[b]);
        if (ctx->stage_done[b]) cudaEventDestroy(ctx->stage_done[b]);
    }
    ctx->disk.close();
    if (ctx->h_stage) cudaFreeHost(ctx->h_stage);
    if (ctx->h_pt) cudaFreeHost(ctx->h_pt);
    for (auto e : ctx->slot_full) cudaEventDestroy(e);
    for (auto e : ctx->raw_done)
        if (e) cudaEventDestroy(e);
    for (auto e : ctx->slot_free) cudaEventDestroy(e);
    for (auto& pr : ctx->copy_events) {
        cudaEventDestroy(pr.a);
        cudaEventDestroy(pr.b);
    }
    for (auto& k : ctx->kernel_events) {
        cudaEventDestroy(k.a);
        cudaEventDestroy(k.b);
    }
    for (auto e : ctx->event_pool) cudaEventDestroy(e);
    for (cudaEvent_t e : {ctx->ev_done, ctx->ev_step0, ctx->ev_step1, ctx->ev_reach, ctx->ev_stage})
        if (e) cudaEventDestroy(e);
    for (int g = 0; g < kPackRingMax; ++g) {
        if (ctx->chunk_ready[g]) cudaEventDestroy(ctx->chunk_ready[g]);
        if (ctx->chunk_free[g]) cudaEventDestroy(ctx->chunk_free[g]);
    }
    if (ctx->compute) cudaStreamDestroy(ctx->compute);
    if (ctx->copy) cudaStreamDestroy(ctx->copy);
    if (ctx->unpack_st) cudaStreamDestroy(ctx->unpack_st);
    delete ctx;
}

extern "C" int loip_create(const loip_model_desc* desc, const loip_config* cfg_in, void* device_arena,
                           uint64_t arena_bytes, loip_ctx** out) {
    if (!out) return LOIP_ERR_INVALID;
    *out = nullptr;
    if (validate_desc(desc) || !cfg_in) {
        g_create_error = "invalid model description";
        return LOIP_ERR_INVALID;
    }
    loip_config cfg = normalized(cfg_in);
    if (cfg.n_slots < 1 || cfg.n_slots > 3 || cfg.max_batch < 1 || cfg.max_batch > 8 || cfg.max_ctx < 1 ||
        cfg.max_ctx > 16384 ||
        cfg.page_tokens != 64 || !device_arena || ((uintptr_t)device_arena % kAlign) ||
        arena_bytes < cfg.device_budget_bytes ||
        (cfg.mode != LOIP_MODE_OVERLAP && cfg.mode != LOIP_MODE_NAIVE && cfg.mode != LOIP_MODE_DIRECT)) {
        g_create_error = "invalid configuration (slots 1..3, batch 1..8, page 64, arena >= budget, aligned)";
        return LOIP_ERR_INVALID;
    }
    if (cfg.mode == LOIP_MODE_NAIVE) cfg.n_slots = 1;
    loip_ctx* c = new loip_ctx();
    c->desc = *desc;
    c->cfg = cfg;
    layout_of(desc, &c->lay);
    c->L = desc->n_layers;
    c->init_packing();
    c->H = desc->hidden;
    c->Hq = desc->n_heads;
    c->Hkv = desc->n_kv_heads;
    c->d = desc->head_dim;
    c->F = desc->ffn;
    c->V = desc->vocab;
    c->qd = c->Hq * c->d;
    c->kvd = c->Hkv * c->d;
    c->arena = reinterpret_cast<char*>(device_arena);
    c->budget = cfg.device_budget_bytes;
    c->fx = fixed_layout(desc, &cfg);
    c->layer_page_bytes = 2ull * c->Hkv * cfg.page_tokens * c->d * 2;
    c->group_bytes = align_up(c->layer_page_bytes * c->L);
    c->kv_tok_bytes = 2ull * c->kvd * 2 * c->L;
    c->max_pages = (cfg.max_ctx + cfg.page_tokens - 1) / cfg.page_tokens;
    c->block_bytes = align_up(c->lay.l_size);
    if (c->group_bytes > c->block_bytes) {
        g_create_error = "a KV page group is larger than a layer block";
        delete c;
        return LOIP_ERR_INVALID;
    }
    // KV region reserved up front
    uint64_t kv_groups = cfg.kv_reserve_bytes ? (cfg.kv_reserve_bytes + c->group_bytes - 1) / c->group_bytes
                                              : (uint64_t)cfg.max_batch * c->max_pages;
    c->kv_region_off = c->fx.total;
    c->kv_region_bytes = kv_groups * c->group_bytes;
    c->blocks_off = align_up(c->kv_region_off + c->kv_region_bytes);
    if (c->budget < c->blocks_off) {
        g_create_error = "budget smaller than the fixed part and the KV reserve";
        delete c;
        return LOIP_ERR_INFEASIBLE;
    }
    c->n_blocks = (int)((c->budget - c->blocks_off) / c->block_bytes);
    // plan (Algorithm 1 memory-first fill with the slot ring)
    std::vector<uint64_t> lb(c->L, c->block_bytes);
    std::vector<uint8_t> res(c->L);
    loip_plan plan{};
    plan.resident = res.data();
    int rc = loip_plan_residency(desc, lb.data(), c->budget, c->kv_region_bytes, c->blocks_off - c->kv_region_bytes,
                                 cfg.n_slots, cfg.hbm_Bps, cfg.link_Bps, &plan);
    if (rc) {
        g_create_error = "budget cannot hold the fixed part, the KV reserve and the slots";
        delete c;
        return rc;
    }
    c->offloaded.assign(c->L, 0);
    c->layer_block.assign(c->L, -1);
    c->res_mask.assign(c->L, 0);
    c->mha_at.assign(c->L, nullptr);
    c->mlp_at.assign(c->L, nullptr);
    c->block_kind.assign(c->n_blocks, B_FREE);
    c->block_owner.assign(c->n_blocks, -1);
    int nb = 0;
    for (int l = 0; l < c->L; ++l) {
        if (res[l]) {
            c->set_resident_block(l, nb);
            c->block_kind[nb] = B_LAYER;
            c->block_owner[nb] = l;
            ++nb;
        } else {
            c->offloaded[l] = 1;
        }
    }
    c->rebuild_order();
    c->slot_block.assign(cfg.n_slots, -1);
    if (!c->off_order.empty()) {
        for (int k = 0; k < cfg.n_slots; ++k) {
            if (nb >= c->n_blocks) {
                g_create_error = "internal: slots do not fit";
                delete c;
                return LOIP_ERR_INFEASIBLE;
            }
            c->slot_block[k] = nb;
            c->block_kind[nb] = B_SLOT;
            c->block_owner[nb] = k;
            ++nb;
        }
    }
    // Algorithm 1's block-level refinement: the memory after the whole blocks
    // keeps blocks of offloaded layers resident (MLP block first)
    c->tail_off = c->blocks_off + (uint64_t)c->n_blocks * c->block_bytes;
    if (!cfg.whole_layers && !c->off_order.empty() && c->budget > c->tail_off) {
        std::vector<uint8_t> masks(c->L);
        refine_blocks(c->budget - c->tail_off, c->L, c->offloaded.data(), c->lay.mha_bytes, c->lay.mlp_bytes,
                      masks.data());
        for (int l = 0; l < c->L; ++l) {
            if (!c->offloaded[l] || masks[l] == 0) continue;
            char* at = c->arena + c->tail_off + c->tail_used;
            if (masks[l] == 2) {
                c->mlp_at[l] = at;
                c->tail_used += c->lay.mlp_bytes;
            } else {
                c->mha_at[l] = at;
                c->tail_used += c->lay.mha_bytes;
            }
            c->res_mask[l] = masks[l];
        }
    }
    for (uint64_t i = 0; i < kv_groups; ++i)
        c->free_groups.push_back((int64_t)(c->kv_region_off + (kv_groups - 1 - i) * c->group_bytes));
    c->kv_groups_total = kv_groups;
    c->reqs.resize(cfg.max_batch);
    c->host_layer.assign(c->L, nullptr);
    // SSD tier: when the host budget cannot hold every streamed layer, the rest
    // (evenly spaced among them) go to a scratch file; kStages staging buffers
    // come out of the host budget
    c->disk_off.assign(c->L, -1);
    if (cfg.host_budget_bytes && !c->off_order.empty()) {
        const uint64_t fit = cfg.host_budget_bytes / c->lay.l_size;
        const int m = (int)c->off_order.size();
        if (fit < (uint64_t)m) {
            if (fit < (uint64_t)loip_ctx::kStages) {
                g_create_error = "host budget cannot hold the SSD tier's staging buffers";
                loip_destroy(c);
                return LOIP_ERR_INFEASIBLE;
            }
            const int nd = m - (int)(fit - loip_ctx::kStages);
            c->disk_stride = (c->lay.l_size + DiskTier::kDiskAlign - 1) / DiskTier::kDiskAlign * DiskTier::kDiskAlign;
            int j = 0;
            for (int i = 0; i < m; ++i)
                if ((int64_t)(i + 1) * nd / m > (int64_t)i * nd / m)
                    c->disk_off[c->off_order[i]] = (int64_t)(j++) * (int64_t)c->disk_stride;
            std::string err;
            if (!c->disk.open(cfg.ssd_dir, &err)) {
                g_create_error = err;
                loip_destroy(c);
                return LOIP_ERR_STATE;
            }
            for (int b = 0; b < loip_ctx::kStages; ++b) {
                if (host_buf_alloc_plain(c->disk_stride, &c->stage[b]) != cudaSuccess ||
                    cudaEventCreateWithFlags(&c->stage_done[b], cudaEventDisableTiming) != cudaSuccess) {
                    g_create_error = "SSD-tier staging buffers";
                    loip_destroy(c);
                    return LOIP_ERR_OOM;
                }
            }
            c->st.n_ssd_layers = j;
        }
    }

    cudaError_t e;
    e = cudaStreamCreateWithFlags(&c->compute, cudaStreamNonBlocking);
    if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&c->copy, cudaStreamNonBlocking);
    if (e == cudaSuccess && c->packing) {  // unpack kernels: short, they gate the staging ring
        int lo = 0, hi = 0;
        e = cudaDeviceGetStreamPriorityRange(&lo, &hi);
        if (e == cudaSuccess) e = cudaStreamCreateWithPriority(&c->unpack_st, cudaStreamNonBlocking, hi);
        for (int g = 0; g < c->ring && e == cudaSuccess; ++g) {
            e = cudaEventCreateWithFlags(&c->chunk_ready[g], cudaEventDisableTiming);
            if (e == cudaSuccess) e = cudaEventCreateWithFlags(&c->chunk_free[g], cudaEventDisableTiming);
        }
        c->slot_inline.assign(cfg.n_slots, 0);
        c->raw_pumped.assign(cfg.n_slots, 1);
        c->inl_left.assign(cfg.n_slots, 0);
        c->inl_chunks.assign(cfg.n_slots, {});
        c->raw_done.assign(cfg.n_slots, nullptr);
        for (int k = 0; k < cfg.n_slots && e == cudaSuccess; ++k)
            e = cudaEventCreateWithFlags(&c->raw_done[k], cudaEventDisableTiming);
    }
    c->slot_full.resize(cfg.n_slots);
    c->slot_free.resize(cfg.n_slots);
    for (int k = 0; k < cfg.n_slots && e == cudaSuccess; ++k) {
        e = cudaEventCreateWithFlags(&c->slot_full[k], cudaEventDisableTiming);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&c->slot_free[k], cudaEventDisableTiming);
    }
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&c->ev_done, cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&c->ev_reach, cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&c->ev_stage, cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreate(&c->ev_step0);
    if (e == cudaSuccess) e = cudaEventCreate(&c->ev_step1);
    // staging: a prefill chunk's tokens, positions, requests and attention tiles;
    // the second quarter also receives the output tokens
    c->h_stage_ints = 8 * (size_t)std::max(cfg.max_batch, cfg.max_prefill_tokens) + 4 * (size_t)cfg.max_batch + 128;
    if (e == cudaSuccess) e = cudaHostAlloc(&c->h_stage, c->h_stage_ints * 4, cudaHostAllocDefault);
    if (e == cudaSuccess) e = cudaHostAlloc(&c->h_pt, (size_t)cfg.max_batch * c->max_pages * 8, cudaHostAllocDefault);
    if (e != cudaSuccess) {
        g_create_error = std::string("CUDA setup failed: ") + cudaGetErrorString(e);
        loip_destroy(c);
        return LOIP_ERR_CUDA;
    }
    // attention completion counters start at zero (each launch leaves them zero)
    e = cudaMemsetAsync(c->arena + c->fx.attn_scratch, 0,
                        attention_scratch_floats(cfg.max_batch, c->Hq, c->d, cfg.max_ctx, cfg.page_tokens) * 4,
                        c->compute);
    if (e == cudaSuccess) e = cudaMemsetAsync(c->arena + c->fx.run_sync, 0, 4 * (2 + 4 * kMaxRunLayers), c->compute);
    c->h_stage[c->h_stage_ints - 1] = 0;
    if (e == cudaSuccess) e = cudaStreamSynchronize(c->compute);
    if (e != cudaSuccess) {
        g_create_error = std::string("CUDA setup failed: ") + cudaGetErrorString(e);
        loip_destroy(c);
        return LOIP_ERR_CUDA;
    }
    c->st.n_resident = c->L - (int)c->off_order.size();
    c->st.n_offloaded = (int)c->off_order.size();
    *out = c;
    return LOIP_OK;
}

extern "C" int loip_get_plan(const loip_ctx* ctx, loip_plan* out) {
    if (!ctx || !out || !out->resident) return LOIP_ERR_INVALID;
    out->n_layers = ctx->L;
    out->n_offloaded = (int)ctx->off_order.size();
    out->n_resident = ctx->L - out->n_offloaded;
    for (int l = 0; l < ctx->L; ++l) out->resident[l] = ctx->offloaded[l] ? 0 : 1;
    std::vector<double> comp(ctx->L), load(ctx->L);
    double copy_s = 0;
    for (int l = 0; l < ctx->L; ++l) {
        comp[l] = (double)ctx->lay.l_size / ctx->cfg.hbm_Bps;
        load[l] = (double)ctx->stream_bytes(l) / ctx->cfg.link_Bps;
        if (ctx->offloaded[l]) copy_s += load[l];
    }
    out->pred_step_s = simulate_step(comp, load, ctx->offloaded.data(), ctx->cfg.n_slots, 4);
    out->eq1_step_s = eq1_single_device(comp, load, ctx->offloaded.data());
    out->pred_copy_s = copy_s;
    out->pred_compute_s = ctx->L * comp[0];
    uint64_t used = ctx->arena_used();
    out->left_bytes = ctx->budget > used ? ctx->budget - used : 0;
    return LOIP_OK;
}

extern "C" int loip_get_block_plan(const loip_ctx* ctx, uint8_t* masks, uint64_t* stream_bytes_per_step) {
    if (!ctx || !masks || !stream_bytes_per_step) return LOIP_ERR_INVALID;
    uint64_t bytes = 0;
    for (int l = 0; l < ctx->L; ++l) {
        masks[l] = ctx->res_mask[l];
        bytes += ctx->stream_bytes(l);
    }
    *stream_bytes_per_step = bytes;
    return LOIP_OK;
}

static int write_layer_generated(loip_ctx* c, char* dst, int l, uint64_t seed) {
    const uint64_t H = c->H, F = c->F, qd = c->qd, kvd = c->kvd;
    auto T = [&](int which) { return (uint32_t)(16 + 16 * l + which); };
    uint16_t* base = reinterpret_cast<uint16_t*>(dst);
    const loip_layer_layout_t& y = c->lay;
    cudaStream_t s = c->compute;
    cudaError_t e = cudaSuccess;
    auto gen = [&](uint64_t off_bytes, uint64_t n, uint32_t tid, int kind) {
        if (e == cudaSuccess) e = launch_generate(base + off_bytes / 2, n, 0, seed, tid, kind, s);
    };
    gen(y.off_g_attn, H, T(0), 1);
    gen(y.off_wqkv, qd * H, T(1), 0);
    gen(y.off_wqkv + qd * H * 2, kvd * H, T(2), 0);
    gen(y.off_wqkv + (qd + kvd) * H * 2, kvd * H, T(3), 0);
    gen(y.off_wo, H * qd, T(4), 0);
    gen(y.off_g_mlp, H, T(5), 1);
    gen(y.off_wg, F * H, T(6), 0);
    gen(y.off_wu, F * H, T(7), 0);
    gen(y.off_wd, H * F, T(8), 0);
    if (c->desc.qk_norm) {
        gen(y.off_g_q, (uint64_t)c->d, T(9), 1);
        gen(y.off_g_k, (uint64_t)c->d, T(10), 1);
    }
    if (e != cudaSuccess) return c->cuda_fail(e, "generator kernel");
    return LOIP_OK;
}

extern "C" int loip_load_weights_generated(loip_ctx* c, uint64_t seed) {
    CTX_GUARD(c);
    int rc = c->sync_all();
    if (rc) return rc;
    rc = c->ensure_embed_host();
    if (rc) return rc;
    // (a host-resident table is written by the generator through its mapping)
    cudaError_t e = launch_generate(const_cast<uint16_t*>(c->embed_table()), (uint64_t)c->V * c->H, 0, seed, 1, 0,
                                    c->compute);
    if (e == cudaSuccess)
        e = launch_generate(c->fixed_ptr<uint16_t>(c->fx.lm_head), (uint64_t)c->V * c->H, 0, seed, 2, 0, c->compute);
    if (e == cudaSuccess)
        e = launch_generate(c->fixed_ptr<uint16_t>(c->fx.g_final), (uint64_t)c->H, 0, seed, 3, 1, c->compute);
    if (e != cudaSuccess) return c->cuda_fail(e, "generator kernel");
    for (int l = 0; l < c->L; ++l) {
        if (c->res_mask[l] == 3) {
            rc = write_layer_generated(c, c->mha_at[l], l, seed);
            if (rc) return rc;
        } else {
            rc = c->ensure_host_pool();
            if (rc) return rc;
            char* tmp = c->slot_ptr(0);
            if (c->packed(l)) {  // defined padding between the tensors (it is packed too)
                e = cudaMemsetAsync(tmp, 0, c->lay.l_size, c->compute);
                if (e != cudaSuccess) return c->cuda_fail(e, "slot clear");
            }
            rc = write_layer_generated(c, tmp, l, seed);
            if (rc) return rc;
            if (c->packed(l)) {
                rc = c->store_packed(l, tmp);
                if (rc) return rc;
            } else if (c->disk_off[l] >= 0) {  // SSD tier: through a staging buffer to the file
                rc = c->sync_all();
                if (rc) return rc;
                rc = c->write_disk_blob(l, tmp, cudaMemcpyDeviceToHost);
                if (rc) return rc;
            } else {
                e = cudaMemcpyAsync(c->host_layer[l], tmp, c->lay.l_size, cudaMemcpyDeviceToHost, c->compute);
            }
            if (e == cudaSuccess && c->mha_at[l])  // its resident block (block-level refinement)
                e = cudaMemcpyAsync(c->mha_at[l], tmp, c->lay.mha_bytes, cudaMemcpyDeviceToDevice, c->compute);
            if (e == cudaSuccess && c->mlp_at[l])
                e = cudaMemcpyAsync(c->mlp_at[l], tmp + c->lay.mha_bytes, c->lay.mlp_bytes, cudaMemcpyDeviceToDevice,
                                    c->compute);
            if (e != cudaSuccess) return c->cuda_fail(e, "host pool copy");
        }
    }
    rc = c->sync_all();
    if (rc) return rc;
    c->weights_loaded = true;
    rc = c->prime_slots();
    if (rc) return rc;
    return c->sync_all();
}

extern "C" int loip_load_layer(loip_ctx* c, int32_t layer, const void* host_blob, uint64_t bytes) {
    CTX_GUARD(c);
    if (layer < 0 || layer >= c->L || !host_blob || bytes != c->lay.l_size)
        return c->fail(LOIP_ERR_INVALID, "layer index or blob size");
    int rc = c->sync_all();
    if (rc) return rc;
    rc = c->ensure_host_pool();  // every offloaded layer gets its pool blob before the ring is primed
    if (rc) return rc;
    cudaError_t e;
    const char* hb = static_cast<const char*>(host_blob);
    if (c->res_mask[layer] != 3 && c->disk_off[layer] >= 0) {
        rc = c->write_disk_blob(layer, hb, cudaMemcpyHostToHost);
        if (rc) return rc;
    } else if (c->res_mask[layer] != 3 && c->packed(layer)) {
        e = cudaMemcpy(c->slot_ptr(0), hb, bytes, cudaMemcpyHostToDevice);
        if (e != cudaSuccess) return c->cuda_fail(e, "layer upload");
        rc = c->store_packed(layer, c->slot_ptr(0));
        if (rc) return rc;
    } else if (c->res_mask[layer] != 3) {
        memcpy(c->host_layer[layer], host_blob, bytes);
    }
    e = cudaSuccess;
    if (c->mha_at[layer]) e = cudaMemcpy(c->mha_at[layer], hb, c->lay.mha_bytes, cudaMemcpyHostToDevice);
    if (e == cudaSuccess && c->mlp_at[layer])
        e = cudaMemcpy(c->mlp_at[layer], hb + c->lay.mha_bytes, c->lay.mlp_bytes, cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return c->cuda_fail(e, "layer upload");
    c->weights_loaded = true;
    rc = c->prime_slots();
    return rc ? rc : c->sync_all();
}

extern "C" int loip_load_globals(loip_ctx* c, const uint16_t* embed, const uint16_t* lm_head, const uint16_t* g_final) {
    CTX_GUARD(c);
    if (!embed || !lm_head || !g_final) return c->fail(LOIP_ERR_INVALID, "null pointer");
    size_t vh = (size_t)c->V * c->H * 2;
    int rc = c->ensure_embed_host();
    if (rc) return rc;
    cudaError_t e = cudaSuccess;
    if (c->cfg.embed_on_host)
        memcpy(c->embed_host.ptr, embed, vh);
    else
        e = cudaMemcpy(c->arena + c->fx.embed, embed, vh, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(c->arena + c->fx.lm_head, lm_head, vh, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(c->arena + c->fx.g_final, g_final, (size_t)c->H * 2, cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return c->cuda_fail(e, "globals upload");
    c->weights_loaded = true;
    return LOIP_OK;
}

extern "C" int loip_stream_layer(loip_ctx* c, int32_t layer, int32_t slot, void* copy_stream) {
    CTX_GUARD(c);
    if (layer < 0 || layer >= c->L || !c->offloaded[layer] || slot < 0 || slot >= c->cfg.n_slots ||
        c->off_order.empty() || !c->host_layer[layer])
        return c->fail(LOIP_ERR_INVALID, "layer is not offloaded or slot out of range");
    cudaStream_t s = copy_stream ? reinterpret_cast<cudaStream_t>(copy_stream) : c->copy;
    int rc = c->flush_inline();
    return rc ? rc : c->enqueue_copy(layer, slot, s);
}

extern "C" int loip_set_batch(loip_ctx* c, int32_t batch, const int32_t* ctx_lens) {
    CTX_GUARD(c);
    if (batch < 1 || batch > c->cfg.max_batch || !ctx_lens) return c->fail(LOIP_ERR_INVALID, "batch size");
    for (int b = 0; b < batch; ++b)
        if (ctx_lens[b] < 0 || ctx_lens[b] >= c->cfg.max_ctx) return c->fail(LOIP_ERR_INVALID, "context length");
    for (int b = 0; b < batch; ++b) {
        int rc = c->ensure_pages(b, ctx_lens[b]);
        if (rc) return rc;
        c->reqs[b].len = ctx_lens[b];
    }
    c->active_batch = batch;
    c->pos_dirty = true;
    return LOIP_OK;
}

extern "C" int loip_layer_forward(loip_ctx* c, int32_t layer, int32_t slot, float* hidden, const int32_t* positions,
                                  int32_t batch, void* compute_stream) {
    CTX_GUARD(c);
    if (layer < 0 || layer >= c->L || !hidden || !positions || batch < 1 || batch > c->cfg.max_batch)
        return c->fail(LOIP_ERR_INVALID, "layer_forward arguments");
    if (c->offloaded[layer] && (slot < 0 || slot >= c->cfg.n_slots))
        return c->fail(LOIP_ERR_INVALID, "offloaded layer needs its slot");
    cudaStream_t s = compute_stream ? reinterpret_cast<cudaStream_t>(compute_stream) : c->compute;
    int rc = c->upload_page_table(s);
    if (rc) return rc;
    float* x = c->fixed_ptr<float>(c->fx.x);
    cudaError_t e = cudaMemcpyAsync(x, hidden, (size_t)batch * c->H * 4, cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) return c->cuda_fail(e, "hidden copy");
    if (c->offloaded[layer] && c->packed(layer)) {
        rc = c->flush_inline();
        if (rc == LOIP_OK) rc = c->wait_packed_slot(slot, s);
        if (rc) return rc;
    } else if (c->offloaded[layer]) {
        e = cudaStreamWaitEvent(s, c->slot_full[slot], 0);
        if (e != cudaSuccess) return c->cuda_fail(e, "slot wait");
    }
    c->chain = false;
    rc = c->decode_layer(layer, batch, positions, s, slot);
    c->chain = false;
    if (rc) return rc;
    if (c->offloaded[layer]) cudaEventRecord(c->slot_free[slot], s);
    e = cudaMemcpyAsync(hidden, x, (size_t)batch * c->H * 4, cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) return c->cuda_fail(e, "hidden copy");
    return LOIP_OK;
}

// One decode step; tokens already on the device (d_tokens), results on device.
static int decode_step_enqueue(loip_ctx* c, const int32_t* d_tokens, int B, int32_t* d_out, float* out_hidden) {
    if (!c->weights_loaded) return c->fail(LOIP_ERR_STATE, "weights not loaded");
    if (B < 1 || B > c->cfg.max_batch) return c->fail(LOIP_ERR_INVALID, "batch size");
    if (B != c->active_batch) {
        // implicit batch: requests 0..B-1 keep their current lengths
        c->active_batch = B;
        c->pos_dirty = true;
    }
    for (int b = 0; b < B; ++b) {
        if (c->reqs[b].len + 1 > c->cfg.max_ctx) return c->fail(LOIP_ERR_INVALID, "context full");
        int rc = c->ensure_pages(b, c->reqs[b].len + 1);
        if (rc) return rc;
    }
    cudaStream_t s = c->compute;
    int rc = c->upload_page_table(s);
    if (rc) return rc;
    rc = c->upload_positions(B, s);
    if (rc) return rc;
    int32_t* pos = c->fixed_ptr<int32_t>(c->fx.dec_pos);
    cudaError_t e;
    cudaEventRecord(c->ev_step0, s);
    c->chain = false;
    float* x = c->fixed_ptr<float>(c->fx.x);
    e = launch_embed(c->embed_table(), d_tokens, B, c->H, c->V, x, s, false);
    if (e != cudaSuccess) return c->cuda_fail(e, "embed kernel");
    c->chain = true;
    // At batch 1 streamed layers unpack inline, on the compute stream (see
    // pump()).  Batched steps compute for much longer per layer (70B, batch 8:
    // 108 ms of kernels per step against 34 ms at batch 1), and inline unpacks
    // would hold the copies back behind them (the link fell to 166 GB/s): their
    // chunks unpack on the unpack stream, between the compute kernels.
    c->inline_unpack = c->packing && c->cfg.mode == LOIP_MODE_OVERLAP && B == 1;
    if (c->cfg.mode == LOIP_MODE_DIRECT)
        rc = c->run_layers_direct(B, pos, s);
    else
        rc = c->run_layers([&](int l, int slot) { return c->decode_layer(l, B, pos, s, slot); },
                           c->fuse_runs(B) ? pos : nullptr);
    if (rc) return rc;
    e = c->timed(5, s, [&] {
        return launch_lm_head(x, c->fixed_ptr<uint16_t>(c->fx.g_final), c->fixed_ptr<uint16_t>(c->fx.lm_head), B, c->H,
                              c->V, c->desc.rms_eps, out_hidden ? out_hidden : c->fixed_ptr<float>(c->fx.z),
                              c->fixed_ptr<float>(c->fx.logits), d_out, c->fixed_ptr<void>(c->fx.lm_scratch), s,
                              c->pdl());
    });
    if (e != cudaSuccess) return c->cuda_fail(e, "lm head kernel");
    e = launch_advance(pos, B, s, !c->ktiming);
    if (e != cudaSuccess) return c->cuda_fail(e, "position advance");
    if (c->run_launched) {  // the layer runs' barrier error word, checked at the next host sync point
        e = cudaMemcpyAsync(c->h_stage + c->h_stage_ints - 1, c->fixed_ptr<unsigned>(c->fx.run_sync) + 1, 4,
                            cudaMemcpyDeviceToHost, s);
        if (e != cudaSuccess) return c->cuda_fail(e, "error word download");
    }
    cudaEventRecord(c->ev_step1, s);
    c->chain = false;
    for (int b = 0; b < B; ++b) c->reqs[b].len += 1;
    c->st.steps += 1;
    c->st.tokens += B;
    return LOIP_OK;
}

extern "C" int loip_decode_step(loip_ctx* c, const int32_t* tokens, int32_t batch, int32_t* out_tokens,
                                float* out_hidden) {
    CTX_GUARD(c);
    if (!tokens || !out_tokens || batch < 1 || batch > c->cfg.max_batch)
        return c->fail(LOIP_ERR_INVALID, "decode_step arguments");
    for (int b = 0; b < batch; ++b)
        if (tokens[b] < 0 || tokens[b] >= c->V) return c->fail(LOIP_ERR_INVALID, "token id out of range");
    auto t0 = std::chrono::steady_clock::now();
    int32_t* hin = c->h_stage;
    int32_t* hout = c->h_stage + c->h_stage_ints / 4;
    int rc0 = c->wait_event(c->ev_stage);
    if (rc0) return rc0;
    memcpy(hin, tokens, (size_t)batch * 4);
    int32_t* d_tok = c->fixed_ptr<int32_t>(c->fx.tokens);
    int32_t* d_out = c->fixed_ptr<int32_t>(c->fx.out_tokens);
    cudaError_t e = cudaMemcpyAsync(d_tok, hin, (size_t)batch * 4, cudaMemcpyHostToDevice, c->compute);
    if (e != cudaSuccess) return c->cuda_fail(e, "token upload");
    cudaEventRecord(c->ev_stage, c->compute);
    int rc = decode_step_enqueue(c, d_tok, batch, d_out, out_hidden);
    if (rc) return rc;
    e = cudaMemcpyAsync(hout, d_out, (size_t)batch * 4, cudaMemcpyDeviceToHost, c->compute);
    if (e != cudaSuccess) return c->cuda_fail(e, "token download");
    e = cudaEventRecord(c->ev_done, c->compute);
    if (e != cudaSuccess) return c->cuda_fail(e, "event record");
    rc = c->wait_event(c->ev_done);
    if (rc) return rc;
    rc = c->check_run_error();
    if (rc) return rc;
    memcpy(out_tokens, hout, (size_t)batch * 4);
    c->collect_kernel_times();
    float ms = 0;
    cudaEventElapsedTime(&ms, c->ev_step0, c->ev_step1);
    c->st.compute_ms = ms;
    c->collect_copy_time();
    c->st.last_step_ms = std::chrono::duration<double, std::milli>(std::chrono::steady_clock::now() - t0).count();
    return LOIP_OK;
}

extern "C" int loip_decode_step_device(loip_ctx* c, const int32_t* tokens_dev, int32_t batch, int32_t* out_tokens_dev,
                                       float* out_hidden) {
    CTX_GUARD(c);
    if (!tokens_dev || !out_tokens_dev) return c->fail(LOIP_ERR_INVALID, "null pointer");
    int rc = decode_step_enqueue(c, tokens_dev, batch, out_tokens_dev, out_hidden);
    if (rc) return rc;
    c->collect_copy_time();
    c->collect_kernel_times();
    return LOIP_OK;
}

extern "C" int loip_prefill(loip_ctx* c, const int32_t* tokens, const int32_t* prompt_lens, int32_t n_prompts,
                            int32_t* out_tokens, float* out_hidden) {
    CTX_GUARD(c);
    if (!tokens || !prompt_lens || !out_tokens || n_prompts < 1 || n_prompts > c->cfg.max_batch)
        return c->fail(LOIP_ERR_INVALID, "prefill arguments");
    if (!c->weights_loaded) return c->fail(LOIP_ERR_STATE, "weights not loaded");
    int64_t M = 0;
    for (int i = 0; i < n_prompts; ++i) {
        if (prompt_lens[i] < 1 || prompt_lens[i] > c->cfg.max_ctx) return c->fail(LOIP_ERR_INVALID, "prompt length");
        M += prompt_lens[i];
    }
    for (int64_t t = 0; t < M; ++t)
        if (tokens[t] < 0 || tokens[t] >= c->V) return c->fail(LOIP_ERR_INVALID, "token id out of range");
    auto t0 = std::chrono::steady_clock::now();
    int rc = c->sync_all();
    if (rc) return rc;
    // the GEMMs hold every SM for ms at a time: streamed layers unpack on their own stream
    c->inline_unpack = false;
    rc = c->flush_inline();
    if (rc) return rc;
    for (int i = 0; i < n_prompts; ++i) {
        c->release_pages(i);
        rc = c->ensure_pages(i, prompt_lens[i]);
        if (rc) return rc;
    }
    cudaStream_t s = c->compute;
    rc = c->upload_page_table(s);
    if (rc) return rc;
    const int Mp = c->cfg.max_prefill_tokens;
    const int tile_pos = attention_tc_tile_positions(c->Hq, c->Hkv);  // positions per attention tile
    // per-token request and position
    std::vector<int32_t> req_of(M), pos_of(M);
    std::vector<int32_t> last_row(n_prompts);
    {
        int64_t t = 0;
        for (int i = 0; i < n_prompts; ++i)
            for (int p = 0; p < prompt_lens[i]; ++p, ++t) {
                req_of[t] = i;
                pos_of[t] = p;
                if (p == prompt_lens[i] - 1) last_row[i] = (int32_t)t;
            }
    }
    float* x = c->fixed_ptr<float>(c->fx.x);
    cudaEventRecord(c->ev_step0, s);
    for (int64_t c0 = 0; c0 < M; c0 += Mp) {
        const int Mc = (int)std::min<int64_t>(Mp, M - c0);
        int32_t* h = c->h_stage;
        // staging: tokens | positions | requests
        rc = c->wait_event(c->ev_stage);  // previous chunk's uploads have been consumed
        if (rc) return rc;
        memcpy(h, tokens + c0, (size_t)Mc * 4);
        memcpy(h + Mc, pos_of.data() + c0, (size_t)Mc * 4);
        memcpy(h + 2 * Mc, req_of.data() + c0, (size_t)Mc * 4);
        // attention query tiles: runs of at most P_T consecutive rows of one request
        int32_t* ht = h + 3 * Mc;
        c->prefill_tiles = 0;
        for (int i = 0; i < Mc;) {
            int n = 1;
            while (i + n < Mc && n < tile_pos && req_of[c0 + i + n] == req_of[c0 + i]) ++n;
            ht[4 * c->prefill_tiles + 0] = i;
            ht[4 * c->prefill_tiles + 1] = n;
            ht[4 * c->prefill_tiles + 2] = req_of[c0 + i];
            ht[4 * c->prefill_tiles + 3] = pos_of[c0 + i];
            ++c->prefill_tiles;
            i += n;
        }
        cudaError_t e = cudaMemcpyAsync(c->arena + c->fx.tokens, h, (size_t)Mc * 4, cudaMemcpyHostToDevice, s);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(c->arena + c->fx.positions, h + Mc, (size_t)Mc * 4, cudaMemcpyHostToDevice, s);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(c->arena + c->fx.row_req, h + 2 * Mc, (size_t)Mc * 4, cudaMemcpyHostToDevice, s);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(c->arena + c->fx.ptiles, ht, (size_t)c->prefill_tiles * 16, cudaMemcpyHostToDevice, s);
        if (e != cudaSuccess) return c->cuda_fail(e, "prefill upload");
        cudaEventRecord(c->ev_stage, s);
        e = launch_embed(c->embed_table(), c->fixed_ptr<int32_t>(c->fx.tokens), Mc, c->H, c->V,
                         c->fixed_ptr<float>(c->fx.px), s);
        if (e != cudaSuccess) return c->cuda_fail(e, "embed kernel");
        rc = c->run_layers([&](int l, int slot) { return c->prefill_layer(l, Mc, s, slot); });
        if (rc) return rc;
        // final rows of prompts ending in this chunk -> decode activations
        for (int i = 0; i < n_prompts; ++i) {
            if (last_row[i] < c0 || last_row[i] >= c0 + Mc) continue;
            e = cudaMemcpyAsync(x + (size_t)i * c->H, c->fixed_ptr<float>(c->fx.px) + (size_t)(last_row[i] - c0) * c->H,
                                (size_t)c->H * 4, cudaMemcpyDeviceToDevice, s);
            if (e != cudaSuccess) return c->cuda_fail(e, "row copy");
        }
    }
    int32_t* d_out = c->fixed_ptr<int32_t>(c->fx.out_tokens);
    cudaError_t e = launch_lm_head(x, c->fixed_ptr<uint16_t>(c->fx.g_final), c->fixed_ptr<uint16_t>(c->fx.lm_head),
                                   n_prompts, c->H, c->V, c->desc.rms_eps,
                                   out_hidden ? out_hidden : c->fixed_ptr<float>(c->fx.z),
                                   c->fixed_ptr<float>(c->fx.logits), d_out, c->fixed_ptr<void>(c->fx.lm_scratch), s);
    if (e != cudaSuccess) return c->cuda_fail(e, "lm head kernel");
    cudaEventRecord(c->ev_step1, s);
    int32_t* hout = c->h_stage + c->h_stage_ints / 4;
    e = cudaMemcpyAsync(hout, d_out, (size_t)n_prompts * 4, cudaMemcpyDeviceToHost, s);
    if (e != cudaSuccess) return c->cuda_fail(e, "token download");
    cudaEventRecord(c->ev_done, s);
    rc = c->wait_event(c->ev_done);
    if (rc) return rc;
    c->collect_kernel_times();
    int tcerr = 0, aterr = 0;
    if (tc_error(&tcerr) != cudaSuccess || tcerr != 0) {
        c->failed = true;
        return c->fail(LOIP_ERR_TIMEOUT, "tensor-core GEMM pipeline did not complete (code " + std::to_string(tcerr) + ")");
    }
    if (attention_tc_error(&aterr) != cudaSuccess || aterr != 0) {
        c->failed = true;
        return c->fail(LOIP_ERR_TIMEOUT, "tensor-core attention did not complete (code " + std::to_string(aterr) + ")");
    }
    memcpy(out_tokens, hout, (size_t)n_prompts * 4);
    for (int i = 0; i < n_prompts; ++i) c->reqs[i].len = prompt_lens[i];
    c->active_batch = n_prompts;
    c->pos_dirty = true;
    float ms = 0;
    cudaEventElapsedTime(&ms, c->ev_step0, c->ev_step1);
    c->st.compute_ms = ms;
    c->collect_copy_time();
    c->st.last_step_ms = std::chrono::duration<double, std::milli>(std::chrono::steady_clock::now() - t0).count();
    return LOIP_OK;
}

extern "C" int32_t loip_get_copy_log(loip_ctx* c, double* ms, uint64_t* bytes, int32_t max_n) {
    if (!c || max_n < 0 || (max_n > 0 && (!ms || !bytes))) return -1;
    c->collect_copy_time();
    const size_t have = std::min<size_t>(c->copy_log_next, loip_ctx::kCopyLog);
    const size_t n = std::min<size_t>(have, (size_t)max_n);
    for (size_t i = 0; i < n; ++i) {  // oldest of the last n first
        const auto& e = c->copy_log[(c->copy_log_next - n + i) % loip_ctx::kCopyLog];
        ms[i] = e.first;
        bytes[i] = e.second;
    }
    return (int32_t)n;
}

extern "C" int loip_get_pool_nodes(loip_ctx* c, int32_t* nodes) {
    if (!c || !nodes) return LOIP_ERR_INVALID;
    for (int l = 0; l < c->L; ++l) nodes[l] = l < (int)c->pool_node.size() ? c->pool_node[l] : -1;
    return LOIP_OK;
}

extern "C" int loip_inject_fault(loip_ctx* c, int32_t kind, int32_t arg) {
    CTX_GUARD(c);
    if (kind != LOIP_FAULT_NONE && kind != LOIP_FAULT_WAIT && kind != LOIP_FAULT_COPY &&
        kind != LOIP_FAULT_HOST_ALLOC && kind != LOIP_FAULT_BARRIER)
        return c->fail(LOIP_ERR_INVALID, "fault kind");
    if (kind == LOIP_FAULT_BARRIER && arg < 0) return c->fail(LOIP_ERR_INVALID, "fault block");
    c->fault_kind = kind;
    c->fault_arg = arg;
    return LOIP_OK;
}

extern "C" int loip_poll_deadline_check(uint32_t timeout_ms, int32_t pending_polls, double* waited_ms) {
    int32_t polls = 0;
    bool timed_out = false;
    const cudaError_t r = poll_until(
        [&] {
            if (pending_polls >= 0 && polls >= pending_polls) return cudaSuccess;
            ++polls;
            return cudaErrorNotReady;
        },
        timeout_ms, &timed_out, waited_ms);
    if (timed_out) return LOIP_ERR_TIMEOUT;
    return r == cudaSuccess ? LOIP_OK : LOIP_ERR_CUDA;
}

extern "C" int loip_replan(loip_ctx* c, int32_t lookahead_tokens) {
    CTX_GUARD(c);
    if (lookahead_tokens < 0) return c->fail(LOIP_ERR_INVALID, "lookahead");
    // pages the active requests need for the lookahead
    uint64_t need = 0;
    for (int b = 0; b < c->active_batch; ++b) {
        int tokens = std::min(c->reqs[b].len + lookahead_tokens, c->cfg.max_ctx);
        int pages = (tokens + c->cfg.page_tokens - 1) / c->cfg.page_tokens;
        need += (uint64_t)std::max(0, pages - (int)c->reqs[b].pages.size());
    }
    while (c->free_groups.size() < need) {
        if (c->grow_kv() >= 0) continue;
        int rc = c->demote_for_kv(need - c->free_groups.size());
        if (rc) return rc;
    }
    return LOIP_OK;
}

extern "C" int loip_get_stats(const loip_ctx* c, loip_stats* out) {
    if (!c || !out) return LOIP_ERR_INVALID;
    *out = c->st;
    out->n_offloaded = (int)c->off_order.size();
    out->n_resident = c->L - out->n_offloaded;
    uint64_t toks = 0;
    uint64_t pages = 0;
    for (auto& r : c->reqs) {
        toks += r.len;
        pages += r.pages.size();
    }
    out->kv_tokens = toks;
    out->kv_bytes = pages * c->group_bytes;
    out->arena_used = c->arena_used();
    return LOIP_OK;
}

extern "C" int loip_synchronize(loip_ctx* c) {
    if (!c) return LOIP_ERR_INVALID;
    int rc = c->sync_all();
    if (rc == LOIP_OK) rc = c->check_run_error();
    c->collect_copy_time();
    c->collect_kernel_times();
    return rc;
}

extern "C" int loip_set_kernel_timing(loip_ctx* c, int32_t enable) {
    CTX_GUARD(c);
    int rc = c->sync_all();
    if (rc) return rc;
    c->collect_kernel_times();
    for (int i = 0; i < 16; ++i) {
        c->st.kernel_ms[i] = 0;
        c->st.kernel_launches[i] = 0;
    }
    c->ktiming = enable != 0;
    return LOIP_OK;
}

extern "C" int loip_measure_h2d(uint64_t bytes, int32_t reps, double* out_Bps) {
    if (!out_Bps || bytes < (1u << 20) || reps < 1) return LOIP_ERR_INVALID;
    HostBuf hb;
    if (host_buf_alloc(bytes, &hb) != cudaSuccess) return LOIP_ERR_OOM;
    memset(hb.ptr, 1, bytes);
    void* d = nullptr;
    cudaStream_t s = nullptr;
    cudaEvent_t a = nullptr, b = nullptr;
    cudaError_t e = cudaMalloc(&d, bytes);
    if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&s, cudaStreamNonBlocking);
    if (e == cudaSuccess) e = cudaEventCreate(&a);
    if (e == cudaSuccess) e = cudaEventCreate(&b);
    double best = 0;
    for (int r = 0; r < reps + 1 && e == cudaSuccess; ++r) {
        cudaEventRecord(a, s);
        e = cudaMemcpyAsync(d, hb.ptr, bytes, cudaMemcpyHostToDevice, s);
        cudaEventRecord(b, s);
        if (e == cudaSuccess) e = cudaEventSynchronize(b);
        float ms = 0;
        if (e == cudaSuccess && r > 0 && cudaEventElapsedTime(&ms, a, b) == cudaSuccess && ms > 0)
            best = std::max(best, (double)bytes / (ms * 1e-3));
    }
    if (a) cudaEventDestroy(a);
    if (b) cudaEventDestroy(b);
    if (s) cudaStreamDestroy(s);
    if (d) cudaFree(d);
    host_buf_free(&hb);
    if (e != cudaSuccess) return LOIP_ERR_CUDA;
    *out_Bps = best;
    return LOIP_OK;
}

extern "C" int loip_measure_direct_read(uint64_t bytes, int32_t reps, double* out_Bps) {
    if (!out_Bps || bytes < (1u << 20) || (bytes & 15) || reps < 1) return LOIP_ERR_INVALID;
    HostBuf hb;
    if (host_buf_alloc(bytes, &hb) != cudaSuccess) return LOIP_ERR_OOM;
    if (!hb.dev) {
        host_buf_free(&hb);
        return LOIP_ERR_CUDA;
    }
    memset(hb.ptr, 1, bytes);
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int blocks = std::max(1, sms) * 4;
    uint32_t* sink = nullptr;
    cudaStream_t s = nullptr;
    cudaEvent_t a = nullptr, b = nullptr;
    cudaError_t e = cudaMalloc(&sink, (size_t)blocks * sizeof(uint32_t));
    if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&s, cudaStreamNonBlocking);
    if (e == cudaSuccess) e = cudaEventCreate(&a);
    if (e == cudaSuccess) e = cudaEventCreate(&b);
    double best = 0;
    for (int r = 0; r < reps + 1 && e == cudaSuccess; ++r) {
        cudaEventRecord(a, s);
        e = launch_read_stream(hb.dev, bytes, blocks, sink, s);
        cudaEventRecord(b, s);
        if (e == cudaSuccess) e = cudaEventSynchronize(b);
        float ms = 0;
        if (e == cudaSuccess && r > 0 && cudaEventElapsedTime(&ms, a, b) == cudaSuccess && ms > 0)
            best = std::max(best, (double)bytes / (ms * 1e-3));
    }
    if (a) cudaEventDestroy(a);
    if (b) cudaEventDestroy(b);
    if (s) cudaStreamDestroy(s);
    if (sink) cudaFree(sink);
    host_buf_free(&hb);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return LOIP_ERR_CUDA;
    }
    *out_Bps = best;
    return LOIP_OK;
}

extern "C" void* loip_compute_stream(loip_ctx* c) { return c ? (void*)c->compute : nullptr; }
extern "C" void* loip_copy_stream(loip_ctx* c) { return c ? (void*)c->copy : nullptr; }

// ============================================================================
// Kernel-level entry points
// ============================================================================
static bool al16(const void* p) { return ((uintptr_t)p & 15) == 0; }
static int cerr(cudaError_t e) {
    if (e == cudaSuccess) return LOIP_OK;
    g_create_error = std::string("kernel launch: ") + cudaGetErrorString(e);  // loip_last_error(NULL)
    cudaGetLastError();  // leave no non-sticky error behind for the next call
    return LOIP_ERR_CUDA;
}

extern "C" int loip_k_generate(uint16_t* out, uint64_t n, uint64_t first, uint64_t seed, uint32_t tensor_id,
                               int32_t kind, void* stream) {
    if ((!out && n) || (kind != 0 && kind != 1) || first + n > (1ull << 40)) return LOIP_ERR_INVALID;
    return cerr(launch_generate(out, n, first, seed, tensor_id, kind, (cudaStream_t)stream));
}

extern "C" int loip_k_embed(const uint16_t* embed, const int32_t* tokens, int32_t B, int32_t H, float* x,
                            void* stream) {
    if (!embed || !tokens || !x || B < 1 || H < 1) return LOIP_ERR_INVALID;
    return cerr(launch_embed(embed, tokens, B, H, 1 << 30, x, (cudaStream_t)stream));
}

extern "C" int loip_k_qkv_rope(const float* x, const uint16_t* g, const uint16_t* wqkv, int32_t B, int32_t H,
                               int32_t Hq, int32_t Hkv, int32_t d, float eps, float theta, const int32_t* positions,
                               float* q_out, const void* kv_base, const int64_t* page_offsets, int32_t max_pages,
                               int32_t page_tokens, int32_t layer, uint64_t layer_page_bytes, void* stream) {
    if (!x || !g || !wqkv || !positions || !q_out || !kv_base || !page_offsets || B < 1 || B > 8 || H % 8 ||
        (d != 64 && d != 128) || Hq % Hkv || page_tokens < 1 || !al16(wqkv) || !al16(x) || !al16(g))
        return LOIP_ERR_INVALID;
    KvView kv{(char*)kv_base, page_offsets, max_pages, page_tokens, layer, layer_page_bytes};
    return cerr(launch_qkv_rope(x, g, wqkv, B, H, Hq, Hkv, d, eps, theta, positions, q_out, kv, nullptr,
                                (cudaStream_t)stream));
}

extern "C" uint64_t loip_k_attention_scratch_floats(int32_t B, int32_t Hq, int32_t d, int32_t max_ctx,
                                                    int32_t page_tokens) {
    if (B < 1 || Hq < 1 || d < 1 || max_ctx < 1 || page_tokens < 1) return 0;
    return attention_scratch_floats(B, Hq, d, max_ctx, page_tokens);
}

extern "C" int loip_k_attention(const float* q, const void* kv_base, const int64_t* page_offsets, int32_t max_pages,
                                const int32_t* ctx_lens, int32_t B, int32_t Hq, int32_t Hkv, int32_t d,
                                int32_t page_tokens, int32_t layer, uint64_t layer_page_bytes, int32_t max_ctx,
                                float* scratch, float* o, void* stream) {
    if (!q || !kv_base || !page_offsets || !ctx_lens || !scratch || !o || B < 1 || (d != 64 && d != 128) ||
        Hq % Hkv || max_ctx < 1 || page_tokens != 64 || (int64_t)max_pages * page_tokens < max_ctx || !al16(q) ||
        ((uintptr_t)kv_base & 15))
        return LOIP_ERR_INVALID;
    if ((max_ctx + page_tokens - 1) / page_tokens > 256) return LOIP_ERR_INVALID;
    KvView kv{(char*)kv_base, page_offsets, max_pages, page_tokens, layer, layer_page_bytes};
    cudaError_t e = cudaMemsetAsync(attention_counters(scratch, B, Hq, d, max_ctx, page_tokens), 0,
                                    (size_t)B * Hq * sizeof(int), (cudaStream_t)stream);
    if (e != cudaSuccess) return LOIP_ERR_CUDA;
    return cerr(launch_attention(q, kv, ctx_lens, nullptr, nullptr, B, Hq, Hkv, d, max_ctx, true, scratch, o, false,
                                 (cudaStream_t)stream, false, 0, true));
}

extern "C" int loip_k_prefill_attention(const float* q, const void* kv_base, const int64_t* page_offsets,
                                        int32_t max_pages, const int32_t* prompt_lens, const int32_t* first_pos,
                                        int32_t n_prompts, int32_t Hq, int32_t Hkv, int32_t d, int32_t page_tokens,
                                        int32_t layer, uint64_t layer_page_bytes, void* tiles, uint16_t* o2,
                                        void* stream) {
    if (!q || !kv_base || !page_offsets || !prompt_lens || !tiles || !o2 || n_prompts < 1 || Hq < 1 || Hkv < 1 ||
        (d != 64 && d != 128) || Hq % Hkv || page_tokens != 64 || max_pages < 1 || !al16(q) || !al16(kv_base) ||
        !al16(o2) || !al16(tiles))
        return LOIP_ERR_INVALID;
    const int G = Hq / Hkv;
    if (G != 1 && G != 2 && G != 4 && G != 8) return LOIP_ERR_INVALID;
    const int tp = attention_tc_tile_positions(Hq, Hkv);
    std::vector<int4> t;
    int M = 0;
    for (int i = 0; i < n_prompts; ++i) {
        const int len = prompt_lens[i], p0 = first_pos ? first_pos[i] : 0;
        if (len < 1 || p0 < 0 || (int64_t)p0 + len > (int64_t)max_pages * page_tokens) return LOIP_ERR_INVALID;
        for (int j = 0; j < len; j += tp) t.push_back(make_int4(M + j, std::min(tp, len - j), i, p0 + j));
        M += len;
    }
    KvView kv{(char*)kv_base, page_offsets, max_pages, page_tokens, layer, layer_page_bytes};
    cudaError_t e = cudaMemcpyAsync(tiles, t.data(), t.size() * sizeof(int4), cudaMemcpyHostToDevice,
                                    (cudaStream_t)stream);
    if (e != cudaSuccess) return cerr(e);
    return cerr(launch_attention_tc(q, kv, static_cast<const int4*>(tiles), (int)t.size(), M, Hq, Hkv, d, o2,
                                    (cudaStream_t)stream));
}

extern "C" int loip_k_attention_tc_status(void) {
    int code = 0;
    if (attention_tc_error(&code) != cudaSuccess) return -1;
    return code;
}

extern "C" int loip_k_oproj(const float* o, const uint16_t* wo, int32_t B, int32_t H, int32_t K, float* x,
                            void* stream) {
    if (!o || !wo || !x || B < 1 || B > 8 || K % 8 || H < 1 || !al16(wo) || !al16(o)) return LOIP_ERR_INVALID;
    return cerr(launch_resid_gemv(o, wo, B, H, K, x, (cudaStream_t)stream, false, false, true));
}

extern "C" int loip_k_gate_up(const float* x, const uint16_t* g, const uint16_t* wg, const uint16_t* wu, int32_t B,
                              int32_t H, int32_t F, float eps, float* a, void* stream) {
    if (!x || !g || !wg || !wu || !a || B < 1 || B > 8 || H % 8 || F < 1 || !al16(wg) || !al16(wu) || !al16(x) ||
        !al16(g))
        return LOIP_ERR_INVALID;
    return cerr(launch_gate_up(x, g, wg, wu, B, H, F, eps, a, (cudaStream_t)stream));
}

extern "C" int loip_k_down(const float* a, const uint16_t* wd, int32_t B, int32_t H, int32_t F, float* x,
                           void* stream) {
    if (!a || !wd || !x || B < 1 || B > 8 || F % 8 || H < 1 || !al16(wd) || !al16(a)) return LOIP_ERR_INVALID;
    return cerr(launch_resid_gemv(a, wd, B, H, F, x, (cudaStream_t)stream));
}

extern "C" int loip_k_gemm_bf16(const uint16_t* A, const uint16_t* W, int32_t M, int32_t N, int32_t K, float* x,
                                void* stream) {
    if (!A || !W || !x || M < 1 || N < 1 || K < 8 || K % 8 || !al16(A) || !al16(W) || !al16(x) || N % 4)
        return LOIP_ERR_INVALID;
    return cerr(launch_tc_gemm_resid(A, false, W, M, N, K, x, (cudaStream_t)stream));
}

extern "C" int loip_k_gemm_split(const uint16_t* A2, const uint16_t* W, int32_t M, int32_t N, int32_t K, float* x,
                                 void* stream) {
    // the lo plane starts M * K elements after the hi plane: 16-byte aligned too
    if (!A2 || !W || !x || M < 1 || N < 1 || K < 8 || K % 8 || !al16(A2) || !al16(W) || !al16(x) || N % 4)
        return LOIP_ERR_INVALID;
    return cerr(launch_tc_gemm_resid(A2, true, W, M, N, K, x, (cudaStream_t)stream));
}

extern "C" int loip_k_pack(const uint16_t* in, uint64_t n_sb, uint8_t* out, uint32_t* raw_list, uint32_t first_sb,
                           uint32_t raw_cap, void* stream) {
    if ((!in || !out) && n_sb) return LOIP_ERR_INVALID;
    if (!al16(in) || !al16(out) || n_sb > (1ull << 32)) return LOIP_ERR_INVALID;
    return cerr(launch_pack(in, n_sb, out, raw_list, first_sb, raw_cap, (cudaStream_t)stream));
}

extern "C" int loip_k_unpack(const uint8_t* in, uint64_t n_sb, uint16_t* out, void* stream) {
    if ((!in || !out) && n_sb) return LOIP_ERR_INVALID;
    if (!al16(in) || !al16(out)) return LOIP_ERR_INVALID;
    return cerr(launch_unpack(in, n_sb, out, (cudaStream_t)stream));
}

extern "C" int loip_k_tc_status(void) {
    int code = 0;
    if (tc_error(&code) != cudaSuccess) return -1;
    return code;
}

extern "C" uint64_t loip_k_lm_head_scratch_bytes(int32_t B, int32_t V) {
    if (B < 1 || V < 1) return 0;
    return lm_head_scratch_bytes(B, V);
}

extern "C" int loip_k_lm_head(const float* x, const uint16_t* g_final, const uint16_t* lm_head, int32_t B, int32_t H,
                              int32_t V, float eps, float* z, float* logits, int32_t* tokens, void* scratch,
                              void* stream) {
    if (!x || !g_final || !lm_head || !tokens || !scratch || B < 1 || B > 8 || H % 8 || V < 1 || !al16(lm_head) ||
        !al16(x) || !al16(g_final))
        return LOIP_ERR_INVALID;
    return cerr(launch_lm_head(x, g_final, lm_head, B, H, V, eps, z, logits, tokens, scratch, (cudaStream_t)stream));
}
