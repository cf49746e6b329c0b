// ra_internal.h -- launch parameters and launchers shared by the library's own
// translation units (host API in ra_api.cu; kernels in ra_evict.cu, ra_attn.cu).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

#include "ra.h"

namespace ra {

constexpr int kHeadDim = 128;            // d; one K or V row is 256 bytes of bf16
constexpr int kRowBytes = kHeadDim * 2;
constexpr int kMaxG = 8;                 // query heads per KV head supported by the kernels
constexpr int kPlanHeader = 8;           // int32 words before the evicted-ordinal list
constexpr int kMaxCandidates = 32768;    // K + r bound (select keeps one u32 key per candidate in smem)
// Split-K partial record of one (warp, KV head) piece: o[G][128], m[G], l[G] in fp32,
// padded to a multiple of 4 floats so that every record starts 16-byte aligned.
__host__ __device__ constexpr int partial_stride(int G) { return G * 128 + ((2 * G + 3) / 4) * 4; }
// Prompt rows live in pages of kPromptPage positions x all KV heads of one sequence (a multiple of
// every kernel's tile height: 48 and 32 rows for attention, 64 for scoring), listed per sequence
// in a page table, so that a finished sequence's slot can take a new request of another length.
constexpr int kPromptPage = 192;
constexpr int kDeviceErrTimeout = 1;     // values of the device error word
constexpr int kDeviceErrPlan = 2;

// Pointers into the bound arena plus the static shape of a context.
struct DevLayout {
    uint16_t* kpool;       // [total_rows][128] bf16: prompt rows of every layer, then generated regions
    uint16_t* vpool;
    int32_t* pos;          // [regions][Cmax] positions of generated slots
    int32_t* region;       // [L][B][KVH] region index currently holding a head's generated slots
    int32_t* spare;        // [B][KVH] the free region that a head's next compaction writes into
    int32_t* seq_lp;       // [B] prompt length
    int32_t* pages;        // [B][max_pages] page of each kPromptPage-position block of a sequence's prompt
    int32_t* plan;         // [B*KVH][kPlanHeader + r] eviction plan of the current layer
    float* partial;        // attention split partials
    int32_t* arrive;       // [B*KVH] split-piece arrival counters
    int32_t* err;          // device error word
    int32_t* evplan;       // [2][L][B][KVH][r + 1] evicted sets computed ahead (plan_kernel)
    // scored policy (null when the context was bound without its buffers)
    uint16_t* qring;       // [L][B][KVH][r][G][128] bf16: query of step s in slot (s - 1) mod r
    float* scores;         // [L][B][KVH][Cmax] raw window score of each candidate of the latest round
    float2* qstats;        // [L][B][KVH][r][G] per window query: (its scale * log2 e, log2 of its softmax sum)
    float* stats;          // [B*KVH][stats_chunks][M][2] restore pass: softmax statistics (max, sum) per chunk
    int stats_chunks;      // chunks per head the stats buffer holds
    long long prompt_rows_per_layer;  // pool pages * KVH * kPromptPage
    int max_pages;
    long long gen_row0;    // first row of the generated regions
    int L, B, KVH, H, G, Cmax, K, r;
    uint64_t seed;
};

// Per-sequence counts come from the host mirror (the single source of truth) as launch parameters.
struct AppendParams {
    DevLayout lay;
    int layer;
    const uint16_t* k_new;  // [B][KVH][128]
    const uint16_t* v_new;
    uint32_t active[RA_MAX_BATCH / 32];
    int32_t seq_c[RA_MAX_BATCH];  // cached generated rows before the append
    int32_t seq_g[RA_MAX_BATCH];  // generated tokens before the append (position = lp + g)
};

struct EvictParams {
    DevLayout lay;
    int layer;
    int policy;    // RA_POLICY_*: how candidates are scored
    int block;     // RA_POLICY_BLOCK: positions per block
    int holefill;  // RA_COMPACT_HOLEFILL: keys per position, evicted slots refilled in place by select
    int early;     // select may compute before its predecessor finishes (it writes only after the wait)
    // Hole-filling with the step's token still pending (the fused step): the cache holds trig_c
    // rows and the token is appended afterwards, into the new last slot; 0: the token is cached.
    int pending;
    int n_trig;
    int16_t trig[RA_MAX_BATCH];    // triggered sequence ids
    int32_t trig_c[RA_MAX_BATCH];  // rows in the cache (a pending new token is not among them)
    int32_t trig_n[RA_MAX_BATCH];  // candidates (all rows but the newest r, counting a pending token)
    int32_t trig_g[RA_MAX_BATCH];  // step of the draw: generated tokens including this step's
    // the host's mirror of the region tables: the triggered sequence's current region and its
    // spare are region_base * KVH + kv_head (one-launch eviction; checked against the tables)
    int32_t trig_src[RA_MAX_BATCH];
    int32_t trig_dst[RA_MAX_BATCH];
    // requests admitted into the slot before the current one: the key stream of a head is
    // (admissions << 16) | head id, so that a new request draws its own numbers
    uint16_t trig_admit[RA_MAX_BATCH];
    // scored policy: tiles (of kScoreTile rows) per CTA of each pass, CTAs per head of each pass
    int ch1, ch2, nch1, nch2;
    float qk_scale_log2;  // restore pass: the scale * log2 e the restored queries are taken at
    // one-launch eviction: clusters per head (each selects on its own, the copy is split over
    // all of them) and whether to skip the sampled cut (exact radix passes only)
    int ev_reps;
    int ev_exact;
    // evicted sets computed ahead by plan_kernel ([2][L][B][KVH][r + 1]: count, then the ordinals
    // ascending) and which half this launch reads; null: the kernel selects itself
    const int32_t* ev_plan;
    int ev_plan_parity;
};

constexpr int kScoreTile = 64;      // key rows per scoring tile
constexpr int kScoreMaxRows = 512;  // r * G window rows the scoring kernels hold
constexpr int kScorePoolRadius = 3; // max-pool width 7 over neighbouring candidates
constexpr int kScoreMaxCandidates = 16384;  // K + r bound of the scored policy (select stages the scores too)

// Attention work is counted in tiles of TILE rows: a head has ceil(lp / TILE) prompt tiles and
// ceil(gen / TILE) tiles of generated rows (gen includes a fused new token, its last row).
struct AttnParams {
    DevLayout lay;
    int layer;
    int tile;               // rows per tile
    const uint16_t* q;      // [B][H][128]
    uint16_t* out;          // [B][H][128]
    const uint16_t* k_new;  // fused append: the step's new rows [B][KVH][128]; null = attention only
    const uint16_t* v_new;
    float* partial;         // split-K partial records (arena or the no-alloc array)
    int32_t* arrive;        // [B*KVH] pieces merged so far per head; zero between launches
    int W;                  // tiles per chunk of the split: warp w takes tiles [w W, (w + 1) W)
    int total;              // total tiles of the layer
    int nchunks;            // ceil(total / W)
    int nwarps;             // warps launched
    float qk_scale_log2;    // scale * log2(e)
    int early;              // 1: the first tiles' K/V may be loaded before the predecessor kernel finishes
    uint32_t active[RA_MAX_BATCH / 32];
    int32_t seq_base[RA_MAX_BATCH + 1];  // KVH * prefix of tiles per head over active sequences
    int32_t seq_gen[RA_MAX_BATCH];       // generated rows attended per head (incl. a fused new token)
    int32_t seq_g[RA_MAX_BATCH];         // tokens generated before this step's (fused) / up to it (separate)
    // From the host mirror, so that entering a head needs no load from memory: the prompt length,
    // the first prompt page when the sequence's pages are consecutive (-1: walk the page table), and
    // this layer's region base (the region of KV head h is base * KVH + h)
    int32_t seq_lp[RA_MAX_BATCH];
    int32_t seq_page0[RA_MAX_BATCH];
    int32_t seq_region[RA_MAX_BATCH];
    uint32_t pending[RA_MAX_BATCH / 32]; // fused step: sequences whose new token this kernel appends
    // fused step: sequences that evicted this step and whose compaction this kernel does -- it reads
    // their old regions (plan header), masks the evicted rows and writes every survivor (and the new
    // token) to its slot in the new region (time order kept)
    uint32_t compacting[RA_MAX_BATCH / 32];
    uint16_t* qring;                     // record each head's query rows in the scored policy's window (or null)
    int ring_off;                        // window slot of sequence b = (seq_g[b] + ring_off) mod r
};

struct CopyRowsParams {
    DevLayout lay;
    int layer;
    const uint16_t* k;  // [B][KVH][row_stride][128] (one sequence's [KVH][row_stride][128] when only_seq >= 0)
    const uint16_t* v;
    const int32_t* pos; // restore only: [B][KVH][row_stride]
    int row_stride;
    int only_seq;       // >= 0: the launch copies that sequence alone (one CTA per KV head)
    int32_t n_rows[RA_MAX_BATCH];  // rows to copy per sequence
};

// Cache row of prompt position `pos` of (layer, KV head h) in `page` (the sequence's page-table
// entry for block pos / kPromptPage).
__host__ __device__ inline long long prompt_row(const DevLayout& L, int layer, int32_t page, int h, int pos)
{
    return (long long)layer * L.prompt_rows_per_layer + ((long long)page * L.KVH + h) * kPromptPage + pos % kPromptPage;
}
__host__ __device__ inline uint32_t key_stream(uint32_t admissions, uint32_t head) { return (admissions << 16) | head; }

// Launchers (return cudaError_t of the launch).
cudaError_t launch_append(const AppendParams& p, int B, cudaStream_t s);
cudaError_t launch_select(const EvictParams& p, cudaStream_t s);
size_t select_smem(int N, int r, bool scored);  // dynamic shared memory of one select CTA
constexpr size_t kSelectSmemLimit = 220 * 1024;
cudaError_t launch_compact(const EvictParams& p, cudaStream_t s);
// Selection and order-preserving compaction in one launch, p.ev_reps clusters of `cluster` CTAs
// per triggered head (random, shared, recency and block policies; ordered compaction).  Each
// CTA holds the keys of at most kEvMaxLocal candidates: cluster >= ceil((K + r) / kEvMaxLocal).
constexpr int kEvMaxLocal = 2112;
constexpr int kEvMaxCluster = 16;
constexpr int kEvMaxEvicted = 512;  // r bound of the one-launch path (the evicted list lives in shared memory)
constexpr int kEvRows = 16;  // rows per copy buffer (8 KB of K and V)
constexpr int kEvBufs = 3;   // copy buffers per warp: 192 KB per CTA, one CTA per SM
cudaError_t launch_evict(const EvictParams& p, int cluster, cudaStream_t s);
// The evicted sets of the triggered sequences' heads in every layer, from the counters alone
// (the random draw reads no cache data), into half p.ev_plan_parity of lay.evplan; one warp per
// CTA, at most `sms` CTAs looping over the (layer, sequence, KV head) items, little shared memory,
// so that it runs beside the attention kernel.
cudaError_t launch_plan(const EvictParams& p, int sms, cudaStream_t s);
// Every layer's round of the triggered sequences (layers 0 .. layers - 1, counters alike in every
// layer), in place, from the evicted sets in half p.ev_plan_parity of lay.evplan: one CTA per
// (layer, sequence, KV head).
cudaError_t launch_compact_stack(const EvictParams& p, int layers, cudaStream_t s);
// The same rounds with order-free slots: the evicted slots of every layer refilled in place from
// the newest ones, the step's token (p.k_new / p.v_new: [layers][B][KVH][d]) included.
cudaError_t launch_fill_stack(const EvictParams& p, int layers, cudaStream_t s);
// One-time attributes; active[cl] (cl = 0..kEvMaxCluster) = clusters of cl CTAs the device runs at once.
cudaError_t evict_prepare(int* active);
cudaError_t launch_timeout_probe(int32_t* err, uint64_t limit_ns, cudaStream_t s);
cudaError_t launch_prefill(const CopyRowsParams& p, cudaStream_t s);
cudaError_t launch_restore(const CopyRowsParams& p, cudaStream_t s);
cudaError_t launch_restore_queries(const DevLayout& lay, int layer, const uint16_t* q, const int32_t* g_dev,
                                   cudaStream_t s);

// Scored policy: pass 1 (restore: softmax statistics of a loaded window, then launch_score_merge)
// or pass 2 (eviction: per-candidate sums with the recorded normalisers).
// The tensor maps cover kpool as [total_rows][128] bf16 and the query windows as
// [L*B*KVH*r*G][128] bf16, both with boxes of kScoreTile rows x 64 channels.
cudaError_t launch_score(const EvictParams& p, int pass, const CUtensorMap* tmap_k, const CUtensorMap* tmap_q,
                         cudaStream_t s);
cudaError_t launch_score_merge(const EvictParams& p, cudaStream_t s);
cudaError_t score_prepare();
int score_row_tiles_per_warp(int M);  // 16-row tiles of the M window rows per warp (1..4)

// Attention comes in two kernel shapes, one build of ra_attn.cu each: wide (48-row tiles, 4 warps
// per CTA) for large layers and narrow (32-row tiles, 6 warps) for small ones, where a finer split
// of a short layer across more warps shortens its tail.  The tensor maps cover kpool / vpool as
// [total_rows][128] bf16 in boxes of the shape's tile rows.
#define RA_ATTN_API                                                                                        \
    int attn_warps_per_cta(int G);                                                                         \
    int attn_tile_rows(int G);                                                                             \
    cudaError_t launch_attention(const AttnParams& p, const CUtensorMap* tmap_k, const CUtensorMap* tmap_v, \
                                 int ctas, cudaStream_t s);                                                \
    cudaError_t attn_prepare(int G); /* one-time function attributes (dynamic smem) */
namespace attn_wide { RA_ATTN_API }
namespace attn_narrow { RA_ATTN_API }
#undef RA_ATTN_API

enum AttnShape { kAttnWide = 0, kAttnNarrow = 1, kAttnShapes = 2 };
#ifndef RA_ATTN_NARROW_ROWS
#define RA_ATTN_NARROW_ROWS (1 << 20)
#endif
constexpr long long kNarrowRows = RA_ATTN_NARROW_ROWS;  // layers attending fewer rows take the narrow shape

inline int attn_warps_per_cta(int shape, int G)
{
    return shape == kAttnNarrow ? attn_narrow::attn_warps_per_cta(G) : attn_wide::attn_warps_per_cta(G);
}
// CTAs of a shape that one SM holds at once (the narrow build may be split into several smaller
// CTAs, so that an SM frees part of its shared memory for the next layer as each CTA finishes).
#ifndef RA_ATTN_NARROW_CTAS
#define RA_ATTN_NARROW_CTAS 1
#endif
inline int attn_ctas_per_sm(int shape) { return shape == kAttnNarrow ? RA_ATTN_NARROW_CTAS : 1; }
inline int attn_tile_rows(int shape, int G)
{
    return shape == kAttnNarrow ? attn_narrow::attn_tile_rows(G) : attn_wide::attn_tile_rows(G);
}
inline cudaError_t launch_attention(int shape, const AttnParams& p, const CUtensorMap* tk, const CUtensorMap* tv,
                                    int ctas, cudaStream_t s)
{
    return shape == kAttnNarrow ? attn_narrow::launch_attention(p, tk, tv, ctas, s)
                                : attn_wide::launch_attention(p, tk, tv, ctas, s);
}
inline cudaError_t attn_prepare(int shape, int G)
{
    return shape == kAttnNarrow ? attn_narrow::attn_prepare(G) : attn_wide::attn_prepare(G);
}

// Launch with programmatic dependent launch: the kernel may be scheduled while its
// predecessor on the stream finishes.  Every kernel waits (griddepcontrol.wait)
// before touching memory its predecessor may write, and lets its successor be
// scheduled only after that wait -- so when a kernel starts, every kernel before
// its predecessor has completed.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s, Args&&... args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

}  // namespace ra
