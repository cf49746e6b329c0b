// ra_api.cu -- host side of the C ABI declared in include/ra.h.
//
// Owns the host mirror of every per-(layer, sequence) counter, so that trigger
// decisions (section 2: every r steps once the candidates exceed K), capacity
// checks and the attention work split are made on the host without reading
// device memory; kernels receive the counts they need as launch parameters.  No call
// allocates device memory or synchronises, except the debug getters.
#include <cuda.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdarg.h>
#include <stdint.h>
#include <stdio.h>
#include <string.h>

#include <algorithm>
#include <mutex>
#include <string>
#include <vector>

#include "ra.h"
#include "ra_internal.h"

using namespace ra;

namespace {

thread_local std::string g_tls_error = "no error";

constexpr int kMaxSMs = 256;       // partial-buffer sizing bound (the GB300 has 152)
constexpr size_t kAlign = 256;

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

struct ProfRec {
    int kind;
    cudaEvent_t start, stop;
    double bytes;
};

}  // namespace

struct ra_ctx {
    // shape
    int L, H, KVH, G, D, B, K, r, Cmax;
    uint64_t seed;
    std::vector<int32_t> lp;       // prompt lengths
    // prompt pages (kPromptPage positions x KVH heads each, every layer alike): the pool, the
    // longest prompt a slot takes, each sequence's pages and the free ones; admissions per slot
    int max_prompt = 0, max_pages = 1;
    long long pool_pages = 0;
    std::vector<int32_t> pages;      // [B][max_pages]
    std::vector<int32_t> free_pages;
    std::vector<int32_t> admits;     // [B]
    long long prompt_rows_per_layer = 0;
    long long total_rows = 0;
    long long gen_rows = 0;
    int regions = 0;
    size_t partial_records = 0;  // split-K partial records the arena holds
    // arena layout (byte offsets)
    size_t off_k, off_v, off_pos, off_region, off_spare, off_lp, off_pages, off_plan, off_partial, off_arrive,
        off_err, off_evplan, bytes;
    // scored policy: query window, scores and pass-1 statistics after the base arena
    bool scoring = false;
    size_t base_bytes = 0, off_qring = 0, off_qstats = 0, off_scores = 0, off_stats = 0;
    int stats_chunks = 0;
    // binding
    bool bound = false;
    int device = -1;
    int sms = 0;
    int evict_active[kEvMaxCluster + 1] = {0};  // clusters of each size the device runs at once
    uint8_t* arena = nullptr;
    DevLayout lay{};
    CUtensorMap tmap_k[kAttnShapes]{}, tmap_v[kAttnShapes]{};  // per attention shape (tile rows)
    CUtensorMap tmap_ks{};  // kpool in kScoreTile-row boxes (scoring kernels)
    CUtensorMap tmap_q{};   // the query windows as [L*B*KVH*r*G][128] rows, same boxes
    // host mirror
    std::vector<int32_t> g, c, nev;  // [L][B]
    std::vector<uint8_t> active;     // [B]
    int policy = RA_POLICY_RANDOM;   // candidate scoring (ra_set_policy)
    int block = 1;
    int compaction = RA_COMPACT_ORDERED;  // ra_set_compaction
    int attn_shape = RA_ATTN_SHAPE_AUTO;  // ra_set_attention_shape
    int evict_mode = RA_EVICT_AUTO;       // ra_set_eviction_kernel
    std::vector<int32_t> score_n;    // [L][B] candidates of the latest scored round
    // Mirror of the device region tables.  Every head of a (layer, seq) evicts together, so the
    // region of (l, b, h) is always region_base * KVH + h: rbase[l * B + b], and the spare of
    // (b, h) is sbase[b] * KVH + h; an ordered compaction swaps the two.
    std::vector<int32_t> rbase, sbase;
    // Evicted sets computed one step ahead (ra_decode_step): plan_kernel runs on a side stream
    // beside the current step's attention and writes half (step parity) of the plan buffer;
    // plan_g / plan_n [2][L * B] record the firing (g, candidates) each half holds (-1: none).
    cudaStream_t side = nullptr;
    cudaEvent_t fork_ev = nullptr, plan_ev = nullptr;
    bool plan_pending = false;
    int parity = 0;
    bool no_early_once = false;  // the next attention launch follows the whole-stack compaction
    bool step_open = false;  // a step's prologue ran (plans launched, stack evicted) and its end has not
    int step_cur = 0;        // the plan half that step reads
    std::vector<int32_t> plan_g, plan_n;
    // profiling
    bool prof = false;
    std::vector<ProfRec> pending;
    std::vector<cudaEvent_t> pool;
    double prof_ms[RA_KERNEL_KINDS] = {0};
    int64_t prof_n[RA_KERNEL_KINDS] = {0};
    double prof_bytes[RA_KERNEL_KINDS] = {0};
    int64_t launch_n[RA_KERNEL_KINDS] = {0};      // always counted
    double launch_bytes[RA_KERNEL_KINDS] = {0};
    std::string err = "no error";
};

namespace {

int fail(ra_ctx* ctx, int code, const char* fmt, ...) __attribute__((format(printf, 3, 4)));
int fail(ra_ctx* ctx, int code, const char* fmt, ...)
{
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    if (ctx) ctx->err = buf;
    g_tls_error = buf;
    return code;
}

int cuda_fail(ra_ctx* ctx, cudaError_t e, const char* what)
{
    return fail(ctx, RA_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

int check_bound(ra_ctx* ctx)
{
    if (!ctx) return fail(nullptr, RA_ERR_INVALID_ARG, "ctx is NULL");
    if (!ctx->bound) return fail(ctx, RA_ERR_STATE, "no device arena bound (call ra_bind first)");
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev != ctx->device)
        return fail(ctx, RA_ERR_STATE, "current device %d is not the bound device %d", dev, ctx->device);
    return RA_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int check_layer(ra_ctx* ctx, int layer)
{
    if (layer < 0 || layer >= ctx->L) return fail(ctx, RA_ERR_INVALID_ARG, "layer %d out of [0, %d)", layer, ctx->L);
    return RA_OK;
}

// --- profiling
cudaEvent_t take_event(ra_ctx* ctx)
{
    if (!ctx->pool.empty()) {
        cudaEvent_t e = ctx->pool.back();
        ctx->pool.pop_back();
        return e;
    }
    cudaEvent_t e = nullptr;
    cudaEventCreate(&e);
    return e;
}

struct ProfScope {
    ra_ctx* ctx;
    int kind;
    double bytes;
    cudaStream_t s;
    cudaEvent_t start = nullptr;
    ProfScope(ra_ctx* c, int k, double b, cudaStream_t st) : ctx(c), kind(k), bytes(b), s(st)
    {
        if (ctx->prof) {
            start = take_event(ctx);
            cudaEventRecord(start, s);
        }
    }
    void done()
    {
        ctx->launch_n[kind] += 1;
        ctx->launch_bytes[kind] += bytes;
        if (ctx->prof && start) {
            cudaEvent_t stop = take_event(ctx);
            cudaEventRecord(stop, s);
            ctx->pending.push_back({kind, start, stop, bytes});
            start = nullptr;
        }
    }
};

int collect_profile(ra_ctx* ctx)
{
    for (auto& pr : ctx->pending) {
        cudaError_t e = cudaEventSynchronize(pr.stop);
        if (e != cudaSuccess) return cuda_fail(ctx, e, "profile event sync");
        float ms = 0.f;
        cudaEventElapsedTime(&ms, pr.start, pr.stop);
        ctx->prof_ms[pr.kind] += ms;
        ctx->prof_n[pr.kind] += 1;
        ctx->prof_bytes[pr.kind] += pr.bytes;
        ctx->pool.push_back(pr.start);
        ctx->pool.push_back(pr.stop);
    }
    ctx->pending.clear();
    return RA_OK;
}

// --- tensor maps over the K and V pools
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

int make_tmap(ra_ctx* ctx, CUtensorMap* map, void* base, long long rows, int box_rows)
{
    static EncodeTiledFn encode = nullptr;
    if (!encode) {
        void* fn = nullptr;
        cudaDriverEntryPointQueryResult q{};
        cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
        if (e != cudaSuccess || !fn || q != cudaDriverEntryPointSuccess)
            return fail(ctx, RA_ERR_CUDA, "cuTensorMapEncodeTiled entry point not available");
        encode = reinterpret_cast<EncodeTiledFn>(fn);
    }
    const cuuint64_t dims[2] = {(cuuint64_t)kHeadDim, (cuuint64_t)rows};
    const cuuint64_t strides[1] = {(cuuint64_t)kRowBytes};
    // boxes of 64 channels (128 bytes) x box_rows rows, stored with the 128-byte swizzle
    const cuuint32_t box[2] = {(cuuint32_t)(kHeadDim / 2), (cuuint32_t)box_rows};
    const cuuint32_t estr[2] = {1, 1};
    CUresult r = encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(ctx, RA_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", (int)r);
    return RA_OK;
}

void fill_active(const ra_ctx* ctx, uint32_t* mask)
{
    for (int i = 0; i < RA_MAX_BATCH / 32; ++i) mask[i] = 0;
    for (int b = 0; b < ctx->B; ++b)
        if (ctx->active[b]) mask[b >> 5] |= 1u << (b & 31);
}

// Work split of one layer's attention from the host mirror, in tiles: a head has
// ceil(lp / TILE) prompt tiles and ceil(gen / TILE) tiles of generated rows, where gen is
// the cached generated rows plus one for a fused new token; the tiles are cut into one equal
// chunk per warp.  *slots = rows attended.
int plan_attention(ra_ctx* ctx, int layer, int fused, AttnParams* p, int* n_active, int* ctas, double* slots,
                   int* shape, const std::vector<int32_t>* old_rows = nullptr)
{
    fill_active(ctx, p->active);
    // sequences whose compaction the launch does: their cached rows are the old region's
    for (int i = 0; i < RA_MAX_BATCH / 32; ++i) p->compacting[i] = 0u;
    if (old_rows)
        for (int b = 0; b < ctx->B; ++b)
            if ((*old_rows)[b] >= 0) p->compacting[b >> 5] |= 1u << (b & 31);
    // fused: every active sequence's token is pending
    for (int i = 0; i < RA_MAX_BATCH / 32; ++i) p->pending[i] = fused ? p->active[i] : 0u;
    long long acc = 0, rows = 0;
    int na = 0;
    for (int b = 0; b < ctx->B; ++b) {
        const int cached = (old_rows && (*old_rows)[b] >= 0) ? (*old_rows)[b] : ctx->c[(size_t)layer * ctx->B + b];
        const int gen = cached + (int)((p->pending[b >> 5] >> (b & 31)) & 1u);
        p->seq_gen[b] = gen;
        p->seq_g[b] = ctx->g[(size_t)layer * ctx->B + b];  // generated tokens before this step's
        p->seq_lp[b] = ctx->lp[b];
        p->seq_region[b] = ctx->rbase[(size_t)layer * ctx->B + b];
        const int32_t* pg = ctx->pages.data() + (size_t)b * ctx->max_pages;
        const int np = (ctx->lp[b] + kPromptPage - 1) / kPromptPage;
        bool consecutive = true;
        for (int j = 1; j < np && consecutive; ++j) consecutive = pg[j] == pg[0] + j;
        p->seq_page0[b] = np == 0 ? 0 : (consecutive ? pg[0] : -1);
        if (ctx->active[b]) {
            rows += (long long)ctx->KVH * (ctx->lp[b] + gen);
            ++na;
        }
    }
    *shape = ctx->attn_shape == RA_ATTN_SHAPE_WIDE     ? kAttnWide
             : ctx->attn_shape == RA_ATTN_SHAPE_NARROW ? kAttnNarrow
             : rows < kNarrowRows                      ? kAttnNarrow
                                                       : kAttnWide;
    const int T = attn_tile_rows(*shape, ctx->G);
    p->tile = T;
    p->seq_base[0] = 0;
    for (int b = 0; b < ctx->B; ++b) {
        if (ctx->active[b]) acc += (long long)ctx->KVH * ((ctx->lp[b] + T - 1) / T + (p->seq_gen[b] + T - 1) / T);
        p->seq_base[b + 1] = (int32_t)acc;
    }
    if (acc >= (1LL << 31)) return fail(ctx, RA_ERR_UNSUPPORTED, "layer holds more than 2^31 tiles");
    p->total = (int)acc;
    const int wpc = attn_warps_per_cta(*shape, ctx->G), cps = attn_ctas_per_sm(*shape);
    const long long nwarps_max = (long long)ctx->sms * cps * wpc;
    const long long W = std::max<long long>(1, (acc + nwarps_max - 1) / nwarps_max);
    const long long nchunks = (acc + W - 1) / W;
    p->W = (int)W;
    p->nchunks = (int)nchunks;
    *ctas = (int)std::min<long long>((long long)ctx->sms * cps, (nchunks + wpc - 1) / wpc);
    p->nwarps = *ctas * wpc;
    *n_active = na;
    *slots = (double)rows;
    // partial records are indexed chunk + head: both bounded by what the arena holds
    if ((size_t)p->nchunks + (size_t)ctx->B * ctx->KVH > ctx->partial_records)
        return fail(ctx, RA_ERR_STATE, "attention split needs more partial records than the arena holds");
    return RA_OK;
}

void layout_scoring(ra_ctx* ctx);

// Arena layout from the shape and the prompt pool (pages, the longest prompt); then the scored
// policy's buffers, if chosen.
int layout_base(ra_ctx* ctx)
{
    const int layers = ctx->L, batch = ctx->B, kv_heads = ctx->KVH, r = ctx->r;
    ctx->max_pages = std::max(1, (ctx->max_prompt + kPromptPage - 1) / kPromptPage);
    ctx->prompt_rows_per_layer = ctx->pool_pages * kv_heads * kPromptPage;
    ctx->regions = (layers + 1) * batch * kv_heads;
    ctx->gen_rows = (long long)ctx->regions * ctx->Cmax;
    ctx->total_rows = ctx->prompt_rows_per_layer * layers + ctx->gen_rows;
    // every slot position and every row index must fit the int32 coordinates the kernels use
    if (ctx->total_rows >= (1LL << 31) || ctx->prompt_rows_per_layer >= (1LL << 31))
        return fail(nullptr, RA_ERR_UNSUPPORTED, "cache too large for 32-bit row coordinates");
    size_t o = 0;
    auto take = [&](size_t n) {
        size_t at = o;
        o = align_up(o + n, kAlign);
        return at;
    };
    const size_t pool_bytes = (size_t)ctx->total_rows * kRowBytes;
    ctx->off_k = take(pool_bytes);
    ctx->off_v = take(pool_bytes);
    ctx->off_pos = take((size_t)ctx->regions * ctx->Cmax * 4);
    ctx->off_region = take((size_t)layers * batch * kv_heads * 4);
    ctx->off_spare = take((size_t)batch * kv_heads * 4);
    ctx->off_lp = take((size_t)batch * 4);
    ctx->off_pages = take((size_t)batch * ctx->max_pages * 4);
    ctx->off_plan = take((size_t)batch * kv_heads * (kPlanHeader + r) * 4);
    // chunks of the attention split: one per warp
    const size_t max_chunks =
        (size_t)kMaxSMs * std::max(attn_warps_per_cta(kAttnWide, ctx->G) * attn_ctas_per_sm(kAttnWide),
                                   attn_warps_per_cta(kAttnNarrow, ctx->G) * attn_ctas_per_sm(kAttnNarrow)) + 1;
    ctx->partial_records = max_chunks + (size_t)batch * kv_heads;
    ctx->off_partial = take(ctx->partial_records * partial_stride(ctx->G) * 4);
    ctx->off_arrive = take((size_t)batch * kv_heads * 4);
    ctx->off_err = take(256);
    ctx->off_evplan = take((size_t)2 * layers * batch * kv_heads * (r + 1) * 4);
    ctx->base_bytes = o;
    // pass-1 chunks per head: at most one per tile of the longest head, capped (the host
    // then takes chunks of several tiles)
    const int tiles1 = (ctx->max_prompt + kScoreTile - 1) / kScoreTile + (ctx->Cmax + kScoreTile - 1) / kScoreTile;
    ctx->stats_chunks = std::min(tiles1, 64);
    layout_scoring(ctx);
    return RA_OK;
}

// Arena size with (or without) the scored policy's buffers after the base layout.
void layout_scoring(ra_ctx* ctx)
{
    if (!ctx->scoring) {
        ctx->bytes = ctx->base_bytes;
        return;
    }
    const size_t heads = (size_t)ctx->B * ctx->KVH;
    const size_t M = (size_t)ctx->r * ctx->G;
    size_t o = ctx->base_bytes;
    ctx->off_qring = o;
    o = align_up(o + (size_t)ctx->L * heads * M * kRowBytes, kAlign);
    ctx->off_qstats = o;
    o = align_up(o + (size_t)ctx->L * heads * M * sizeof(float2), kAlign);
    ctx->off_scores = o;
    o = align_up(o + (size_t)ctx->L * heads * ctx->Cmax * sizeof(float), kAlign);
    ctx->off_stats = o;
    o = align_up(o + heads * ctx->stats_chunks * M * 2 * sizeof(float), kAlign);
    ctx->bytes = o;
}

// Launch shape of a scoring pass over the heads of the sequences in p (pass 1: prompt + the
// trig_n cached rows each; pass 2: the trig_n candidate rows each): about two waves of CTAs
// (one per SM when the window needs more than half the shared memory), each taking a run of
// consecutive tiles of one head.  Returns the algorithmic bytes: the key rows read (every
// one is contracted with the M = r * G window rows, so flops = bytes * M).
double plan_scoring(ra_ctx* ctx, EvictParams* p, int pass)
{
    const int M = ctx->r * ctx->G;
    // pass 2 runs on tcgen05 with all of an SM's tensor memory: one CTA per SM, and runs of
    // whole 128-row tiles (two scoring tiles)
    const int per_sm = pass == 2 ? 1 : (score_row_tiles_per_warp(M) <= 2 ? 2 : 1);
    long long work = 0;
    int most = 1;
    double rows = 0;
    for (int i = 0; i < p->n_trig; ++i) {
        const int lp = pass == 1 ? ctx->lp[p->trig[i]] : 0, n = p->trig_n[i];
        const int t = (lp + kScoreTile - 1) / kScoreTile + (n + kScoreTile - 1) / kScoreTile;
        work += (long long)ctx->KVH * t;
        most = std::max(most, t);
        rows += (double)ctx->KVH * (lp + n);
    }
    const long long target = (long long)ctx->sms * per_sm;
    long long ch = std::max<long long>((work + target - 1) / target, 1);
    if (pass == 1) ch = std::max<long long>(ch, (most + ctx->stats_chunks - 1) / ctx->stats_chunks);
    if (pass == 2) ch = (ch + 1) / 2 * 2;
    const int nch = (int)((most + ch - 1) / ch);
    if (pass == 1) {
        p->ch1 = (int)ch;
        p->nch1 = nch;
    } else {
        p->ch2 = (int)ch;
        p->nch2 = nch;
    }
    return rows * kRowBytes;
}

int run_eviction_launches(ra_ctx* ctx, EvictParams& p, double moved, cudaStream_t s, bool compact_in_attention,
                          int score_early);

// Evicted sets can be computed ahead for the policies whose keys need no scores (random, shared,
// recency, block), with ordered compaction outside the attention pass (the one-launch kernels) or
// order-free slots.  Keys that follow positions (order-free slots, block draws) are read from the
// cache, so their plans also need r >= 2: the next step's candidates then exclude the slot the
// current step appends.
bool keys_read_positions(const ra_ctx* ctx)
{
    return ctx->compaction == RA_COMPACT_HOLEFILL || ctx->policy == RA_POLICY_BLOCK;
}

bool plan_usable(const ra_ctx* ctx)
{
    if (ctx->r > kEvMaxEvicted || (ctx->evict_mode & ~RA_EVICT_EXACT) == RA_EVICT_TWO_KERNELS) return false;
    if (ctx->policy == RA_POLICY_SNAPKV || (keys_read_positions(ctx) && ctx->r < 2)) return false;
    if (ctx->compaction == RA_COMPACT_HOLEFILL) return true;
    return ctx->compaction == RA_COMPACT_ORDERED && ctx->evict_active[1] > 0;
}

// One eviction round of the triggered sequences in p: [score passes,] select, compact (unless
// the caller's attention launch does the compaction).
int run_eviction(ra_ctx* ctx, EvictParams& p, double moved, cudaStream_t s, bool compact_in_attention = false,
                 int score_early = 0)
{
    for (int i = 0; i < p.n_trig; ++i) {
        p.trig_src[i] = ctx->rbase[(size_t)p.layer * ctx->B + p.trig[i]];
        p.trig_dst[i] = ctx->sbase[p.trig[i]];
        p.trig_admit[i] = (uint16_t)ctx->admits[p.trig[i]];
    }
    int rc = run_eviction_launches(ctx, p, moved, s, compact_in_attention, score_early);
    if (rc == RA_OK && !p.holefill)  // every ordered compaction (any kernel) swaps region and spare
        for (int i = 0; i < p.n_trig; ++i)
            std::swap(ctx->rbase[(size_t)p.layer * ctx->B + p.trig[i]], ctx->sbase[p.trig[i]]);
    return rc;
}

int run_eviction_launches(ra_ctx* ctx, EvictParams& p, double moved, cudaStream_t s, bool compact_in_attention,
                          int score_early)
{
    cudaError_t e;
    if (p.policy == RA_POLICY_SNAPKV) {  // window scores with the normalisers recorded at decode time
        for (int i = 0; i < p.n_trig; ++i) ctx->score_n[(size_t)p.layer * ctx->B + p.trig[i]] = p.trig_n[i];
        const double bytes = plan_scoring(ctx, &p, 2);
        ProfScope ps(ctx, RA_KERNEL_SCORE_SUM, bytes, s);
        const int select_early = p.early;
        p.early = score_early;  // the scoring pass's own flag; the selection after it waits first
        e = launch_score(p, 2, &ctx->tmap_ks, &ctx->tmap_q, s);
        p.early = select_early;
        ps.done();
        if (e != cudaSuccess) return cuda_fail(ctx, e, "score launch");
    }
    // The random policy and its key-per-ordinal variants with ordered compaction: one launch,
    // a cluster per triggered head.
    // A head's candidates are split over the CTAs of a cluster (at most kEvMaxLocal keys each);
    // each of a head's `reps` clusters selects on its own and the copy is split over all of
    // them.  The automatic shape maximises the CTAs working on each head at once,
    // cl x reps / waves, from the device's cluster occupancy (a GPC holds a whole cluster, so
    // sizes that pack its SMs win; ties go to the larger cluster, which draws fewer keys per
    // CTA).  A device that cannot schedule a usable size takes the two kernels.
    const int least = std::max(1, (ctx->K + ctx->r + kEvMaxLocal - 1) / kEvMaxLocal);
    const int heads = std::max(1, p.n_trig * ctx->KVH);
    const int forced = ctx->evict_mode & ~RA_EVICT_EXACT;
    int cl = 0, reps = 1;
    double best = 0;
    if (p.ev_plan) {  // the evicted sets are known: no cluster, the copy spread over about one CTA per SM
        cl = 1;
        reps = std::max(1, std::min(64, ctx->evict_active[1] / heads));
    }
    for (int x = std::max(least, forced >= 2 ? forced : least); x <= kEvMaxCluster && !p.ev_plan; ++x) {
        const int act = ctx->evict_active[x];
        if (act <= 0) continue;
        const int rp = std::max(1, std::min(act / heads, 64));
        const double waves = std::ceil((double)heads * rp / act);
        const double score = x * rp / waves;
        if (score >= best) {
            best = score;
            cl = x;
            reps = rp;
        }
        if (forced >= 2) break;  // the forced size (or the next one the device can schedule)
    }
    const bool one_launch = !p.holefill && !compact_in_attention && p.policy != RA_POLICY_SNAPKV &&
                            forced != RA_EVICT_TWO_KERNELS && cl > 0 && ctx->r <= kEvMaxEvicted;
    if (one_launch) {
        p.ev_reps = reps;
        p.ev_exact = (ctx->evict_mode & RA_EVICT_EXACT) ? 1 : 0;
        ProfScope ps(ctx, RA_KERNEL_EVICT, moved * 2.0 * (2 * kRowBytes + 4), s);
        e = launch_evict(p, cl, s);
        ps.done();
        if (e != cudaSuccess) return cuda_fail(ctx, e, "evict launch");
        return RA_OK;
    }
    {
        // with order-free compaction the select kernel also moves m rows per head (read and write)
        double fill = 0;
        if (p.holefill)
            for (int i = 0; i < p.n_trig; ++i) fill += (double)(p.trig_n[i] - ctx->K) * ctx->KVH * 2.0 * (2 * kRowBytes + 4);
        ProfScope ps(ctx, RA_KERNEL_SELECT, fill, s);
        e = launch_select(p, s);
        ps.done();
    }
    if (e != cudaSuccess) return cuda_fail(ctx, e, "select launch");
    if (p.holefill || compact_in_attention) return RA_OK;  // done by select / by the attention launch
    {
        ProfScope ps(ctx, RA_KERNEL_COMPACT, moved * 2.0 * (2 * kRowBytes + 4), s);
        e = launch_compact(p, s);
        ps.done();
    }
    if (e != cudaSuccess) return cuda_fail(ctx, e, "compact launch");
    return RA_OK;
}

void set_scale(AttnParams* p, float scale)
{
    const float sc = scale > 0.f ? scale : 1.0f / sqrtf((float)kHeadDim);
    p->qk_scale_log2 = sc * 1.4426950408889634f;
}

}  // namespace

extern "C" {

const char* ra_last_error(const ra_ctx* ctx) { return ctx ? ctx->err.c_str() : g_tls_error.c_str(); }

int ra_create_batched(ra_ctx** out, int layers, int q_heads, int kv_heads, int head_dim, int batch,
                      const int32_t* prompt_lens, int K, int r, uint64_t seed)
{
    if (!out) return fail(nullptr, RA_ERR_INVALID_ARG, "out is NULL");
    *out = nullptr;
    if (layers < 1) return fail(nullptr, RA_ERR_INVALID_ARG, "layers must be >= 1");
    if (kv_heads < 1 || kv_heads > 32) return fail(nullptr, RA_ERR_INVALID_ARG, "kv_heads must be in [1, 32]");
    if (q_heads < kv_heads || q_heads % kv_heads != 0)
        return fail(nullptr, RA_ERR_INVALID_ARG, "q_heads must be a positive multiple of kv_heads");
    if (q_heads / kv_heads > kMaxG) return fail(nullptr, RA_ERR_UNSUPPORTED, "q_heads / kv_heads must be <= 8");
    if (head_dim != kHeadDim) return fail(nullptr, RA_ERR_UNSUPPORTED, "head_dim must be 128");
    if (batch < 1 || batch > RA_MAX_BATCH) return fail(nullptr, RA_ERR_INVALID_ARG, "batch must be in [1, %d]", RA_MAX_BATCH);
    if (!prompt_lens) return fail(nullptr, RA_ERR_INVALID_ARG, "prompt_lens is NULL");
    if (K < 0 || r < 1) return fail(nullptr, RA_ERR_INVALID_ARG, "need K >= 0 and r >= 1");
    if ((long long)K + r > kMaxCandidates) return fail(nullptr, RA_ERR_UNSUPPORTED, "K + r must be <= %d", kMaxCandidates);
    if (select_smem(K + r, r, false) > kSelectSmemLimit)
        return fail(nullptr, RA_ERR_UNSUPPORTED, "K + 2r too large for the selection's shared memory");

    ra_ctx* ctx = new ra_ctx();
    ctx->L = layers;
    ctx->H = q_heads;
    ctx->KVH = kv_heads;
    ctx->G = q_heads / kv_heads;
    ctx->D = head_dim;
    ctx->B = batch;
    ctx->K = K;
    ctx->r = r;
    ctx->Cmax = K + 2 * r;
    ctx->seed = seed;
    ctx->lp.assign(prompt_lens, prompt_lens + batch);
    for (int b = 0; b < batch; ++b) {
        if (prompt_lens[b] < 0) {
            delete ctx;
            return fail(nullptr, RA_ERR_INVALID_ARG, "prompt_lens[%d] < 0", b);
        }
        ctx->max_prompt = std::max(ctx->max_prompt, (int)prompt_lens[b]);
        ctx->pool_pages += (prompt_lens[b] + kPromptPage - 1) / kPromptPage;
    }
    int rc = layout_base(ctx);
    if (rc != RA_OK) {
        delete ctx;
        return rc;
    }
    ctx->g.assign((size_t)layers * batch, 0);
    ctx->c.assign((size_t)layers * batch, 0);
    ctx->nev.assign((size_t)layers * batch, 0);
    ctx->active.assign(batch, 1);
    ctx->score_n.assign((size_t)layers * batch, 0);
    *out = ctx;
    return RA_OK;
}

int ra_create(ra_ctx** out, int layers, int q_heads, int kv_heads, int head_dim, int prompt_len, int K, int r,
              uint64_t seed)
{
    const int32_t lp = prompt_len;
    if (prompt_len < 0) return fail(nullptr, RA_ERR_INVALID_ARG, "prompt_len < 0");
    return ra_create_batched(out, layers, q_heads, kv_heads, head_dim, 1, &lp, K, r, seed);
}

size_t ra_device_bytes(const ra_ctx* ctx) { return ctx ? ctx->bytes : 0; }

int ra_bind(ra_ctx* ctx, void* device_arena, size_t bytes, void* stream)
{
    if (!ctx) return fail(nullptr, RA_ERR_INVALID_ARG, "ctx is NULL");
    if (!device_arena || (reinterpret_cast<uintptr_t>(device_arena) & (kAlign - 1)))
        return fail(ctx, RA_ERR_INVALID_ARG, "arena must be a non-NULL 256-byte aligned device pointer");
    if (bytes < ctx->bytes) return fail(ctx, RA_ERR_INVALID_ARG, "arena has %zu bytes, need %zu", bytes, ctx->bytes);
    cudaError_t e;
    cudaPointerAttributes attr{};
    if ((e = cudaPointerGetAttributes(&attr, device_arena)) != cudaSuccess) return cuda_fail(ctx, e, "arena attributes");
    if (attr.type != cudaMemoryTypeDevice) return fail(ctx, RA_ERR_INVALID_ARG, "arena is not device memory");
    int dev = -1;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return cuda_fail(ctx, e, "cudaGetDevice");
    if (attr.device != dev) return fail(ctx, RA_ERR_INVALID_ARG, "arena lives on device %d, current is %d", attr.device, dev);
    int sms = 0;
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
        return cuda_fail(ctx, e, "SM count");
    if (sms > kMaxSMs) return fail(ctx, RA_ERR_UNSUPPORTED, "more than %d SMs", kMaxSMs);
    cudaStream_t s = (cudaStream_t)stream;

    uint8_t* a = (uint8_t*)device_arena;
    DevLayout& Ly = ctx->lay;
    Ly.kpool = (uint16_t*)(a + ctx->off_k);
    Ly.vpool = (uint16_t*)(a + ctx->off_v);
    Ly.pos = (int32_t*)(a + ctx->off_pos);
    Ly.region = (int32_t*)(a + ctx->off_region);
    Ly.spare = (int32_t*)(a + ctx->off_spare);
    Ly.seq_lp = (int32_t*)(a + ctx->off_lp);
    Ly.pages = (int32_t*)(a + ctx->off_pages);
    Ly.max_pages = ctx->max_pages;
    Ly.plan = (int32_t*)(a + ctx->off_plan);
    Ly.partial = (float*)(a + ctx->off_partial);
    Ly.arrive = (int32_t*)(a + ctx->off_arrive);
    Ly.err = (int32_t*)(a + ctx->off_err);
    Ly.evplan = (int32_t*)(a + ctx->off_evplan);
    Ly.qring = ctx->scoring ? (uint16_t*)(a + ctx->off_qring) : nullptr;
    Ly.qstats = ctx->scoring ? (float2*)(a + ctx->off_qstats) : nullptr;
    Ly.scores = ctx->scoring ? (float*)(a + ctx->off_scores) : nullptr;
    Ly.stats = ctx->scoring ? (float*)(a + ctx->off_stats) : nullptr;
    Ly.stats_chunks = ctx->stats_chunks;
    Ly.prompt_rows_per_layer = ctx->prompt_rows_per_layer;
    Ly.gen_row0 = ctx->prompt_rows_per_layer * ctx->L;
    Ly.L = ctx->L;
    Ly.B = ctx->B;
    Ly.KVH = ctx->KVH;
    Ly.H = ctx->H;
    Ly.G = ctx->G;
    Ly.Cmax = ctx->Cmax;
    Ly.K = ctx->K;
    Ly.r = ctx->r;
    Ly.seed = ctx->seed;

    // Prompt pages in sequence order, the rest of the pool free; no admissions yet.
    ctx->pages.assign((size_t)ctx->B * ctx->max_pages, 0);
    ctx->free_pages.clear();
    {
        long long next = 0;
        for (int b = 0; b < ctx->B; ++b)
            for (int j = 0; j < (ctx->lp[b] + kPromptPage - 1) / kPromptPage; ++j)
                ctx->pages[(size_t)b * ctx->max_pages + j] = (int32_t)next++;
        if (next > ctx->pool_pages) return fail(ctx, RA_ERR_CAPACITY, "prompts need more pages than the pool holds");
        for (long long pg = ctx->pool_pages - 1; pg >= next; --pg) ctx->free_pages.push_back((int32_t)pg);
    }
    ctx->admits.assign(ctx->B, 0);
    // Tables: regions of (layer, seq, head) in order, one spare per (seq, head).
    const int BH = ctx->B * ctx->KVH;
    std::vector<int32_t> region((size_t)ctx->L * BH), spare(BH);
    for (size_t i = 0; i < region.size(); ++i) region[i] = (int32_t)i;
    for (int i = 0; i < BH; ++i) spare[i] = ctx->L * BH + i;
    int32_t zero = 0;
    // Pageable host sources: cudaMemcpyAsync returns once the data is staged, so the vectors may die here.
    if ((e = cudaMemcpyAsync(Ly.region, region.data(), region.size() * 4, cudaMemcpyHostToDevice, s)) != cudaSuccess ||
        (e = cudaMemcpyAsync(Ly.spare, spare.data(), spare.size() * 4, cudaMemcpyHostToDevice, s)) != cudaSuccess ||
        (e = cudaMemcpyAsync(Ly.seq_lp, ctx->lp.data(), ctx->B * 4, cudaMemcpyHostToDevice, s)) != cudaSuccess ||
        (e = cudaMemcpyAsync(Ly.pages, ctx->pages.data(), ctx->pages.size() * 4, cudaMemcpyHostToDevice, s)) !=
            cudaSuccess ||
        (e = cudaMemcpyAsync(Ly.err, &zero, 4, cudaMemcpyHostToDevice, s)) != cudaSuccess ||
        (e = cudaMemsetAsync(Ly.arrive, 0, (size_t)BH * 4, s)) != cudaSuccess)
        return cuda_fail(ctx, e, "table initialisation");
    // rows that were never written (past a head's cached slots) then read as zeros, never as stale NaNs
    if ((e = cudaMemsetAsync(a, 0, ctx->off_pos, s)) != cudaSuccess) return cuda_fail(ctx, e, "cache clear");
    // an empty query window and no scores yet
    if (ctx->scoring && (e = cudaMemsetAsync(a + ctx->off_qring, 0, ctx->off_stats - ctx->off_qring, s)) != cudaSuccess)
        return cuda_fail(ctx, e, "query window clear");
    if ((e = cudaStreamSynchronize(s)) != cudaSuccess) return cuda_fail(ctx, e, "table initialisation sync");

    int rc;
    for (int sh = 0; sh < kAttnShapes; ++sh) {
        const int tile = attn_tile_rows(sh, ctx->G);
        if ((rc = make_tmap(ctx, &ctx->tmap_k[sh], Ly.kpool, ctx->total_rows, tile)) != RA_OK) return rc;
        if ((rc = make_tmap(ctx, &ctx->tmap_v[sh], Ly.vpool, ctx->total_rows, tile)) != RA_OK) return rc;
        if ((e = attn_prepare(sh, ctx->G)) != cudaSuccess) return cuda_fail(ctx, e, "attention kernel attributes");
    }
    if ((e = evict_prepare(ctx->evict_active)) != cudaSuccess) return cuda_fail(ctx, e, "eviction kernel attributes");
    if (ctx->scoring) {
        if ((rc = make_tmap(ctx, &ctx->tmap_ks, Ly.kpool, ctx->total_rows, kScoreTile)) != RA_OK) return rc;
        const long long win_rows = (long long)ctx->L * ctx->B * ctx->KVH * ctx->r * ctx->G;
        if ((rc = make_tmap(ctx, &ctx->tmap_q, Ly.qring, win_rows, kScoreTile)) != RA_OK) return rc;
        if ((e = score_prepare()) != cudaSuccess) return cuda_fail(ctx, e, "score kernel attributes");
    }

    ctx->arena = a;
    ctx->device = dev;
    ctx->sms = sms;
    ctx->bound = true;
    std::fill(ctx->g.begin(), ctx->g.end(), 0);
    std::fill(ctx->c.begin(), ctx->c.end(), 0);
    std::fill(ctx->nev.begin(), ctx->nev.end(), 0);
    std::fill(ctx->score_n.begin(), ctx->score_n.end(), 0);
    if (!ctx->side) {
        if ((e = cudaStreamCreateWithFlags(&ctx->side, cudaStreamNonBlocking)) != cudaSuccess ||
            (e = cudaEventCreateWithFlags(&ctx->fork_ev, cudaEventDisableTiming)) != cudaSuccess ||
            (e = cudaEventCreateWithFlags(&ctx->plan_ev, cudaEventDisableTiming)) != cudaSuccess)
            return cuda_fail(ctx, e, "side stream");
    }
    ctx->plan_pending = false;
    ctx->parity = 0;
    ctx->plan_g.assign((size_t)2 * ctx->L * ctx->B, -1);
    ctx->plan_n.assign((size_t)2 * ctx->L * ctx->B, -1);
    ctx->rbase.resize((size_t)ctx->L * ctx->B);
    ctx->sbase.resize((size_t)ctx->B);
    for (size_t i = 0; i < ctx->rbase.size(); ++i) ctx->rbase[i] = (int32_t)i;
    for (int b = 0; b < ctx->B; ++b) ctx->sbase[b] = ctx->L * ctx->B + b;
    return RA_OK;
}

int ra_prefill(ra_ctx* ctx, int layer, const uint16_t* k, const uint16_t* v, int row_stride, void* stream)
{
    int rc;
    if ((rc = check_bound(ctx)) != RA_OK) return rc;
    if ((rc = check_layer(ctx, layer)) != RA_OK) return rc;
    if (!k || !v || !aligned16(k) || !aligned16(v)) return fail(ctx, RA_ERR_INVALID_ARG, "k/v must be 16-byte aligned");
    int maxlp = 0;
    for (int b = 0; b < ctx->B; ++b) maxlp = std::max(maxlp, (int)ctx->lp[b]);
    if (row_stride < maxlp) return fail(ctx, RA_ERR_INVALID_ARG, "row_stride %d < max prompt length %d", row_stride, maxlp);
    if (maxlp == 0) return RA_OK;
    CopyRowsParams p{};
    p.lay = ctx->lay;
    p.layer = layer;
    p.k = k;
    p.v = v;
    p.row_stride = row_stride;
    p.only_seq = -1;
    for (int b = 0; b < ctx->B; ++b) p.n_rows[b] = ctx->lp[b];
    cudaError_t e = launch_prefill(p, (cudaStream_t)stream);
    return e == cudaSuccess ? RA_OK : cuda_fail(ctx, e, "prefill launch");
}

int ra_restore(ra_ctx* ctx, int layer, const int32_t* g_host, const int32_t* c_host, const int32_t* pos,
               const uint16_t* k, const uint16_t* v, int row_stride, void* stream)
{
    int rc;
    if ((rc = check_bound(ctx)) != RA_OK) return rc;
    if ((rc = check_layer(ctx, layer)) != RA_OK) return rc;
    if (!g_host || !c_host || !pos || !k || !v) return fail(ctx, RA_ERR_INVALID_ARG, "NULL argument");
    if (!aligned16(k) || !aligned16(v)) return fail(ctx, RA_ERR_INVALID_ARG, "k/v must be 16-byte aligned");
    int maxc = 0;
    for (int b = 0; b < ctx->B; ++b) {
        if (c_host[b] < 0 || c_host[b] > ctx->Cmax || c_host[b] > g_host[b])
            return fail(ctx, RA_ERR_INVALID_ARG, "seq %d: need 0 <= c <= min(g, K + 2r)", b);
        maxc = std::max(maxc, (int)c_host[b]);
    }
    if (row_stride < maxc) return fail(ctx, RA_ERR_INVALID_ARG, "row_stride %d < max c %d", row_stride, maxc);
    cudaStream_t s = (cudaStream_t)stream;
    CopyRowsParams p{};
    p.lay = ctx->lay;
    p.layer = layer;
    p.k = k;
    p.v = v;
    p.pos = pos;
    p.row_stride = row_stride;
    p.only_seq = -1;
    for (int b = 0; b < ctx->B; ++b) p.n_rows[b] = c_host[b];
    cudaError_t e;
    if (maxc > 0 && (e = launch_restore(p, s)) != cudaSuccess) return cuda_fail(ctx, e, "restore launch");
    for (int b = 0; b < ctx->B; ++b) {
        const size_t i = (size_t)layer * ctx->B + b;
        ctx->g[i] = g_host[b];
        ctx->c[i] = c_host[b];
        ctx->plan_g[i] = ctx->plan_g[(size_t)ctx->L * ctx->B + i] = -1;  // positions replaced
    }
    return RA_OK;
}

int ra_set_policy(ra_ctx* ctx, int policy, int block)
{
    if (!ctx) return fail(nullptr, RA_ERR_INVALID_ARG, "ctx is NULL");
    if (policy < RA_POLICY_RANDOM || policy > RA_POLICY_SNAPKV)
        return fail(ctx, RA_ERR_INVALID_ARG, "unknown policy %d", policy);
    if (policy == RA_POLICY_BLOCK && block < 1) return fail(ctx, RA_ERR_INVALID_ARG, "block must be >= 1");
    if (policy == RA_POLICY_SNAPKV && ctx->compaction == RA_COMPACT_HOLEFILL)
        return fail(ctx, RA_ERR_UNSUPPORTED, "the scored policy needs ordered compaction");
    if (policy == RA_POLICY_SNAPKV && !ctx->scoring) {
        if (ctx->bound)
            return fail(ctx, RA_ERR_STATE, "the scored policy must be set before ra_device_bytes / ra_bind");
        if (ctx->r * ctx->G > kScoreMaxRows)
            return fail(ctx, RA_ERR_UNSUPPORTED, "scored policy needs r * G <= %d (have %d)", kScoreMaxRows,
                        ctx->r * ctx->G);
        if (ctx->K + ctx->r > kScoreMaxCandidates)
            return fail(ctx, RA_ERR_UNSUPPORTED, "scored policy needs K + r <= %d", kScoreMaxCandidates);
        ctx->scoring = true;
        layout_scoring(ctx);
    }
    ctx->policy = policy;
    ctx->block = policy == RA_POLICY_BLOCK ? block : 1;
    std::fill(ctx->plan_g.begin(), ctx->plan_g.end(), -1);  // sets computed ahead under another policy
    return RA_OK;
}

int ra_set_compaction(ra_ctx* ctx, int mode)
{
    if (!ctx) return fail(nullptr, RA_ERR_INVALID_ARG, "ctx is NULL");
    if (mode != RA_COMPACT_ORDERED && mode != RA_COMPACT_HOLEFILL && mode != RA_COMPACT_FUSED)
        return fail(ctx, RA_ERR_INVALID_ARG, "unknown compaction %d", mode);
    if (mode == RA_COMPACT_HOLEFILL && ctx->policy == RA_POLICY_SNAPKV)
        return fail(ctx, RA_ERR_UNSUPPORTED, "the scored policy needs ordered compaction");
    ctx->compaction = mode;
    std::fill(ctx->plan_g.begin(), ctx->plan_g.end(), -1);  // keys per ordinal or per position
    return RA_OK;
}

int ra_set_attention_shape(ra_ctx* ctx, int shape)
{
    if (!ctx) return fail(nullptr, RA_ERR_INVALID_ARG, "ctx is NULL");
    if (shape < RA_ATTN_SHAPE_AUTO || shape > RA_ATTN_SHAPE_NARROW)
        return fail(ctx, RA_ERR_INVALID_ARG, "unknown attention shape %d", shape);
    ctx->attn_shape = shape;
    return RA_OK;
}

int ra_set_prompt_pool(ra_ctx* ctx, int max_prompt_len, long long pool_positions)
{
    if (!ctx) return fail(nullptr, RA_ERR_INVALID_ARG, "ctx is NULL");
    if (ctx->bound) return fail(ctx, RA_ERR_STATE, "the prompt pool must be set before ra_device_bytes / ra_bind");
    if (max_prompt_len < 0 || pool_positions < 0) return fail(ctx, RA_ERR_INVALID_ARG, "negative size");
    long long need = 0;
    int longest = 0;
    for (int b = 0; b < ctx->B; ++b) {
        need += (ctx->lp[b] + kPromptPage - 1) / kPromptPage;
        longest = std::max(longest, (int)ctx->lp[b]);
    }
    const int old_max = ctx->max_prompt;
    const long long old_pool = ctx->pool_pages;
    ctx->max_prompt = std::max(longest, max_prompt_len);
    ctx->pool_pages = std::max(need, (pool_positions + kPromptPage - 1) / kPromptPage);
    int rc = layout_base(ctx);
    if (rc != RA_OK) {  // too large: keep the previous pool
        ctx->max_prompt = old_max;
        ctx->pool_pages = old_pool;
        layout_base(ctx);
        return fail(ctx, rc, "%s", ra_last_error(nullptr));
    }
    return RA_OK;
}

int ra_admit(ra_ctx* ctx, int seq, int prompt_len, const uint16_t* k, const uint16_t* v, int row_stride, void* stream)
{
    int rc;
    if ((rc = check_bound(ctx)) != RA_OK) return rc;
    if (seq < 0 || seq >= ctx->B) return fail(ctx, RA_ERR_INVALID_ARG, "seq %d out of range", seq);
    if (ctx->active[seq]) return fail(ctx, RA_ERR_STATE, "seq %d is active: finish it (ra_set_active 0) first", seq);
    if (prompt_len < 0 || prompt_len > ctx->max_prompt)
        return fail(ctx, RA_ERR_CAPACITY, "prompt of %d tokens: the slots take up to %d (ra_set_prompt_pool)", prompt_len,
                    ctx->max_prompt);
    if (prompt_len > 0 && (!k || !v || !aligned16(k) || !aligned16(v) || row_stride < prompt_len))
        return fail(ctx, RA_ERR_INVALID_ARG, "k/v must be 16-byte aligned with row_stride >= prompt_len");
    if (ctx->admits[seq] >= 0xFFFF) return fail(ctx, RA_ERR_CAPACITY, "slot %d has taken 65535 requests", seq);
    const int old_n = (ctx->lp[seq] + kPromptPage - 1) / kPromptPage, new_n = (prompt_len + kPromptPage - 1) / kPromptPage;
    if ((long long)ctx->free_pages.size() + old_n < new_n)
        return fail(ctx, RA_ERR_CAPACITY, "prompt pool has %zu free pages, the request needs %d",
                    ctx->free_pages.size() + old_n, new_n);
    cudaStream_t s = (cudaStream_t)stream;
    int32_t* row = ctx->pages.data() + (size_t)seq * ctx->max_pages;
    for (int j = 0; j < old_n; ++j) ctx->free_pages.push_back(row[j]);
    for (int j = 0; j < new_n; ++j) {
        row[j] = ctx->free_pages.back();
        ctx->free_pages.pop_back();
    }
    ctx->lp[seq] = prompt_len;
    cudaError_t e;
    // (pageable sources: the calls return once the values are staged)
    if ((e = cudaMemcpyAsync(ctx->lay.pages + (size_t)seq * ctx->max_pages, row, (size_t)ctx->max_pages * 4,
                             cudaMemcpyHostToDevice, s)) != cudaSuccess ||
        (e = cudaMemcpyAsync(ctx->lay.seq_lp + seq, &ctx->lp[seq], 4, cudaMemcpyHostToDevice, s)) != cudaSuccess)
        return cuda_fail(ctx, e, "page table update");
    if (prompt_len > 0) {
        CopyRowsParams p{};
        p.lay = ctx->lay;
        p.k = k;
        p.v = v;
        p.row_stride = row_stride;
        p.only_seq = seq;
        p.n_rows[seq] = prompt_len;
        for (int l = 0; l < ctx->L; ++l) {
            p.layer = l;
            p.k = k + (size_t)l * ctx->KVH * row_stride * kHeadDim;
            p.v = v + (size_t)l * ctx->KVH * row_stride * kHeadDim;
            if ((e = launch_prefill(p, s)) != cudaSuccess) return cuda_fail(ctx, e, "admit prefill launch");
        }
    }
    // a fresh request: nothing generated, nothing cached, its own random stream
    for (int l = 0; l < ctx->L; ++l) {
        const size_t i = (size_t)l * ctx->B + seq;
        ctx->g[i] = ctx->c[i] = ctx->nev[i] = 0;
        ctx->score_n[i] = 0;
        ctx->plan_g[i] = ctx->plan_g[(size_t)ctx->L * ctx->B + i] = -1;
    }
    ctx->admits[seq] += 1;
    ctx->active[seq] = 1;
    return RA_OK;
}

int ra_set_eviction_kernel(ra_ctx* ctx, int mode)
{
    if (!ctx) return fail(nullptr, RA_ERR_INVALID_ARG, "ctx is NULL");
    const int base = mode & ~RA_EVICT_EXACT;
    if (mode < 0 || base > kEvMaxCluster || (mode & ~(RA_EVICT_EXACT | 31)))
        return fail(ctx, RA_ERR_INVALID_ARG, "eviction kernel mode %d: expected [0, %d], optionally | RA_EVICT_EXACT",
                    mode, kEvMaxCluster);
    ctx->evict_mode = mode;
    return RA_OK;
}

int ra_set_active(ra_ctx* ctx, int seq, int active)
{
    if (!ctx) return fail(nullptr, RA_ERR_INVALID_ARG, "ctx is NULL");
    if (seq < 0 || seq >= ctx->B) return fail(ctx, RA_ERR_INVALID_ARG, "seq %d out of range", seq);
    ctx->active[seq] = active ? 1 : 0;
    return RA_OK;
}

int ra_restore_queries(ra_ctx* ctx, int layer, const uint16_t* q, float scale, void* stream)
{
    int rc;
    if ((rc = check_bound(ctx)) != RA_OK) return rc;
    if ((rc = check_layer(ctx, layer)) != RA_OK) return rc;
    if (!ctx->scoring) return fail(ctx, RA_ERR_STATE, "context bound without the scored policy's query window");
    if (!q || !aligned16(q)) return fail(ctx, RA_ERR_INVALID_ARG, "q must be non-NULL and 16-byte aligned");
    cudaStream_t s = (cudaStream_t)stream;
    const size_t base = (size_t)layer * ctx->B;
    cudaError_t e = launch_restore_queries(ctx->lay, layer, q, ctx->g.data() + base, s);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "query window restore launch");
    // The normalisers of the loaded queries: each over the prompt and the cached rows at
    // positions up to its own (what it attended to at its step, as no eviction can come between).
    EvictParams p{};
    p.lay = ctx->lay;
    p.layer = layer;
    int n = 0;
    for (int b = 0; b < ctx->B; ++b) {
        if (ctx->g[base + b] < 1) continue;
        p.trig[n] = (int16_t)b;
        p.trig_c[n] = ctx->c[base + b];
        p.trig_n[n] = ctx->c[base + b];
        p.trig_g[n] = ctx->g[base + b];
        ++n;
    }
    if (n == 0) return RA_OK;
    p.n_trig = n;
    AttnParams sp{};
    set_scale(&sp, scale);
    p.qk_scale_log2 = sp.qk_scale_log2;
    const double bytes = plan_scoring(ctx, &p, 1);
    {
        ProfScope ps(ctx, RA_KERNEL_SCORE_STATS, bytes, s);
        e = launch_score(p, 1, &ctx->tmap_ks, &ctx->tmap_q, s);
        ps.done();
    }
    if (e != cudaSuccess) return cuda_fail(ctx, e, "window normaliser launch");
    if ((e = launch_score_merge(p, s)) != cudaSuccess) return cuda_fail(ctx, e, "window normaliser merge launch");
    return RA_OK;
}

int ra_append_kv(ra_ctx* ctx, int layer, const uint16_t* k_new, const uint16_t* v_new, void* stream)
{
    int rc;
    if ((rc = check_bound(ctx)) != RA_OK) return rc;
    if ((rc = check_layer(ctx, layer)) != RA_OK) return rc;
    if (!k_new || !v_new || !aligned16(k_new) || !aligned16(v_new))
        return fail(ctx, RA_ERR_INVALID_ARG, "k_new/v_new must be non-NULL and 16-byte aligned");
    int n_active = 0;
    for (int b = 0; b < ctx->B; ++b) {
        if (!ctx->active[b]) continue;
        ++n_active;
        if (ctx->c[(size_t)layer * ctx->B + b] >= ctx->Cmax)
            return fail(ctx, RA_ERR_CAPACITY, "layer %d seq %d already caches K + 2r = %d generated tokens", layer, b,
                        ctx->Cmax);
    }
    if (n_active == 0) return RA_OK;
    AppendParams p{};
    p.lay = ctx->lay;
    p.layer = layer;
    p.k_new = k_new;
    p.v_new = v_new;
    fill_active(ctx, p.active);
    for (int b = 0; b < ctx->B; ++b) {
        p.seq_c[b] = ctx->c[(size_t)layer * ctx->B + b];
        p.seq_g[b] = ctx->g[(size_t)layer * ctx->B + b];
    }
    cudaStream_t s = (cudaStream_t)stream;
    ProfScope ps(ctx, RA_KERNEL_APPEND, 2.0 * n_active * ctx->KVH * kRowBytes * 2, s);
    cudaError_t e = launch_append(p, ctx->B, s);
    ps.done();
    if (e != cudaSuccess) return cuda_fail(ctx, e, "append launch");
    for (int b = 0; b < ctx->B; ++b) {
        if (!ctx->active[b]) continue;
        ctx->c[(size_t)layer * ctx->B + b] += 1;
        ctx->g[(size_t)layer * ctx->B + b] += 1;
    }
    return RA_OK;
}

int ra_evict(ra_ctx* ctx, int layer, int* n_fired, void* stream)
{
    int rc;
    if (n_fired) *n_fired = 0;
    if ((rc = check_bound(ctx)) != RA_OK) return rc;
    if ((rc = check_layer(ctx, layer)) != RA_OK) return rc;
    EvictParams p{};
    p.lay = ctx->lay;
    p.layer = layer;
    p.policy = ctx->policy;
    p.block = ctx->block;
    p.holefill = ctx->compaction == RA_COMPACT_HOLEFILL;
    int n = 0;
    double moved = 0;
    for (int b = 0; b < ctx->B; ++b) {
        if (!ctx->active[b]) continue;
        const int g = ctx->g[(size_t)layer * ctx->B + b], c = ctx->c[(size_t)layer * ctx->B + b];
        // section 2 / Appendix F trigger: every r steps, once the candidates exceed the budget
        if (g > 0 && g % ctx->r == 0 && c - ctx->r > ctx->K) {
            p.trig[n] = (int16_t)b;
            p.trig_c[n] = c;
            p.trig_n[n] = c - ctx->r;
            p.trig_g[n] = g;
            ++n;
            moved += (double)(ctx->K + ctx->r) * ctx->KVH;
        }
    }
    if (n == 0) return RA_OK;
    p.n_trig = n;
    if ((rc = run_eviction(ctx, p, moved, (cudaStream_t)stream)) != RA_OK) return rc;
    for (int i = 0; i < n; ++i) {
        const int b = p.trig[i];
        ctx->c[(size_t)layer * ctx->B + b] = ctx->K + ctx->r;
        ctx->nev[(size_t)layer * ctx->B + b] += 1;
    }
    if (n_fired) *n_fired = n;
    return RA_OK;
}

int ra_decode_attn(ra_ctx* ctx, int layer, const uint16_t* q, uint16_t* out, float scale, void* stream)
{
    int rc;
    if ((rc = check_bound(ctx)) != RA_OK) return rc;
    if ((rc = check_layer(ctx, layer)) != RA_OK) return rc;
    if (!q || !out || !aligned16(q) || !aligned16(out))
        return fail(ctx, RA_ERR_INVALID_ARG, "q/out must be non-NULL and 16-byte aligned");
    AttnParams p{};
    p.lay = ctx->lay;
    p.layer = layer;
    p.q = q;
    p.out = out;
    p.partial = ctx->lay.partial;
    p.arrive = ctx->lay.arrive;
    p.qring = ctx->lay.qring;
    p.ring_off = -1;  // the step's token is already appended: its query is step g
    int n_active = 0;
    int ctas = 0;
    double rows = 0;
    int shape = kAttnWide;
    if ((rc = plan_attention(ctx, layer, 0, &p, &n_active, &ctas, &rows, &shape)) != RA_OK) return rc;
    if (n_active == 0) return RA_OK;
    set_scale(&p, scale);
    cudaStream_t s = (cudaStream_t)stream;
    ProfScope ps(ctx, RA_KERNEL_ATTN, rows * 2 * kRowBytes + 2.0 * n_active * ctx->H * kRowBytes, s);
    cudaError_t e = launch_attention(shape, p, &ctx->tmap_k[shape], &ctx->tmap_v[shape], ctas, s);
    ps.done();
    if (e != cudaSuccess) return cuda_fail(ctx, e, "attention launch");
    return RA_OK;
}

namespace {
int decode_layer_impl(ra_ctx* ctx, int layer, const uint16_t* q, const uint16_t* k_new, const uint16_t* v_new,
                      uint16_t* out, float scale, void* stream, int plan_parity);
}

namespace {
// The host-side checks of one fused layer step (before anything changes).
int check_layer_call(ra_ctx* ctx, int layer, const uint16_t* q, const uint16_t* k_new, const uint16_t* v_new,
                     const uint16_t* out)
{
    int rc;
    if ((rc = check_bound(ctx)) != RA_OK) return rc;
    if ((rc = check_layer(ctx, layer)) != RA_OK) return rc;
    if (!q || !out || !k_new || !v_new || !aligned16(q) || !aligned16(out) || !aligned16(k_new) || !aligned16(v_new))
        return fail(ctx, RA_ERR_INVALID_ARG, "q/k_new/v_new/out must be non-NULL and 16-byte aligned");
    const size_t base = (size_t)layer * ctx->B;
    for (int b = 0; b < ctx->B; ++b)
        if (ctx->active[b] && ctx->c[base + b] >= ctx->Cmax)
            return fail(ctx, RA_ERR_CAPACITY, "layer %d seq %d already caches K + 2r = %d generated tokens", layer, b,
                        ctx->Cmax);
    return RA_OK;
}

// The start of a decode step of the whole stack (ra_decode_step, or ra_decode_layer of layer 0):
// wait for the evicted sets computed during the previous step, launch the next step's on the
// side stream, and run every layer's round of the sequences that fire now and have those sets,
// in one launch.  It needs none of the step's rows: in both layouts each layer's attention then
// appends its token into the last slot, as after an eviction inside the layer's own call.
int step_prologue(ra_ctx* ctx, cudaStream_t s)
{
    cudaError_t e;
    const bool serve = plan_usable(ctx);
    if (ctx->plan_pending) {  // the evicted sets of this step, computed during the previous one
        if ((e = cudaStreamWaitEvent(s, ctx->plan_ev, 0)) != cudaSuccess) return cuda_fail(ctx, e, "plan wait");
        ctx->plan_pending = false;
    }
    const int cur = ctx->parity, nxt = 1 - cur;
    std::fill(ctx->plan_g.begin() + (size_t)nxt * ctx->L * ctx->B, ctx->plan_g.begin() + (size_t)(nxt + 1) * ctx->L * ctx->B,
              -1);
    if (serve) {
        // The sequences whose trigger fires at the next step (from layer 0's counters after this
        // step): their evicted sets in every layer, computed on the side stream beside this step.
        // The fork orders the plan after the previous step, the last reader of half nxt.
        EvictParams pp{};
        pp.lay = ctx->lay;
        pp.policy = ctx->policy;
        pp.block = ctx->block;
        pp.holefill = ctx->compaction == RA_COMPACT_HOLEFILL;
        pp.ev_exact = (ctx->evict_mode & RA_EVICT_EXACT) ? 1 : 0;
        pp.ev_plan_parity = nxt;
        const bool read_pos = keys_read_positions(ctx);
        int n = 0;
        for (int b = 0; b < ctx->B; ++b) {
            if (!ctx->active[b]) continue;
            const int g1 = ctx->g[b] + 1, c1 = ctx->c[b] + 1;
            const bool fires = g1 % ctx->r == 0 && c1 - ctx->r > ctx->K;
            if (fires && read_pos) continue;  // this step rewrites the positions the keys would read
            const int g2 = g1 + 1, c2 = (fires ? ctx->K + ctx->r : c1) + 1;
            if (g2 % ctx->r == 0 && c2 - ctx->r > ctx->K && c2 - ctx->r <= ctx->K + ctx->r) {
                pp.trig[n] = (int16_t)b;
                pp.trig_admit[n] = (uint16_t)ctx->admits[b];
                pp.trig_g[n] = g2;
                pp.trig_n[n] = c2 - ctx->r;
                ++n;
            }
        }
        if (n > 0) {
            pp.n_trig = n;
            if ((e = cudaEventRecord(ctx->fork_ev, s)) != cudaSuccess ||
                (e = cudaStreamWaitEvent(ctx->side, ctx->fork_ev, 0)) != cudaSuccess)
                return cuda_fail(ctx, e, "plan fork");
            {
                ProfScope ps(ctx, RA_KERNEL_PLAN, 0.0, ctx->side);
                e = launch_plan(pp, ctx->sms, ctx->side);
                ps.done();
            }
            if (e != cudaSuccess) return cuda_fail(ctx, e, "plan launch");
            if ((e = cudaEventRecord(ctx->plan_ev, ctx->side)) != cudaSuccess) return cuda_fail(ctx, e, "plan record");
            ctx->plan_pending = true;
            for (int i = 0; i < n; ++i)
                for (int l = 0; l < ctx->L; ++l) {
                    const size_t k = (size_t)nxt * ctx->L * ctx->B + (size_t)l * ctx->B + pp.trig[i];
                    ctx->plan_g[k] = pp.trig_g[i];
                    ctx->plan_n[k] = pp.trig_n[i];
                }
        }
    }
    // The sequences that fire at this step in every layer alike, with every layer's evicted set
    // computed ahead: all their rounds in one launch, in place, before the first layer: the
    // survivors move down (ordered) or the evicted slots are refilled from the newest rows
    // (order-free), and the layers then append the token as usual.
    if (serve) {
        const bool fill = ctx->compaction == RA_COMPACT_HOLEFILL;
        EvictParams sp{};
        sp.lay = ctx->lay;
        sp.ev_plan_parity = cur;
        sp.holefill = fill ? 1 : 0;
        sp.pending = 1;
        int n = 0;
        double moved = 0;
        for (int b = 0; b < ctx->B; ++b) {
            if (!ctx->active[b]) continue;
            const int g = ctx->g[b], c = ctx->c[b];
            if ((g + 1) % ctx->r != 0 || c + 1 - ctx->r <= ctx->K) continue;
            bool all = true;
            for (int l = 0; l < ctx->L && all; ++l) {
                const size_t i = (size_t)l * ctx->B + b, k = (size_t)cur * ctx->L * ctx->B + i;
                all = ctx->g[i] == g && ctx->c[i] == c && ctx->plan_g[k] == g + 1 && ctx->plan_n[k] == c + 1 - ctx->r;
            }
            if (!all) continue;
            sp.trig[n] = (int16_t)b;
            sp.trig_c[n] = c;
            sp.trig_n[n] = c + 1 - ctx->r;
            sp.trig_g[n] = g + 1;
            ++n;
            // rows moved per head: the survivors below the token (ordered), the m refills (order-free)
            moved += (double)(fill ? c + 1 - ctx->r - ctx->K : ctx->K + ctx->r - 1) * ctx->KVH * ctx->L;
        }
        if (n > 0) {
            sp.n_trig = n;
            {
                ProfScope ps(ctx, RA_KERNEL_STACK, moved * 2.0 * (2 * kRowBytes + 4), s);
                e = fill ? launch_fill_stack(sp, ctx->L, s) : launch_compact_stack(sp, ctx->L, s);
                ps.done();
            }
            if (e != cudaSuccess) return cuda_fail(ctx, e, "whole-stack compaction launch");
            for (int i = 0; i < n; ++i)
                for (int l = 0; l < ctx->L; ++l) {
                    const size_t k = (size_t)l * ctx->B + sp.trig[i];
                    ctx->c[k] = ctx->K + ctx->r - 1;  // rows left before the step's token is written (last)
                    ctx->nev[k] += 1;
                }
            ctx->no_early_once = true;
        }
    }
    ctx->step_open = true;
    ctx->step_cur = cur;
    return RA_OK;
}

// The end of the step: join the side stream (the plan finished long before the last layer), so
// that once the caller's stream completes, so has everything the step launched; then the plan
// halves swap roles.
int step_epilogue(ra_ctx* ctx, cudaStream_t s)
{
    if (!ctx->step_open) return RA_OK;
    ctx->step_open = false;
    ctx->parity = 1 - ctx->step_cur;
    if (ctx->plan_pending) {
        const cudaError_t e = cudaStreamWaitEvent(s, ctx->plan_ev, 0);
        if (e != cudaSuccess) return cuda_fail(ctx, e, "plan join");
        ctx->plan_pending = false;
    }
    return RA_OK;
}
}  // namespace

int ra_decode_layer(ra_ctx* ctx, int layer, const uint16_t* q, const uint16_t* k_new, const uint16_t* v_new,
                    uint16_t* out, float scale, void* stream)
{
    // Layers called in order 0 .. L-1 form a step: layer 0 opens it (the evicted sets computed
    // during the previous step; with ordered compaction every layer's round of the firing
    // sequences in one launch), layer L-1 closes it.  Any other order is still correct: the
    // sets computed ahead are used only where the counters they assumed still hold.
    int rc;
    if ((rc = check_layer_call(ctx, layer, q, k_new, v_new, out)) != RA_OK) return rc;
    cudaStream_t s = (cudaStream_t)stream;
    if (layer == 0) {
        if (ctx->step_open && (rc = step_epilogue(ctx, s)) != RA_OK) return rc;
        if ((rc = step_prologue(ctx, s)) != RA_OK) return rc;
    }
    rc = decode_layer_impl(ctx, layer, q, k_new, v_new, out, scale, stream, ctx->step_open ? ctx->step_cur : -1);
    if (layer == ctx->L - 1 && ctx->step_open) {
        const int rc_end = step_epilogue(ctx, s);
        if (rc == RA_OK) rc = rc_end;
    }
    return rc;
}

namespace {
// plan_parity >= 0: evicted sets computed ahead into that half of the plan buffer may be used
// (inside a step whose prologue has ordered the stream after their computation)
int decode_layer_impl(ra_ctx* ctx, int layer, const uint16_t* q, const uint16_t* k_new, const uint16_t* v_new,
                      uint16_t* out, float scale, void* stream, int plan_parity)
{
    int rc;
    if ((rc = check_layer_call(ctx, layer, q, k_new, v_new, out)) != RA_OK) return rc;
    const size_t base = (size_t)layer * ctx->B;
    cudaStream_t s = (cudaStream_t)stream;
    cudaError_t e;
    std::vector<int32_t> old_rows((size_t)ctx->B, -1);  // sequences the attention launch compacts: rows before
    // The attention pass compacts (time order kept) when each tile's evicted rows fit its 64-bit mask.
    const bool fuse_compaction = ctx->compaction == RA_COMPACT_FUSED && ctx->r <= 64;  // tiles have <= 64 rows
    // 1. Eviction first, with the step's token pending: it is the newest slot, so it is never a
    //    candidate, and evicting before writing it gives the same state as append-then-evict.
    //    With ordered compaction only the selection runs here: the attention pass below reads
    //    the old region anyway and writes the survivors to the new one as it goes.
    EvictParams ep{};
    ep.lay = ctx->lay;
    ep.layer = layer;
    ep.policy = ctx->policy;
    ep.block = ctx->block;
    ep.holefill = ctx->compaction == RA_COMPACT_HOLEFILL;
    // The selection reads nothing its predecessor (the previous layer's attention) writes: Philox
    // needs no input, and positions were last written by this layer's previous step, which has
    // completed (every kernel before the predecessor has).  The scored policy reads scores its
    // predecessor computes, and with one layer the predecessor is this layer's previous step.
    ep.early = (ctx->policy != RA_POLICY_SNAPKV && ctx->L >= 2) ? 1 : 0;
    const int score_early = ctx->L >= 2 ? 1 : 0;  // the scoring pass reads only older kernels' output
    ep.pending = 1;  // the step's token is appended by the attention launch below
    int n = 0;
    double moved = 0;
    for (int b = 0; b < ctx->B; ++b) {
        if (!ctx->active[b]) continue;
        const int g1 = ctx->g[base + b] + 1, c1 = ctx->c[base + b] + 1;
        if (g1 % ctx->r == 0 && c1 - ctx->r > ctx->K) {
            ep.trig[n] = (int16_t)b;
            ep.trig_c[n] = c1 - 1;
            ep.trig_n[n] = c1 - ctx->r;
            ep.trig_g[n] = g1;
            ++n;
            moved += (double)(ctx->K + ctx->r - 1) * ctx->KVH;
        }
    }
    double compacted = 0;  // rows the attention launch writes as compaction
    if (n > 0 && plan_parity >= 0 && !ep.holefill && !fuse_compaction && plan_usable(ctx)) {
        bool all = true;  // every triggered sequence's evicted sets were computed ahead for this round
        for (int i = 0; i < n && all; ++i) {
            const size_t k = (size_t)plan_parity * ctx->L * ctx->B + (size_t)layer * ctx->B + ep.trig[i];
            all = ctx->plan_g[k] == ep.trig_g[i] && ctx->plan_n[k] == ep.trig_n[i];
        }
        if (all) {
            ep.ev_plan = ctx->lay.evplan;
            ep.ev_plan_parity = plan_parity;
        }
    }
    if (n > 0) {
        ep.n_trig = n;
        if ((rc = run_eviction(ctx, ep, moved, s, fuse_compaction, score_early)) != RA_OK) return rc;
        for (int i = 0; i < n; ++i) {
            const int b = ep.trig[i];
            ctx->nev[base + b] += 1;
            if (fuse_compaction) {
                old_rows[b] = ep.trig_c[i];
                compacted += (double)(ctx->K + ctx->r) * ctx->KVH;
            }
            ctx->c[base + b] = ctx->K + ctx->r - 1;  // rows left before the token is written (last)
        }
    }
    // 2. Fused append + attention (+ merge of the split pieces).
    AttnParams p{};
    p.lay = ctx->lay;
    p.layer = layer;
    p.q = q;
    p.out = out;
    p.k_new = k_new;
    p.v_new = v_new;
    p.partial = ctx->lay.partial;
    p.arrive = ctx->lay.arrive;
    p.qring = ctx->lay.qring;
    p.ring_off = 0;  // the query of step g + 1
    int n_active = 0, ctas = 0;
    double rows = 0;
    int shape = kAttnWide;
    if ((rc = plan_attention(ctx, layer, 1, &p, &n_active, &ctas, &rows, &shape, &old_rows)) != RA_OK)
        return rc;
    if (n_active == 0) return RA_OK;
    set_scale(&p, scale);
    // The kernel may request its first K/V tiles before its predecessor finishes when that
    // predecessor cannot be writing this layer's cache or tables: no eviction of this layer at
    // this step (else it is this layer's compaction) and more than one layer (else it is this
    // layer's previous step).  Kernels let successors start only after their own wait, so
    // everything older than the predecessor has completed.
    p.early = (n == 0 && ctx->L >= 2 && !ctx->no_early_once) ? 1 : 0;
    ctx->no_early_once = false;
    {
        // rows read (a new token's from the caller), a new token's row written, q read, out written
        int n_pending = 0;
        for (int b = 0; b < ctx->B; ++b) n_pending += (int)((p.pending[b >> 5] >> (b & 31)) & 1u);
        // (a compacting head's survivors are written once more, with their positions)
        ProfScope ps(ctx, RA_KERNEL_ATTN,
                     rows * 2 * kRowBytes + 2.0 * n_active * ctx->H * kRowBytes +
                         (double)n_pending * ctx->KVH * 2 * kRowBytes + compacted * (2 * kRowBytes + 8),
                     s);
        e = launch_attention(shape, p, &ctx->tmap_k[shape], &ctx->tmap_v[shape], ctas, s);
        ps.done();
    }
    if (e != cudaSuccess) return cuda_fail(ctx, e, "attention launch");
    for (int b = 0; b < ctx->B; ++b) {
        if (!ctx->active[b]) continue;
        ctx->c[base + b] += 1;
        ctx->g[base + b] += 1;
    }
    return RA_OK;
}

}  // namespace

int ra_decode_step(ra_ctx* ctx, const uint16_t* q_all, const uint16_t* k_all, const uint16_t* v_all, uint16_t* out_all,
                   float scale, void* stream)
{
    int rc;
    if ((rc = check_bound(ctx)) != RA_OK) return rc;
    if (!q_all || !k_all || !v_all || !out_all) return fail(ctx, RA_ERR_INVALID_ARG, "NULL argument");
    // validate every layer's capacity first so that a failing step changes nothing
    for (int l = 0; l < ctx->L; ++l)
        for (int b = 0; b < ctx->B; ++b)
            if (ctx->active[b] && ctx->c[(size_t)l * ctx->B + b] >= ctx->Cmax)
                return fail(ctx, RA_ERR_CAPACITY, "layer %d seq %d is full (evict not called)", l, b);
    const size_t qs = (size_t)ctx->B * ctx->H * kHeadDim, ks = (size_t)ctx->B * ctx->KVH * kHeadDim;
    cudaStream_t s = (cudaStream_t)stream;
    if (ctx->step_open && (rc = step_epilogue(ctx, s)) != RA_OK) return rc;  // a per-layer step left open
    if ((rc = step_prologue(ctx, s)) != RA_OK) return rc;
    for (int l = 0; l < ctx->L; ++l)
        if ((rc = decode_layer_impl(ctx, l, q_all + l * qs, k_all + l * ks, v_all + l * ks, out_all + l * qs, scale,
                                    stream, ctx->step_cur)) != RA_OK)
            break;
    const int rc_end = step_epilogue(ctx, s);
    return rc != RA_OK ? rc : rc_end;
}

int ra_get_counters(const ra_ctx* ctx, int seq, int layer, int32_t* g, int32_t* c, int32_t* n_evictions)
{
    if (!ctx) return fail(nullptr, RA_ERR_INVALID_ARG, "ctx is NULL");
    if (seq < 0 || seq >= ctx->B || layer < 0 || layer >= ctx->L)
        return fail(const_cast<ra_ctx*>(ctx), RA_ERR_INVALID_ARG, "seq/layer out of range");
    const size_t i = (size_t)layer * ctx->B + seq;
    if (g) *g = ctx->g[i];
    if (c) *c = ctx->c[i];
    if (n_evictions) *n_evictions = ctx->nev[i];
    return RA_OK;
}

static int read_region(ra_ctx* ctx, int layer, int seq, int kv_head, int32_t* reg, cudaStream_t s)
{
    cudaError_t e;
    if ((e = cudaStreamSynchronize(s)) != cudaSuccess) return cuda_fail(ctx, e, "stream sync");
    if ((e = cudaMemcpy(reg, ctx->lay.region + ((size_t)layer * ctx->B + seq) * ctx->KVH + kv_head, 4,
                        cudaMemcpyDeviceToHost)) != cudaSuccess)
        return cuda_fail(ctx, e, "region read");
    return RA_OK;
}

int ra_get_positions(ra_ctx* ctx, int layer, int seq, int kv_head, int32_t* host_pos, int capacity, int* n,
                     void* stream)
{
    int rc;
    if ((rc = check_bound(ctx)) != RA_OK) return rc;
    if ((rc = check_layer(ctx, layer)) != RA_OK) return rc;
    if (seq < 0 || seq >= ctx->B || kv_head < 0 || kv_head >= ctx->KVH || !n)
        return fail(ctx, RA_ERR_INVALID_ARG, "seq/kv_head out of range or n NULL");
    const int c = ctx->c[(size_t)layer * ctx->B + seq];
    *n = c;
    if (capacity < c || (c > 0 && !host_pos)) return fail(ctx, RA_ERR_INVALID_ARG, "capacity %d < %d", capacity, c);
    int32_t reg;
    if ((rc = read_region(ctx, layer, seq, kv_head, &reg, (cudaStream_t)stream)) != RA_OK) return rc;
    cudaError_t e;
    if (c > 0 && (e = cudaMemcpy(host_pos, ctx->lay.pos + (size_t)reg * ctx->Cmax, (size_t)c * 4,
                                 cudaMemcpyDeviceToHost)) != cudaSuccess)
        return cuda_fail(ctx, e, "positions read");
    return RA_OK;
}

int ra_get_kv(ra_ctx* ctx, int layer, int seq, int kv_head, uint16_t* host_k, uint16_t* host_v, int capacity_rows,
              int* n_rows, void* stream)
{
    int rc;
    if ((rc = check_bound(ctx)) != RA_OK) return rc;
    if ((rc = check_layer(ctx, layer)) != RA_OK) return rc;
    if (seq < 0 || seq >= ctx->B || kv_head < 0 || kv_head >= ctx->KVH || !n_rows)
        return fail(ctx, RA_ERR_INVALID_ARG, "seq/kv_head out of range or n_rows NULL");
    const int lp = ctx->lp[seq], c = ctx->c[(size_t)layer * ctx->B + seq];
    *n_rows = lp + c;
    if (capacity_rows < lp + c || !host_k || !host_v)
        return fail(ctx, RA_ERR_INVALID_ARG, "capacity %d < %d rows", capacity_rows, lp + c);
    int32_t reg;
    if ((rc = read_region(ctx, layer, seq, kv_head, &reg, (cudaStream_t)stream)) != RA_OK) return rc;
    const long long grow = ctx->lay.gen_row0 + (long long)reg * ctx->Cmax;
    cudaError_t e;
    for (int w = 0; w < 2; ++w) {
        const uint16_t* pool = w ? ctx->lay.vpool : ctx->lay.kpool;
        uint16_t* dst = w ? host_v : host_k;
        for (int p0 = 0; p0 < lp; p0 += kPromptPage) {  // the prompt, page by page
            const int32_t page = ctx->pages[(size_t)seq * ctx->max_pages + p0 / kPromptPage];
            const long long prow = prompt_row(ctx->lay, layer, page, kv_head, 0);
            const int n = std::min(kPromptPage, lp - p0);
            if ((e = cudaMemcpy(dst + (size_t)p0 * kHeadDim, pool + prow * kHeadDim, (size_t)n * kRowBytes,
                                cudaMemcpyDeviceToHost)) != cudaSuccess)
                return cuda_fail(ctx, e, "prompt rows read");
        }
        if (c > 0 && (e = cudaMemcpy(dst + (size_t)lp * kHeadDim, pool + grow * kHeadDim, (size_t)c * kRowBytes,
                                     cudaMemcpyDeviceToHost)) != cudaSuccess)
            return cuda_fail(ctx, e, "generated rows read");
    }
    return RA_OK;
}

int ra_get_scores(ra_ctx* ctx, int layer, int seq, int kv_head, float* host_scores, int capacity, int* n,
                  void* stream)
{
    int rc;
    if ((rc = check_bound(ctx)) != RA_OK) return rc;
    if ((rc = check_layer(ctx, layer)) != RA_OK) return rc;
    if (seq < 0 || seq >= ctx->B || kv_head < 0 || kv_head >= ctx->KVH || !n)
        return fail(ctx, RA_ERR_INVALID_ARG, "seq/kv_head out of range or n NULL");
    if (!ctx->scoring) return fail(ctx, RA_ERR_STATE, "context bound without the scored policy's buffers");
    const int N = ctx->score_n[(size_t)layer * ctx->B + seq];
    *n = N;
    if (capacity < N || (N > 0 && !host_scores)) return fail(ctx, RA_ERR_INVALID_ARG, "capacity %d < %d", capacity, N);
    cudaError_t e;
    if ((e = cudaStreamSynchronize((cudaStream_t)stream)) != cudaSuccess) return cuda_fail(ctx, e, "stream sync");
    const float* src = ctx->lay.scores + (((size_t)layer * ctx->B + seq) * ctx->KVH + kv_head) * ctx->Cmax;
    if (N > 0 && (e = cudaMemcpy(host_scores, src, (size_t)N * 4, cudaMemcpyDeviceToHost)) != cudaSuccess)
        return cuda_fail(ctx, e, "scores read");
    return RA_OK;
}

int ra_check_device(ra_ctx* ctx, void* stream)
{
    int rc;
    if ((rc = check_bound(ctx)) != RA_OK) return rc;
    cudaError_t e;
    if ((e = cudaStreamSynchronize((cudaStream_t)stream)) != cudaSuccess) return cuda_fail(ctx, e, "stream sync");
    int32_t w = 0;
    if ((e = cudaMemcpy(&w, ctx->lay.err, 4, cudaMemcpyDeviceToHost)) != cudaSuccess) return cuda_fail(ctx, e, "err read");
    if (w != 0) {  // reported once: clear it (the stream is idle, nothing else writes it now)
        const int32_t zero = 0;
        if ((e = cudaMemcpy(ctx->lay.err, &zero, 4, cudaMemcpyHostToDevice)) != cudaSuccess)
            return cuda_fail(ctx, e, "err clear");
    }
    if (w == kDeviceErrTimeout) return fail(ctx, RA_ERR_DEVICE_TIMEOUT, "a kernel gave up a bounded wait");
    if (w == kDeviceErrPlan) return fail(ctx, RA_ERR_STATE, "device eviction plan inconsistent with host counters");
    if (w != 0) return fail(ctx, RA_ERR_STATE, "device error word %d", w);
    return RA_OK;
}

int ra_debug_timeout_probe(ra_ctx* ctx, uint64_t limit_ns, void* stream)
{
    int rc;
    if ((rc = check_bound(ctx)) != RA_OK) return rc;
    if (limit_ns < 1000ull || limit_ns > 100000000ull)
        return fail(ctx, RA_ERR_INVALID_ARG, "limit_ns %llu outside [1e3, 1e8]", (unsigned long long)limit_ns);
    cudaError_t e = launch_timeout_probe(ctx->lay.err, limit_ns, (cudaStream_t)stream);
    return e == cudaSuccess ? RA_OK : cuda_fail(ctx, e, "timeout probe launch");
}

int ra_profile_enable(ra_ctx* ctx, int on)
{
    if (!ctx) return fail(nullptr, RA_ERR_INVALID_ARG, "ctx is NULL");
    ctx->prof = on != 0;
    return RA_OK;
}

int ra_profile_reset(ra_ctx* ctx)
{
    if (!ctx) return fail(nullptr, RA_ERR_INVALID_ARG, "ctx is NULL");
    int rc = collect_profile(ctx);
    for (int k = 0; k < RA_KERNEL_KINDS; ++k) {
        ctx->prof_ms[k] = 0;
        ctx->prof_n[k] = 0;
        ctx->prof_bytes[k] = 0;
        ctx->launch_n[k] = 0;
        ctx->launch_bytes[k] = 0;
    }
    return rc;
}

int ra_profile_read(ra_ctx* ctx, int kind, double* total_ms, int64_t* launches, double* algorithmic_bytes)
{
    if (!ctx) return fail(nullptr, RA_ERR_INVALID_ARG, "ctx is NULL");
    if (kind < 0 || kind >= RA_KERNEL_KINDS) return fail(ctx, RA_ERR_INVALID_ARG, "bad kernel kind %d", kind);
    int rc = collect_profile(ctx);
    if (rc != RA_OK) return rc;
    if (total_ms) *total_ms = ctx->prof_ms[kind];
    if (launches) *launches = ctx->launch_n[kind];
    if (algorithmic_bytes) *algorithmic_bytes = ctx->launch_bytes[kind];
    return RA_OK;
}

void ra_destroy(ra_ctx* ctx)
{
    if (!ctx) return;
    if (ctx->side) {
        cudaStreamSynchronize(ctx->side);
        cudaStreamDestroy(ctx->side);
        cudaEventDestroy(ctx->fork_ev);
        cudaEventDestroy(ctx->plan_ev);
    }
    for (auto& pr : ctx->pending) {
        cudaEventSynchronize(pr.stop);
        cudaEventDestroy(pr.start);
        cudaEventDestroy(pr.stop);
    }
    for (auto e : ctx->pool) cudaEventDestroy(e);
    delete ctx;
}

}  // extern "C"

// ----------------------------------------------------------------------------
// ra_decode_attn_noalloc: decode attention whose split-K scratch lives in a
// fixed device array of this library instead of the caller's arena.
//
// The array below is allocated by the CUDA module loader when the library is
// loaded on a device and is held until the process exits.  Host code must not
// pass the symbol itself to a kernel (on the host it names a shadow, not device
// memory): its device address is looked up once per device with
// cudaGetSymbolAddress while that device is current, and that address is what
// the kernels receive.
// ----------------------------------------------------------------------------
namespace {

constexpr size_t kNoAllocScratchBytes = 8u << 20;  // 8 MiB per device
constexpr int kNoAllocMaxDevices = 64;

static __device__ __align__(256) float g_noalloc_scratch[kNoAllocScratchBytes / sizeof(float)];

std::mutex g_noalloc_mu;
float* g_noalloc_ptr[kNoAllocMaxDevices] = {nullptr};

int noalloc_scratch(ra_ctx* ctx, int dev, float** out)
{
    if (dev < 0 || dev >= kNoAllocMaxDevices) return fail(ctx, RA_ERR_UNSUPPORTED, "device %d out of range", dev);
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (!g_noalloc_ptr[dev]) {
        void* p = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess || !p) return cuda_fail(ctx, e, "cudaGetSymbolAddress(scratch)");
        g_noalloc_ptr[dev] = static_cast<float*>(p);
    }
    *out = g_noalloc_ptr[dev];
    return RA_OK;
}

}  // namespace

extern "C" int ra_decode_attn_noalloc(ra_ctx* ctx, int layer, const uint16_t* q, uint16_t* out, float scale,
                                      void* stream)
{
    int rc;
    if ((rc = check_bound(ctx)) != RA_OK) return rc;
    if ((rc = check_layer(ctx, layer)) != RA_OK) return rc;
    if (!q || !out || !aligned16(q) || !aligned16(out))
        return fail(ctx, RA_ERR_INVALID_ARG, "q/out must be non-NULL and 16-byte aligned");
    AttnParams p{};
    p.lay = ctx->lay;
    p.layer = layer;
    p.q = q;
    p.out = out;
    p.qring = ctx->lay.qring;
    p.ring_off = -1;
    int n_active = 0, ctas = 0;
    double rows = 0;
    int shape = kAttnWide;
    if ((rc = plan_attention(ctx, layer, 0, &p, &n_active, &ctas, &rows, &shape)) != RA_OK) return rc;
    if (n_active == 0) return RA_OK;
    set_scale(&p, scale);
    // [arrival counters, one int per (seq, KV head)][partial records, one per (chunk, head) piece]
    const size_t counters = align_up((size_t)ctx->B * ctx->KVH * sizeof(int32_t), kAlign);
    const size_t need =
        counters + (size_t)(p.nchunks + (long long)ctx->B * ctx->KVH) * partial_stride(ctx->G) * sizeof(float);
    if (need > kNoAllocScratchBytes)
        return fail(ctx, RA_ERR_CAPACITY, "layer needs %zu bytes of split-K scratch; the fixed array holds %zu", need,
                    kNoAllocScratchBytes);
    float* scratch = nullptr;
    if ((rc = noalloc_scratch(ctx, ctx->device, &scratch)) != RA_OK) return rc;
    cudaStream_t s = (cudaStream_t)stream;
    p.arrive = reinterpret_cast<int32_t*>(scratch);
    p.partial = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(scratch) + counters);
    // the counters must start at zero; the array keeps whatever the previous call left
    cudaError_t e = cudaMemsetAsync(scratch, 0, counters, s);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "scratch counter clear");
    e = launch_attention(shape, p, &ctx->tmap_k[shape], &ctx->tmap_v[shape], ctas, s);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "attention launch");
    return RA_OK;
}
