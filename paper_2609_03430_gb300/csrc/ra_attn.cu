// ra_attn.cu -- GQA split-K flash-decode attention over the per-head caches (sm_103a).
//
// Computes, for every active sequence b and query head qh (KV head h = qh / G),
//     o = sum_i softmax_i(scale * q . k_i) v_i
// over the prompt rows and the cached generated rows of (b, h) -- section 2
// ("Notation"), with the grouped-query sharing of Appendix F.  In the fused
// form the step's new token (Appendix F: appended post-RoPE every step) is the
// last generated row: it is read from the caller's k_new/v_new rows, placed in
// its head's last tile, attended, and written into the cache by the warp that
// consumes that tile.
//
// Work split: every head is cut into tiles of TILE rows (its prompt rows, then
// its generated rows); the tiles of all heads of the layer are laid end to end
// (sequence-major, then KV head) and cut into equal chunks of W tiles, one per
// warp, so every warp makes the same number of pipeline trips.  A
// warp runs its own pipeline: lane 0 streams the tiles of K and V -- each as
// two 64-channel boxes stored with the 128-byte swizzle -- plus, at the first
// tile of each head piece, the G query rows, into a ring of SPW shared-memory
// stages with 2-D TMA loads completing on per-stage mbarriers; all 32 lanes
// consume.  A head that fits in one chunk is finished in registers.  Otherwise
// each (head, chunk) piece writes an fp32 partial (unnormalised o, running max
// m, sum l) to record `chunk + head` -- unique because chunks and heads both
// advance monotonically through the tile order -- and the last warp to finish
// a piece of that head (an arrival counter per head) merges all of them.
//
// With the scored comparator's buffers bound, the warp that consumes a head's
// first tile also copies the head's G query rows into the query window, and
// whoever finishes a head records each query's softmax normaliser beside it:
// until the next eviction, the window score needs exactly these normalisers.
//
// Per-warp compute: the contraction of the G query rows with a tile of cache
// rows runs on the tensor cores (mma.sync m16n8k16, bf16 in, fp32 accumulate):
// S = Q K^T takes the query heads as the 16 M rows (G <= 8 used, the rest
// zero) and 8 cache rows per N tile; O += P V reuses the S accumulator
// fragments as the A operand (P rounded to bf16).  Q fragments stay in
// registers for a whole head piece; K and V are read with ldmatrix from TMA
// tiles stored with the 128-byte swizzle, so the reads are bank-conflict free.
// Each lane owns one query head (lane / 4): the softmax statistics need only
// two shuffles per 16 rows, and O needs no cross-lane reduction.  The softmax
// is online in base 2 with the scale folded into one multiply; the running max
// is only raised when a batch exceeds it by more than 2^8 (the result is
// unchanged up to rounding, as softmax is shift invariant), so rescaling the
// accumulators is rare.
//
// The narrow build (RA_ATTN_TRANSPOSED) takes the products transposed, so
// that the 16-row M side holds cache rows and the 8-wide N side the query
// heads: S^T = K Q^T (A = 16 cache rows x 16 channels of K; B = the same Q
// fragments), then O^T += V^T P^T (A = V read transposed; B = P^T, the S^T
// accumulators rounded to bf16 and transposed in registers with movmatrix).
// That is half the products per row.  A lane then holds rows lane / 4 and
// lane / 4 + 8 of a batch for query heads 2 (lane % 4) and 2 (lane % 4) + 1,
// and a raised max needs a reduction over the 8 lanes of a head pair.  On
// small layers, where warps share sub-partitions, it measured 1.5% faster;
// the wide build keeps the other layout, which measured 2-4% faster there.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <limits.h>
#include <math.h>
#include <stdint.h>

#include "ra_internal.h"
#include "ra_ptx.cuh"

namespace ra {
namespace {

constexpr float kTau = 8.0f;                       // lazy-rescale threshold (log2 units)
constexpr uint64_t kWaitLimitNs = 2000000000ull;   // bounded mbarrier waits: 2 s
constexpr int kSmemBudget = 220 * 1024;
constexpr int kHalfCh = 64;                        // channels per swizzled TMA box (128 bytes)

// Kernel shape: rows per stage (a multiple of 16), stages per warp, warps per CTA
// (one CTA per SM; the warp count is capped by what fits in shared memory).  The library
// builds this file twice, into the namespaces attn_wide (48-row tiles, 4 warps: large
// layers) and attn_narrow (32-row tiles, 6 warps: small layers, finer work split).
#ifndef RA_ATTN_NS
#define RA_ATTN_NS attn_wide
#endif
#ifndef RA_ATTN_TILE
#define RA_ATTN_TILE 48
#endif
#ifndef RA_ATTN_SPW
#define RA_ATTN_SPW 2
#endif
#ifndef RA_ATTN_WARPS
#define RA_ATTN_WARPS 4
#endif
// Contraction layout: 0 = the query heads are the MMA's M rows (the wide shape); 1 = the cache rows
// are, transposed (the narrow shape).  See the comment at the top of the file.
#ifndef RA_ATTN_TRANSPOSED
#define RA_ATTN_TRANSPOSED 0
#endif

template <int G>
struct Cfg {
    static constexpr int TILE = RA_ATTN_TILE;                                // rows per stage
    static constexpr int HALF_BYTES = TILE * 128;                            // one 64-channel half of K or V
    static constexpr int KV_BYTES = 2 * HALF_BYTES;                          // a K (or V) tile
    static constexpr int Q_BYTES = G * kRowBytes;
    static constexpr int NT_OFF = 2 * KV_BYTES + Q_BYTES;  // the fused new token's K and V rows (unswizzled)
    static constexpr int STAGE_BYTES = (NT_OFF + 2 * kRowBytes + 1023) / 1024 * 1024;
    static constexpr int SPW = RA_ATTN_SPW;
    static constexpr int WARPS_FIT = kSmemBudget / (SPW * STAGE_BYTES);
    static constexpr int WARPS = WARPS_FIT < RA_ATTN_WARPS ? WARPS_FIT : RA_ATTN_WARPS;
    static constexpr int NSTAGE = WARPS * SPW;
    static constexpr size_t SMEM = 1024 + (size_t)NSTAGE * STAGE_BYTES + (size_t)NSTAGE * (16 + 8);
    // merge layout: LG lanes per query head, MCH channels per lane
    static constexpr int GP = G <= 1 ? 1 : (G <= 2 ? 2 : (G <= 4 ? 4 : 8));
    static constexpr int LG = 32 / GP;
    static constexpr int MCH = kHeadDim / LG;
    static_assert(G >= 1 && G <= 8, "the 16-row MMA holds up to 8 query heads");
    static_assert(TILE % 16 == 0 && TILE <= 256, "whole 16-row MMA batches; TMA box rows <= 256");
    static_assert(kPromptPage % TILE == 0, "a prompt tile lies inside one page");
    static_assert(HALF_BYTES % 1024 == 0, "128-byte-swizzled TMA boxes start 1024-byte aligned");
    static_assert(WARPS >= 2, "shared-memory budget too small");
    static_assert(SMEM <= 232448, "fits the 227 KB opt-in shared memory of sm_100+");
};

// Tile header flags; the chunk index sits above them (<< kFlagBits).
constexpr int kFirst = 1, kLast = 2, kNewTok = 4, kHead0 = 8, kCompact = 16, kFlagBits = 5;

// Producer-side walk over the warp's chunks (chunks and cursors count tiles).
struct TileIter {
    int chunk;                       // this warp's chunk (-1: not started)
    int f, end;                      // flattened tile cursor and end of the current chunk
    int b, h, k;                     // current sequence, KV head, tile within the head
    int nt, tp;                      // tiles in the head, prompt tiles among them
    int lp, gen;                     // prompt rows, generated rows (incl. a fused new token)
    bool comp;                       // the head compacts in this launch: its generated rows are the old region's
    long long pbase, grow;           // the head's prompt rows: pbase + page * KVH * kPromptPage + offset; first generated row
    const int32_t* ptab;             // the sequence's page table (null: its pages are page0, page0 + 1, ...)
    int page0;
    int pg_i, pg_cur, pg_next;       // page-table entry i of the current prompt tile, and entry i + 1 (read ahead)
    bool piece_start;
};

struct TileDesc {
    long long row;  // first cache row of the tile
    int n, hid, flags, chunk;
};

__device__ __forceinline__ int seq_head_tiles(const AttnParams& p, int b)
{
    return (p.seq_base[b + 1] - p.seq_base[b]) / p.lay.KVH;
}

template <bool COMPACT>
__device__ __forceinline__ void enter_head(TileIter& it, const AttnParams& p)
{
    const DevLayout& L = p.lay;
    it.lp = p.seq_lp[it.b];
    it.gen = p.seq_gen[it.b];
    it.tp = (it.lp + p.tile - 1) / p.tile;
    it.pbase = prompt_row(L, p.layer, 0, it.h, 0);
    it.page0 = p.seq_page0[it.b];
    it.ptab = it.page0 >= 0 ? nullptr : L.pages + (size_t)it.b * L.max_pages;
    it.pg_i = 0;
    if (it.lp > 0) {
        it.pg_cur = it.ptab ? __ldg(it.ptab) : it.page0;
        it.pg_next = it.lp > kPromptPage ? (it.ptab ? __ldg(it.ptab + 1) : it.page0 + 1) : 0;
    }
    it.comp = COMPACT && ((p.compacting[it.b >> 5] >> (it.b & 31)) & 1u);
    const int reg = it.comp ? L.plan[(size_t)(it.b * L.KVH + it.h) * (kPlanHeader + L.r)]  // the old region
                            : p.seq_region[it.b] * L.KVH + it.h;
    it.grow = L.gen_row0 + (long long)reg * L.Cmax;
    it.piece_start = true;
}

template <bool COMPACT>
__device__ void iter_init(TileIter& it, const AttnParams& p, int R0, int R1)
{
    it.f = R0;
    it.end = R1;
    int lo = 0, hi = p.lay.B - 1;  // largest b with seq_base[b] <= R0 (empty sequences skipped below)
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (p.seq_base[mid] <= R0) lo = mid; else hi = mid - 1;
    }
    int b = lo;
    while (b < p.lay.B && p.seq_base[b + 1] <= R0) ++b;
    it.b = b;
    it.nt = seq_head_tiles(p, b);
    const int off = R0 - p.seq_base[b];
    it.h = off / it.nt;
    it.k = off - it.h * it.nt;
    enter_head<COMPACT>(it, p);
}

// The warp's chunk (its index): false once it is done.
template <bool COMPACT>
__device__ bool iter_next_chunk(TileIter& it, const AttnParams& p, int warp_id)
{
    if (it.chunk >= 0 || warp_id >= p.nchunks) return false;
    it.chunk = warp_id;
    const int R0 = warp_id * p.W;
    iter_init<COMPACT>(it, p, R0, min(p.total, R0 + p.W));
    return true;
}

template <bool COMPACT>
__device__ bool iter_next(TileIter& it, const AttnParams& p, TileDesc& d, int warp_id)
{
    if (it.f >= it.end && !iter_next_chunk<COMPACT>(it, p, warp_id)) return false;
    const int T = p.tile;
    d.flags = (it.piece_start ? kFirst : 0) | (it.k == 0 ? kHead0 : 0);
    if (it.k < it.tp) {  // a prompt tile lies inside one page (kPromptPage is a multiple of T)
        const int p0 = it.k * T, pi = p0 / kPromptPage;
        if (pi != it.pg_i) {  // another page: the next one's entry was read ahead (a chunk may start mid-prompt)
            it.pg_cur = pi == it.pg_i + 1 ? it.pg_next : (it.ptab ? __ldg(it.ptab + pi) : it.page0 + pi);
            it.pg_i = pi;
            it.pg_next = (pi + 1) * kPromptPage < it.lp ? (it.ptab ? __ldg(it.ptab + pi + 1) : it.page0 + pi + 1) : 0;
        }
        d.row = it.pbase + (long long)it.pg_cur * p.lay.KVH * kPromptPage + p0 % kPromptPage;
        d.n = min(T, it.lp - p0);
    } else {
        const int kg = it.k - it.tp;
        d.row = it.grow + (long long)kg * T;
        d.n = min(T, it.gen - kg * T);
        if (p.k_new && ((p.pending[it.b >> 5] >> (it.b & 31)) & 1u) && kg * T + d.n == it.gen)
            d.flags |= kNewTok;  // its last row is the step's new token
        if (COMPACT && it.comp) d.flags |= kCompact;
    }
    if (it.k + 1 == it.nt || it.f + 1 == it.end) d.flags |= kLast;
    d.hid = it.b * p.lay.KVH + it.h;
    d.chunk = it.chunk;
    it.piece_start = false;
    ++it.k;
    ++it.f;
    if (it.k == it.nt && it.f < it.end) {  // next head (skipping finished sequences)
        if (++it.h == p.lay.KVH) {
            it.h = 0;
            do {
                ++it.b;
            } while (seq_head_tiles(p, it.b) == 0);
            it.nt = seq_head_tiles(p, it.b);
        }
        it.k = 0;
        enter_head<COMPACT>(it, p);
    }
    return true;
}

// Byte offset of (row j, 16-byte chunk c of 16) inside a swizzled K or V tile:
// two boxes of 64 channels; within a box the chunk index is xored with j mod 8.
template <int G>
__device__ __forceinline__ uint32_t swz(int j, int c)
{
    return (uint32_t)((c >> 3) * Cfg<G>::HALF_BYTES + j * 128 + (((c & 7) ^ (j & 7)) << 4));
}

__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], uint32_t addr)
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}

__device__ __forceinline__ void ldsm_x4_t(uint32_t (&r)[4], uint32_t addr)
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}

#if !RA_ATTN_TRANSPOSED
#pragma nv_diag_suppress 550  // d2, d3: the product's padding rows, discarded
// D[16x8] += A[16x16] B[16x8], bf16 inputs, fp32 accumulators.  Only rows 0..7 of A
// (the query heads) are nonzero, so only c0/c1 of the accumulator are kept.
__device__ __forceinline__ void mma_rows8(float& c0, float& c1, uint32_t a0, uint32_t a2, uint32_t b0, uint32_t b1)
{
    float d2, d3;
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%10, %11, %12, %13};"
        : "=f"(c0), "=f"(c1), "=f"(d2), "=f"(d3)
        : "r"(a0), "r"(0u), "r"(a2), "r"(0u), "r"(b0), "r"(b1), "f"(c0), "f"(c1), "f"(0.f), "f"(0.f));
    (void)d2;  // rows 8..15 of the product: padding
    (void)d3;
}
#pragma nv_diag_default 550
#endif

#if RA_ATTN_TRANSPOSED
// C[16x8] += A[16x16] B[16x8], bf16 inputs, fp32 accumulators (register-only: not volatile, so the
// compiler may interleave independent products).
__device__ __forceinline__ void mma16816(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1)
{
    asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Transpose of an 8x8 bf16 matrix held in fragment layout (lane l: row l / 4, columns 2 (l % 4) + {0, 1}).
__device__ __forceinline__ uint32_t movtrans(uint32_t x)
{
    uint32_t y;
    asm("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(y) : "r"(x));
    return y;
}
#endif

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi)
{
    return (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(lo)) |
           ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(hi)) << 16);
}

// The scored policy's window: the softmax normaliser of query head g of (b, KV head h) at this
// step, as (scale * log2 e, log2 sum_i exp2(scale * log2 e * q.k_i)), beside its query rows.
template <int G>
__device__ __forceinline__ void record_stats(const AttnParams& p, int b, int h, int g, float lse2)
{
    const int r = p.lay.r;
    int slot = (p.seq_g[b] + p.ring_off) % r;
    if (slot < 0) slot += r;
    p.lay.qstats[((((size_t)p.layer * p.lay.B + b) * p.lay.KVH + h) * r + slot) * G + g] =
        make_float2(p.qk_scale_log2, lse2);
}

// Merge every piece of head `hid` (pieces are partial records c0 + q + hid, q < P) into the
// bf16 output rows of its G query heads.  One warp, two rounds of L2 reads: first every lane
// reads the statistics of its pieces (lane q: piece q, q + 32, ...) and the warp reduces them
// to each query head's max M and normaliser L; then lanes split as (query head g, channel
// group), and for every piece load its max (one address per head: a broadcast) and their
// channels together, so the loads of all pieces are independent.  Partials come from other
// SMs: read through L2.
template <int G>
__device__ void merge_head(const AttnParams& p, int hid, int c0, int P, int lane)
{
    using C = Cfg<G>;
    const size_t rs = (size_t)partial_stride(G);
    const float* base = p.partial + (size_t)(c0 + hid) * rs;
    float M[G], Lh[G];
#pragma unroll
    for (int g = 0; g < G; ++g) {
        M[g] = -INFINITY;
        Lh[g] = 0.f;
    }
    for (int q = lane; q < P; q += 32)
#pragma unroll
        for (int g = 0; g < G; ++g) M[g] = fmaxf(M[g], __ldcg(base + q * rs + G * kHeadDim + g));
#pragma unroll
    for (int g = 0; g < G; ++g)
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) M[g] = fmaxf(M[g], __shfl_xor_sync(0xffffffffu, M[g], o));
    for (int q = lane; q < P; q += 32)
#pragma unroll
        for (int g = 0; g < G; ++g) {
            const float* st = base + q * rs + G * kHeadDim;
            Lh[g] = fmaf(exp2f(__ldcg(st + g) - M[g]), __ldcg(st + G + g), Lh[g]);
        }
#pragma unroll
    for (int g = 0; g < G; ++g)
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) Lh[g] += __shfl_xor_sync(0xffffffffu, Lh[g], o);

    const int g = lane / C::LG, sub = lane % C::LG;
    const int gg = g < G ? g : 0;  // lanes of padding heads shadow head 0 (results unused)
    float Mg = M[0], Lg = Lh[0];
#pragma unroll
    for (int k = 1; k < G; ++k)
        if (gg == k) {
            Mg = M[k];
            Lg = Lh[k];
        }
    const int ch0 = sub * C::MCH;
    float4 acc[C::MCH / 4];
#pragma unroll
    for (int j = 0; j < C::MCH / 4; ++j) acc[j] = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 4
    for (int q = 0; q < P; ++q) {
        const float* rec = base + q * rs;
        const float a = exp2f(__ldcg(rec + G * kHeadDim + gg) - Mg);
        const float4* o = reinterpret_cast<const float4*>(rec + gg * kHeadDim + ch0);
#pragma unroll
        for (int k = 0; k < C::MCH / 4; ++k) {
            const float4 v = __ldcg(o + k);
            acc[k].x = fmaf(a, v.x, acc[k].x);
            acc[k].y = fmaf(a, v.y, acc[k].y);
            acc[k].z = fmaf(a, v.z, acc[k].z);
            acc[k].w = fmaf(a, v.w, acc[k].w);
        }
    }
    if (g >= G) return;
    const float inv = 1.f / Lg;
    const int b = hid / p.lay.KVH, h = hid - b * p.lay.KVH;
    if (p.qring && sub == 0) record_stats<G>(p, b, h, g, Mg + log2f(Lg));
    uint16_t* out = p.out + ((size_t)b * p.lay.H + (size_t)h * G + g) * kHeadDim + ch0;
#pragma unroll
    for (int k = 0; k < C::MCH / 4; ++k) {
        const uint2 w = make_uint2(pack_bf16x2(acc[k].x * inv, acc[k].y * inv), pack_bf16x2(acc[k].z * inv, acc[k].w * inv));
        *reinterpret_cast<uint2*>(out + 4 * k) = w;
    }
}

// COMPACT: the launch also does the compaction of the heads in p.compacting (a separate
// instantiation, so that launches without it run code free of its branches and registers).
template <int G, bool COMPACT>
__global__ void __launch_bounds__(Cfg<G>::WARPS * 32, 1)
    attn_kernel(const __grid_constant__ AttnParams p, const __grid_constant__ CUtensorMap tk,
                const __grid_constant__ CUtensorMap tv)
{
    using C = Cfg<G>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    uint8_t* wstage = smem + (size_t)warp * C::SPW * C::STAGE_BYTES;
    // [stages (1024-byte aligned)][tile headers, 16 bytes each][mbarriers, 8 bytes each]
    int4* hdrs = reinterpret_cast<int4*>(smem + (size_t)C::NSTAGE * C::STAGE_BYTES) + warp * C::SPW;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + (size_t)C::NSTAGE * C::STAGE_BYTES + C::NSTAGE * 16) + warp * C::SPW;

    const int gw = blockIdx.x * C::WARPS + warp;
    if (gw >= p.nchunks) {  // no chunk for this warp
        pdl_wait();
        pdl_launch_dependents();
        return;
    }

    if (lane == 0) {
        for (int s = 0; s < C::SPW; ++s) mbar_init(&bars[s], 1);
        fence_mbar_init();
        prefetch_tensormap(&tk);
        prefetch_tensormap(&tv);
    }
    __syncwarp();
    // The cache, the region table and the inputs may come from the previous kernel.  With
    // p.early (the host has checked that the previous kernel writes none of this layer's
    // cache or tables) the first tiles' K and V are requested before waiting; the query
    // rows and the new token's row, which the caller may have just produced, come after.
    if (!p.early) pdl_wait();

    TileIter it;
    it.chunk = -1;
    it.f = it.end = 0;
    int issued = 0;
    // The caller's rows of a stage: the query rows (first tile of a piece), the new token's row.
    auto issue_inputs = [&](int s) {
        const int4 hd = hdrs[s];
        uint8_t* st = wstage + (size_t)s * C::STAGE_BYTES;
        const int b = hd.z / p.lay.KVH, h = hd.z - b * p.lay.KVH;
        if (hd.y & kNewTok) {
            const size_t src = ((size_t)b * p.lay.KVH + h) * kHeadDim;
            bulk_load(st + C::NT_OFF, p.k_new + src, (uint32_t)kRowBytes, &bars[s]);
            bulk_load(st + C::NT_OFF + kRowBytes, p.v_new + src, (uint32_t)kRowBytes, &bars[s]);
        }
        if (hd.y & kFirst)
            bulk_load(st + 2 * C::KV_BYTES, p.q + ((size_t)b * p.lay.H + (size_t)h * G) * kHeadDim,
                      (uint32_t)C::Q_BYTES, &bars[s]);
    };
    auto issue = [&](int t, bool inputs) -> bool {
        TileDesc d;
        if (!iter_next<COMPACT>(it, p, d, gw)) return false;
        const int s = t % C::SPW;
        if (lane == 0) {
            uint8_t* st = wstage + (size_t)s * C::STAGE_BYTES;
            hdrs[s] = make_int4(d.n, d.flags | (d.chunk << kFlagBits), d.hid, (int)d.row);
            const bool first = d.flags & kFirst;
            const bool newtok = d.flags & kNewTok;
            mbar_arrive_expect_tx(&bars[s], 2u * C::KV_BYTES + (first ? (uint32_t)C::Q_BYTES : 0u) +
                                                (newtok ? 2u * kRowBytes : 0u));
            tma_load_2d(st, &tk, 0, (int)d.row, &bars[s]);
            tma_load_2d(st + C::HALF_BYTES, &tk, kHalfCh, (int)d.row, &bars[s]);
            tma_load_2d(st + C::KV_BYTES, &tv, 0, (int)d.row, &bars[s]);
            tma_load_2d(st + C::KV_BYTES + C::HALF_BYTES, &tv, kHalfCh, (int)d.row, &bars[s]);
            if (inputs) issue_inputs(s);
        }
        return true;
    };
    bool more = true;
    for (int t = 0; t < C::SPW && more; ++t) {
        more = issue(t, !p.early);
        if (more) ++issued;
    }
    if (p.early) {
        pdl_wait();
        if (lane == 0)
            for (int t = 0; t < issued; ++t) issue_inputs(t);
    }
    pdl_launch_dependents();  // only now: the successor may assume our predecessor has completed

    const int gq = lane >> 2;  // this lane's query head (rows >= G are padding)
    const int tq = lane & 3;
    const int mi = lane >> 3, ri = lane & 7;  // ldmatrix: matrix and row this lane addresses

    uint32_t qa[8][2];  // fragments of Q (rows 0..7) for the 8 k-steps of 16 channels (A, or B of Q^T)
#if RA_ATTN_TRANSPOSED
    const int hA = 2 * tq, hB = 2 * tq + 1;  // the query heads of this lane's accumulator columns
    float O[8][4];      // O^T: m-tile mt = channels 16 mt..; {ch 16mt+gq: hA, hB; ch 16mt+gq+8: hA, hB}
    float mA = -INFINITY, mB = -INFINITY, lA = 0.f, lB = 0.f;  // running max and (lane-partial) sum per head
#pragma unroll
    for (int mt = 0; mt < 8; ++mt) O[mt][0] = O[mt][1] = O[mt][2] = O[mt][3] = 0.f;
#else
    float O[16][2];     // O[head gq][n-tile * 8 + 2 tq + {0, 1}]
    float m_run = -INFINITY, l_run = 0.f;
#pragma unroll
    for (int nt = 0; nt < 16; ++nt) O[nt][0] = O[nt][1] = 0.f;
#endif

    for (int t = 0; t < issued; ++t) {
        const int s = t % C::SPW;
        if (!mbar_wait_bounded(&bars[s], (uint32_t)((t / C::SPW) & 1), kWaitLimitNs)) {
            // Give up: flag it, let the copies already issued land (bounded), leave.
            if (lane == 0) atomicExch(p.lay.err, kDeviceErrTimeout);
            for (int u = t + 1; u < issued; ++u)
                (void)mbar_wait_bounded(&bars[u % C::SPW], (uint32_t)((u / C::SPW) & 1), kWaitLimitNs);
            return;
        }
        const int4 hd = hdrs[s];
        const int n = hd.x;
        uint8_t* Ks = wstage + (size_t)s * C::STAGE_BYTES;
        uint8_t* Vs = Ks + C::KV_BYTES;
        const uint32_t ks = smem_u32(Ks), vs = smem_u32(Vs);
        if (hd.y & kFirst) {  // first tile of a head piece: fresh query fragments
            const uint8_t* Qs = Vs + C::KV_BYTES;
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
                qa[kk][0] = gq < G ? *reinterpret_cast<const uint32_t*>(Qs + gq * kRowBytes + (16 * kk + 2 * tq) * 2) : 0u;
                qa[kk][1] = gq < G ? *reinterpret_cast<const uint32_t*>(Qs + gq * kRowBytes + (16 * kk + 8 + 2 * tq) * 2) : 0u;
            }
            if ((hd.y & kHead0) && p.qring) {  // the scored policy's window: this step's query rows of the head
                const int b = hd.z / p.lay.KVH, h = hd.z - b * p.lay.KVH, r = p.lay.r;
                int slot = (p.seq_g[b] + p.ring_off) % r;
                if (slot < 0) slot += r;
                uint4* dst = reinterpret_cast<uint4*>(
                    p.qring + ((((size_t)p.layer * p.lay.B + b) * p.lay.KVH + h) * r + slot) * (size_t)(G * kHeadDim));
                for (int i = lane; i < G * 16; i += 32) dst[i] = lds128(Qs + i * 16);
            }
        }
        // A tile of a head that compacts in this launch: which of its rows were evicted (a 64-bit
        // mask, from the ascending list of at most 64 evicted ordinals) and how many before it.
        uint32_t ev_lo = 0u, ev_hi = 0u;
        int ev_before = 0, j0 = 0;
        if (COMPACT && (hd.y & kCompact)) {
            const int32_t* plan = p.lay.plan + (size_t)hd.z * (kPlanHeader + p.lay.r);
            const int m = plan[3];
            j0 = (int)((long long)hd.w - p.lay.gen_row0 - (long long)plan[0] * p.lay.Cmax);
            const int e0 = lane < m ? plan[kPlanHeader + lane] - j0 : INT_MAX;
            const int e1 = lane + 32 < m ? plan[kPlanHeader + 32 + lane] - j0 : INT_MAX;
            ev_before = __popc(__ballot_sync(0xffffffffu, e0 < 0)) + __popc(__ballot_sync(0xffffffffu, e1 < 0));
            const uint32_t lo = ((e0 >= 0 && e0 < 32) ? 1u << e0 : 0u) | ((e1 >= 0 && e1 < 32) ? 1u << e1 : 0u);
            const uint32_t hi = ((e0 >= 32 && e0 < 64) ? 1u << (e0 - 32) : 0u) | ((e1 >= 32 && e1 < 64) ? 1u << (e1 - 32) : 0u);
            ev_lo = __reduce_or_sync(0xffffffffu, lo);
            ev_hi = __reduce_or_sync(0xffffffffu, hi);
        }
        if (hd.y & kNewTok) {  // fused append: put the new token in row n-1 of the tile and into the cache
            const int b = hd.z / p.lay.KVH;
            const int c = lane & 15;
            const uint4 v = lds128(Ks + C::NT_OFF + (lane >> 4) * kRowBytes + c * 16);
            *reinterpret_cast<uint4*>((lane < 16 ? Ks : Vs) + swz<G>(n - 1, c)) = v;
            if (!(COMPACT && (hd.y & kCompact))) {  // (a compacting head writes it with its survivors)
                const long long row = (long long)hd.w + n - 1;
                reinterpret_cast<uint4*>((lane < 16 ? p.lay.kpool : p.lay.vpool) + row * kHeadDim)[c] = v;
                if (lane == 0) p.lay.pos[row - p.lay.gen_row0] = p.seq_lp[b] + p.seq_g[b];
            }
            __syncwarp();
        }
        if (n < C::TILE) {  // rows past the valid ones hold stale data: zero V there so 0 * V stays 0
            const int nb = (n + 15) & ~15;  // only rows inside the last used 16-row batch matter
            for (int idx = lane; idx < (nb - n) * 16; idx += 32) {
                const int j = n + (idx >> 4), c = idx & 15;
                *reinterpret_cast<uint4*>(Vs + swz<G>(j, c)) = make_uint4(0u, 0u, 0u, 0u);
            }
            __syncwarp();
        }

#if RA_ATTN_TRANSPOSED
        // per 16-row batch: S^T = K Q^T (two accumulator chains), online softmax, O^T += V^T P^T
        const float sl = p.qk_scale_log2;
        for (int bs = 0; bs < n; bs += 16) {
            float x[4] = {0.f, 0.f, 0.f, 0.f}, y[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
            for (int kk = 0; kk < 8; kk += 2) {
                uint32_t a0[4], a1[4];
                ldsm_x4(a0, ks + swz<G>(bs + (mi & 1) * 8 + ri, 2 * kk + (mi >> 1)));
                ldsm_x4(a1, ks + swz<G>(bs + (mi & 1) * 8 + ri, 2 * kk + 2 + (mi >> 1)));
                mma16816(x, a0, qa[kk][0], qa[kk][1]);
                mma16816(y, a1, qa[kk + 1][0], qa[kk + 1][1]);
            }
            const int r0 = bs + gq, r1 = r0 + 8;  // this lane's rows; heads hA, hB
            bool v0 = r0 < n, v1 = r1 < n;
            if (COMPACT && (hd.y & kCompact)) {  // evicted rows get no weight
                v0 = v0 && !(((r0 < 32 ? ev_lo >> r0 : ev_hi >> (r0 - 32)) & 1u));
                v1 = v1 && !(((r1 < 32 ? ev_lo >> r1 : ev_hi >> (r1 - 32)) & 1u));
            }
            float sv[4] = {v0 ? (x[0] + y[0]) * sl : -INFINITY, v0 ? (x[1] + y[1]) * sl : -INFINITY,
                           v1 ? (x[2] + y[2]) * sl : -INFINITY, v1 ? (x[3] + y[3]) * sl : -INFINITY};
            float xA = fmaxf(sv[0], sv[2]), xB = fmaxf(sv[1], sv[3]);
            if (__any_sync(0xffffffffu, xA > mA + kTau || xB > mB + kTau)) {
#pragma unroll
                for (int o = 4; o < 32; o <<= 1) {  // over the 8 lanes that share a head pair
                    xA = fmaxf(xA, __shfl_xor_sync(0xffffffffu, xA, o));
                    xB = fmaxf(xB, __shfl_xor_sync(0xffffffffu, xB, o));
                }
                const float nA = xA > mA + kTau ? xA : mA, nB = xB > mB + kTau ? xB : mB;
                const float aA = (nA == mA) ? 1.f : exp2f(mA - nA), aB = (nB == mB) ? 1.f : exp2f(mB - nB);
                mA = nA;
                mB = nB;
                lA *= aA;
                lB *= aB;
#pragma unroll
                for (int mt = 0; mt < 8; ++mt) {
                    O[mt][0] *= aA;
                    O[mt][2] *= aA;
                    O[mt][1] *= aB;
                    O[mt][3] *= aB;
                }
            }
            float pr[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const float m = (e & 1) ? mB : mA;
                pr[e] = (COMPACT && sv[e] == -INFINITY) ? 0.f : exp2f(sv[e] - m);
            }
            lA += pr[0] + pr[2];
            lB += pr[1] + pr[3];
            const uint32_t b0 = movtrans(pack_bf16x2(pr[0], pr[1])), b1 = movtrans(pack_bf16x2(pr[2], pr[3]));
#pragma unroll
            for (int mt = 0; mt < 8; ++mt) {
                uint32_t v4[4];
                ldsm_x4_t(v4, vs + swz<G>(bs + (mi >> 1) * 8 + ri, 2 * mt + (mi & 1)));
                mma16816(O[mt], v4, b0, b1);
            }
        }

        if (hd.y & kLast) {  // last tile of the piece
            float la = lA, lb = lB;
#pragma unroll
            for (int o = 4; o < 32; o <<= 1) {
                la += __shfl_xor_sync(0xffffffffu, la, o);
                lb += __shfl_xor_sync(0xffffffffu, lb, o);
            }
            const int hid = hd.z;
            const int b = hid / p.lay.KVH, h = hid - b * p.lay.KVH;
            const int nth = seq_head_tiles(p, b);
            const long long A = p.seq_base[b] + (long long)h * nth;
            const int w0 = (int)(A / p.W), w1 = (int)((A + nth - 1) / p.W);
            if (w0 == w1) {  // the whole head was this warp's: normalise and write the output
                if (p.qring && gq == 0) {
                    if (hA < G) record_stats<G>(p, b, h, hA, mA + log2f(la));
                    if (hB < G) record_stats<G>(p, b, h, hB, mB + log2f(lb));
                }
                const float iA = 1.f / la, iB = 1.f / lb;
                __nv_bfloat16* ob = reinterpret_cast<__nv_bfloat16*>(p.out + ((size_t)b * p.lay.H + (size_t)h * G) * kHeadDim);
#pragma unroll
                for (int mt = 0; mt < 8; ++mt) {
                    const int ch = 16 * mt + gq;
                    if (hA < G) {
                        ob[hA * kHeadDim + ch] = __float2bfloat16_rn(O[mt][0] * iA);
                        ob[hA * kHeadDim + ch + 8] = __float2bfloat16_rn(O[mt][2] * iA);
                    }
                    if (hB < G) {
                        ob[hB * kHeadDim + ch] = __float2bfloat16_rn(O[mt][1] * iB);
                        ob[hB * kHeadDim + ch + 8] = __float2bfloat16_rn(O[mt][3] * iB);
                    }
                }
            } else {
                float* rec = p.partial + (size_t)((hd.y >> kFlagBits) + hid) * partial_stride(G);
#pragma unroll
                for (int mt = 0; mt < 8; ++mt) {
                    const int ch = 16 * mt + gq;
                    if (hA < G) {
                        rec[hA * kHeadDim + ch] = O[mt][0];
                        rec[hA * kHeadDim + ch + 8] = O[mt][2];
                    }
                    if (hB < G) {
                        rec[hB * kHeadDim + ch] = O[mt][1];
                        rec[hB * kHeadDim + ch + 8] = O[mt][3];
                    }
                }
                if (gq == 0) {
                    if (hA < G) {
                        rec[G * kHeadDim + hA] = mA;
                        rec[G * kHeadDim + G + hA] = la;
                    }
                    if (hB < G) {
                        rec[G * kHeadDim + hB] = mB;
                        rec[G * kHeadDim + G + hB] = lb;
                    }
                }
                __threadfence();
                __syncwarp();
                int old = 0;
                if (lane == 0) old = atomicAdd(p.arrive + hid, 1);
                old = __shfl_sync(0xffffffffu, old, 0);
                if (old == w1 - w0) {  // every other piece of this head is already written
                    __threadfence();
                    merge_head<G>(p, hid, w0, w1 - w0 + 1, lane);
                    if (lane == 0) p.arrive[hid] = 0;  // ready for the next launch
                }
            }
            mA = mB = -INFINITY;
            lA = lB = 0.f;
#pragma unroll
            for (int mt = 0; mt < 8; ++mt) O[mt][0] = O[mt][1] = O[mt][2] = O[mt][3] = 0.f;
        }
#else
        for (int bs = 0; bs < n; bs += 16) {
            // S = Q K^T for rows bs..bs+15: n-tile 0 = rows bs..bs+7, n-tile 1 = rows bs+8..bs+15
            float s0a = 0.f, s0b = 0.f, s1a = 0.f, s1b = 0.f;
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
                uint32_t b[4];
                ldsm_x4(b, ks + swz<G>(bs + (mi >> 1) * 8 + ri, 2 * kk + (mi & 1)));
                mma_rows8(s0a, s0b, qa[kk][0], qa[kk][1], b[0], b[1]);
                mma_rows8(s1a, s1b, qa[kk][0], qa[kk][1], b[2], b[3]);
            }
            // this lane: head gq, rows bs + 2tq + {0,1} and bs + 8 + 2tq + {0,1}
            const int r0 = bs + 2 * tq;
            const float sl = p.qk_scale_log2;
            float sc[4] = {r0 < n ? s0a * sl : -INFINITY, r0 + 1 < n ? s0b * sl : -INFINITY,
                           r0 + 8 < n ? s1a * sl : -INFINITY, r0 + 9 < n ? s1b * sl : -INFINITY};
            if (COMPACT && (hd.y & kCompact)) {  // evicted rows get no weight
                const int rr[4] = {r0, r0 + 1, r0 + 8, r0 + 9};
#pragma unroll
                for (int e = 0; e < 4; ++e)
                    if (((rr[e] < 32 ? ev_lo >> rr[e] : ev_hi >> (rr[e] - 32)) & 1u)) sc[e] = -INFINITY;
            }
            float bm = fmaxf(fmaxf(sc[0], sc[1]), fmaxf(sc[2], sc[3]));
            bm = fmaxf(bm, __shfl_xor_sync(0xffffffffu, bm, 1));
            bm = fmaxf(bm, __shfl_xor_sync(0xffffffffu, bm, 2));
            const bool need = bm > m_run + kTau;
            if (__any_sync(0xffffffffu, need)) {
                const float m_new = need ? bm : m_run;
                const float a = (m_new == m_run) ? 1.f : exp2f(m_run - m_new);
                l_run *= a;
                m_run = m_new;
#pragma unroll
                for (int nt = 0; nt < 16; ++nt) {
                    O[nt][0] *= a;
                    O[nt][1] *= a;
                }
            }
            float pr[4];
#pragma unroll
            // masked rows: exp2(-inf) = 0; a compacting head can have a whole batch evicted, with
            // m_run still -inf (the difference would be NaN), so there a masked row weighs 0 outright
            for (int e = 0; e < 4; ++e) pr[e] = (COMPACT && sc[e] == -INFINITY) ? 0.f : exp2f(sc[e] - m_run);
            l_run += (pr[0] + pr[1]) + (pr[2] + pr[3]);
            const uint32_t pa0 = pack_bf16x2(pr[0], pr[1]), pa2 = pack_bf16x2(pr[2], pr[3]);
            // O += P V: 16 n-tiles of 8 channels, k = the 16 rows
#pragma unroll
            for (int np = 0; np < 8; ++np) {
                uint32_t b[4];
                ldsm_x4_t(b, vs + swz<G>(bs + (mi & 1) * 8 + ri, 2 * np + (mi >> 1)));
                mma_rows8(O[2 * np][0], O[2 * np][1], pa0, pa2, b[0], b[1]);
                mma_rows8(O[2 * np + 1][0], O[2 * np + 1][1], pa0, pa2, b[2], b[3]);
            }
        }

        if (hd.y & kLast) {  // last tile of the piece
            float l = l_run;
            l += __shfl_xor_sync(0xffffffffu, l, 1);
            l += __shfl_xor_sync(0xffffffffu, l, 2);
            const int hid = hd.z;
            const int b = hid / p.lay.KVH, h = hid - b * p.lay.KVH;
            const int nth = seq_head_tiles(p, b);
            const long long A = p.seq_base[b] + (long long)h * nth;
            const int w0 = (int)(A / p.W), w1 = (int)((A + nth - 1) / p.W);
            if (w0 == w1) {  // the whole head was this warp's: normalise and write the output
                if (gq < G) {
                    if (p.qring && tq == 0) record_stats<G>(p, b, h, gq, m_run + log2f(l));
                    const float inv = 1.f / l;
                    uint32_t* out = reinterpret_cast<uint32_t*>(p.out + ((size_t)b * p.lay.H + (size_t)h * G + gq) * kHeadDim);
#pragma unroll
                    for (int nt = 0; nt < 16; ++nt) out[nt * 4 + tq] = pack_bf16x2(O[nt][0] * inv, O[nt][1] * inv);
                }
            } else {
                float* rec = p.partial + (size_t)((hd.y >> kFlagBits) + hid) * partial_stride(G);
                if (gq < G) {
#pragma unroll
                    for (int nt = 0; nt < 16; ++nt)
                        *reinterpret_cast<float2*>(rec + gq * kHeadDim + nt * 8 + 2 * tq) = make_float2(O[nt][0], O[nt][1]);
                    if (tq == 0) {
                        rec[G * kHeadDim + gq] = m_run;
                        rec[G * kHeadDim + G + gq] = l;
                    }
                }
                __threadfence();
                __syncwarp();
                int old = 0;
                if (lane == 0) old = atomicAdd(p.arrive + hid, 1);
                old = __shfl_sync(0xffffffffu, old, 0);
                if (old == w1 - w0) {  // every other piece of this head is already written
                    __threadfence();
                    merge_head<G>(p, hid, w0, w1 - w0 + 1, lane);
                    if (lane == 0) p.arrive[hid] = 0;  // ready for the next launch
                }
            }
            m_run = -INFINITY;
            l_run = 0.f;
#pragma unroll
            for (int nt = 0; nt < 16; ++nt) O[nt][0] = O[nt][1] = 0.f;
        }
#endif

        if (COMPACT && (hd.y & kCompact)) {
            // Compaction fused into the pass: every surviving row of the tile (the new token
            // included) goes from the staged tile to its slot in the new region, ordinal
            // j - (evicted before j); positions follow.  One row per step, 16-byte lanes
            // (0-15: K, 16-31: V).
            const int32_t* plan = p.lay.plan + (size_t)hd.z * (kPlanHeader + p.lay.r);
            const long long drow0 = p.lay.gen_row0 + (long long)plan[1] * p.lay.Cmax;
            const int32_t* spos = p.lay.pos + (size_t)plan[0] * p.lay.Cmax;
            int32_t* dpos = p.lay.pos + (size_t)plan[1] * p.lay.Cmax;
            const int c = lane & 15;
            uint16_t* pool = lane < 16 ? p.lay.kpool : p.lay.vpool;
            const uint8_t* tile = lane < 16 ? Ks : Vs;
            auto evicted = [&](int jj) { return ((jj < 32 ? ev_lo >> jj : ev_hi >> (jj - 32)) & 1u) != 0u; };
            auto dest = [&](int jj) {
                const int below = jj < 32 ? __popc(ev_lo & ((1u << jj) - 1u))
                                          : __popc(ev_lo) + __popc(ev_hi & ((1u << (jj - 32)) - 1u));
                return j0 + jj - ev_before - below;
            };
            for (int jj = 0; jj < n; ++jj) {
                if (evicted(jj)) continue;
                reinterpret_cast<uint4*>(pool + (drow0 + dest(jj)) * kHeadDim)[c] = lds128(tile + swz<G>(jj, c));
            }
            for (int jj = lane; jj < n; jj += 32) {
                if (evicted(jj)) continue;
                const int b = hd.z / p.lay.KVH;
                const bool newtok = (hd.y & kNewTok) && jj == n - 1;
                dpos[dest(jj)] = newtok ? p.seq_lp[b] + p.seq_g[b] : __ldg(spos + j0 + jj);
            }
        }

        __syncwarp();
        if (more) {
            if (lane == 0) fence_proxy_async_smem();
            more = issue(t + C::SPW, true);
            if (more) ++issued;
        }
    }
}

// Active sequences whose heads hold no slot at all (empty prompt, nothing generated)
// attend over nothing: their output rows are zero.
__global__ void __launch_bounds__(256) zero_empty_kernel(const __grid_constant__ AttnParams p)
{
    pdl_wait();
    pdl_launch_dependents();
    const int b = blockIdx.x;
    if (!((p.active[b >> 5] >> (b & 31)) & 1u) || p.seq_base[b + 1] != p.seq_base[b]) return;
    uint16_t* out = p.out + (size_t)b * p.lay.H * kHeadDim;
    for (int i = threadIdx.x; i < p.lay.H * kHeadDim / 8; i += blockDim.x)
        reinterpret_cast<uint4*>(out)[i] = make_uint4(0u, 0u, 0u, 0u);
}

template <int G>
cudaError_t launch_attn_g(const AttnParams& p, const CUtensorMap* tk, const CUtensorMap* tv, int ctas, cudaStream_t s)
{
    using C = Cfg<G>;
    bool compact = false;
    for (int i = 0; i < RA_MAX_BATCH / 32; ++i) compact |= p.compacting[i] != 0u;
    if (compact) return launch_pdl(attn_kernel<G, true>, dim3(ctas), dim3(C::WARPS * 32), C::SMEM, s, p, *tk, *tv);
    return launch_pdl(attn_kernel<G, false>, dim3(ctas), dim3(C::WARPS * 32), C::SMEM, s, p, *tk, *tv);
}

template <int G>
cudaError_t prepare_g()
{
    cudaError_t e = cudaFuncSetAttribute(attn_kernel<G, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)Cfg<G>::SMEM);
    if (e != cudaSuccess) return e;
    return cudaFuncSetAttribute(attn_kernel<G, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg<G>::SMEM);
}

}  // namespace

namespace RA_ATTN_NS {

int attn_warps_per_cta(int G)
{
    switch (G) {
        case 1: return Cfg<1>::WARPS;
        case 2: return Cfg<2>::WARPS;
        case 3: return Cfg<3>::WARPS;
        case 4: return Cfg<4>::WARPS;
        case 5: return Cfg<5>::WARPS;
        case 6: return Cfg<6>::WARPS;
        case 7: return Cfg<7>::WARPS;
        case 8: return Cfg<8>::WARPS;
    }
    return 0;
}

int attn_tile_rows(int G)
{
    switch (G) {
        case 1: return Cfg<1>::TILE;
        case 2: return Cfg<2>::TILE;
        case 3: return Cfg<3>::TILE;
        case 4: return Cfg<4>::TILE;
        case 5: return Cfg<5>::TILE;
        case 6: return Cfg<6>::TILE;
        case 7: return Cfg<7>::TILE;
        case 8: return Cfg<8>::TILE;
    }
    return 0;
}

cudaError_t attn_prepare(int G)
{
    switch (G) {
        case 1: return prepare_g<1>();
        case 2: return prepare_g<2>();
        case 3: return prepare_g<3>();
        case 4: return prepare_g<4>();
        case 5: return prepare_g<5>();
        case 6: return prepare_g<6>();
        case 7: return prepare_g<7>();
        case 8: return prepare_g<8>();
    }
    return cudaErrorInvalidValue;
}

cudaError_t launch_attention(const AttnParams& p, const CUtensorMap* tk, const CUtensorMap* tv, int ctas,
                             cudaStream_t s)
{
    bool any_empty = false;
    for (int b = 0; b < p.lay.B; ++b)
        if (((p.active[b >> 5] >> (b & 31)) & 1u) && p.seq_base[b + 1] == p.seq_base[b]) any_empty = true;
    if (any_empty) {
        cudaError_t e = launch_pdl(zero_empty_kernel, dim3(p.lay.B), dim3(256), 0, s, p);
        if (e != cudaSuccess) return e;
    }
    if (p.total == 0) return cudaSuccess;
    switch (p.lay.G) {
        case 1: return launch_attn_g<1>(p, tk, tv, ctas, s);
        case 2: return launch_attn_g<2>(p, tk, tv, ctas, s);
        case 3: return launch_attn_g<3>(p, tk, tv, ctas, s);
        case 4: return launch_attn_g<4>(p, tk, tv, ctas, s);
        case 5: return launch_attn_g<5>(p, tk, tv, ctas, s);
        case 6: return launch_attn_g<6>(p, tk, tv, ctas, s);
        case 7: return launch_attn_g<7>(p, tk, tv, ctas, s);
        case 8: return launch_attn_g<8>(p, tk, tv, ctas, s);
    }
    return cudaErrorInvalidValue;
}

}  // namespace RA_ATTN_NS
}  // namespace ra
