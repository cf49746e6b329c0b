// ra_attn.cu -- GQA split-K flash-decode attention over the per-head caches (sm_103a).
//
// Computes, for every active sequence b and query head qh (KV head h = qh / G),
//     o = sum_i softmax_i(scale * q . k_i) v_i
// over the prompt rows and the cached generated rows of (b, h) -- section 2
// ("Notation"), with the grouped-query sharing of Appendix F.  In the fused
// form the step's new token (Appendix F: appended post-RoPE every step) is one
// more slot: it is read from the caller's k_new/v_new rows, attended, and
// written into the cache by the warp that consumes it.
//
// Work split ("stream-K" by warp): the slots of all heads of the layer are laid
// end to end (sequence-major, then KV head; within a head the prompt rows, the
// cached generated rows, then the new token) and every warp of the grid takes
// one contiguous range of W slots.  A warp runs its own pipeline: lane 0
// streams tiles of TILE rows of K and of V (and, at the first tile of each head
// piece, the G query rows) into a ring of SPW shared-memory stages with 2-D TMA
// loads completing on per-stage mbarriers; all 32 lanes consume.  A head that
// fits in one warp's range is finished in registers.  Otherwise each (head,
// warp) piece writes an fp32 partial (unnormalised o, running max m, sum l) to
// slot `warp + head` -- unique because warps and heads both advance
// monotonically through the slot order -- and the last warp to finish a piece
// of that head (an arrival counter per head) merges all of them.
//
// Per-warp compute layout: LPS lanes share one cache row (each lane owns
// 16 bytes -- 8 channels -- of every LPS-th 16-byte chunk, so a row read is
// bank-conflict free); the warp works on 32/LPS rows at once.  The G query rows
// live in fp32 registers; each K row is read once from shared memory and used
// by all G heads (G flop per byte), with packed two-wide fp32 FMAs.  Partial
// dot products are summed across the LPS lanes with a butterfly reduce-scatter
// (each exchange halves the vector), which leaves exactly one (row, head) score
// per lane.  The softmax is online in base 2 with the scale folded into one
// multiply; the running max is only raised when a batch exceeds it by more than
// 2^8 (results are unchanged up to rounding, as softmax is shift invariant), so
// rescaling the accumulators is rare.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "ra_internal.h"
#include "ra_ptx.cuh"

namespace ra {
namespace {

constexpr float kTau = 8.0f;                       // lazy-rescale threshold (log2 units)
constexpr uint64_t kWaitLimitNs = 2000000000ull;   // bounded mbarrier waits: 2 s
constexpr int kSmemBudget = 220 * 1024;

template <int G>
struct Cfg {
    static constexpr int GP = G <= 1 ? 1 : (G <= 2 ? 2 : (G <= 4 ? 4 : 8));  // G padded to a power of two
    static constexpr int LPS = G <= 4 ? 8 : 16;                              // lanes per cache row
    static constexpr int SG = 32 / LPS;                                      // rows per warp step
    static constexpr int NB = LPS / GP;                                      // steps per reduce batch
    static constexpr int BATCH = SG * NB;                                    // rows per batch
    static constexpr int NCH = 16 / LPS;                                     // 16-byte chunks per lane per row
    static constexpr int CPL = NCH * 8;                                      // channels per lane
    static constexpr int CP2 = CPL / 2;                                      // channel pairs per lane
    static constexpr int TILE = BATCH > 16 ? BATCH : 16;                     // rows per stage
    static constexpr int KV_BYTES = TILE * kRowBytes;
    static constexpr int Q_BYTES = G * kRowBytes;
    static constexpr int STAGE_BYTES = ((2 * KV_BYTES + Q_BYTES) + 127) / 128 * 128;
    static constexpr int W3 = kSmemBudget / (3 * STAGE_BYTES);
    static constexpr int SPW = W3 >= 6 ? 3 : 2;
    static constexpr int WARPS_RAW = SPW == 3 ? W3 : kSmemBudget / (2 * STAGE_BYTES);
    static constexpr int WARPS = WARPS_RAW > 8 ? 8 : WARPS_RAW;
    static constexpr int NSTAGE = WARPS * SPW;
    static constexpr size_t SMEM = 128 + (size_t)NSTAGE * STAGE_BYTES + (size_t)NSTAGE * (16 + 8);
    // merge layout: LG lanes per query head, MCH channels per lane
    static constexpr int LG = 32 / GP;
    static constexpr int MCH = kHeadDim / LG;
    static_assert(LPS == NB * GP, "one reduced score per lane");
    static_assert(TILE % BATCH == 0, "tile holds whole batches");
    static_assert(WARPS >= 4, "shared-memory budget too small");
    static_assert(STAGE_BYTES % 128 == 0, "TMA destinations stay 128-byte aligned");
    static_assert(SMEM <= 232448, "fits the 227 KB opt-in shared memory of sm_100+");
};

constexpr int kFirst = 1, kLast = 2, kNewTok = 4;

// Producer-side walk over the warp's slot range.
struct TileIter {
    int f, end;           // flattened cursor and end of the warp's range
    int b, h, pos;        // current sequence, KV head, slot within the head
    int hl, lp, cg;       // head length, prompt length, cached generated rows (excl. a fused new token)
    long long prow, grow; // first prompt row / first generated row of the head
    bool piece_start;
};

struct TileDesc {
    long long row;  // first cache row (TMA) or the cache row the new token goes to
    int n, hid, flags;
};

__device__ __forceinline__ int seq_head_len(const AttnParams& p, int b)
{
    return (p.seq_base[b + 1] - p.seq_base[b]) / p.lay.KVH;
}

__device__ __forceinline__ void enter_head(TileIter& it, const AttnParams& p)
{
    const DevLayout& L = p.lay;
    const int lp = L.seq_lp[it.b];
    it.lp = lp < it.hl ? lp : it.hl;
    it.cg = it.hl - it.lp - (p.k_new ? 1 : 0);
    it.prow = (long long)p.layer * L.prompt_rows_per_layer + L.seq_poff[it.b] + (long long)it.h * lp;
    const int reg = L.region[((size_t)p.layer * L.B + it.b) * L.KVH + it.h];
    it.grow = L.gen_row0 + (long long)reg * L.Cmax;
    it.piece_start = true;
}

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
    it.hl = seq_head_len(p, b);
    const int off = R0 - p.seq_base[b];
    it.h = off / it.hl;
    it.pos = off - it.h * it.hl;
    enter_head(it, p);
}

__device__ bool iter_next(TileIter& it, const AttnParams& p, int tile, TileDesc& d)
{
    if (it.f >= it.end) return false;
    const int gen_end = it.lp + it.cg;  // slots [gen_end, hl) hold the fused new token
    const int seg_end = it.pos < it.lp ? it.lp : (it.pos < gen_end ? gen_end : it.hl);
    const int rem = it.end - it.f;
    const int piece_end = (it.hl - it.pos < rem) ? it.hl : it.pos + rem;
    int n = (seg_end < piece_end ? seg_end : piece_end) - it.pos;
    if (n > tile) n = tile;
    d.flags = (it.piece_start ? kFirst : 0) | (it.pos + n == piece_end ? kLast : 0);
    if (it.pos < it.lp) {
        d.row = it.prow + it.pos;
    } else {
        d.row = it.grow + (it.pos - it.lp);
        if (it.pos >= gen_end) d.flags |= kNewTok;  // row = its destination slot in the cache
    }
    d.n = n;
    d.hid = it.b * p.lay.KVH + it.h;
    it.piece_start = false;
    it.pos += n;
    it.f += n;
    if (it.pos == it.hl && it.f < it.end) {  // next head (skipping finished sequences)
        if (++it.h == p.lay.KVH) {
            it.h = 0;
            do {
                ++it.b;
            } while (seq_head_len(p, it.b) == 0);
            it.hl = seq_head_len(p, it.b);
        }
        it.pos = 0;
        enter_head(it, p);
    }
    return true;
}

__device__ __forceinline__ void unpack8(const uint4 u, float2* f)
{
    f[0] = make_float2(bf16lo(u.x), bf16hi(u.x));
    f[1] = make_float2(bf16lo(u.y), bf16hi(u.y));
    f[2] = make_float2(bf16lo(u.z), bf16hi(u.z));
    f[3] = make_float2(bf16lo(u.w), bf16hi(u.w));
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi)
{
    return (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(lo)) |
           ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(hi)) << 16);
}

// Merge every piece of head `hid` (pieces are partial records w0 + p + hid, p < P)
// into the bf16 output rows of its G query heads.  One warp; lanes split as
// (query head, channel block).  Partials come from other SMs: read through L2.
template <int G>
__device__ void merge_head(const AttnParams& p, int hid, int w0, int P, int lane)
{
    using C = Cfg<G>;
    const int g = lane / C::LG;
    const int c0 = (lane % C::LG) * C::MCH;
    if (g >= G) return;
    const size_t rs = (size_t)partial_stride(G);
    const float* base = p.partial + (size_t)(w0 + hid) * rs;
    float M = -INFINITY;
#pragma unroll 4
    for (int q = 0; q < P; ++q) M = fmaxf(M, __ldcg(base + q * rs + G * kHeadDim + g));
    float Lsum = 0.f;
    float4 acc[C::MCH / 4];
#pragma unroll
    for (int j = 0; j < C::MCH / 4; ++j) acc[j] = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 2
    for (int q = 0; q < P; ++q) {
        const float* rec = base + q * rs;
        const float a = exp2f(__ldcg(rec + G * kHeadDim + g) - M);
        Lsum = fmaf(a, __ldcg(rec + G * kHeadDim + G + g), Lsum);
        const float4* o = reinterpret_cast<const float4*>(rec + g * kHeadDim + c0);
#pragma unroll
        for (int j = 0; j < C::MCH / 4; ++j) {
            const float4 v = __ldcg(o + j);
            acc[j].x = fmaf(a, v.x, acc[j].x);
            acc[j].y = fmaf(a, v.y, acc[j].y);
            acc[j].z = fmaf(a, v.z, acc[j].z);
            acc[j].w = fmaf(a, v.w, acc[j].w);
        }
    }
    const float inv = 1.f / Lsum;
    const int b = hid / p.lay.KVH, h = hid - b * p.lay.KVH;
    uint16_t* out = p.out + ((size_t)b * p.lay.H + (size_t)h * G + g) * kHeadDim + c0;
#pragma unroll
    for (int j = 0; j < C::MCH / 4; ++j) {
        const uint2 w = make_uint2(pack_bf16x2(acc[j].x * inv, acc[j].y * inv), pack_bf16x2(acc[j].z * inv, acc[j].w * inv));
        *reinterpret_cast<uint2*>(out + 4 * j) = w;
    }
}

template <int G>
__global__ void __launch_bounds__(Cfg<G>::WARPS * 32, 1)
    attn_kernel(const __grid_constant__ AttnParams p, const __grid_constant__ CUtensorMap tk,
                const __grid_constant__ CUtensorMap tv)
{
    using C = Cfg<G>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 127) & ~uintptr_t(127));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    uint8_t* wstage = smem + (size_t)warp * C::SPW * C::STAGE_BYTES;
    // [stages (128-byte aligned)][tile headers, 16 bytes each][mbarriers, 8 bytes each]
    int4* hdrs = reinterpret_cast<int4*>(smem + (size_t)C::NSTAGE * C::STAGE_BYTES) + warp * C::SPW;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + (size_t)C::NSTAGE * C::STAGE_BYTES + C::NSTAGE * 16) + warp * C::SPW;

    pdl_launch_dependents();
    const int gw = blockIdx.x * C::WARPS + warp;
    const long long R0l = (long long)gw * p.W;
    if (R0l >= p.total) return;
    const int R0 = (int)R0l;
    const int R1 = (int)min((long long)p.total, R0l + p.W);

    if (lane == 0) {
        for (int s = 0; s < C::SPW; ++s) mbar_init(&bars[s], 1);
        fence_mbar_init();
        prefetch_tensormap(&tk);
        prefetch_tensormap(&tv);
    }
    __syncwarp();
    pdl_wait();  // the cache, the region table and the inputs may come from the previous kernel

    TileIter it;
    iter_init(it, p, R0, R1);
    int issued = 0;
    auto issue = [&](int t) -> bool {
        TileDesc d;
        if (!iter_next(it, p, C::TILE, d)) return false;
        const int s = t % C::SPW;
        if (lane == 0) {
            uint8_t* st = wstage + (size_t)s * C::STAGE_BYTES;
            hdrs[s] = make_int4(d.n, d.flags, d.hid, (int)d.row);
            const bool first = d.flags & kFirst;
            const uint32_t kv = (d.flags & kNewTok) ? 2u * kRowBytes : 2u * C::KV_BYTES;
            mbar_arrive_expect_tx(&bars[s], kv + (first ? (uint32_t)C::Q_BYTES : 0u));
            const int b = d.hid / p.lay.KVH, h = d.hid - b * p.lay.KVH;
            if (d.flags & kNewTok) {  // the step's new token comes from the caller's rows
                const size_t src = ((size_t)b * p.lay.KVH + h) * kHeadDim;
                bulk_load(st, p.k_new + src, (uint32_t)kRowBytes, &bars[s]);
                bulk_load(st + C::KV_BYTES, p.v_new + src, (uint32_t)kRowBytes, &bars[s]);
            } else {
                tma_load_2d(st, &tk, 0, (int)d.row, &bars[s]);
                tma_load_2d(st + C::KV_BYTES, &tv, 0, (int)d.row, &bars[s]);
            }
            if (first)
                bulk_load(st + 2 * C::KV_BYTES, p.q + ((size_t)b * p.lay.H + (size_t)h * G) * kHeadDim,
                          (uint32_t)C::Q_BYTES, &bars[s]);
        }
        return true;
    };
    bool more = true;
    for (int t = 0; t < C::SPW && more; ++t) {
        more = issue(t);
        if (more) ++issued;
    }

    const int k = lane % C::LPS;
    const int grp = lane / C::LPS;
    const int g_own = lane % C::GP;
    const int i_own = k / C::GP;

    float2 qf[G][C::CP2];
    float2 O[G][C::CP2];
    float m_own = -INFINITY, l_own = 0.f;
#pragma unroll
    for (int g = 0; g < G; ++g)
#pragma unroll
        for (int c = 0; c < C::CP2; ++c) O[g][c] = make_float2(0.f, 0.f);

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
        const uint8_t* Ks = wstage + (size_t)s * C::STAGE_BYTES;
        const uint8_t* Vs = Ks + C::KV_BYTES;
        if (hd.y & kFirst) {  // first tile of a head piece: fresh query rows
            const uint8_t* Qs = Vs + C::KV_BYTES;
#pragma unroll
            for (int g = 0; g < G; ++g)
#pragma unroll
                for (int cc = 0; cc < C::NCH; ++cc) unpack8(lds128(Qs + g * kRowBytes + (k + cc * C::LPS) * 16), &qf[g][cc * 4]);
        }

        for (int bs = 0; bs < n; bs += C::BATCH) {
            float vals[C::LPS];
#pragma unroll
            for (int i = 0; i < C::NB; ++i) {
                const int slot = bs + i * C::SG + grp;
                const int row = slot < n ? slot : n - 1;
                float2 acc[G];
#pragma unroll
                for (int g = 0; g < G; ++g) acc[g] = make_float2(0.f, 0.f);
#pragma unroll
                for (int cc = 0; cc < C::NCH; ++cc) {
                    float2 kf[4];
                    unpack8(lds128(Ks + row * kRowBytes + (k + cc * C::LPS) * 16), kf);
#pragma unroll
                    for (int e = 0; e < 4; ++e)
#pragma unroll
                        for (int g = 0; g < G; ++g) acc[g] = __ffma2_rn(qf[g][cc * 4 + e], kf[e], acc[g]);
                }
#pragma unroll
                for (int g = 0; g < C::GP; ++g) vals[i * C::GP + g] = g < G ? acc[g < G ? g : 0].x + acc[g < G ? g : 0].y : 0.f;
            }
            // Butterfly reduce-scatter over the LPS lanes of a row group:
            // afterwards lane k holds the full dot product of value k = (i_own, g_own).
#pragma unroll
            for (int msk = C::LPS / 2; msk >= 1; msk >>= 1) {
                const bool up = (lane & msk) != 0;
#pragma unroll
                for (int t2 = 0; t2 < msk; ++t2) {
                    const float send = up ? vals[t2] : vals[t2 + msk];
                    const float keep = up ? vals[t2 + msk] : vals[t2];
                    vals[t2] = keep + __shfl_xor_sync(0xffffffffu, send, msk);
                }
            }
            float sc = vals[0] * p.qk_scale_log2;
            const int slot_own = bs + i_own * C::SG + grp;
            if (slot_own >= n || g_own >= G) sc = -INFINITY;
            float bm = sc;
#pragma unroll
            for (int msk = C::GP; msk < 32; msk <<= 1) bm = fmaxf(bm, __shfl_xor_sync(0xffffffffu, bm, msk));
            const bool need = bm > m_own + kTau;
            if (__any_sync(0xffffffffu, need)) {
                const float m_new = need ? bm : m_own;
                const float a_own = (m_new == m_own) ? 1.f : exp2f(m_own - m_new);
                l_own *= a_own;
                m_own = m_new;
#pragma unroll
                for (int g = 0; g < G; ++g) {
                    const float a = __shfl_sync(0xffffffffu, a_own, g);
                    const float2 a2 = make_float2(a, a);
#pragma unroll
                    for (int c = 0; c < C::CP2; ++c) O[g][c] = __fmul2_rn(O[g][c], a2);
                }
            }
            const float pr = (g_own < G) ? exp2f(sc - m_own) : 0.f;
            l_own += pr;
#pragma unroll
            for (int i = 0; i < C::NB; ++i) {
                const int slot = bs + i * C::SG + grp;
                const int row = slot < n ? slot : n - 1;
                float2 pb[G];
#pragma unroll
                for (int g = 0; g < G; ++g) {
                    const float pg = __shfl_sync(0xffffffffu, pr, grp * C::LPS + i * C::GP + g);
                    pb[g] = make_float2(pg, pg);
                }
#pragma unroll
                for (int cc = 0; cc < C::NCH; ++cc) {
                    float2 vf[4];
                    unpack8(lds128(Vs + row * kRowBytes + (k + cc * C::LPS) * 16), vf);
#pragma unroll
                    for (int e = 0; e < 4; ++e)
#pragma unroll
                        for (int g = 0; g < G; ++g) O[g][cc * 4 + e] = __ffma2_rn(pb[g], vf[e], O[g][cc * 4 + e]);
                }
            }
        }

        if (hd.y & kNewTok) {  // fused append: the new token's K/V row and position go into the cache
            const int b = hd.z / p.lay.KVH, h = hd.z - b * p.lay.KVH;
            const long long row = hd.w;
            const uint4 v = lds128((lane < 16 ? Ks : Vs) + (lane & 15) * 16);
            reinterpret_cast<uint4*>((lane < 16 ? p.lay.kpool : p.lay.vpool) + row * kHeadDim)[lane & 15] = v;
            if (lane == 0) {
                const long long slot = row - p.lay.gen_row0;  // region * Cmax + cached index
                const int g0 = p.seq_g[b];
                p.lay.pos[slot] = p.lay.seq_lp[b] + g0;
                if (h == 0) {
                    DevCounters* cnt = p.lay.counters + (size_t)p.layer * p.lay.B + b;
                    cnt->c = (int)(slot % p.lay.Cmax) + 1;
                    cnt->g = g0 + 1;
                }
            }
        }

        if (hd.y & kLast) {  // last tile of the piece
            float l = l_own;
#pragma unroll
            for (int msk = C::GP; msk < 32; msk <<= 1) l += __shfl_xor_sync(0xffffffffu, l, msk);
#pragma unroll
            for (int g = 0; g < G; ++g)
#pragma unroll
                for (int c = 0; c < C::CP2; ++c)
#pragma unroll
                    for (int msk = C::LPS; msk < 32; msk <<= 1) {
                        O[g][c].x += __shfl_xor_sync(0xffffffffu, O[g][c].x, msk);
                        O[g][c].y += __shfl_xor_sync(0xffffffffu, O[g][c].y, msk);
                    }
            const int hid = hd.z;
            const int b = hid / p.lay.KVH, h = hid - b * p.lay.KVH;
            const int hl = seq_head_len(p, b);
            const long long A = p.seq_base[b] + (long long)h * hl;
            const int w0 = (int)(A / p.W), w1 = (int)((A + hl - 1) / p.W);
            // l of head g sits in lane g (lanes 0..G-1 have g_own = lane)
            float lg[G];
#pragma unroll
            for (int g = 0; g < G; ++g) lg[g] = __shfl_sync(0xffffffffu, l, g);
            if (w0 == w1) {  // the whole head was this warp's: normalise and write the output
                if (grp == 0) {
#pragma unroll
                    for (int g = 0; g < G; ++g) {
                        const float inv = 1.f / lg[g];
                        uint16_t* out = p.out + ((size_t)b * p.lay.H + (size_t)h * G + g) * kHeadDim;
#pragma unroll
                        for (int cc = 0; cc < C::NCH; ++cc) {
                            const float2* o = &O[g][cc * 4];
                            uint4 w;
                            w.x = pack_bf16x2(o[0].x * inv, o[0].y * inv);
                            w.y = pack_bf16x2(o[1].x * inv, o[1].y * inv);
                            w.z = pack_bf16x2(o[2].x * inv, o[2].y * inv);
                            w.w = pack_bf16x2(o[3].x * inv, o[3].y * inv);
                            reinterpret_cast<uint4*>(out)[k + cc * C::LPS] = w;
                        }
                    }
                }
            } else {
                float* rec = p.partial + (size_t)(gw + hid) * partial_stride(G);
                if (grp == 0) {
#pragma unroll
                    for (int g = 0; g < G; ++g)
#pragma unroll
                        for (int cc = 0; cc < C::NCH; ++cc) {
                            float4* dst = reinterpret_cast<float4*>(rec + g * kHeadDim + (k + cc * C::LPS) * 8);
                            const float2* o = &O[g][cc * 4];
                            dst[0] = make_float4(o[0].x, o[0].y, o[1].x, o[1].y);
                            dst[1] = make_float4(o[2].x, o[2].y, o[3].x, o[3].y);
                        }
                }
                if (lane < G) {
                    rec[G * kHeadDim + lane] = m_own;
                    rec[G * kHeadDim + G + lane] = l;
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
            m_own = -INFINITY;
            l_own = 0.f;
#pragma unroll
            for (int g = 0; g < G; ++g)
#pragma unroll
                for (int c = 0; c < C::CP2; ++c) O[g][c] = make_float2(0.f, 0.f);
        }

        __syncwarp();
        if (more) {  // refill the stage just consumed with the tile SPW ahead
            if (lane == 0) fence_proxy_async_smem();
            more = issue(t + C::SPW);
            if (more) ++issued;
        }
    }
}

// Active sequences whose heads hold no slot at all (empty prompt, nothing generated)
// attend over nothing: their output rows are zero.
__global__ void __launch_bounds__(256) zero_empty_kernel(const __grid_constant__ AttnParams p)
{
    pdl_launch_dependents();
    pdl_wait();
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
    return launch_pdl(attn_kernel<G>, dim3(ctas), dim3(C::WARPS * 32), C::SMEM, s, p, *tk, *tv);
}

template <int G>
cudaError_t prepare_g()
{
    return cudaFuncSetAttribute(attn_kernel<G>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg<G>::SMEM);
}

}  // namespace

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

}  // namespace ra
