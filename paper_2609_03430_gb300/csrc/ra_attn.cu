// ra_attn.cu -- GQA split-K flash-decode attention over the per-head caches (sm_103a).
//
// Computes, for every active sequence b and query head qh (KV head h = qh / G),
//     o = sum_i softmax_i(scale * q . k_i) v_i
// over the prompt rows and the cached generated rows of (b, h) -- section 2
// ("Notation"), with the grouped-query sharing of Appendix F.
//
// Work split ("stream-K" by warp): the slots of all heads of the layer are laid
// end to end (sequence-major, then KV head, then prompt slots, then generated
// slots) and every warp of the grid takes one contiguous range of W slots.  A
// warp runs its own pipeline: lane 0 streams tiles of TILE rows of K and of V
// (and, at the first tile of each head piece, the G query rows) into a ring of
// SPW shared-memory stages with 2-D TMA loads completing on per-stage
// mbarriers; all 32 lanes consume.  At the end of each (head, warp) piece the
// warp writes an fp32 partial (unnormalised o, running max m, sum l) to slot
// `warp + head` of the partial buffer -- unique because warps and heads both
// advance monotonically through the slot order -- and combine_kernel merges
// the pieces of every head.
//
// Per-warp compute layout: LPS lanes share one cache row (each lane owns
// 16 bytes -- 8 channels -- of every LPS-th 16-byte chunk, so a row read is
// bank-conflict free); the warp works on 32/LPS rows at once.  The G query rows
// live in fp32 registers; each K row is read once from shared memory and used
// by all G heads (G flop per byte).  Partial dot products are summed across the
// LPS lanes with a butterfly reduce-scatter (each exchange halves the vector),
// which leaves exactly one (row, head) score per lane.  The softmax is online
// in base 2 with the scale folded into one multiply; the running max is only
// raised when a batch exceeds it by more than 2^8 (results are unchanged up to
// rounding, as softmax is shift invariant), so rescaling the accumulators is
// rare.
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
    static_assert(STAGE_BYTES % 128 == 0, "TMA destinations stay 128-byte aligned");
    static_assert(SMEM <= 232448, "fits the 227 KB opt-in shared memory of sm_100+");
    static_assert(LPS * 1 == NB * GP, "one reduced score per lane");
    static_assert(TILE % BATCH == 0, "tile holds whole batches");
    static_assert(WARPS >= 4, "shared-memory budget too small");
};

// Producer-side walk over the warp's slot range.
struct TileIter {
    int f, end;          // flattened cursor and end of the warp's range
    int b, h, pos;       // current sequence, KV head, slot within the head
    int hl, lp;          // head length (prompt + generated) and prompt length
    long long prow, grow;// first prompt row / first generated row of the head
    bool piece_start;
};

struct TileDesc {
    long long row;
    int n, hid;
    bool first, last;
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
    it.prow = (long long)p.layer * L.prompt_rows_per_layer + L.seq_poff[it.b] + (long long)it.h * lp;
    const int reg = L.region[((size_t)p.layer * L.B + it.b) * L.KVH + it.h];
    it.grow = L.gen_row0 + (long long)reg * L.Cmax;
    it.piece_start = true;
}

__device__ void iter_init(TileIter& it, const AttnParams& p, int R0, int R1)
{
    it.f = R0;
    it.end = R1;
    // largest b with seq_base[b] <= R0 and a non-empty head range
    int lo = 0, hi = p.lay.B - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (p.seq_base[mid] <= R0) lo = mid; else hi = mid - 1;
    }
    int b = lo;
    while (b < p.lay.B && p.seq_base[b + 1] <= R0) ++b;  // skip empty sequences at the boundary
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
    const int seg_end = it.pos < it.lp ? it.lp : it.hl;
    const int rem = it.end - it.f;
    const int piece_end = (it.hl - it.pos < rem) ? it.hl : it.pos + rem;
    int n = (seg_end < piece_end ? seg_end : piece_end) - it.pos;
    if (n > tile) n = tile;
    d.row = it.pos < it.lp ? it.prow + it.pos : it.grow + (it.pos - it.lp);
    d.n = n;
    d.hid = it.b * p.lay.KVH + it.h;
    d.first = it.piece_start;
    d.last = (it.pos + n == piece_end);
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

template <int G>
__device__ __forceinline__ void unpack8(const uint4 u, float* f)
{
    f[0] = bf16lo(u.x); f[1] = bf16hi(u.x);
    f[2] = bf16lo(u.y); f[3] = bf16hi(u.y);
    f[4] = bf16lo(u.z); f[5] = bf16hi(u.z);
    f[6] = bf16lo(u.w); f[7] = bf16hi(u.w);
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

    TileIter it;
    iter_init(it, p, R0, R1);
    int issued = 0;
    auto issue = [&](int t) -> bool {
        TileDesc d;
        if (!iter_next(it, p, C::TILE, d)) return false;
        const int s = t % C::SPW;
        if (lane == 0) {
            uint8_t* st = wstage + (size_t)s * C::STAGE_BYTES;
            hdrs[s] = make_int4(d.n, (d.first ? 1 : 0) | (d.last ? 2 : 0), d.hid, 0);
            const uint32_t bytes = 2u * C::KV_BYTES + (d.first ? (uint32_t)C::Q_BYTES : 0u);
            mbar_arrive_expect_tx(&bars[s], bytes);
            tma_load_2d(st, &tk, 0, (int)d.row, &bars[s]);
            tma_load_2d(st + C::KV_BYTES, &tv, 0, (int)d.row, &bars[s]);
            if (d.first) {
                const int b = d.hid / p.lay.KVH, h = d.hid - b * p.lay.KVH;
                bulk_load(st + 2 * C::KV_BYTES, p.q + ((size_t)b * p.lay.H + (size_t)h * G) * kHeadDim,
                          (uint32_t)C::Q_BYTES, &bars[s]);
            }
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

    float qf[G][C::CPL];
    float O[G][C::CPL];
    float m_own = -INFINITY, l_own = 0.f;
#pragma unroll
    for (int g = 0; g < G; ++g)
#pragma unroll
        for (int c = 0; c < C::CPL; ++c) O[g][c] = 0.f;

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
        if (hd.y & 1) {  // first tile of a head piece: fresh query rows
            const uint8_t* Qs = Vs + C::KV_BYTES;
#pragma unroll
            for (int g = 0; g < G; ++g)
#pragma unroll
                for (int cc = 0; cc < C::NCH; ++cc) unpack8<G>(lds128(Qs + g * kRowBytes + (k + cc * C::LPS) * 16), &qf[g][cc * 8]);
        }

        for (int bs = 0; bs < n; bs += C::BATCH) {
            float vals[C::LPS];
#pragma unroll
            for (int v = 0; v < C::LPS; ++v) vals[v] = 0.f;
#pragma unroll
            for (int i = 0; i < C::NB; ++i) {
                const int slot = bs + i * C::SG + grp;
                const int row = slot < n ? slot : n - 1;
#pragma unroll
                for (int cc = 0; cc < C::NCH; ++cc) {
                    float kf[8];
                    unpack8<G>(lds128(Ks + row * kRowBytes + (k + cc * C::LPS) * 16), kf);
#pragma unroll
                    for (int g = 0; g < G; ++g)
#pragma unroll
                        for (int e = 0; e < 8; ++e) vals[i * C::GP + g] = fmaf(qf[g][cc * 8 + e], kf[e], vals[i * C::GP + g]);
                }
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
#pragma unroll
                    for (int c = 0; c < C::CPL; ++c) O[g][c] *= a;
                }
            }
            const float pr = (g_own < G) ? exp2f(sc - m_own) : 0.f;
            l_own += pr;
#pragma unroll
            for (int i = 0; i < C::NB; ++i) {
                const int slot = bs + i * C::SG + grp;
                const int row = slot < n ? slot : n - 1;
                float pb[G];
#pragma unroll
                for (int g = 0; g < G; ++g) pb[g] = __shfl_sync(0xffffffffu, pr, grp * C::LPS + i * C::GP + g);
#pragma unroll
                for (int cc = 0; cc < C::NCH; ++cc) {
                    float vf[8];
                    unpack8<G>(lds128(Vs + row * kRowBytes + (k + cc * C::LPS) * 16), vf);
#pragma unroll
                    for (int g = 0; g < G; ++g)
#pragma unroll
                        for (int e = 0; e < 8; ++e) O[g][cc * 8 + e] = fmaf(pb[g], vf[e], O[g][cc * 8 + e]);
                }
            }
        }

        if (hd.y & 2) {  // last tile of the piece: reduce across row groups and write the partial
            float l = l_own;
#pragma unroll
            for (int msk = C::GP; msk < 32; msk <<= 1) l += __shfl_xor_sync(0xffffffffu, l, msk);
#pragma unroll
            for (int g = 0; g < G; ++g)
#pragma unroll
                for (int c = 0; c < C::CPL; ++c)
#pragma unroll
                    for (int msk = C::LPS; msk < 32; msk <<= 1) O[g][c] += __shfl_xor_sync(0xffffffffu, O[g][c], msk);
            float* rec = p.lay.partial + (size_t)(gw + hd.z) * partial_stride(G);
            if (grp == 0) {
#pragma unroll
                for (int g = 0; g < G; ++g)
#pragma unroll
                    for (int cc = 0; cc < C::NCH; ++cc) {
                        float4* dst = reinterpret_cast<float4*>(rec + g * kHeadDim + (k + cc * C::LPS) * 8);
                        dst[0] = make_float4(O[g][cc * 8 + 0], O[g][cc * 8 + 1], O[g][cc * 8 + 2], O[g][cc * 8 + 3]);
                        dst[1] = make_float4(O[g][cc * 8 + 4], O[g][cc * 8 + 5], O[g][cc * 8 + 6], O[g][cc * 8 + 7]);
                    }
            }
            if (lane < G) {
                rec[G * kHeadDim + lane] = m_own;
                rec[G * kHeadDim + G + lane] = l;
            }
            m_own = -INFINITY;
            l_own = 0.f;
#pragma unroll
            for (int g = 0; g < G; ++g)
#pragma unroll
                for (int c = 0; c < C::CPL; ++c) O[g][c] = 0.f;
        }

        __syncwarp();
        if (more) {  // refill the stage just consumed with the tile SPW ahead
            if (lane == 0) fence_proxy_async_smem();
            more = issue(t + C::SPW);
            if (more) ++issued;
        }
    }
}

template <int G>
__global__ void __launch_bounds__(256) combine_kernel(const __grid_constant__ AttnParams p)
{
    const int wid = (int)((blockIdx.x * blockDim.x + threadIdx.x) >> 5);
    const int lane = threadIdx.x & 31;
    const DevLayout& L = p.lay;
    const int per_seq = L.KVH * G;
    const int b = wid / per_seq;
    if (b >= L.B) return;
    if (!((p.active[b >> 5] >> (b & 31)) & 1u)) return;
    const int rem = wid - b * per_seq;
    const int h = rem / G, g = rem - h * G;
    uint16_t* o = p.out + ((size_t)b * L.H + (size_t)h * G + g) * kHeadDim + lane * 4;
    const int hl = (p.seq_base[b + 1] - p.seq_base[b]) / L.KVH;
    if (hl == 0) {
        *reinterpret_cast<uint2*>(o) = make_uint2(0u, 0u);
        return;
    }
    const long long A = p.seq_base[b] + (long long)h * hl;
    const int w0 = (int)(A / p.W), w1 = (int)((A + hl - 1) / p.W);
    const int hid = b * L.KVH + h;
    const size_t rs = (size_t)partial_stride(G);
    float M = -INFINITY;
    for (int w = w0; w <= w1; ++w) M = fmaxf(M, p.lay.partial[(size_t)(w + hid) * rs + G * kHeadDim + g]);
    float Lsum = 0.f, acc[4] = {0.f, 0.f, 0.f, 0.f};
    for (int w = w0; w <= w1; ++w) {
        const float* rec = p.lay.partial + (size_t)(w + hid) * rs;
        const float a = exp2f(rec[G * kHeadDim + g] - M);
        Lsum = fmaf(a, rec[G * kHeadDim + G + g], Lsum);
        const float4 v = *reinterpret_cast<const float4*>(rec + g * kHeadDim + lane * 4);
        acc[0] = fmaf(a, v.x, acc[0]);
        acc[1] = fmaf(a, v.y, acc[1]);
        acc[2] = fmaf(a, v.z, acc[2]);
        acc[3] = fmaf(a, v.w, acc[3]);
    }
    const float inv = 1.f / Lsum;
    uint32_t packed[2];
#pragma unroll
    for (int j = 0; j < 2; ++j) {
        const uint32_t lo = __bfloat16_as_ushort(__float2bfloat16_rn(acc[2 * j] * inv));
        const uint32_t hi = __bfloat16_as_ushort(__float2bfloat16_rn(acc[2 * j + 1] * inv));
        packed[j] = lo | (hi << 16);
    }
    *reinterpret_cast<uint2*>(o) = make_uint2(packed[0], packed[1]);
}

template <int G>
cudaError_t launch_attn_g(const AttnParams& p, const CUtensorMap* tk, const CUtensorMap* tv, int ctas, cudaStream_t s)
{
    using C = Cfg<G>;
    attn_kernel<G><<<ctas, C::WARPS * 32, C::SMEM, s>>>(p, *tk, *tv);
    return cudaGetLastError();
}

template <int G>
cudaError_t prepare_g()
{
    return cudaFuncSetAttribute(attn_kernel<G>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg<G>::SMEM);
}

template <int G>
cudaError_t launch_combine_g(const AttnParams& p, cudaStream_t s)
{
    const long long warps = (long long)p.lay.B * p.lay.KVH * G;
    const int blocks = (int)((warps * 32 + 255) / 256);
    combine_kernel<G><<<blocks, 256, 0, s>>>(p);
    return cudaGetLastError();
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

cudaError_t launch_combine(const AttnParams& p, cudaStream_t s)
{
    switch (p.lay.G) {
        case 1: return launch_combine_g<1>(p, s);
        case 2: return launch_combine_g<2>(p, s);
        case 3: return launch_combine_g<3>(p, s);
        case 4: return launch_combine_g<4>(p, s);
        case 5: return launch_combine_g<5>(p, s);
        case 6: return launch_combine_g<6>(p, s);
        case 7: return launch_combine_g<7>(p, s);
        case 8: return launch_combine_g<8>(p, s);
    }
    return cudaErrorInvalidValue;
}

}  // namespace ra
