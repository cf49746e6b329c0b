// ra_evict.cu -- cache writes and Random Attention eviction on sm_103a.
//
//   append_kernel   one warp per (seq, KV head): the step's post-RoPE K/V row
//                   and its position go to slot c of the head's region
//                   (Appendix F: keys stored post-RoPE, cumulative counter).
//   select_kernel   one CTA per triggered (seq, KV head): Philox4x32-10 score
//                   per candidate (section 3's i.i.d. uniform draw; or one of
//                   the variants the paper contrasts: a draw shared by all heads,
//                   protected recency, block-contiguous draws), radix select of
//                   the K smallest (score, ordinal) -- Eq. 1 -- and a
//                   ballot-compacted, ascending list of the evicted ordinals.
//                   Under the scored comparator the score is the max-pooled
//                   window attention that ra_score.cu computed; with order-free
//                   slots every key follows the candidate's position.
//                   With order-free slots the select CTA also refills the
//                   evicted slots in place from the newest ones (no compact).
//   compact_kernel  many CTAs per triggered head: order-preserving move of the
//                   survivors (kept candidates, then the buffer rows) into
//                   the head's spare region with coalesced 16-byte copies
//                   (Appendix F keeps each keep-set in time order and gathers
//                   the cache into it).  Out of place, so CTAs never wait on
//                   each other; the old region becomes the spare.
#include <cuda_runtime.h>
#include <stdint.h>

#include "ra_internal.h"
#include "ra_ptx.cuh"

namespace ra {
namespace {

// Philox4x32-10, Salmon et al. (SC'11): ten rounds of two 32x32->64-bit
// multiplies; the high halves are xored with the other two counter words and
// the round key; the key advances by the two Weyl constants between rounds.
// Returns word 0 of the output block.
__device__ __forceinline__ uint32_t philox4x32_10_w0(uint32_t x0, uint32_t x1, uint32_t x2, uint32_t x3,
                                                     uint32_t k0, uint32_t k1)
{
#pragma unroll
    for (int round = 0; round < 10; ++round) {
        const uint32_t p_hi = __umulhi(0xD2511F53u, x0), p_lo = 0xD2511F53u * x0;
        const uint32_t q_hi = __umulhi(0xCD9E8D57u, x2), q_lo = 0xCD9E8D57u * x2;
        const uint32_t n0 = q_hi ^ x1 ^ k0;
        const uint32_t n2 = p_hi ^ x3 ^ k1;
        x0 = n0;
        x1 = q_lo;
        x2 = n2;
        x3 = p_lo;
        k0 += 0x9E3779B9u;
        k1 += 0xBB67AE85u;
    }
    return x0;
}

__device__ __forceinline__ bool bit_on(const uint32_t* mask, int b) { return (mask[b >> 5] >> (b & 31)) & 1u; }

// ----------------------------------------------------------------------------- append
__global__ void __launch_bounds__(1024) append_kernel(const __grid_constant__ AppendParams p)
{
    pdl_wait();
    pdl_launch_dependents();
    const int b = blockIdx.x;
    if (!bit_on(p.active, b)) return;
    const DevLayout& L = p.lay;
    const int h = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int c = p.seq_c[b], g = p.seq_g[b];
    const int reg = L.region[((size_t)p.layer * L.B + b) * L.KVH + h];
    const long long row = L.gen_row0 + (long long)reg * L.Cmax + c;
    const size_t src = ((size_t)b * L.KVH + h) * kHeadDim;
    if (lane < 16) {
        const uint4 v = reinterpret_cast<const uint4*>(p.k_new + src)[lane];
        reinterpret_cast<uint4*>(L.kpool + row * kHeadDim)[lane] = v;
    } else {
        const uint4 v = reinterpret_cast<const uint4*>(p.v_new + src)[lane - 16];
        reinterpret_cast<uint4*>(L.vpool + row * kHeadDim)[lane - 16] = v;
    }
    if (lane == 0) L.pos[(size_t)reg * L.Cmax + c] = L.seq_lp[b] + g;
}

// ----------------------------------------------------------------------------- select
constexpr int kSelThreads = 256;

__global__ void __launch_bounds__(kSelThreads) select_kernel(const __grid_constant__ EvictParams p)
{
    extern __shared__ uint32_t sm[];
    __shared__ uint32_t hist[3][256];
    __shared__ uint32_t s_total;
    // With p.early the keys, the radix select and the evicted list are computed before waiting for
    // the previous kernel (their inputs come from kernels that completed earlier); everything this
    // kernel writes to global memory comes after the wait.
    if (!p.early) {
        pdl_wait();
        pdl_launch_dependents();
    }
    const DevLayout& L = p.lay;
    const int b = p.trig[blockIdx.x], h = blockIdx.y;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    // With a pending token (fused step) the cache holds c rows and the token about to be
    // appended is the newest slot: the candidate count and the step include it.
    const int c = p.trig_c[blockIdx.x], N = p.trig_n[blockIdx.x], g = p.trig_g[blockIdx.x];
    const int K = L.K, r = L.r;
    const int m = N - K;
    const int head_id = b * L.KVH + h;
    int32_t* plan = L.plan + (size_t)head_id * (kPlanHeader + r);
    if (m <= 0 || m > r || N > kMaxCandidates || N > c) {  // the host mirror rules this out; never move data on a bad plan
        if (p.early) {
            pdl_wait();
            pdl_launch_dependents();
        }
        if (tid == 0) {
            atomicExch(L.err, kDeviceErrPlan);
            plan[3] = 0;
        }
        return;
    }
    const int nwords = (N + 31) >> 5;
    uint32_t* keys = sm;                       // [N]
    uint32_t* evbits = sm + nwords * 32;       // [nwords]
    int32_t* s_ev = reinterpret_cast<int32_t*>(evbits + nwords);  // [r] evicted ordinals, ascending
    // (under the scored policy the raw scores follow s_ev)

    if (tid < 256) hist[0][tid] = 0;  // the first digit's histogram (the fill's barrier publishes it)
    const uint32_t k0 = (uint32_t)L.seed, k1 = (uint32_t)(L.seed >> 32);
    const int32_t* pos = L.pos + (size_t)L.region[((size_t)p.layer * L.B + b) * L.KVH + h] * L.Cmax;
    if (p.holefill && p.policy != RA_POLICY_BLOCK) {  // order-free slots: every key follows the position
        const uint32_t id = p.policy == RA_POLICY_SHARED ? (uint32_t)(b * L.KVH) : (uint32_t)head_id;
#pragma unroll 8
        for (int j = tid; j < N; j += kSelThreads) {
            const uint32_t pj = (uint32_t)__ldg(pos + j);
            keys[j] = p.policy == RA_POLICY_RECENCY ? 0xFFFFFFFFu - pj
                                                    : philox4x32_10_w0(pj, (uint32_t)g, (uint32_t)p.layer, id, k0, k1);
        }
    } else if (p.policy == RA_POLICY_RECENCY) {  // protected recency: the K newest candidates score lowest
        for (int j = tid; j < N; j += kSelThreads) keys[j] = (uint32_t)(N - 1 - j);
    } else if (p.policy == RA_POLICY_BLOCK) {  // one draw per block of consecutive positions
        for (int j = tid; j < N; j += kSelThreads)
            keys[j] = philox4x32_10_w0((uint32_t)(pos[j] / p.block), (uint32_t)g, (uint32_t)p.layer, (uint32_t)head_id,
                                       k0, k1);
    } else if (p.policy == RA_POLICY_SNAPKV) {
        // scored comparator: the window score max-pooled over +-kScorePoolRadius candidates;
        // larger scores must sort first, so the key is the order-reversed float
        const float* sc = L.scores + (((size_t)p.layer * L.B + b) * L.KVH + h) * L.Cmax;
        float* raw = reinterpret_cast<float*>(s_ev + r);  // [N], staged once
#pragma unroll 4
        for (int j = tid; j < N; j += kSelThreads) raw[j] = __ldcg(sc + j);
        __syncthreads();
        for (int j = tid; j < N; j += kSelThreads) {
            float m = raw[j];
#pragma unroll
            for (int d = 1; d <= kScorePoolRadius; ++d) {
                if (j - d >= 0) m = fmaxf(m, raw[j - d]);
                if (j + d < N) m = fmaxf(m, raw[j + d]);
            }
            const uint32_t u = __float_as_uint(m);
            const uint32_t asc = (u & 0x80000000u) ? ~u : (u | 0x80000000u);  // ascending with the float
            keys[j] = ~asc;
        }
    } else {  // random: an independent draw per KV head; shared: one draw for all heads of the sequence
        const uint32_t id = p.policy == RA_POLICY_SHARED ? (uint32_t)(b * L.KVH) : (uint32_t)head_id;
        for (int j = tid; j < N; j += kSelThreads)
            keys[j] = philox4x32_10_w0((uint32_t)j, (uint32_t)g, (uint32_t)p.layer, id, k0, k1);
    }
    __syncthreads();

    // Radix select of the element at rank K (0-based) of the (key, ordinal) order:
    // 8 bits at a time from the top.  Afterwards T is its key and `rank` is its
    // rank among the keys equal to T, i.e. the number of ties that are kept.
    // One barrier per digit: every warp scans the histogram itself, and the
    // histograms rotate over three buffers -- the one a pass fills was last read
    // two passes earlier, before the previous barrier, so it is cleared
    // (during the pass before) without a barrier of its own.
    uint32_t prefix = 0, mask = 0;
    uint32_t rank = (uint32_t)K;
    for (int pass = 0; pass < 4; ++pass) {
        const int shift = 24 - 8 * pass;
        uint32_t* H = hist[pass % 3];
        if (tid < 256) hist[(pass + 1) % 3][tid] = 0;
        // A warp whose in-prefix keys all share one bin (the common case for the scored
        // policy's first digits, and once few keys remain) adds once; otherwise each lane adds.
        for (int j0 = warp * 32; j0 < N; j0 += kSelThreads) {
            const int j = j0 + lane;
            const uint32_t kk = j < N ? keys[j] : 0u;
            const bool in = j < N && (kk & mask) == prefix;
            const uint32_t bin = (kk >> shift) & 255u;
            const uint32_t inb = __ballot_sync(0xffffffffu, in);
            if (inb == 0u) continue;
            const int leader = __ffs(inb) - 1;
            const uint32_t b0 = __shfl_sync(0xffffffffu, bin, leader);
            if (__all_sync(0xffffffffu, !in || bin == b0)) {
                if (lane == leader) atomicAdd(&H[b0], (uint32_t)__popc(inb));
            } else if (in) {
                atomicAdd(&H[bin], 1u);
            }
        }
        __syncthreads();
        uint32_t loc[8], sum = 0;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            loc[q] = H[lane * 8 + q];
            sum += loc[q];
        }
        uint32_t incl = sum;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t t = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += t;
        }
        const uint32_t excl = incl - sum;
        uint32_t bin = 0, before = 0;
        if (excl <= rank && rank < incl) {
            uint32_t cum = excl;
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                if (rank < cum + loc[q]) {
                    bin = (uint32_t)(lane * 8 + q);
                    before = cum;
                    break;
                }
                cum += loc[q];
            }
        }
        const int src = __ffs(__ballot_sync(0xffffffffu, excl <= rank && rank < incl)) - 1;
        bin = __shfl_sync(0xffffffffu, bin, src);
        before = __shfl_sync(0xffffffffu, before, src);
        rank -= before;
        prefix |= bin << shift;
        mask |= 255u << shift;
    }
    const uint32_t T = prefix;
    const uint32_t kept_ties = rank;

    // Evicted: key > T, and the ties beyond the first `kept_ties` (in ordinal order).
    for (int w = warp; w < nwords; w += kSelThreads / 32) {
        const int j = w * 32 + lane;
        const bool ev = (j < N) && keys[j] >= T;
        const uint32_t bits = __ballot_sync(0xffffffffu, ev);
        if (lane == 0) evbits[w] = bits;
    }
    __syncthreads();
    if (kept_ties > 0 && warp == 0) {  // rare: give the lowest-ordinal ties back to the keep-set
        uint32_t remaining = kept_ties;
        for (int w = 0; w < nwords && remaining > 0; ++w) {
            const int j = w * 32 + lane;
            const uint32_t eq = __ballot_sync(0xffffffffu, (j < N) && keys[j] == T);
            uint32_t clear = 0, e = eq;
            while (e && remaining > 0) {
                const uint32_t low = e & (~e + 1u);
                clear |= low;
                e ^= low;
                --remaining;
            }
            if (lane == 0) evbits[w] &= ~clear;
        }
    }
    __syncthreads();

    // Ascending list of evicted ordinals: warp 0 walks the bitmap 32 words at a time.
    if (warp == 0) {
        uint32_t off = 0;
        for (int base = 0; base < nwords; base += 32) {
            const int w = base + lane;
            uint32_t bits = (w < nwords) ? evbits[w] : 0u;
            const uint32_t cntb = __popc(bits);
            uint32_t incl = cntb;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const uint32_t t = __shfl_up_sync(0xffffffffu, incl, o);
                if (lane >= o) incl += t;
            }
            uint32_t pos = off + incl - cntb;
            while (bits) {
                const int bit = __ffs(bits) - 1;
                bits &= bits - 1;
                if (pos < (uint32_t)r) s_ev[pos] = w * 32 + bit;
                ++pos;
            }
            off += __shfl_sync(0xffffffffu, incl, 31);
        }
        if (lane == 0) s_total = off;
    }
    __syncthreads();
    if (p.early) {
        pdl_wait();
        pdl_launch_dependents();
    }
    for (int i = tid; i < min((int)s_total, r); i += kSelThreads) plan[kPlanHeader + i] = s_ev[i];
    if (tid == 0) {
        const int32_t* regp = L.region + ((size_t)p.layer * L.B + b) * L.KVH + h;
        const int src = *regp, dst = p.holefill ? src : L.spare[b * L.KVH + h];  // hole-filling works in place
        const bool ok = (s_total == (uint32_t)m);
        plan[0] = src;
        plan[1] = dst;
        plan[2] = c;
        plan[3] = ok ? m : 0;
        if (ok && !p.holefill) {
            L.region[((size_t)p.layer * L.B + b) * L.KVH + h] = dst;
            L.spare[b * L.KVH + h] = src;
        } else if (!ok) {
            atomicExch(L.err, kDeviceErrPlan);
        }
    }
    if (!p.holefill) return;
    // Order-free compaction, in place: evicted slot e_i takes the row of slot top - m + i, where
    // top is the slot count including a pending token (the newest slot, taken from the caller's
    // rows).  Those m <= r slots are all buffer slots, so sources and destinations never overlap.
    if (s_total != (uint32_t)m) return;
    const int top = p.k_new ? c + 1 : c;
    const long long row0 = L.gen_row0 + (long long)L.region[((size_t)p.layer * L.B + b) * L.KVH + h] * L.Cmax;
    int32_t* gpos = L.pos + (size_t)L.region[((size_t)p.layer * L.B + b) * L.KVH + h] * L.Cmax;
    const int part = lane & 15;
    uint16_t* pool = lane < 16 ? L.kpool : L.vpool;
    constexpr int kWarpsSel = kSelThreads / 32, kBatch = 8;  // rows a warp has in flight
    for (int i0 = warp; i0 < m; i0 += kWarpsSel * kBatch) {
        uint4 v[kBatch];
        int32_t pv[kBatch];
        int to[kBatch];
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {  // every load of the batch first ...
            const int i = i0 + u * kWarpsSel;
            to[u] = -1;
            if (i < m) {
                const int from = top - m + i;
                to[u] = s_ev[i];
                if (from == c) {  // the step's pending token
                    const uint16_t* src = (lane < 16 ? p.k_new : p.v_new) + ((size_t)b * L.KVH + h) * kHeadDim;
                    v[u] = reinterpret_cast<const uint4*>(src)[part];
                    pv[u] = L.seq_lp[b] + g - 1;
                } else {
                    v[u] = reinterpret_cast<const uint4*>(pool + (row0 + from) * kHeadDim)[part];
                    pv[u] = gpos[from];
                }
            }
        }
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {  // ... then the stores
            if (to[u] < 0) continue;
            reinterpret_cast<uint4*>(pool + (row0 + to[u]) * kHeadDim)[part] = v[u];
            if (lane == 0) gpos[to[u]] = pv[u];
        }
    }
}

// ----------------------------------------------------------------------------- compact
constexpr int kCompactThreads = 256;
constexpr int kCompactUnroll = 4;
constexpr int kCompactChunk = 256;  // slots per CTA

__global__ void __launch_bounds__(kCompactThreads) compact_kernel(const __grid_constant__ EvictParams p)
{
    extern __shared__ int32_t s_ev[];
    __shared__ int32_t s_hdr[4];
    __shared__ int32_t s_dst[kCompactChunk];
    pdl_wait();
    pdl_launch_dependents();
    const DevLayout& L = p.lay;
    const int t = blockIdx.y / L.KVH, h = blockIdx.y % L.KVH;
    const int b = p.trig[t];
    const int head_id = b * L.KVH + h;
    const int32_t* plan = L.plan + (size_t)head_id * (kPlanHeader + L.r);
    if (threadIdx.x < 4) s_hdr[threadIdx.x] = plan[threadIdx.x];
    __syncthreads();
    const int src = s_hdr[0], dst = s_hdr[1], c = s_hdr[2], m = s_hdr[3];
    if (m <= 0) return;  // select flagged a bad plan: region table untouched, nothing moves
    for (int i = threadIdx.x; i < m; i += kCompactThreads) s_ev[i] = plan[kPlanHeader + i];
    __syncthreads();
    const int s0 = blockIdx.x * kCompactChunk;
    if (s0 >= c) return;
    const int s1 = min(c, s0 + kCompactChunk);
    // destination of every slot of the chunk: j - #evicted(< j), or -1 if j is evicted
    for (int t = threadIdx.x; t < s1 - s0; t += kCompactThreads) {
        const int j = s0 + t;
        int lo = 0, hi = m;
        while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (s_ev[mid] < j) lo = mid + 1; else hi = mid;
        }
        s_dst[t] = (lo < m && s_ev[lo] == j) ? -1 : j - lo;
    }
    __syncthreads();
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const uint16_t* sbase = (lane < 16 ? L.kpool : L.vpool) + (L.gen_row0 + (long long)src * L.Cmax) * kHeadDim;
    uint16_t* dbase = (lane < 16 ? L.kpool : L.vpool) + (L.gen_row0 + (long long)dst * L.Cmax) * kHeadDim;
    const int part = lane & 15;
    const int32_t* spos = L.pos + (size_t)src * L.Cmax;
    int32_t* dpos = L.pos + (size_t)dst * L.Cmax;
    for (int base = s0 + warp * kCompactUnroll; base < s1; base += (kCompactThreads / 32) * kCompactUnroll) {
        uint4 val[kCompactUnroll];
        int dj[kCompactUnroll];
        int pv[kCompactUnroll];
#pragma unroll
        for (int u = 0; u < kCompactUnroll; ++u) {
            const int j = base + u;
            dj[u] = j < s1 ? s_dst[j - s0] : -1;
            if (dj[u] >= 0) {
                val[u] = __ldg(reinterpret_cast<const uint4*>(sbase + (size_t)j * kHeadDim) + part);
                if (lane == 0) pv[u] = __ldg(spos + j);
            }
        }
#pragma unroll
        for (int u = 0; u < kCompactUnroll; ++u) {
            if (dj[u] >= 0) {
                reinterpret_cast<uint4*>(dbase + (size_t)dj[u] * kHeadDim)[part] = val[u];
                if (lane == 0) dpos[dj[u]] = pv[u];
            }
        }
    }
}

// ----------------------------------------------------------------------------- timeout probe
// The failure path of every bounded wait, run on purpose: one arrival with 16 bytes of
// transfer expected, and no copy ever issued, so the barrier's phase cannot complete; the
// bounded wait gives up after limit_ns and the error word is flagged as the pipelines do.
__global__ void __launch_bounds__(32) timeout_probe_kernel(int32_t* err, uint64_t limit_ns)
{
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x != 0) return;
    mbar_init(&bar, 1);
    fence_mbar_init();
    mbar_arrive_expect_tx(&bar, 16u);
    if (!mbar_wait_bounded(&bar, 0u, limit_ns)) atomicExch(err, kDeviceErrTimeout);
    mbar_inval(&bar);
}

// ----------------------------------------------------------------------------- prefill / restore
__global__ void __launch_bounds__(256) copy_rows_kernel(const __grid_constant__ CopyRowsParams p, int restore)
{
    const DevLayout& L = p.lay;
    const int b = blockIdx.x / L.KVH, h = blockIdx.x % L.KVH;
    const int n = p.n_rows[b];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    long long row0;
    int32_t* dpos = nullptr;
    if (restore) {
        const int reg = L.region[((size_t)p.layer * L.B + b) * L.KVH + h];
        row0 = L.gen_row0 + (long long)reg * L.Cmax;
        dpos = L.pos + (size_t)reg * L.Cmax;
    } else {
        row0 = (long long)p.layer * L.prompt_rows_per_layer + L.seq_poff[b] + (long long)h * L.seq_lp[b];
    }
    const size_t src0 = ((size_t)b * L.KVH + h) * (size_t)p.row_stride;
    const uint16_t* sb = (lane < 16 ? p.k : p.v);
    uint16_t* db = (lane < 16 ? L.kpool : L.vpool);
    for (int i = warp; i < n; i += 8) {
        const uint4 v = reinterpret_cast<const uint4*>(sb + (src0 + i) * kHeadDim)[lane & 15];
        reinterpret_cast<uint4*>(db + (row0 + i) * kHeadDim)[lane & 15] = v;
        if (restore && lane == 0) dpos[i] = p.pos[src0 + i];
    }
}

}  // namespace

// Scored policy, warm start: the r latest queries of every (seq, query head), oldest first,
// into the window slots of their steps.
struct RestoreQParams {
    DevLayout lay;
    int layer;
    const uint16_t* q;  // [B][H][r][128]
    int32_t g[RA_MAX_BATCH];
};

__global__ void __launch_bounds__(256) restore_queries_kernel(const __grid_constant__ RestoreQParams p)
{
    const DevLayout& L = p.lay;
    const int b = blockIdx.x / L.H, qh = blockIdx.x - b * L.H;
    const int h = qh / L.G, gq = qh - h * L.G;
    const int r = L.r;
    uint16_t* win = L.qring + (((size_t)p.layer * L.B + b) * L.KVH + h) * (size_t)r * L.G * kHeadDim;
    const uint16_t* src = p.q + ((size_t)b * L.H + qh) * (size_t)r * kHeadDim;
    for (int i = threadIdx.x; i < r * 16; i += blockDim.x) {
        const int u = i >> 4, c = i & 15;
        const int step = p.g[b] - r + 1 + u;  // 1-based decode step of row u
        if (step < 1) continue;
        const int slot = (step - 1) % r;
        reinterpret_cast<uint4*>(win + ((size_t)slot * L.G + gq) * kHeadDim)[c] =
            reinterpret_cast<const uint4*>(src + (size_t)u * kHeadDim)[c];
    }
}

cudaError_t launch_restore_queries(const DevLayout& lay, int layer, const uint16_t* q, const int32_t* g_host,
                                   cudaStream_t s)
{
    RestoreQParams p{};
    p.lay = lay;
    p.layer = layer;
    p.q = q;
    for (int b = 0; b < lay.B; ++b) p.g[b] = g_host[b];
    restore_queries_kernel<<<lay.B * lay.H, 256, 0, s>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_append(const AppendParams& p, int B, cudaStream_t s)
{
    return launch_pdl(append_kernel, dim3(B), dim3(p.lay.KVH * 32), 0, s, p);
}

// keys [N rounded to 32], the evicted bitmap, the evicted list [r], and under the scored policy
// the raw scores [N]
size_t select_smem(int N, int r, bool scored)
{
    const size_t words = (size_t)(N + 31) / 32;
    return (words * 32 + words + (size_t)r + (scored ? words * 32 : 0)) * sizeof(uint32_t);
}

cudaError_t launch_select(const EvictParams& p, cudaStream_t s)
{
    const int N = p.lay.K + p.lay.r;  // candidates at a firing step never exceed K + r
    const size_t smem = select_smem(N, p.lay.r, p.policy == RA_POLICY_SNAPKV);
    static size_t configured = 0;
    if (smem > 48 * 1024 && smem > configured) {
        cudaError_t e = cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        configured = smem;
    }
    return launch_pdl(select_kernel, dim3(p.n_trig, p.lay.KVH), dim3(kSelThreads), smem, s, p);
}

cudaError_t launch_compact(const EvictParams& p, cudaStream_t s)
{
    const int Cmax = p.lay.Cmax;
    const int chunks = (Cmax + kCompactChunk - 1) / kCompactChunk;
    return launch_pdl(compact_kernel, dim3(chunks, p.n_trig * p.lay.KVH), dim3(kCompactThreads),
                      p.lay.r * sizeof(int32_t), s, p);
}

cudaError_t launch_timeout_probe(int32_t* err, uint64_t limit_ns, cudaStream_t s)
{
    timeout_probe_kernel<<<1, 32, 0, s>>>(err, limit_ns);
    return cudaGetLastError();
}

cudaError_t launch_prefill(const CopyRowsParams& p, cudaStream_t s)
{
    copy_rows_kernel<<<p.lay.B * p.lay.KVH, 256, 0, s>>>(p, 0);
    return cudaGetLastError();
}

cudaError_t launch_restore(const CopyRowsParams& p, cudaStream_t s)
{
    copy_rows_kernel<<<p.lay.B * p.lay.KVH, 256, 0, s>>>(p, 1);
    return cudaGetLastError();
}

}  // namespace ra
