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
//   evict_kernel    the random policy and its key-per-ordinal variants in one
//                   launch: a thread-block cluster per triggered head draws the
//                   keys, selects the evicted set exactly across the cluster
//                   through distributed shared memory, and moves the survivors
//                   order-preserving with bulk copies (details below).
//   compact_kernel  many CTAs per triggered head: order-preserving move of the
//                   survivors (kept candidates, then the buffer rows) into
//                   the head's spare region with coalesced 16-byte copies
//                   (Appendix F keeps each keep-set in time order and gathers
//                   the cache into it).  Out of place, so CTAs never wait on
//                   each other; the old region becomes the spare.
//   plan_kernel     the next step's evicted sets in every layer, beside the
//                   current step (the draw needs no cache data but positions).
//   compact_stack_kernel / fill_stack_kernel
//                   at a whole-stack step, every layer's round of the firing
//                   sequences in one launch, in place, from those sets:
//                   order-preserving, or refilling the evicted slots.
#include <cuda_runtime.h>
#include <limits.h>

#include <algorithm>
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
        const uint32_t id = key_stream(p.trig_admit[blockIdx.x],
                                       p.policy == RA_POLICY_SHARED ? (uint32_t)(b * L.KVH) : (uint32_t)head_id);
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
            keys[j] = philox4x32_10_w0((uint32_t)(pos[j] / p.block), (uint32_t)g, (uint32_t)p.layer,
                                       key_stream(p.trig_admit[blockIdx.x], (uint32_t)head_id), k0, k1);
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
        const uint32_t id = key_stream(p.trig_admit[blockIdx.x],
                                       p.policy == RA_POLICY_SHARED ? (uint32_t)(b * L.KVH) : (uint32_t)head_id);
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
    // Order-free compaction, in place.  With top the slot count including a pending token: evicted
    // slot e_i takes the row of slot top - m + i for i < m - 1, and the newest row ends in the new
    // last slot top - m - 1, whose own row, unless e_{m-1} is that slot, fills e_{m-1}.  A pending
    // token is the newest row: the attention kernel appends it into the new last slot afterwards.
    // Slots top - m .. top - 1 are buffer slots, so no move reads a slot that another writes.
    if (s_total != (uint32_t)m) return;
    const int top = p.pending ? c + 1 : c, last = top - m - 1;
    const long long row0 = L.gen_row0 + (long long)L.region[((size_t)p.layer * L.B + b) * L.KVH + h] * L.Cmax;
    int32_t* gpos = L.pos + (size_t)L.region[((size_t)p.layer * L.B + b) * L.KVH + h] * L.Cmax;
    const int part = lane & 15;
    uint16_t* pool = lane < 16 ? L.kpool : L.vpool;  // lanes 0-15 move K, 16-31 V, 16 bytes each
    auto row = [&](int slot) { return reinterpret_cast<uint4*>(pool + (row0 + slot) * kHeadDim) + part; };
    constexpr int kWarpsSel = kSelThreads / 32, kBatch = 8;  // rows a warp has in flight
    for (int i0 = warp; i0 < m - 1; i0 += kWarpsSel * kBatch) {
        uint4 v[kBatch];
        int32_t pv[kBatch];
        int to[kBatch];
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {  // every load of the batch first ...
            const int i = i0 + u * kWarpsSel;
            to[u] = -1;
            if (i < m - 1) {
                to[u] = s_ev[i];
                v[u] = *row(top - m + i);
                pv[u] = gpos[top - m + i];
            }
        }
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {  // ... then the stores
            if (to[u] < 0) continue;
            *row(to[u]) = v[u];
            if (lane == 0) gpos[to[u]] = pv[u];
        }
    }
    if (warp == kWarpsSel - 1) {  // the last evicted slot and the new last slot
        const int e = s_ev[m - 1];
        const bool fill_e = e != last, newest = !p.pending;
        uint4 a = make_uint4(0u, 0u, 0u, 0u), n = a;
        int32_t pa = 0, pn = 0;
        if (fill_e) {
            a = *row(last);
            pa = gpos[last];
        }
        if (newest) {
            n = *row(top - 1);
            pn = gpos[top - 1];
        }
        if (fill_e) {
            *row(e) = a;
            if (lane == 0) gpos[e] = pa;
        }
        if (newest) {
            *row(last) = n;
            if (lane == 0) gpos[last] = pn;
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

// ----------------------------------------------------------------------------- evict (select + compact)
// One launch per eviction round: for every triggered (seq, KV head), `reps` thread-block clusters
// of CL CTAs.  Each cluster selects the head's evicted set on its own (the replicas of a head
// compute the same set); the head's cached slots are cut into reps x CL equal row ranges, one
// per CTA, for the copy.  CTA k of a cluster draws the keys of the candidates
// [k N / CL, (k + 1) N / CL).
//
//   1. Keys of the own candidates (the same key rules as select_kernel), while the region
//      tables load; then every warp starts TMA bulk copies of its first chunks of K and V rows
//      into shared memory: the rows are read whatever the draw decides (about r of K + r are
//      evicted), so the copies overlap the selection, and with early = 1 the previous kernel's
//      tail too.
//   2. The evicted set is the m = N - K largest (key, ordinal) pairs, found exactly.
//      Random and shared draws (uniform 32-bit keys) first try a cut: only keys >= tau, with
//      tau set so that about 2m + 32 of the N candidates pass; each CTA lists its passing
//      candidates, the cluster exchanges the lists through distributed shared memory (one
//      barrier) and ranks them exactly.  If at least m passed (all but certainly), the top m
//      are the evicted set, since every candidate below the cut ranks lower.  Otherwise, and
//      for the other policies, radix passes over 8-bit digits from the top: each CTA's
//      histogram is summed by every CTA through distributed shared memory until the digit bin
//      holding the boundary has at most kEvCap candidates, which are gathered and ranked; if
//      all 32 bits tie, the largest ordinals are evicted first, CTA by CTA.  The CTAs then
//      exchange their evicted ordinals.  Either way every CTA ends with the whole ascending
//      list of evicted ordinals.
//   3. Slot j moves to j - (evicted ordinals below j); each warp stores the runs of surviving
//      rows of its chunks with bulk copies shared -> global (positions by plain stores),
//      refilling its buffers as they drain.  Out of place into the head's spare region, as
//      compact_kernel; CTA 0 of replica 0 swaps the region tables.
constexpr int kEvThreads = 256;
constexpr int kEvWarps = kEvThreads / 32;
constexpr int kEvCap = kEvMaxEvicted;  // candidates gathered for an exact ranking; also the most a round evicts
constexpr uint64_t kEvWaitLimitNs = 2000000000ull;
static_assert(kEvThreads == 256, "one thread per histogram bin");
static_assert(kEvCap <= 2 * kEvThreads, "a plan's ordinals are read two per thread");
static_assert(kEvMaxLocal % 32 == 0, "whole bitmap words");
static_assert(kMaxCandidates + 128 <= 65536, "ordinals and the CTA rank share one 32-bit word");

struct EvShared {
    uint32_t keys[kEvMaxLocal];
    uint32_t hist[2][256];            // this CTA's histogram of the current digit (double-buffered)
    uint32_t tot[256];                // the cluster's
    uint2 blist[kEvCap];              // own listed candidates: (key, ordinal)
    uint2 ball[kEvCap];               // everyone's: (key, rank << 16 | ordinal), ordered as (key, ordinal)
    int32_t evlist[kEvCap];           // every evicted ordinal, ascending
    int32_t evown[kEvCap];            // the cut: the evicted ordinals in any order; radix passes: own, ascending
    uint32_t evown_n;
    uint32_t bcnt, nev;
    uint32_t sel[6];
    uint32_t cnt[kEvMaxCluster];
    uint64_t bar[kEvWarps][kEvBufs];
};

// Gather the cluster's lists (S.blist of every CTA, S.bcnt entries each) into S.ball, tagging
// each entry with its CTA's rank; returns the total.  Entries keep the (key, ordinal) order.
__device__ __forceinline__ int gather_lists(EvShared& S, int CL, int tid)
{
    if (tid < CL) S.cnt[tid] = ld_dsmem_u32(dsmem_addr(&S.bcnt, tid));
    __syncthreads();
    int total = 0;
    for (int k = 0; k < CL; ++k) total += (int)S.cnt[k];
    if (total > kEvCap) return total;
    for (int e = tid; e < total; e += kEvThreads) {
        int k = 0, off = 0;
        while (e >= off + (int)S.cnt[k]) off += (int)S.cnt[k++];
        const uint2 x = ld_dsmem_u32x2(dsmem_addr(&S.blist[e - off], k));
        S.ball[e] = make_uint2(x.x, ((uint32_t)k << 16) | x.y);  // ranks grow with ordinals: order kept
    }
    return total;
}

// Number of evicted ordinals below j (S.evlist ascending, n entries).
__device__ __forceinline__ int ev_below(const EvShared& S, int n, int j)
{
    int lo = 0, hi = n;
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (S.evlist[mid] < j) lo = mid + 1; else hi = mid;
    }
    return lo;
}

template <int R, int NB>
__global__ void __launch_bounds__(kEvThreads, 1) evict_kernel(const __grid_constant__ EvictParams p)
{
    static_assert(R <= 32 && NB >= 3 && NB == kEvBufs, "a lane per row of a chunk; refills trail by one chunk");
    extern __shared__ __align__(128) uint8_t ev_dyn[];  // [warp][buffer][K rows R][V rows R]
    __shared__ EvShared S;
    constexpr int kBufBytes = 2 * R * kRowBytes;
    const DevLayout& L = p.lay;
    const int CL = (int)gridDim.x, reps = p.ev_reps;
    const uint32_t rank = cluster_ctarank();
    const int h = blockIdx.y / reps, rep = blockIdx.y - h * reps, t = blockIdx.z;
    const int b = p.trig[t];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int c = p.trig_c[t], N = p.trig_n[t], g = p.trig_g[t];
    const int m = N - L.K;
    const int head_id = b * L.KVH + h;
    // The host mirror rules these out; every CTA of the launch decides alike, so they leave together.
    // (a CTA keeps the keys of its candidates only when it selects itself, without a plan)
    if (m < 1 || m > L.r || m > kEvCap || N > c || N > kMaxCandidates ||
        (!p.ev_plan && (N + CL - 1) / CL > kEvMaxLocal) || CL > kEvMaxCluster || reps < 1) {
        pdl_wait();
        pdl_launch_dependents();
        if (tid == 0 && rank == 0 && rep == 0) atomicExch(L.err, kDeviceErrPlan);
        return;
    }
    const int j0 = (int)((long long)rank * N / CL), nloc = (int)((long long)(rank + 1) * N / CL) - j0;
    const int U = reps * CL, u = rep * CL + (int)rank;  // this CTA's share of the copy
    const int s0 = (int)((long long)u * c / U), s1 = (int)((long long)(u + 1) * c / U);
    uint8_t* wbuf = ev_dyn + (size_t)warp * NB * kBufBytes;
    uint64_t* wbar = S.bar[warp];
    S.hist[0][tid] = 0;
    if (tid == 0) S.bcnt = 0;
    __syncthreads();
    // With p.early the host has checked that the previous kernel writes none of this layer's
    // rows or positions: the copies and the selection start before waiting for it.  The regions
    // come from the host's mirror of the tables (checked against them below).
    if (!p.early) pdl_wait();
    const int src = p.trig_src[t] * L.KVH + h, dst = p.trig_dst[t] * L.KVH + h;

    // 1. keys (random / shared / recency keys need no memory, so they overlap the table loads),
    //    the cut's list or the first digit's histogram, then the first copies
    const bool cut = (p.policy == RA_POLICY_RANDOM || p.policy == RA_POLICY_SHARED) && !p.ev_exact;
    // tau = 2^32 (1 - E / N) with E = 2m + 32 expected to pass (all of them when E >= N)
    const uint64_t E = 2ull * (uint64_t)m + 32ull;
    const uint32_t tau = E >= (uint64_t)N ? 0u : (uint32_t)(((uint64_t)(N - E) << 32) / (uint64_t)N);
    const uint32_t k0 = (uint32_t)L.seed, k1 = (uint32_t)(L.seed >> 32);
    const uint32_t id =
        key_stream(p.trig_admit[t], p.policy == RA_POLICY_SHARED ? (uint32_t)(b * L.KVH) : (uint32_t)head_id);
    const int32_t* spos = L.pos + (size_t)src * L.Cmax;
    auto record = [&](int i, uint32_t key) {  // the key of local candidate i: kept, listed or counted
        S.keys[i] = key;
        if (!cut) {
            atomicAdd(&S.hist[0][key >> 24], 1u);
        } else if (key >= tau) {
            const uint32_t at = atomicAdd(&S.bcnt, 1u);
            if (at < (uint32_t)kEvCap) S.blist[at] = make_uint2(key, (uint32_t)(j0 + i));
        }
    };
    // a precomputed plan: the evicted ordinals of this head, [count][ordinals ascending]
    const int32_t* plan = p.ev_plan ? p.ev_plan + (size_t)(((size_t)p.ev_plan_parity * L.L + p.layer) * L.B * L.KVH +
                                                           (size_t)b * L.KVH + h) * (L.r + 1)
                                    : nullptr;
    // the plan's count and this thread's share of its ordinals, read before the row copies
    // start, so that the reads do not queue behind them
    int plan_n = 0, plan_v0 = 0, plan_v1 = 0;
    if (plan) {
        plan_n = __ldcg(plan);
        if (tid < m) plan_v0 = __ldcg(plan + 1 + tid);
        if (tid + kEvThreads < m) plan_v1 = __ldcg(plan + 1 + tid + kEvThreads);
    } else if (p.policy == RA_POLICY_RANDOM || p.policy == RA_POLICY_SHARED) {
        // four independent Philox chains per thread at a time (each chain is 10 serial rounds)
        for (int i0 = tid; i0 < nloc; i0 += 4 * kEvThreads) {
            uint32_t kq[4];
#pragma unroll
            for (int q = 0; q < 4; ++q)
                kq[q] = philox4x32_10_w0((uint32_t)(j0 + i0 + q * kEvThreads), (uint32_t)g, (uint32_t)p.layer, id, k0, k1);
#pragma unroll
            for (int q = 0; q < 4; ++q)
                if (i0 + q * kEvThreads < nloc) record(i0 + q * kEvThreads, kq[q]);
        }
    } else {
        for (int i = tid; i < nloc; i += kEvThreads) {
            const int j = j0 + i;
            record(i, p.policy == RA_POLICY_RECENCY  // the K newest candidates score lowest
                          ? (uint32_t)(N - 1 - j)
                          : philox4x32_10_w0((uint32_t)(__ldg(spos + j) / p.block), (uint32_t)g, (uint32_t)p.layer,
                                             key_stream(p.trig_admit[t], (uint32_t)head_id), k0, k1));
        }
    }
    if (lane == 0) {  // this warp's copy barriers
        for (int i = 0; i < NB; ++i) mbar_init(&wbar[i], 1);
        fence_mbar_init();
    }
    __syncwarp();
    const long long srow0 = L.gen_row0 + (long long)src * L.Cmax, drow0 = L.gen_row0 + (long long)dst * L.Cmax;
    int32_t* dpos = L.pos + (size_t)dst * L.Cmax;
    // chunk w + k * kEvWarps of the CTA's rows goes to buffer k % NB of warp w
    const int nch = (s1 - s0 + R - 1) / R;
    auto issue_load = [&](int k) {
        const int a = s0 + (warp + k * kEvWarps) * R, n = min(R, s1 - a);
        uint8_t* buf = wbuf + (k % NB) * kBufBytes;
        mbar_arrive_expect_tx(&wbar[k % NB], 2u * (uint32_t)n * kRowBytes);
        bulk_load(buf, L.kpool + (srow0 + a) * kHeadDim, (uint32_t)n * kRowBytes, &wbar[k % NB]);
        bulk_load(buf + R * kRowBytes, L.vpool + (srow0 + a) * kHeadDim, (uint32_t)n * kRowBytes, &wbar[k % NB]);
    };
    const int mine = nch > warp ? (nch - warp + kEvWarps - 1) / kEvWarps : 0;  // this warp's chunks
    int issued = min(NB, mine);
    if (lane == 0)
        for (int k = 0; k < issued; ++k) issue_load(k);

    // 2. the selection
    bool done = false;  // S.evlist holds the evicted set
    if (plan) {  // computed ahead: check that it is an ascending list of m candidates
        if (tid == 0) S.bcnt = 0;
        const int n = plan_n;
        if (n == m) {
            if (tid < m) S.evlist[tid] = plan_v0;
            if (tid + kEvThreads < m) S.evlist[tid + kEvThreads] = plan_v1;
        }
        __syncthreads();
        bool bad = n != m;
        for (int i = tid; i < m && !bad; i += kEvThreads)
            bad = S.evlist[i] < 0 || S.evlist[i] >= N || (i + 1 < m && S.evlist[i] >= S.evlist[i + 1]);
        if (bad) S.bcnt = 1;
        __syncthreads();
        if (tid == 0) S.nev = S.bcnt ? 0u : (uint32_t)m;  // a bad plan fails the check below
        done = true;
    }
    if (!done && cut) {
        cluster_sync();  // every CTA's list is complete
        const int total = gather_lists(S, CL, tid);
        __syncthreads();
        if (total >= m && total <= kEvCap) {  // the top m of the list are the evicted set
            if (tid == 0) S.nev = 0;
            __syncthreads();
            for (int e = warp; e < total; e += kEvWarps) {  // rank among the listed pairs, a warp per pair
                const uint2 x = S.ball[e];
                int above = 0;
                for (int f = lane; f < total; f += 32) {
                    const uint2 y = S.ball[f];
                    above += (y.x > x.x || (y.x == x.x && y.y > x.y)) ? 1 : 0;
                }
                above = __reduce_add_sync(0xffffffffu, above);
                if (lane == 0 && above < m) S.evown[atomicAdd(&S.nev, 1u)] = (int32_t)(x.y & 0xFFFFu);  // evicted
            }
            __syncthreads();
            for (int e = warp; e < m; e += kEvWarps) {  // position among the m evicted, by ordinal
                const int je = S.evown[e];
                int below = 0;
                for (int f = lane; f < m; f += 32) below += S.evown[f] < je ? 1 : 0;
                below = __reduce_add_sync(0xffffffffu, below);
                if (lane == 0) S.evlist[below] = je;
            }
            done = true;
        }
        // (otherwise: the radix passes below, from the first digit's histogram)
        if (!done) {
            for (int i = tid; i < nloc; i += kEvThreads) atomicAdd(&S.hist[0][S.keys[i] >> 24], 1u);
        }
    }
    if (!done) {
        uint32_t prefix = 0, mask = 0, need = (uint32_t)m;  // evicted still to find at or below the prefix
        uint32_t T = 0xFFFFFFFFu;
        int jT = INT_MAX;
        int hb = 0;
        for (int d = 0; d < 4; ++d) {
            const int shift = 24 - 8 * d;
            cluster_sync();  // every CTA's S.hist[hb] is complete (and, after the cut, no list is read any more)
            uint32_t v[kEvMaxCluster];  // bin tid of every CTA's histogram, all loads in flight at once
#pragma unroll
            for (int k = 0; k < kEvMaxCluster; ++k) v[k] = k < CL ? ld_dsmem_u32(dsmem_addr(&S.hist[hb][tid], k)) : 0u;
            {
                uint32_t sum = 0;
#pragma unroll
                for (int k = 0; k < kEvMaxCluster; ++k) sum += v[k];
                S.tot[tid] = sum;
            }
            __syncthreads();
            if (warp == 0) {  // the bin of the need-th largest, scanning from the top
                uint32_t loc[8], sum = 0;
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                    loc[q] = S.tot[255 - (8 * lane + q)];
                    sum += loc[q];
                }
                uint32_t incl = sum;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const uint32_t x = __shfl_up_sync(0xffffffffu, incl, o);
                    if (lane >= o) incl += x;
                }
                const uint32_t excl = incl - sum;
                if (excl < need && need <= incl) {
                    uint32_t cum = excl;
#pragma unroll
                    for (int q = 0; q < 8; ++q) {
                        if (need <= cum + loc[q]) {
                            S.sel[0] = 255u - (uint32_t)(8 * lane + q);
                            S.sel[1] = cum;
                            S.sel[2] = loc[q];
                            break;
                        }
                        cum += loc[q];
                    }
                }
            }
            __syncthreads();
            const uint32_t B = S.sel[0], cnt = S.sel[2];
            need -= S.sel[1];
            prefix |= B << shift;
            mask |= 0xFFu << shift;
            if (cnt <= (uint32_t)kEvCap) {  // gather the boundary candidates and rank them exactly
                if (tid == 0) S.bcnt = 0;
                __syncthreads();
                for (int i = tid; i < nloc; i += kEvThreads) {
                    const uint32_t key = S.keys[i];
                    if ((key & mask) == prefix) S.blist[atomicAdd(&S.bcnt, 1u)] = make_uint2(key, (uint32_t)(j0 + i));
                }
                cluster_sync();
                const int total = gather_lists(S, CL, tid);
                __syncthreads();
                for (int e = warp; e < total; e += kEvWarps) {  // a warp per pair
                    const uint2 x = S.ball[e];
                    uint32_t above = 0;
                    for (int f = lane; f < total; f += 32) {
                        const uint2 y = S.ball[f];
                        above += (y.x > x.x || (y.x == x.x && y.y > x.y)) ? 1u : 0u;
                    }
                    above = __reduce_add_sync(0xffffffffu, above);
                    if (lane == 0 && above == need - 1) {  // the smallest evicted pair
                        S.sel[3] = x.x;
                        S.sel[4] = x.y & 0xFFFFu;
                    }
                }
                __syncthreads();
                T = S.sel[3];
                jT = (int)S.sel[4];
                break;
            }
            if (d == 3) {  // more than kEvCap candidates share all 32 bits: the largest ordinals go first
                if (tid == (int)B) {  // this thread read bin B of every CTA: their tie counts
                    uint32_t after = 0;
#pragma unroll
                    for (int k = kEvMaxCluster - 1; k >= 0; --k) {
                        if (k >= CL) continue;
                        const uint32_t e = need > after ? min(need - after, v[k]) : 0u;  // ties CTA k evicts
                        if (k == (int)rank) {
                            S.sel[3] = v[k] - e;  // local index of the first evicted tie
                            S.sel[4] = e;
                        }
                        after += v[k];
                    }
                }
                __syncthreads();
                T = prefix;
                if (S.sel[4] > 0 && warp == 0) {  // ordinal of local tie number S.sel[3]
                    uint32_t seen = 0;
                    const uint32_t want = S.sel[3];
                    for (int i0 = 0; i0 < nloc; i0 += 32) {
                        const int i = i0 + lane;
                        const uint32_t eq = __ballot_sync(0xffffffffu, i < nloc && S.keys[i] == T);
                        if (seen + __popc(eq) > want) {
                            uint32_t e = eq;
                            for (uint32_t q = seen; q < want; ++q) e &= e - 1u;
                            if (lane == 0) S.sel[5] = (uint32_t)(j0 + i0 + __ffs(e) - 1);
                            break;
                        }
                        seen += __popc(eq);
                    }
                }
                __syncthreads();
                jT = S.sel[4] > 0 ? (int)S.sel[5] : INT_MAX;
                break;
            }
            hb ^= 1;  // this buffer was last read by the other CTAs before the barrier above
            S.hist[hb][tid] = 0;
            __syncthreads();
            for (int i = tid; i < nloc; i += kEvThreads) {
                const uint32_t key = S.keys[i];
                if ((key & mask) == prefix) atomicAdd(&S.hist[hb][(key >> (shift - 8)) & 255u], 1u);
            }
        }
        // own evicted ordinals, ascending (ballot compaction), then every CTA's, in rank order
        // (into lists of their own: other CTAs may still be reading the boundary lists)
        if (warp == 0) {
            uint32_t off = 0;
            for (int i0 = 0; i0 < nloc; i0 += 32) {
                const int i = i0 + lane;
                const uint32_t key = i < nloc ? S.keys[i] : 0u;
                const bool ev = i < nloc && (key > T || (key == T && j0 + i >= jT));
                const uint32_t bits = __ballot_sync(0xffffffffu, ev);
                const uint32_t at = off + __popc(bits & ((1u << lane) - 1u));
                if (ev && at < (uint32_t)kEvCap) S.evown[at] = j0 + i;
                off += __popc(bits);
            }
            if (lane == 0) S.evown_n = off;
        }
        cluster_sync();  // every CTA's evicted list is complete
        if (tid < CL) S.cnt[tid] = ld_dsmem_u32(dsmem_addr(&S.evown_n, tid));
        __syncthreads();
        int total = 0;
        for (int k = 0; k < CL; ++k) total += (int)S.cnt[k];
        if (total <= kEvCap) {
            for (int e = tid; e < total; e += kEvThreads) {
                int k = 0, off = 0;
                while (e >= off + (int)S.cnt[k]) off += (int)S.cnt[k++];
                S.evlist[e] = (int32_t)ld_dsmem_u32(dsmem_addr(&S.evown[e - off], k));
            }
        }
        if (tid == 0) S.nev = (uint32_t)total;  // (a total other than m fails the check below)
    }
    cluster_arrive();  // the last read of another CTA's shared memory; waited for before exit
    __syncthreads();
    const int nev = (int)S.nev;
    const bool ok = nev == m;  // the same in every CTA of the launch

    if (p.early) pdl_wait();
    pdl_launch_dependents();
    if (tid == 0 && rank == 0 && rep == 0) {
        int32_t* reg = L.region + ((size_t)p.layer * L.B + b) * L.KVH + h;
        int32_t* spr = L.spare + b * L.KVH + h;
        if (ok && *reg == src && *spr == dst) {
            *reg = dst;
            *spr = src;
        } else {
            atomicExch(L.err, kDeviceErrPlan);
        }
    }
    // 3. the survivors' rows, chunk by chunk as their copies land; a buffer is refilled one chunk
    //    later, once its stores have read it
    for (int k = 0; k < issued; ++k) {
        const int a = s0 + (warp + k * kEvWarps) * R, n = min(R, s1 - a);
        const uint8_t* buf = wbuf + (k % NB) * kBufBytes;
        // lane 0 alone reads the buffer (its bulk stores), so lane 0 alone waits; the verdict is the warp's
        bool landed = true;
        if (lane == 0) landed = mbar_wait_bounded(&wbar[k % NB], (uint32_t)((k / NB) & 1), kEvWaitLimitNs);
        if (!__shfl_sync(0xffffffffu, (int)landed, 0)) {
            if (lane == 0) {
                atomicExch(L.err, kDeviceErrTimeout);
                for (int q = k + 1; q < issued; ++q)  // let the copies already issued land (bounded)
                    (void)mbar_wait_bounded(&wbar[q % NB], (uint32_t)((q / NB) & 1), kEvWaitLimitNs);
            }
            break;
        }
        if (ok) {
            if (lane < n) {
                const int j = a + lane, e = ev_below(S, nev, j);
                if (e == nev || S.evlist[e] != j) dpos[j - e] = spos[j];
            }
            if (lane == 0) {
                int e = ev_below(S, nev, a);  // evicted ordinals below the run start
                for (int q = a; q < a + n;) {
                    const int nx = e < nev ? S.evlist[e] : INT_MAX;
                    const int v = min(a + n, nx);
                    if (v > q) {
                        const long long drow = drow0 + (q - e);
                        bulk_store(L.kpool + drow * kHeadDim, buf + (q - a) * kRowBytes, (uint32_t)(v - q) * kRowBytes);
                        bulk_store(L.vpool + drow * kHeadDim, buf + (R + q - a) * kRowBytes, (uint32_t)(v - q) * kRowBytes);
                    }
                    if (nx < a + n) {  // skip the evicted row
                        q = nx + 1;
                        ++e;
                    } else {
                        q = v;
                    }
                }
                bulk_commit();
                if (k >= 1 && issued < mine) {  // chunk issued = k + NB - 1 into the buffer of chunk k - 1
                    asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
                    issue_load(issued);
                }
            }
            if (k >= 1 && issued < mine) ++issued;  // warp-uniform
        }
        __syncwarp();
    }
    if (lane == 0) bulk_wait_all();
    cluster_wait();
}

// ----------------------------------------------------------------------------- plan (evicted sets ahead)
// The random draw reads no cache data: a candidate's key depends only on (ordinal, step, layer,
// head), so the evicted set of a firing step is known as soon as the counters are.  (Keys that
// follow positions -- order-free slots, block draws -- read the candidates' positions, which no
// kernel of the step before rewrites for a sequence that fires only at the next one.)  plan_kernel
// computes it ahead, beside the attention of the step before: one warp per CTA and about one CTA
// per SM, each looping over (layer, sequence, KV head) items, so that it takes a sliver of each
// SM's issue slots (7 KB of shared memory: it fits beside an attention CTA).  Per item, the
// same exact rules as evict_kernel: the sampled cut and an exact ranking of the listed pairs, or
// -- when fewer than m pass, for recency keys, or with RA_EVICT_EXACT -- four radix passes over
// recomputed keys (none is stored) and one ascending sweep that writes the evicted ordinals in
// order, ties at the threshold evicted from the largest ordinal down.  Output per item:
// [m][ordinals ascending] (-1 if the item is out of range).
struct PlanShared {
    uint2 list[kEvCap];
    int32_t ev[kEvCap];
    uint32_t hist[256];
    uint32_t cnt, nev;
};

// The key of candidate j, by the rules of select_kernel: per ordinal, or per position (pos: the
// head's positions) for order-free slots and block draws.
__device__ __forceinline__ uint32_t plan_key(const EvictParams& p, int layer, uint32_t id, int N, int g, int j,
                                             const int32_t* pos)
{
    const uint32_t k0 = (uint32_t)p.lay.seed, k1 = (uint32_t)(p.lay.seed >> 32);
    if (p.policy == RA_POLICY_BLOCK)
        return philox4x32_10_w0((uint32_t)(__ldcg(pos + j) / p.block), (uint32_t)g, (uint32_t)layer, id, k0, k1);
    if (p.holefill) {
        const uint32_t pj = (uint32_t)__ldcg(pos + j);
        return p.policy == RA_POLICY_RECENCY ? 0xFFFFFFFFu - pj : philox4x32_10_w0(pj, (uint32_t)g, (uint32_t)layer, id, k0, k1);
    }
    if (p.policy == RA_POLICY_RECENCY) return (uint32_t)(N - 1 - j);
    return philox4x32_10_w0((uint32_t)j, (uint32_t)g, (uint32_t)layer, id, k0, k1);
}

__global__ void __launch_bounds__(32) plan_kernel(const __grid_constant__ EvictParams p)
{
    __shared__ PlanShared S;
    const DevLayout& L = p.lay;
    const int lane = threadIdx.x;
    const int items = L.L * p.n_trig * L.KVH;
    for (int item = blockIdx.x; item < items; item += gridDim.x) {
        const int h = item % L.KVH, t = (item / L.KVH) % p.n_trig, layer = item / (L.KVH * p.n_trig);
        const int b = p.trig[t], N = p.trig_n[t], g = p.trig_g[t];
        const int m = N - L.K;
        int32_t* out =
            L.evplan + (size_t)((((size_t)p.ev_plan_parity * L.L + layer) * L.B + b) * L.KVH + h) * (L.r + 1);
        if (m < 1 || m > L.r || m > kEvCap || N > kMaxCandidates) {  // the host rules this out; the copy rejects it
            if (lane == 0) out[0] = -1;
            continue;
        }
        const uint32_t id = key_stream(p.trig_admit[t],
                                       p.policy == RA_POLICY_SHARED ? (uint32_t)(b * L.KVH) : (uint32_t)(b * L.KVH + h));
        const int32_t* pos = L.pos + (size_t)L.region[((size_t)layer * L.B + b) * L.KVH + h] * L.Cmax;
        const bool cut = (p.policy == RA_POLICY_RANDOM || p.policy == RA_POLICY_SHARED) && !p.ev_exact;
        bool done = false;
        if (cut) {
            const uint64_t E = 2ull * (uint64_t)m + 32ull;
            const uint32_t tau = E >= (uint64_t)N ? 0u : (uint32_t)(((uint64_t)(N - E) << 32) / (uint64_t)N);
            uint32_t cnt = 0;  // warp-uniform
            // independent Philox chains (and position loads) in flight per lane: 4 measured faster than 8
            constexpr int kChains = 4;
            // (warp-uniform trip count: every lane reaches each ballot, also when N < 32)
            for (int c0 = 0; c0 < N; c0 += kChains * 32) {
                uint32_t kq[kChains];
#pragma unroll
                for (int q = 0; q < kChains; ++q)
                    kq[q] = plan_key(p, layer, id, N, g, min(c0 + q * 32 + lane, N - 1), pos);
#pragma unroll
                for (int q = 0; q < kChains; ++q) {
                    const int j = c0 + q * 32 + lane;
                    const bool pass = j < N && kq[q] >= tau;
                    const uint32_t bits = __ballot_sync(0xffffffffu, pass);
                    const uint32_t at = cnt + __popc(bits & ((1u << lane) - 1u));
                    if (pass && at < (uint32_t)kEvCap) S.list[at] = make_uint2(kq[q], (uint32_t)j);
                    cnt += __popc(bits);
                }
            }
            __syncwarp();
            const int total = (int)cnt;
            if (total >= m && total <= kEvCap) {  // the top m of the list are the evicted set
                uint32_t nev = 0;
                for (int e0 = 0; e0 < total; e0 += 32) {
                    const int e = e0 + lane;
                    bool ev = false;
                    if (e < total) {
                        const uint2 x = S.list[e];
                        int above = 0;
#pragma unroll 8
                        for (int f = 0; f < total; ++f) {
                            const uint2 y = S.list[f];
                            above += (y.x > x.x || (y.x == x.x && y.y > x.y)) ? 1 : 0;
                        }
                        ev = above < m;
                    }
                    const uint32_t bits = __ballot_sync(0xffffffffu, ev);
                    if (ev) S.ev[nev + __popc(bits & ((1u << lane) - 1u))] = (int32_t)S.list[e].y;
                    nev += __popc(bits);
                }
                __syncwarp();
                for (int e = lane; e < m; e += 32) {  // ascending by ordinal
                    const int je = S.ev[e];
                    int below = 0;
#pragma unroll 8
                    for (int f = 0; f < m; ++f) below += S.ev[f] < je ? 1 : 0;
                    out[1 + below] = je;
                }
                if (lane == 0) out[0] = m;
                done = true;
            }
            __syncwarp();  // S.list and S.ev are rewritten by the next item
        }
        if (done) continue;
        // exact radix passes over recomputed keys: the need-th largest key T after four digits
        uint32_t prefix = 0, mask = 0, need = (uint32_t)m, ties = 0;
        for (int d = 0; d < 4; ++d) {
            const int shift = 24 - 8 * d;
            for (int i = lane; i < 256; i += 32) S.hist[i] = 0;
            __syncwarp();
            for (int j = lane; j < N; j += 32) {
                const uint32_t key = plan_key(p, layer, id, N, g, j, pos);
                if ((key & mask) == prefix) atomicAdd(&S.hist[(key >> shift) & 255u], 1u);
            }
            __syncwarp();
            uint32_t loc[8], sum = 0;
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                loc[q] = S.hist[255 - (8 * lane + q)];
                sum += loc[q];
            }
            uint32_t incl = sum;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const uint32_t x = __shfl_up_sync(0xffffffffu, incl, o);
                if (lane >= o) incl += x;
            }
            const uint32_t excl = incl - sum;
            uint32_t bin = 0, above = 0, cnt = 0;
            const bool mine = excl < need && need <= incl;
            if (mine) {
                uint32_t cum = excl;
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                    if (need <= cum + loc[q]) {
                        bin = 255u - (uint32_t)(8 * lane + q);
                        above = cum;
                        cnt = loc[q];
                        break;
                    }
                    cum += loc[q];
                }
            }
            const int src = __ffs(__ballot_sync(0xffffffffu, mine)) - 1;
            bin = __shfl_sync(0xffffffffu, bin, src);
            above = __shfl_sync(0xffffffffu, above, src);
            ties = __shfl_sync(0xffffffffu, cnt, src);
            need -= above;
            prefix |= bin << shift;
            mask |= 0xFFu << shift;
            __syncwarp();  // S.hist is rewritten by the next pass
        }
        // evicted: key > T, and among the `ties` keys equal to T the `need` largest ordinals;
        // an ascending sweep writes them in order
        const uint32_t T = prefix, tie_from = ties - need;
        uint32_t base_ev = 0, base_tie = 0;
        for (int c0 = 0; c0 < N; c0 += 32) {
            const int j = c0 + lane;
            const uint32_t key = j < N ? plan_key(p, layer, id, N, g, j, pos) : 0u;
            const bool eq = j < N && key == T, gt = j < N && key > T;
            const uint32_t eqb = __ballot_sync(0xffffffffu, eq);
            const bool ev = gt || (eq && base_tie + __popc(eqb & ((1u << lane) - 1u)) >= tie_from);
            const uint32_t evb = __ballot_sync(0xffffffffu, ev);
            const uint32_t pos = base_ev + __popc(evb & ((1u << lane) - 1u));
            if (ev && pos < (uint32_t)m) out[1 + pos] = j;
            base_ev += __popc(evb);
            base_tie += __popc(eqb);
        }
        if (lane == 0) out[0] = base_ev == (uint32_t)m ? m : -1;
    }
}

// ----------------------------------------------------------------------------- compact_stack (in place)
// At the start of a whole-stack step, every layer's round of the sequences that fire, in one
// launch, from evicted sets computed ahead (plan_kernel): one CTA per (layer, sequence, KV head)
// and array (K with the positions, or V) compacts the head's rows of that array in place.  A
// survivor moves down by the evicted ordinals below it (at most m <= r rows), so a CTA that copies
// its rows in ascending chunks never overwrites a row it has not read yet: every store of chunk i
// lands below chunk i + 1, and every later load reads at or above it (and the two arrays are
// separate, so their CTAs are independent).  Chunks of kStkRows rows stream through a ring of
// stages with TMA bulk copies; the survivors' runs go back with bulk stores, positions by plain
// stores.
constexpr int kStkThreads = 128;
constexpr int kStkRows = 128;   // rows per stage: 32 KB of K or V
constexpr int kStkStages = 3;   // 96 KB of stages: two CTAs per SM
constexpr size_t kStkSmem = (size_t)kStkStages * kStkRows * kRowBytes;
static_assert(kStkStages >= 2 && kStkRows <= kStkThreads, "refills trail by one chunk; a thread per row");
static_assert(((kStkRows + 4) * 4) % 16 == 0, "every stage's positions start 16-byte aligned");

struct StkShared {
    int32_t ev[kEvCap];                  // the evicted ordinals, ascending
    __align__(16) int32_t pos[kStkStages][kStkRows + 4];  // (bulk copy destinations: 16-byte aligned)
    uint64_t bar[kStkStages];
    int bad;
};

__global__ void __launch_bounds__(kStkThreads) compact_stack_kernel(const __grid_constant__ EvictParams p)
{
    extern __shared__ __align__(128) uint8_t stk_dyn[];  // [stage][rows of K or V]
    __shared__ __align__(16) StkShared S;
    constexpr int kStageBytes = kStkRows * kRowBytes;
    const DevLayout& L = p.lay;
    const int tid = threadIdx.x;
    const int item = blockIdx.x >> 1, part = blockIdx.x & 1;  // layer-major (layer, sequence, KV head); 0: K, 1: V
    uint16_t* pool = part ? L.vpool : L.kpool;
    const int h = item % L.KVH, t = (item / L.KVH) % p.n_trig, layer = item / (L.KVH * p.n_trig);
    const int b = p.trig[t], c = p.trig_c[t], N = p.trig_n[t];
    const int m = N - L.K;
    pdl_wait();  // the rows were written by the previous step's attention
    pdl_launch_dependents();
    if (m < 1 || m > L.r || m > kEvCap || N > c || c > L.Cmax) {  // the host rules this out
        if (tid == 0) atomicExch(L.err, kDeviceErrPlan);
        return;
    }
    const int reg = L.region[((size_t)layer * L.B + b) * L.KVH + h];
    const long long row0 = L.gen_row0 + (long long)reg * L.Cmax;
    int32_t* gpos = L.pos + (size_t)reg * L.Cmax;
    const int32_t* plan =
        L.evplan + (size_t)((((size_t)p.ev_plan_parity * L.L + layer) * L.B + b) * L.KVH + h) * (L.r + 1);
    const bool with_pos = part == 0;
    const bool pos_bulk = with_pos && (L.Cmax & 3) == 0;  // position chunks are 16-byte aligned
    const int nch = (c + kStkRows - 1) / kStkRows;
    auto issue = [&](int i) {  // chunk i into stage i % kStkStages (thread 0)
        const int s = i % kStkStages, a = i * kStkRows, n = min(kStkRows, c - a);
        uint8_t* st = stk_dyn + (size_t)s * kStageBytes;
        const uint32_t pbytes = pos_bulk ? (uint32_t)min((n + 3) & ~3, L.Cmax - a) * 4u : 0u;
        mbar_arrive_expect_tx(&S.bar[s], (uint32_t)n * kRowBytes + pbytes);
        bulk_load(st, pool + (row0 + a) * kHeadDim, (uint32_t)n * kRowBytes, &S.bar[s]);
        if (pbytes) bulk_load(S.pos[s], gpos + a, pbytes, &S.bar[s]);
    };
    int issued = 0;  // thread 0's count of chunks whose copies are issued
    if (tid == 0) {
        S.bad = 0;
        for (int s = 0; s < kStkStages; ++s) mbar_init(&S.bar[s], 1);
        fence_mbar_init();
        issued = min(kStkStages, nch);
        for (int i = 0; i < issued; ++i) issue(i);
    }
    // the plan: m ordinals, ascending, below N
    const int n_plan = __ldcg(plan);
    for (int i = tid; i < m; i += kStkThreads) S.ev[i] = __ldcg(plan + 1 + i);
    __syncthreads();
    bool bad = n_plan != m;
    for (int i = tid; i < m && !bad; i += kStkThreads)
        bad = S.ev[i] < 0 || S.ev[i] >= N || (i + 1 < m && S.ev[i] >= S.ev[i + 1]);
    if (bad) S.bad = 1;
    __syncthreads();
    if (S.bad) {  // a bad plan moves nothing: wait (bounded) for the copies issued, and leave
        if (tid == 0) {
            atomicExch(L.err, kDeviceErrPlan);
            for (int q = 0; q < issued; ++q)
                (void)mbar_wait_bounded(&S.bar[q % kStkStages], (uint32_t)((q / kStkStages) & 1), kEvWaitLimitNs);
        }
        return;
    }
    auto ev_below = [&](int j) {  // evicted ordinals below j
        int lo = 0, hi = m;
        while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (S.ev[mid] < j) lo = mid + 1; else hi = mid;
        }
        return lo;
    };
    for (int i = 0; i < nch; ++i) {  // every chunk's copies are issued by the time it is reached
        const int s = i % kStkStages, a = i * kStkRows, n = min(kStkRows, c - a);
        if (tid == 0 && !mbar_wait_bounded(&S.bar[s], (uint32_t)((i / kStkStages) & 1), kEvWaitLimitNs)) {
            atomicExch(L.err, kDeviceErrTimeout);
            for (int q = i + 1; q < issued; ++q)  // let the copies already issued land (bounded)
                (void)mbar_wait_bounded(&S.bar[q % kStkStages], (uint32_t)((q / kStkStages) & 1), kEvWaitLimitNs);
            S.bad = 2;
        }
        if (with_pos && !pos_bulk && tid < n) S.pos[s][tid] = __ldcg(gpos + a + tid);  // (all read before any is written)
        __syncthreads();
        if (S.bad) break;
        if (with_pos && tid < n) {  // positions of the chunk's survivors
            const int j = a + tid, e = ev_below(j);
            if (e == m || S.ev[e] != j) gpos[j - e] = S.pos[s][tid];
        }
        if (tid == 0) {  // the runs of survivors, each to its place below
            const uint8_t* st = stk_dyn + (size_t)s * kStageBytes;
            int e = ev_below(a);
            for (int q = a; q < a + n;) {
                const int nx = e < m ? S.ev[e] : INT_MAX;
                const int v = min(a + n, nx);
                if (v > q) {
                    const long long drow = row0 + (q - e);
                    bulk_store(pool + drow * kHeadDim, st + (q - a) * kRowBytes, (uint32_t)(v - q) * kRowBytes);
                }
                if (nx < a + n) {
                    q = nx + 1;
                    ++e;
                } else {
                    q = v;
                }
            }
            bulk_commit();
        }
        __syncthreads();  // the stage's positions are read
        if (tid == 0 && i >= 1 && issued < nch) {  // chunk i + 2 into chunk i - 1's stage once its stores read it
            asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
            issue(issued);
            ++issued;
        }
    }
    if (tid == 0) bulk_wait_all();
}

// ----------------------------------------------------------------------------- fill_stack (order-free, in place)
// The order-free counterpart of compact_stack_kernel: at the start of a whole-stack step, every
// layer's round of the sequences that fire, in one launch, from evicted sets computed ahead.  One
// CTA per (layer, sequence, KV head) moves rows as select_kernel does with the step's token
// pending: evicted slot e_i takes the row of slot c + 1 - m + i for i < m - 1, and the row of the
// new last slot c - m, unless e_{m-1} is that slot, fills e_{m-1}; each layer's attention then
// appends its token into the new last slot.  Slots c - m .. c - 1 are buffer slots, so no move
// reads a slot that another writes.
constexpr int kFillThreads = 256;

__global__ void __launch_bounds__(kFillThreads) fill_stack_kernel(const __grid_constant__ EvictParams p)
{
    __shared__ int32_t ev[kEvCap];
    __shared__ int bad;
    const DevLayout& L = p.lay;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int item = blockIdx.x;  // layer-major (layer, sequence, KV head)
    const int h = item % L.KVH, t = (item / L.KVH) % p.n_trig, layer = item / (L.KVH * p.n_trig);
    const int b = p.trig[t], c = p.trig_c[t], N = p.trig_n[t];
    const int m = N - L.K;
    // The plan (complete: the stream waited for it) and the tables are read before waiting for
    // the predecessor; the rows and positions it may have written, after.  Every exit waits
    // first, so that no successor starts before the predecessor completes.
    if (m < 1 || m > L.r || m > kEvCap || N > c || c + 1 > L.Cmax) {  // the host rules this out
        pdl_wait();
        pdl_launch_dependents();
        if (tid == 0) atomicExch(L.err, kDeviceErrPlan);
        return;
    }
    const int32_t* plan =
        L.evplan + (size_t)((((size_t)p.ev_plan_parity * L.L + layer) * L.B + b) * L.KVH + h) * (L.r + 1);
    if (tid == 0) bad = __ldcg(plan) != m;
    for (int i = tid; i < m; i += kFillThreads) ev[i] = __ldcg(plan + 1 + i);
    const int reg = L.region[((size_t)layer * L.B + b) * L.KVH + h];
    __syncthreads();
    bool wrong = false;  // the plan: m ordinals, ascending, below N
    for (int i = tid; i < m; i += kFillThreads) wrong = wrong || ev[i] < 0 || ev[i] >= N || (i + 1 < m && ev[i] >= ev[i + 1]);
    if (wrong) bad = 1;
    __syncthreads();
    pdl_wait();  // the buffer rows were written by earlier steps' attention
    pdl_launch_dependents();
    if (bad) {  // a bad plan moves nothing
        if (tid == 0) atomicExch(L.err, kDeviceErrPlan);
        return;
    }
    const long long row0 = L.gen_row0 + (long long)reg * L.Cmax;
    int32_t* gpos = L.pos + (size_t)reg * L.Cmax;
    const int top = c + 1, last = c - m, part = lane & 15;
    uint16_t* pool = lane < 16 ? L.kpool : L.vpool;  // lanes 0-15 move K, 16-31 V, 16 bytes each
    constexpr int kWarps = kFillThreads / 32, kBatch = 8;  // rows a warp has in flight
    // moves i < m - 1: slot top - m + i to e_i; move m - 1: the new last slot to e_{m-1}, if they differ
    for (int i0 = warp; i0 < m; i0 += kWarps * kBatch) {
        uint4 v[kBatch];
        int32_t pv[kBatch];
        int to[kBatch];
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {  // every load of the batch first ...
            const int i = i0 + u * kWarps;
            to[u] = -1;
            if (i < m && (i < m - 1 || ev[i] != last)) {
                const int from = i < m - 1 ? top - m + i : last;
                to[u] = ev[i];
                v[u] = reinterpret_cast<const uint4*>(pool + (row0 + from) * kHeadDim)[part];
                pv[u] = gpos[from];
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
    const int b = p.only_seq >= 0 ? p.only_seq : (int)blockIdx.x / L.KVH, h = blockIdx.x % L.KVH;
    const int n = p.n_rows[b];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    long long row0 = 0;
    int32_t* dpos = nullptr;
    const int32_t* ptab = L.pages + (size_t)b * L.max_pages;
    if (restore) {
        const int reg = L.region[((size_t)p.layer * L.B + b) * L.KVH + h];
        row0 = L.gen_row0 + (long long)reg * L.Cmax;
        dpos = L.pos + (size_t)reg * L.Cmax;
    }
    const size_t src0 = ((p.only_seq >= 0 ? 0 : (size_t)b * L.KVH) + h) * (size_t)p.row_stride;
    const uint16_t* sb = (lane < 16 ? p.k : p.v);
    uint16_t* db = (lane < 16 ? L.kpool : L.vpool);
    for (int i = warp; i < n; i += 8) {
        const uint4 v = reinterpret_cast<const uint4*>(sb + (src0 + i) * kHeadDim)[lane & 15];
        const long long row = restore ? row0 + i : prompt_row(L, p.layer, ptab[i / kPromptPage], h, i);
        reinterpret_cast<uint4*>(db + row * kHeadDim)[lane & 15] = v;
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

namespace {
constexpr size_t kEvSmem = (size_t)kEvWarps * kEvBufs * 2 * kEvRows * kRowBytes;

cudaLaunchConfig_t evict_config(int cluster, int heads_reps, int n_trig, cudaStream_t s, cudaLaunchAttribute* attr)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)cluster, (unsigned)heads_reps, (unsigned)n_trig);
    cfg.blockDim = dim3(kEvThreads);
    cfg.dynamicSmemBytes = kEvSmem;
    cfg.stream = s;
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)cluster;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cfg;
}
}  // namespace

// One-time attributes, and how many clusters of each size 1..kEvMaxCluster the device runs at
// once (active[cl], 0 where that size cannot be scheduled).
cudaError_t evict_prepare(int* active)
{
    auto kernel = evict_kernel<kEvRows, kEvBufs>;
    cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kEvSmem);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
    bool any = false;
    active[0] = 0;
    for (int cl = 1; cl <= kEvMaxCluster; ++cl) {
        cudaLaunchAttribute attr[2];
        cudaLaunchConfig_t cfg = evict_config(cl, 1, 1, 0, attr);
        cfg.numAttrs = 1;  // the cluster shape only
        int n = 0;
        if (cudaOccupancyMaxActiveClusters(&n, kernel, &cfg) != cudaSuccess) {
            (void)cudaGetLastError();
            n = 0;
        }
        active[cl] = n;
        any = any || n > 0;
    }
    return any ? cudaSuccess : cudaErrorInvalidConfiguration;
}

cudaError_t launch_evict(const EvictParams& p, int cluster, cudaStream_t s)
{
    if (cluster < 1 || cluster > kEvMaxCluster) return cudaErrorInvalidValue;
    cudaLaunchAttribute attr[2];
    cudaLaunchConfig_t cfg = evict_config(cluster, p.lay.KVH * p.ev_reps, p.n_trig, s, attr);
    return cudaLaunchKernelEx(&cfg, evict_kernel<kEvRows, kEvBufs>, p);
}

cudaError_t launch_plan(const EvictParams& p, int sms, cudaStream_t s)
{
    const int items = p.lay.L * p.n_trig * p.lay.KVH;
    plan_kernel<<<(unsigned)std::min(items, std::max(sms, 1)), 32, 0, s>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_compact_stack(const EvictParams& p, int layers, cudaStream_t s)
{
    static bool configured = false;
    if (!configured) {
        cudaError_t e = cudaFuncSetAttribute(compact_stack_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kStkSmem);
        if (e != cudaSuccess) return e;
        configured = true;
    }
    return launch_pdl(compact_stack_kernel, dim3((unsigned)(2 * layers * p.n_trig * p.lay.KVH)), dim3(kStkThreads),
                      kStkSmem, s, p);
}

cudaError_t launch_fill_stack(const EvictParams& p, int layers, cudaStream_t s)
{
    return launch_pdl(fill_stack_kernel, dim3((unsigned)(layers * p.n_trig * p.lay.KVH)), dim3(kFillThreads), 0, s, p);
}

cudaError_t launch_timeout_probe(int32_t* err, uint64_t limit_ns, cudaStream_t s)
{
    timeout_probe_kernel<<<1, 32, 0, s>>>(err, limit_ns);
    return cudaGetLastError();
}

cudaError_t launch_prefill(const CopyRowsParams& p, cudaStream_t s)
{
    copy_rows_kernel<<<(p.only_seq >= 0 ? 1 : p.lay.B) * p.lay.KVH, 256, 0, s>>>(p, 0);
    return cudaGetLastError();
}

cudaError_t launch_restore(const CopyRowsParams& p, cudaStream_t s)
{
    copy_rows_kernel<<<p.lay.B * p.lay.KVH, 256, 0, s>>>(p, 1);
    return cudaGetLastError();
}

}  // namespace ra
