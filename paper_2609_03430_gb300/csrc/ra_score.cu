// ra_score.cu -- window attention of the scored comparator on sm_103a.
//
// The comparator ranks a head's eviction candidates by the SnapKV score of
// section 2 ("Baselines as choices of s"): the attention that the window of
// the last r decode queries gives each candidate, summed over the window and
// over the G query heads of the KV group (max-pooling and top-K happen in the
// select kernel).  A window query attends, as at its own decode step, to the
// keys at positions up to its own: the prompt, every candidate, and the first
// u buffer rows, u = its rank in the window.
//
// Between two eviction rounds the cache only grows, so each window query saw
// at its own step exactly the keys it sees now, and the decode attention
// kernel records its softmax normaliser beside it.  The eviction therefore
// needs one pass over the candidate rows only:
//   summation pass (score_kernel<2, MT>)  per triggered (sequence, KV head),
//       the logits of the M = r * G window rows against the candidate tiles,
//       normalised by the recorded normalisers and summed over all M rows:
//       one fp32 score per candidate.  Each CTA holds all M rows, so every
//       column sum is complete inside it -- no atomics, and the result does
//       not depend on the launch shape.
//   restore pass (score_kernel<1, MT> + score_merge_kernel)  only when a
//       window is loaded from outside (ra_restore_queries): the normalisers,
//       recomputed over the prompt and the cached rows each query sees (by
//       position), split over chunks of key tiles and merged.
// The contraction of the window rows with the key rows is a dense GEMM
// (M x keys x 128), so it runs on the tensor cores (mma.sync m16n8k16, bf16
// in, fp32 accumulate).  CTA layout: 8 warps; warp w owns the 16-row M tiles
// w, w + 8, ... (MT of them).  The M rows arrive by 2-D TMA (64-row x
// 64-channel boxes, 128-byte swizzle) with the first key tile and are read as
// A fragments with ldmatrix; key tiles of 64 rows x 128 channels arrive the
// same way into a two-stage ring on mbarriers and are read as B fragments.  Logits are in base 2 with the scale folded in.
#include <cuda.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "ra_internal.h"
#include "ra_ptx.cuh"

namespace ra {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kStages = 2;
constexpr int kHalfBytes = kScoreTile * 128;      // one 64-channel box of a key tile
constexpr int kTileBytes = 2 * kHalfBytes;        // a key tile: 64 rows x 256 bytes
constexpr uint64_t kWaitLimitNs = 2000000000ull;  // bounded mbarrier waits: 2 s
static_assert(kScoreTile == 64, "eight 8-column MMA tiles per key tile");
static_assert(kHalfBytes % 1024 == 0, "128-byte-swizzled TMA boxes start 1024-byte aligned");

template <int MT>
struct SCfg {
    static constexpr int ROWS = 16 * kWarps * MT;                 // window rows held (M padded)
    static constexpr int Q_HALF = ROWS * 128;                     // one 64-channel half of the window
    static constexpr int Q_OFF = kStages * kTileBytes;            // after the key stages
    static constexpr int STAT_OFF = Q_OFF + ROWS * kRowBytes;     // pass 2: row max and 1/sum
    static constexpr int RED_OFF = STAT_OFF + 2 * ROWS * 4;       // pass 2: column sums per warp
    static constexpr int BAR_OFF = RED_OFF + kWarps * kScoreTile * 4;
    static constexpr size_t SMEM = 1024 + (size_t)BAR_OFF + kStages * 8;
    static_assert(ROWS <= kScoreMaxRows || MT == 1, "window rows");
    static_assert(ROWS % kScoreTile == 0 && Q_HALF % 1024 == 0, "whole TMA boxes, 1024-byte aligned");
    static_assert(SMEM <= 232448, "fits the 227 KB opt-in shared memory");
};

// Byte offset of (window row R, 16-byte chunk c) of the window block: two 64-channel halves of
// `half` bytes each, rows of 128 bytes, chunks xored with R mod 8 (the TMA 128-byte swizzle).
__device__ __forceinline__ uint32_t qswz(int R, int c, int half)
{
    return (uint32_t)((c >> 3) * half + R * 128 + (((c & 7) ^ (R & 7)) << 4));
}

// Byte offset of (key row j, 16-byte chunk c) inside a 128-byte-swizzled key tile.
__device__ __forceinline__ uint32_t kswz(int j, int c)
{
    return (uint32_t)((c >> 3) * kHalfBytes + j * 128 + (((c & 7) ^ (j & 7)) << 4));
}

__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], uint32_t addr)
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}

// D[16x8] += A[16x16] B[16x8], bf16 in, fp32 accumulate.
__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1)
{
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Tiles of one head: restore pass -- its prompt rows, then its c cached generated rows;
// summation pass -- its N candidate rows.
__device__ __forceinline__ int head_tiles(int pass, int lp, int n_gen, int* tp)
{
    *tp = pass == 1 ? (lp + kScoreTile - 1) / kScoreTile : 0;
    return *tp + (n_gen + kScoreTile - 1) / kScoreTile;
}

// Restore pass: the decode step whose query sits in window slot `slot` when g tokens have been
// generated (the r latest steps fill the r slots), and how many of the head's c cached generated
// rows (positions pos[0..c), increasing) that query sees: those at positions up to its own.
__device__ __forceinline__ int visible_rows(const int32_t* pos, int c, int lp, int g, int r, int slot)
{
    const int d = ((g - 1 - slot) % r + r) % r;
    const int step = g - d;
    if (step < 1) return 0;  // no such step yet: the slot is never read before a real query fills it
    const int qpos = lp + step - 1;
    int lo = 0, hi = c;      // first ordinal whose position is after qpos
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (__ldcg(pos + mid) <= qpos) lo = mid + 1; else hi = mid;
    }
    return lo;
}

// PASS 1 (restore): per window row, (max, sum of exp2) over one chunk of the keys it sees.
// PASS 2 (eviction): per candidate, the sum over window rows of exp2(logit - log2 normaliser).
template <int PASS, int MT>
__global__ void __launch_bounds__(kThreads, MT <= 2 ? 2 : 1) score_kernel(const __grid_constant__ EvictParams p,
                                                                        const __grid_constant__ CUtensorMap tk,
                                                                        const __grid_constant__ CUtensorMap tw)
{
    using C = SCfg<MT>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::BAR_OFF);
    float* s_sl = reinterpret_cast<float*>(smem + C::STAT_OFF);  // pass 2: each row's scale * log2 e
    float* s_lse = s_sl + C::ROWS;                               // pass 2: each row's log2 normaliser
    float* red = reinterpret_cast<float*>(smem + C::RED_OFF);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    // The window, the cache and the tables come from earlier kernels.  With p.early (pass 2 inside
    // the fused step) they were all written by kernels that completed before the predecessor (the
    // previous layer's attention) started, and the scores are read only by the successor: the pass
    // computes before waiting, and lets its successor start only after the wait, at its end.
    if (!(PASS == 2 && p.early)) {
        pdl_wait();
        pdl_launch_dependents();
    }

    const DevLayout& L = p.lay;
    const int t = blockIdx.y / L.KVH, h = blockIdx.y - t * L.KVH;
    const int b = p.trig[t];
    const int N = p.trig_n[t], r = L.r, G = L.G, M = r * G;
    const int lp = L.seq_lp[b];
    int tp;
    const int nt_head = head_tiles(PASS, lp, N, &tp);
    const int ch = PASS == 1 ? p.ch1 : p.ch2;
    const int t0 = blockIdx.x * ch;
    if (t0 >= nt_head) return;  // (exiting counts as letting the successor start)
    const int ntile = min(ch, nt_head - t0);
    const long long prow = (long long)p.layer * L.prompt_rows_per_layer + L.seq_poff[b] + (long long)h * lp;
    const size_t lbh = ((size_t)p.layer * L.B + b) * L.KVH + h;
    const int reg = L.region[lbh];
    const long long grow = L.gen_row0 + (long long)reg * L.Cmax;
    const int hid = b * L.KVH + h;

    auto tile_row = [&](int k) -> long long {  // first cache row of the head's tile k
        return k < tp ? prow + (long long)k * kScoreTile : grow + (long long)(k - tp) * kScoreTile;
    };
    // thread 0: tile t0 + i into stage i % 2 (one arrival per phase: `extra` bytes of other copies
    // completing on the same barrier are expected together with the tile)
    auto issue = [&](int i, uint32_t extra) {
        const int s = i % kStages;
        uint8_t* st = smem + (size_t)s * kTileBytes;
        const int row = (int)tile_row(t0 + i);
        mbar_arrive_expect_tx(&bars[s], (uint32_t)kTileBytes + extra);
        tma_load_2d(st, &tk, 0, row, &bars[s]);
        tma_load_2d(st + kHalfBytes, &tk, 64, row, &bars[s]);
    };
    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) mbar_init(&bars[s], 1);
        fence_mbar_init();
        prefetch_tensormap(&tk);
        prefetch_tensormap(&tw);
        // The window rows (row R = slot * G + g) complete on stage 0's barrier with the first
        // key tile.  Rows past M belong to the next head's window (or lie past the end and
        // read as zero): finite, and given no weight.
        issue(0, (uint32_t)(C::ROWS * kRowBytes));
        const int row0 = (int)(lbh * (size_t)M);
        for (int rb = 0; rb < C::ROWS; rb += kScoreTile) {
            tma_load_2d(smem + C::Q_OFF + rb * 128, &tw, 0, row0 + rb, &bars[0]);
            tma_load_2d(smem + C::Q_OFF + C::Q_HALF + rb * 128, &tw, 64, row0 + rb, &bars[0]);
        }
        for (int i = 1; i < kStages && i < ntile; ++i) issue(i, 0u);
    }
    if (PASS == 2) {  // the normaliser each window query had at its decode step
        const float2* qst = L.qstats + lbh * (size_t)M;
        for (int R = tid; R < C::ROWS; R += kThreads) {
            const float2 f = R < M ? __ldcg(qst + R) : make_float2(0.f, INFINITY);  // padding rows weigh 0
            s_sl[R] = f.x;
            s_lse[R] = f.y;
        }
    }
    __syncthreads();

    // This lane's rows: R = 16 * (warp + 8 i) + (lane / 4) + 8 hf; its columns: 8 nt + 2 (lane % 4) + e.
    const int tq = lane & 3;
    const int mi = lane >> 3, ri = lane & 7;
    int lim[MT][2];  // pass 1: generated rows the row sees
    // pass 1: running max and (per-lane partial) sum of exp2; pass 2: the row's scale and normaliser
    float mrow[MT][2], lrow[MT][2];
#pragma unroll
    for (int i = 0; i < MT; ++i)
#pragma unroll
        for (int hf = 0; hf < 2; ++hf) {
            const int R = 16 * (warp + kWarps * i) + (lane >> 2) + 8 * hf;
            if (PASS == 1) {
                lim[i][hf] = R < M ? visible_rows(L.pos + (size_t)reg * L.Cmax, N, lp, p.trig_g[t], r, R / G) : 0;
                mrow[i][hf] = -INFINITY;
                lrow[i][hf] = 0.f;
            } else {
                lim[i][hf] = 0;
                mrow[i][hf] = s_sl[R];
                lrow[i][hf] = s_lse[R];
            }
        }
    const float sl = p.qk_scale_log2;  // pass 1: the scale the restored queries are taken at
    const uint32_t qs = smem_u32(smem + C::Q_OFF);
    float* scores = L.scores + lbh * L.Cmax;

    for (int i = 0; i < ntile; ++i) {
        const int s = i % kStages;
        const bool ok = mbar_wait_bounded(&bars[s], (uint32_t)((i / kStages) & 1), kWaitLimitNs);
        if (!__syncthreads_and(ok)) {  // give up together; let the copies in flight land first
            if (tid == 0) {
                atomicExch(L.err, kDeviceErrTimeout);
                for (int j = i + 1; j < ntile && j < i + kStages; ++j)
                    (void)mbar_wait_bounded(&bars[j % kStages], (uint32_t)((j / kStages) & 1), kWaitLimitNs);
            }
            if (PASS == 2 && p.early) pdl_wait();  // the successor still starts only after the predecessor
            return;
        }
        const uint32_t ks = smem_u32(smem + (size_t)s * kTileBytes);
        float acc[MT][8][4];
#pragma unroll
        for (int a = 0; a < MT; ++a)
#pragma unroll
            for (int n = 0; n < 8; ++n) acc[a][n][0] = acc[a][n][1] = acc[a][n][2] = acc[a][n][3] = 0.f;
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
            uint32_t af[MT][4];
#pragma unroll
            for (int a = 0; a < MT; ++a)
                ldsm_x4(af[a], qs + qswz(16 * (warp + kWarps * a) + (lane & 15), 2 * kk + (lane >> 4), C::Q_HALF));
#pragma unroll
            for (int np = 0; np < 4; ++np) {
                uint32_t bf[4];
                ldsm_x4(bf, ks + kswz(16 * np + (mi >> 1) * 8 + ri, 2 * kk + (mi & 1)));
#pragma unroll
                for (int a = 0; a < MT; ++a) {
                    mma16816(acc[a][2 * np], af[a], bf[0], bf[1]);
                    mma16816(acc[a][2 * np + 1], af[a], bf[2], bf[3]);
                }
            }
        }
        const int k = t0 + i;
        if (PASS == 1) {
            const bool prompt = k < tp;
            const int base = (prompt ? k : k - tp) * kScoreTile;  // index of column 0 within its segment
#pragma unroll
            for (int a = 0; a < MT; ++a)
#pragma unroll
                for (int hf = 0; hf < 2; ++hf) {
                    const int nvalid = (prompt ? lp : lim[a][hf]) - base;  // columns this row sees
                    float bm = -INFINITY;
#pragma unroll
                    for (int n = 0; n < 8; ++n)
#pragma unroll
                        for (int e = 0; e < 2; ++e) {
                            const int col = 8 * n + 2 * tq + e;
                            const float v = col < nvalid ? acc[a][n][2 * hf + e] * sl : -INFINITY;
                            acc[a][n][2 * hf + e] = v;
                            bm = fmaxf(bm, v);
                        }
                    bm = fmaxf(bm, __shfl_xor_sync(0xffffffffu, bm, 1));
                    bm = fmaxf(bm, __shfl_xor_sync(0xffffffffu, bm, 2));
                    const float mn = fmaxf(mrow[a][hf], bm);
                    if (mn != -INFINITY) {
                        float sum = mrow[a][hf] == -INFINITY ? 0.f : lrow[a][hf] * exp2f(mrow[a][hf] - mn);
#pragma unroll
                        for (int n = 0; n < 8; ++n)
#pragma unroll
                            for (int e = 0; e < 2; ++e) sum += exp2f(acc[a][n][2 * hf + e] - mn);
                        lrow[a][hf] = sum;
                        mrow[a][hf] = mn;
                    }
                }
        } else {
            float cs[8][2];
#pragma unroll
            for (int n = 0; n < 8; ++n) cs[n][0] = cs[n][1] = 0.f;
#pragma unroll
            for (int a = 0; a < MT; ++a)
#pragma unroll
                for (int hf = 0; hf < 2; ++hf)
#pragma unroll
                    for (int n = 0; n < 8; ++n)
#pragma unroll
                        for (int e = 0; e < 2; ++e)
                            cs[n][e] += exp2f(fmaf(acc[a][n][2 * hf + e], mrow[a][hf], -lrow[a][hf]));
#pragma unroll
            for (int n = 0; n < 8; ++n)
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                    float v = cs[n][e];
                    v += __shfl_xor_sync(0xffffffffu, v, 4);
                    v += __shfl_xor_sync(0xffffffffu, v, 8);
                    v += __shfl_xor_sync(0xffffffffu, v, 16);
                    if (lane < 4) red[warp * kScoreTile + 8 * n + 2 * tq + e] = v;
                }
            __syncthreads();
            if (tid < kScoreTile) {
                float v = 0.f;
#pragma unroll
                for (int w = 0; w < kWarps; ++w) v += red[w * kScoreTile + tid];
                const int j = k * kScoreTile + tid;
                if (j < N) scores[j] = v;
            }
        }
        __syncthreads();  // stage s (and the column-sum buffer) free again
        if (tid == 0 && i + kStages < ntile) {
            fence_proxy_async_smem();
            issue(i + kStages, 0u);
        }
    }

    if (PASS == 2 && p.early) {
        pdl_wait();
        pdl_launch_dependents();
    }
    if (PASS == 1) {  // this chunk's statistics of every real row
        float* out = L.stats + ((size_t)hid * L.stats_chunks + blockIdx.x) * M * 2;
#pragma unroll
        for (int a = 0; a < MT; ++a)
#pragma unroll
            for (int hf = 0; hf < 2; ++hf) {
                float l = lrow[a][hf];
                l += __shfl_xor_sync(0xffffffffu, l, 1);
                l += __shfl_xor_sync(0xffffffffu, l, 2);
                const int R = 16 * (warp + kWarps * a) + (lane >> 2) + 8 * hf;
                if (tq == 0 && R < M) *reinterpret_cast<float2*>(out + (size_t)R * 2) = make_float2(mrow[a][hf], l);
            }
    }
}

// Restore pass, last step: merge each window row's chunk statistics into its normaliser.
__global__ void __launch_bounds__(256) score_merge_kernel(const __grid_constant__ EvictParams p)
{
    pdl_wait();
    pdl_launch_dependents();
    const DevLayout& L = p.lay;
    const int t = blockIdx.x / L.KVH, h = blockIdx.x - t * L.KVH;
    const int b = p.trig[t];
    const int M = L.r * L.G;
    int tp;
    const int nch = (head_tiles(1, L.seq_lp[b], p.trig_n[t], &tp) + p.ch1 - 1) / p.ch1;
    const float* st = L.stats + (size_t)(b * L.KVH + h) * L.stats_chunks * M * 2;
    float2* qst = L.qstats + (((size_t)p.layer * L.B + b) * L.KVH + h) * (size_t)M;
    for (int R = threadIdx.x; R < M; R += blockDim.x) {
        float mx = -INFINITY;
        for (int k = 0; k < nch; ++k) mx = fmaxf(mx, st[((size_t)k * M + R) * 2]);
        float sum = 0.f;
        if (mx != -INFINITY)
            for (int k = 0; k < nch; ++k) {
                const float mk = st[((size_t)k * M + R) * 2];
                if (mk != -INFINITY) sum += st[((size_t)k * M + R) * 2 + 1] * exp2f(mk - mx);
            }
        qst[R] = make_float2(p.qk_scale_log2, mx + log2f(sum));
    }
}

template <int PASS, int MT>
cudaError_t launch_mt(const EvictParams& p, const CUtensorMap* tk, const CUtensorMap* tq, cudaStream_t s)
{
    const dim3 grid(PASS == 1 ? p.nch1 : p.nch2, p.n_trig * p.lay.KVH);
    return launch_pdl(score_kernel<PASS, MT>, grid, dim3(kThreads), SCfg<MT>::SMEM, s, p, *tk, *tq);
}

template <int MT>
cudaError_t prepare_mt()
{
    cudaError_t e = cudaFuncSetAttribute(score_kernel<1, MT>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SCfg<MT>::SMEM);
    if (e != cudaSuccess) return e;
    return cudaFuncSetAttribute(score_kernel<2, MT>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SCfg<MT>::SMEM);
}

}  // namespace

int score_row_tiles_per_warp(int M) { return ((M + 15) / 16 + kWarps - 1) / kWarps; }

cudaError_t score_prepare()
{
    cudaError_t e;
    if ((e = prepare_mt<1>()) != cudaSuccess) return e;
    if ((e = prepare_mt<2>()) != cudaSuccess) return e;
    if ((e = prepare_mt<3>()) != cudaSuccess) return e;
    return prepare_mt<4>();
}

cudaError_t launch_score_merge(const EvictParams& p, cudaStream_t s)
{
    return launch_pdl(score_merge_kernel, dim3(p.n_trig * p.lay.KVH), dim3(256), 0, s, p);
}

cudaError_t launch_score(const EvictParams& p, int pass, const CUtensorMap* tk, const CUtensorMap* tq, cudaStream_t s)
{
    const int MT = score_row_tiles_per_warp(p.lay.r * p.lay.G);
    if (pass == 1) {
        switch (MT) {
            case 1: return launch_mt<1, 1>(p, tk, tq, s);
            case 2: return launch_mt<1, 2>(p, tk, tq, s);
            case 3: return launch_mt<1, 3>(p, tk, tq, s);
            case 4: return launch_mt<1, 4>(p, tk, tq, s);
        }
    } else {
        switch (MT) {
            case 1: return launch_mt<2, 1>(p, tk, tq, s);
            case 2: return launch_mt<2, 2>(p, tk, tq, s);
            case 3: return launch_mt<2, 3>(p, tk, tq, s);
            case 4: return launch_mt<2, 4>(p, tk, tq, s);
        }
    }
    return cudaErrorInvalidValue;
}

}  // namespace ra
