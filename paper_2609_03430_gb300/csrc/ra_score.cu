// ra_score.cu -- window attention of the scored comparator on sm_103a.
//
// The comparator ranks a head's eviction candidates by the SnapKV score of
// section 2 ("Baselines as choices of s"): the attention that the window of
// the last r decode queries gives each candidate, summed over the window and
// over the G query heads of the KV group (max-pooling and top-K happen in the
// select kernel).  A window query of step s attends, like the decode step it
// came from, to the keys at positions up to its own: the prompt, every
// candidate, and the first u buffer rows, u = its rank in the window.
//
// Per triggered (sequence, KV head) the window is M = r * G query rows.  The
// contraction of those rows with every key row is a dense GEMM (M x keys x 128),
// so it runs on the tensor cores (mma.sync m16n8k16, bf16 in, fp32 accumulate):
//   pass 1 (score_kernel<1, MT>)  per row, the running max and sum of exp of
//       the scaled logits over the keys it sees, over one chunk of key tiles;
//       one (max, sum) pair per row and chunk goes to the statistics buffer.
//   pass 2 (score_kernel<2, MT>)  merges a head's chunk statistics, recomputes
//       the logits of the candidate tiles, normalises them and sums the weights
//       over all M rows: one fp32 score per candidate.  Each CTA holds all M
//       rows, so every column sum is complete inside it -- no atomics, and the
//       result does not depend on the launch shape.
// CTA layout: 8 warps; warp w owns the 16-row M tiles w, w + 8, ... (MT of
// them).  The M rows sit in shared memory with a 16-byte-chunk xor swizzle and
// are read as A fragments with ldmatrix; key tiles of 64 rows x 128 channels
// arrive by 2-D TMA (two 64-channel boxes, 128-byte swizzle) into a two-stage
// ring on mbarriers, and are read as B fragments with ldmatrix.  Logits are in
// base 2 with the scale folded into one multiply.
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
    static constexpr int Q_OFF = kStages * kTileBytes;            // after the key stages
    static constexpr int STAT_OFF = Q_OFF + ROWS * kRowBytes;     // pass 2: row max and 1/sum
    static constexpr int RED_OFF = STAT_OFF + 2 * ROWS * 4;       // pass 2: column sums per warp
    static constexpr int BAR_OFF = RED_OFF + kWarps * kScoreTile * 4;
    static constexpr size_t SMEM = 1024 + (size_t)BAR_OFF + kStages * 8;
    static_assert(ROWS <= kScoreMaxRows || MT == 1, "window rows");
    static_assert(SMEM <= 232448, "fits the 227 KB opt-in shared memory");
};

// Byte offset of (window row R, 16-byte chunk c) of the M x 128 query block:
// chunks are xored with R mod 8 within each 128-byte half of a row.
__device__ __forceinline__ uint32_t qswz(int R, int c) { return (uint32_t)(R * kRowBytes + ((c & 8) | ((c ^ R) & 7)) * 16); }

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

// Tiles of one head in pass 1: its prompt rows, then its generated rows up to the
// newest any window query sees (ordinal N + r - 2); in pass 2: the candidate rows.
__device__ __forceinline__ int head_tiles(int pass, int lp, int N, int r, int* tp)
{
    if (pass == 2) {
        *tp = 0;
        return (N + kScoreTile - 1) / kScoreTile;
    }
    *tp = (lp + kScoreTile - 1) / kScoreTile;
    return *tp + (N + r - 1 + kScoreTile - 1) / kScoreTile;
}

template <int PASS, int MT>
__global__ void __launch_bounds__(kThreads, MT <= 2 ? 2 : 1) score_kernel(const __grid_constant__ EvictParams p,
                                                            const __grid_constant__ CUtensorMap tk)
{
    using C = SCfg<MT>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::BAR_OFF);
    float* s_m = reinterpret_cast<float*>(smem + C::STAT_OFF);
    float* s_il = s_m + C::ROWS;
    float* red = reinterpret_cast<float*>(smem + C::RED_OFF);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    pdl_wait();  // the window, the cache and the tables come from earlier kernels
    pdl_launch_dependents();

    const DevLayout& L = p.lay;
    const int t = blockIdx.y / L.KVH, h = blockIdx.y - t * L.KVH;
    const int b = p.trig[t];
    const int N = p.trig_n[t], r = L.r, G = L.G, M = r * G;
    const int lp = L.seq_lp[b];
    int tp;
    const int nt_head = head_tiles(PASS, lp, N, r, &tp);
    const int ch = PASS == 1 ? p.ch1 : p.ch2;
    const int t0 = blockIdx.x * ch;
    if (t0 >= nt_head) return;
    const int ntile = min(ch, nt_head - t0);
    const long long prow = (long long)p.layer * L.prompt_rows_per_layer + L.seq_poff[b] + (long long)h * lp;
    const int reg = L.region[((size_t)p.layer * L.B + b) * L.KVH + h];
    const long long grow = L.gen_row0 + (long long)reg * L.Cmax;
    const int hid = b * L.KVH + h;

    auto tile_row = [&](int k) -> long long {  // first cache row of the head's tile k
        return k < tp ? prow + (long long)k * kScoreTile : grow + (long long)(k - tp) * kScoreTile;
    };
    auto issue = [&](int i) {  // thread 0: tile t0 + i into stage i % 2
        const int s = i % kStages;
        uint8_t* st = smem + (size_t)s * kTileBytes;
        const int row = (int)tile_row(t0 + i);
        mbar_arrive_expect_tx(&bars[s], (uint32_t)kTileBytes);
        tma_load_2d(st, &tk, 0, row, &bars[s]);
        tma_load_2d(st + kHalfBytes, &tk, 64, row, &bars[s]);
    };
    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) mbar_init(&bars[s], 1);
        fence_mbar_init();
        prefetch_tensormap(&tk);
        for (int i = 0; i < kStages && i < ntile; ++i) issue(i);
    }

    // The window rows (row R = slot * G + g), zero past M.
    const uint16_t* win = L.qring + (((size_t)p.layer * L.B + b) * L.KVH + h) * (size_t)M * kHeadDim;
    for (int i = tid; i < C::ROWS * 16; i += kThreads) {
        const int R = i >> 4, c = i & 15;
        const uint4 v = R < M ? __ldcg(reinterpret_cast<const uint4*>(win) + i) : make_uint4(0u, 0u, 0u, 0u);
        *reinterpret_cast<uint4*>(smem + C::Q_OFF + qswz(R, c)) = v;
    }
    float* stats = L.stats + (size_t)hid * L.stats_chunks * M * 2;
    if (PASS == 2) {  // merge the chunk statistics of pass 1 into each row's max and 1/sum
        int tp1;
        const int nch = (head_tiles(1, lp, N, r, &tp1) + p.ch1 - 1) / p.ch1;
        for (int R = tid; R < C::ROWS; R += kThreads) {
            float mx = 0.f, il = 0.f;
            if (R < M) {
                mx = -INFINITY;
                for (int k = 0; k < nch; ++k) mx = fmaxf(mx, __ldcg(stats + ((size_t)k * M + R) * 2));
                float sum = 0.f;
                for (int k = 0; k < nch; ++k) {
                    const float mk = __ldcg(stats + ((size_t)k * M + R) * 2);
                    if (mk != -INFINITY) sum += __ldcg(stats + ((size_t)k * M + R) * 2 + 1) * exp2f(mk - mx);
                }
                il = 1.f / sum;
            }
            s_m[R] = mx;
            s_il[R] = il;
        }
    }
    __syncthreads();

    // This lane's rows: R = 16 * (warp + 8 i) + (lane / 4) + 8 hf; its columns: 8 nt + 2 (lane % 4) + e.
    const int tq = lane & 3;
    const int mi = lane >> 3, ri = lane & 7;
    const float sl = p.qk_scale_log2;
    int lim[MT][2];  // pass 1: generated ordinals this row sees (N + its rank in the window)
    // pass 1: running max and (per-lane partial) sum of exp2; pass 2: the row's max and 1/sum
    float mrow[MT][2], lrow[MT][2];
#pragma unroll
    for (int i = 0; i < MT; ++i)
#pragma unroll
        for (int hf = 0; hf < 2; ++hf) {
            const int R = 16 * (warp + kWarps * i) + (lane >> 2) + 8 * hf;
            lim[i][hf] = N + ((R / G) + 1) % r;
            if (PASS == 1) {
                mrow[i][hf] = -INFINITY;
                lrow[i][hf] = 0.f;
            } else {
                mrow[i][hf] = s_m[R];
                lrow[i][hf] = s_il[R];
            }
        }
    const uint32_t qs = smem_u32(smem + C::Q_OFF);
    float* scores = L.scores + (((size_t)p.layer * L.B + b) * L.KVH + h) * L.Cmax;

    for (int i = 0; i < ntile; ++i) {
        const int s = i % kStages;
        const bool ok = mbar_wait_bounded(&bars[s], (uint32_t)((i / kStages) & 1), kWaitLimitNs);
        if (!__syncthreads_and(ok)) {  // give up together; let the copies in flight land first
            if (tid == 0) {
                atomicExch(L.err, kDeviceErrTimeout);
                for (int j = i + 1; j < ntile && j < i + kStages; ++j)
                    (void)mbar_wait_bounded(&bars[j % kStages], (uint32_t)((j / kStages) & 1), kWaitLimitNs);
            }
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
            for (int a = 0; a < MT; ++a) ldsm_x4(af[a], qs + qswz(16 * (warp + kWarps * a) + (lane & 15), 2 * kk + (lane >> 4)));
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
                            cs[n][e] += exp2f(acc[a][n][2 * hf + e] * sl - mrow[a][hf]) * lrow[a][hf];
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
            issue(i + kStages);
        }
    }

    if (PASS == 1) {  // this chunk's statistics of every real row
        float* out = stats + (size_t)blockIdx.x * M * 2;
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

template <int PASS, int MT>
cudaError_t launch_mt(const EvictParams& p, const CUtensorMap* tk, cudaStream_t s)
{
    const dim3 grid(PASS == 1 ? p.nch1 : p.nch2, p.n_trig * p.lay.KVH);
    return launch_pdl(score_kernel<PASS, MT>, grid, dim3(kThreads), SCfg<MT>::SMEM, s, p, *tk);
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

cudaError_t launch_score(const EvictParams& p, int pass, const CUtensorMap* tk, cudaStream_t s)
{
    const int MT = score_row_tiles_per_warp(p.lay.r * p.lay.G);
    if (pass == 1) {
        switch (MT) {
            case 1: return launch_mt<1, 1>(p, tk, s);
            case 2: return launch_mt<1, 2>(p, tk, s);
            case 3: return launch_mt<1, 3>(p, tk, s);
            case 4: return launch_mt<1, 4>(p, tk, s);
        }
    } else {
        switch (MT) {
            case 1: return launch_mt<2, 1>(p, tk, s);
            case 2: return launch_mt<2, 2>(p, tk, s);
            case 3: return launch_mt<2, 3>(p, tk, s);
            case 4: return launch_mt<2, 4>(p, tk, s);
        }
    }
    return cudaErrorInvalidValue;
}

}  // namespace ra
