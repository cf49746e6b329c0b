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
//   summation pass (score_sum_tc_kernel<ROWS>)  per triggered (sequence, KV
//       head), the logits of the M = r * G window rows against the candidate
//       tiles, normalised by the recorded normalisers and summed over all M
//       rows: one fp32 score per candidate.  Each CTA holds all M rows, so
//       every candidate's sum is complete inside it -- no atomics, and the
//       result does not depend on the launch shape.  It runs on tcgen05 with
//       the accumulators in tensor memory (see the kernel).
//   restore pass (score_stats_kernel<MT> + score_merge_kernel)  only when a
//       window is loaded from outside (ra_restore_queries): the normalisers,
//       recomputed over the prompt and the cached rows each query sees (by
//       position), split over chunks of key tiles and merged.
// The contraction of the window rows with the key rows is a dense GEMM
// (M x keys x 128), so both passes run on the tensor cores.  The restore pass
// (a warm start only) uses mma.sync m16n8k16 (bf16 in, fp32 accumulate);
// its CTA layout: 8 warps; warp w owns the 16-row M tiles
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
static_assert(kPromptPage % kScoreTile == 0, "a scoring tile of the prompt lies inside one page");
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
    static constexpr int BAR_OFF = Q_OFF + ROWS * kRowBytes;
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

// Tiles of one head in the restore pass: its prompt rows, then its c cached generated rows.
__device__ __forceinline__ int head_tiles(int lp, int n_gen, int* tp)
{
    *tp = (lp + kScoreTile - 1) / kScoreTile;
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

// Restore pass: per window row, (max, sum of exp2) over one chunk of the keys it sees.
template <int MT>
__global__ void __launch_bounds__(kThreads, MT <= 2 ? 2 : 1) score_stats_kernel(const __grid_constant__ EvictParams p,
                                                                              const __grid_constant__ CUtensorMap tk,
                                                                              const __grid_constant__ CUtensorMap tw)
{
    using C = SCfg<MT>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::BAR_OFF);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    pdl_wait();  // the window, the cache and the tables come from earlier kernels
    pdl_launch_dependents();

    const DevLayout& L = p.lay;
    const int t = blockIdx.y / L.KVH, h = blockIdx.y - t * L.KVH;
    const int b = p.trig[t];
    const int N = p.trig_n[t], r = L.r, G = L.G, M = r * G;
    const int lp = L.seq_lp[b];
    int tp;
    const int nt_head = head_tiles(lp, N, &tp);
    const int ch = p.ch1;
    const int t0 = blockIdx.x * ch;
    if (t0 >= nt_head) return;  // (exiting counts as letting the successor start)
    const int ntile = min(ch, nt_head - t0);
    const long long pbase = prompt_row(L, p.layer, 0, h, 0);
    const int32_t* ptab = L.pages + (size_t)b * L.max_pages;
    const size_t lbh = ((size_t)p.layer * L.B + b) * L.KVH + h;
    const int reg = L.region[lbh];
    const long long grow = L.gen_row0 + (long long)reg * L.Cmax;
    const int hid = b * L.KVH + h;

    auto tile_row = [&](int k) -> long long {  // first cache row of the head's tile k
        // (a prompt tile lies inside one page: kPromptPage is a multiple of kScoreTile)
        return k < tp ? pbase + (long long)__ldg(ptab + k * kScoreTile / kPromptPage) * L.KVH * kPromptPage +
                            (k * kScoreTile) % kPromptPage
                      : grow + (long long)(k - tp) * kScoreTile;
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
    __syncthreads();

    // This lane's rows: R = 16 * (warp + 8 i) + (lane / 4) + 8 hf; its columns: 8 nt + 2 (lane % 4) + e.
    const int tq = lane & 3;
    const int mi = lane >> 3, ri = lane & 7;
    int lim[MT][2];  // generated rows the row sees
    float mrow[MT][2], lrow[MT][2];  // running max and (per-lane partial) sum of exp2
#pragma unroll
    for (int i = 0; i < MT; ++i)
#pragma unroll
        for (int hf = 0; hf < 2; ++hf) {
            const int R = 16 * (warp + kWarps * i) + (lane >> 2) + 8 * hf;
            lim[i][hf] = R < M ? visible_rows(L.pos + (size_t)reg * L.Cmax, N, lp, p.trig_g[t], r, R / G) : 0;
            mrow[i][hf] = -INFINITY;
            lrow[i][hf] = 0.f;
        }
    const float sl = p.qk_scale_log2;  // the scale the restored queries are taken at
    const uint32_t qs = smem_u32(smem + C::Q_OFF);

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
        {
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
        }
        __syncthreads();  // stage s free again
        if (tid == 0 && i + kStages < ntile) {
            fence_proxy_async_smem();
            issue(i + kStages, 0u);
        }
    }

    {  // this chunk's statistics of every real row
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

// ---------------------------------------------------------------------------------------------
// Summation pass on the 5th-generation tensor cores (tcgen05, accumulators in tensor memory).
//
// The product is taken transposed, D = K Q^T: the 128 candidate key rows of a tile are the M
// side of the MMA and the window rows are the N side (up to 256 per instruction), so that TMEM
// lane j holds every window row's logit against key j.  The thread that reads lane j then sums
// its own key's weights exp2(logit * scale_R - lse_R) over the window rows R, with no
// cross-thread reduction; the two warpgroups take half of the window rows each.  Both operands
// are K-major in shared memory with the 128-byte swizzle the TMA copies already produce (rows of
// 128 bytes, 8-row groups 1024 bytes apart, the two 64-channel halves one after the other); a
// K-step of 16 channels advances the descriptors' start address by 32 bytes.  One thread issues
// the MMAs and commits them to an mbarrier.  With a window of at most 256 rows the accumulator
// is double-buffered in TMEM, so the MMAs of tile i + 1 run while tile i's weights are summed.

constexpr int kTcRows = 128;                        // key rows per tile: the MMA's M
constexpr int kTcHalf = kTcRows * 128;              // one 64-channel half of a key tile
constexpr int kTcStage = 2 * kTcHalf;               // a key tile: 128 rows x 256 bytes

template <int ROWS>  // window rows held: r * G padded to a multiple of 128, at most 512
struct TcCfg {
    static constexpr int NCH = ROWS > 256 ? 2 : 1;             // MMAs per K-step (N <= 256 each)
    static constexpr int NC = ROWS / NCH;                      // N of each MMA
    static constexpr int NBUF = 2 * ROWS <= 512 ? 2 : 1;      // accumulator buffers in TMEM (512 columns)
    static constexpr uint32_t COLS = NBUF * ROWS <= 256 ? 256u : 512u;  // columns allocated (a power of 2)
    static constexpr int Q_OFF = 2 * kTcStage;                 // after the two key stages
    static constexpr int Q_HALF = ROWS * 128;
    static constexpr int STAT_OFF = Q_OFF + ROWS * kRowBytes;
    static constexpr int RED_OFF = STAT_OFF + 2 * ROWS * 4;
    static constexpr int BAR_OFF = RED_OFF + 2 * kTcRows * 4;  // full[2], mma_done[2], TMEM base
    static constexpr size_t SMEM = 1024 + (size_t)BAR_OFF + 4 * 8 + 16;
    static_assert(ROWS % 128 == 0 && ROWS <= 512, "window rows");
    static_assert(NC % 16 == 0 && NC <= 256, "UMMA N for M = 128");
    static_assert(SMEM <= 232448, "fits the 227 KB opt-in shared memory");
};

// Shared-memory matrix descriptor: K-major, 128-byte swizzle, 8-row groups 1024 bytes apart.
__device__ __forceinline__ uint64_t umma_desc_sw128(uint32_t saddr)
{
    uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);  // bits 0-13: start address >> 4
    d |= (uint64_t)1 << 16;                            // bits 16-29: leading byte offset (unused here)
    d |= (uint64_t)(1024 >> 4) << 32;                  // bits 32-45: stride byte offset >> 4
    d |= (uint64_t)1 << 46;                            // bits 46-48: fixed 0b001
    d |= (uint64_t)2 << 61;                            // bits 61-63: 128-byte swizzle
    return d;
}

// Instruction descriptor of kind::f16: fp32 accumulate, bf16 A and B, both K-major, M x N.
__device__ __forceinline__ uint32_t umma_idesc_bf16(int M, int N)
{
    return (1u << 4)                        // D: f32
           | (1u << 7) | (1u << 10)         // A, B: bf16
           | ((uint32_t)(N >> 3) << 17)     // N / 8
           | ((uint32_t)(M >> 4) << 24);    // M / 16
}

__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc, int accum)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accum)
        : "memory");
}

__device__ __forceinline__ void umma_commit(uint64_t* bar)
{
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
                 : "memory");
}

__device__ __forceinline__ void tmem_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tmem_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// 32 consecutive fp32 columns of this warp's 32 TMEM lanes (one lane per thread).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&v)[32])
{
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
        "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];\n\t"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
          "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]),
          "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]),
          "=r"(v[24]), "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
        : "r"(taddr)
        : "memory");
}

template <int ROWS>
__global__ void __launch_bounds__(kThreads, 1) score_sum_tc_kernel(const __grid_constant__ EvictParams p,
                                                                  const __grid_constant__ CUtensorMap tk,
                                                                  const __grid_constant__ CUtensorMap tw)
{
    using C = TcCfg<ROWS>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::BAR_OFF);  // key tile (and the window) landed
    uint64_t* mdone = full + 2;                                          // the tile's MMAs completed
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(full + 4);
    float* s_sl = reinterpret_cast<float*>(smem + C::STAT_OFF);
    float* s_lse = s_sl + ROWS;
    float* red = reinterpret_cast<float*>(smem + C::RED_OFF);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    // As the mma.sync pass: with p.early everything read here was written by kernels that
    // completed before the predecessor started, and the scores are read only by the successor.
    if (!p.early) {
        pdl_wait();
        pdl_launch_dependents();
    }
    const DevLayout& L = p.lay;
    const int t = blockIdx.y / L.KVH, h = blockIdx.y - t * L.KVH;
    const int b = p.trig[t];
    const int N = p.trig_n[t], M = L.r * L.G;
    const int r_lo = blockIdx.x * p.ch2 * kScoreTile;  // this CTA's candidate rows [r_lo, r_hi)
    if (r_lo >= N) {
        if (p.early) {
            pdl_wait();
            pdl_launch_dependents();
        }
        return;
    }
    const int r_hi = min(N, r_lo + p.ch2 * kScoreTile);
    const int ntile = (r_hi - r_lo + kTcRows - 1) / kTcRows;
    const size_t lbh = ((size_t)p.layer * L.B + b) * L.KVH + h;
    const long long grow = L.gen_row0 + (long long)L.region[lbh] * L.Cmax;

    auto issue_tile = [&](int i, uint32_t extra) {  // thread 0: key tile i into stage i % 2
        const int s = i % 2;
        uint8_t* st = smem + (size_t)s * kTcStage;
        const int row = (int)(grow + r_lo + (long long)i * kTcRows);
        mbar_arrive_expect_tx(&full[s], (uint32_t)kTcStage + extra);
        for (int q = 0; q < kTcRows; q += kScoreTile) {
            tma_load_2d(st + q * 128, &tk, 0, row + q, &full[s]);
            tma_load_2d(st + kTcHalf + q * 128, &tk, 64, row + q, &full[s]);
        }
    };
    if (warp == 0) {  // the accumulators' tensor memory (held until the end)
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                     "r"(C::COLS)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    if (tid == 0) {
        for (int s = 0; s < 2; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&mdone[s], 1);
        }
        fence_mbar_init();
        prefetch_tensormap(&tk);
        prefetch_tensormap(&tw);
        // The window rows (row R = slot * G + g) complete on full[0] with the first key tile;
        // rows past M are another head's (or read as zero): finite, and given no weight below.
        issue_tile(0, (uint32_t)(ROWS * kRowBytes));
        const int row0 = (int)(lbh * (size_t)M);
        for (int rb = 0; rb < ROWS; rb += kScoreTile) {
            tma_load_2d(smem + C::Q_OFF + rb * 128, &tw, 0, row0 + rb, &full[0]);
            tma_load_2d(smem + C::Q_OFF + C::Q_HALF + rb * 128, &tw, 64, row0 + rb, &full[0]);
        }
        if (ntile > 1) issue_tile(1, 0u);
    }
    // thread 0's counts of tiles: copies issued, MMAs issued, MMAs waited for
    int n_loaded = min(ntile, 2), n_mma = 0, done = 0;
    {  // the normaliser each window query had at its decode step
        const float2* qst = L.qstats + lbh * (size_t)M;
        for (int R = tid; R < ROWS; R += kThreads) {
            const float2 f = R < M ? __ldcg(qst + R) : make_float2(0.f, INFINITY);  // padding rows weigh 0
            s_sl[R] = f.x;
            s_lse[R] = f.y;
        }
    }
    tmem_fence_before();
    __syncthreads();
    tmem_fence_after();
    const uint32_t tmem = *tmem_slot;
    const uint32_t idesc = umma_idesc_bf16(kTcRows, C::NC);
    const uint32_t sbase = smem_u32(smem);

    // Thread 0: the MMAs of tile i into accumulator buffer i % NBUF, committed to mdone[i % 2].
    auto issue_mma = [&](int i) -> bool {
        if (!mbar_wait_bounded(&full[i % 2], (uint32_t)((i / 2) & 1), kWaitLimitNs)) return false;
        tmem_fence_after();
        const uint32_t d0 = tmem + (uint32_t)((i % C::NBUF) * ROWS);
        const uint32_t a0 = sbase + (uint32_t)((i % 2) * kTcStage);
#pragma unroll
        for (int kh = 0; kh < 2; ++kh)        // 64-channel half
#pragma unroll
            for (int kk = 0; kk < 4; ++kk) {  // 16-channel K-step inside the half
                const uint64_t ad = umma_desc_sw128(a0 + kh * kTcHalf + kk * 32);
#pragma unroll
                for (int c = 0; c < C::NCH; ++c) {
                    const uint64_t bd = umma_desc_sw128(sbase + C::Q_OFF + kh * C::Q_HALF + c * C::NC * 128 + kk * 32);
                    umma_bf16(d0 + c * C::NC, ad, bd, idesc, (kh | kk) != 0);
                }
            }
        umma_commit(&mdone[i % 2]);
        n_mma = i + 1;
        return true;
    };

    float* scores = L.scores + lbh * L.Cmax;
    const int wg = warp >> 2, wq = warp & 3;  // warpgroup (half of the window rows), TMEM lane quarter
    bool ok = true;
    if (tid == 0) ok = issue_mma(0);
    for (int i = 0; i < ntile; ++i) {
        if (C::NBUF == 2 && tid == 0 && ok && i + 1 < ntile) ok = issue_mma(i + 1);
        const bool got = mbar_wait_bounded(&mdone[i % 2], (uint32_t)((i / 2) & 1), kWaitLimitNs);
        if (!__syncthreads_and(got && ok)) {  // give up together
            if (tid == 0) atomicExch(L.err, kDeviceErrTimeout);
            break;
        }
        done = i + 1;
        tmem_fence_after();
        if (tid == 0 && i + 2 < ntile) {  // the tile's MMAs have read stage i % 2: refill it
            fence_proxy_async_smem();
            issue_tile(i + 2, 0u);
            n_loaded = i + 3;
        }
        // this thread: key row wq * 32 + lane of the tile, window rows [wg * ROWS / 2, (wg + 1) * ROWS / 2)
        const uint32_t tl = tmem + ((uint32_t)(wq * 32) << 16) + (uint32_t)((i % C::NBUF) * ROWS);
        float sum = 0.f;
#pragma unroll 1
        for (int c0 = wg * (ROWS / 2); c0 < (wg + 1) * (ROWS / 2); c0 += 32) {
            uint32_t v[32];
            tmem_ld32(tl + c0, v);
#pragma unroll
            for (int j = 0; j < 32; ++j) sum += exp2f(fmaf(__uint_as_float(v[j]), s_sl[c0 + j], -s_lse[c0 + j]));
        }
        red[wg * kTcRows + wq * 32 + lane] = sum;
        tmem_fence_before();
        __syncthreads();  // both halves summed; the accumulator buffer is free again
        if (tid < kTcRows) {
            const int row = r_lo + i * kTcRows + tid;
            if (row < r_hi) scores[row] = red[tid] + red[kTcRows + tid];
        }
        if (C::NBUF == 1 && tid == 0 && ok && i + 1 < ntile) {
            tmem_fence_after();
            ok = issue_mma(i + 1);
        }
        __syncthreads();  // red is rewritten by the next tile
    }
    // Leave only with nothing in flight: after a timeout, the MMAs issued but not waited for and
    // the copies issued but not consumed are waited for once more, bounded.
    if (tid == 0) {
        for (int i = done; i < n_mma; ++i) (void)mbar_wait_bounded(&mdone[i % 2], (uint32_t)((i / 2) & 1), kWaitLimitNs);
        for (int i = n_mma; i < n_loaded; ++i) (void)mbar_wait_bounded(&full[i % 2], (uint32_t)((i / 2) & 1), kWaitLimitNs);
    }
    tmem_fence_before();
    __syncthreads();
    if (warp == 0) {
        tmem_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(C::COLS) : "memory");
    }
    if (p.early) {
        pdl_wait();
        pdl_launch_dependents();
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
    const int nch = (head_tiles(L.seq_lp[b], p.trig_n[t], &tp) + p.ch1 - 1) / p.ch1;
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

template <int MT>
cudaError_t launch_stats(const EvictParams& p, const CUtensorMap* tk, const CUtensorMap* tq, cudaStream_t s)
{
    const dim3 grid(p.nch1, p.n_trig * p.lay.KVH);
    return launch_pdl(score_stats_kernel<MT>, grid, dim3(kThreads), SCfg<MT>::SMEM, s, p, *tk, *tq);
}

template <int MT>
cudaError_t prepare_mt()
{
    cudaError_t e = cudaFuncSetAttribute(score_stats_kernel<MT>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SCfg<MT>::SMEM);
    if (e != cudaSuccess) return e;
    return cudaFuncSetAttribute(score_sum_tc_kernel<128 * MT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)TcCfg<128 * MT>::SMEM);
}

template <int MT>
cudaError_t launch_sum_tc(const EvictParams& p, const CUtensorMap* tk, const CUtensorMap* tq, cudaStream_t s)
{
    const dim3 grid(p.nch2, p.n_trig * p.lay.KVH);
    return launch_pdl(score_sum_tc_kernel<128 * MT>, grid, dim3(kThreads), TcCfg<128 * MT>::SMEM, s, p, *tk, *tq);
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
            case 1: return launch_stats<1>(p, tk, tq, s);
            case 2: return launch_stats<2>(p, tk, tq, s);
            case 3: return launch_stats<3>(p, tk, tq, s);
            case 4: return launch_stats<4>(p, tk, tq, s);
        }
    } else {
        switch (MT) {
            case 1: return launch_sum_tc<1>(p, tk, tq, s);
            case 2: return launch_sum_tc<2>(p, tk, tq, s);
            case 3: return launch_sum_tc<3>(p, tk, tq, s);
            case 4: return launch_sum_tc<4>(p, tk, tq, s);
        }
    }
    return cudaErrorInvalidValue;
}

}  // namespace ra
