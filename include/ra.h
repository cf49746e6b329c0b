/*
 * ra.h -- C ABI of the GB300 (sm_103a) Random Attention decode library.
 *
 * Random Attention (arXiv 2609.03430) evicts KV-cache entries during decoding
 * with no score: the prompt is always kept, the newest r tokens form a buffer
 * that is never a candidate, and among the older generated tokens every KV head
 * independently keeps a budget of K drawn uniformly at random (section 3,
 * applied through Eq. 1 of section 2).  This library owns the per-(sequence,
 * layer, KV head) caches and runs the decode hot path on the GPU:
 *
 *   ra_append_kv    write the step's new post-RoPE K/V          (Appendix F)
 *   ra_evict        periodic random eviction + compaction       (sections 2-3)
 *   ra_decode_attn  GQA decode attention over the caches        (section 2)
 *
 * Conventions (every entry point):
 *   - Return RA_OK (0) or a negative RA_ERR_* code; ra_last_error() gives text.
 *     Argument and state errors are detected on the host before any launch
 *     and leave the state unchanged.
 *   - `stream` is a cudaStream_t (NULL = legacy default stream).  All calls are
 *     asynchronous on it and never synchronise, except the debug getters
 *     (ra_get_*) and ra_check_device, which synchronise that stream.  Issue all
 *     calls of one context on one stream (or order them yourself).
 *   - Device pointers are caller-owned and must stay valid until the stream
 *     work that uses them has finished.  bf16 tensors are passed as uint16_t
 *     bit patterns.  Every device pointer must be 16-byte aligned.
 *   - The library never allocates device memory: the caller sizes one arena
 *     with ra_device_bytes() (e.g. a torch uint8 CUDA tensor) and binds it.
 *   - head_dim must be 128; G = q_heads / kv_heads must be an integer in
 *     [1, 8]; query head qh reads KV head qh / G (consecutive grouping; the
 *     paper's GQA models share a KV head's keep-set across its query group,
 *     Appendix F).
 *
 * Budget convention: K counts the retained *generated* tokens of a head.  The
 * paper's budget holds the prompt too (prompt entries score +inf, section 3),
 * so K_paper = prompt_len + K.
 *
 * Random draw (the paper fixes none; this is the library's mapping): the score
 * of candidate j (its ordinal in slot order among the c - r candidates) is
 * word 0 of Philox4x32-10 (Salmon et al., SC'11) with
 *     counter = (j, g, layer, (a << 16) | (seq * kv_heads + kv_head)),  key = (seed lo, seed hi),
 * where g is the number of generated tokens appended when the eviction fires
 * and a the number of requests admitted into slot seq before the current one
 * (0 for the batch given at creation; see ra_admit), so that every request
 * draws its own numbers (a per-request stream, as the paper's per-request
 * seed).  The K smallest (score, j) survive.
 */
#ifndef RA_H_
#define RA_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define RA_OK 0
#define RA_ERR_INVALID_ARG (-1)    /* bad argument (range, alignment, NULL) */
#define RA_ERR_STATE (-2)          /* call not valid in the current state (e.g. no arena bound) */
#define RA_ERR_CAPACITY (-3)       /* append would exceed prompt_len + K + 2r slots (evict not called) */
#define RA_ERR_CUDA (-4)           /* a CUDA runtime call or launch failed */
#define RA_ERR_DEVICE_TIMEOUT (-5) /* a kernel gave up a bounded wait and flagged it (ra_check_device) */
#define RA_ERR_UNSUPPORTED (-6)    /* shape outside what the kernels implement */

#define RA_MAX_BATCH 512

typedef struct ra_ctx ra_ctx;

/* Per-kernel timing classes for ra_profile_read. */
enum ra_kernel_kind {
    RA_KERNEL_APPEND = 0,
    RA_KERNEL_SELECT = 1,
    RA_KERNEL_COMPACT = 2,
    RA_KERNEL_ATTN = 3,
    RA_KERNEL_SCORE_STATS = 4, /* scored comparator: normalisers of a restored query window */
    RA_KERNEL_SCORE_SUM = 5,   /* scored comparator: window attention summed per candidate */
    RA_KERNEL_EVICT = 6,       /* selection and order-preserving compaction in one launch */
    RA_KERNEL_PLAN = 7,        /* evicted sets of the next step, computed beside the current one */
    RA_KERNEL_STACK = 8,       /* every layer's in-place compaction of the sequences firing at a whole-stack step */
    RA_KERNEL_KINDS = 9
};

/*
 * Create a batch-1 context: `layers` layers of `q_heads` query / `kv_heads` KV
 * heads of size head_dim, a prompt of prompt_len tokens, budget K >= 0 and
 * buffer r >= 1 (the paper uses r = 64, Appendix F), eviction seed `seed`.
 * Host-only; bind an arena before any other call.
 */
int ra_create(ra_ctx** out, int layers, int q_heads, int kv_heads, int head_dim, int prompt_len, int K, int r,
              uint64_t seed);

/*
 * Same for `batch` sequences with their own prompt lengths
 * (prompt_lens: host array [batch], each >= 0).  batch <= RA_MAX_BATCH.
 */
int ra_create_batched(ra_ctx** out, int layers, int q_heads, int kv_heads, int head_dim, int batch,
                      const int32_t* prompt_lens, int K, int r, uint64_t seed);

/* Bytes of device memory the context needs (caches, tables, scratch). */
size_t ra_device_bytes(const ra_ctx* ctx);

/*
 * Bind `bytes` >= ra_device_bytes() of caller-owned device memory (256-byte
 * aligned) on the current device and initialise the tables on `stream`.
 * All caches start empty (g = c = 0 for every sequence and layer).
 */
int ra_bind(ra_ctx* ctx, void* device_arena, size_t bytes, void* stream);

/*
 * Fill layer `layer`'s prompt caches: k, v device [batch][kv_heads][row_stride][head_dim],
 * of which rows [0, prompt_len(seq)) are used; row_stride >= max prompt_len.
 */
int ra_prefill(ra_ctx* ctx, int layer, const uint16_t* k, const uint16_t* v, int row_stride, void* stream);

/*
 * Restore the generated part of layer `layer` (warm start / checkpoint load):
 * for every sequence b, g_host[b] tokens have been generated and c_host[b]
 * (<= K + 2r, <= g_host[b]) of them are cached, at positions
 * pos[b][h][0..c) (device int32 [batch][kv_heads][row_stride], strictly
 * increasing, in [prompt_len(b), prompt_len(b) + g)) with rows k, v
 * (device [batch][kv_heads][row_stride][head_dim]).
 */
int ra_restore(ra_ctx* ctx, int layer, const int32_t* g_host, const int32_t* c_host, const int32_t* pos,
               const uint16_t* k, const uint16_t* v, int row_stride, void* stream);

/*
 * Candidate scoring policy (default RA_POLICY_RANDOM, the method).  The others
 * are the controls the paper contrasts with it, kept through the same Eq. 1
 * top-K and compaction:
 *   RA_POLICY_SHARED   one draw per (sequence, layer) used by every KV head --
 *                      the shared-draw control (section 5, Appendix D);
 *   RA_POLICY_RECENCY  keep the K newest candidates -- protected recency, the
 *                      prompt plus a contiguous recent window (section 4.1, 5);
 *   RA_POLICY_BLOCK    one draw per block of `block` consecutive positions, so
 *                      the history is kept in contiguous blocks (section 5).
 *   RA_POLICY_SNAPKV   the scored comparator: a candidate's score is the
 *                      attention it receives from the window of the last r
 *                      decode queries, summed over the query heads of its KV
 *                      group and max-pooled over the 3 candidates on either
 *                      side (SnapKV as section 2 writes it, with the prompt
 *                      pinned and the buffer unscored as for the method); the
 *                      K best survive, ties to the earlier position.  Each
 *                      window query's weights are those of its own decode
 *                      step: the same scale, over the keys at positions up
 *                      to its own (the cache only grows between rounds, so
 *                      that is what it saw; the attention calls record each
 *                      query's softmax normaliser for this).
 * Takes effect from the next eviction; `block` >= 1 is used by RA_POLICY_BLOCK.
 *
 * The scored policy needs a per-layer window of recent queries, which the
 * attention calls record: set it BEFORE ra_device_bytes / ra_bind (the arena
 * then also holds the window, the scores and their scratch, and the context
 * keeps recording the window under every policy); on a context bound without
 * them it fails with RA_ERR_STATE.  It requires r * G <= 512 and K + r <= 16384.
 */
#define RA_POLICY_RANDOM 0
#define RA_POLICY_SHARED 1
#define RA_POLICY_RECENCY 2
#define RA_POLICY_BLOCK 3
#define RA_POLICY_SNAPKV 4
int ra_set_policy(ra_ctx* ctx, int policy, int block);

/*
 * Compaction of an eviction round (default RA_COMPACT_ORDERED):
 *   RA_COMPACT_ORDERED  the survivors stay in time order: kept candidates, then
 *                       the buffer, moved into a fresh region (Appendix F keeps
 *                       each keep-set in time order and gathers the cache into
 *                       it).  Moves about K + r rows per head and round.
 *   RA_COMPACT_HOLEFILL order-free: attention is a sum over the cached set
 *                       (section 2), so slots need no order -- in Appendix G's
 *                       terms a keep-set is a random permutation of slot
 *                       indices.  Each candidate's key is drawn per position
 *                       (counter word 0 = its position instead of its ordinal;
 *                       recency keeps the largest positions), so the kept set
 *                       does not depend on the layout.  The m evicted slots
 *                       e_0 < ... < e_{m-1} are refilled in place and the
 *                       cache shrinks to c - m slots, c counting the step's
 *                       token: slot e_i takes slot c - m + i for i < m - 1,
 *                       and the newest row (the token) ends in the new last
 *                       slot c - m - 1, whose own row, unless e_{m-1} is that
 *                       slot, fills e_{m-1}.  At most m + 1 <= r + 1 row moves
 *                       per head and round, done by the selection kernel (in
 *                       a whole-stack step, for every layer of the firing
 *                       sequences in one launch); in the fused forms the
 *                       attention kernel appends the token into the last
 *                       slot, as in the ordered layout.  ra_get_positions then
 *                       lists positions in slot order, which is no longer
 *                       time order.
 *   RA_COMPACT_FUSED    the ordered layout, but in ra_decode_layer the attention
 *                       pass itself does the compaction: it reads each evicting
 *                       head's old region (as it must read every survivor
 *                       anyway), gives the evicted rows no weight, and writes
 *                       each survivor and the step's token to its slot in the
 *                       new region -- one read of the old rows instead of two.
 *                       Needs r <= 64; otherwise, and in ra_evict, the
 *                       separate compaction runs.  Results are identical to
 *                       RA_COMPACT_ORDERED (slower on the measured workloads:
 *                       the copy is done by the attention warps).
 * Takes effect from the next eviction.  RA_COMPACT_HOLEFILL cannot be combined
 * with RA_POLICY_SNAPKV (its pooling runs over neighbouring positions, which
 * needs time order): that combination fails with RA_ERR_UNSUPPORTED.
 */
#define RA_COMPACT_ORDERED 0
#define RA_COMPACT_HOLEFILL 1
#define RA_COMPACT_FUSED 2
int ra_set_compaction(ra_ctx* ctx, int mode);

/*
 * Scored policy, warm start: load the query window of layer `layer` from q,
 * device [batch][q_heads][r][head_dim] bf16, where row u of (b, qh) is the
 * query of decode step g_b - r + 1 + u (g_b = the sequence's generated count,
 * so row r - 1 is the latest step), attended at `scale` (<= 0: 1/sqrt(d)).
 * Call it after ra_prefill / ra_restore of the layer: it also recomputes each
 * loaded query's softmax normaliser over the prompt and the cached rows at
 * positions up to its own.  Steps before the first are never read.
 * RA_ERR_STATE unless the context was bound with the scored policy's buffers.
 */
int ra_restore_queries(ra_ctx* ctx, int layer, const uint16_t* q, float scale, void* stream);

/*
 * Debug (scored policy): copy the raw window scores (before pooling) that the
 * latest scored eviction of (layer, seq, kv_head) computed, one fp32 per
 * candidate in slot order, to host (synchronises).  *n = the candidate count
 * of that eviction (0 if none happened yet); capacity must be >= *n.
 */
int ra_get_scores(ra_ctx* ctx, int layer, int seq, int kv_head, float* host_scores, int capacity, int* n,
                  void* stream);

/*
 * Tuning: the decode-attention kernel shape.  RA_ATTN_SHAPE_AUTO (default)
 * picks per launch: layers attending fewer than 2^20 cache rows take the
 * narrow shape (32-row tiles, 6 warps per SM: a finer split of a short layer),
 * larger ones the wide shape (48-row tiles, 4 warps).  Outputs agree within
 * fp32 rounding (the split, hence the summation order, differs).
 */
#define RA_ATTN_SHAPE_AUTO 0
#define RA_ATTN_SHAPE_WIDE 1
#define RA_ATTN_SHAPE_NARROW 2
int ra_set_attention_shape(ra_ctx* ctx, int shape);

/*
 * Tuning: how an ordered-compaction round of the random policy (and of the shared, recency and
 * block variants) runs.  RA_EVICT_AUTO (default) launches one kernel: for every triggered head
 * one or more thread-block clusters each draw the keys, select the evicted set exactly across
 * the cluster through distributed shared memory, and move their share of the survivors; the
 * cluster size and the clusters per head are chosen from the number of triggered heads and the
 * device's cluster occupancy.  For the random and shared draws the selection first takes the
 * candidates above a cut that about 2m + 32 of them pass (m = candidates - K evicted) and ranks
 * those exactly; if fewer than m pass it falls back to exact radix passes over the keys, which
 * RA_EVICT_EXACT (or-ed into the mode) forces.  RA_EVICT_TWO_KERNELS runs the selection kernel
 * (one CTA per head, writing the evicted list to global memory) and then the compaction kernel.
 * A value in [2, 16] forces that cluster size (raised to the minimum that holds a head's keys,
 * ceil((K + r) / 2112) CTAs, or to the next size the device can schedule).  Results are
 * identical in every mode.  The scored policy, order-free and in-attention compaction, and
 * buffers of r > 512 always use the selection kernel in the per-layer calls.  RA_EVICT_TWO_KERNELS
 * also turns off the sets computed ahead in ra_decode_step, so every round selects in step.
 */
#define RA_EVICT_AUTO 0
#define RA_EVICT_TWO_KERNELS 1
#define RA_EVICT_EXACT 256
int ra_set_eviction_kernel(ra_ctx* ctx, int mode);

/*
 * Prompt pool; set it BEFORE ra_device_bytes / ra_bind (default: exactly the prompts given at
 * creation).  Prompt rows live in pages of 192 positions (all KV heads of one sequence, in every
 * layer), listed per sequence in a page table that the kernels read tile by tile, so that a
 * finished sequence's slot can take a new request with a prompt of another length (ra_admit).
 * max_prompt_len: the longest prompt a slot will take; pool_positions: the prompt positions the
 * pool holds over all slots (per layer and KV head), rounded up to pages and at least what the
 * creation prompts use.  RA_ERR_STATE once bound.
 */
int ra_set_prompt_pool(ra_ctx* ctx, int max_prompt_len, long long pool_positions);

/*
 * Admit a new request into slot `seq`, which must be finished (ra_set_active(seq, 0)): the slot's
 * prompt pages return to the pool and ceil(prompt_len / 192) pages are taken, the prompt rows
 * k, v (device [layers][kv_heads][row_stride][head_dim], rows [0, prompt_len) used; post-RoPE
 * keys, Appendix F) are written on `stream`, the slot's counters restart at g = c = 0 in every
 * layer, and the slot is active again.  The generated regions are reused as they are; positions
 * restart at 0 for the new request.  Its random stream is the slot's next one (admission count
 * in the key; see the mapping above).  Errors leave the state unchanged: RA_ERR_STATE if the slot
 * is active, RA_ERR_CAPACITY if prompt_len exceeds the pool's longest prompt or its free pages.
 * (The paper's serving runs use vLLM's paged cache; this is that capability for the prompt.)
 */
int ra_admit(ra_ctx* ctx, int seq, int prompt_len, const uint16_t* k, const uint16_t* v, int row_stride, void* stream);

/* Mark sequence `seq` active (1) or finished (0); finished ones are skipped by every call. */
int ra_set_active(ra_ctx* ctx, int seq, int active);

/*
 * Append the step's new token of every active sequence to layer `layer`:
 * k_new, v_new device [batch][kv_heads][head_dim] (post-RoPE keys, Appendix F).
 * The token's position is prompt_len + g; g and c advance by one.
 * RA_ERR_CAPACITY if a cache already holds K + 2r generated tokens.
 */
int ra_append_kv(ra_ctx* ctx, int layer, const uint16_t* k_new, const uint16_t* v_new, void* stream);

/*
 * Random Attention eviction of layer `layer` (sections 2-3, Appendix F).  Runs
 * after the step's append.  For every active sequence whose trigger fires --
 * g is a multiple of r and the candidates (all cached generated tokens but the
 * newest r) exceed K -- each KV head keeps the K candidates with the smallest
 * Philox scores (see above), in their original order, followed by the r buffer
 * tokens; K/V rows and positions are compacted order-preserving.  A no-op for
 * sequences whose trigger does not fire.  *n_fired (may be NULL) receives the
 * number of sequences that evicted.
 */
int ra_evict(ra_ctx* ctx, int layer, int* n_fired, void* stream);

/*
 * GQA decode attention of layer `layer` (section 2, "Notation"):
 * out[b][qh] = sum_i softmax_i(scale * q[b][qh] . k_i) v_i over the prompt and
 * the cached generated tokens of KV head qh / G.  q, out: device
 * [batch][q_heads][head_dim] bf16; fp32 accumulation, bf16 round-to-nearest
 * output.  scale <= 0 means 1/sqrt(head_dim).  Rows of inactive sequences are
 * not written.
 */
int ra_decode_attn(ra_ctx* ctx, int layer, const uint16_t* q, uint16_t* out, float scale, void* stream);

/*
 * One decode step of one layer, fused; same result as ra_append_kv ->
 * ra_evict -> ra_decode_attn with the same arguments.  The eviction runs first
 * with the step's token pending: the newest slot is never a candidate, so
 * evicting before writing it leaves the identical cache.  One attention kernel
 * then writes the new token's row and position, attends over prompt + cache +
 * new token, and merges its own split pieces.  k_new, v_new: device
 * [batch][kv_heads][head_dim]; q, out: device [batch][q_heads][head_dim].
 * RA_ERR_CAPACITY as for ra_append_kv.  Layers called in order 0 .. layers-1
 * form a step, as in ra_decode_step: with ordered or order-free compaction and
 * a policy other than the scored one, layer 0's call also runs every layer's
 * round of the sequences that fire, from evicted sets computed during the
 * previous step (same result as each layer evicting in its own call), and
 * layer layers-1's call joins the library's stream back.
 */
int ra_decode_layer(ra_ctx* ctx, int layer, const uint16_t* q, const uint16_t* k_new, const uint16_t* v_new,
                    uint16_t* out, float scale, void* stream);

/*
 * One decode step of the whole layer stack: ra_decode_layer for l = 0..layers-1,
 * with q_all [layers][batch][q_heads][d], k_all / v_all [layers][batch][kv_heads][d],
 * out_all [layers][batch][q_heads][d].  Capacity is checked for every layer first,
 * so a step that fails changes nothing.  Same result as the per-layer calls, by a
 * faster route: the keys of the random policy and its variants (not the scored
 * one) need no cache data beyond positions, so during each step a kernel on a
 * stream of the library's own (forked from `stream` at the step's start and
 * joined to it at its end, by events: once `stream` completes, so has all the
 * step's work) computes the next step's evicted sets in every layer, and at that step one
 * launch compacts every layer of the sequences that fire (ordered or order-free,
 * in place) before the first layer runs.  Sets computed ahead are used only
 * where the counters they were computed from still hold; elsewhere the layers
 * select as ra_decode_layer does.
 */
int ra_decode_step(ra_ctx* ctx, const uint16_t* q_all, const uint16_t* k_all, const uint16_t* v_all,
                   uint16_t* out_all, float scale, void* stream);

/*
 * Same computation and result as ra_decode_attn, for callers that cannot supply
 * device scratch memory at call time -- e.g. code that runs while another
 * framework owns all device allocation, or inside a region where cudaMalloc is
 * not allowed.  The split-K partials go to a fixed 8 MiB device array inside
 * this library (one per GPU that loads it, held until the process exits)
 * instead of the bound arena; this call allocates nothing.  (The paper has no
 * counterpart: this is an interface convenience.)
 *   - Layers whose split needs more than 8 MiB of partials (roughly more than
 *     (8 MiB / (G*128*4 B)) warps-plus-heads) are rejected with RA_ERR_CAPACITY.
 *   - The first call on a device looks up the array's device address; make that
 *     first call before any stream capture.
 *   - Every call shares the one array: calls whose work overlaps on the GPU
 *     (different streams, or different contexts on one device) race.  Calls
 *     ordered on one stream are safe; no state is carried between calls.
 */
int ra_decode_attn_noalloc(ra_ctx* ctx, int layer, const uint16_t* q, uint16_t* out, float scale, void* stream);

/* Host-mirrored counters of (seq, layer): generated tokens g, cached generated c, evictions so far. */
int ra_get_counters(const ra_ctx* ctx, int seq, int layer, int32_t* g, int32_t* c, int32_t* n_evictions);

/* Debug: copy the c cached generated positions of (layer, seq, kv_head) to host (synchronises). */
int ra_get_positions(ra_ctx* ctx, int layer, int seq, int kv_head, int32_t* host_pos, int capacity, int* n,
                     void* stream);

/* Debug: copy all rows (prompt, then cached generated) of (layer, seq, kv_head) to host (synchronises). */
int ra_get_kv(ra_ctx* ctx, int layer, int seq, int kv_head, uint16_t* host_k, uint16_t* host_v, int capacity_rows,
              int* n_rows, void* stream);

/*
 * Synchronise `stream` and report what the kernels flagged in the context's device error word:
 * RA_ERR_DEVICE_TIMEOUT if a kernel gave up a bounded wait (every mbarrier wait of the pipelines
 * is bounded at 2 s; the kernel then lets its own copies land, releases what it holds and
 * returns), RA_ERR_STATE if an eviction plan disagreed with the host counters.  The word is
 * cleared once reported, so a later call reports only new events.
 */
int ra_check_device(ra_ctx* ctx, void* stream);

/*
 * Test hook of the device-timeout path: launch one CTA on `stream` that arms an mbarrier for 16
 * bytes of transfer that nothing ever issues, waits on it with its wait bounded at limit_ns
 * nanoseconds (1 000 .. 100 000 000), then flags the timeout in the device error word exactly as
 * the pipeline kernels do, and returns.  It touches no memory but its own shared memory and the
 * error word, so the context stays usable: ra_check_device then returns RA_ERR_DEVICE_TIMEOUT
 * once.  (The paper has no counterpart: failure detection of this library.)
 */
int ra_debug_timeout_probe(ra_ctx* ctx, uint64_t limit_ns, void* stream);

/*
 * Per-kernel accounting.  Launch counts and algorithmic bytes (the bytes each
 * kernel must move by definition: cache rows read, rows moved, q/out rows) are
 * always counted; CUDA-event timing of every launch is recorded only while
 * enabled (ra_profile_enable).  ra_profile_read synchronises on the recorded
 * events and returns the totals of one ra_kernel_kind since the last reset.
 * For the two scoring kinds (RA_KERNEL_SCORE_STATS runs only in
 * ra_restore_queries) the bytes are the key rows read (256 bytes each, every
 * one contracted with the M = r * G window rows: flops = bytes * M).
 */
int ra_profile_enable(ra_ctx* ctx, int on);
int ra_profile_read(ra_ctx* ctx, int kind, double* total_ms, int64_t* launches, double* algorithmic_bytes);
int ra_profile_reset(ra_ctx* ctx);

/* Static message for the last error of ctx (or of the calling thread if ctx is NULL). */
const char* ra_last_error(const ra_ctx* ctx);

/* Release the context (host memory only; the arena stays the caller's). */
void ra_destroy(ra_ctx* ctx);

#ifdef __cplusplus
}
#endif

#endif /* RA_H_ */
