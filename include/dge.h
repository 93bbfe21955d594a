/*
 * dge.h -- C ABI of the Draft-Guided Eviction (DGE) score -> select -> compact
 * pass on one GPU (sm_103a).
 *
 * The paper (Alg. 1) drafts k answer tokens on the full KV cache, then, once
 * per layer and KV head: scores every past position with the observation
 * queries (line B: the k draft queries; DGE-W: the base evictor's window), keeps
 * the per-head budget (retention rule R_E: SnapKV top-B after max-pooling,
 * PyramidKV per-layer budgets, H2O's accumulated attention, StreamingLLM's sinks
 * + recency), and edits the cache keeping temporal order (App. E implementation
 * notes: sort indices, gather [retained past] || [window + draft tail]).
 *
 * Conventions shared by every call:
 *   - Caches are bf16, GQA ("kv_head") layout as in App. G: K, V are indexed
 *     [layer][batch][kv_head][position][d] through the element strides of a
 *     dge_tensor; d is contiguous.  Query rows are [layer][batch][q_head][row][d].
 *     Query head g belongs to KV head g / (Hq / Hkv).
 *   - A "unit" is one (layer, batch, kv_head).  Units are ordered
 *     u = (layer * batch + b) * Hkv + h.
 *   - Positions are int32 in [0, n).  Scored positions of a unit are [0, P) with
 *     P = n - tail.  Scores are float32, [unit][P], contiguous.
 *   - Packed outputs (idx, Kc, Vc) hold budgets[l] rows per unit, units in
 *     order, so unit (l, b, h) starts at row
 *       row_base(l) + (b * Hkv + h) * budgets[l],
 *       row_base(l) = batch * Hkv * (budgets[0] + ... + budgets[l-1]).
 *     Kc, Vc are [rows][d] bf16, contiguous.  idx rows are ascending positions.
 *   - Every device pointer is caller-owned.  The library allocates no device
 *     memory and never synchronises the caller's stream (except
 *     dge_get_device_status and dge_noalloc_status).  It keeps no device state
 *     between calls, with one exception: the fixed scratch array of
 *     dge_score_noalloc, which is part of the library's device image (every GPU
 *     that loads the library holds it until exit).  All work is enqueued on
 *     `stream` (a cudaStream_t passed as void*; NULL = legacy default stream).
 *   - Which scoring kernels run is decided per call from the problem and the
 *     device (tcgen05 kernels where they apply, warp-level kernels otherwise);
 *     the environment variable DGE_SCORE_KERNEL=mma, read on every scoring
 *     call, forces the warp-level kernels (a check of one path against the
 *     other; the results agree within the score tolerance, not bit for bit).
 *   - Outputs must not alias inputs.
 *   - Validation errors are returned before anything is enqueued.  Launch
 *     failures return DGE_ERR_CUDA; dge_last_error() then holds the CUDA error
 *     text for the calling thread.
 */
#ifndef DGE_H
#define DGE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Status codes. */
enum {
    DGE_OK = 0,
    DGE_ERR_INVALID_ARG = 1,         /* null pointer, inconsistent sizes, bad budget */
    DGE_ERR_UNSUPPORTED = 2,         /* head_dim, alignment or size outside what the kernels take */
    DGE_ERR_WORKSPACE_TOO_SMALL = 3, /* ws_bytes below dge_workspace_size() */
    DGE_ERR_CUDA = 4,                /* a CUDA launch or runtime call failed */
    DGE_ERR_DEVICE_TIMEOUT = 5       /* a device-side bounded wait gave up (status word) */
};

/* Scoring variant (Alg. 1 line B and the retention rules of App. L). */
enum {
    DGE_VARIANT_SCORED = 0,    /* SnapKV / PyramidKV / DGE: the caller's m observation rows
                                  per query head, row i at position n - m + i */
    DGE_VARIANT_H2O = 1,       /* H2O accumulator: all n rows, row i at position i, causal */
    DGE_VARIANT_STREAMING = 2  /* StreamingLLM: sinks + recency, no scores */
};

/* Pooling along positions before selection (App. B: max-pool, kernel 7). */
enum {
    DGE_POOL_NONE = 0,
    DGE_POOL_MAX = 1,  /* max over the in-range cells of [j - r, j + r], r = kernel / 2 */
    DGE_POOL_AVG = 2   /* sum over the in-range cells / kernel (zero padding) */
};

/*
 * The eviction problem (Alg. 1 inputs: per-head budget B, draft length k,
 * base evictor E with window w).
 */
typedef struct dge_problem {
    int32_t num_layers;    /* L >= 1 (at most 256) */
    int32_t batch;         /* b >= 1 */
    int32_t num_q_heads;   /* Hq >= 1 */
    int32_t num_kv_heads;  /* Hkv >= 1, divides Hq */
    int32_t head_dim;      /* d: 64 or 128 */
    int32_t obs_rows;      /* SCORED: m = w + k >= 1 rows per query head; ignored otherwise */
    int64_t seq_len;       /* n >= 1, < 2^31: cache length incl. window and draft rows */
    int32_t tail;          /* protected tail [n - tail, n): SCORED t (normally m), H2O the
                              recent window; ignored by STREAMING */
    int32_t sinks;         /* protected head [0, sinks) */
    int32_t variant;       /* DGE_VARIANT_* */
    int32_t pool;          /* DGE_POOL_* (SCORED only; H2O and STREAMING do not pool) */
    int32_t pool_kernel;   /* odd, 1..31, when pool != NONE */
    float scale;           /* logit scale; 0 means 1/sqrt(head_dim) */
    int32_t select_block;  /* 0 (or 1): keep the best positions.  2..64: block-granular
                              selection, the selection ladder's fixed-block rung (Table
                              "Selection decomposition"; sizes 8/16/32 in App. "Diagnostic
                              details"), read as: candidates [sinks, P) in consecutive blocks of
                              this many positions from `sinks` (the last may be shorter), ranked
                              by the sum of their scores (ties: lower block first), taken whole
                              while they fit; the first block that does not fit gives its
                              lowest positions, so the budget is met exactly.  At most 16384
                              blocks per unit.  SCORED and H2O. */
    const int32_t *budgets;/* HOST array [L]: kept rows per unit of layer l, counting the
                              protected sinks and tail: sinks + tail <= budgets[l] <= n
                              (STREAMING: sinks <= budgets[l] <= n) */
} dge_problem;

/* A bf16 tensor in device memory with element strides; d is contiguous.
 * data must be 16-byte aligned and every stride a multiple of 8 elements. */
typedef struct dge_tensor {
    const void *data;
    int64_t stride_layer, stride_batch, stride_head, stride_pos;
} dge_tensor;

/*
 * A paged KV cache (block table), the layout paged-attention serving engines keep (the paper
 * names paged-attention batching as the route to throughput, Sec. "Limitations"): every
 * layer's K (and V) lives in a pool of fixed-size pages, and a sequence's positions are the
 * concatenation of the pages its block table lists.  With paging, the dge_tensor of K and of
 * V describes its pools: data = slot 0 of page 0 of layer 0's pool, stride_layer = elements
 * between the layers' pools, stride_head = between the KV heads of a slot, stride_pos = between
 * the slots of a page (stride_batch is unused); position p of sequence b is slot
 * p % page_size of page block_table[b * pages_per_seq + p / page_size].  K and V share the
 * block table and the page geometry.  Q is never paged.
 *   block_table: device int32 [b][pages_per_seq], 4-byte aligned; the entries covering
 *     positions [0, n) must lie in [0, num_pages) (an entry outside is read as page 0);
 *   page_size: 16, 32 or 64, or a multiple of 128;
 *   pages_per_seq >= ceil(n / page_size); num_pages >= 1 (pages in each layer's pool);
 *   stride_page: elements between pages, a positive multiple of 8.
 * Every call that takes K / V accepts it: scoring reads the pages (one TMA box per page of a
 * 128-key tile), the packed gather reads them, the in-place gather moves row r of every
 * unit to position r of the same sequence's pages (so its first ceil(B / page_size) pages
 * hold the kept cache and the rest can be returned to the pool).
 */
typedef struct dge_paging {
    const int32_t *block_table;
    int32_t page_size;
    int32_t pages_per_seq;
    int32_t num_pages;
    int32_t reserved;     /* 0 */
    int64_t stride_page;
} dge_paging;

/* Inputs and outputs of dge_evict / dge_score. */
typedef struct dge_buffers {
    dge_tensor K;        /* [L][b][Hkv][n][d] */
    dge_tensor V;        /* [L][b][Hkv][n][d] (dge_evict only) */
    dge_tensor Q;        /* [L][b][Hq][m][d] (SCORED) or [L][b][Hq][n][d] (H2O); unused by
                            STREAMING */
    float *scores;       /* [unit][P] final (pooled) scores; required by dge_score, optional
                            (NULL) for dge_evict */
    int32_t *idx;        /* packed kept positions (dge_evict) */
    void *Kc;            /* packed [rows][d] bf16 (dge_evict) */
    void *Vc;            /* packed [rows][d] bf16 (dge_evict) */
    /* Row normalisers, fp32, natural log, dense [L][b][Hq][rows] (rows = m for SCORED, n for
     * H2O), row i of query head h at position pos_i:
     *   lse[l][b][h][i] = log sum_{j <= pos_i} exp(scale * q . k_j)   (scale as in the problem).
     * lse_in (optional): supplied by the caller -- the attention pass that produced the draft
     * (or window) rows already forms this normaliser (flash attention returns it), which is
     * why the paper counts the draft's scores as free (Sec. "Draft-Guided Eviction", phase B;
     * App. "Complexity and overheads").  With lse_in the scoring skips its normaliser pass
     * and reads K once.  The caller vouches for the values: they must be finite, and scores
     * are exp(s - lse) summed as given.
     * lse_out (optional, ignored when lse_in is set): receives the normalisers the scoring
     * computed.  Both 4-byte aligned; NULL to leave unused. */
    const float *lse_in;
    float *lse_out;
    /* K and V as a paged cache (NULL: the [L][b][Hkv][n][d] layout above); see dge_paging. */
    const dge_paging *paging;
} dge_buffers;

/*
 * Bytes of device workspace that dge_score / dge_evict need for this problem
 * (for STREAMING only the 256-byte status region).  The workspace is
 * caller-allocated, 256-byte aligned, and may be reused across calls on the
 * same stream; its contents need no initialisation.  Its first 4 bytes are the
 * device status word: dge_score and dge_evict clear it when they start,
 * device-side checks set it, dge_get_device_status reads and clears it.
 * Returns DGE_OK or DGE_ERR_INVALID_ARG / DGE_ERR_UNSUPPORTED.
 */
int dge_workspace_size(const dge_problem *p, size_t *bytes);

/* Total rows of the packed outputs: batch * Hkv * sum(budgets). */
int dge_packed_rows(const dge_problem *p, int64_t *rows);

/*
 * Scores (Alg. 1 line B; App. B): for every unit, over the stacked rows of its
 * G = Hq / Hkv query heads,
 *   raw[j] = sum_rows exp(s_rj - lse_r),  s_rj = scale * q_r . k_j  (j <= pos_r),
 *   lse_r  = log sum_{j <= pos_r} exp(s_rj),
 * for j in [0, P), then pooled along positions (SCORED only) and written to
 * bufs->scores.  Uses bufs->K, bufs->Q, bufs->scores.  SCORED and H2O only.
 */
int dge_score(const dge_problem *p, const dge_buffers *bufs, void *ws, size_t ws_bytes,
              void *stream);

/*
 * dge_score without a workspace argument and without allocating anything, for
 * callers that are not allowed to allocate device memory: code embedded in a
 * serving runtime that owns the whole device-memory plan and rejects any
 * allocation on its request path, or code that must not call cudaMalloc /
 * cudaFree because those can synchronise the whole device while other streams
 * are running.  The paper has no counterpart; this is a deployment convenience.
 *
 * Scratch is a fixed device array built into the library,
 * DGE_NOALLOC_SCRATCH_BYTES (32 MiB); every GPU that loads the library holds
 * it until the process exits.  A problem whose dge_workspace_size() exceeds it
 * is rejected with DGE_ERR_WORKSPACE_TOO_SMALL before anything is enqueued
 * (dge_last_error() then states both sizes).  The first call on each device
 * looks up the array's device address with that device current, so make that
 * first call before any stream capture.  The address is kept for the life of
 * the process: do not use this call on a device after cudaDeviceReset() (the
 * array may then live elsewhere).  Every call uses the same array and it
 * keeps the previous call's contents (the call itself clears what must start
 * at zero), so calls that can overlap on the GPU -- on different streams or
 * from different host threads -- race; serialise them.  Inputs, outputs and
 * scores are those of dge_score.  Device-side reports (a bounded wait that
 * gave up) land in the status word at the start of the built-in array, which
 * the caller cannot address: read them with dge_noalloc_status before the
 * next dge_score_noalloc call, which clears the word when it starts.
 */
#define DGE_NOALLOC_SCRATCH_BYTES ((size_t)32 << 20)
int dge_score_noalloc(const dge_problem *p, const dge_buffers *bufs, void *stream);

/*
 * The device status word of dge_score_noalloc's built-in array on the current
 * device: synchronises `stream`, reads the word, clears it and returns it, as
 * dge_get_device_status does for a caller's workspace (DGE_OK when nothing
 * was reported).  Returns DGE_ERR_INVALID_ARG if dge_score_noalloc has not run
 * on this device.  Allocates nothing.
 */
int dge_noalloc_status(void *stream);

/*
 * Retention (Alg. 1: I <- R_E(s, B - w); App. E: sort to keep temporal order).
 * Takes no workspace: the selection runs in shared memory and reads the scores
 * from global memory, so it needs no device scratch and reports no
 * device-side status.
 * For every unit keeps [0, sinks), the budgets[l] - sinks - tail positions of
 * [sinks, P) with the largest scores (equal scores: lower position first), and
 * [P, n); writes them ascending to the packed idx.  STREAMING ignores scores
 * (may be NULL) and keeps [0, sinks) and the last budgets[l] - sinks positions.
 */
int dge_select(const dge_problem *p, const float *scores, int32_t *idx, void *stream);

/*
 * Compaction (App. E: gather [retained past] || [window + draft tail]):
 * Kc[r] = K[idx[r]], Vc[r] = V[idx[r]] for every packed row, a bit copy.
 * idx values must lie in [0, n) (out-of-range rows are left unwritten and
 * reported through dge_get_device_status as DGE_ERR_INVALID_ARG when a
 * workspace is given; pass ws = NULL to skip that report).
 */
int dge_compact(const dge_problem *p, const int32_t *idx, const dge_tensor *K,
                const dge_tensor *V, void *Kc, void *Vc, void *ws, void *stream);

/* dge_compact over a paged cache (K, V describe the pools; see dge_paging). */
int dge_compact_paged(const dge_problem *p, const dge_paging *paging, const int32_t *idx,
                      const dge_tensor *K, const dge_tensor *V, void *Kc, void *Vc, void *ws,
                      void *stream);

/*
 * The whole pass, score -> pool -> select -> compact, enqueued on one stream
 * with no host synchronisation.  Writes bufs->idx, Kc, Vc and, when not NULL,
 * bufs->scores.  STREAMING needs no workspace (ws may be NULL).
 */
int dge_evict(const dge_problem *p, const dge_buffers *bufs, void *ws, size_t ws_bytes,
              void *stream);

/*
 * In-place compaction (Alg. 1: each head's cache is edited once, in place, temporal order
 * kept; App. E sorts the kept indices before the gather): rows [0, B_l) of every unit of K
 * and V become the kept rows, in ascending position order; rows [B_l, n) keep their old
 * contents.  K->data and V->data are WRITTEN (the cache the caller decodes from next).
 * idx: packed kept positions as dge_select writes them; each unit's must ascend (then
 * idx[r] >= r and the forward copy is safe).  A position outside [r, n) is skipped and
 * reported in the status word of ws (DGE_ERR_INVALID_ARG; like dge_compact, this call does
 * not clear the word first); ws may be NULL.
 */
int dge_compact_inplace(const dge_problem *p, const int32_t *idx, const dge_tensor *K,
                        const dge_tensor *V, void *ws, void *stream);

/* dge_compact_inplace over a paged cache: row r of every unit moves to position r of the same
 * sequence through the block table (see dge_paging). */
int dge_compact_inplace_paged(const dge_problem *p, const dge_paging *paging, const int32_t *idx,
                              const dge_tensor *K, const dge_tensor *V, void *ws, void *stream);

/*
 * dge_evict with the in-place compaction: score -> pool -> select, then the kept rows move
 * to the front of every unit of bufs->K and bufs->V (their data is WRITTEN).  bufs->Kc and
 * bufs->Vc are ignored; bufs->idx, scores, lse_in and lse_out as for dge_evict.  The scoring
 * finishes before the gather starts (same stream), so the scores see the cache as it was.
 */
int dge_evict_inplace(const dge_problem *p, const dge_buffers *bufs, void *ws, size_t ws_bytes,
                      void *stream);

/*
 * Eviction diagnostics (Sec. "Attention-Mass Analysis"; Eq. evict-mass and Eq. match), SCORED
 * only, for an eviction already done by dge_evict:
 *   evicted_mass [L][b][Hq][m] (required): rho of every observation row, the share of its
 *     softmax (over its visible keys) that falls on evicted keys: 1 - Z_hat / Z, where Z_hat
 *     is the same sum over the retained keys only;
 *   l_match [unit] (optional): the attention-matching loss of Eq. match, the mean over the
 *     unit's rows of log Z - log Z_hat = -log(1 - rho);
 *   run_length [unit] (optional): the mean contiguous run of retained positions,
 *     B_l / (number of maximal runs of consecutive kept positions).
 * Uses bufs->Q, bufs->Kc and bufs->idx as dge_evict wrote them, and bufs->lse_in = the rows'
 * full-cache normalisers (dge_evict's lse_out, or the caller's own); bufs->K and bufs->V only
 * for the held-out queries below.
 * log Z_hat comes from the scoring run on each layer's packed kept keys as a cache of length
 * B_l (the observation rows keep their relative positions), so the observation rows must lie
 * in the protected tail (m <= tail; otherwise DGE_ERR_UNSUPPORTED).  ws: dge_workspace_size(p)
 * bytes.
 */
typedef struct dge_diag {
    float *evicted_mass;
    float *l_match;
    float *run_length;
    /* Optional held-out decode queries (heldout_q.data NULL: skipped): bf16 [L][b][Hq][d]
     * through the tensor's strides (stride_pos unused), one query per head at position n, so
     * it attends over all n keys of bufs->K / bufs->V (the cache before compaction).  With
     * weights a_j = softmax_j(scale q.k_j), kept set R = the head's idx and evicted set E:
     *   heldout_mass [L][b][Hq]: m(E) = sum_{j in E} a_j,
     *   heldout_err  [L][b][Hq]: |o - o~|, o = sum_j a_j v_j, o~ = sum_{j in R} a_j v_j/(1-m),
     *   heldout_gap  [L][b][Hq]: m(E) |mu_E - mu_R| with mu the a-weighted value means over
     *     E and R; Eq. evict-mass says heldout_err equals it exactly.
     * The three outputs are required when heldout_q.data is set. */
    dge_tensor heldout_q;
    float *heldout_mass;
    float *heldout_err;
    float *heldout_gap;
} dge_diag;
int dge_diagnostics(const dge_problem *p, const dge_buffers *bufs, const dge_diag *out,
                    void *ws, size_t ws_bytes, void *stream);

/*
 * PyramidKV's per-layer past budgets (App. L): c = B - w, min = floor(c/20),
 * max = 2c - min, steps = floor((max - min)/(L - 1)), out[l] = max - l*steps.
 * These are past tokens only; add the protected tail to get dge budgets.
 * Host only.  Needs L >= 2 and B > w.
 */
int dge_pyramid_budgets(int32_t B, int32_t w, int32_t L, int32_t *out);

/*
 * Synchronises `stream`, reads the device status word in `ws` (written by
 * bounded device waits and device-side checks), clears it, and returns it
 * (DGE_OK when nothing was reported).
 */
int dge_get_device_status(void *ws, void *stream);

/*
 * Kernel timing (tracing).  Between dge_profile_begin() and dge_profile_end(),
 * every kernel the library enqueues is bracketed by two CUDA events on the
 * call's stream (the GPU's own order is unchanged).  dge_profile_end() waits
 * for those events, then writes up to `capacity` entries, one per kernel
 * name, with the number of launches and their summed device time, and sets
 * *count to the number of distinct kernels.  Host-side state is per process
 * and guarded by a mutex; begin clears it.
 */
typedef struct dge_kernel_time {
    char name[48];
    int64_t launches;
    double total_ms;
} dge_kernel_time;

int dge_profile_begin(void);
int dge_profile_end(dge_kernel_time *out, int capacity, int *count);

/*
 * Cycle accounting of the tensor-core scoring kernel (tracing).  When `buffer`
 * (device memory, caller-owned) is not NULL, every CTA of later launches writes
 * per-role sums of SM clock cycles into it, slot-major: entry
 * slot * DGE_TRACE_LEN + cta.  Slots: 0 MMA waiting for the query block, 1 MMA
 * waiting for key tiles, 2 MMA waiting for a free accumulator, 3 MMA issuing, 4 MMA
 * committing, 5 MMA total, 6 producer waiting for a query buffer, 7 producer waiting
 * for a key stage, 8 producer total, 9 first epilogue warp waiting for accumulators,
 * 10 its phase-2 cycles reading accumulators and adding exponentials, 11 its
 * phase-1 task ends (row-sum hand-off), 12 its phase-2 task starts (waiting for the
 * staged lse), 13 timeline (below), 14 its total, 15 tiles issued.  Timelines hold
 * global-timer stamps (ns).  Slot 13, for CTA `cta` only: entry 4i .. 4i+3 when
 * its coordinator starts staging phase-2 task i, has the buffer, sees every chunk
 * of the unit counted and has staged lse; entry 2048 + 2i / 2i+1 when its first
 * epilogue warp starts / ends waiting for that lse.  Slots 17 .. 19: the first
 * epilogue warp's phase-1 cycles reading accumulators and adding exponentials, its
 * cycles in the phase-2 exchange and in releasing accumulators.  Per-tile timelines of CTA `cta`,
 * entry i for its i-th key tile: slot 16 when the producer issues its copy, 20 when
 * the MMA warp sees it landed, 21 when its accumulator is free, 22 when its MMAs
 * are issued and committed, 23 when the first epilogue warp has the result.  `bytes`
 * must cover the slots;
 * pass NULL to stop.  Host-side state, per process.  Only launches that take a
 * unit's query rows whole are traced; a launch split into row blocks (more stacked
 * rows than one accumulator holds) writes nothing.
 */
#define DGE_TRACE_SLOTS 24
#define DGE_TRACE_LEN 4096
int dge_trace_set(void *buffer, size_t bytes, int cta);

/*
 * Test hook of the device-side failure detection, off by default.  limit_ns
 * bounds every later device-side wait of the tcgen05 kernels (0 restores the
 * default, 4 s).  extra_chunks > 0 makes the tensor-core scoring kernel's wait
 * for a unit's row sums expect that many key chunks more than exist, so the
 * wait can only run out: the kernel then records DGE_ERR_DEVICE_TIMEOUT in the
 * status word, stops, drains its copies and MMAs, frees its tensor memory and
 * returns (results of that call are undefined; the context stays usable).
 * Host-side state, per process; not for production use.
 */
int dge_debug_set_waits(uint64_t limit_ns, int32_t extra_chunks);

/* Static text for a status code. */
const char *dge_status_string(int code);

/* Text of the last CUDA error seen by a call on this thread ("" if none). */
const char *dge_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* DGE_H */
