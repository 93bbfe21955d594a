// dge_api.cu -- the C ABI declared in include/dge.h: argument validation,
// workspace layout and the launch sequence of the score -> select -> compact
// pass.  Host code only; kernels live in score_mma.cu and select_compact.cu.
#include <math.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <map>
#include <mutex>
#include <string>
#include <vector>

#include "common.cuh"
#include "kernels.h"

using namespace dge;

namespace {

thread_local char g_last_error[512] = "";

int cuda_fail(cudaError_t err, const char *where)
{
    snprintf(g_last_error, sizeof g_last_error, "%s: %s (%s)", where, cudaGetErrorName(err),
             cudaGetErrorString(err));
    return DGE_ERR_CUDA;
}

#define DGE_CHECK_CUDA(expr, where)                  \
    do {                                             \
        cudaError_t e_ = (expr);                     \
        if (e_ != cudaSuccess)                       \
            return cuda_fail(e_, where);             \
    } while (0)

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

// ---------------------------------------------------------------------------
// Kernel timing: events around launches while profiling is on.
struct ProfRecord {
    const char *name;
    cudaEvent_t start, stop;
};

struct Profiler {
    std::mutex mu;
    bool on = false;
    std::vector<ProfRecord> records;
    std::vector<cudaEvent_t> pool;

    cudaEvent_t take()
    {
        if (!pool.empty()) {
            cudaEvent_t e = pool.back();
            pool.pop_back();
            return e;
        }
        cudaEvent_t e = nullptr;
        if (cudaEventCreate(&e) != cudaSuccess)
            return nullptr;
        return e;
    }
};

Profiler &profiler()
{
    static Profiler p;
    return p;
}

// Records a start event at construction and a stop event at destruction.
class ProfScope {
  public:
    ProfScope(const char *name, cudaStream_t stream) : name_(name), stream_(stream)
    {
        Profiler &p = profiler();
        std::lock_guard<std::mutex> lk(p.mu);
        if (!p.on)
            return;
        start_ = p.take();
        stop_ = p.take();
        if (start_ && stop_ && cudaEventRecord(start_, stream_) == cudaSuccess)
            active_ = true;
    }
    ~ProfScope()
    {
        if (!active_)
            return;
        Profiler &p = profiler();
        std::lock_guard<std::mutex> lk(p.mu);
        if (cudaEventRecord(stop_, stream_) == cudaSuccess)
            p.records.push_back({name_, start_, stop_});
    }

  private:
    const char *name_;
    cudaStream_t stream_;
    cudaEvent_t start_ = nullptr, stop_ = nullptr;
    bool active_ = false;
};

#define DGE_LAUNCH(name, stream, expr)                                \
    do {                                                              \
        cudaError_t e_;                                               \
        {                                                             \
            ProfScope ps_(name, stream);                              \
            e_ = (expr);                                              \
        }                                                             \
        if (e_ != cudaSuccess)                                        \
            return cuda_fail(e_, name);                               \
    } while (0)

// Work decomposition and workspace layout of one problem.
struct Plan {
    Geometry g;
    LayerTable layers;
    int64_t packed_rows = 0;
    int rows_per_block = 0;  // phase-1 row block (all rows for SCORED)
    int chunk_keys = 0;      // phase-1 key chunk
    int nchunks = 0;
    TcPlan tc = {};          // tensor-core path decomposition (SCORED only)
    size_t off_partial = 0, off_lse = 0, off_raw = 0, off_pooled = 0, off_claim = 0, off_count = 0,
           off_ready = 0, off_rawfx = 0, off_units = 0, off_rpart = 0, ws_bytes = 0;
    size_t flags_clear = 0;  // bytes from off_claim that a tensor-core scoring call zeroes
};

constexpr int kScoredChunkKeys = 2048;
constexpr int kH2ORowBlock = 128;

int make_plan(const dge_problem *p, Plan &plan)
{
    if (!p || !p->budgets)
        return DGE_ERR_INVALID_ARG;
    const int64_t n = p->seq_len;
    if (p->num_layers < 1 || p->num_layers > kMaxLayers || p->batch < 1 || p->num_q_heads < 1 ||
        p->num_kv_heads < 1 || p->num_q_heads % p->num_kv_heads != 0 || n < 1 ||
        n >= (int64_t)INT32_MAX || p->sinks < 0 || p->sinks > n)
        return DGE_ERR_INVALID_ARG;
    if (p->variant != DGE_VARIANT_SCORED && p->variant != DGE_VARIANT_H2O &&
        p->variant != DGE_VARIANT_STREAMING)
        return DGE_ERR_INVALID_ARG;
    if (p->head_dim != 64 && p->head_dim != 128)
        return DGE_ERR_UNSUPPORTED;
    if (!isfinite(p->scale))
        return DGE_ERR_INVALID_ARG;

    Geometry &g = plan.g;
    memset(&g, 0, sizeof g);
    g.L = p->num_layers;
    g.b = p->batch;
    g.Hq = p->num_q_heads;
    g.Hkv = p->num_kv_heads;
    g.G = g.Hq / g.Hkv;
    g.d = p->head_dim;
    g.n = (int)n;
    g.sinks = p->sinks;
    g.variant = p->variant;
    g.pool = DGE_POOL_NONE;
    g.pool_kernel = 1;
    g.U = (int64_t)g.L * g.b * g.Hkv;
    const float scale = p->scale != 0.f ? p->scale : 1.f / sqrtf((float)g.d);
    g.scale_log2 = scale * 1.4426950408889634f;

    if (p->variant == DGE_VARIANT_STREAMING) {
        g.tail = 0;
        g.P = g.n;
        g.m = 0;
        g.R = 0;
    } else {
        if (p->tail < 0 || (int64_t)p->tail + p->sinks > n)
            return DGE_ERR_INVALID_ARG;
        g.tail = p->tail;
        g.P = g.n - g.tail;
        if (p->variant == DGE_VARIANT_SCORED) {
            if (p->obs_rows < 1 || p->obs_rows > n)
                return DGE_ERR_INVALID_ARG;
            g.m = p->obs_rows;
            if ((int64_t)g.G * g.m > kMaxRows)
                return DGE_ERR_UNSUPPORTED;
            g.R = g.G * g.m;
            if (p->pool != DGE_POOL_NONE && p->pool != DGE_POOL_MAX && p->pool != DGE_POOL_AVG)
                return DGE_ERR_INVALID_ARG;
            if (p->pool != DGE_POOL_NONE &&
                (p->pool_kernel < 1 || p->pool_kernel > 31 || p->pool_kernel % 2 == 0))
                return DGE_ERR_INVALID_ARG;
            g.pool = p->pool;
            g.pool_kernel = p->pool == DGE_POOL_NONE ? 1 : p->pool_kernel;
        } else {
            g.m = 0;
            if ((int64_t)g.G * n >= (int64_t)INT32_MAX)
                return DGE_ERR_UNSUPPORTED;
            g.R = (int)(g.G * n);
        }
    }

    g.select_block = 0;
    if (p->variant != DGE_VARIANT_STREAMING) {
        if (p->select_block < 0 || p->select_block > kMaxSelectBlock)
            return DGE_ERR_INVALID_ARG;
        if (p->select_block >= 2) {
            const int64_t C = (int64_t)g.P - g.sinks;
            if ((C + p->select_block - 1) / p->select_block > kMaxSelectBlocks)
                return DGE_ERR_UNSUPPORTED;
            g.select_block = p->select_block;
        }
    }

    int64_t acc = 0;
    for (int l = 0; l < g.L; ++l) {
        const int32_t B = p->budgets[l];
        const int64_t lo = (p->variant == DGE_VARIANT_STREAMING) ? g.sinks
                                                                 : (int64_t)g.sinks + g.tail;
        if (B < lo || B > n)
            return DGE_ERR_INVALID_ARG;
        plan.layers.budget[l] = B;
        plan.layers.row_base[l] = acc;
        acc += (int64_t)g.b * g.Hkv * B;
    }
    plan.packed_rows = acc;

    if (p->variant == DGE_VARIANT_SCORED) {
        plan.rows_per_block = g.R;
        plan.chunk_keys = kScoredChunkKeys;
    } else if (p->variant == DGE_VARIANT_H2O) {
        plan.rows_per_block = kH2ORowBlock;
        plan.chunk_keys = g.n;
    }
    size_t off = kStatusBytes;
    if (p->variant != DGE_VARIANT_STREAMING) {
        plan.nchunks = (g.n + plan.chunk_keys - 1) / plan.chunk_keys;
        // The partial region serves both scoring paths (the larger of the two layouts).
        size_t part_bytes = (size_t)g.U * g.R * plan.nchunks * sizeof(float2);
        int nrb = 1;
        if (p->variant == DGE_VARIANT_SCORED) {
            plan.tc = tc_plan(g);
            nrb = plan.tc.nrb;
            const size_t tc_bytes =
                (size_t)g.U * nrb * plan.tc.r4 * plan.tc.nparts * sizeof(float);
            if (tc_bytes > part_bytes)
                part_bytes = tc_bytes;
        }
        plan.off_partial = off;
        off = align256(off + part_bytes);
        plan.off_lse = off;
        off = align256(off + (size_t)g.U * g.R * sizeof(float));
        plan.off_raw = off;
        off = align256(off + (size_t)g.U * g.P * sizeof(float));
        plan.off_pooled = off;
        if (g.pool != DGE_POOL_NONE)
            off = align256(off + (size_t)g.U * g.P * sizeof(float));
        // Flags, one region: the task claim counter (tensor-core path; 16 bytes), chunk
        // counters [U*nrb], per-unit range flags [U], then the list of units to recompute
        // ([0] = count, [1 ..] = ids).  Everything up to the list count is zeroed with one
        // memset before a scoring launch.
        plan.off_claim = off;
        plan.off_count = off + 16;
        plan.off_ready = plan.off_count + (size_t)g.U * nrb * sizeof(uint32_t);
        plan.off_units = plan.off_ready + (size_t)g.U * sizeof(uint32_t);
        plan.flags_clear = plan.off_units + sizeof(uint32_t) - plan.off_claim;
        off = align256(plan.off_units + (size_t)(g.U + 1) * sizeof(uint32_t));
        if (nrb > 1) {
            // Row blocks of one unit add their column sums in fixed point (exact, so the
            // order of the additions does not matter).
            plan.off_rawfx = off;
            off = align256(off + (size_t)g.U * g.P * sizeof(unsigned long long));
        }
        if (p->variant == DGE_VARIANT_SCORED) {
            // Row partials of the units recomputed with running maxima ([U][R] float2): apart
            // from the tensor-core chunk sums, which the normaliser export still reads.
            plan.off_rpart = off;
            off = align256(off + (size_t)g.U * g.R * sizeof(float2));
        }
    }
    plan.ws_bytes = off;
    return DGE_OK;
}

int check_tensor(const dge_tensor &t)
{
    if (!t.data)
        return DGE_ERR_INVALID_ARG;
    if (((uintptr_t)t.data & 15) != 0)
        return DGE_ERR_UNSUPPORTED;
    if (t.stride_layer < 0 || t.stride_batch < 0 || t.stride_head < 0 || t.stride_pos < 0)
        return DGE_ERR_INVALID_ARG;
    if ((t.stride_layer | t.stride_batch | t.stride_head | t.stride_pos) & 7)
        return DGE_ERR_UNSUPPORTED;
    return DGE_OK;
}

TensorDesc desc(const dge_tensor &t)
{
    TensorDesc d;
    d.data = static_cast<const __nv_bfloat16 *>(t.data);
    d.s_layer = t.stride_layer;
    d.s_batch = t.stride_batch;
    d.s_head = t.stride_head;
    d.s_pos = t.stride_pos;
    return d;
}

// A paged cache's geometry (NULL: contiguous).  page_size: 16, 32, 64 or a multiple of 128,
// so a 128-key tile spans at most 8 pages and every TMA box starts 1024-byte aligned.
int check_paging(const dge_paging *pg, int64_t n)
{
    if (!pg)
        return DGE_OK;
    if (!pg->block_table || pg->num_pages < 1 || pg->stride_page <= 0 || pg->reserved != 0)
        return DGE_ERR_INVALID_ARG;
    const int ps = pg->page_size;
    if (!(ps == 16 || ps == 32 || ps == 64 || (ps >= 128 && ps % 128 == 0)))
        return DGE_ERR_UNSUPPORTED;
    if ((int64_t)pg->pages_per_seq * ps < n)
        return DGE_ERR_INVALID_ARG;
    if (((uintptr_t)pg->block_table & 3) || (pg->stride_page & 7))
        return DGE_ERR_UNSUPPORTED;
    return DGE_OK;
}

// K or V, contiguous or paged.
TensorDesc kv_desc(const dge_tensor &t, const dge_paging *pg)
{
    TensorDesc d = desc(t);
    if (pg) {
        d.bt = pg->block_table;
        d.page_size = pg->page_size;
        d.pps = pg->pages_per_seq;
        d.num_pages = pg->num_pages;
        d.s_page = pg->stride_page;
        d.s_batch = 0;
    }
    return d;
}

int check_ws(const Plan &plan, void *ws, size_t ws_bytes)
{
    if (!ws)
        return DGE_ERR_INVALID_ARG;
    if (((uintptr_t)ws & 255) != 0)
        return DGE_ERR_UNSUPPORTED;
    if (ws_bytes < plan.ws_bytes)
        return DGE_ERR_WORKSPACE_TOO_SMALL;
    return DGE_OK;
}

template <typename T>
T *ws_at(void *ws, size_t off)
{
    return reinterpret_cast<T *>(static_cast<uint8_t *>(ws) + off);
}

// Which scoring kernels to use: the tcgen05 path when the problem and device allow it,
// unless DGE_SCORE_KERNEL=mma asks for the warp-level path.
bool want_tc(const Geometry &g)
{
    const char *env = getenv("DGE_SCORE_KERNEL");
    if (env && strcmp(env, "mma") == 0)
        return false;
    return g.variant == DGE_VARIANT_H2O ? h2o_tc_supported(g) : tc_supported(g);
}

// H2O on the tensor cores: phase 1 (unless the normalisers are supplied: lse2 already holds
// them), phase 2, then the warp-level kernels for units whose row sums left fp32's range.
// False when the tensors cannot be described to TMA (nothing launched: use the warp path).
int run_h2o_tc(const Plan &plan, const TensorDesc &K, const TensorDesc &Q, void *ws,
               cudaStream_t stream, bool supplied, float *lse_out, bool *done)
{
    const Geometry &g = plan.g;
    const H2oPlan hp = h2o_tc_plan(g);
    float2 *partial = ws_at<float2>(ws, plan.off_partial);
    float *lse2 = ws_at<float>(ws, plan.off_lse);
    float *raw = ws_at<float>(ws, plan.off_raw);
    uint32_t *ready = ws_at<uint32_t>(ws, plan.off_ready);
    uint32_t *status = static_cast<uint32_t *>(ws);
    bool encoded = false;
    *done = false;
    if (!supplied) {
        DGE_CHECK_CUDA(cudaMemsetAsync(ready, 0, (size_t)g.U * sizeof(uint32_t), stream),
                       "flag clear");
        DGE_LAUNCH("h2o_tc_lse", stream,
                   launch_h2o_tc(1, K, Q, g, hp, lse2, raw, ready, status, stream, &encoded));
        if (!encoded)
            return DGE_OK;
    }
    DGE_LAUNCH("h2o_tc_colsum", stream,
               launch_h2o_tc(2, K, Q, g, hp, lse2, raw, ready, status, stream, &encoded));
    if (!encoded)
        return DGE_OK;
    *done = true;
    if (supplied)
        return DGE_OK;
    // Every row of every unit is a query row here, so the per-unit grids are large: the
    // recompute runs over a device-side list of the flagged units (usually empty).
    UnitSel units;
    units.sel = ws_at<uint32_t>(ws, plan.off_units);
    units.list = true;
    DGE_LAUNCH("recompute_list", stream,
               launch_collect_units(ready, g.U, ws_at<uint32_t>(ws, plan.off_units), stream));
    DGE_LAUNCH("recompute_lse", stream,
               launch_lse_partial(K, Q, g, plan.rows_per_block, plan.chunk_keys, partial, stream,
                                  units));
    DGE_LAUNCH("recompute_combine", stream,
               launch_combine_lse(partial, g.U * g.R, plan.nchunks, lse2, stream, units, g.R));
    DGE_LAUNCH("recompute_colsum", stream,
               launch_colsum_keys(K, Q, g, lse2, raw, stream, units));
    if (lse_out)
        DGE_LAUNCH("lse_export", stream,
                   launch_lse_export(nullptr, 0, 0, 0, lse2, nullptr, g.U, g.R, g.R, lse_out,
                                     stream));
    return DGE_OK;
}

// raw scores of every unit into the workspace.  lse_in (nullable): the caller's natural-log
// row normalisers, so only the column-sum pass runs; lse_out (nullable, ignored with lse_in):
// receives the normalisers computed here.
int run_scoring(const Plan &plan, const TensorDesc &K, const TensorDesc &Q, void *ws,
                cudaStream_t stream, const float *lse_in, float *lse_out)
{
    const Geometry &g = plan.g;
    float2 *partial = ws_at<float2>(ws, plan.off_partial);
    float *lse2 = ws_at<float>(ws, plan.off_lse);
    float *raw = ws_at<float>(ws, plan.off_raw);
    if (lse_in) {
        if (g.variant == DGE_VARIANT_SCORED && want_tc(g)) {
            TcBuffers tb;
            tb.part = nullptr;
            tb.lse2 = lse2;
            tb.raw = raw;
            tb.count = nullptr;
            tb.ready = nullptr;
            tb.status = static_cast<uint32_t *>(ws);
            tb.lse_in = lse_in;
            tb.claim = ws_at<uint32_t>(ws, plan.off_claim);
            DGE_CHECK_CUDA(cudaMemsetAsync(tb.claim, 0, sizeof(uint32_t), stream), "claim clear");
            unsigned long long *raw_fx = nullptr;
            if (plan.tc.nrb > 1) {
                raw_fx = ws_at<unsigned long long>(ws, plan.off_rawfx);
                DGE_CHECK_CUDA(cudaMemsetAsync(raw_fx, 0, (size_t)g.U * g.P * 8, stream),
                               "sum clear");
                tb.raw_fx = raw_fx;
            }
            bool encoded = false;
            DGE_LAUNCH("score_tc_lse", stream,
                       launch_score_tc(K, Q, g, plan.tc, tb, stream, &encoded));
            if (encoded) {
                if (raw_fx)
                    DGE_LAUNCH("fixed_to_float", stream,
                               launch_fixed_to_float(raw_fx, raw, g.U * g.P, stream));
                return DGE_OK;
            }
        }
        DGE_LAUNCH("lse_import", stream, launch_lse_import(lse_in, lse2, g.U * g.R, stream));
        if (g.variant == DGE_VARIANT_H2O && want_tc(g)) {
            bool done = false;
            const int rc = run_h2o_tc(plan, K, Q, ws, stream, true, nullptr, &done);
            if (rc != DGE_OK || done)
                return rc;
        }
        if (g.variant == DGE_VARIANT_H2O)
            DGE_LAUNCH("colsum_keys", stream, launch_colsum_keys(K, Q, g, lse2, raw, stream));
        else
            DGE_LAUNCH("colsum_rows", stream,
                       launch_colsum_rows(K, Q, g, kScoredChunkKeys, lse2, raw, stream));
        return DGE_OK;
    }
    if (g.variant == DGE_VARIANT_SCORED && want_tc(g)) {
        DGE_CHECK_CUDA(cudaMemsetAsync(ws_at<uint8_t>(ws, plan.off_claim), 0, plan.flags_clear,
                                       stream),
                       "flag clear");
        TcBuffers tb;
        tb.claim = ws_at<uint32_t>(ws, plan.off_claim);
        tb.part = reinterpret_cast<float *>(partial);
        tb.lse2 = lse2;
        tb.raw = raw;
        tb.count = ws_at<uint32_t>(ws, plan.off_count);
        tb.ready = ws_at<uint32_t>(ws, plan.off_ready);
        tb.list = ws_at<uint32_t>(ws, plan.off_units);
        tb.status = static_cast<uint32_t *>(ws);
        const int nrb = plan.tc.nrb;
        unsigned long long *raw_fx = nullptr;
        if (nrb > 1) {
            raw_fx = ws_at<unsigned long long>(ws, plan.off_rawfx);
            DGE_CHECK_CUDA(cudaMemsetAsync(raw_fx, 0, (size_t)g.U * g.P * 8, stream),
                           "sum clear");
            tb.raw_fx = raw_fx;
        }
        // The observation rows' own positions (causally masked), as the last chunk-sum slot;
        // the main kernel covers the keys every row sees.
        DGE_LAUNCH("score_tail", stream,
                   launch_tail_rows(K, Q, g, plan.tc.rows, nrb, tb.part, plan.tc.nparts,
                                    plan.tc.nchunks, plan.tc.r4, stream));
        bool encoded = false;
        DGE_LAUNCH("score_tc", stream,
                   launch_score_tc(K, Q, g, plan.tc, tb, stream, &encoded));
        if (encoded) {
            if (nrb > 1)
                DGE_LAUNCH("fixed_to_float", stream,
                           launch_fixed_to_float(raw_fx, raw, g.U * g.P, stream));
            // Units whose row sums left fp32's safe range were listed by the kernel; one CTA
            // per listed unit recomputes it with running maxima (an empty list: one read).
            DGE_LAUNCH("recompute", stream,
                       launch_recompute_units(K, Q, g, ws_at<float2>(ws, plan.off_rpart), lse2,
                                              raw, tb.list, stream));
            if (lse_out)
                DGE_LAUNCH("lse_export", stream,
                           launch_lse_export(tb.part, plan.tc.nparts, plan.tc.p1_chunks,
                                             plan.tc.r4, lse2,
                                             tb.ready, g.U, g.R, plan.tc.rows, lse_out, stream));
            return DGE_OK;
        }
    }
    if (g.variant == DGE_VARIANT_H2O && want_tc(g)) {
        bool done = false;
        const int rc = run_h2o_tc(plan, K, Q, ws, stream, false, lse_out, &done);
        if (rc != DGE_OK || done)
            return rc;
    }
    DGE_LAUNCH("lse_partial", stream,
               launch_lse_partial(K, Q, g, plan.rows_per_block, plan.chunk_keys, partial, stream));
    DGE_LAUNCH("combine_lse", stream,
               launch_combine_lse(partial, g.U * g.R, plan.nchunks, lse2, stream));
    if (g.variant == DGE_VARIANT_H2O)
        DGE_LAUNCH("colsum_keys", stream, launch_colsum_keys(K, Q, g, lse2, raw, stream));
    else
        DGE_LAUNCH("colsum_rows", stream,
                   launch_colsum_rows(K, Q, g, kScoredChunkKeys, lse2, raw, stream));
    if (lse_out)
        DGE_LAUNCH("lse_export", stream,
                   launch_lse_export(nullptr, 0, 0, 0, lse2, nullptr, g.U, g.R, g.R, lse_out,
                                     stream));
    return DGE_OK;
}

// Row normaliser pointers: 4-byte aligned or NULL.
bool lse_ptrs_ok(const dge_buffers *bufs)
{
    return ((uintptr_t)bufs->lse_in & 3) == 0 && ((uintptr_t)bufs->lse_out & 3) == 0;
}

}  // namespace

void dge::record_error_text(const char *text)
{
    snprintf(g_last_error, sizeof g_last_error, "%s", text);
}

extern "C" {

int dge_workspace_size(const dge_problem *p, size_t *bytes)
{
    if (!bytes)
        return DGE_ERR_INVALID_ARG;
    Plan plan;
    const int rc = make_plan(p, plan);
    if (rc != DGE_OK)
        return rc;
    *bytes = plan.ws_bytes;
    return DGE_OK;
}

int dge_packed_rows(const dge_problem *p, int64_t *rows)
{
    if (!rows)
        return DGE_ERR_INVALID_ARG;
    Plan plan;
    const int rc = make_plan(p, plan);
    if (rc != DGE_OK)
        return rc;
    *rows = plan.packed_rows;
    return DGE_OK;
}

int dge_score(const dge_problem *p, const dge_buffers *bufs, void *ws, size_t ws_bytes,
              void *stream_)
{
    Plan plan;
    int rc = make_plan(p, plan);
    if (rc != DGE_OK)
        return rc;
    if (plan.g.variant == DGE_VARIANT_STREAMING || !bufs || !bufs->scores)
        return DGE_ERR_INVALID_ARG;
    if ((rc = check_tensor(bufs->K)) != DGE_OK || (rc = check_tensor(bufs->Q)) != DGE_OK ||
        (rc = check_paging(bufs->paging, plan.g.n)) != DGE_OK ||
        (rc = check_ws(plan, ws, ws_bytes)) != DGE_OK)
        return rc;
    if (((uintptr_t)bufs->scores & 3) != 0 || !lse_ptrs_ok(bufs))
        return DGE_ERR_UNSUPPORTED;
    cudaStream_t stream = static_cast<cudaStream_t>(stream_);
    DGE_CHECK_CUDA(cudaMemsetAsync(ws, 0, sizeof(uint32_t), stream), "status clear");
    if ((rc = run_scoring(plan, kv_desc(bufs->K, bufs->paging), desc(bufs->Q), ws, stream,
                          bufs->lse_in, bufs->lse_out)) != DGE_OK)
        return rc;
    DGE_LAUNCH("pool", stream,
               launch_pool(ws_at<float>(ws, plan.off_raw), bufs->scores, plan.g.U, plan.g.P,
                           plan.g.pool, plan.g.pool_kernel, stream));
    return DGE_OK;
}

int dge_select(const dge_problem *p, const float *scores, int32_t *idx, void *stream_)
{
    Plan plan;
    const int rc = make_plan(p, plan);
    if (rc != DGE_OK)
        return rc;
    if (!idx || ((uintptr_t)idx & 3) != 0)
        return DGE_ERR_INVALID_ARG;
    cudaStream_t stream = static_cast<cudaStream_t>(stream_);
    if (plan.g.variant == DGE_VARIANT_STREAMING) {
        DGE_LAUNCH("streaming", stream, launch_streaming_indices(plan.g, plan.layers, idx, stream));
        return DGE_OK;
    }
    if (!scores || ((uintptr_t)scores & 3) != 0)
        return DGE_ERR_INVALID_ARG;
    if (plan.g.select_block >= 2)
        DGE_LAUNCH("block_select", stream,
                   launch_block_select(plan.g, plan.layers, scores, idx, stream));
    else
        DGE_LAUNCH("select", stream, launch_select(plan.g, plan.layers, scores, idx, stream));
    return DGE_OK;
}

int dge_compact_paged(const dge_problem *p, const dge_paging *paging, const int32_t *idx,
                      const dge_tensor *K, const dge_tensor *V, void *Kc, void *Vc, void *ws,
                      void *stream_)
{
    Plan plan;
    int rc = make_plan(p, plan);
    if (rc != DGE_OK)
        return rc;
    if (!idx || !K || !V || !Kc || !Vc)
        return DGE_ERR_INVALID_ARG;
    if ((rc = check_tensor(*K)) != DGE_OK || (rc = check_tensor(*V)) != DGE_OK ||
        (rc = check_paging(paging, plan.g.n)) != DGE_OK)
        return rc;
    if (((uintptr_t)Kc & 15) || ((uintptr_t)Vc & 15) || ((uintptr_t)idx & 3) ||
        ((uintptr_t)ws & 255))
        return DGE_ERR_UNSUPPORTED;
    cudaStream_t stream = static_cast<cudaStream_t>(stream_);
    DGE_LAUNCH("compact", stream,
               launch_compact(plan.g, plan.layers, idx, nullptr, kv_desc(*K, paging),
                              kv_desc(*V, paging), Kc, Vc, false, static_cast<uint32_t *>(ws),
                              stream));
    return DGE_OK;
}

int dge_compact(const dge_problem *p, const int32_t *idx, const dge_tensor *K,
                const dge_tensor *V, void *Kc, void *Vc, void *ws, void *stream)
{
    return dge_compact_paged(p, nullptr, idx, K, V, Kc, Vc, ws, stream);
}

}  // extern "C"

namespace {

// dge_evict and dge_evict_inplace: validation, scores, selection, then the gather into the
// packed outputs or into the cache itself.
int evict_impl(const dge_problem *p, const dge_buffers *bufs, void *ws, size_t ws_bytes,
               void *stream_, bool inplace)
{
    Plan plan;
    int rc = make_plan(p, plan);
    if (rc != DGE_OK)
        return rc;
    if (!bufs || !bufs->idx || (!inplace && (!bufs->Kc || !bufs->Vc)))
        return DGE_ERR_INVALID_ARG;
    if ((rc = check_tensor(bufs->K)) != DGE_OK || (rc = check_tensor(bufs->V)) != DGE_OK ||
        (rc = check_paging(bufs->paging, plan.g.n)) != DGE_OK)
        return rc;
    if ((!inplace && (((uintptr_t)bufs->Kc & 15) || ((uintptr_t)bufs->Vc & 15))) ||
        ((uintptr_t)bufs->idx & 3) || ((uintptr_t)bufs->scores & 3) || !lse_ptrs_ok(bufs))
        return DGE_ERR_UNSUPPORTED;
    const Geometry &g = plan.g;
    cudaStream_t stream = static_cast<cudaStream_t>(stream_);
    const TensorDesc K = kv_desc(bufs->K, bufs->paging), V = kv_desc(bufs->V, bufs->paging);
    uint32_t *status = static_cast<uint32_t *>(ws);
    if (g.variant == DGE_VARIANT_STREAMING) {
        if (ws && ((uintptr_t)ws & 255))
            return DGE_ERR_UNSUPPORTED;
        if (ws)
            DGE_CHECK_CUDA(cudaMemsetAsync(ws, 0, sizeof(uint32_t), stream), "status clear");
        if (inplace)
            DGE_LAUNCH("compact_inplace", stream,
                       launch_compact_inplace(g, plan.layers, nullptr, bufs->idx, K, V, true,
                                              status, stream));
        else
            DGE_LAUNCH("compact", stream,
                       launch_compact(g, plan.layers, nullptr, bufs->idx, K, V, bufs->Kc,
                                      bufs->Vc, true, status, stream));
        return DGE_OK;
    }
    if ((rc = check_tensor(bufs->Q)) != DGE_OK || (rc = check_ws(plan, ws, ws_bytes)) != DGE_OK)
        return rc;
    DGE_CHECK_CUDA(cudaMemsetAsync(ws, 0, sizeof(uint32_t), stream), "status clear");
    const TensorDesc Q = desc(bufs->Q);
    if ((rc = run_scoring(plan, K, Q, ws, stream, bufs->lse_in, bufs->lse_out)) != DGE_OK)
        return rc;
    float *raw = ws_at<float>(ws, plan.off_raw);
    const float *sel = raw;
    const bool fused = g.select_block < 2 && pool_select_supported(g);
    const bool fused_large = !fused && g.select_block < 2 && pool_select_large_supported(g);
    if (fused) {
        DGE_LAUNCH("pool_select", stream,
                   launch_pool_select(g, plan.layers, raw, bufs->scores, bufs->idx, stream));
    } else if (fused_large) {
        float *pooled = bufs->scores ? bufs->scores : ws_at<float>(ws, plan.off_pooled);
        DGE_LAUNCH("pool_select", stream,
                   launch_pool_select_large(g, plan.layers, raw, pooled, bufs->idx, stream));
    } else if (g.pool != DGE_POOL_NONE) {
        float *pooled = bufs->scores ? bufs->scores : ws_at<float>(ws, plan.off_pooled);
        DGE_LAUNCH("pool", stream,
                   launch_pool(raw, pooled, g.U, g.P, g.pool, g.pool_kernel, stream));
        sel = pooled;
    } else if (bufs->scores) {
        DGE_CHECK_CUDA(cudaMemcpyAsync(bufs->scores, raw, (size_t)g.U * g.P * sizeof(float),
                                       cudaMemcpyDeviceToDevice, stream),
                       "scores copy");
    }
    if (g.select_block >= 2)
        DGE_LAUNCH("block_select", stream,
                   launch_block_select(g, plan.layers, sel, bufs->idx, stream));
    else if (!fused && !fused_large)
        DGE_LAUNCH("select", stream, launch_select(g, plan.layers, sel, bufs->idx, stream));
    if (inplace)
        DGE_LAUNCH("compact_inplace", stream,
                   launch_compact_inplace(g, plan.layers, bufs->idx, nullptr, K, V, false, status,
                                          stream));
    else
        DGE_LAUNCH("compact", stream,
                   launch_compact(g, plan.layers, bufs->idx, nullptr, K, V, bufs->Kc, bufs->Vc,
                                  false, status, stream));
    return DGE_OK;
}

}  // namespace

extern "C" {

int dge_evict(const dge_problem *p, const dge_buffers *bufs, void *ws, size_t ws_bytes,
              void *stream)
{
    return evict_impl(p, bufs, ws, ws_bytes, stream, false);
}

int dge_evict_inplace(const dge_problem *p, const dge_buffers *bufs, void *ws, size_t ws_bytes,
                      void *stream)
{
    return evict_impl(p, bufs, ws, ws_bytes, stream, true);
}

int dge_diagnostics(const dge_problem *p, const dge_buffers *bufs, const dge_diag *out,
                    void *ws, size_t ws_bytes, void *stream_)
{
    Plan plan;
    int rc = make_plan(p, plan);
    if (rc != DGE_OK)
        return rc;
    const Geometry &g = plan.g;
    if (g.variant != DGE_VARIANT_SCORED || !bufs || !out || !out->evicted_mass || !bufs->Kc ||
        !bufs->idx || !bufs->lse_in)
        return DGE_ERR_INVALID_ARG;
    // The observation rows must lie in the protected tail, so that they are the last m rows of
    // every layer's kept cache.
    if (g.m > g.tail)
        return DGE_ERR_UNSUPPORTED;
    if ((rc = check_tensor(bufs->Q)) != DGE_OK || (rc = check_ws(plan, ws, ws_bytes)) != DGE_OK)
        return rc;
    if (((uintptr_t)bufs->Kc & 15) || ((uintptr_t)bufs->idx & 3) ||
        ((uintptr_t)bufs->lse_in & 3) || ((uintptr_t)out->evicted_mass & 3) ||
        ((uintptr_t)out->l_match & 3) || ((uintptr_t)out->run_length & 3))
        return DGE_ERR_UNSUPPORTED;
    if (out->heldout_q.data) {
        if (!out->heldout_mass || !out->heldout_err || !out->heldout_gap)
            return DGE_ERR_INVALID_ARG;
        if ((rc = check_tensor(out->heldout_q)) != DGE_OK ||
            (rc = check_tensor(bufs->K)) != DGE_OK || (rc = check_tensor(bufs->V)) != DGE_OK ||
            (rc = check_paging(bufs->paging, g.n)) != DGE_OK)
            return rc;
        if (((uintptr_t)out->heldout_mass & 3) || ((uintptr_t)out->heldout_err & 3) ||
            ((uintptr_t)out->heldout_gap & 3) || !heldout_supported(g))
            return DGE_ERR_UNSUPPORTED;
    }
    // Each layer's kept keys as a cache of its own: n' = B_l rows, every one kept.
    Plan sub[kMaxLayers];
    for (int l = 0; l < g.L; ++l) {
        dge_problem q = *p;
        const int32_t B = plan.layers.budget[l];
        q.num_layers = 1;
        q.seq_len = B;
        q.budgets = &plan.layers.budget[l];
        q.pool = DGE_POOL_NONE;
        q.pool_kernel = 1;
        if ((rc = make_plan(&q, sub[l])) != DGE_OK)
            return rc;
        if (sub[l].ws_bytes > ws_bytes)
            return DGE_ERR_WORKSPACE_TOO_SMALL;
    }
    cudaStream_t stream = static_cast<cudaStream_t>(stream_);
    DGE_CHECK_CUDA(cudaMemsetAsync(ws, 0, sizeof(uint32_t), stream), "status clear");
    const int64_t rows_per_layer = (int64_t)g.b * g.Hkv * g.R;  // lse entries of one layer
    for (int l = 0; l < g.L; ++l) {
        const int64_t B = plan.layers.budget[l];
        dge_tensor kl;
        kl.data = static_cast<const __nv_bfloat16 *>(bufs->Kc) + plan.layers.row_base[l] * g.d;
        kl.stride_pos = g.d;
        kl.stride_head = B * g.d;
        kl.stride_batch = (int64_t)g.Hkv * B * g.d;
        kl.stride_layer = (int64_t)g.b * g.Hkv * B * g.d;
        TensorDesc Ql = desc(bufs->Q);
        Ql.data += (int64_t)l * bufs->Q.stride_layer;
        if ((rc = run_scoring(sub[l], desc(kl), Ql, ws, stream, nullptr,
                              out->evicted_mass + (int64_t)l * rows_per_layer)) != DGE_OK)
            return rc;
    }
    DGE_LAUNCH("diagnostics", stream,
               launch_diag(bufs->lse_in, out->evicted_mass, bufs->idx, g, plan.layers,
                           out->l_match, out->run_length, stream));
    if (out->heldout_q.data)
        DGE_LAUNCH("heldout", stream,
                   launch_heldout(desc(out->heldout_q), kv_desc(bufs->K, bufs->paging),
                                  kv_desc(bufs->V, bufs->paging), bufs->idx,
                                  g, plan.layers, out->heldout_mass, out->heldout_err,
                                  out->heldout_gap, stream));
    return DGE_OK;
}

int dge_compact_inplace_paged(const dge_problem *p, const dge_paging *paging, const int32_t *idx,
                              const dge_tensor *K, const dge_tensor *V, void *ws, void *stream_)
{
    Plan plan;
    int rc = make_plan(p, plan);
    if (rc != DGE_OK)
        return rc;
    if (!idx || !K || !V)
        return DGE_ERR_INVALID_ARG;
    if ((rc = check_tensor(*K)) != DGE_OK || (rc = check_tensor(*V)) != DGE_OK ||
        (rc = check_paging(paging, plan.g.n)) != DGE_OK)
        return rc;
    if (((uintptr_t)idx & 3) || ((uintptr_t)ws & 255))
        return DGE_ERR_UNSUPPORTED;
    cudaStream_t stream = static_cast<cudaStream_t>(stream_);
    DGE_LAUNCH("compact_inplace", stream,
               launch_compact_inplace(plan.g, plan.layers, idx, nullptr, kv_desc(*K, paging),
                                      kv_desc(*V, paging), false, static_cast<uint32_t *>(ws),
                                      stream));
    return DGE_OK;
}

int dge_compact_inplace(const dge_problem *p, const int32_t *idx, const dge_tensor *K,
                        const dge_tensor *V, void *ws, void *stream)
{
    return dge_compact_inplace_paged(p, nullptr, idx, K, V, ws, stream);
}

int dge_pyramid_budgets(int32_t B, int32_t w, int32_t L, int32_t *out)
{
    if (!out || L < 2 || B <= w)
        return DGE_ERR_INVALID_ARG;
    const int32_t c = B - w;
    const int32_t lo = c / 20;
    const int32_t hi = 2 * c - lo;
    const int32_t step = (hi - lo) / (L - 1);
    for (int32_t l = 0; l < L; ++l)
        out[l] = hi - l * step;
    return DGE_OK;
}

int dge_get_device_status(void *ws, void *stream_)
{
    if (!ws)
        return DGE_ERR_INVALID_ARG;
    cudaStream_t stream = static_cast<cudaStream_t>(stream_);
    DGE_CHECK_CUDA(cudaStreamSynchronize(stream), "stream sync");
    uint32_t v = 0;
    DGE_CHECK_CUDA(cudaMemcpy(&v, ws, sizeof v, cudaMemcpyDeviceToHost), "status read");
    DGE_CHECK_CUDA(cudaMemset(ws, 0, sizeof v), "status clear");
    return (int)v;
}

const char *dge_status_string(int code)
{
    switch (code) {
    case DGE_OK: return "ok";
    case DGE_ERR_INVALID_ARG: return "invalid argument";
    case DGE_ERR_UNSUPPORTED: return "unsupported (head_dim, alignment or size)";
    case DGE_ERR_WORKSPACE_TOO_SMALL: return "workspace too small";
    case DGE_ERR_CUDA: return "CUDA error";
    case DGE_ERR_DEVICE_TIMEOUT: return "device-side wait timed out";
    default: return "unknown status";
    }
}

const char *dge_last_error(void) { return g_last_error; }

int dge_debug_set_waits(uint64_t limit_ns, int32_t extra_chunks)
{
    if (extra_chunks < 0)
        return DGE_ERR_INVALID_ARG;
    tc_set_waits(limit_ns, extra_chunks);
    return DGE_OK;
}

int dge_trace_set(void *buffer, size_t bytes, int cta)
{
    if (buffer && (bytes < (size_t)DGE_TRACE_SLOTS * DGE_TRACE_LEN * sizeof(uint64_t) ||
                   ((uintptr_t)buffer & 7) || cta < 0))
        return DGE_ERR_INVALID_ARG;
    tc_set_trace(static_cast<unsigned long long *>(buffer), cta);
    return DGE_OK;
}

int dge_profile_begin(void)
{
    Profiler &p = profiler();
    std::lock_guard<std::mutex> lk(p.mu);
    for (auto &r : p.records) {
        p.pool.push_back(r.start);
        p.pool.push_back(r.stop);
    }
    p.records.clear();
    p.on = true;
    return DGE_OK;
}

int dge_profile_end(dge_kernel_time *out, int capacity, int *count)
{
    Profiler &p = profiler();
    std::lock_guard<std::mutex> lk(p.mu);
    p.on = false;
    std::map<std::string, std::pair<int64_t, double>> acc;
    std::vector<std::string> order;
    int rc = DGE_OK;
    for (auto &r : p.records) {
        float ms = 0.f;
        cudaError_t e = cudaEventSynchronize(r.stop);
        if (e == cudaSuccess)
            e = cudaEventElapsedTime(&ms, r.start, r.stop);
        if (e != cudaSuccess && rc == DGE_OK)
            rc = cuda_fail(e, "profile");
        auto it = acc.find(r.name);
        if (it == acc.end()) {
            order.push_back(r.name);
            it = acc.emplace(r.name, std::make_pair((int64_t)0, 0.0)).first;
        }
        it->second.first += 1;
        it->second.second += ms;
        p.pool.push_back(r.start);
        p.pool.push_back(r.stop);
    }
    p.records.clear();
    if (count)
        *count = (int)order.size();
    for (int i = 0; i < (int)order.size() && i < capacity && out; ++i) {
        snprintf(out[i].name, sizeof out[i].name, "%s", order[i].c_str());
        out[i].launches = acc[order[i]].first;
        out[i].total_ms = acc[order[i]].second;
    }
    return rc;
}

}  // extern "C"
