// kernels.h -- internal launchers of libdge (not part of the ABI).
#pragma once

#include "common.cuh"

namespace dge {

// Scoring on the warp-level tensor core path (score_mma.cu).  A UnitSel restricts the work:
// sel == nullptr, every unit; list false, the units whose flag sel[u] equals kUnitRecompute;
// list true, the units of a device-side list (sel[0] = count, sel[1 ..] = ids, as written by
// launch_collect_units), taken by a capped grid, so that an empty list costs little however
// many units there are.
constexpr uint32_t kUnitRecompute = 2;
struct UnitSel {
    const uint32_t *sel = nullptr;
    bool list = false;
};
cudaError_t launch_lse_partial(const TensorDesc &K, const TensorDesc &Q, const Geometry &g,
                               int rows_per_block, int chunk_keys, float2 *partial,
                               cudaStream_t stream, UnitSel units = {});
cudaError_t launch_combine_lse(const float2 *partial, int64_t total_rows, int nchunks,
                               float *lse2, cudaStream_t stream, UnitSel units = {},
                               int rows_per_unit = 1);
cudaError_t launch_colsum_rows(const TensorDesc &K, const TensorDesc &Q, const Geometry &g,
                               int chunk_keys, const float *lse2, float *raw,
                               cudaStream_t stream, UnitSel units = {});
// The units whose flag (flags[U]) equals kUnitRecompute into units[1 + U] (count first).
cudaError_t launch_collect_units(const uint32_t *flags, int64_t U, uint32_t *units,
                                 cudaStream_t stream);
// Tensor-core scoring: the row sums of every sub-unit over the observation rows' own
// positions [n - m, n) (masked causally), into chunk-sum slot `slot` of
// part[U*nrb][nparts][r4].
cudaError_t launch_tail_rows(const TensorDesc &K, const TensorDesc &Q, const Geometry &g,
                             int rows, int nrb, float *part, int nparts, int slot, int r4,
                             cudaStream_t stream);
// SCORED units of a device-side list (list[0] = count, then ids), each recomputed whole by
// one CTA with running maxima: row normalisers into lse2 (partial: [U][R] float2 scratch),
// then the column sums into raw.  A capped grid: an empty list costs one read per CTA.
cudaError_t launch_recompute_units(const TensorDesc &K, const TensorDesc &Q, const Geometry &g,
                                   float2 *partial, float *lse2, float *raw, const uint32_t *list,
                                   cudaStream_t stream);

// Scoring on the tcgen05 path (score_tc.cu).
struct TcPlan {
    int r_pad, nslab, chunk_keys, nchunks, kstages;
    int p1_chunks;     // chunks with keys below n - m (phase 1 covers [0, n - m))
    int nparts;        // chunk-sum slots per sub-unit: nchunks + 1 (slot nchunks: the tail)
    int r4;            // row stride of the chunk sums: rows rounded up to 4 (16-byte rows)
    int gsub = 1;      // query heads per sub-unit (row block)
    int nrb = 1;       // sub-units per unit: G / gsub
    int rows = 0;      // stacked rows of a sub-unit: gsub * m
    size_t smem;
};
struct TcBuffers {
    float *part;       // [U*nrb][nparts][r4] row sums of each key chunk, then of the tail
    float *lse2;       // [U][R]
    float *raw;        // [U][P]
    unsigned long long *raw_fx = nullptr;  // [U][P], nrb > 1: fixed-point sums (2^-40)
    uint32_t *count = nullptr;  // [U*nrb], zero before the launch
    uint32_t *ready = nullptr;  // [U], zero before the launch; 2 = recompute
    uint32_t *list = nullptr;   // [1 + U], list[0] zero before the launch: the units flagged 2
    uint32_t *status = nullptr;
    uint32_t *claim = nullptr;  // task claim counter, zero before the launch
    const float *lse_in = nullptr;  // [U][R] supplied natural-log normalisers (one pass)
};
bool tc_supported(const Geometry &g);
// Trace buffer of the tensor-core scoring kernel (see dge_trace_set); nullptr = off.
void tc_set_trace(unsigned long long *buffer, int cta);
// Test hook (see dge_debug_set_waits): the bound of the tcgen05 kernels' device-side waits
// (0 = the default) and extra chunks the scoring kernel's unit-count wait expects.
void tc_set_waits(unsigned long long limit_ns, int count_extra);
unsigned long long tc_wait_limit_ns();
TcPlan tc_plan(const Geometry &g);
// Both phases in one launch.  *encoded is false when the tensors cannot be described
// to TMA (nothing is launched then).
cudaError_t launch_score_tc(const TensorDesc &K, const TensorDesc &Q, const Geometry &g,
                            const TcPlan &plan, const TcBuffers &buf, cudaStream_t stream,
                            bool *encoded);
cudaError_t launch_colsum_keys(const TensorDesc &K, const TensorDesc &Q, const Geometry &g,
                               const float *lse2, float *raw, cudaStream_t stream,
                               UnitSel units = {});

// H2O scoring on the tcgen05 path (h2o_tc.cu): query blocks of pb positions x G heads.
struct H2oPhase {
    int pb;            // positions per query block
    int rows;          // G * pb stacked rows of a block
    int r_pad;         // rows rounded up to 16 (the MMA's N)
    int nqb;           // query blocks per unit
    size_t smem;       // dynamic shared memory
};
struct H2oPlan {
    H2oPhase ph[2];    // phase 1 (row normalisers), phase 2 (column sums)
    int nslab;         // d / 64
    int nkt;           // 128-key tiles of past keys per unit
};
bool h2o_tc_supported(const Geometry &g);
H2oPlan h2o_tc_plan(const Geometry &g);
// phase 1: lse2 [U][R] (base 2) and ready [U] (2 = recompute; zero before the launch);
// phase 2: raw [U][P] from lse2.  *encoded is false when the tensors cannot be described to
// TMA (nothing is launched then).
cudaError_t launch_h2o_tc(int phase, const TensorDesc &K, const TensorDesc &Q, const Geometry &g,
                          const H2oPlan &plan, float *lse2, float *raw, uint32_t *ready,
                          uint32_t *status, cudaStream_t stream, bool *encoded);

// Pooling, selection, gather (select_compact.cu).
cudaError_t launch_pool(const float *raw, float *out, int64_t U, int P, int pool, int kernel,
                        cudaStream_t stream);
// Row normalisers: caller's natural-log [U][R] -> base-2 lse2; lse2 (or, on the tensor-core
// path, its chunk sums part [U*nrb][nparts][r4] -- slots 0 .. p1_chunks-1, then the tail's slot
// nparts-1, in that order -- for units with ready != 2) -> natural-log out.
cudaError_t launch_lse_import(const float *lse_in, float *lse2, int64_t total, cudaStream_t stream);
cudaError_t launch_lse_export(const float *part, int nparts, int p1_chunks, int r4,
                              const float *lse2,
                              const uint32_t *ready, int64_t U, int R, int rows, float *lse_out,
                              cudaStream_t stream);
// Fixed-point (2^-40) column sums of row blocks -> float.
cudaError_t launch_fixed_to_float(const unsigned long long *fx, float *out, int64_t total,
                                  cudaStream_t stream);

// Diagnostics of one eviction from lse (full cache) and lse_hat (kept keys), both [U][R]
// natural log: rho_io holds lse_hat on entry and the evicted mass on return; l_match and
// run_length [U] (nullable).
cudaError_t launch_diag(const float *lse, float *rho_io, const int32_t *idx, const Geometry &g,
                        const LayerTable &layers, float *l_match, float *run_length,
                        cudaStream_t stream);
// Held-out decode queries (one per query head, position n) against a kept set: evicted mass,
// |o - o~| and m |mu_E - mu_R| per head (Eq. evict-mass).  n <= 131072.
bool heldout_supported(const Geometry &g);
cudaError_t launch_heldout(const TensorDesc &Qh, const TensorDesc &K, const TensorDesc &V,
                           const int32_t *idx, const Geometry &g, const LayerTable &layers,
                           float *mass, float *err, float *gap, cudaStream_t stream);
// Pooling and selection in one kernel (the evict path), for P <= 32768 positions per unit.
// pooled_out (nullable) receives the pooled scores.
bool pool_select_supported(const Geometry &g);
cudaError_t launch_pool_select(const Geometry &g, const LayerTable &layers, const float *raw,
                               float *pooled_out, int32_t *idx, cudaStream_t stream);
// The same for longer rows (P > 32768; avg or max pooling of radius <= 4): the pooled scores
// go to `pooled` (required: the selection reads them back).
bool pool_select_large_supported(const Geometry &g);
cudaError_t launch_pool_select_large(const Geometry &g, const LayerTable &layers, const float *raw,
                                     float *pooled, int32_t *idx, cudaStream_t stream);
// Block-granular selection (g.select_block >= 2) from final scores [U][P].
cudaError_t launch_block_select(const Geometry &g, const LayerTable &layers, const float *scores,
                                int32_t *idx, cudaStream_t stream);
cudaError_t launch_select(const Geometry &g, const LayerTable &layers, const float *scores,
                          int32_t *idx, cudaStream_t stream);
cudaError_t launch_streaming_indices(const Geometry &g, const LayerTable &layers, int32_t *idx,
                                     cudaStream_t stream);
// In-place gather: rows [0, B_l) of every unit of K and V become the kept rows (idx ascending
// per unit, as the selection writes it; implicit = StreamingLLM positions, written to idx_out).
cudaError_t launch_compact_inplace(const Geometry &g, const LayerTable &layers,
                                   const int32_t *idx_in, int32_t *idx_out, const TensorDesc &K,
                                   const TensorDesc &V, bool implicit, uint32_t *status,
                                   cudaStream_t stream);
cudaError_t launch_compact(const Geometry &g, const LayerTable &layers, const int32_t *idx_in,
                           int32_t *idx_out, const TensorDesc &K, const TensorDesc &V, void *Kc,
                           void *Vc, bool implicit, uint32_t *status, cudaStream_t stream);

// Stores `text` as the calling thread's dge_last_error() message.
void record_error_text(const char *text);

}  // namespace dge
