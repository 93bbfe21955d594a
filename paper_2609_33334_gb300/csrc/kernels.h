// kernels.h -- internal launchers of libdge (not part of the ABI).
#pragma once

#include "common.cuh"

namespace dge {

// Scoring (score_mma.cu).
cudaError_t launch_lse_partial(const TensorDesc &K, const TensorDesc &Q, const Geometry &g,
                               int rows_per_block, int chunk_keys, float2 *partial,
                               cudaStream_t stream);
cudaError_t launch_combine_lse(const float2 *partial, int64_t total_rows, int nchunks,
                               float *lse2, cudaStream_t stream);
cudaError_t launch_colsum_rows(const TensorDesc &K, const TensorDesc &Q, const Geometry &g,
                               int chunk_keys, const float *lse2, float *raw,
                               cudaStream_t stream);
cudaError_t launch_colsum_keys(const TensorDesc &K, const TensorDesc &Q, const Geometry &g,
                               const float *lse2, float *raw, cudaStream_t stream);

// Pooling, selection, gather (select_compact.cu).
cudaError_t launch_pool(const float *raw, float *out, int64_t U, int P, int pool, int kernel,
                        cudaStream_t stream);
cudaError_t launch_select(const Geometry &g, const LayerTable &layers, const float *scores,
                          int32_t *idx, cudaStream_t stream);
cudaError_t launch_streaming_indices(const Geometry &g, const LayerTable &layers, int32_t *idx,
                                     cudaStream_t stream);
cudaError_t launch_compact(const Geometry &g, const LayerTable &layers, const int32_t *idx_in,
                           int32_t *idx_out, const TensorDesc &K, const TensorDesc &V, void *Kc,
                           void *Vc, bool implicit, uint32_t *status, cudaStream_t stream);

// Stores `text` as the calling thread's dge_last_error() message.
void record_error_text(const char *text);

}  // namespace dge
