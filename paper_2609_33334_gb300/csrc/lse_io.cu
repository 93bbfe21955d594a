// lse_io.cu -- row normalisers in and out of the scoring.
//
// The caller's normalisers (dge_buffers.lse_in / lse_out) are natural-log, fp32, dense
// [L][b][Hq][rows], which is the kernels' [U][R] order (unit u = (l*b + batch)*Hkv + h,
// stacked row r = g*rows + i of query head h*G + g).  The kernels keep lse in base 2
// (x = log2(e) * scale * q.k).  Row normaliser: App. B ("float32 softmax"); supplying it from
// the attention pass that produced the rows: Sec. "Draft-Guided Eviction" (phase B).
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace dge {

namespace {

__global__ void lse_import_kernel(const float *__restrict__ in, float *__restrict__ lse2,
                                  int64_t total)
{
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x)
        lse2[i] = in[i] * 1.4426950408889634f;
}

// out[u][r] = ln 2 * lse2 of the row: from the tensor-core path's chunk sums (added in chunk
// order, as that kernel merges them; row r of unit u is row r % rows of sub-unit
// u * (R / rows) + r / rows) unless the unit was recomputed (ready == 2) or there are no chunk
// sums (warp-level path), then from lse2.
__global__ void lse_export_kernel(const float *__restrict__ part, int nparts, int p1_chunks,
                                  int r4,
                                  const float *__restrict__ lse2,
                                  const uint32_t *__restrict__ ready, int64_t U, int R, int rows,
                                  float *__restrict__ out)
{
    const int64_t total = U * (int64_t)R;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t u = i / R;
        const int r = (int)(i - u * R);
        float l2;
        if (part && !(ready && ready[u] == 2)) {
            float Z = 0.f;
            const int64_t sub = u * (R / rows) + r / rows;
            const float *pu = part + sub * (int64_t)nparts * r4 + r % rows;
            for (int c = 0; c < p1_chunks; ++c)
                Z += pu[(int64_t)c * r4];
            Z += pu[(int64_t)(nparts - 1) * r4];   // the tail, added last as the kernel does
            l2 = log2f(Z);
        } else {
            l2 = lse2[i];
        }
        out[i] = l2 * 0.69314718055994531f;
    }
}

// Column sums of row blocks, added in fixed point (2^-40 units), back to float.
__global__ void fixed_to_float_kernel(const unsigned long long *__restrict__ fx,
                                      float *__restrict__ out, int64_t total)
{
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x)
        out[i] = __ll2float_rn((long long)fx[i]) * 0x1p-40f;   // one rounding, exact scaling
}

int blocks_for(int64_t total)
{
    const int64_t b = (total + 255) / 256;
    return (int)(b < 152 * 16 ? (b < 1 ? 1 : b) : 152 * 16);
}

}  // namespace

cudaError_t launch_lse_import(const float *lse_in, float *lse2, int64_t total, cudaStream_t stream)
{
    lse_import_kernel<<<blocks_for(total), 256, 0, stream>>>(lse_in, lse2, total);
    return cudaGetLastError();
}

cudaError_t launch_lse_export(const float *part, int nparts, int p1_chunks, int r4,
                              const float *lse2,
                              const uint32_t *ready, int64_t U, int R, int rows, float *lse_out,
                              cudaStream_t stream)
{
    lse_export_kernel<<<blocks_for(U * (int64_t)R), 256, 0, stream>>>(part, nparts, p1_chunks, r4, lse2,
                                                                       ready, U, R, rows, lse_out);
    return cudaGetLastError();
}

cudaError_t launch_fixed_to_float(const unsigned long long *fx, float *out, int64_t total,
                                  cudaStream_t stream)
{
    fixed_to_float_kernel<<<blocks_for(total), 256, 0, stream>>>(fx, out, total);
    return cudaGetLastError();
}


}  // namespace dge
