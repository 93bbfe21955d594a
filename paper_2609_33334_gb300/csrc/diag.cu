// diag.cu -- eviction diagnostics from the normalisers (Sec. "Attention-Mass Analysis";
// App. "Why deferral can recover FullKV": Eq. evict-mass and Eq. match).
//
// For an observation row with full-cache normaliser lse = log Z and kept-set normaliser
// lse_hat = log Z_hat (the same sum over the retained keys only):
//   evicted mass  rho = 1 - Z_hat / Z = -expm1(lse_hat - lse)     (Eq. match's rho_q),
//   L_match of a unit = mean over its rows of lse - lse_hat = -log(1 - rho),
// and the retained-run length of a unit = B / (number of maximal runs of consecutive kept
// positions) -- the "mean contiguous run of retained tokens".
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace dge {

namespace {

constexpr int kDiagThreads = 256;

// Fixed-order block sum (deterministic): per-thread partial, then a tree in shared memory.
__device__ float block_sum(float v, float *red)
{
    red[threadIdx.x] = v;
    __syncthreads();
    for (int o = kDiagThreads / 2; o > 0; o >>= 1) {
        if ((int)threadIdx.x < o)
            red[threadIdx.x] += red[threadIdx.x + o];
        __syncthreads();
    }
    const float s = red[0];
    __syncthreads();
    return s;
}

__global__ void __launch_bounds__(kDiagThreads)
diag_kernel(const float *__restrict__ lse, float *__restrict__ rho_io,
            const int32_t *__restrict__ idx, Geometry g, LayerTable layers,
            float *__restrict__ l_match, float *__restrict__ run_length)
{
    __shared__ float red[kDiagThreads];
    const int64_t u = blockIdx.x;
    int l, bb, h;
    unit_coords(g, u, l, bb, h);
    // rho in place of lse_hat; the deficit lse - lse_hat summed for L_match.
    float dsum = 0.f;
    for (int r = threadIdx.x; r < g.R; r += kDiagThreads) {
        const int64_t i = u * g.R + r;
        const float d = fmaxf(lse[i] - rho_io[i], 0.f);
        rho_io[i] = -expm1f(-d);
        dsum += d;
    }
    const float tot = block_sum(dsum, red);
    if (l_match && threadIdx.x == 0)
        l_match[u] = tot / (float)g.R;
    if (run_length) {
        const int B = layers.budget[l];
        const int32_t *ui = idx + layers.row_base[l] + (int64_t)(bb * g.Hkv + h) * B;
        float breaks = 0.f;
        for (int j = 1 + threadIdx.x; j < B; j += kDiagThreads)
            breaks += ui[j] != ui[j - 1] + 1 ? 1.f : 0.f;
        const float runs = 1.f + block_sum(breaks, red);
        if (threadIdx.x == 0)
            run_length[u] = (float)B / runs;
    }
}

}  // namespace

cudaError_t launch_diag(const float *lse, float *rho_io, const int32_t *idx, const Geometry &g,
                        const LayerTable &layers, float *l_match, float *run_length,
                        cudaStream_t stream)
{
    if (g.U == 0)
        return cudaSuccess;
    diag_kernel<<<(unsigned)g.U, kDiagThreads, 0, stream>>>(lse, rho_io, idx, g, layers, l_match,
                                                           run_length);
    return cudaGetLastError();
}

}  // namespace dge
