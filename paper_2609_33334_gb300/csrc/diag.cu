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

namespace dge {

namespace {

constexpr int kHoThreads = 256;
constexpr int kHoWarps = kHoThreads / 32;
constexpr int kHoMaxWords = 4096;         // kept-position bitmask: n <= 131072

// One held-out decode query per CTA (query head h of (l, b)), attending over all n keys of its
// KV head: an online softmax per warp (keys j = warp, warp + 8, ...; lanes split d), with the
// kept keys and the evicted keys in separate sums, merged across warps at the end.
template <int D>
__global__ void __launch_bounds__(kHoThreads)
heldout_kernel(TensorDesc Qh, TensorDesc K, TensorDesc V, const int32_t *__restrict__ idx,
               Geometry g, LayerTable layers, float *__restrict__ mass, float *__restrict__ err,
               float *__restrict__ gap)
{
    constexpr int E = D / 32;                 // elements of d per lane
    __shared__ uint32_t keep_bits[kHoMaxWords];
    __shared__ float w_max[kHoWarps], w_z[2][kHoWarps];
    __shared__ float w_o[2][kHoWarps][D];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t qh = blockIdx.x;            // (l * b + bb) * Hq + hq
    const int hq = (int)(qh % g.Hq);
    const int bb = (int)((qh / g.Hq) % g.b);
    const int l = (int)(qh / ((int64_t)g.Hq * g.b));
    const int h = hq / g.G;
    const int n = g.n, B = layers.budget[l];
    const int32_t *ui = idx + layers.row_base[l] + (int64_t)(bb * g.Hkv + h) * B;
    const int words = (n + 31) / 32;
    for (int i = threadIdx.x; i < words; i += kHoThreads)
        keep_bits[i] = 0;
    __syncthreads();
    for (int r = threadIdx.x; r < B; r += kHoThreads) {
        const int j = ui[r];
        if (j >= 0 && j < n)
            atomicOr(&keep_bits[j >> 5], 1u << (j & 31));
    }
    __syncthreads();

    const __nv_bfloat16 *q = Qh.data + l * Qh.s_layer + bb * Qh.s_batch + hq * Qh.s_head;
    float qv[E];
#pragma unroll
    for (int e = 0; e < E; ++e)
        qv[e] = __bfloat162float(q[lane * E + e]) * g.scale_log2;
    float mx = -INFINITY, z[2] = {0.f, 0.f}, o[2][E];
#pragma unroll
    for (int e = 0; e < E; ++e)
        o[0][e] = o[1][e] = 0.f;
    for (int j = warp; j < n; j += kHoWarps) {
        const __nv_bfloat16 *kr = kv_row_ptr(K, l, bb, h, j) + lane * E;
        float s = 0.f;
#pragma unroll
        for (int e = 0; e < E; ++e)
            s = fmaf(qv[e], __bfloat162float(kr[e]), s);
#pragma unroll
        for (int off = 16; off > 0; off >>= 1)
            s += __shfl_xor_sync(0xffffffffu, s, off);
        if (s > mx) {                         // rescale both sums to the new maximum
            const float c = ex2(mx - s);
            z[0] *= c;
            z[1] *= c;
#pragma unroll
            for (int e = 0; e < E; ++e) {
                o[0][e] *= c;
                o[1][e] *= c;
            }
            mx = s;
        }
        const float w = ex2(s - mx);
        const int set = (keep_bits[j >> 5] >> (j & 31)) & 1u ? 0 : 1;   // 0 kept, 1 evicted
        z[set] += w;
        const __nv_bfloat16 *vr = kv_row_ptr(V, l, bb, h, j) + lane * E;
#pragma unroll
        for (int e = 0; e < E; ++e)
            o[set][e] = fmaf(w, __bfloat162float(vr[e]), o[set][e]);
    }
    if (lane == 0) {
        w_max[warp] = mx;
        w_z[0][warp] = z[0];
        w_z[1][warp] = z[1];
    }
#pragma unroll
    for (int e = 0; e < E; ++e) {
        w_o[0][warp][lane * E + e] = o[0][e];
        w_o[1][warp][lane * E + e] = o[1][e];
    }
    __syncthreads();
    if (warp == 0) {
        float M = -INFINITY;
        for (int w = 0; w < kHoWarps; ++w)
            M = fmaxf(M, w_max[w]);
        float Z[2] = {0.f, 0.f}, O[2][E];
#pragma unroll
        for (int e = 0; e < E; ++e)
            O[0][e] = O[1][e] = 0.f;
        for (int w = 0; w < kHoWarps; ++w) {
            const float c = w_max[w] == -INFINITY ? 0.f : ex2(w_max[w] - M);
            for (int t = 0; t < 2; ++t) {
                Z[t] += c * w_z[t][w];
#pragma unroll
                for (int e = 0; e < E; ++e)
                    O[t][e] += c * w_o[t][w][lane * E + e];
            }
        }
        const float Zt = Z[0] + Z[1];
        const float m = Z[1] / Zt;
        // o - o~ = (O_R + O_E)/Z - O_R/Z_R;  mu_E - mu_R = O_E/Z_E - O_R/Z_R.
        float e2 = 0.f, g2 = 0.f;
#pragma unroll
        for (int e = 0; e < E; ++e) {
            const float muR = Z[0] > 0.f ? O[0][e] / Z[0] : 0.f;
            const float muE = Z[1] > 0.f ? O[1][e] / Z[1] : 0.f;
            const float dv = (O[0][e] + O[1][e]) / Zt - muR;
            const float gv = muE - muR;
            e2 = fmaf(dv, dv, e2);
            g2 = fmaf(gv, gv, g2);
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
            e2 += __shfl_xor_sync(0xffffffffu, e2, off);
            g2 += __shfl_xor_sync(0xffffffffu, g2, off);
        }
        if (lane == 0) {
            mass[qh] = m;
            err[qh] = sqrtf(e2);
            gap[qh] = m * sqrtf(g2);
        }
    }
}

}  // namespace

bool heldout_supported(const Geometry &g) { return (g.n + 31) / 32 <= kHoMaxWords; }

cudaError_t launch_heldout(const TensorDesc &Qh, const TensorDesc &K, const TensorDesc &V,
                           const int32_t *idx, const Geometry &g, const LayerTable &layers,
                           float *mass, float *err, float *gap, cudaStream_t stream)
{
    const int64_t heads = (int64_t)g.L * g.b * g.Hq;
    if (heads == 0)
        return cudaSuccess;
    if (g.d == 128)
        heldout_kernel<128><<<(unsigned)heads, kHoThreads, 0, stream>>>(Qh, K, V, idx, g, layers,
                                                                        mass, err, gap);
    else
        heldout_kernel<64><<<(unsigned)heads, kHoThreads, 0, stream>>>(Qh, K, V, idx, g, layers,
                                                                       mass, err, gap);
    return cudaGetLastError();
}

}  // namespace dge
