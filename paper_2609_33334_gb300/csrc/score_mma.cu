// score_mma.cu -- attention-score kernels on the warp-level tensor core path.
//
// Computes, per unit (layer, batch, KV head), over the stacked rows r of the
// group's G query heads (Alg. 1 line B; App. B; App. G):
//   x_rj  = log2(e) * scale * q_r . k_j                      (base-2 logits)
//   lse_r = log2 sum_{j <= pos_r} 2^{x_rj}                    (row normaliser)
//   raw_j = sum_r 2^{x_rj - lse_r}   over rows with j <= pos_r (column sum)
//
// The normaliser couples a whole row, so the pass has two phases:
//   phase 1 (lse_partial_kernel): rows resident in shared memory, keys
//     streamed; each CTA emits per-row (max, sum) partials for its key chunk;
//   combine_lse_kernel: merges the chunk partials into lse_r;
//   phase 2 (colsum_rows_kernel / colsum_keys_kernel): recomputes the logits
//     and sums 2^{x - lse} over rows for every key.
// The products use mma.sync m16n8k16 with keys as the M dimension and rows as
// N (the "transposed" product S^T = K Q^T), so each lane holds 2 keys x 2 rows
// of every 16x8 tile: row sums reduce across 8 lanes and column sums across 4.
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace dge {

constexpr int kThreads = 256;   // 8 warps
constexpr int kTileKeys = 64;   // keys per staged K tile = 4 m-tiles of 16
constexpr int kRowTile = 64;    // query rows per streamed tile (keys-resident kernel)
constexpr int kKeyBlock = 128;  // keys per CTA of the keys-resident kernel (8 warps x 16)

template <int D>
struct Pad {
    static constexpr int kStride = D + 8;  // padded smem row: conflict-free ldmatrix
};

__device__ __forceinline__ float neg_inf() { return -INFINITY; }

// Stage `rows` query rows (stacked index r0 + r) into smem, zero rows up to rows_pad.
template <int D>
__device__ void stage_rows(__nv_bfloat16 *sQ, const TensorDesc &Q, const Geometry &g, int l,
                           int bb, int h, int r0, int rows, int rows_pad, int rows_per_head)
{
    constexpr int V = D / 8;
    for (int i = threadIdx.x; i < rows_pad * V; i += blockDim.x) {
        const int r = i / V, c = i % V;
        __nv_bfloat16 *dst = sQ + r * Pad<D>::kStride + c * 8;
        if (r < rows)
            cp_async_16(dst, q_row_ptr(Q, g, l, bb, h, r0 + r, rows_per_head) + c * 8, 16);
        else
            *reinterpret_cast<int4 *>(dst) = make_int4(0, 0, 0, 0);
    }
}

// Stage keys [k0, k0 + kTileKeys) of one unit, zero-filling keys >= k_lim.
template <int D, int KEYS>
__device__ void stage_keys(__nv_bfloat16 *sK, const TensorDesc &K, int l, int bb, int h, int k0,
                           int k_lim)
{
    constexpr int V = D / 8;
    for (int i = threadIdx.x; i < KEYS * V; i += blockDim.x) {
        const int r = i / V, c = i % V;
        const int key = k0 + r;
        __nv_bfloat16 *dst = sK + r * Pad<D>::kStride + c * 8;
        if (key < k_lim)
            cp_async_16(dst, kv_row_ptr(K, l, bb, h, key) + c * 8, 16);
        else
            *reinterpret_cast<int4 *>(dst) = make_int4(0, 0, 0, 0);
    }
}

// A fragments (16 keys x D) of m-tile `mt` of a staged key tile.
template <int D>
__device__ __forceinline__ void load_a(uint32_t (&a)[D / 16][4], const __nv_bfloat16 *sK, int mt,
                                       int lane)
{
    const __nv_bfloat16 *base =
        sK + (mt * 16 + (lane & 7) + 8 * ((lane >> 3) & 1)) * Pad<D>::kStride + 8 * (lane >> 4);
#pragma unroll
    for (int ks = 0; ks < D / 16; ++ks)
        ldmatrix_x4(a[ks], base + ks * 16);
}

// acc = S^T tile (16 keys x 8 rows) of n-tile `nt` of the staged rows.
template <int D>
__device__ __forceinline__ void tile_product(float (&acc)[4], const uint32_t (&a)[D / 16][4],
                                             const __nv_bfloat16 *sQ, int nt, int lane)
{
    acc[0] = acc[1] = acc[2] = acc[3] = 0.f;
    const __nv_bfloat16 *base = sQ + (nt * 8 + (lane & 7)) * Pad<D>::kStride + 8 * (lane >> 3);
#pragma unroll
    for (int k2 = 0; k2 < D / 32; ++k2) {
        uint32_t b[4];
        ldmatrix_x4(b, base + k2 * 32);
        mma_bf16_16816(acc, a[2 * k2], b[0], b[1]);
        mma_bf16_16816(acc, a[2 * k2 + 1], b[2], b[3]);
    }
}

// Highest position seen by stacked rows [r0, r1) of one unit.
__device__ __forceinline__ int max_row_position(const Geometry &g, int r0, int r1)
{
    if (g.variant != DGE_VARIANT_H2O)
        return g.n - 1;
    if (r0 / g.n == (r1 - 1) / g.n)
        return (r1 - 1) % g.n;
    return g.n - 1;
}

// The units a launch covers (UnitSel): every unit, one CTA per block of work (sel ==
// nullptr); the units whose flag sel[u] equals kUnitRecompute (the other CTAs return at
// once); or the units of a list (units[0] = count, units[1 ..] = ids), whose blocks the CTAs
// of a capped grid take in turn -- a launch for an empty list costs one read per CTA however
// large the problem.  vblocks is the number of blocks of work, vblock_id the global block
// index of the vb-th, vblock_skip whether a block of unit u has nothing to do.
__device__ __forceinline__ int64_t vblocks(const UnitSel &us, int64_t U, int64_t per_unit)
{
    return (us.sel && us.list ? (int64_t)us.sel[0] : U) * per_unit;
}
__device__ __forceinline__ int64_t vblock_id(const UnitSel &us, int64_t per_unit, int64_t vb)
{
    return us.sel && us.list ? (int64_t)us.sel[1 + vb / per_unit] * per_unit + vb % per_unit
                             : vb;
}
__device__ __forceinline__ bool vblock_skip(const UnitSel &us, int64_t u)
{
    return us.sel && !us.list && us.sel[u] != kUnitRecompute;
}
constexpr int64_t kListGrid = 1024;   // CTAs of a launch over a unit list
__host__ inline int64_t grid_for(const UnitSel &us, int64_t blocks)
{
    return us.sel && us.list && blocks > kListGrid ? kListGrid : blocks;
}

// ---------------------------------------------------------------------------
// Phase 1: per-row (max, sum) partials over one key chunk.
// Block = (unit, row block, key chunk), flattened as ((u * nrb) + rb) * nchunks + chunk.
// partial layout: [u][R][nchunks] float2 (max in base-2 units, sum of 2^{x - max}).
template <int D, int MAX_NTW>
__device__ void lse_partial_block(const TensorDesc &K, const TensorDesc &Q, const Geometry &g,
                                  int rows_per_block, int nrb, int chunk_keys, int nchunks,
                                  float2 *__restrict__ partial, int64_t bid)
{
    extern __shared__ __align__(16) uint8_t smem[];
    const int chunk = (int)(bid % nchunks);
    const int rb = (int)((bid / nchunks) % nrb);
    const int64_t u = bid / ((int64_t)nchunks * nrb);
    int l, bb, h;
    unit_coords(g, u, l, bb, h);
    const int r0 = rb * rows_per_block;
    const int rows = min(rows_per_block, g.R - r0);
    const int rows_pad = (rows + 7) & ~7;
    const int rows_per_head = g.variant == DGE_VARIANT_H2O ? g.n : g.m;
    const int NT = rows_pad / 8;

    const int k_lo = chunk * chunk_keys;
    const int k_hi = min(min(k_lo + chunk_keys, g.n), max_row_position(g, r0, r0 + rows) + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int gq = lane >> 2, tq = lane & 3;

    float rm[MAX_NTW][2], rz[MAX_NTW][2];
    int lim[MAX_NTW][2];
#pragma unroll
    for (int i = 0; i < MAX_NTW; ++i)
#pragma unroll
        for (int c = 0; c < 2; ++c) {
            const int nt = warp + 8 * i;
            const int r = nt * 8 + 2 * tq + c;
            rm[i][c] = neg_inf();
            rz[i][c] = 0.f;
            lim[i][c] = (nt < NT && r < rows) ? min(row_position(g, r0 + r), k_hi - 1) : -1;
        }

    if (k_lo < k_hi) {
        __nv_bfloat16 *sQ = reinterpret_cast<__nv_bfloat16 *>(smem);
        __nv_bfloat16 *sK = sQ + rows_pad * Pad<D>::kStride;
        stage_rows<D>(sQ, Q, g, l, bb, h, r0, rows, rows_pad, rows_per_head);
        stage_keys<D, kTileKeys>(sK, K, l, bb, h, k_lo, k_hi);
        cp_async_commit();
        const int ntiles = (k_hi - k_lo + kTileKeys - 1) / kTileKeys;
        for (int t = 0; t < ntiles; ++t) {
            if (t + 1 < ntiles) {
                stage_keys<D, kTileKeys>(sK + ((t + 1) & 1) * kTileKeys * Pad<D>::kStride, K, l,
                                         bb, h, k_lo + (t + 1) * kTileKeys, k_hi);
                cp_async_commit();
                cp_async_wait<1>();
            } else {
                cp_async_wait<0>();
            }
            __syncthreads();
            const __nv_bfloat16 *sKt = sK + (t & 1) * kTileKeys * Pad<D>::kStride;
            const int tile0 = k_lo + t * kTileKeys;
#pragma unroll 1
            for (int mt = 0; mt < kTileKeys / 16; ++mt) {
                uint32_t a[D / 16][4];
                load_a<D>(a, sKt, mt, lane);
                const int key0 = tile0 + mt * 16 + gq, key1 = key0 + 8;
#pragma unroll
                for (int i = 0; i < MAX_NTW; ++i) {
                    const int nt = warp + 8 * i;
                    if (nt < NT) {
                        float acc[4];
                        tile_product<D>(acc, a, sQ, nt, lane);
#pragma unroll
                        for (int c = 0; c < 2; ++c) {
                            const float xa = key0 <= lim[i][c] ? acc[c] * g.scale_log2 : neg_inf();
                            const float xb =
                                key1 <= lim[i][c] ? acc[2 + c] * g.scale_log2 : neg_inf();
                            const float mx = fmaxf(xa, xb);
                            if (mx > rm[i][c]) {
                                rz[i][c] *= ex2(rm[i][c] - mx);
                                rm[i][c] = mx;
                            }
                            if (mx != neg_inf())
                                rz[i][c] += ex2(xa - rm[i][c]) + ex2(xb - rm[i][c]);
                        }
                    }
                }
            }
            __syncthreads();
        }
    }

    // Merge the 8 lanes that share each row (lane bits 2..4), then write.
#pragma unroll
    for (int i = 0; i < MAX_NTW; ++i)
#pragma unroll
        for (int c = 0; c < 2; ++c) {
            float m = rm[i][c], z = rz[i][c];
#pragma unroll
            for (int off = 4; off < 32; off <<= 1) {
                const float m2 = __shfl_xor_sync(0xffffffffu, m, off);
                const float z2 = __shfl_xor_sync(0xffffffffu, z, off);
                const float M = fmaxf(m, m2);
                z = (M == neg_inf()) ? 0.f : z * ex2(m - M) + z2 * ex2(m2 - M);
                m = M;
            }
            const int nt = warp + 8 * i;
            const int r = nt * 8 + 2 * tq + c;
            if (gq == 0 && nt < NT && r < rows)
                partial[((u * g.R) + r0 + r) * nchunks + chunk] = make_float2(m, z);
        }
}

template <int D, int MAX_NTW>
__global__ void __launch_bounds__(kThreads)
lse_partial_kernel(TensorDesc K, TensorDesc Q, Geometry g, int rows_per_block, int nrb,
                   int chunk_keys, int nchunks, float2 *__restrict__ partial, UnitSel us)
{
    const int64_t per = (int64_t)nrb * nchunks;
    const int64_t total = vblocks(us, g.U, per);
    for (int64_t vb = blockIdx.x; vb < total; vb += gridDim.x) {
        const int64_t bid = vblock_id(us, per, vb);
        if (vblock_skip(us, bid / per))
            continue;
        lse_partial_block<D, MAX_NTW>(K, Q, g, rows_per_block, nrb, chunk_keys, nchunks, partial,
                                      bid);
        __syncthreads();   // shared memory is reused by the next block of work
    }
}

// lse_r = M + log2(sum_c z_c 2^{m_c - M}) over the chunks of row r.
__global__ void combine_lse_kernel(const float2 *__restrict__ partial, int64_t total_rows,
                                   int nchunks, float *__restrict__ lse2, UnitSel us,
                                   int rows_per_unit)
{
    const int64_t total = us.sel && us.list ? (int64_t)us.sel[0] * rows_per_unit : total_rows;
    for (int64_t v = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; v < total;
         v += (int64_t)gridDim.x * blockDim.x) {
        const int64_t i = vblock_id(us, rows_per_unit, v);
        if (vblock_skip(us, i / rows_per_unit))
            continue;
        const float2 *p = partial + i * nchunks;
        float M = neg_inf();
        for (int c = 0; c < nchunks; ++c)
            M = fmaxf(M, p[c].x);
        float Z = 0.f;
        for (int c = 0; c < nchunks; ++c)
            Z += p[c].y * ex2(p[c].x - M);
        lse2[i] = M + log2f(Z);
    }
}

// ---------------------------------------------------------------------------
// Phase 2 (rows resident): raw_j = sum_r 2^{x_rj - lse_r} for keys of one chunk
// of [0, P).  Block = (unit, chunk) flattened as u * nchunks + chunk.
template <int D, int MAX_NTW>
__device__ void colsum_rows_block(const TensorDesc &K, const TensorDesc &Q, const Geometry &g,
                                  int chunk_keys, int nchunks, const float *__restrict__ lse2,
                                  float *__restrict__ raw, int64_t bid)
{
    extern __shared__ __align__(16) uint8_t smem[];
    __shared__ float sCol[kThreads / 32][kTileKeys];
    const int64_t u = bid / nchunks;
    const int chunk = (int)(bid % nchunks);
    int l, bb, h;
    unit_coords(g, u, l, bb, h);
    const int rows = g.R;
    const int rows_pad = (rows + 7) & ~7;
    const int NT = rows_pad / 8;
    const int k_lo = chunk * chunk_keys;
    const int k_hi = min(k_lo + chunk_keys, g.P);
    if (k_lo >= k_hi)
        return;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int gq = lane >> 2, tq = lane & 3;
    float L2[MAX_NTW][2];
    int lim[MAX_NTW][2];
#pragma unroll
    for (int i = 0; i < MAX_NTW; ++i)
#pragma unroll
        for (int c = 0; c < 2; ++c) {
            const int nt = warp + 8 * i;
            const int r = nt * 8 + 2 * tq + c;
            const bool ok = nt < NT && r < rows;
            L2[i][c] = ok ? lse2[u * g.R + r] : 0.f;
            lim[i][c] = ok ? min(row_position(g, r), k_hi - 1) : -1;
        }

    __nv_bfloat16 *sQ = reinterpret_cast<__nv_bfloat16 *>(smem);
    __nv_bfloat16 *sK = sQ + rows_pad * Pad<D>::kStride;
    stage_rows<D>(sQ, Q, g, l, bb, h, 0, rows, rows_pad, g.m);
    stage_keys<D, kTileKeys>(sK, K, l, bb, h, k_lo, k_hi);
    cp_async_commit();
    const int ntiles = (k_hi - k_lo + kTileKeys - 1) / kTileKeys;
    for (int t = 0; t < ntiles; ++t) {
        if (t + 1 < ntiles) {
            stage_keys<D, kTileKeys>(sK + ((t + 1) & 1) * kTileKeys * Pad<D>::kStride, K, l, bb,
                                     h, k_lo + (t + 1) * kTileKeys, k_hi);
            cp_async_commit();
            cp_async_wait<1>();
        } else {
            cp_async_wait<0>();
        }
        __syncthreads();
        const __nv_bfloat16 *sKt = sK + (t & 1) * kTileKeys * Pad<D>::kStride;
        const int tile0 = k_lo + t * kTileKeys;
#pragma unroll 1
        for (int mt = 0; mt < kTileKeys / 16; ++mt) {
            uint32_t a[D / 16][4];
            load_a<D>(a, sKt, mt, lane);
            const int key0 = tile0 + mt * 16 + gq, key1 = key0 + 8;
            float cs0 = 0.f, cs1 = 0.f;
#pragma unroll
            for (int i = 0; i < MAX_NTW; ++i) {
                const int nt = warp + 8 * i;
                if (nt < NT) {
                    float acc[4];
                    tile_product<D>(acc, a, sQ, nt, lane);
#pragma unroll
                    for (int c = 0; c < 2; ++c) {
                        cs0 += key0 <= lim[i][c] ? ex2(acc[c] * g.scale_log2 - L2[i][c]) : 0.f;
                        cs1 += key1 <= lim[i][c] ? ex2(acc[2 + c] * g.scale_log2 - L2[i][c]) : 0.f;
                    }
                }
            }
            cs0 += __shfl_xor_sync(0xffffffffu, cs0, 1);
            cs0 += __shfl_xor_sync(0xffffffffu, cs0, 2);
            cs1 += __shfl_xor_sync(0xffffffffu, cs1, 1);
            cs1 += __shfl_xor_sync(0xffffffffu, cs1, 2);
            if (tq == 0) {
                sCol[warp][mt * 16 + gq] = cs0;
                sCol[warp][mt * 16 + gq + 8] = cs1;
            }
        }
        __syncthreads();
        if (threadIdx.x < kTileKeys) {
            const int key = tile0 + threadIdx.x;
            if (key < k_hi) {
                float s = 0.f;
#pragma unroll
                for (int w = 0; w < kThreads / 32; ++w)
                    s += sCol[w][threadIdx.x];
                raw[u * g.P + key] = s;
            }
        }
        __syncthreads();
    }
}

template <int D, int MAX_NTW>
__global__ void __launch_bounds__(kThreads)
colsum_rows_kernel(TensorDesc K, TensorDesc Q, Geometry g, int chunk_keys, int nchunks,
                   const float *__restrict__ lse2, float *__restrict__ raw, UnitSel us)
{
    const int64_t total = vblocks(us, g.U, nchunks);
    for (int64_t vb = blockIdx.x; vb < total; vb += gridDim.x) {
        const int64_t bid = vblock_id(us, nchunks, vb);
        if (vblock_skip(us, bid / nchunks))
            continue;
        colsum_rows_block<D, MAX_NTW>(K, Q, g, chunk_keys, nchunks, lse2, raw, bid);
        __syncthreads();
    }
}

// ---------------------------------------------------------------------------
// Phase 2 (keys resident, rows streamed) for H2O: CTA owns kKeyBlock keys,
// warp w owns keys [16w, 16w + 16) with its A fragments in registers, and the
// rows that can see those keys (position >= first key) stream through smem.
// Block = (unit, key block) flattened as u * nkb + kb.
template <int D>
__device__ void colsum_keys_block(const TensorDesc &K, const TensorDesc &Q, const Geometry &g,
                                  int nkb, const float *__restrict__ lse2,
                                  float *__restrict__ raw, int64_t bid)
{
    extern __shared__ __align__(16) uint8_t smem[];
    __shared__ float sL[2][kRowTile];
    __shared__ int sPos[2][kRowTile];
    const int64_t u = bid / nkb;
    const int kb = (int)(bid % nkb);
    int l, bb, h;
    unit_coords(g, u, l, bb, h);
    const int k_lo = kb * kKeyBlock;
    const int k_hi = min(k_lo + kKeyBlock, g.P);
    if (k_lo >= k_hi)
        return;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int gq = lane >> 2, tq = lane & 3;

    __nv_bfloat16 *sK = reinterpret_cast<__nv_bfloat16 *>(smem);
    __nv_bfloat16 *sQ = sK + kKeyBlock * Pad<D>::kStride;  // [2][kRowTile][stride]
    stage_keys<D, kKeyBlock>(sK, K, l, bb, h, k_lo, k_hi);
    cp_async_commit();

    // Row tiles: for every query head of the group, positions from the tile
    // containing k_lo up to n - 1 (rows at earlier positions cannot see these keys).
    const int first = (k_lo / kRowTile) * kRowTile;
    const int tiles_per_head = (g.n - first + kRowTile - 1) / kRowTile;
    const int ntiles = tiles_per_head * g.G;

    auto stage_tile = [&](int t, int buf) {
        const int gh = t / tiles_per_head;
        const int i0 = first + (t % tiles_per_head) * kRowTile;
        const int rows = min(kRowTile, g.n - i0);
        stage_rows<D>(sQ + buf * kRowTile * Pad<D>::kStride, Q, g, l, bb, h, gh * g.n + i0, rows,
                      kRowTile, g.n);
        if (threadIdx.x < kRowTile) {
            const int r = threadIdx.x;
            sL[buf][r] = r < rows ? lse2[u * g.R + gh * g.n + i0 + r] : 0.f;
            sPos[buf][r] = r < rows ? i0 + r : -1;
        }
    };

    stage_tile(0, 0);
    cp_async_commit();
    cp_async_wait<0>();
    __syncthreads();
    uint32_t a[D / 16][4];
    load_a<D>(a, sK, warp, lane);
    const int key0 = k_lo + warp * 16 + gq, key1 = key0 + 8;
    const bool v0 = key0 < k_hi, v1 = key1 < k_hi;
    float cs0 = 0.f, cs1 = 0.f;
    for (int t = 0; t < ntiles; ++t) {
        if (t + 1 < ntiles) {
            stage_tile(t + 1, (t + 1) & 1);
            cp_async_commit();
            cp_async_wait<1>();
        } else {
            cp_async_wait<0>();
        }
        __syncthreads();
        const int buf = t & 1;
        const __nv_bfloat16 *sQt = sQ + buf * kRowTile * Pad<D>::kStride;
#pragma unroll
        for (int nt = 0; nt < kRowTile / 8; ++nt) {
            float acc[4];
            tile_product<D>(acc, a, sQt, nt, lane);
#pragma unroll
            for (int c = 0; c < 2; ++c) {
                const int r = nt * 8 + 2 * tq + c;
                const int p = sPos[buf][r];
                const float L = sL[buf][r];
                cs0 += (v0 && key0 <= p) ? ex2(acc[c] * g.scale_log2 - L) : 0.f;
                cs1 += (v1 && key1 <= p) ? ex2(acc[2 + c] * g.scale_log2 - L) : 0.f;
            }
        }
        __syncthreads();
    }
    cs0 += __shfl_xor_sync(0xffffffffu, cs0, 1);
    cs0 += __shfl_xor_sync(0xffffffffu, cs0, 2);
    cs1 += __shfl_xor_sync(0xffffffffu, cs1, 1);
    cs1 += __shfl_xor_sync(0xffffffffu, cs1, 2);
    if (tq == 0) {
        if (v0)
            raw[u * g.P + key0] = cs0;
        if (v1)
            raw[u * g.P + key1] = cs1;
    }
}

template <int D>
__global__ void __launch_bounds__(kThreads)
colsum_keys_kernel(TensorDesc K, TensorDesc Q, Geometry g, int nkb,
                   const float *__restrict__ lse2, float *__restrict__ raw, UnitSel us)
{
    const int64_t total = vblocks(us, g.U, nkb);
    for (int64_t vb = blockIdx.x; vb < total; vb += gridDim.x) {
        const int64_t bid = vblock_id(us, nkb, vb);
        if (vblock_skip(us, bid / nkb))
            continue;
        colsum_keys_block<D>(K, Q, g, nkb, lse2, raw, bid);
        __syncthreads();
    }
}

// Units of a list (list[0] = count, list[1 ..] = ids), each recomputed whole by one CTA:
// the row normalisers over all keys with running maxima (one chunk, all rows), then the
// column sums over [0, P).  The merge of a single chunk is the combine step's: lse = m +
// log2(z).  The CTA's own global writes of lse2 are visible to it after the barrier.
template <int D, int MAX_NTW>
__global__ void __launch_bounds__(kThreads)
recompute_units_kernel(TensorDesc K, TensorDesc Q, Geometry g, float2 *__restrict__ partial,
                       float *__restrict__ lse2, float *__restrict__ raw,
                       const uint32_t *__restrict__ list)
{
    const uint32_t count = list[0];
    for (uint32_t i = blockIdx.x; i < count; i += gridDim.x) {
        const int64_t u = list[1 + i];
        lse_partial_block<D, MAX_NTW>(K, Q, g, g.R, 1, g.n, 1, partial, u);
        __syncthreads();
        for (int r = threadIdx.x; r < g.R; r += blockDim.x) {
            const float2 p = partial[u * g.R + r];
            lse2[u * g.R + r] = p.x + log2f(p.y);
        }
        __syncthreads();
        colsum_rows_block<D, MAX_NTW>(K, Q, g, g.P, 1, lse2, raw, u);
        __syncthreads();
    }
}

// Row sums over the observation rows' own positions, for the tensor-core scoring, whose main
// kernel covers only the keys every row sees ([0, n - m)): sub-unit s = u * nrb + rb holds
// rows rb * rows .. of unit u; row r sits at n - m + r % m and sees the keys n - m .. n - m +
// r % m.  z_r = sum of 2^{x_rj} over them, in fp32 with no running maximum (the tensor-core
// kernel's sums are plain too; its range check covers these), written to chunk-sum slot `slot`
// of the sub-unit: part[(s * nparts + slot) * r4 + r].
template <int D, int MAX_NTW>
__global__ void __launch_bounds__(kThreads)
tail_rows_kernel(TensorDesc K, TensorDesc Q, Geometry g, int rows, int nrb,
                 float *__restrict__ part, int nparts, int slot, int r4)
{
    extern __shared__ __align__(16) uint8_t smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int gq = lane >> 2, tq = lane & 3;
    const int rows_pad = (rows + 7) & ~7;
    const int NT = rows_pad / 8;
    const int first = g.n - g.m;
    __nv_bfloat16 *sQ = reinterpret_cast<__nv_bfloat16 *>(smem);
    __nv_bfloat16 *sK = sQ + rows_pad * Pad<D>::kStride;
    for (int64_t s = blockIdx.x; s < g.U * nrb; s += gridDim.x) {
        const int64_t u = s / nrb;
        const int rb = (int)(s % nrb);
        int l, bb, h;
        unit_coords(g, u, l, bb, h);
        stage_rows<D>(sQ, Q, g, l, bb, h, rb * rows, rows, rows_pad, g.m);
        float z[MAX_NTW][2];
        int lim[MAX_NTW][2];
#pragma unroll
        for (int i = 0; i < MAX_NTW; ++i)
#pragma unroll
            for (int c = 0; c < 2; ++c) {
                const int nt = warp + 8 * i;
                const int r = nt * 8 + 2 * tq + c;
                z[i][c] = 0.f;
                lim[i][c] = (nt < NT && r < rows) ? first + r % g.m : -1;
            }
        for (int k0 = first; k0 < g.n; k0 += kTileKeys) {
            stage_keys<D, kTileKeys>(sK, K, l, bb, h, k0, g.n);
            cp_async_commit();
            cp_async_wait<0>();
            __syncthreads();
#pragma unroll 1
            for (int mt = 0; mt < kTileKeys / 16; ++mt) {
                if (k0 + mt * 16 >= g.n)
                    break;
                uint32_t a[D / 16][4];
                load_a<D>(a, sK, mt, lane);
                const int key0 = k0 + mt * 16 + gq, key1 = key0 + 8;
#pragma unroll
                for (int i = 0; i < MAX_NTW; ++i) {
                    const int nt = warp + 8 * i;
                    if (nt < NT) {
                        float acc[4];
                        tile_product<D>(acc, a, sQ, nt, lane);
#pragma unroll
                        for (int c = 0; c < 2; ++c) {
                            const float ea = key0 <= lim[i][c] ? ex2(acc[c] * g.scale_log2) : 0.f;
                            const float eb = key1 <= lim[i][c] ? ex2(acc[2 + c] * g.scale_log2)
                                                               : 0.f;
                            z[i][c] += ea + eb;
                        }
                    }
                }
            }
            __syncthreads();
        }
        // The 8 lanes that share each row (lane bits 2..4), in a fixed order.
#pragma unroll
        for (int i = 0; i < MAX_NTW; ++i)
#pragma unroll
            for (int c = 0; c < 2; ++c) {
                float v = z[i][c];
                v += __shfl_xor_sync(0xffffffffu, v, 4);
                v += __shfl_xor_sync(0xffffffffu, v, 8);
                v += __shfl_xor_sync(0xffffffffu, v, 16);
                const int nt = warp + 8 * i;
                const int r = nt * 8 + 2 * tq + c;
                if (gq == 0 && nt < NT && r < rows)
                    part[(s * nparts + slot) * r4 + r] = v;
            }
    }
}

// The units flagged kUnitRecompute, as a list (units[0] = count, then the ids in any order:
// every unit is recomputed on its own).  One CTA.
__global__ void collect_units_kernel(const uint32_t *__restrict__ flags, int64_t U,
                                     uint32_t *__restrict__ units)
{
    __shared__ uint32_t count;
    if (threadIdx.x == 0)
        count = 0;
    __syncthreads();
    for (int64_t u = threadIdx.x; u < U; u += blockDim.x)
        if (flags[u] == kUnitRecompute)
            units[1 + atomicAdd(&count, 1u)] = (uint32_t)u;
    __syncthreads();
    if (threadIdx.x == 0)
        units[0] = count;
}

// ---------------------------------------------------------------------------
// Host launchers.

static int max_ntw_bucket(int rows)
{
    const int ntw = ((rows + 7) / 8 + 7) / 8;
    if (ntw <= 1) return 1;
    if (ntw <= 2) return 2;
    if (ntw <= 4) return 4;
    if (ntw <= 8) return 8;
    return 16;
}

template <typename KernelT>
static cudaError_t prepare(KernelT kernel, size_t smem)
{
    if (smem > 48 * 1024)
        return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)smem);
    return cudaSuccess;
}

#define DGE_DISPATCH_NTW(bucket, D, KERNEL, ...)                         \
    switch (bucket) {                                                     \
    case 1: { auto k = KERNEL<D, 1>; __VA_ARGS__; break; }               \
    case 2: { auto k = KERNEL<D, 2>; __VA_ARGS__; break; }               \
    case 4: { auto k = KERNEL<D, 4>; __VA_ARGS__; break; }               \
    case 8: { auto k = KERNEL<D, 8>; __VA_ARGS__; break; }               \
    default: { auto k = KERNEL<D, 16>; __VA_ARGS__; break; }             \
    }

cudaError_t launch_lse_partial(const TensorDesc &K, const TensorDesc &Q, const Geometry &g,
                               int rows_per_block, int chunk_keys, float2 *partial,
                               cudaStream_t stream, UnitSel units)
{
    const int nrb = (g.R + rows_per_block - 1) / rows_per_block;
    const int nchunks = (g.n + chunk_keys - 1) / chunk_keys;
    const int rows_pad = (min(rows_per_block, g.R) + 7) & ~7;
    const int64_t blocks = grid_for(units, g.U * nrb * nchunks);
    cudaError_t err = cudaSuccess;
    const int bucket = max_ntw_bucket(rows_pad);
    if (g.d == 128) {
        const size_t smem = (size_t)(rows_pad + 2 * kTileKeys) * Pad<128>::kStride * 2;
        DGE_DISPATCH_NTW(bucket, 128, lse_partial_kernel,
                         err = prepare(k, smem);
                         if (err == cudaSuccess) {
                             k<<<(unsigned)blocks, kThreads, smem, stream>>>(
                                 K, Q, g, rows_per_block, nrb, chunk_keys, nchunks, partial,
                                 units);
                             err = cudaGetLastError();
                         })
    } else {
        const size_t smem = (size_t)(rows_pad + 2 * kTileKeys) * Pad<64>::kStride * 2;
        DGE_DISPATCH_NTW(bucket, 64, lse_partial_kernel,
                         err = prepare(k, smem);
                         if (err == cudaSuccess) {
                             k<<<(unsigned)blocks, kThreads, smem, stream>>>(
                                 K, Q, g, rows_per_block, nrb, chunk_keys, nchunks, partial,
                                 units);
                             err = cudaGetLastError();
                         })
    }
    return err;
}

cudaError_t launch_combine_lse(const float2 *partial, int64_t total_rows, int nchunks,
                               float *lse2, cudaStream_t stream, UnitSel units,
                               int rows_per_unit)
{
    const int threads = 256;
    const int64_t blocks = grid_for(units, (total_rows + threads - 1) / threads);
    combine_lse_kernel<<<(unsigned)blocks, threads, 0, stream>>>(partial, total_rows, nchunks,
                                                                  lse2, units, rows_per_unit);
    return cudaGetLastError();
}

cudaError_t launch_colsum_rows(const TensorDesc &K, const TensorDesc &Q, const Geometry &g,
                               int chunk_keys, const float *lse2, float *raw,
                               cudaStream_t stream, UnitSel units)
{
    const int nchunks = (g.P + chunk_keys - 1) / chunk_keys;
    const int rows_pad = (g.R + 7) & ~7;
    const int64_t blocks = grid_for(units, g.U * nchunks);
    cudaError_t err = cudaSuccess;
    const int bucket = max_ntw_bucket(rows_pad);
    if (g.d == 128) {
        const size_t smem = (size_t)(rows_pad + 2 * kTileKeys) * Pad<128>::kStride * 2;
        DGE_DISPATCH_NTW(bucket, 128, colsum_rows_kernel,
                         err = prepare(k, smem);
                         if (err == cudaSuccess) {
                             k<<<(unsigned)blocks, kThreads, smem, stream>>>(
                                 K, Q, g, chunk_keys, nchunks, lse2, raw, units);
                             err = cudaGetLastError();
                         })
    } else {
        const size_t smem = (size_t)(rows_pad + 2 * kTileKeys) * Pad<64>::kStride * 2;
        DGE_DISPATCH_NTW(bucket, 64, colsum_rows_kernel,
                         err = prepare(k, smem);
                         if (err == cudaSuccess) {
                             k<<<(unsigned)blocks, kThreads, smem, stream>>>(
                                 K, Q, g, chunk_keys, nchunks, lse2, raw, units);
                             err = cudaGetLastError();
                         })
    }
    return err;
}

cudaError_t launch_colsum_keys(const TensorDesc &K, const TensorDesc &Q, const Geometry &g,
                               const float *lse2, float *raw, cudaStream_t stream,
                               UnitSel units)
{
    const int nkb = (g.P + kKeyBlock - 1) / kKeyBlock;
    const int64_t blocks = grid_for(units, g.U * nkb);
    cudaError_t err;
    if (g.d == 128) {
        const size_t smem = (size_t)(kKeyBlock + 2 * kRowTile) * Pad<128>::kStride * 2;
        err = prepare(colsum_keys_kernel<128>, smem);
        if (err != cudaSuccess)
            return err;
        colsum_keys_kernel<128><<<(unsigned)blocks, kThreads, smem, stream>>>(K, Q, g, nkb, lse2,
                                                                              raw, units);
    } else {
        const size_t smem = (size_t)(kKeyBlock + 2 * kRowTile) * Pad<64>::kStride * 2;
        err = prepare(colsum_keys_kernel<64>, smem);
        if (err != cudaSuccess)
            return err;
        colsum_keys_kernel<64><<<(unsigned)blocks, kThreads, smem, stream>>>(K, Q, g, nkb, lse2,
                                                                             raw, units);
    }
    return cudaGetLastError();
}

cudaError_t launch_recompute_units(const TensorDesc &K, const TensorDesc &Q, const Geometry &g,
                                   float2 *partial, float *lse2, float *raw, const uint32_t *list,
                                   cudaStream_t stream)
{
    int dev = 0, sms = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err == cudaSuccess)
        err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (err != cudaSuccess)
        return err;
    const int64_t blocks = g.U < sms ? g.U : sms;
    const int rows_pad = (g.R + 7) & ~7;
    const int bucket = max_ntw_bucket(rows_pad);
    if (g.d == 128) {
        const size_t smem = (size_t)(rows_pad + 2 * kTileKeys) * Pad<128>::kStride * 2;
        DGE_DISPATCH_NTW(bucket, 128, recompute_units_kernel,
                         err = prepare(k, smem);
                         if (err == cudaSuccess) {
                             k<<<(unsigned)blocks, kThreads, smem, stream>>>(K, Q, g, partial,
                                                                             lse2, raw, list);
                             err = cudaGetLastError();
                         })
    } else {
        const size_t smem = (size_t)(rows_pad + 2 * kTileKeys) * Pad<64>::kStride * 2;
        DGE_DISPATCH_NTW(bucket, 64, recompute_units_kernel,
                         err = prepare(k, smem);
                         if (err == cudaSuccess) {
                             k<<<(unsigned)blocks, kThreads, smem, stream>>>(K, Q, g, partial,
                                                                             lse2, raw, list);
                             err = cudaGetLastError();
                         })
    }
    return err;
}

cudaError_t launch_tail_rows(const TensorDesc &K, const TensorDesc &Q, const Geometry &g,
                             int rows, int nrb, float *part, int nparts, int slot, int r4,
                             cudaStream_t stream)
{
    int dev = 0, sms = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err == cudaSuccess)
        err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (err != cudaSuccess)
        return err;
    const int64_t subs = g.U * nrb;
    const int64_t blocks = subs < (int64_t)sms * 8 ? subs : (int64_t)sms * 8;
    const int rows_pad = (rows + 7) & ~7;
    const int bucket = max_ntw_bucket(rows_pad);
    if (g.d == 128) {
        const size_t smem = (size_t)(rows_pad + kTileKeys) * Pad<128>::kStride * 2;
        DGE_DISPATCH_NTW(bucket, 128, tail_rows_kernel,
                         err = prepare(k, smem);
                         if (err == cudaSuccess) {
                             k<<<(unsigned)blocks, kThreads, smem, stream>>>(
                                 K, Q, g, rows, nrb, part, nparts, slot, r4);
                             err = cudaGetLastError();
                         })
    } else {
        const size_t smem = (size_t)(rows_pad + kTileKeys) * Pad<64>::kStride * 2;
        DGE_DISPATCH_NTW(bucket, 64, tail_rows_kernel,
                         err = prepare(k, smem);
                         if (err == cudaSuccess) {
                             k<<<(unsigned)blocks, kThreads, smem, stream>>>(
                                 K, Q, g, rows, nrb, part, nparts, slot, r4);
                             err = cudaGetLastError();
                         })
    }
    return err;
}

cudaError_t launch_collect_units(const uint32_t *flags, int64_t U, uint32_t *units,
                                 cudaStream_t stream)
{
    collect_units_kernel<<<1, 1024, 0, stream>>>(flags, U, units);
    return cudaGetLastError();
}

}  // namespace dge
