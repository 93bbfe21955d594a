// select_compact.cu -- pooling, per-unit top-B selection, and the K/V gather.
//
// Pooling (App. B, max-pool kernel 7; avg-pool for PyramidKV's workload) runs
// along positions of [0, P).  Selection is the retention rule of Alg. 1
// (I <- R_E(s, B - w)) with the kept set written in temporal order (App. E):
// a radix select finds the exact (B - sinks - tail)-th largest score, then a
// stable, position-ordered compaction keeps every larger score and the lowest
// positions among the scores equal to it.  The gather copies K and V rows at
// the kept positions into the packed compact cache (App. E).
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace dge {

// ---------------------------------------------------------------------------
// Pooling: out[u][j] = pool over raw[u][max(0, j - r) .. min(P - 1, j + r)].
__global__ void pool_kernel(const float *__restrict__ raw, float *__restrict__ out, int64_t U,
                            int P, int pool, int kernel)
{
    const int64_t total = U * (int64_t)P;
    const int r = kernel / 2;
    const float inv_kernel = 1.0f / (float)kernel;  // avg-pool: in-range sum times 1/K
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t u = i / P;
        const int j = (int)(i - u * P);
        const float *row = raw + u * P;
        if (pool == DGE_POOL_NONE) {
            out[i] = row[j];
            continue;
        }
        const int lo = max(0, j - r), hi = min(P - 1, j + r);
        if (pool == DGE_POOL_MAX) {
            float m = -INFINITY;
            for (int q = lo; q <= hi; ++q)
                m = fmaxf(m, row[q]);
            out[i] = m;
        } else {
            float s = 0.f;
            for (int q = lo; q <= hi; ++q)
                s += row[q];
            out[i] = s * inv_kernel;
        }
    }
}

cudaError_t launch_pool(const float *raw, float *out, int64_t U, int P, int pool, int kernel,
                        cudaStream_t stream)
{
    const int64_t total = U * (int64_t)P;
    if (total == 0)
        return cudaSuccess;
    const int threads = 256;
    const int64_t want = (total + threads - 1) / threads;
    const int64_t blocks = want < 152 * 64 ? want : 152 * 64;
    pool_kernel<<<(unsigned)blocks, threads, 0, stream>>>(raw, out, U, P, pool, kernel);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Selection.  One CTA of kSelThreads per unit.

constexpr int kSelThreads = 1024;
constexpr int kSelWarps = kSelThreads / 32;
constexpr int kSmemKeys = 53248;  // candidates held in shared memory (208 KiB)

struct SelectParams {
    Geometry g;
    LayerTable layers;
    int64_t lead = 0;   // pool_select: a CTA prefetches the raw scores of unit u + lead into L2
};

__device__ __forceinline__ int64_t unit_row_base(const SelectParams &p, int64_t u, int &budget)
{
    int l, bb, h;
    unit_coords(p.g, u, l, bb, h);
    budget = p.layers.budget[l];
    return p.layers.row_base[l] + (int64_t)(bb * p.g.Hkv + h) * budget;
}

// Exclusive scan of one int per warp (cnt[0..kSelWarps)) into base[], by warp 0.
__device__ __forceinline__ void scan_warp_counts(const int *cnt, int *base)
{
    if (threadIdx.x < 32) {
        const int lane = threadIdx.x;
        const int v = lane < kSelWarps ? cnt[lane] : 0;
        int incl = v;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const int o = __shfl_up_sync(0xffffffffu, incl, off);
            if (lane >= off)
                incl += o;
        }
        if (lane < kSelWarps)
            base[lane] = incl - v;
    }
}

constexpr int kRadixBits = 11;
constexpr int kRadixBins = 1 << kRadixBits;
static_assert(kRadixBins == 2 * kSelThreads, "two bins per thread in the bin search");

// Shared-memory scratch of the selection helpers.
struct SelScratch {
    uint32_t hist[kRadixBins];
    uint32_t bincnt;   // keys in the bin a pass selected
    int warp_a[kSelWarps], warp_b[kSelWarps], warp_c[kSelWarps];
    uint32_t prefix;
    int rank;
};

// T = the keep-th largest of the C keys key_at(0 .. C-1) (1 <= keep < C) and need_eq = how
// many keys equal to T are kept (those at the lowest positions).  Radix select from the
// highest bit in which the smallest and the largest key differ (the bits above are common to
// every key), kRadixBits a pass: the scores of one unit share a few exponents, so histograms
// of the top bits would put nearly every key in a handful of bins, whose shared-memory atomics
// serialise.  The passes stop early when every key of the selected bin is kept (its count is
// the rank still wanted): T is then the bin's lowest possible key (the prefix, lower bits
// zero) and need_eq = C, which keeps exactly the keys >= T.  After two 11-bit passes the bin
// nearly always holds one key, so the third pass is skipped.  kBatch > 1 (keys in global
// memory): each thread loads kBatch keys before it uses any, so their latencies overlap
// instead of adding up between the shared-memory atomics.  Called by every thread of a block
// of kSelThreads.
template <int kBatch = 1, typename KeyAt>
__device__ void radix_threshold(KeyAt key_at, int C, int keep, SelScratch &sc, uint32_t &T,
                                int &need_eq, uint32_t kmin = 0xffffffffu, uint32_t kmax = 0u,
                                bool have_range = false)
{
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (!have_range)
        for (int j0 = tid; j0 < C; j0 += kBatch * kSelThreads) {
            uint32_t kb[kBatch];
#pragma unroll
            for (int q = 0; q < kBatch; ++q) {
                const int j = j0 + q * kSelThreads;
                kb[q] = j < C ? key_at(j) : 0u;
            }
#pragma unroll
            for (int q = 0; q < kBatch; ++q)
                if (j0 + q * kSelThreads < C) {
                    kmin = min(kmin, kb[q]);
                    kmax = max(kmax, kb[q]);
                }
        }
    kmin = __reduce_min_sync(0xffffffffu, kmin);
    kmax = __reduce_max_sync(0xffffffffu, kmax);
    if (lane == 0) {
        sc.warp_a[warp] = (int)kmin;
        sc.warp_b[warp] = (int)kmax;
    }
    __syncthreads();
    if (warp == 0) {
        const uint32_t a = __reduce_min_sync(0xffffffffu, (uint32_t)sc.warp_a[lane]);
        const uint32_t b = __reduce_max_sync(0xffffffffu, (uint32_t)sc.warp_b[lane]);
        if (lane == 0) {
            sc.warp_c[0] = (int)a;
            sc.warp_c[1] = (int)b;
        }
    }
    __syncthreads();
    kmin = (uint32_t)sc.warp_c[0];
    kmax = (uint32_t)sc.warp_c[1];
    const uint32_t diff = kmin ^ kmax;
    const int top = diff ? 31 - __clz(diff) : -1;   // bits [0, top] vary
    uint32_t mask = top >= 31 ? 0u : ~((2u << top) - 1u);
    uint32_t prefix = kmax & mask;
    int rank = keep;  // 1-based rank of T among the keys matching `prefix`, from the top
    const int npass = (top + kRadixBits) / kRadixBits;
    bool whole_bin = false;
#pragma unroll 1
    for (int pass = 0; pass < npass; ++pass) {
        const int hi = top - kRadixBits * pass;         // highest bit of this pass
        const int shift = hi >= kRadixBits - 1 ? hi - (kRadixBits - 1) : 0;
        const uint32_t bmask = (2u << (hi - shift)) - 1u;
        for (int i = tid; i < kRadixBins; i += kSelThreads)
            sc.hist[i] = 0;
        __syncthreads();
        for (int j0 = tid; j0 < C; j0 += kBatch * kSelThreads) {
            uint32_t kb[kBatch];
#pragma unroll
            for (int q = 0; q < kBatch; ++q) {
                const int j = j0 + q * kSelThreads;
                kb[q] = j < C ? key_at(j) : 0u;
            }
#pragma unroll
            for (int q = 0; q < kBatch; ++q)
                if (j0 + q * kSelThreads < C && (kb[q] & mask) == prefix)
                    atomicAdd(&sc.hist[(kb[q] >> shift) & bmask], 1u);
        }
        __syncthreads();
        {
            // Counts from the top bin down: thread t holds bins tb and tb - 1, tb = top - 2t
            // (bins above bmask are empty); a block scan gives the count above each pair.
            const int tb = kRadixBins - 1 - 2 * tid;
            const uint32_t c_hi = sc.hist[tb], c_lo = sc.hist[tb - 1];
            const uint32_t local = c_hi + c_lo;
            uint32_t incl = local;
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const uint32_t o = __shfl_up_sync(0xffffffffu, incl, off);
                if (lane >= off)
                    incl += o;
            }
            if (lane == 31)
                sc.warp_a[warp] = (int)incl;
            __syncthreads();
            if (warp == 0) {
                const uint32_t v = (uint32_t)sc.warp_a[lane];
                uint32_t wi = v;
#pragma unroll
                for (int off = 1; off < 32; off <<= 1) {
                    const uint32_t o = __shfl_up_sync(0xffffffffu, wi, off);
                    if (lane >= off)
                        wi += o;
                }
                sc.warp_b[lane] = (int)(wi - v);
            }
            __syncthreads();
            const uint32_t run = (uint32_t)sc.warp_b[warp] + incl - local;
            if (run < (uint32_t)rank && run + local >= (uint32_t)rank) {
                const bool hi_bin = run + c_hi >= (uint32_t)rank;
                sc.prefix = prefix | ((uint32_t)(hi_bin ? tb : tb - 1) << shift);
                sc.rank = rank - (int)(hi_bin ? run : run + c_hi);
                sc.bincnt = hi_bin ? c_hi : c_lo;
            }
        }
        __syncthreads();
        prefix = sc.prefix;
        rank = sc.rank;
        mask |= bmask << shift;
        if ((uint32_t)rank == sc.bincnt) {   // the whole bin is kept
            whole_bin = true;
            break;
        }
    }
    T = npass == 0 ? kmax : prefix;   // npass == 0: every key is equal
    need_eq = whole_bin ? C : rank;
}

// Writes the positions s0 + j of the kept keys -- every key above T and the first need_eq keys
// equal to T -- in ascending order to out[0 .. keep).  Warp w walks a contiguous range of the
// candidates twice: it counts its keys above and equal to T, then (after two scans over the
// warps) writes its kept positions; the equal keys a warp keeps follow from the equal keys
// before its range.  kBatch as for radix_threshold (a warp loads kBatch rows of 32 keys, then
// uses them in order).  Called by every thread of a block of kSelThreads.
template <int kBatch = 1, typename KeyAt>
__device__ void ordered_compaction(KeyAt key_at, int C, uint32_t T, int need_eq, int keep, int s0,
                                   int32_t *out, SelScratch &sc)
{
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const uint32_t lt_mask = (1u << lane) - 1u;
    const int per_w = ((C + kSelWarps - 1) / kSelWarps + 31) & ~31;
    const int w_lo = min(C, warp * per_w), w_hi = min(C, w_lo + per_w);
    int eq_cnt = 0, gt_cnt = 0;
    for (int c0 = w_lo; c0 < w_hi; c0 += 32 * kBatch) {
        uint32_t kb[kBatch];
#pragma unroll
        for (int q = 0; q < kBatch; ++q) {
            const int j = c0 + 32 * q + lane;
            kb[q] = j < w_hi ? key_at(j) : 0u;
        }
#pragma unroll
        for (int q = 0; q < kBatch; ++q) {
            const int j = c0 + 32 * q + lane;
            eq_cnt += __popc(__ballot_sync(0xffffffffu, j < w_hi && kb[q] == T));
            gt_cnt += __popc(__ballot_sync(0xffffffffu, j < w_hi && kb[q] > T));
        }
    }
    if (lane == 0) {
        sc.warp_a[warp] = eq_cnt;
        sc.warp_b[warp] = gt_cnt;
    }
    __syncthreads();
    scan_warp_counts(sc.warp_a, sc.warp_c);
    __syncthreads();
    const int eq_base = sc.warp_c[warp];
    const int eq_kept = min(eq_cnt, max(0, need_eq - eq_base));
    __syncthreads();                      // every warp has read its equal-key offset
    if (lane == 0)
        sc.warp_a[warp] = sc.warp_b[warp] + eq_kept;
    __syncthreads();
    scan_warp_counts(sc.warp_a, sc.warp_c);
    __syncthreads();
    int sel_run = sc.warp_c[warp], eq_run = eq_base;
    for (int c0 = w_lo; c0 < w_hi; c0 += 32 * kBatch) {
        uint32_t kb[kBatch];
#pragma unroll
        for (int q = 0; q < kBatch; ++q) {
            const int j = c0 + 32 * q + lane;
            kb[q] = j < w_hi ? key_at(j) : 0u;
        }
#pragma unroll
        for (int q = 0; q < kBatch; ++q) {
            const int j = c0 + 32 * q + lane;
            const uint32_t k = kb[q];
            const bool eq = j < w_hi && k == T;
            const uint32_t eqb = __ballot_sync(0xffffffffu, eq);
            const bool sel =
                j < w_hi && (k > T || (eq && eq_run + __popc(eqb & lt_mask) < need_eq));
            const uint32_t selb = __ballot_sync(0xffffffffu, sel);
            const int pos = sel_run + __popc(selb & lt_mask);
            if (sel && pos < keep)
                out[pos] = s0 + j;
            sel_run += __popc(selb);
            eq_run += __popc(eqb);
        }
    }
}

// Block-wide exclusive scan of one value per thread (thread order); every thread of a block
// of kSelThreads calls it.  Returns the sum over lower threads; *total (nullable) = the sum.
__device__ __forceinline__ int block_exclusive_scan(int v, SelScratch &sc, int *total = nullptr)
{
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    int incl = v;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const int o = __shfl_up_sync(0xffffffffu, incl, off);
        if (lane >= off)
            incl += o;
    }
    if (lane == 31)
        sc.warp_a[warp] = incl;
    __syncthreads();
    const int wv = lane < kSelWarps ? sc.warp_a[lane] : 0;
    int wi = wv;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const int o = __shfl_up_sync(0xffffffffu, wi, off);
        if (lane >= off)
            wi += o;
    }
    const int before = __shfl_sync(0xffffffffu, wi - wv, warp);
    if (total)
        *total = __shfl_sync(0xffffffffu, wi, 31);
    __syncthreads();   // warp_a is free again
    return before + incl - v;
}

// ordered_compaction for C <= 32 * kSelThreads in one pass over the keys: warp w's range is
// cut into 32-key segments, and a ballot per segment hands lane s the masks of segment s (keys
// above T, keys equal to T).  Two block scans give each lane its share of the equal keys and
// its first output slot; it then writes its kept positions in order.
template <typename KeyAt>
__device__ void ordered_compaction_masks(KeyAt key_at, int C, uint32_t T, int need_eq, int keep,
                                         int s0, int32_t *out, SelScratch &sc)
{
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int per_w = ((C + kSelWarps - 1) / kSelWarps + 31) & ~31;   // <= 1024
    const int w_lo = min(C, warp * per_w), w_hi = min(C, w_lo + per_w);
    uint32_t gtm = 0, eqm = 0;
    for (int q = 0; q < per_w / 32; ++q) {
        const int j = w_lo + 32 * q + lane;
        const uint32_t k = j < w_hi ? key_at(j) : 0u;
        const uint32_t gb = __ballot_sync(0xffffffffu, j < w_hi && k > T);
        const uint32_t eb = __ballot_sync(0xffffffffu, j < w_hi && k == T);
        if (lane == q) {
            gtm = gb;
            eqm = eb;
        }
    }
    // Equal keys before this segment; this lane keeps the lowest of its own up to need_eq.
    const int eq_before = block_exclusive_scan(__popc(eqm), sc);
    int take = min(__popc(eqm), max(0, need_eq - eq_before));
    uint32_t sel = gtm;
    for (uint32_t e = eqm; take > 0; --take) {
        const uint32_t low = e & (0u - e);
        sel |= low;
        e ^= low;
    }
    int pos = block_exclusive_scan(__popc(sel), sc);
    const int seg0 = s0 + w_lo + 32 * lane;
    while (sel) {
        const int b = __ffs(sel) - 1;
        if (pos < keep)
            out[pos] = seg0 + b;
        ++pos;
        sel &= sel - 1;
    }
}

template <bool SMEM>
__global__ void __launch_bounds__(kSelThreads)
select_kernel(const float *__restrict__ scores, int32_t *__restrict__ idx, SelectParams p)
{
    extern __shared__ __align__(16) uint32_t skeys[];
    __shared__ SelScratch scr;

    const int64_t u = blockIdx.x;
    const Geometry &g = p.g;
    int budget;
    int32_t *out = idx + unit_row_base(p, u, budget);
    const int P = g.P, s0 = g.sinks, tail = g.n - g.P;
    const int C = P - s0;                    // candidates [s0, P)
    const int keep = budget - s0 - tail;     // candidates to keep
    const float *sc = scores + u * (int64_t)P + s0;

    for (int j = threadIdx.x; j < s0; j += kSelThreads)
        out[j] = j;
    for (int j = threadIdx.x; j < tail; j += kSelThreads)
        out[s0 + keep + j] = P + j;
    if (keep <= 0)
        return;
    if (keep >= C) {
        for (int j = threadIdx.x; j < C; j += kSelThreads)
            out[s0 + j] = s0 + j;
        return;
    }

    if (SMEM) {
        for (int j = threadIdx.x; j < C; j += kSelThreads)
            skeys[j] = float_key(sc[j]);
        __syncthreads();
    }
    auto key_at = [&](int j) -> uint32_t { return SMEM ? skeys[j] : float_key(sc[j]); };

    uint32_t T;
    int need_eq;
    constexpr int kBatch = SMEM ? 1 : 8;   // keys in global memory: batched loads
    radix_threshold<kBatch>(key_at, C, keep, scr, T, need_eq);
    if (C <= 32 * kSelThreads)
        ordered_compaction_masks(key_at, C, T, need_eq, keep, s0, out + s0, scr);
    else
        ordered_compaction<kBatch>(key_at, C, T, need_eq, keep, s0, out + s0, scr);
}

cudaError_t launch_select(const Geometry &g, const LayerTable &layers, const float *scores,
                          int32_t *idx, cudaStream_t stream)
{
    SelectParams p;
    p.g = g;
    p.layers = layers;
    const int C = g.P - g.sinks;
    if (C <= kSmemKeys) {
        const size_t smem = (size_t)max(C, 1) * sizeof(uint32_t);
        if (smem > 48 * 1024) {
            cudaError_t err = cudaFuncSetAttribute(
                select_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            if (err != cudaSuccess)
                return err;
        }
        select_kernel<true><<<(unsigned)g.U, kSelThreads, smem, stream>>>(scores, idx, p);
    } else {
        select_kernel<false><<<(unsigned)g.U, kSelThreads, 0, stream>>>(scores, idx, p);
    }
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Pooling and selection fused (the evict path, P <= kPsMaxP): one CTA per unit loads the
// unit's raw scores into shared memory once, pools them (the same arithmetic and order as
// pool_kernel, so the pooled values are bit-identical), optionally writes them out, and
// selects from the shared-memory copy.  The kernel is latency- and issue-bound (one CTA per
// SM, block barriers between its steps): pooling reads each score once from shared memory (a
// 16-byte load gives a lane four consecutive positions, the neighbours come by shuffles; R
// guard cells of the pool's neutral value on each side of the row leave every window sum or
// max bit-identical to the clipped one), the key range comes with the key write, the radix
// select's bin search is a block scan, and the position-ordered compaction reads the keys
// once.

constexpr int kPsThreads = 1024;
constexpr int kPsPer = 32;                       // positions pooled per thread (registers)
constexpr int kPsMaxP = kPsThreads * kPsPer;     // 32768

// Pooled value at position j of a row of P raw scores in shared memory.  R > 0: the pool
// radius known at compile time (interior positions unrolled); R < 0: radius r at run time.
template <int POOL, int R>
__device__ __forceinline__ float pool_at(const float *sraw, int j, int P, int r, int kernel)
{
    if (POOL == DGE_POOL_NONE)
        return sraw[j];
    const int rr = R > 0 ? R : r;
    const int lo = max(0, j - rr), hi = min(P - 1, j + rr);
    float x = POOL == DGE_POOL_MAX ? -INFINITY : 0.f;
    if (R > 0 && j >= R && j + R < P) {
#pragma unroll
        for (int q = -R; q <= R; ++q)
            x = POOL == DGE_POOL_MAX ? fmaxf(x, sraw[j + q]) : x + sraw[j + q];
    } else {
        for (int q = lo; q <= hi; ++q)
            x = POOL == DGE_POOL_MAX ? fmaxf(x, sraw[q]) : x + sraw[q];
    }
    return POOL == DGE_POOL_AVG ? x * (1.0f / (float)kernel) : x;
}

constexpr int kPsGuard = 4;                      // guard cells on each side of the row

template <int POOL, int R>
__global__ void __launch_bounds__(kPsThreads, 1)
pool_select_kernel(const float *__restrict__ raw, float *__restrict__ pooled_out,
                   int32_t *__restrict__ idx, SelectParams p, int kernel)
{
    // [guard][P rounded up to 128][guard]: raw scores, then pooled keys in place
    extern __shared__ __align__(16) uint32_t sbuf[];
    __shared__ SelScratch sc;

    const int tid = threadIdx.x;
    const int64_t u = blockIdx.x;
    const Geometry &g = p.g;
    int budget;
    int32_t *out = idx + unit_row_base(p, u, budget);
    const int P = g.P, s0 = g.sinks, tail = g.n - g.P;
    const int C = P - s0;                    // candidates [s0, P)
    const int keep = budget - s0 - tail;     // candidates to keep

    // Raw scores to shared memory, pooled values to registers, then keys in place.
    const float *row = raw + u * (int64_t)P;
    // The unit that will most likely take this SM next (one CTA per SM: u + the SM count) has
    // its raw scores prefetched into L2 now, so its load comes from L2.  Only whole 16-byte
    // pieces inside that row are named (the bulk prefetch's alignment rule).
    if (tid == 0 && p.lead > 0 && u + p.lead < g.U) {
        const uintptr_t a0 = reinterpret_cast<uintptr_t>(raw + (u + p.lead) * (int64_t)P);
        const uintptr_t lo = (a0 + 15) & ~uintptr_t(15);
        const uintptr_t hi = (a0 + (uintptr_t)P * 4) & ~uintptr_t(15);
        if (hi > lo)
            asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(lo),
                         "r"((uint32_t)(hi - lo))
                         : "memory");
    }
    uint32_t *skey = sbuf + kPsGuard;
    float *sraw = reinterpret_cast<float *>(skey);
    for (int j = tid; j < P; j += kPsThreads)
        sraw[j] = row[j];
    if (tid < kPsGuard) {
        const float neutral = POOL == DGE_POOL_MAX ? -INFINITY : 0.f;
        sraw[-1 - tid] = neutral;
        sraw[P + tid] = neutral;
    }
    __syncthreads();
    // Position of value i of this thread: chunks of 128 positions, chunk c to warp c % 32;
    // a lane holds 4 consecutive positions of each of its chunks (compile-time radius), or
    // positions tid + 1024 i (run-time radius).
    constexpr bool kChunked = R >= 0 && R <= kPsGuard;
    const int lane = tid & 31, warp = tid >> 5;
    auto pos_of = [&](int i) {
        return kChunked ? 128 * (warp + 32 * (i >> 2)) + 4 * lane + (i & 3) : tid + i * kPsThreads;
    };
    float v[kPsPer];
    if constexpr (kChunked) {
        constexpr int RR = R > 0 ? R : 0;
#pragma unroll
        for (int c = 0; c < kPsPer / 4; ++c) {
            const int base = 128 * (warp + 32 * c);
            if (base < P) {   // warp-uniform
                const float4 a = *reinterpret_cast<const float4 *>(sraw + base + 4 * lane);
                // w[4 + t] = position 4 * lane + t of the chunk, t = -4 .. 7.
                float w[12];
                w[4] = a.x;
                w[5] = a.y;
                w[6] = a.z;
                w[7] = a.w;
#pragma unroll
                for (int t = 1; t <= RR; ++t) {
                    const float left = __shfl_up_sync(0xffffffffu, w[8 - t], 1);
                    const float right = __shfl_down_sync(0xffffffffu, w[3 + t], 1);
                    w[4 - t] = lane == 0 ? sraw[base - t] : left;
                    w[7 + t] = lane == 31 ? sraw[base + 127 + t] : right;
                }
#pragma unroll
                for (int t = 0; t < 4; ++t) {
                    if (POOL == DGE_POOL_NONE) {
                        v[4 * c + t] = w[4 + t];
                        continue;
                    }
                    float x = POOL == DGE_POOL_MAX ? -INFINITY : 0.f;
#pragma unroll
                    for (int q = -RR; q <= RR; ++q)
                        x = POOL == DGE_POOL_MAX ? fmaxf(x, w[4 + t + q]) : x + w[4 + t + q];
                    v[4 * c + t] = POOL == DGE_POOL_AVG ? x * (1.0f / (float)(2 * RR + 1)) : x;
                }
            } else {
#pragma unroll
                for (int t = 0; t < 4; ++t)
                    v[4 * c + t] = 0.f;
            }
        }
    } else {
#pragma unroll
        for (int i = 0; i < kPsPer; ++i) {
            const int j = tid + i * kPsThreads;
            v[i] = j < P ? pool_at<POOL, R>(sraw, j, P, kernel / 2, kernel) : 0.f;
        }
    }
    __syncthreads();
    float *pout = pooled_out ? pooled_out + u * (int64_t)P : nullptr;
    uint32_t kmin = 0xffffffffu, kmax = 0u;   // range of the candidate keys [s0, P)
    uint32_t kv[kPsPer];
#pragma unroll
    for (int i = 0; i < kPsPer; ++i) {
        const int j = pos_of(i);
        kv[i] = float_key(v[i]);
        if (j < P) {
            if (pout)
                pout[j] = v[i];
            if (j >= s0) {
                kmin = min(kmin, kv[i]);
                kmax = max(kmax, kv[i]);
            }
        }
    }
    if constexpr (kChunked) {
        // Four consecutive keys at once (positions past P land in the chunk padding).
#pragma unroll
        for (int c = 0; c < kPsPer / 4; ++c)
            if (pos_of(4 * c) < P)
                *reinterpret_cast<uint4 *>(skey + pos_of(4 * c)) =
                    make_uint4(kv[4 * c], kv[4 * c + 1], kv[4 * c + 2], kv[4 * c + 3]);
    } else {
#pragma unroll
        for (int i = 0; i < kPsPer; ++i)
            if (pos_of(i) < P)
                skey[pos_of(i)] = kv[i];
    }
    __syncthreads();

    for (int j = tid; j < s0; j += kPsThreads)
        out[j] = j;
    for (int j = tid; j < tail; j += kPsThreads)
        out[s0 + keep + j] = P + j;
    if (keep <= 0)
        return;
    if (keep >= C) {
        for (int j = tid; j < C; j += kPsThreads)
            out[s0 + j] = s0 + j;
        return;
    }
    const uint32_t *keys = skey + s0;
    auto key_at = [&](int j) -> uint32_t { return keys[j]; };
    uint32_t T;
    int need_eq;
    radix_threshold(key_at, C, keep, sc, T, need_eq, kmin, kmax, true);
    ordered_compaction_masks(key_at, C, T, need_eq, keep, s0, out + s0, sc);
}

bool pool_select_supported(const Geometry &g) { return g.P <= kPsMaxP; }

cudaError_t launch_pool_select(const Geometry &g, const LayerTable &layers, const float *raw,
                               float *pooled_out, int32_t *idx, cudaStream_t stream)
{
    SelectParams p;
    p.g = g;
    p.layers = layers;
    int dev = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess)
        e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess)
        return e;
    p.lead = sms;
    // The row rounded up to whole 128-position chunks, with guard cells on both sides.
    const size_t smem = (size_t)(((max(g.P, 1) + 127) & ~127) + 2 * kPsGuard) * sizeof(uint32_t);
    using KernT = void (*)(const float *, float *, int32_t *, SelectParams, int);
    KernT kern;
    if (g.pool == DGE_POOL_MAX)
        kern = g.pool_kernel == 7 ? pool_select_kernel<DGE_POOL_MAX, 3>
                                  : pool_select_kernel<DGE_POOL_MAX, -1>;
    else if (g.pool == DGE_POOL_AVG)
        kern = g.pool_kernel == 7 ? pool_select_kernel<DGE_POOL_AVG, 3>
                                  : pool_select_kernel<DGE_POOL_AVG, -1>;
    else
        kern = pool_select_kernel<DGE_POOL_NONE, 0>;
    cudaError_t err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)smem);
    if (err != cudaSuccess)
        return err;
    kern<<<(unsigned)g.U, kPsThreads, smem, stream>>>(raw, pooled_out, idx, p, g.pool_kernel);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Pooling and selection fused for rows longer than kPsMaxP (the 128K-key caches), where the
// keys do not fit in shared memory: one CTA per unit pools its row tile by tile through
// shared memory (kPlTile positions and kPsGuard guard cells of the pool's neutral value on
// each side, the same arithmetic and order as pool_kernel, so the pooled values are
// bit-identical), writes the pooled row out and tracks the candidates' key range on the way,
// then runs the radix select and the ordered compaction on keys read back from global memory
// (L2: the CTA has just written them), kBatch at a time.  This replaces pool_kernel plus
// select_kernel, whose selection read each key with its own memory latency.

constexpr int kPlTile = 32768;   // positions pooled per shared-memory tile (128 KB)

template <int POOL, int R>
__global__ void __launch_bounds__(kSelThreads, 1)
pool_select_large_kernel(const float *__restrict__ raw, float *pooled, int32_t *__restrict__ idx,
                         SelectParams p, int kernel)
{
    extern __shared__ __align__(16) float stile[];   // [kPsGuard][kPlTile][kPsGuard]
    __shared__ SelScratch sc;

    const int tid = threadIdx.x;
    const int64_t u = blockIdx.x;
    const Geometry &g = p.g;
    int budget;
    int32_t *out = idx + unit_row_base(p, u, budget);
    const int P = g.P, s0 = g.sinks, tail = g.n - g.P;
    const int C = P - s0;                    // candidates [s0, P)
    const int keep = budget - s0 - tail;     // candidates to keep
    const float *row = raw + u * (int64_t)P;
    float *prow = pooled + u * (int64_t)P;
    const int r = R >= 0 ? R : kernel / 2;   // <= kPsGuard (the launcher checks)
    const float neutral = POOL == DGE_POOL_MAX ? -INFINITY : 0.f;
    const float inv_kernel = 1.0f / (float)kernel;

    uint32_t kmin = 0xffffffffu, kmax = 0u;   // range of the candidate keys [s0, P)
    for (int t0 = 0; t0 < P; t0 += kPlTile) {
        const int len = min(kPlTile, P - t0);
        for (int i = tid; i < len + 2 * kPsGuard; i += kSelThreads) {
            const int j = t0 - kPsGuard + i;
            stile[i] = j >= 0 && j < P ? row[j] : neutral;
        }
        __syncthreads();
        for (int i = tid; i < len; i += kSelThreads) {
            const float *w = stile + kPsGuard + i;
            float x = neutral;
            if (R > 0) {
#pragma unroll
                for (int q = -(R > 0 ? R : 0); q <= (R > 0 ? R : 0); ++q)
                    x = POOL == DGE_POOL_MAX ? fmaxf(x, w[q]) : x + w[q];
            } else {
                for (int q = -r; q <= r; ++q)
                    x = POOL == DGE_POOL_MAX ? fmaxf(x, w[q]) : x + w[q];
            }
            if (POOL == DGE_POOL_AVG)
                x *= inv_kernel;
            const int j = t0 + i;
            prow[j] = x;
            if (j >= s0) {
                const uint32_t k = float_key(x);
                kmin = min(kmin, k);
                kmax = max(kmax, k);
            }
        }
        __syncthreads();   // the tile is read before the next one overwrites it
    }

    for (int j = tid; j < s0; j += kSelThreads)
        out[j] = j;
    for (int j = tid; j < tail; j += kSelThreads)
        out[s0 + keep + j] = P + j;
    if (keep <= 0)
        return;
    if (keep >= C) {
        for (int j = tid; j < C; j += kSelThreads)
            out[s0 + j] = s0 + j;
        return;
    }
    // Keys from the pooled row this CTA has just written: loads through L2 (ld.global.cg),
    // never the read-only path, which need not see this kernel's own stores.
    const float *keys = prow + s0;
    auto key_at = [&](int j) -> uint32_t { return float_key(__ldcg(keys + j)); };
    uint32_t T;
    int need_eq;
    radix_threshold<8>(key_at, C, keep, sc, T, need_eq, kmin, kmax, true);
    if (C <= 32 * kSelThreads)
        ordered_compaction_masks(key_at, C, T, need_eq, keep, s0, out + s0, sc);
    else
        ordered_compaction<8>(key_at, C, T, need_eq, keep, s0, out + s0, sc);
}

bool pool_select_large_supported(const Geometry &g)
{
    return g.P > kPsMaxP && (g.pool == DGE_POOL_AVG || g.pool == DGE_POOL_MAX) &&
           g.pool_kernel >= 1 && g.pool_kernel / 2 <= kPsGuard;
}

cudaError_t launch_pool_select_large(const Geometry &g, const LayerTable &layers, const float *raw,
                                     float *pooled, int32_t *idx, cudaStream_t stream)
{
    SelectParams p;
    p.g = g;
    p.layers = layers;
    const size_t smem = (size_t)(kPlTile + 2 * kPsGuard) * sizeof(float);
    using KernT = void (*)(const float *, float *, int32_t *, SelectParams, int);
    KernT kern;
    if (g.pool == DGE_POOL_MAX)
        kern = g.pool_kernel == 7 ? pool_select_large_kernel<DGE_POOL_MAX, 3>
                                  : pool_select_large_kernel<DGE_POOL_MAX, -1>;
    else
        kern = g.pool_kernel == 7 ? pool_select_large_kernel<DGE_POOL_AVG, 3>
                                  : pool_select_large_kernel<DGE_POOL_AVG, -1>;
    cudaError_t err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)smem);
    if (err != cudaSuccess)
        return err;
    kern<<<(unsigned)g.U, kSelThreads, smem, stream>>>(raw, pooled, idx, p, g.pool_kernel);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Block-granular selection (the selection ladder's fixed-block rung; the rule as read in
// dge.h): one CTA per unit forms the block sums (fp32, positions in order), sorts the
// (sum key, block index) pairs descending in shared memory (bitonic; pairs are unique, so the
// order is deterministic), walks the ranking to take whole blocks while they fit and a prefix
// of the first that does not, and writes the taken positions in block order (ascending).

constexpr int kBsThreads = 1024;

__global__ void __launch_bounds__(kBsThreads, 1)
block_select_kernel(const float *__restrict__ scores, int32_t *__restrict__ idx, SelectParams p,
                    int bs, int n2)
{
    extern __shared__ __align__(16) uint64_t items[];          // [n2]
    int *take = reinterpret_cast<int *>(items + n2);           // [nb]
    __shared__ int warp_tot[kSelWarps], warp_base[kSelWarps];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int64_t u = blockIdx.x;
    const Geometry &g = p.g;
    int budget;
    int32_t *out = idx + unit_row_base(p, u, budget);
    const int P = g.P, s0 = g.sinks, tail = g.n - g.P;
    const int C = P - s0;
    const int keep = budget - s0 - tail;
    for (int j = tid; j < s0; j += kBsThreads)
        out[j] = j;
    for (int j = tid; j < tail; j += kBsThreads)
        out[s0 + keep + j] = P + j;
    if (keep <= 0)
        return;
    if (keep >= C) {
        for (int j = tid; j < C; j += kBsThreads)
            out[s0 + j] = s0 + j;
        return;
    }
    const int nb = (C + bs - 1) / bs;
    const float *sc = scores + u * (int64_t)P + s0;
    for (int k = tid; k < n2; k += kBsThreads) {
        uint64_t item = 0;
        if (k < nb) {
            const int lo = k * bs, hi = min(lo + bs, C);
            float sum = 0.f;
            for (int j = lo; j < hi; ++j)
                sum += sc[j];
            item = ((uint64_t)float_key(sum) << 32) | (uint32_t)(0xFFFFFFFFu - (uint32_t)k);
            take[k] = 0;
        }
        items[k] = item;
    }
    __syncthreads();
    // Bitonic sort, descending: the largest sum first, then the lowest block index.
    for (int size = 2; size <= n2; size <<= 1)
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            for (int i = tid; i < (n2 >> 1); i += kBsThreads) {
                const int pos = 2 * i - (i & (stride - 1));
                const uint64_t a = items[pos], b = items[pos + stride];
                const bool down = (pos & size) == 0;
                if ((a < b) == down) {
                    items[pos] = b;
                    items[pos + stride] = a;
                }
            }
            __syncthreads();
        }
    if (tid == 0) {
        int left = keep;
        for (int i = 0; i < nb && left > 0; ++i) {
            const int k = (int)(0xFFFFFFFFu - (uint32_t)items[i]);
            const int size = min(bs, C - k * bs);
            const int t = size <= left ? size : left;
            take[k] = t;
            left -= t;
        }
    }
    __syncthreads();
    // Positions in block order: thread t owns blocks [t*per, (t+1)*per).
    const int per = (nb + kBsThreads - 1) / kBsThreads;
    const int k0 = min(nb, tid * per), k1 = min(nb, k0 + per);
    int mine = 0;
    for (int k = k0; k < k1; ++k)
        mine += take[k];
    int incl = mine;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const int o = __shfl_up_sync(0xffffffffu, incl, off);
        if (lane >= off)
            incl += o;
    }
    if (lane == 31)
        warp_tot[warp] = incl;
    __syncthreads();
    scan_warp_counts(warp_tot, warp_base);
    __syncthreads();
    int o = warp_base[warp] + incl - mine;
    for (int k = k0; k < k1; ++k)
        for (int q = 0; q < take[k]; ++q)
            out[s0 + o++] = s0 + k * bs + q;
}

cudaError_t launch_block_select(const Geometry &g, const LayerTable &layers, const float *scores,
                                int32_t *idx, cudaStream_t stream)
{
    SelectParams p;
    p.g = g;
    p.layers = layers;
    const int C = g.P - g.sinks;
    const int nb = max(1, (C + g.select_block - 1) / g.select_block);
    int n2 = 1;
    while (n2 < nb)
        n2 <<= 1;
    const size_t smem = (size_t)n2 * sizeof(uint64_t) + (size_t)nb * sizeof(int);
    cudaError_t err = cudaFuncSetAttribute(block_select_kernel,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (err != cudaSuccess)
        return err;
    block_select_kernel<<<(unsigned)g.U, kBsThreads, smem, stream>>>(scores, idx, p,
                                                                    g.select_block, n2);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// StreamingLLM indices: [0, sinks) then the last budget - sinks positions.
__global__ void streaming_index_kernel(int32_t *__restrict__ idx, SelectParams p)
{
    const int64_t u = blockIdx.x;
    int budget;
    int32_t *out = idx + unit_row_base(p, u, budget);
    const int s0 = p.g.sinks, n = p.g.n;
    for (int r = threadIdx.x; r < budget; r += blockDim.x)
        out[r] = r < s0 ? r : n - budget + r;
}

cudaError_t launch_streaming_indices(const Geometry &g, const LayerTable &layers, int32_t *idx,
                                     cudaStream_t stream)
{
    SelectParams p;
    p.g = g;
    p.layers = layers;
    streaming_index_kernel<<<(unsigned)g.U, 256, 0, stream>>>(idx, p);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Gather: Kc[row] = K[idx[row]], Vc[row] = V[idx[row]], 16-byte vectors.
// Block = (unit, row block of kGatherRows); implicit = StreamingLLM indices
// computed in place (and written to idx).
constexpr int kGatherRows = 64;

// Row `pos` of a unit: contiguous (from the unit's base) or through the block table.
template <bool kPaged>
__device__ __forceinline__ const __nv_bfloat16 *gather_row(const TensorDesc &T,
                                                           const __nv_bfloat16 *unit, int l,
                                                           int bb, int h, int pos)
{
    if constexpr (kPaged)
        return kv_row_ptr(T, l, bb, h, pos);
    return unit + (int64_t)pos * T.s_pos;
}

template <int D, bool kPaged>
__global__ void __launch_bounds__(256)
compact_kernel(const int32_t *__restrict__ idx_in, int32_t *__restrict__ idx_out, TensorDesc K,
               TensorDesc V, __nv_bfloat16 *__restrict__ Kc, __nv_bfloat16 *__restrict__ Vc,
               SelectParams p, int nrb, int implicit, uint32_t *status)
{
    constexpr int TPR = D / 8;             // threads per row (16 B each)
    constexpr int RPI = 256 / TPR;          // rows per iteration
    const int64_t u = blockIdx.x / nrb;
    const int rb = (int)(blockIdx.x % nrb);
    int l, bb, h;
    unit_coords(p.g, u, l, bb, h);
    int budget;
    const int64_t base = unit_row_base(p, u, budget);
    const int r_lo = rb * kGatherRows;
    const int r_hi = min(r_lo + kGatherRows, budget);
    const __nv_bfloat16 *Ku = kv_unit_ptr(K, l, bb, h);
    const __nv_bfloat16 *Vu = kv_unit_ptr(V, l, bb, h);
    const int part = threadIdx.x % TPR;
    for (int r = r_lo + threadIdx.x / TPR; r < r_hi; r += RPI) {
        int pos;
        if (implicit) {
            pos = r < p.g.sinks ? r : p.g.n - budget + r;
            if (part == 0 && idx_out)
                idx_out[base + r] = pos;
        } else {
            pos = idx_in[base + r];
        }
        if (pos < 0 || pos >= p.g.n) {
            if (part == 0)
                set_status(status, DGE_ERR_INVALID_ARG);
            continue;
        }
        const int4 kv = *reinterpret_cast<const int4 *>(
            gather_row<kPaged>(K, Ku, l, bb, h, pos) + part * 8);
        const int4 vv = *reinterpret_cast<const int4 *>(
            gather_row<kPaged>(V, Vu, l, bb, h, pos) + part * 8);
        *reinterpret_cast<int4 *>(Kc + (base + r) * D + part * 8) = kv;
        *reinterpret_cast<int4 *>(Vc + (base + r) * D + part * 8) = vv;
    }
}

// In-place gather into the cache itself (Alg. 1: the cache of every head is edited once, in
// place, temporal order kept): rows [0, B) of a unit become the kept rows.  Kept positions
// ascend, so idx[r] >= r and a forward copy never overwrites a row still to be read.  One
// CTA per unit walks its rows in chunks; inside a chunk every source row is read into
// registers before the block barrier and written after it, so a row that is both read and
// written within the chunk is read first; rows written by earlier chunks lie below every
// later source row.  A position outside [r, n) is reported (DGE_ERR_INVALID_ARG) and skipped.
// A paged cache keeps the same order on the sequence's positions: row r of the unit goes to
// position r through the block table.
template <int D, bool kPaged>
__global__ void __launch_bounds__(256)
compact_inplace_kernel(const int32_t *__restrict__ idx_in, int32_t *__restrict__ idx_out,
                       TensorDesc K, TensorDesc V, SelectParams p, int implicit, uint32_t *status)
{
    constexpr int TPR = D / 8;             // threads per row (16 B each)
    constexpr int RPI = 256 / TPR;          // rows per pass
    constexpr int kPasses = 4;              // rows of a chunk: kPasses * RPI, in registers
    const int64_t u = blockIdx.x;
    int l, bb, h;
    unit_coords(p.g, u, l, bb, h);
    int budget;
    const int64_t base = unit_row_base(p, u, budget);
    __nv_bfloat16 *Ku = const_cast<__nv_bfloat16 *>(kv_unit_ptr(K, l, bb, h));
    __nv_bfloat16 *Vu = const_cast<__nv_bfloat16 *>(kv_unit_ptr(V, l, bb, h));
    const int part = threadIdx.x % TPR, rsub = threadIdx.x / TPR;
    for (int r0 = 0; r0 < budget; r0 += kPasses * RPI) {
        int4 kv[kPasses], vv[kPasses];
        int dst[kPasses];
#pragma unroll
        for (int i = 0; i < kPasses; ++i) {
            const int r = r0 + i * RPI + rsub;
            dst[i] = -1;
            if (r < budget) {
                int pos;
                if (implicit) {
                    pos = r < p.g.sinks ? r : p.g.n - budget + r;
                    if (part == 0 && idx_out)
                        idx_out[base + r] = pos;
                } else {
                    pos = idx_in[base + r];
                }
                if (pos < r || pos >= p.g.n) {
                    if (part == 0)
                        set_status(status, DGE_ERR_INVALID_ARG);
                } else if (pos != r) {
                    kv[i] = *reinterpret_cast<const int4 *>(
                        gather_row<kPaged>(K, Ku, l, bb, h, pos) + part * 8);
                    vv[i] = *reinterpret_cast<const int4 *>(
                        gather_row<kPaged>(V, Vu, l, bb, h, pos) + part * 8);
                    dst[i] = r;
                }
            }
        }
        __syncthreads();
#pragma unroll
        for (int i = 0; i < kPasses; ++i)
            if (dst[i] >= 0) {
                *reinterpret_cast<int4 *>(
                    const_cast<__nv_bfloat16 *>(gather_row<kPaged>(K, Ku, l, bb, h, dst[i])) +
                    part * 8) = kv[i];
                *reinterpret_cast<int4 *>(
                    const_cast<__nv_bfloat16 *>(gather_row<kPaged>(V, Vu, l, bb, h, dst[i])) +
                    part * 8) = vv[i];
            }
    }
}

cudaError_t launch_compact_inplace(const Geometry &g, const LayerTable &layers,
                                   const int32_t *idx_in, int32_t *idx_out, const TensorDesc &K,
                                   const TensorDesc &V, bool implicit, uint32_t *status,
                                   cudaStream_t stream)
{
    SelectParams p;
    p.g = g;
    p.layers = layers;
    if (g.U == 0)
        return cudaSuccess;
    auto kernel = g.d == 128 ? (K.bt ? compact_inplace_kernel<128, true>
                                     : compact_inplace_kernel<128, false>)
                             : (K.bt ? compact_inplace_kernel<64, true>
                                     : compact_inplace_kernel<64, false>);
    kernel<<<(unsigned)g.U, 256, 0, stream>>>(idx_in, idx_out, K, V, p, implicit ? 1 : 0, status);
    return cudaGetLastError();
}

cudaError_t launch_compact(const Geometry &g, const LayerTable &layers, const int32_t *idx_in,
                           int32_t *idx_out, const TensorDesc &K, const TensorDesc &V, void *Kc,
                           void *Vc, bool implicit, uint32_t *status, cudaStream_t stream)
{
    SelectParams p;
    p.g = g;
    p.layers = layers;
    int maxb = 0;
    for (int l = 0; l < g.L; ++l)
        maxb = max(maxb, layers.budget[l]);
    const int nrb = (maxb + kGatherRows - 1) / kGatherRows;
    if (nrb == 0)
        return cudaSuccess;
    const int64_t blocks = g.U * nrb;
    auto kernel = g.d == 128 ? (K.bt ? compact_kernel<128, true> : compact_kernel<128, false>)
                             : (K.bt ? compact_kernel<64, true> : compact_kernel<64, false>);
    kernel<<<(unsigned)blocks, 256, 0, stream>>>(idx_in, idx_out, K, V,
                                                 static_cast<__nv_bfloat16 *>(Kc),
                                                 static_cast<__nv_bfloat16 *>(Vc), p, nrb,
                                                 implicit ? 1 : 0, status);
    return cudaGetLastError();
}

}  // namespace dge
