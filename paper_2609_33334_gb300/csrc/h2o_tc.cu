// h2o_tc.cu -- H2O accumulated attention scores on the 5th-generation tensor cores.
//
// The H2O score of a past key j (App. B's H2O note, the accumulated-attention evictor that Alg. 1
// applies after drafting) sums, over every query row of the cache -- all n positions of the G
// query heads of the key's group, each row causal -- the softmax probability the row gives j.
// In base 2:
//   x_rj = log2(e) * scale * q_r . k_j,   row r = (g, p) sees keys j <= p,
//   lse_r = log2 sum_{j <= p} 2^{x_rj},   raw_j = sum_{r : p_r >= j} 2^{x_rj - lse_r}.
// A unit's rows form query blocks of pb positions x G heads (stacked head-major, one 5-D TMA
// box; at most 128 rows in phase 1 and 144 in phase 2).  Two launches of one persistent,
// warp-specialised kernel, one CTA per SM, tasks dealt round-robin:
//   phase 1, task (unit, query block): the block stays in shared memory while the key tiles it
//     can see stream through a ring; the epilogue keeps every row's sum of 2^x in registers,
//     and warp 3 turns the block's sums into lse_r;
//   phase 2, task (unit, 128-key tile): the key tile stays while the query blocks that can
//     see it stream through the ring with their -lse (staged by warp 2); every epilogue thread
//     keeps one key's column sum for the whole task, and the three warpgroups' partial sums
//     meet once, at the end of the task.
// Both phases compute D[128 keys x R_pad rows] = K_tile . Q_block^T with tcgen05.mma (M = 128,
// bf16 -> fp32) into one of four (phase 1) or three (phase 2) TMEM accumulators: warp 0 issues
// the TMA copies, warp 1 the MMAs, warps 4..15 (three warpgroups, a third of the columns each,
// one key per thread) read the accumulators.  Row sums carry no running maximum: fp32 holds
// 2^x for |x| < 126, and a unit whose sums leave [2^-60, 2^126) is flagged (ready = 2) and
// recomputed by the warp-level kernels.  Every wait is bounded: on expiry the CTA records
// DGE_ERR_DEVICE_TIMEOUT, stops issuing work, drains its own copies and MMAs and frees TMEM.
#include <cuda.h>
#include <math.h>
#include <string.h>

#include <type_traits>

#include "common.cuh"
#include "kernels.h"
#include "tc_common.cuh"
#include "tc_ptx.cuh"

namespace dge {

namespace {

constexpr int kTile = 128;
constexpr int kEpiWG = 3;                 // epilogue warpgroups
constexpr int kEpiWarps = 4 * kEpiWG;
constexpr int kEpiWarp0 = 4;              // epilogue warps are 4 .. 15 (aligned warpgroups)
constexpr int kThreads = (kEpiWarp0 + kEpiWarps) * 32;
// Registers after reallocation: warpgroup 0 (producer, MMA, two staging warps) gives up
// registers to the epilogue; 4*32*56 + 12*32*152 = 512 threads x 128 at launch.
constexpr int kRegsControl = 56, kRegsEpilogue = 152;
static_assert(4 * 32 * kRegsControl + kEpiWarps * 32 * kRegsEpilogue <= kThreads * 128,
              "register split");
constexpr int kMaxGroups = 3;             // 16-column groups per epilogue warpgroup
constexpr int kMaxBlockRows = kEpiWG * kMaxGroups * 16;
// Rows of a query block and TMEM accumulators, per phase: phase 1 takes blocks of up to 128
// rows (four accumulators of 128 columns, so its MMAs run one more tile ahead of the
// epilogue), phase 2 blocks of up to 144 rows (three of 160 columns).  Measured with 128-row
// blocks on 32 layers x 8 sequences x 8 KV heads of 8K positions, G = 4: phase 1 101 -> 85 ms,
// phase 2 96.5 -> 103.6 ms (12 % more tiles for it).
constexpr int kBlockRows1 = 128, kAccBufs1 = 4;
constexpr int kBlockRows2 = kMaxBlockRows, kAccBufs2 = 3;
constexpr int kMaxAccBufs = 4;
static_assert(kAccBufs1 * ((kBlockRows1 + 31) & ~31) <= 512 &&
                  kAccBufs2 * ((kBlockRows2 + 31) & ~31) <= 512,
              "TMEM columns");
constexpr int kStages = 4;                // streamed operand ring
constexpr int kTmemCols = 512;
constexpr int kKSlab = kTile * 128;       // 128 keys x 64 bf16
constexpr int kXchBufs = 4;               // phase-2 end-of-task exchange areas
// -lse of the streamed query blocks, staged kLseGroup blocks at a time into one of two slots:
// a hand-off (one wait, one arrival) every kLseGroup tiles rather than every tile.
constexpr int kLseGroup = 4;
constexpr int kLseSlots = 2;
constexpr int kLseBlock = 160;            // floats per block (>= rows, 16-byte multiple)
constexpr int kLseLoads = (kBlockRows2 + 31) / 32;     // staged rows per lane (phase 2)
constexpr uint32_t kReadyBad = 2;

// Barrier slots.
constexpr int kBarRingFull = 0, kBarRingEmpty = 4, kBarStatFull = 8, kBarStatEmpty = 10,
              kBarAccFull = 12, kBarAccEmpty = kBarAccFull + kMaxAccBufs,
              kBarDrain = kBarAccEmpty + kMaxAccBufs, kBarRedFull = kBarDrain + 1,
              kBarRedEmpty = kBarRedFull + 2, kBarLseFull = kBarRedEmpty + 2,
              kBarLseEmpty = kBarLseFull + kLseSlots, kBarXch = kBarLseEmpty + kLseSlots,
              kNumBars = kBarXch + kXchBufs * 4;
constexpr int kCtrlBytes = 512;           // barriers, TMEM address, flags (16-byte multiple)
// Flag slots (ints): abort, then the parity of the last arm of every ring stage and
// stationary buffer (-1 = never armed) for the drain.
constexpr int kFlagAbort = tc::kFlagAbort, kFlagRingArm = 4, kFlagStatArm = 8;
static_assert(kNumBars * 8 + 16 + 16 * 4 <= kCtrlBytes, "control block");

struct H2oArgs {
    Geometry g;
    tc::KPaging kp;    // K through a block table (kp.bt != nullptr)
    int phase;         // 1: row normalisers, 2: column sums
    int pb;            // positions per query block
    int rows;          // G * pb
    int r_pad;         // rows rounded up to 16
    int nslab;         // d / 64
    int acc_stride;    // TMEM columns between accumulators
    int nqb, nkt;      // query blocks, past-key tiles per unit
    int64_t items;     // tasks of this launch
    int ng[kEpiWG], gbase[kEpiWG];   // 16-column groups of each epilogue warpgroup
    float *lse2;       // [U][R], row r = g * n + p
    float *raw;        // [U][P]
    uint32_t *ready;   // [U]
    uint32_t *status;
    unsigned long long timeout_ns;
};

__host__ __device__ inline uint32_t q_slab(int r_pad) { return (uint32_t)r_pad * 128u; }
__host__ __device__ inline uint32_t stat_slab(int phase, int r_pad)
{
    return phase == 1 ? q_slab(r_pad) : (uint32_t)kKSlab;
}
__host__ __device__ inline uint32_t ring_slab(int phase, int r_pad)
{
    return phase == 1 ? (uint32_t)kKSlab : q_slab(r_pad);
}

__host__ __device__ inline size_t smem_bytes(int phase, int r_pad, int nslab)
{
    return 1024                                                 // alignment slack
           + (size_t)2 * nslab * stat_slab(phase, r_pad)        // stationary operand
           + (size_t)kStages * nslab * ring_slab(phase, r_pad)  // streamed operand
           + kCtrlBytes + (size_t)kLseSlots * kLseGroup * kLseBlock * 4
           + (size_t)2 * kEpiWG * 4 * kMaxGroups * 16 * 4 + (size_t)kXchBufs * kEpiWG * kTile * 4
           + (size_t)(tc::kPageWindow + 4) * 4;
}

struct Smem {
    uint8_t *stat;     // [2][nslab][stat_slab]
    uint8_t *ring;     // [kStages][nslab][ring_slab]
    uint64_t *bar;     // [kNumBars]
    uint32_t *tmem;    // allocation result
    int *flag;         // [16]
    float *lse;        // [kLseSlots][kLseGroup][kLseBlock] -lse of streamed blocks (phase 2)
    float *red;        // [2][kEpiWG][4][kMaxGroups * 16] per-warp row sums (phase 1)
    float *xch;        // [kXchBufs][kEpiWG][128] per-warpgroup column sums (phase 2)
    int *pages;        // [tc::kPageWindow] page ids of the producer's window (paged caches)
};

__device__ __forceinline__ Smem carve(uint8_t *raw, int phase, int r_pad, int nslab)
{
    const uint32_t base = ptx::smem_addr(raw);
    uint32_t off = ((base + 1023u) & ~1023u) - base;
    Smem s;
    s.stat = raw + off;
    off += 2u * nslab * stat_slab(phase, r_pad);
    s.ring = raw + off;
    off += (uint32_t)kStages * nslab * ring_slab(phase, r_pad);
    s.bar = reinterpret_cast<uint64_t *>(raw + off);
    s.tmem = reinterpret_cast<uint32_t *>(raw + off + kNumBars * 8);
    s.flag = reinterpret_cast<int *>(raw + off + kNumBars * 8 + 16);
    off += kCtrlBytes;
    s.lse = reinterpret_cast<float *>(raw + off);
    off += kLseSlots * kLseGroup * kLseBlock * 4;
    s.red = reinterpret_cast<float *>(raw + off);
    off += 2 * kEpiWG * 4 * kMaxGroups * 16 * 4;
    s.xch = reinterpret_cast<float *>(raw + off);
    off += kXchBufs * kEpiWG * kTile * 4;
    s.pages = reinterpret_cast<int *>(raw + off);
    return s;
}

struct Task {
    int64_t u;
    int blk;      // phase 1: query block; phase 2: key tile
    int first;    // first streamed tile (phase 2: first query block that sees the key tile)
    int ntiles;   // streamed tiles
};

// Task `item` of this launch.  Phase 1: the key tiles 0 .. that the block's last visible
// position needs.  Phase 2: the query blocks from the one holding the tile's first key on
// (earlier positions cannot see any key of the tile).
__device__ __forceinline__ void get_task(const H2oArgs &a, int64_t item, Task &T)
{
    if (a.phase == 1) {
        T.u = item / a.nqb;
        T.blk = (int)(item % a.nqb);
        const int p_end = min((T.blk + 1) * a.pb, a.g.n);
        T.first = 0;
        T.ntiles = (p_end + kTile - 1) / kTile;
    } else {
        T.u = item / a.nkt;
        T.blk = (int)(item % a.nkt);
        T.first = T.blk * kTile / a.pb;
        T.ntiles = a.nqb - T.first;
    }
}

// Visibility of key `key` to the 16 columns cb .. cb+15 of a query block starting at
// position p0: column c is row (c / pb, p0 + c % pb).
__device__ __forceinline__ uint32_t causal_mask(int key, int p0, int pb, int cb)
{
    int i = cb % pb;
    uint32_t mask = 0;
#pragma unroll
    for (int c = 0; c < 16; ++c) {
        mask |= (key <= p0 + i ? 1u : 0u) << c;
        if (++i == pb)
            i = 0;
    }
    return mask;
}

// Phase 1 for one 16-column group: z[c] += 2^{x_c} (keys after a row's position add nothing).
// kDiag: the tile reaches the block's own positions (masked); a compile-time choice, so the
// loop over the other tiles carries no mask code.
template <bool kDiag>
__device__ __forceinline__ void rows_add(float (&z)[16], const float (&v)[16], float s2, int key,
                                         int p0, int pb, int cb)
{
    if constexpr (!kDiag) {
        const float2 sc = make_float2(s2, s2);
#pragma unroll
        for (int c = 0; c < 16; c += 2) {
            const float2 x = __fmul2_rn(make_float2(v[c], v[c + 1]), sc);
            const float2 acc = __fadd2_rn(make_float2(z[c], z[c + 1]),
                                          make_float2(ex2(x.x), ex2(x.y)));
            z[c] = acc.x;
            z[c + 1] = acc.y;
        }
    } else {
        const uint32_t mask = causal_mask(key, p0, pb, cb);
#pragma unroll
        for (int c = 0; c < 16; ++c) {
            const float e = ex2(v[c] * s2);
            z[c] += ((mask >> c) & 1u) ? e : 0.f;
        }
    }
}

// Phase 2 for one 16-column group: adds 2^{x_c - lse_c} over the rows that see `key`.  nL
// holds -lse (rows past the cache or padding: -inf).  Columns 2q, 2q+1 go to acc[q % 4]: four
// independent chains of additions instead of one (the epilogue is latency-bound), added
// together in a fixed order at the end of the task.
template <bool kDiag>
__device__ __forceinline__ void col_add(float2 (&acc)[4], const float (&v)[16],
                                        const float (&nL)[16], float s2, int key, int p0, int pb,
                                        int cb)
{
    if constexpr (!kDiag) {
        const float2 sc = make_float2(s2, s2);
#pragma unroll
        for (int c = 0; c < 16; c += 2) {
            const float2 x = __ffma2_rn(make_float2(v[c], v[c + 1]), sc,
                                        make_float2(nL[c], nL[c + 1]));
            acc[(c >> 1) & 3] = __fadd2_rn(acc[(c >> 1) & 3], make_float2(ex2(x.x), ex2(x.y)));
        }
    } else {
        const uint32_t mask = causal_mask(key, p0, pb, cb);
#pragma unroll
        for (int c = 0; c < 16; ++c) {
            const float p = ex2(v[c] * s2 + nL[c]);
            acc[(c >> 1) & 3].x += ((mask >> c) & 1u) ? p : 0.f;
        }
    }
}

// f(gi, v) over this warp's 16-column groups gi = 0 .. ng-1, one TMEM round trip each.
template <typename F>
__device__ __forceinline__ void for_groups(uint32_t tbase, int ng, F &&f)
{
#pragma unroll
    for (int gi = 0; gi < kMaxGroups; ++gi)
        if (gi < ng) {
            float v[16];
            ptx::tmem_ld16(tbase + gi * 16, v);
            ptx::tmem_ld_wait_dep(v);
            f(gi, v);
        }
}

template <bool kPaged, int kAccBufs>
__global__ void __launch_bounds__(kThreads, 1)
h2o_tc_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmQ,
              const __grid_constant__ CUtensorMap tmKm, const H2oArgs a)
{
    extern __shared__ uint8_t smem_raw[];
    const Smem sm = carve(smem_raw, a.phase, a.r_pad, a.nslab);
    volatile int *flag = sm.flag;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const Geometry &g = a.g;
    const uint32_t sslab = stat_slab(a.phase, a.r_pad), rslab = ring_slab(a.phase, a.r_pad);
    const uint32_t qbytes = (uint32_t)a.nslab * 128u * (uint32_t)a.rows;  // one query block
    const uint32_t kbytes = (uint32_t)a.nslab * (uint32_t)kKSlab;         // one key tile
    const int64_t S = gridDim.x;
    auto wait = [&](uint64_t *bar, uint32_t parity) {
        return tc::wait_bar(bar, parity, flag, a.timeout_ns, a.status);
    };

    // ---- set-up -------------------------------------------------------------------
    if (threadIdx.x == 0) {
        for (int i = 0; i < kStages; ++i) {
            ptx::mbar_init(&sm.bar[kBarRingFull + i], 1);
            ptx::mbar_init(&sm.bar[kBarRingEmpty + i], 1);
        }
        for (int i = 0; i < kLseSlots; ++i) {
            ptx::mbar_init(&sm.bar[kBarLseFull + i], 1);
            ptx::mbar_init(&sm.bar[kBarLseEmpty + i], kEpiWarps);
        }
        for (int i = 0; i < 2; ++i) {
            ptx::mbar_init(&sm.bar[kBarStatFull + i], 1);
            ptx::mbar_init(&sm.bar[kBarStatEmpty + i], 1);
            ptx::mbar_init(&sm.bar[kBarRedFull + i], kEpiWarps);
            ptx::mbar_init(&sm.bar[kBarRedEmpty + i], 1);
        }
        for (int i = 0; i < kAccBufs; ++i) {
            ptx::mbar_init(&sm.bar[kBarAccFull + i], 1);
            ptx::mbar_init(&sm.bar[kBarAccEmpty + i], kEpiWarps);
        }
        ptx::mbar_init(&sm.bar[kBarDrain], 1);
        // End-of-task exchange: one barrier per area and lane quarter, one arrival per
        // warpgroup.
        for (int i = 0; i < kXchBufs * 4; ++i)
            ptx::mbar_init(&sm.bar[kBarXch + i], kEpiWG);
        flag[kFlagAbort] = 0;
        for (int i = 0; i < kStages; ++i)
            flag[kFlagRingArm + i] = -1;
        flag[kFlagStatArm] = flag[kFlagStatArm + 1] = -1;
        ptx::fence_mbar_init();
    }
    // Query rows `rows` .. r_pad-1 are never written by TMA: zero them once so the padded
    // accumulator columns are exactly 0.
    {
        const int pad_rows = a.r_pad - a.rows;
        uint8_t *qbuf = a.phase == 1 ? sm.stat : sm.ring;
        const int nbuf = a.phase == 1 ? 2 : kStages;
        const int words = pad_rows * 128 / 16;
        for (int b = 0; b < nbuf; ++b)
            for (int s = 0; s < a.nslab; ++s) {
                int4 *p = reinterpret_cast<int4 *>(qbuf + ((size_t)b * a.nslab + s) * q_slab(a.r_pad) +
                                                   (size_t)a.rows * 128);
                for (int i = threadIdx.x; i < words; i += blockDim.x)
                    p[i] = make_int4(0, 0, 0, 0);
            }
        ptx::fence_proxy_async_smem();
    }
    if (warp == 1) {
        ptx::tmem_alloc(sm.tmem, kTmemCols);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem_base = *sm.tmem;

    if (warp < kEpiWarp0) {
        ptx::regs_dec<kRegsControl>();
        if (warp == 0) {
            // ---- TMA producer -----------------------------------------------------------
            if (lane == 0) {
                ptx::prefetch_tmap(&tmK);
                ptx::prefetch_tmap(&tmQ);
                // The streamed operand is read by the other CTAs working on the same unit;
                // the stationary one by this task alone.
                const uint64_t shared_pol = ptx::make_policy_evict_last();
                const uint64_t once_pol = ptx::make_policy_evict_first();
                int rs = 0, sb = 0;
                uint32_t rph = 0, sph = 0;
                bool ok = true;
                for (int64_t item = blockIdx.x; ok && item < a.items; item += S) {
                    Task T;
                    get_task(a, item, T);
                    int l, bb, h;
                    unit_coords(g, T.u, l, bb, h);
                    if (!wait(&sm.bar[kBarStatEmpty + sb], sph ^ 1)) {
                        ok = false;
                        break;
                    }
                    uint8_t *sdst = sm.stat + (size_t)sb * a.nslab * sslab;
                    ptx::mbar_arrive_expect_tx(&sm.bar[kBarStatFull + sb],
                                               a.phase == 1 ? qbytes : kbytes);
                    flag[kFlagStatArm + sb] = (int)sph;
                    for (int s = 0; s < a.nslab && a.phase == 1; ++s) {
                        ptx::tma_load_5d_hint(sdst + s * sslab, &tmQ, &sm.bar[kBarStatFull + sb],
                                              s * 64, T.blk * a.pb, h * g.G, bb, l, once_pol);
                    }
                    if (a.phase == 2) {
                        const int *ids = sm.pages;
                        if constexpr (kPaged)
                            ids = tc::fetch_pages(sm.pages, a.kp, bb, T.blk * kTile, 1);
                        tc::load_k_tile<kPaged>(sdst, sslab, a.nslab, &tmK, &tmKm,
                                                &sm.bar[kBarStatFull + sb], T.blk * kTile, l, bb,
                                                h, a.kp, ids, T.blk * kTile, once_pol);
                    }
                    if (++sb == 2) {
                        sb = 0;
                        sph ^= 1;
                    }
                    int w0 = 0;               // first key of the page-id window (paged caches)
                    const int *ids = sm.pages;
                    for (int i = 0; i < T.ntiles; ++i) {
                        if constexpr (kPaged) {
                            if (a.phase == 1 && i % tc::kPageWindowTiles == 0) {
                                w0 = i * kTile;
                                ids = tc::fetch_pages(sm.pages, a.kp, bb, w0,
                                                      min(T.ntiles - i, tc::kPageWindowTiles));
                            }
                        }
                        if (!wait(&sm.bar[kBarRingEmpty + rs], rph ^ 1)) {
                            ok = false;
                            break;
                        }
                        uint8_t *rdst = sm.ring + (size_t)rs * a.nslab * rslab;
                        ptx::mbar_arrive_expect_tx(&sm.bar[kBarRingFull + rs],
                                                   a.phase == 1 ? kbytes : qbytes);
                        flag[kFlagRingArm + rs] = (int)rph;
                        if (a.phase == 1)
                            tc::load_k_tile<kPaged>(rdst, rslab, a.nslab, &tmK, &tmKm,
                                                    &sm.bar[kBarRingFull + rs], i * kTile, l, bb,
                                                    h, a.kp, ids, w0, shared_pol);
                        else
                            for (int s = 0; s < a.nslab; ++s)
                                ptx::tma_load_5d_hint(rdst + s * rslab, &tmQ,
                                                      &sm.bar[kBarRingFull + rs], s * 64,
                                                      (T.first + i) * a.pb, h * g.G, bb, l,
                                                      shared_pol);
                        if (++rs == kStages) {
                            rs = 0;
                            rph ^= 1;
                        }
                    }
                }
            }
        } else if (warp == 1) {
            // ---- MMA issuer -------------------------------------------------------------
            if (lane == 0) {
                const uint32_t idesc = ptx::idesc_bf16_f32(kTile, a.r_pad);
                const uint32_t qs = q_slab(a.r_pad);
                int rs = 0, sb = 0;
                uint32_t rph = 0, sph = 0;
                int64_t tc = 0;  // accumulator sequence number: buffer tc % 3, use tc / 3
                bool ok = true;
                for (int64_t item = blockIdx.x; ok && item < a.items; item += S) {
                    Task T;
                    get_task(a, item, T);
                    if (!wait(&sm.bar[kBarStatFull + sb], sph)) {
                        ok = false;
                        break;
                    }
                    const uint32_t stat_addr = ptx::smem_addr(sm.stat + (size_t)sb * a.nslab * sslab);
                    for (int i = 0; i < T.ntiles; ++i, ++tc) {
                        const int ab = (int)(tc % kAccBufs);
                        const uint32_t aph = (uint32_t)((tc / kAccBufs) & 1);
                        if (!wait(&sm.bar[kBarRingFull + rs], rph) ||
                            !wait(&sm.bar[kBarAccEmpty + ab], aph ^ 1)) {
                            ok = false;
                            break;
                        }
                        ptx::tc_fence_after();
                        const uint32_t ring_addr =
                            ptx::smem_addr(sm.ring + (size_t)rs * a.nslab * rslab);
                        // A = the key tile (128 rows), B = the query block (r_pad rows).
                        const uint64_t ad0 = ptx::smem_desc_sw128(a.phase == 1 ? ring_addr : stat_addr);
                        const uint64_t bd0 = ptx::smem_desc_sw128(a.phase == 1 ? stat_addr : ring_addr);
                        const uint32_t d_tmem = tmem_base + (uint32_t)(ab * a.acc_stride);
#pragma unroll
                        for (int kk = 0; kk < 8; ++kk) {
                            if (kk < a.nslab * 4) {
                                const uint32_t a_off =
                                    ((uint32_t)(kk >> 2) * kKSlab + (uint32_t)(kk & 3) * 32u) >> 4;
                                const uint32_t b_off =
                                    ((uint32_t)(kk >> 2) * qs + (uint32_t)(kk & 3) * 32u) >> 4;
                                ptx::mma_bf16(d_tmem, ad0 + a_off, bd0 + b_off, idesc,
                                              kk > 0 ? 1u : 0u);
                            }
                        }
                        ptx::mma_commit(&sm.bar[kBarRingEmpty + rs]);
                        ptx::mma_commit(&sm.bar[kBarAccFull + ab]);
                        if (++rs == kStages) {
                            rs = 0;
                            rph ^= 1;
                        }
                    }
                    if (!ok)
                        break;
                    ptx::mma_commit(&sm.bar[kBarStatEmpty + sb]);
                    if (++sb == 2) {
                        sb = 0;
                        sph ^= 1;
                    }
                }
                // Every MMA issued so far completes before the drain barrier fires.
                ptx::mma_commit(&sm.bar[kBarDrain]);
                tc::drain_bar(&sm.bar[kBarDrain], 0, 2000000000ull);
            }
        } else {
            bool dead = false;
            auto wait_w = [&](uint64_t *bar, uint32_t parity) {
                if (!dead) {
                    const bool got = wait(bar, parity);
                    dead = !__all_sync(0xffffffffu, got);
                }
                return !dead;
            };
            if (warp == 2 && a.phase == 2) {
                // ---- -lse of every streamed query block, per row: -inf past the cache ------
                // A group of kLseGroup blocks (they may straddle tasks) at a time: every lse of
                // the group is copied to shared memory asynchronously, all in flight at once
                // (one L2 round trip per group), then each lane negates its own entries.
                int hd[kLseLoads];   // query head of each of this lane's rows
#pragma unroll
                for (int j = 0; j < kLseLoads; ++j)
                    hd[j] = (lane + 32 * j) / a.pb;
                int64_t item = blockIdx.x;   // cursor: block i of task `item`
                int i = 0;
                Task T;
                bool more = item < a.items;
                if (more)
                    get_task(a, item, T);
                uint32_t copied[kLseGroup];  // per block: bit j = this lane's row lane + 32 j
                for (int64_t grp = 0; more && !dead; ++grp) {
                    const int slot = (int)(grp % kLseSlots);
                    if (!wait_w(&sm.bar[kBarLseEmpty + slot],
                                (uint32_t)((grp / kLseSlots) & 1) ^ 1))
                        break;
                    float *L = sm.lse + slot * kLseGroup * kLseBlock;
#pragma unroll
                    for (int c = 0; c < kLseGroup; ++c) {
                        copied[c] = 0;
                        if (!more)
                            continue;
                        const float *src = a.lse2 + T.u * g.R;
                        const int p0 = (T.first + i) * a.pb;
#pragma unroll
                        for (int j = 0; j < kLseLoads; ++j) {
                            const int r = lane + 32 * j;
                            const int pos = p0 + r - hd[j] * a.pb;
                            float *dst = L + c * kLseBlock + r;
                            if (r < a.rows && pos < g.n) {
                                asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(
                                                 ptx::smem_addr(dst)),
                                             "l"(src + (int64_t)hd[j] * g.n + pos)
                                             : "memory");
                                copied[c] |= 1u << j;
                            } else if (r < a.r_pad) {
                                *dst = -INFINITY;
                            }
                        }
                        if (++i == T.ntiles) {
                            i = 0;
                            item += S;
                            more = item < a.items;
                            if (more)
                                get_task(a, item, T);
                        }
                    }
                    asm volatile("cp.async.wait_all;" ::: "memory");
#pragma unroll
                    for (int c = 0; c < kLseGroup; ++c)
#pragma unroll
                        for (int j = 0; j < kLseLoads; ++j)
                            if (copied[c] >> j & 1u) {
                                float *dst = L + c * kLseBlock + lane + 32 * j;
                                *dst = -*dst;
                            }
                    // A last group may be partly filled: its consumers stop at the last block.
                    __syncwarp();
                    if (lane == 0)
                        ptx::mbar_arrive(&sm.bar[kBarLseFull + slot]);
                }
            } else if (warp == 3 && a.phase == 1) {
                // ---- row sums of a query block -> lse_r ---------------------------------------
                constexpr int W = kMaxGroups * 16;
                int rb = 0;
                uint32_t rph = 0;
                for (int64_t item = blockIdx.x; !dead && item < a.items; item += S) {
                    Task T;
                    get_task(a, item, T);
                    if (wait_w(&sm.bar[kBarRedFull + rb], rph)) {
                        const int p0 = T.blk * a.pb;
                        float *dst = a.lse2 + T.u * g.R;
                        bool bad = false;
                        for (int col = lane; col < a.rows; col += 32) {
                            int w = 0;
                            while (w + 1 < kEpiWG && col >= a.gbase[w + 1] * 16)
                                ++w;
                            const int lc = col - a.gbase[w] * 16;
                            const float *rbuf = sm.red + (rb * kEpiWG + w) * 4 * W;
                            const float Z = rbuf[lc] + rbuf[W + lc] + rbuf[2 * W + lc] +
                                            rbuf[3 * W + lc];
                            const int gh = col / a.pb;
                            const int pos = p0 + col - gh * a.pb;
                            if (pos < g.n) {
                                if (!(Z >= 0x1p-60f && Z < 0x1p126f))
                                    bad = true;
                                dst[(int64_t)gh * g.n + pos] = log2f(Z);
                            }
                        }
                        bad = __any_sync(0xffffffffu, bad);
                        if (lane == 0 && bad)
                            a.ready[T.u] = kReadyBad;  // recomputed after the kernel
                    }
                    __syncwarp();
                    if (lane == 0)
                        ptx::mbar_arrive(&sm.bar[kBarRedEmpty + rb]);
                    if (++rb == 2) {
                        rb = 0;
                        rph ^= 1;
                    }
                }
            }
        }
    } else {
        ptx::regs_inc<kRegsEpilogue>();
        // ---- epilogue -------------------------------------------------------------------
        const int ew = warp - kEpiWarp0;         // 0 .. kEpiWarps-1
        const int wg = ew >> 2;                  // warpgroup
        const int quarter = warp & 3;            // TMEM lane quarter of this warp
        const int kl = quarter * 32 + lane;      // key within the tile
        const int ng = a.ng[wg];
        const int col_base = a.gbase[wg] * 16;
        const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
        const float s2 = g.scale_log2;
        int tc = 0;
        bool dead = false;
        auto acquire_acc = [&](int ab, uint32_t aph) {
            if (!dead) {
                const bool got = wait(&sm.bar[kBarAccFull + ab], aph);
                dead = !__all_sync(0xffffffffu, got);
            }
            if (!dead)
                ptx::tc_fence_after();
            return !dead;
        };
        auto wait_uniform = [&](uint64_t *bar, uint32_t parity) {
            if (!dead) {
                const bool got = wait(bar, parity);
                dead = !__all_sync(0xffffffffu, got);
            }
            return !dead;
        };
        auto release_acc = [&](int ab) {
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0 && !dead)
                ptx::mbar_arrive(&sm.bar[kBarAccEmpty + ab]);
        };

        if (a.phase == 1) {
            int rb = 0;
            uint32_t rph = 0;
            for (int64_t item = blockIdx.x; item < a.items; item += S) {
                Task T;
                get_task(a, item, T);
                const int p0 = T.blk * a.pb;
                float z[kMaxGroups][16];
#pragma unroll
                for (int i = 0; i < kMaxGroups; ++i)
#pragma unroll
                    for (int c = 0; c < 16; ++c)
                        z[i][c] = 0.f;
                // Tiles below the block's first position are seen by every row (no mask); the
                // rest reach the block's own positions.  Two loops, each with its own body.
                auto tile1 = [&](int i, auto diag_c) {
                    constexpr bool kDiag = decltype(diag_c)::value;
                    const int ab = tc % kAccBufs;
                    const uint32_t aph = (uint32_t)((tc / kAccBufs) & 1);
                    const int key = i * kTile + kl;
                    if (acquire_acc(ab, aph)) {
                        const uint32_t tbase =
                            tmem_base + (uint32_t)(ab * a.acc_stride + col_base) + lane_off;
                        for_groups(tbase, ng, [&](int gi, const float(&v)[16]) {
#pragma unroll
                            for (int gj = 0; gj < kMaxGroups; ++gj)
                                if (gj == gi)
                                    rows_add<kDiag>(z[gj], v, s2, key, p0, a.pb,
                                                    col_base + gj * 16);
                        });
                    }
                    release_acc(ab);
                    ++tc;
                };
                const int nplain = min(T.ntiles, p0 / kTile);
                for (int i = 0; i < nplain; ++i)
                    tile1(i, std::false_type());
                for (int i = nplain; i < T.ntiles; ++i)
                    tile1(i, std::true_type());
                // Sums over this warp's 32 keys, handed to warp 3 through a double-buffered
                // area (it adds the lane quarters in a fixed order).
#pragma unroll
                for (int gi = 0; gi < kMaxGroups; gi += 2) {
                    if (gi < ng) {
                        if (gi + 1 < kMaxGroups && gi + 1 < ng)
                            tc::transpose_sum32(z[gi], z[gi + 1 < kMaxGroups ? gi + 1 : gi], lane);
                        else
                            tc::transpose_sum16(z[gi], lane);
                    }
                }
                if (wait_uniform(&sm.bar[kBarRedEmpty + rb], rph ^ 1)) {
                    float *red = sm.red + ((rb * kEpiWG + wg) * 4 + quarter) * (kMaxGroups * 16);
#pragma unroll
                    for (int gi = 0; gi < kMaxGroups; gi += 2) {
                        if (gi < ng) {
                            if (gi + 1 < kMaxGroups && gi + 1 < ng)
                                red[gi * 16 + lane] = z[gi][0];
                            else if (lane < 16)
                                red[gi * 16 + lane] = z[gi][0];
                        }
                    }
                    __syncwarp();
                    if (lane == 0)
                        ptx::mbar_arrive(&sm.bar[kBarRedFull + rb]);
                }
                if (++rb == 2) {
                    rb = 0;
                    rph ^= 1;
                }
            }
        } else {
            int xc = 0;
            int64_t nb = 0;      // streamed blocks so far (the stager's count)
            bool lse_ok = false;
            for (int64_t item = blockIdx.x; item < a.items; item += S) {
                Task T;
                get_task(a, item, T);
                const int k0 = T.blk * kTile;
                const int key = k0 + kl;
                float2 acc[4];
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    acc[q] = make_float2(0.f, 0.f);
                // The first blocks hold rows before some of the tile's keys (masked); the rest see
                // every key.  Two loops, each with its own body.
                auto tile2 = [&](int i, auto diag_c) {
                    constexpr bool kDiag = decltype(diag_c)::value;
                    const int ab = tc % kAccBufs;
                    const uint32_t aph = (uint32_t)((tc / kAccBufs) & 1);
                    const int p0 = (T.first + i) * a.pb;
                    const int sub = (int)(nb % kLseGroup);
                    const int slot = (int)((nb / kLseGroup) % kLseSlots);
                    if (sub == 0)
                        lse_ok = wait_uniform(&sm.bar[kBarLseFull + slot],
                                              (uint32_t)((nb / (kLseGroup * kLseSlots)) & 1));
                    ++nb;
                    if (acquire_acc(ab, aph)) {
                        const uint32_t tbase =
                            tmem_base + (uint32_t)(ab * a.acc_stride + col_base) + lane_off;
                        const float4 *L4 = reinterpret_cast<const float4 *>(
                            sm.lse + (slot * kLseGroup + sub) * kLseBlock + col_base);
                        // Per 16-column group: the TMEM read and the group's -lse (shared
                        // memory) in flight together.
#pragma unroll
                        for (int gi = 0; gi < kMaxGroups; ++gi)
                            if (gi < ng) {
                                float v[16], nl[16];
                                ptx::tmem_ld16(tbase + gi * 16, v);
#pragma unroll
                                for (int q = 0; q < 4; ++q) {
                                    const float4 f = lse_ok ? L4[gi * 4 + q]
                                                            : make_float4(-INFINITY, -INFINITY,
                                                                          -INFINITY, -INFINITY);
                                    nl[4 * q] = f.x;
                                    nl[4 * q + 1] = f.y;
                                    nl[4 * q + 2] = f.z;
                                    nl[4 * q + 3] = f.w;
                                }
                                ptx::tmem_ld_wait_dep(v);
                                col_add<kDiag>(acc, v, nl, s2, key, p0, a.pb, col_base + gi * 16);
                            }
                    }
                    // Every warp has read this block's -lse: the fourth block of a group frees
                    // the slot.
                    if (lse_ok && sub == kLseGroup - 1) {
                        __syncwarp();
                        if (lane == 0)
                            ptx::mbar_arrive(&sm.bar[kBarLseEmpty + slot]);
                    }
                    release_acc(ab);
                    ++tc;
                };
                // Block i is masked while its first position precedes the tile's last key.
                const int ndiag =
                    min(T.ntiles, max(0, (k0 + kTile + a.pb - 1) / a.pb - T.first));
                for (int i = 0; i < ndiag; ++i)
                    tile2(i, std::true_type());
                for (int i = ndiag; i < T.ntiles; ++i)
                    tile2(i, std::false_type());
                // The three warps of this lane quarter (one per warpgroup) leave their sums in
                // shared memory; a warp whose arrival completes the phase adds them in
                // warpgroup order and stores the key's score (two may both see it complete:
                // they store the same value).  An area is rewritten four tasks later, which
                // needs every warp past the first tile of the next task.
                const int xb = xc % kXchBufs;
                ++xc;
                float *xs = sm.xch + xb * kEpiWG * kTile;
                xs[wg * kTile + kl] =
                    ((acc[0].x + acc[0].y) + (acc[1].x + acc[1].y)) +
                    ((acc[2].x + acc[2].y) + (acc[3].x + acc[3].y));
                __syncwarp();
                int last = 0;
                if (lane == 0) {
                    uint64_t *b = &sm.bar[kBarXch + xb * 4 + quarter];
                    last = ptx::mbar_test_token(b, ptx::mbar_arrive_token(b)) ? 1 : 0;
                }
                last = __shfl_sync(0xffffffffu, last, 0);
                __syncwarp();
                if (last && !dead && key < g.P) {
                    float total = xs[kl];
#pragma unroll
                    for (int w = 1; w < kEpiWG; ++w)
                        total += xs[w * kTile + kl];
                    a.raw[T.u * g.P + key] = total;
                }
            }
        }
    }

    // ---- teardown ------------------------------------------------------------------------
    __syncthreads();
    if (warp == 0 && lane == 0) {
        // Copies still in flight (only after an abort) land before the CTA leaves.
        for (int i = 0; i < kStages; ++i)
            if (flag[kFlagRingArm + i] >= 0)
                tc::drain_bar(&sm.bar[kBarRingFull + i], (uint32_t)flag[kFlagRingArm + i],
                              1000000000ull);
        for (int i = 0; i < 2; ++i)
            if (flag[kFlagStatArm + i] >= 0)
                tc::drain_bar(&sm.bar[kBarStatFull + i], (uint32_t)flag[kFlagStatArm + i],
                              1000000000ull);
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    if (warp == 1)
        ptx::tmem_dealloc(tmem_base, kTmemCols);
}

}  // namespace

bool h2o_tc_supported(const Geometry &g)
{
    if (g.variant != DGE_VARIANT_H2O || (g.d != 64 && g.d != 128) || g.G < 1)
        return false;
    // At least 16 positions per block: the causal mask of a 16-column group then wraps to the
    // next head at most once, and every block keeps the tensor pipe busy.
    if (kBlockRows1 / g.G < 16 || kBlockRows2 / g.G < 16)
        return false;
    int dev = 0, major = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess)
        return false;
    return major == 10 && tc::have_tensor_maps();
}

H2oPlan h2o_tc_plan(const Geometry &g)
{
    H2oPlan p;
    p.nslab = g.d / 64;
    p.nkt = (g.P + kTile - 1) / kTile;
    for (int ph = 1; ph <= 2; ++ph) {
        H2oPhase &q = p.ph[ph - 1];
        q.pb = (ph == 1 ? kBlockRows1 : kBlockRows2) / g.G;
        if (q.pb > g.n)
            q.pb = g.n;
        q.rows = g.G * q.pb;
        q.r_pad = (q.rows + 15) & ~15;
        q.nqb = (g.n + q.pb - 1) / q.pb;
        const size_t s = smem_bytes(ph, q.r_pad, p.nslab);
        // At least half of the SM's shared memory: one CTA per SM, so a CTA's TMEM
        // allocation (all 512 columns) never waits for another CTA of this kernel.
        q.smem = s < 120 * 1024 ? 120 * 1024 : s;
    }
    return p;
}

cudaError_t launch_h2o_tc(int phase, const TensorDesc &K, const TensorDesc &Q, const Geometry &g,
                          const H2oPlan &plan, float *lse2, float *raw, uint32_t *ready,
                          uint32_t *status, cudaStream_t stream, bool *encoded)
{
    CUtensorMap tmK, tmQ, tmKm;
    memset(&tmKm, 0, sizeof tmKm);
    const bool merged = K.bt && tc::encode_k_merged_map(&tmKm, K, g.L, g.Hkv, g.d);
    *encoded = tc::encode_k_map(&tmK, K, g.L, g.b, g.Hkv, g.n, g.d) &&
               tc::encode_5d(&tmQ, Q, g.L, g.b, g.Hq, g.n, g.d, plan.ph[phase - 1].pb, g.G);
    if (!*encoded)
        return cudaSuccess;
    int dev = 0, sms = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err == cudaSuccess)
        err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (err != cudaSuccess)
        return err;

    H2oArgs a;
    a.g = g;
    a.kp = tc::k_paging(K, g.n);
    a.kp.merged = merged ? 1 : 0;
    const H2oPhase &q = plan.ph[phase - 1];
    a.phase = phase;
    a.pb = q.pb;
    a.rows = q.rows;
    a.r_pad = q.r_pad;
    a.nslab = plan.nslab;
    a.acc_stride = (q.r_pad + 31) & ~31;
    a.nqb = q.nqb;
    a.nkt = plan.nkt;
    a.items = g.U * (phase == 1 ? (int64_t)q.nqb : (int64_t)plan.nkt);
    const int NG = q.r_pad / 16;
    for (int w = 0, base = 0; w < kEpiWG; ++w) {
        a.ng[w] = NG / kEpiWG + (w < NG % kEpiWG ? 1 : 0);
        a.gbase[w] = base;
        base += a.ng[w];
    }
    a.lse2 = lse2;
    a.raw = raw;
    a.ready = ready;
    a.status = status;
    a.timeout_ns = tc_wait_limit_ns();
    if (a.items == 0)
        return cudaSuccess;
    const size_t smem = q.smem;
    auto kernel = phase == 1
                      ? (K.bt ? h2o_tc_kernel<true, kAccBufs1> : h2o_tc_kernel<false, kAccBufs1>)
                      : (K.bt ? h2o_tc_kernel<true, kAccBufs2> : h2o_tc_kernel<false, kAccBufs2>);
    err = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (err != cudaSuccess)
        return err;
    const int64_t grid = a.items < sms ? a.items : sms;
    kernel<<<(unsigned)grid, kThreads, smem, stream>>>(tmK, tmQ, tmKm, a);
    return cudaGetLastError();
}

}  // namespace dge
