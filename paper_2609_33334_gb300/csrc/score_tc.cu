// score_tc.cu -- the attention-score pass on the 5th-generation tensor cores.
//
// Same quantities as score_mma.cu (Alg. 1 line B; App. B; App. G), in base 2:
//   x_rj = log2(e) * scale * q_r . k_j,  lse_r = log2 sum_{j <= pos_r} 2^{x_rj},
//   raw_j = sum_r 2^{x_rj - lse_r}.
//
// One persistent CTA per SM, warp-specialised:
//   warp 0      TMA producer: the unit's stacked query block (5-D box, G heads x m
//               rows) and 128-key tiles of K, 128-byte swizzled, into a ring;
//   warp 1      MMA issuer: D[128 keys x R_pad rows] = K_tile . Q^T with
//               tcgen05.mma (M = 128, N = R_pad, bf16 -> fp32) into one of three
//               TMEM accumulators; also owns the TMEM allocation;
//   warps 2-3   coordinator: warp 3 publishes the phase-1 chunk sums and counts
//               them into the unit; warp 2 merges a finished unit's chunk sums
//               (bulk-copied to shared memory) into -lse for this CTA's phase-2
//               tasks;
//   warps 4-15  epilogue: three warpgroups, each thread one key (TMEM lane),
//               each warpgroup a third of the row columns.
// Work items are (unit, key chunk).  Tasks -- phase 1 of an item (per-row sums 2^x over the
// chunk) or phase 2 (2^{x - lse} summed over rows per key) -- form one sequence in which
// phase 1 of item lag + j and phase 2 of item j alternate; each CTA's producer claims the
// next task from a global counter when it needs one, and hands it to the other roles
// through a ring in shared memory.  Claiming in sequence order keeps the CTAs together (a
// slow CTA claims fewer tasks, so no CTA falls behind the others), so phase 2 re-reads a
// chunk about `lag` items after its phase-1 read, while it is still in L2, and a task only
// ever waits for tasks claimed before it.  Row sums use no running maximum: fp32 holds 2^x
// for |x| < 126, and a unit whose sums leave [2^-60, 2^126) is flagged (ready = 2) and
// recomputed by the warp-level path.
//
// Every wait is bounded: on expiry the CTA records DGE_ERR_DEVICE_TIMEOUT in the
// status word, stops issuing work, waits (bounded) for its own copies and MMAs,
// frees TMEM and returns.
#include <cuda.h>
#include <math.h>
#include <string.h>


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
// Registers per thread after reallocation: warpgroup 0 (producer, MMA, coordinators) gives
// up registers to the epilogue warpgroups.  The block launches with 512 threads x 128
// registers; 4*32*64 + 12*32*144 fits in that.  (56 / 152 left the producer spilling:
// c3 1 % and 16-slot pages 5 % slower.)
constexpr int kRegsLaunch = 128, kRegsControl = 64, kRegsEpilogue = 144;
static_assert(4 * 32 * kRegsControl + kEpiWarps * 32 * kRegsEpilogue <= kThreads * kRegsLaunch,
              "register split");
constexpr int kMaxGroups = 3;             // 16-column groups per epilogue warpgroup
constexpr int kMaxKStages = 4;
constexpr int kAccBufs = 3;               // TMEM accumulators
constexpr int kTmemCols = 512;
constexpr int kSlabBytes = kTile * 128;  // 128 rows x 64 bf16
constexpr uint32_t kReadyBad = 2;          // unit left fp32's range: recomputed afterwards

// Barrier slots.
constexpr int kBarKFull = 0, kBarKEmpty = 4, kBarQFull = 8, kBarQEmpty = 10, kBarAccFull = 12,
              kBarAccEmpty = 15, kBarDrain = 18, kBarRedFull = 19, kBarRedEmpty = 21,
              kBarLseFull = 23, kBarLseEmpty = 25, kBarStage = 27, kBarXch = 28,
              kBarRingFull = 40, kBarRingEmpty = 48, kNumBars = 56;
constexpr int kRing = 8;                  // claimed tasks handed from the producer to the others
// Lag of the claim sequence in tenths of the grid (see launch_score_tc) and the key tiles of a
// task of whole units (see tc_plan).
#ifndef DGE_TC_LAG_GRID_X10
#define DGE_TC_LAG_GRID_X10 15
#endif
#ifndef DGE_TC_CHUNK_TILES
#define DGE_TC_CHUNK_TILES 128
#endif
constexpr int kLagGridX10 = DGE_TC_LAG_GRID_X10;
// The producer claims the next task this many tiles before the current task's last copy.
#ifndef DGE_TC_CLAIM_AHEAD
#define DGE_TC_CLAIM_AHEAD 4
#endif
constexpr int kClaimAhead = DGE_TC_CLAIM_AHEAD;
constexpr int kChunkTiles = DGE_TC_CHUNK_TILES;
constexpr int kPageBuf = tc::kPageWindow + 4;   // ints of one page-id window buffer
// Fewest items (unit, chunk) of a launch of whole units: about three per SM of a 152-SM GB300.
constexpr int kMinItems = 456;
// Arrivals that free a ring slot: the MMA warp, the two coordinator warps, the epilogue warps.
constexpr int kRingConsumers = 3 + 12;
constexpr int kStageBytes = 12288;        // chunk sums of a unit, staged for the lse merge
constexpr int kCtrlBytes = 640;            // barriers, TMEM address, flags, ring (16-byte multiple)
constexpr int kRowsPerLane = 5;           // rows of the lse merge per lane (R <= 160)
// Flag slots (ints): abort, then the parity of the last arm of every key stage, query
// buffer and the staging buffer (-1 = never armed) for the drain.
constexpr int kFlagAbort = tc::kFlagAbort, kFlagKArm = 4, kFlagQArm = 8, kFlagSArm = 10;

struct TcArgs {
    Geometry g;
    tc::KPaging kp;    // K through a block table (kp.bt != nullptr)
    int rows;          // stacked rows of a sub-unit: gsub heads x m (all of R when nrb == 1)
    int nrb, gsub;     // sub-units (row blocks) per unit, query heads per sub-unit
    int r_pad, r4, nslab, kstages;
    int acc_stride;    // TMEM columns between accumulator buffers
    int unit_tiles, nchunks;   // key tiles of a unit; chunk c = tiles [c*T/nc, (c+1)*T/nc)
    int p1_chunks;     // chunks with phase-1 keys (the first ones: they start below n - m)
    int nparts;        // chunk-sum slots per sub-unit: nchunks, then the tail's (slot nchunks)
    int64_t items;
    int64_t lag;       // items between an item's phase-1 and phase-2 tasks (>= nchunks - 1)
    int64_t total;     // tasks in the claim sequence
    uint32_t *claim;   // claim counter, zero before the launch
    const float *lse_in;  // [U][R] natural-log row normalisers supplied by the caller: then
                          // there is no phase 1 and phase 2 of item t*S + s runs in step t
    int ng[kEpiWG];    // 16-column groups of each epilogue warpgroup
    int gbase[kEpiWG]; // first group of each epilogue warpgroup
    float *part;       // [U][nchunks][r4]
    float *lse2;       // [U][R]
    float *raw;        // [U][P] (nrb == 1)
    unsigned long long *raw_fx;  // [U][P] fixed point, 2^-40 units (nrb > 1): row blocks add
    uint32_t *count;   // [U*nrb] phase-1 chunks counted in, per sub-unit
    uint32_t *ready;   // [U] 2 = the unit left fp32's range (recomputed afterwards)
    uint32_t *list;    // [1 + U] units to recompute: count, then ids
    uint32_t *status;
    unsigned long long timeout_ns;
    int count_extra;   // chunks a unit's count must exceed nchunks by (0; > 0 only in tests)
    unsigned long long *trace;  // see dge_trace_set; nullptr = off
    int trace_cta;
};

// Cycle accounting (see dge_trace_set): per-role sums of SM clock cycles, written once per
// CTA at the end into trace[slot * DGE_TRACE_LEN + blockIdx.x].
enum TraceSlot {
    kTrMmaWaitQ = 0, kTrMmaWaitK, kTrMmaWaitAcc, kTrMmaIssue, kTrMmaCommit, kTrMmaTotal,
    kTrProdWaitQ, kTrProdWaitK, kTrProdTotal, kTrEpiWaitAcc, kTrEpiMathP2, kTrEpiP1End,
    kTrEpiP2Start, kTrTimeline, kTrEpiTotal, kTrTiles, kTrTileIssue, kTrEpiMath, kTrEpiXch,
    kTrEpiRelease, kTrTileKReady, kTrTileAccFree, kTrTileIssued, kTrTileEpi
};

template <bool kTr>
__device__ __forceinline__ void trace_put(const TcArgs &a, int slot, long long v)
{
    if (kTr && a.trace && blockIdx.x < DGE_TRACE_LEN)
        a.trace[slot * DGE_TRACE_LEN + blockIdx.x] = (unsigned long long)v;
}

// Timeline of CTA a.trace_cta: global-timer stamps (ns) at index i of a timeline slot.
template <bool kTr>
__device__ __forceinline__ void trace_at(const TcArgs &a, int slot, int i)
{
    if (kTr && a.trace && (int)blockIdx.x == a.trace_cta && i >= 0 && i < DGE_TRACE_LEN)
        a.trace[slot * DGE_TRACE_LEN + i] = ptx::globaltimer();
}


// SM clock for the cycle accounting; a constant 0 in the kernel built without it.
template <bool kTr>
__device__ __forceinline__ long long tclock()
{
    if (kTr)
        return clock64();
    return 0;
}

struct Task {
    int phase;
    int64_t u;
    int chunk, k_lo, k_hi, ntiles;
};

// Task p of the claim sequence.  Items are item = u * nchunks + chunk.  Positions 0 .. lag-1
// are phase 1 of items 0 .. lag-1; then phase 1 of item lag + j and phase 2 of item j
// alternate; the last lag positions are phase 2 of the last lag items.  A unit's last chunk
// is at most nchunks - 1 items after any of its chunks, so with lag >= nchunks - 1 phase 2 of
// every chunk of a unit comes after phase 1 of all of them.  With normalisers supplied
// (lse_in) the sequence is phase 2 of every item in order.  False when p is past the end or
// the task covers no keys.
__device__ __forceinline__ bool task_at(const TcArgs &a, int64_t p, Task &T)
{
    int64_t item;
    if (a.lse_in) {
        item = p;
        T.phase = 2;
    } else if (p < a.lag) {
        item = p;
        T.phase = 1;
    } else {
        const int64_t q = p - a.lag, mid = 2 * (a.items - a.lag);
        if (q < mid) {
            item = (q & 1) ? (q >> 1) : a.lag + (q >> 1);
            T.phase = (q & 1) ? 2 : 1;
        } else {
            item = a.items - a.lag + (q - mid);
            T.phase = 2;
        }
    }
    if (p < 0 || p >= a.total || item < 0 || item >= a.items)
        return false;
    T.u = item / a.nchunks;
    T.chunk = (int)(item % a.nchunks);
    T.k_lo = (int)((int64_t)T.chunk * a.unit_tiles / a.nchunks) * kTile;
    const int k_end = (int)((int64_t)(T.chunk + 1) * a.unit_tiles / a.nchunks) * kTile;
    // Phase 1 covers the keys every observation row sees, [0, n - m); the rows' own positions
    // [n - m, n) are added by the tail kernel (masked there).  Phase 2 covers [0, P), P <= n - m.
    const int end = T.phase == 1 ? a.g.n - a.g.m : a.g.P;
    T.k_hi = min(k_end, end);
    if (T.k_lo >= T.k_hi)
        return false;
    T.ntiles = (T.k_hi - T.k_lo + kTile - 1) / kTile;
    return true;
}

struct Smem {
    uint8_t *q;          // [2][nslab][r_pad * 128]
    uint8_t *k;          // [kstages][nslab][kSlabBytes]
    float *stage;        // [kStageBytes / 4] chunk sums of one unit (lse merge)
    uint64_t *bar;       // [kNumBars]
    uint32_t *tmem;      // allocation result
    int *flag;           // [16]
    volatile int64_t *ring;  // [kRing] claimed task positions (-1: no more tasks)
    float *sL;           // [2][256] -lse of the rows of a phase-2 task (padding: -inf)
    float *red;          // [2][kEpiWG][4][kMaxGroups * 16] per-warp phase-1 row sums
    int *sLbad;          // [2] that task's unit is recomputed elsewhere
    float *xch;          // [kAccBufs][kEpiWG][128] phase-2 partial column sums
    int *pages;          // [2][kPageBuf] page ids of the producer's current and next window (paged caches)
};

__host__ __device__ inline size_t smem_bytes(int r_pad, int nslab, int kstages)
{
    return 1024                                   // alignment slack
           + (size_t)2 * nslab * r_pad * 128      // query buffers
           + (size_t)kstages * nslab * kSlabBytes // key ring
           + kStageBytes                          // lse merge staging
           + kCtrlBytes                           // barriers, tmem holder, flags
           + (2 * 256 + 2 * kEpiWG * 4 * kMaxGroups * 16) * 4 + 16
           + kAccBufs * kEpiWG * kTile * 4 + 2 * kPageBuf * 4;
}

__device__ __forceinline__ Smem carve(uint8_t *raw, int r_pad, int nslab, int kstages)
{
    // Offsets from the shared-memory symbol itself, so every pointer stays a shared-space
    // pointer (32-bit addressing) rather than a generic one.
    const uint32_t base = ptx::smem_addr(raw);
    uint32_t off = ((base + 1023u) & ~1023u) - base;
    Smem s;
    s.q = raw + off;
    off += (uint32_t)(2 * nslab * r_pad * 128);
    s.k = raw + off;
    off += (uint32_t)(kstages * nslab * kSlabBytes);
    s.stage = reinterpret_cast<float *>(raw + off);
    off += kStageBytes;
    s.bar = reinterpret_cast<uint64_t *>(raw + off);
    s.tmem = reinterpret_cast<uint32_t *>(raw + off + kNumBars * 8);
    s.flag = reinterpret_cast<int *>(raw + off + kNumBars * 8 + 16);
    s.ring = reinterpret_cast<int64_t *>(raw + off + kNumBars * 8 + 16 + 64);
    static_assert(kNumBars * 8 + 16 + 64 + kRing * 8 <= kCtrlBytes, "control block");
    off += kCtrlBytes;
    s.sL = reinterpret_cast<float *>(raw + off);  // 16-byte aligned: read as float4
    off += 2 * 256 * 4;
    s.red = reinterpret_cast<float *>(raw + off);
    off += 2 * kEpiWG * 4 * kMaxGroups * 16 * 4;
    s.sLbad = reinterpret_cast<int *>(raw + off);
    off += 16;
    s.xch = reinterpret_cast<float *>(raw + off);
    off += kAccBufs * kEpiWG * kTile * 4;
    s.pages = reinterpret_cast<int *>(raw + off);
    return s;
}

// Bounded wait on an mbarrier phase (false once the CTA has aborted or timed out).
__device__ __forceinline__ bool wait_bar(uint64_t *bar, uint32_t parity, volatile int *flag,
                                         const TcArgs &a)
{
    return tc::wait_bar(bar, parity, flag, a.timeout_ns, a.status);
}

using tc::drain_bar;
using tc::transpose_sum16;
using tc::transpose_sum32;


// Phase 1 for one 16-column group: z[c] += 2^{x_c} (every row sees every key of phase 1).
// Padding columns (no query row) are computed too: skipping them measured slower (one more
// branch in the loop) than their exponentials cost.
__device__ __forceinline__ void rows_add(float (&z)[16], const float (&w)[16], float s2, bool valid)
{
    if (!valid)
        return;
    const float2 sc = make_float2(s2, s2);
#pragma unroll
    for (int c = 0; c < 16; c += 2) {
        const float2 x = __fmul2_rn(make_float2(w[c], w[c + 1]), sc);
        const float2 acc = __fadd2_rn(make_float2(z[c], z[c + 1]),
                                      make_float2(ex2(x.x), ex2(x.y)));
        z[c] = acc.x;
        z[c + 1] = acc.y;
    }
}

// Phase 2 for one 16-column group: adds 2^{x_c - lse_c} over the group's rows into the
// pair accumulator.  nL holds -lse (padded columns: -inf, so they add exactly 0).
__device__ __forceinline__ void col_add(float2 &acc, const float (&w)[16], const float (&nL)[16],
                                        float s2)
{
    const float2 sc = make_float2(s2, s2);
#pragma unroll
    for (int c = 0; c < 16; c += 2) {
        const float2 x = __ffma2_rn(make_float2(w[c], w[c + 1]), sc,
                                    make_float2(nL[c], nL[c + 1]));
        acc = __fadd2_rn(acc, make_float2(ex2(x.x), ex2(x.y)));
    }
}

// Runs f(gi, v) over this warp's lane quarter of 16-column groups gi = 0 .. ng-1 (ng <=
// kMaxGroups, warp-uniform) read from TMEM, one group per round trip.  (Keeping the next
// group's load in flight while f runs measured markedly slower.)
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



// kTr: with the cycle accounting and timelines of dge_trace_set (a separate build, so the
// clock reads cost nothing when tracing is off).  kFx: units split into row blocks whose
// column sums meet in fixed point (a separate build, so the whole-unit path carries none of
// it: its epilogue is latency-bound and slowed by 5% with it).
template <bool kTr, bool kFx, bool kPaged>
__global__ void __launch_bounds__(kThreads, 1)
score_tc_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmQ,
                const __grid_constant__ CUtensorMap tmKm, const TcArgs a)
{
    extern __shared__ uint8_t smem_raw[];
    const Smem sm = carve(smem_raw, a.r_pad, a.nslab, a.kstages);
    volatile int *flag = sm.flag;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const Geometry &g = a.g;
    const uint32_t q_slab_bytes = (uint32_t)a.r_pad * 128;

    // ---- set-up -------------------------------------------------------------------
    if (threadIdx.x == 0) {
        for (int i = 0; i < a.kstages; ++i) {
            ptx::mbar_init(&sm.bar[kBarKFull + i], 1);
            ptx::mbar_init(&sm.bar[kBarKEmpty + i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            ptx::mbar_init(&sm.bar[kBarQFull + i], 1);
            ptx::mbar_init(&sm.bar[kBarQEmpty + i], 1);
        }
        for (int i = 0; i < kAccBufs; ++i) {
            ptx::mbar_init(&sm.bar[kBarAccFull + i], 1);
            ptx::mbar_init(&sm.bar[kBarAccEmpty + i], kEpiWarps);
        }
        ptx::mbar_init(&sm.bar[kBarDrain], 1);
        ptx::mbar_init(&sm.bar[kBarStage], 1);
        for (int i = 0; i < 2; ++i) {
            ptx::mbar_init(&sm.bar[kBarRedFull + i], kEpiWarps);
            ptx::mbar_init(&sm.bar[kBarRedEmpty + i], 1);
            ptx::mbar_init(&sm.bar[kBarLseFull + i], 1);
            ptx::mbar_init(&sm.bar[kBarLseEmpty + i], kEpiWarps);
        }
        flag[kFlagAbort] = 0;
        for (int i = 0; i < kMaxKStages; ++i)
            flag[kFlagKArm + i] = -1;
        flag[kFlagQArm] = flag[kFlagQArm + 1] = -1;
        flag[kFlagSArm] = -1;
        // Phase-2 exchange: one barrier per accumulator and lane quarter, one arrival per
        // warpgroup.
        for (int i = 0; i < kAccBufs * 4; ++i)
            ptx::mbar_init(&sm.bar[kBarXch + i], kEpiWG);
        for (int i = 0; i < kRing; ++i) {
            ptx::mbar_init(&sm.bar[kBarRingFull + i], 1);
            ptx::mbar_init(&sm.bar[kBarRingEmpty + i], kRingConsumers);
        }
        ptx::fence_mbar_init();
    }
    // Query rows R .. r_pad-1 are never written by TMA: zero them once so the padded
    // accumulator columns are exactly 0.
    {
        const int pad_rows = a.r_pad - a.rows;
        const int words = pad_rows * 128 / 16;
        for (int b = 0; b < 2; ++b)
            for (int s = 0; s < a.nslab; ++s) {
                int4 *base = reinterpret_cast<int4 *>(sm.q + ((size_t)b * a.nslab + s) * q_slab_bytes +
                                                      (size_t)a.rows * 128);
                for (int i = threadIdx.x; i < words; i += blockDim.x)
                    base[i] = make_int4(0, 0, 0, 0);
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
        // ---- TMA producer (the whole warp: lane 0 claims, arms the barriers and publishes;
        // the boxes of a copy are spread over the lanes, one box each) ----------------------
        if (lane == 0) {
            ptx::prefetch_tmap(&tmK);
            ptx::prefetch_tmap(&tmQ);
        }
        // Phase-1 tiles stay in L2 for the phase-2 re-read; the re-read marks them first to go.
        const uint64_t keep = ptx::make_policy_evict_last();
        const uint64_t drop = ptx::make_policy_evict_first();
        int ks = 0, ptc = 0;
        uint32_t kph = 0;
        long long cy_wq = 0, cy_wk = 0;
        const long long cy0 = tclock<kTr>();
        bool ok = true;
        // A bounded wait with a warp-uniform outcome.
        auto wait_w0 = [&](uint64_t *bar, uint32_t parity) -> bool {
            const bool got = wait_bar(bar, parity, flag, a);
            return __all_sync(0xffffffffu, got);
        };
        // Tasks are handed on one ahead: the next task is claimed kClaimAhead tiles before the
        // current one's last copy (lane 0's atomic; its value is read one tile later, so the
        // round trip is hidden), published to the ring then, and its query block loaded as
        // soon as that buffer is free, so neither the claim nor the query copy falls between
        // two tasks.  Task k uses query buffer k & 1.
        auto claim_one = [&]() -> uint32_t {
            uint32_t c = 0;
            if (lane == 0)
                c = atomicAdd(a.claim, 1u);
            return __shfl_sync(0xffffffffu, c, 0);
        };
        auto claim_next = [&](uint32_t first, Task &N) -> int64_t {
            for (uint32_t c = first; (int64_t)c < a.total; c = claim_one())
                if (task_at(a, c, N))
                    return c;
            return -1;
        };
        auto publish = [&](int k, int64_t pos) -> bool {
            const int slot = k % kRing;
            if (!wait_w0(&sm.bar[kBarRingEmpty + slot], (uint32_t)((k / kRing) & 1) ^ 1u))
                return false;
            if (lane == 0) {
                sm.ring[slot] = pos;
                ptx::mbar_arrive(&sm.bar[kBarRingFull + slot]);
            }
            return true;
        };
        auto load_q = [&](const Task &N, int b, uint32_t ph) {
            int l, bb, h;
            unit_coords(g, kFx ? N.u / a.nrb : N.u, l, bb, h);
            const int qhead = h * g.G + (kFx ? (int)(N.u % a.nrb) * a.gsub : 0);
            if (lane == 0) {
                ptx::mbar_arrive_expect_tx(&sm.bar[kBarQFull + b],
                                           (uint32_t)a.nslab * 128u * (uint32_t)a.rows);
                flag[kFlagQArm + b] = (int)ph;
            }
            __syncwarp();
            if (lane < a.nslab)
                ptx::tma_load_5d_hint(sm.q + ((size_t)b * a.nslab + lane) * q_slab_bytes, &tmQ,
                                      &sm.bar[kBarQFull + b], lane * 64, 0, qhead, bb, l, keep);
        };
        Task T;
        int64_t p = claim_next(claim_one(), T);
        ok = publish(0, p);
        bool q_ready = false;  // the current task's query block is already on its way
        for (int k = 0; ok && p >= 0; ++k) {
            const int qb = k & 1;
            const uint32_t qph = (uint32_t)((k >> 1) & 1);
            if (!q_ready) {
                long long c0 = tclock<kTr>();
                if (!wait_w0(&sm.bar[kBarQEmpty + qb], qph ^ 1)) {
                    ok = false;
                    break;
                }
                cy_wq += tclock<kTr>() - c0;
                load_q(T, qb, qph);
            }
            int l, bb, h;
            unit_coords(g, kFx ? T.u / a.nrb : T.u, l, bb, h);
            Task N;
            int64_t np = -1;
            uint32_t pend = 0;  // lane 0's claimed position (valid once read after a tile)
            bool claimed = false, pushed = false, nq = false;
            const int claim_at = max(T.ntiles - kClaimAhead, 0);
            const int nqb = qb ^ 1;
            const uint32_t nqph = (uint32_t)(((k + 1) >> 1) & 1);
            const uint64_t pol = T.phase == 2 ? drop : keep;
            int w0 = 0;               // first key of the page-id window (paged caches)
            const int *ids = sm.pages;
            int wrun = -1;            // lane t: tile t of the window as one run of pages, or -1
            for (int tile = 0; tile < T.ntiles; ++tile) {
                if (tile == claim_at) {
                    if (lane == 0)
                        pend = atomicAdd(a.claim, 1u);
                    claimed = true;
                } else if (claimed && !pushed) {
                    np = claim_next(__shfl_sync(0xffffffffu, pend, 0), N);
                    if (!publish(k + 1, np)) {
                        ok = false;
                        break;
                    }
                    pushed = true;
                }
                if (pushed && np >= 0 && !nq &&
                    __shfl_sync(0xffffffffu,
                                ptx::mbar_test_parity(&sm.bar[kBarQEmpty + nqb], nqph ^ 1) ? 1
                                                                                            : 0,
                                0)) {
                    load_q(N, nqb, nqph);
                    nq = true;
                }
                if constexpr (kPaged) {
                    // Page ids a window of kPageWindowTiles tiles at a time, double buffered:
                    // at a window's first tile the next window's ids are requested into the
                    // other buffer (whose window is done), and only this window's are waited
                    // for -- in flight since the previous window began, except for a task's
                    // first window.
                    constexpr int W = tc::kPageWindowTiles;
                    if (tile % W == 0) {
                        const int wi = tile / W;
                        int *buf = sm.pages + (wi & 1) * kPageBuf;
                        if (wi == 0) {
                            tc::fetch_pages_issue_warp(buf, a.kp, bb, T.k_lo, min(T.ntiles, W),
                                                       lane);
                            tc::fetch_pages_commit();
                        }
                        if (tile + W < T.ntiles) {
                            tc::fetch_pages_issue_warp(sm.pages + ((wi + 1) & 1) * kPageBuf,
                                                       a.kp, bb, T.k_lo + (tile + W) * kTile,
                                                       min(T.ntiles - tile - W, W), lane);
                            tc::fetch_pages_commit();
                            tc::fetch_pages_wait_group<1>();
                        } else {
                            tc::fetch_pages_wait_group<0>();
                        }
                        __syncwarp();
                        w0 = T.k_lo + tile * kTile;
                        ids = tc::page_ids_at(buf, a.kp, bb, w0);
                        wrun = tc::tile_runs(a.kp, ids, w0, min(T.ntiles - tile, W), lane);
                    }
                }
                long long c0 = tclock<kTr>();
                if (!wait_w0(&sm.bar[kBarKEmpty + ks], kph ^ 1)) {
                    ok = false;
                    break;
                }
                cy_wk += tclock<kTr>() - c0;
                if (lane == 0) {
                    trace_at<kTr>(a, kTrTileIssue, ptc);
                    ptx::mbar_arrive_expect_tx(&sm.bar[kBarKFull + ks],
                                               (uint32_t)a.nslab * kSlabBytes);
                    flag[kFlagKArm + ks] = (int)kph;
                }
                ++ptc;
                __syncwarp();
                tc::load_k_tile_warp<kPaged>(sm.k + (size_t)ks * a.nslab * kSlabBytes,
                                             kSlabBytes, a.nslab, &tmK, &tmKm,
                                             &sm.bar[kBarKFull + ks], T.k_lo + tile * kTile, l,
                                             bb, h, a.kp, ids, w0, pol, lane,
                                             kPaged ? __shfl_sync(0xffffffffu, wrun,
                                                                  tile % tc::kPageWindowTiles)
                                                    : -1);
                if (++ks == a.kstages) {
                    ks = 0;
                    kph ^= 1;
                }
            }
            if (!ok)
                break;
            if (!claimed && lane == 0)
                pend = atomicAdd(a.claim, 1u);
            if (!pushed) {
                np = claim_next(__shfl_sync(0xffffffffu, pend, 0), N);
                if (!publish(k + 1, np)) {
                    ok = false;
                    break;
                }
            }
            T = N;
            p = np;
            q_ready = nq;
        }
        if constexpr (kPaged)
            tc::fetch_pages_wait_group<0>();   // no page-id copy outlives the loop (aborts)
        if (lane == 0) {
            trace_put<kTr>(a, kTrProdWaitQ, cy_wq);
            trace_put<kTr>(a, kTrProdWaitK, cy_wk);
            trace_put<kTr>(a, kTrProdTotal, tclock<kTr>() - cy0);
        }
    } else if (warp == 1) {
        // ---- MMA issuer -----------------------------------------------------------------
        if (lane == 0) {
            const uint32_t idesc = ptx::idesc_bf16_f32(kTile, a.r_pad);
            int ks = 0, qb = 0;
            uint32_t kph = 0, qph = 0;
            int64_t tc = 0;  // accumulator sequence number: buffer tc % 3, use tc / 3
            long long cy_wq = 0, cy_wk = 0, cy_wa = 0, cy_is = 0, cy_cm = 0;
            const long long cy0 = tclock<kTr>();
            bool ok = true;
            for (int k = 0; ok; ++k) {
                    const int slot = k % kRing;
                    if (!wait_bar(&sm.bar[kBarRingFull + slot], (uint32_t)((k / kRing) & 1), flag,
                                  a))
                        break;
                    const int64_t p = sm.ring[slot];
                    ptx::mbar_arrive(&sm.bar[kBarRingEmpty + slot]);
                    Task T;
                    if (p < 0 || !task_at(a, p, T))
                        break;
                    long long c0 = tclock<kTr>();
                    if (!wait_bar(&sm.bar[kBarQFull + qb], qph, flag, a)) {
                        ok = false;
                        break;
                    }
                    cy_wq += tclock<kTr>() - c0;
                    const uint32_t qbase = ptx::smem_addr(sm.q + (size_t)qb * a.nslab * q_slab_bytes);
                    for (int tile = 0; tile < T.ntiles; ++tile, ++tc) {
                        const int ab = (int)(tc % kAccBufs);
                        const uint32_t aph = (uint32_t)((tc / kAccBufs) & 1);
                        c0 = tclock<kTr>();
                        if (!wait_bar(&sm.bar[kBarKFull + ks], kph, flag, a)) {
                            ok = false;
                            break;
                        }
                        long long c1 = tclock<kTr>();
                        cy_wk += c1 - c0;
                        trace_at<kTr>(a, kTrTileKReady, (int)tc);
                        if (!wait_bar(&sm.bar[kBarAccEmpty + ab], aph ^ 1, flag, a)) {
                            ok = false;
                            break;
                        }
                        trace_at<kTr>(a, kTrTileAccFree, (int)tc);
                        c0 = tclock<kTr>();
                        cy_wa += c0 - c1;
                        ptx::tc_fence_after();
                        // Descriptors are linear in the start address (bits 0..13 hold
                        // addr >> 4), so each K step adds its byte offset / 16.
                        const uint64_t ad0 = ptx::smem_desc_sw128(
                            ptx::smem_addr(sm.k + (size_t)ks * a.nslab * kSlabBytes));
                        const uint64_t bd0 = ptx::smem_desc_sw128(qbase);
                        const uint32_t d_tmem = tmem_base + (uint32_t)(ab * a.acc_stride);
#pragma unroll
                        for (int kk = 0; kk < 8; ++kk) {
                            if (kk < a.nslab * 4) {
                                const uint32_t a_off = ((uint32_t)(kk >> 2) * kSlabBytes +
                                                        (uint32_t)(kk & 3) * 32u) >> 4;
                                const uint32_t b_off = ((uint32_t)(kk >> 2) * q_slab_bytes +
                                                        (uint32_t)(kk & 3) * 32u) >> 4;
                                ptx::mma_bf16(d_tmem, ad0 + a_off, bd0 + b_off, idesc,
                                              kk > 0 ? 1u : 0u);
                            }
                        }
                        c1 = tclock<kTr>();
                        cy_is += c1 - c0;
                        ptx::mma_commit(&sm.bar[kBarKEmpty + ks]);
                        ptx::mma_commit(&sm.bar[kBarAccFull + ab]);
                        cy_cm += tclock<kTr>() - c1;
                        trace_at<kTr>(a, kTrTileIssued, (int)tc);
                        if (++ks == a.kstages) {
                            ks = 0;
                            kph ^= 1;
                        }
                    }
                    if (!ok)
                        break;
                    ptx::mma_commit(&sm.bar[kBarQEmpty + qb]);
                    qb ^= 1;
                    if (qb == 0)
                        qph ^= 1;
                }
            trace_put<kTr>(a, kTrMmaWaitQ, cy_wq);
            trace_put<kTr>(a, kTrMmaWaitK, cy_wk);
            trace_put<kTr>(a, kTrMmaWaitAcc, cy_wa);
            trace_put<kTr>(a, kTrMmaIssue, cy_is);
            trace_put<kTr>(a, kTrMmaCommit, cy_cm);
            trace_put<kTr>(a, kTrMmaTotal, tclock<kTr>() - cy0);
            trace_put<kTr>(a, kTrTiles, tc);
            // Every MMA issued so far completes before the drain barrier fires.
            ptx::mma_commit(&sm.bar[kBarDrain]);
            drain_bar(&sm.bar[kBarDrain], 0, 2000000000ull);
        }
    } else {
        // ---- coordinator: warp 2 stages lse, warp 3 hands off row sums ---------------------
        // Warp 3, per phase-1 task: adds the epilogue warps' row sums of the chunk, publishes
        // them and counts the chunk into its unit.  Warp 2, per phase-2 task: waits until
        // every chunk of the task's unit is counted, brings the unit's chunk sums into
        // shared memory with bulk copies, adds them in chunk order (the same result in every
        // CTA that needs the unit) and stages -lse for the epilogue.  The two warps never
        // wait on each other, and a phase-2 task needs only phase-1 tasks claimed before it,
        // so the waits cannot form a cycle.
        bool dead = false;
        auto wait_w = [&](uint64_t *bar, uint32_t parity) {
            if (!dead) {
                const bool got = wait_bar(bar, parity, flag, a);
                dead = !__all_sync(0xffffffffu, got);
            }
            return !dead;
        };
        // This CTA's k-th claimed task from the ring (the whole warp reads it; lane 0 frees
        // the slot).  False at the end of the sequence or once the CTA is dead.
        auto ring_task = [&](int k, Task &T) -> bool {
            const int slot = k % kRing;
            if (!wait_w(&sm.bar[kBarRingFull + slot], (uint32_t)((k / kRing) & 1)))
                return false;
            const int64_t p = sm.ring[slot];
            __syncwarp();
            if (lane == 0)
                ptx::mbar_arrive(&sm.bar[kBarRingEmpty + slot]);
            return p >= 0 && task_at(a, p, T);
        };
        if (warp == 2) {
            // Bounded spin of one lane until every chunk of unit u is counted.
            auto spin_count = [&](const uint32_t *p) -> bool {
                const uint64_t t0 = ptx::globaltimer();
                const uint32_t need = (uint32_t)(a.p1_chunks + a.count_extra);
                while (ptx::ld_acquire_u32(p) < need) {
                    __nanosleep(64);
                    if (flag[kFlagAbort] || *(volatile uint32_t *)a.status != 0) {
                        flag[kFlagAbort] = 1;
                        return false;
                    }
                    if (ptx::globaltimer() - t0 > a.timeout_ns) {
                        flag[kFlagAbort] = 1;
                        set_status(a.status, DGE_ERR_DEVICE_TIMEOUT);
                        return false;
                    }
                }
                return true;
            };
            const int per_piece = kStageBytes / (a.r4 * 4);  // chunks per bulk copy
            uint32_t sph = 0;
            int p2c = 0;
            for (int k = 0;; ++k) {
                Task T;
                if (!ring_task(k, T))
                    break;
                if (T.phase != 2)
                    continue;
                const int lb = p2c & 1;
                const uint32_t lph = (uint32_t)((p2c >> 1) & 1);
                ++p2c;
                if (lane == 0)
                    trace_at<kTr>(a, kTrTimeline, 4 * (p2c - 1));
                int got = wait_w(&sm.bar[kBarLseEmpty + lb], lph ^ 1) ? 1 : 0;
                if (a.lse_in) {
                    // Supplied normalisers: -lse in base 2, straight from the caller's array.
                    float *L = sm.sL + lb * 256;
                    const float *src = a.lse_in + T.u * a.rows;
                    for (int r = lane; r < a.r_pad; r += 32)
                        L[r] = (got && r < a.rows) ? -__ldg(src + r) * 1.4426950408889634f
                                                : -INFINITY;
                    __syncwarp();
                    if (lane == 0) {
                        sm.sLbad[lb] = (!got || flag[kFlagAbort]) ? 1 : 0;
                        ptx::mbar_arrive(&sm.bar[kBarLseFull + lb]);
                    }
                    continue;
                }
                if (lane == 0) {
                    trace_at<kTr>(a, kTrTimeline, 4 * (p2c - 1) + 1);
                    got = got && spin_count(&a.count[T.u]);
                    // The acquire above saw every chunk's sums; the bulk copies below read
                    // them through the async proxy.
                    ptx::fence_proxy_async_global();
                    trace_at<kTr>(a, kTrTimeline, 4 * (p2c - 1) + 2);
                }
                got = __shfl_sync(0xffffffffu, got, 0);
                float Z[kRowsPerLane];
#pragma unroll
                for (int i = 0; i < kRowsPerLane; ++i)
                    Z[i] = 0.f;
                // Slots 0 .. p1_chunks-1 (chunk order), then the tail's slot nchunks; the
                // slots in between belong to chunks with no phase-1 keys and are skipped.
                const float *src = a.part + T.u * a.nparts * a.r4;
                for (int c0 = 0; got && c0 < a.nparts; c0 += per_piece) {
                    const int nc = min(per_piece, a.nparts - c0);
                    __syncwarp();
                    if (lane == 0) {
                        // The previous piece's reads (generic proxy) come before the copy.
                        ptx::fence_proxy_async_smem();
                        const uint32_t bytes = (uint32_t)(nc * a.r4 * 4);
                        ptx::mbar_arrive_expect_tx(&sm.bar[kBarStage], bytes);
                        flag[kFlagSArm] = (int)sph;
                        ptx::bulk_load(sm.stage, src + (int64_t)c0 * a.r4, bytes, &sm.bar[kBarStage]);
                    }
                    if (!wait_w(&sm.bar[kBarStage], sph)) {
                        got = 0;
                        break;
                    }
                    sph ^= 1;
                    for (int c = 0; c < nc; ++c) {
                        if (c0 + c >= a.p1_chunks && c0 + c < a.nchunks)
                            continue;
#pragma unroll
                        for (int i = 0; i < kRowsPerLane; ++i) {
                            const int r = lane + 32 * i;
                            if (r < a.rows)
                                Z[i] += sm.stage[c * a.r4 + r];
                        }
                    }
                }
                bool bad = false;
                float *L = sm.sL + lb * 256;
#pragma unroll
                for (int i = 0; i < kRowsPerLane; ++i) {
                    const int r = lane + 32 * i;
                    if (r < a.r_pad) {
                        float v = -INFINITY;
                        if (got && r < a.rows) {
                            if (!(Z[i] >= 0x1p-60f && Z[i] < 0x1p126f))
                                bad = true;
                            v = -log2f(Z[i]);
                        }
                        L[r] = v;
                    }
                }
                bad = __any_sync(0xffffffffu, bad);
                __syncwarp();
                if (lane == 0) {
                    sm.sLbad[lb] = (!got || bad || flag[kFlagAbort]) ? 1 : 0;
                    if (got && bad) {
                        // The unit (all of its row blocks) is recomputed after the kernel;
                        // the first CTA to flag it lists it.
                        const int64_t unit = T.u / a.nrb;
                        if (atomicExch(&a.ready[unit], kReadyBad) != kReadyBad)
                            a.list[1 + atomicAdd(a.list, 1u)] = (uint32_t)unit;
                    }
                    trace_at<kTr>(a, kTrTimeline, 4 * (p2c - 1) + 3);
                    ptx::mbar_arrive(&sm.bar[kBarLseFull + lb]);
                }
            }
        } else {
            int p1c = 0;
            for (int k = 0;; ++k) {
                Task T;
                if (!ring_task(k, T))
                    break;
                if (T.phase != 1)
                    continue;
                const int rb = p1c & 1;
                const uint32_t rph = (uint32_t)((p1c >> 1) & 1);
                ++p1c;
                const bool ok = wait_w(&sm.bar[kBarRedFull + rb], rph);
                if (ok) {
                    constexpr int W = kMaxGroups * 16;
                    float *dst = a.part + (T.u * a.nparts + T.chunk) * a.r4;
                    for (int col = lane; col < a.rows; col += 32) {
                        int w = 0;
                        while (w + 1 < kEpiWG && col >= a.gbase[w + 1] * 16)
                            ++w;
                        const int lc = col - a.gbase[w] * 16;
                        const float *rbuf = sm.red + (rb * kEpiWG + w) * 4 * W;
                        dst[col] = rbuf[lc] + rbuf[W + lc] + rbuf[2 * W + lc] + rbuf[3 * W + lc];
                    }
                    __threadfence();
                }
                __syncwarp();
                if (lane == 0) {
                    if (ok) {
                        // Cumulative release of every lane's sums with the chunk count.
                        ptx::fence_acq_rel_gpu();
                        atomicAdd(&a.count[T.u], 1u);
                    }
                    ptx::mbar_arrive(&sm.bar[kBarRedEmpty + rb]);
                }
            }
        }
    }
    } else {
        ptx::regs_inc<kRegsEpilogue>();
        // ---- epilogue -------------------------------------------------------------------
        // Every warpgroup reads every tile, its own 16-column groups: phase 1 keeps the row
        // sums in registers, phase 2 forms partial column sums that the three warps of a
        // lane quarter combine through shared memory.
        const int ew = warp - kEpiWarp0;         // 0 .. kEpiWarps-1
        const int wg = ew >> 2;                  // warpgroup
        const int quarter = warp & 3;            // TMEM lane quarter of this warp
        const int kl = quarter * 32 + lane;      // key within the tile
        const int ng = a.ng[wg];
        const int col_base = a.gbase[wg] * 16;
        const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
        const float s2 = g.scale_log2;
        int tc = 0;   // accumulator tiles consumed (buffer tc % 3, use tc / 3)
        int p1c = 0;  // phase-1 tasks (row-sum hand-off buffer p1c % 2)
        int p2c = 0;  // phase-2 tasks (-lse buffer p2c % 2)
        bool dead = false;

        long long cy_wa = 0, cy_p1e = 0, cy_p2s = 0, cy_math = 0, cy_math2 = 0, cy_xch = 0, cy_rel = 0;
        const long long cy0 = tclock<kTr>();
        // Waits for this thread's accumulator and returns false once the CTA is dead
        // (the outcome is warp-uniform: the TMEM loads after it are warp-collective).
        auto acquire_acc = [&](int ab, uint32_t aph) {
            const long long c0 = tclock<kTr>();
            if (!dead) {
                const bool got = wait_bar(&sm.bar[kBarAccFull + ab], aph, flag, a);
                dead = !__all_sync(0xffffffffu, got);
            }
            if (!dead)
                ptx::tc_fence_after();
            cy_wa += tclock<kTr>() - c0;
            if (ew == 0 && lane == 0)
                trace_at<kTr>(a, kTrTileEpi, tc);
            return !dead;
        };
        // A bounded, warp-uniform wait on a CTA barrier (false once the CTA is dead).
        auto wait_uniform = [&](uint64_t *bar, uint32_t parity) {
            if (!dead) {
                const bool got = wait_bar(bar, parity, flag, a);
                dead = !__all_sync(0xffffffffu, got);
            }
            return !dead;
        };
        auto release_acc = [&](int ab, uint32_t count) {
            const long long c0 = tclock<kTr>();
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0 && !dead)
                ptx::mbar_arrive_cnt(&sm.bar[kBarAccEmpty + ab], count);
            cy_rel += tclock<kTr>() - c0;
        };

        for (int k = 0;; ++k) {
                Task T;
                {
                    // This CTA's k-th claimed task (every epilogue warp frees the slot once).
                    const int slot = k % kRing;
                    if (!wait_uniform(&sm.bar[kBarRingFull + slot], (uint32_t)((k / kRing) & 1)))
                        break;
                    const int64_t p = sm.ring[slot];
                    __syncwarp();
                    if (lane == 0)
                        ptx::mbar_arrive(&sm.bar[kBarRingEmpty + slot]);
                    if (p < 0 || !task_at(a, p, T))
                        break;
                }
                if (ew == 0 && lane == 0)
                    trace_at<kTr>(a, kTrTimeline, 3072 + 4 * k);
                if (T.phase == 1) {
                    // ---------------- phase 1: row sums over this chunk ----------------
                    float z[kMaxGroups][16];
#pragma unroll
                    for (int i = 0; i < kMaxGroups; ++i)
#pragma unroll
                        for (int c = 0; c < 16; ++c)
                            z[i][c] = 0.f;
                    for (int tile = 0; tile < T.ntiles; ++tile, ++tc) {
                        const int ab = tc % kAccBufs;
                        const uint32_t aph = (uint32_t)((tc / kAccBufs) & 1);
                        const int tile0 = T.k_lo + tile * kTile;
                        const int key = tile0 + kl;
                        const bool valid = key < T.k_hi;
                        if (acquire_acc(ab, aph)) {
                            // All of this warp's columns in one TMEM round trip.
                            const uint32_t tbase =
                                tmem_base + (uint32_t)(ab * a.acc_stride + col_base) + lane_off;
                            const long long c0 = tclock<kTr>();
                            auto f1 = [&](int gi, const float(&v)[16]) {
#pragma unroll
                                for (int gj = 0; gj < kMaxGroups; ++gj)
                                    if (gj == gi)
                                        rows_add(z[gj], v, s2, valid);
                            };
                            for_groups(tbase, ng, f1);
                            cy_math += tclock<kTr>() - c0;
                        }
                        release_acc(ab, 1u);
                    }
                    const long long c_end = tclock<kTr>();
                    if (ew == 0 && lane == 0)
                        trace_at<kTr>(a, kTrTimeline, 3072 + 4 * k + 1);
                    // Sums over this warp's 32 keys, handed to the coordinator warps through
                    // a double-buffered area (they add the warps in a fixed order).
                    const int rb = p1c & 1;
                    const uint32_t rph = (uint32_t)((p1c >> 1) & 1);
#pragma unroll
                    for (int gi = 0; gi < kMaxGroups; gi += 2) {
                        if (gi < ng) {
                            if (gi + 1 < kMaxGroups && gi + 1 < ng)
                                transpose_sum32(z[gi], z[gi + 1 < kMaxGroups ? gi + 1 : gi], lane);
                            else
                                transpose_sum16(z[gi], lane);
                        }
                    }
                    if (ew == 0 && lane == 0)
                        trace_at<kTr>(a, kTrTimeline, 3072 + 4 * k + 2);
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
                        if (ew == 0 && lane == 0)
                            trace_at<kTr>(a, kTrTimeline, 3072 + 4 * k + 3);
                    }
                    ++p1c;
                    cy_p1e += tclock<kTr>() - c_end;
                } else {
                    const long long c_start = tclock<kTr>();
                    // ---------------- phase 2: column sums of this chunk ----------------
                    // The coordinator warp has put -lse of this unit's rows in sL[lb]; this
                    // warpgroup's columns go to registers and the buffer is released.
                    const int lb = p2c & 1;
                    const uint32_t lph = (uint32_t)((p2c >> 1) & 1);
                    ++p2c;
                    if (ew == 0 && lane == 0)
                        trace_at<kTr>(a, kTrTimeline, 2048 + 2 * (p2c - 1));
                    // -lse of this warpgroup's columns into registers for the whole task; the
                    // staging buffer is then free for the coordinator's next-but-one task.
                    // (Reading it from shared memory per group instead measured 1 % slower.)
                    float nL[kMaxGroups][16];
                    bool task_ok = false;
                    if (wait_uniform(&sm.bar[kBarLseFull + lb], lph)) {
                        const float4 *L4 =
                            reinterpret_cast<const float4 *>(sm.sL + lb * 256 + col_base);
#pragma unroll
                        for (int gi = 0; gi < kMaxGroups; ++gi)
#pragma unroll
                            for (int i = 0; i < 4; ++i) {
                                const float4 q = gi < ng ? L4[gi * 4 + i]
                                                         : make_float4(-INFINITY, -INFINITY,
                                                                       -INFINITY, -INFINITY);
                                nL[gi][4 * i] = q.x;
                                nL[gi][4 * i + 1] = q.y;
                                nL[gi][4 * i + 2] = q.z;
                                nL[gi][4 * i + 3] = q.w;
                            }
                        task_ok = sm.sLbad[lb] == 0;
                        __syncwarp();
                        if (lane == 0)
                            ptx::mbar_arrive(&sm.bar[kBarLseEmpty + lb]);
                    } else {
#pragma unroll
                        for (int gi = 0; gi < kMaxGroups; ++gi)
#pragma unroll
                            for (int c = 0; c < 16; ++c)
                                nL[gi][c] = -INFINITY;
                    }
                    if (ew == 0 && lane == 0)
                        trace_at<kTr>(a, kTrTimeline, 2048 + 2 * (p2c - 1) + 1);
                    task_ok = task_ok && !dead;
                    // This unit's score row: plain stores, or fixed-point adds when it is
                    // split into row blocks.
                    const int64_t row_at = (int64_t)(kFx ? T.u / a.nrb : T.u) * g.P;
                    float *const raw_row = kFx ? nullptr : a.raw + row_at;
                    unsigned long long *const fx_row = kFx ? a.raw_fx + row_at : nullptr;
                    cy_p2s += tclock<kTr>() - c_start;
                    for (int tile = 0; tile < T.ntiles; ++tile, ++tc) {
                        const int ab = tc % kAccBufs;
                        const uint32_t aph = (uint32_t)((tc / kAccBufs) & 1);
                        const int tile0 = T.k_lo + tile * kTile;
                        const int key = tile0 + kl;
                        float2 acc = make_float2(0.f, 0.f);
                        if (acquire_acc(ab, aph)) {
                            const uint32_t tbase =
                                tmem_base + (uint32_t)(ab * a.acc_stride + col_base) + lane_off;
                            const long long c0 = tclock<kTr>();
                            auto f2 = [&](int gi, const float(&v)[16]) {
#pragma unroll
                                for (int gj = 0; gj < kMaxGroups; ++gj)
                                    if (gj == gi)
                                        col_add(acc, v, nL[gj], s2);
                            };
                            for_groups(tbase, ng, f2);
                            cy_math2 += tclock<kTr>() - c0;
                        }
                        // The three warps of this lane quarter (one per warpgroup) leave their
                        // partial sums in shared memory; whichever comes last adds them in
                        // warpgroup order and stores the key's score.  Nobody waits: a slot is
                        // rewritten only after accumulator ab is refilled, which needs every
                        // warp's release below, the last warp's after its reads.
                        const long long cx = tclock<kTr>();
                        if constexpr (kFx) {
                            // Row blocks add into the unit's score row in integers (2^-40
                            // units), so every warpgroup adds its own partial sum: the order of
                            // the additions does not matter and no warp waits for another.
                            // The scaling by 2^40 is exact in fp32, so this is a rounding of
                            // the exact product.
                            if (task_ok && key < T.k_hi)
                                atomicAdd(fx_row + key, (unsigned long long)__float2ll_rn(
                                                            (acc.x + acc.y) * 0x1p40f));
                            cy_xch += tclock<kTr>() - cx;
                            release_acc(ab, 1u);
                            continue;
                        }
                        float *xs = sm.xch + ab * kEpiWG * kTile;
                        xs[wg * kTile + kl] = acc.x + acc.y;
                        __syncwarp();
                        // The arrival releases this warp's sums; a warp that finds the phase
                        // complete right after its own arrival has all three (two warps may
                        // both find it so: they store the same value).
                        int last = 0;
                        if (lane == 0) {
                            uint64_t *xb = &sm.bar[kBarXch + ab * 4 + quarter];
                            last = ptx::mbar_test_token(xb, ptx::mbar_arrive_token(xb)) ? 1 : 0;
                        }
                        last = __shfl_sync(0xffffffffu, last, 0);
                        __syncwarp();  // lane 0's acquire orders the other lanes' reads
                        if (last) {
                            float total = xs[kl];
#pragma unroll
                            for (int w = 1; w < kEpiWG; ++w)
                                total += xs[w * kTile + kl];
                            if (task_ok && key < T.k_hi)
                                raw_row[key] = total;
                        }
                        cy_xch += tclock<kTr>() - cx;
                        release_acc(ab, 1u);
                    }
                }
            }
        if (ew == 0 && lane == 0) {
            trace_put<kTr>(a, kTrEpiWaitAcc, cy_wa);
            trace_put<kTr>(a, kTrEpiP1End, cy_p1e);
            trace_put<kTr>(a, kTrEpiP2Start, cy_p2s);
            trace_put<kTr>(a, kTrEpiMath, cy_math);
            trace_put<kTr>(a, kTrEpiMathP2, cy_math2);
            trace_put<kTr>(a, kTrEpiXch, cy_xch);
            trace_put<kTr>(a, kTrEpiRelease, cy_rel);
            trace_put<kTr>(a, kTrEpiTotal, tclock<kTr>() - cy0);
        }
    }

    // ---- teardown ------------------------------------------------------------------------
    __syncthreads();
    if (warp == 0 && lane == 0) {
        // Copies still in flight (only after an abort) land before the CTA leaves.
        for (int i = 0; i < a.kstages; ++i)
            if (flag[kFlagKArm + i] >= 0)
                drain_bar(&sm.bar[kBarKFull + i], (uint32_t)flag[kFlagKArm + i], 1000000000ull);
        for (int i = 0; i < 2; ++i)
            if (flag[kFlagQArm + i] >= 0)
                drain_bar(&sm.bar[kBarQFull + i], (uint32_t)flag[kFlagQArm + i], 1000000000ull);
        if (flag[kFlagSArm] >= 0)
            drain_bar(&sm.bar[kBarStage], (uint32_t)flag[kFlagSArm], 1000000000ull);
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    if (warp == 1)
        ptx::tmem_dealloc(tmem_base, kTmemCols);
}

unsigned long long *g_trace = nullptr;
int g_trace_cta = 0;
unsigned long long g_wait_limit_ns = tc::kDefaultWaitLimitNs;
int g_count_extra = 0;

}  // namespace

namespace tc {

using Encode = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                            const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                            const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                            CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

Encode encode_fn_impl()
{
    static Encode fn = nullptr;
    static bool tried = false;
    if (!tried) {
        tried = true;
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<Encode>(p);
    }
    return fn;
}

bool encode_5d(CUtensorMap *map, const TensorDesc &t, int L, int b, int heads, int rows, int d,
               int box_rows, int box_heads)
{
    Encode fn = encode_fn_impl();
    if (!fn)
        return false;
    const cuuint64_t dims[5] = {(cuuint64_t)d, (cuuint64_t)rows, (cuuint64_t)heads, (cuuint64_t)b,
                                (cuuint64_t)L};
    const cuuint64_t strides[4] = {(cuuint64_t)t.s_pos * 2, (cuuint64_t)t.s_head * 2,
                                   (cuuint64_t)t.s_batch * 2, (cuuint64_t)t.s_layer * 2};
    const cuuint32_t box[5] = {64, (cuuint32_t)box_rows, (cuuint32_t)box_heads, 1, 1};
    const cuuint32_t estr[5] = {1, 1, 1, 1, 1};
    for (int i = 0; i < 4; ++i)
        if (strides[i] == 0 || strides[i] % 16 != 0)
            return false;
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<__nv_bfloat16 *>(t.data), dims,
              strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool have_tensor_maps()
{
    return encode_fn_impl() != nullptr;
}

bool encode_k_map(CUtensorMap *map, const TensorDesc &t, int L, int b, int Hkv, int n, int d)
{
    if (!t.bt)
        return encode_5d(map, t, L, b, Hkv, n, d, 128, 1);
    Encode fn = encode_fn_impl();
    if (!fn)
        return false;
    // [L][page][slot][head][d]: boxes of one head, min(page_size, 128) slots.  A pool of one
    // layer may carry any layer stride; give the map a nonzero one.
    const int64_t s_layer = t.s_layer != 0 ? t.s_layer : t.s_page * t.num_pages;
    const cuuint64_t dims[5] = {(cuuint64_t)d, (cuuint64_t)Hkv, (cuuint64_t)t.page_size,
                                (cuuint64_t)t.num_pages, (cuuint64_t)L};
    const cuuint64_t strides[4] = {(cuuint64_t)t.s_head * 2, (cuuint64_t)t.s_pos * 2,
                                   (cuuint64_t)t.s_page * 2, (cuuint64_t)s_layer * 2};
    const cuuint32_t box[5] = {64, 1, (cuuint32_t)(t.page_size < 128 ? t.page_size : 128), 1, 1};
    const cuuint32_t estr[5] = {1, 1, 1, 1, 1};
    for (int i = 0; i < 4; ++i)
        if (strides[i] == 0 || strides[i] % 16 != 0)
            return false;
    (void)b;
    (void)n;
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<__nv_bfloat16 *>(t.data), dims,
              strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Slots of consecutive pages adjacent in memory: page stride = page_size * slot stride.
static bool slots_run_on(const TensorDesc &t)
{
    return t.bt && t.s_page == (int64_t)t.page_size * t.s_pos;
}

bool encode_k_merged_map(CUtensorMap *map, const TensorDesc &t, int L, int Hkv, int d)
{
    Encode fn = encode_fn_impl();
    if (!fn || !slots_run_on(t))
        return false;
    // [L][slot over all pages][head][d], plus a unit outer dimension.
    const int64_t slots = (int64_t)t.num_pages * t.page_size;
    const int64_t s_layer = t.s_layer != 0 ? t.s_layer : t.s_page * t.num_pages;
    const cuuint64_t dims[5] = {(cuuint64_t)d, (cuuint64_t)Hkv, (cuuint64_t)slots, (cuuint64_t)L, 1};
    const cuuint64_t strides[4] = {(cuuint64_t)t.s_head * 2, (cuuint64_t)t.s_pos * 2,
                                   (cuuint64_t)s_layer * 2, (cuuint64_t)s_layer * L * 2};
    const cuuint32_t box[5] = {64, 1, 128, 1, 1};
    const cuuint32_t estr[5] = {1, 1, 1, 1, 1};
    for (int i = 0; i < 4; ++i)
        if (strides[i] == 0 || strides[i] % 16 != 0)
            return false;
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<__nv_bfloat16 *>(t.data), dims,
              strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

KPaging k_paging(const TensorDesc &t, int n)
{
    KPaging p;
    p.bt = t.bt;
    p.page_size = t.page_size;
    p.pps = t.pps;
    p.num_pages = t.num_pages;
    p.n = n;
    p.merged = 0;
    p.ps_shift = 0;
    while (p.ps_shift < 30 && (1 << p.ps_shift) < t.page_size)
        ++p.ps_shift;
    return p;
}

}  // namespace tc

void tc_set_trace(unsigned long long *buffer, int cta)
{
    g_trace = buffer;
    g_trace_cta = cta;
}

void tc_set_waits(unsigned long long limit_ns, int count_extra)
{
    g_wait_limit_ns = limit_ns ? limit_ns : tc::kDefaultWaitLimitNs;
    g_count_extra = count_extra;
}

unsigned long long tc_wait_limit_ns()
{
    return g_wait_limit_ns;
}

// Query heads per sub-unit: the most heads of a KV group (a divisor of G) whose stacked rows
// still fit one accumulator and the lse stager.
int tc_gsub(const Geometry &g)
{
    const int cap = kEpiWG * kMaxGroups * 16 < 32 * kRowsPerLane ? kEpiWG * kMaxGroups * 16
                                                                 : 32 * kRowsPerLane;
    for (int gs = g.G; gs >= 1; --gs)
        if (g.G % gs == 0 && gs * g.m <= cap)
            return gs;
    return 0;
}

bool tc_supported(const Geometry &g)
{
    // The observation rows must lie in the protected tail (t >= m), so that phase 2 needs no
    // causal mask; the caller's rare t < m goes to the warp-level kernels.
    if (g.variant != DGE_VARIANT_SCORED || (g.d != 64 && g.d != 128) || g.m > 256 || g.G > 256 ||
        g.tail < g.m)
        return false;
    const int gs = tc_gsub(g);
    if (gs == 0 || (size_t)((gs * g.m + 3) & ~3) * 4 > (size_t)kStageBytes)
        return false;
    int dev = 0, major = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess)
        return false;
    return major == 10 && tc::have_tensor_maps();
}

TcPlan tc_plan(const Geometry &g)
{
    TcPlan p;
    p.gsub = tc_gsub(g);
    p.nrb = p.gsub > 0 ? g.G / p.gsub : 1;
    p.rows = p.gsub * g.m;
    p.r_pad = (p.rows + 15) & ~15;
    p.r4 = (p.rows + 3) & ~3;
    p.nslab = g.d / 64;
    // Key chunk (one task).  The phase-1 data read between an item's two phases is about
    // (lag + nchunks) chunks, so only chunks of about 8 tiles keep the phase-2 re-read in L2,
    // and those pay the per-task hand-offs (the row-sum reduction, the lse staging, a
    // query-block load) too often: at 32K keys, 8 tiles 3.09 ms, 16 tiles 2.71, 48 tiles 2.56,
    // 128 tiles 2.51 (K read twice at the copy rate).  Whole units take chunks of at most
    // kChunkTiles tiles, but at least kMinItems items in all when the units are few and short
    // (8K keys, 256 units: two chunks of 32 tiles, 0.189 ms against 0.203 for whole units),
    // never below 16 tiles; a unit is split into chunks of equal length (within a tile).
    const int unit_tiles = (g.n + kTile - 1) / kTile;
    int nch = (unit_tiles + kChunkTiles - 1) / kChunkTiles;
    const int64_t want = (kMinItems + g.U - 1) / (g.U > 0 ? g.U : 1);
    const int cap = unit_tiles / 16 > 1 ? unit_tiles / 16 : 1;
    if (want > nch)
        nch = want < cap ? (int)want : (cap > nch ? cap : nch);
    int tiles = nch > 0 && unit_tiles > 0 ? (unit_tiles + nch - 1) / nch : 1;
    // Row blocks (R > 144) make the kernel bound by the tensor pipe and the epilogue, not by
    // DRAM, so the L2 fit does not matter and the longest chunk wins: at 128K keys and four
    // row blocks (70B shape), quarter-unit chunks (256 tiles) took 25.4 ms against 26.7 ms
    // for 16-tile ones.
    const int quarter = (unit_tiles / 4) / 8 * 8;
    if (p.nrb > 1)
        tiles = quarter < 8 ? (unit_tiles < 8 ? unit_tiles : 8) : quarter;
    p.chunk_keys = tiles * kTile;
    p.nchunks = (unit_tiles + tiles - 1) / tiles;
    // Chunks whose keys start below n - m carry phase-1 keys (the first p1_chunks ones).
    const int first_obs = g.n - g.m;
    p.p1_chunks = 0;
    for (int c = 0; c < p.nchunks; ++c)
        if ((int)((int64_t)c * unit_tiles / p.nchunks) * kTile < first_obs)
            p.p1_chunks = c + 1;
    p.nparts = p.nchunks + 1;

    p.kstages = kMaxKStages;
    while (p.kstages > 2 && smem_bytes(p.r_pad, p.nslab, p.kstages) > 232448)
        --p.kstages;
    p.smem = smem_bytes(p.r_pad, p.nslab, p.kstages);
    // At least half of the SM's shared memory: one CTA per SM, so a CTA's TMEM allocation
    // (all 512 columns) never waits for another CTA of this kernel.
    if (p.smem < 120 * 1024)
        p.smem = 120 * 1024;
    return p;
}

cudaError_t launch_score_tc(const TensorDesc &K, const TensorDesc &Q, const Geometry &g,
                            const TcPlan &plan, const TcBuffers &buf, cudaStream_t stream,
                            bool *encoded)
{
    CUtensorMap tmK, tmQ, tmKm;
    memset(&tmKm, 0, sizeof tmKm);
    const bool merged = K.bt && tc::encode_k_merged_map(&tmKm, K, g.L, g.Hkv, g.d);
    *encoded = tc::encode_k_map(&tmK, K, g.L, g.b, g.Hkv, g.n, g.d) &&
               tc::encode_5d(&tmQ, Q, g.L, g.b, g.Hq, g.m, g.d, g.m, plan.gsub);
    if (!*encoded)
        return cudaSuccess;
    int dev = 0, sms = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err == cudaSuccess)
        err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (err != cudaSuccess)
        return err;

    TcArgs a;
    a.g = g;
    a.kp = tc::k_paging(K, g.n);
    a.kp.merged = merged ? 1 : 0;
    a.rows = plan.rows;
    a.nrb = plan.nrb;
    a.gsub = plan.gsub;
    a.r_pad = plan.r_pad;
    a.r4 = plan.r4;
    a.acc_stride = (plan.r_pad + 31) & ~31;
    a.nslab = plan.nslab;
    a.kstages = plan.kstages;
    a.unit_tiles = (g.n + kTile - 1) / kTile;
    a.nchunks = plan.nchunks;
    a.p1_chunks = plan.p1_chunks;
    a.nparts = plan.nparts;
    a.lse_in = buf.lse_in;
    if (a.lse_in) {
        // One pass, nothing to keep in L2: tasks of up to 32 tiles.
        a.nchunks = (a.unit_tiles + 31) / 32;
    }
    a.items = g.U * a.nrb * a.nchunks;
    const int NG = plan.r_pad / 16;
    for (int w = 0, base = 0; w < kEpiWG; ++w) {
        a.ng[w] = NG / kEpiWG + (w < NG % kEpiWG ? 1 : 0);
        a.gbase[w] = base;
        base += a.ng[w];
    }
    const int64_t grid = a.items < sms ? a.items : sms;
    if (a.lse_in) {
        a.lag = 0;
        a.total = a.items;
    } else {
        // Phase 2 of an item is claimed `lag` items after its phase 1: the whole unit's
        // chunks (nchunks - 1) plus about one and a half rounds of the grid, so that the
        // phase-1 tasks it needs, claimed that much earlier, have finished (each CTA holds at
        // most about two tasks between claiming and finishing them) while the chunk is still
        // in L2.
        const int64_t lag = (int64_t)kLagGridX10 * grid / 10 + a.nchunks - 1;
        a.lag = lag < a.items ? lag : a.items;
        a.total = 2 * a.items;
    }
    a.claim = buf.claim;
    a.part = buf.part;
    a.lse2 = buf.lse2;
    a.raw = buf.raw;
    a.raw_fx = plan.nrb > 1 ? buf.raw_fx : nullptr;
    a.count = buf.count;
    a.ready = buf.ready;
    a.list = buf.list;
    a.status = buf.status;
    a.timeout_ns = g_wait_limit_ns;
    a.count_extra = a.lse_in ? 0 : g_count_extra;
    a.trace = g_trace;
    a.trace_cta = g_trace_cta;

    // The traced build covers whole, contiguous units only; row blocks and paged caches run
    // untraced.
    void (*kernel)(const CUtensorMap, const CUtensorMap, const CUtensorMap, const TcArgs) =
        K.bt ? (plan.nrb > 1 ? score_tc_kernel<false, true, true>
                             : score_tc_kernel<false, false, true>)
             : (plan.nrb > 1 ? score_tc_kernel<false, true, false>
                             : (a.trace ? score_tc_kernel<true, false, false>
                                        : score_tc_kernel<false, false, false>));
    err = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               (int)plan.smem);
    if (err != cudaSuccess)
        return err;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = plan.smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, tmK, tmQ, tmKm, a);
}

}  // namespace dge
