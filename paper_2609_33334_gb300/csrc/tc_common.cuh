// tc_common.cuh -- device helpers shared by the tcgen05 kernels (score_tc.cu, h2o_tc.cu):
// bounded mbarrier waits and the warp transpose-and-add used to reduce per-lane row sums.
#pragma once

#include <cuda.h>

#include "common.cuh"
#include "tc_ptx.cuh"

namespace dge {
namespace tc {

// Slot 0 of a kernel's shared flag block: set once the CTA has aborted.
constexpr int kFlagAbort = 0;

// Bound of every device-side wait of the tcgen05 kernels unless a test shortens it.
constexpr unsigned long long kDefaultWaitLimitNs = 4000000000ull;

// Bounded wait on an mbarrier phase.  Returns false when the CTA has aborted or the wait
// outlived `timeout_ns` (then it aborts the CTA and records DGE_ERR_DEVICE_TIMEOUT).
__device__ inline bool wait_bar(uint64_t *bar, uint32_t parity, volatile int *flag,
                                unsigned long long timeout_ns, uint32_t *status)
{
    uint64_t t0 = 0;
    uint32_t spins = 0;
    while (!ptx::mbar_try_wait(bar, parity)) {
        if ((++spins & 63) == 0) {
            if (flag[kFlagAbort])
                return false;
            const uint64_t now = ptx::globaltimer();
            if (t0 == 0) {
                t0 = now;
            } else if (now - t0 > timeout_ns) {
                flag[kFlagAbort] = 1;
                set_status(status, DGE_ERR_DEVICE_TIMEOUT);
                return false;
            }
        }
    }
    return true;
}

// Bounded wait that ignores the abort flag (teardown drains).
__device__ inline void drain_bar(uint64_t *bar, uint32_t parity, unsigned long long limit_ns)
{
    const uint64_t t0 = ptx::globaltimer();
    while (!ptx::mbar_try_wait(bar, parity))
        if (ptx::globaltimer() - t0 > limit_ns)
            return;
}

// In-place sums over the 32 lanes of a warp, for 32 per-lane values held as two
// 16-value groups a (columns 0..15) and b (16..31): afterwards a[0] of lane l holds
// the total of column l.  Each step halves the values a lane keeps: the lane whose
// bit o is set keeps the upper half, its partner the lower half.
__device__ __forceinline__ void transpose_sum32(float (&a)[16], float (&b)[16], int lane)
{
    const bool up16 = (lane & 16) != 0;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
        const float send = up16 ? a[i] : b[i];
        const float keep = up16 ? b[i] : a[i];
        a[i] = keep + __shfl_xor_sync(0xffffffffu, send, 16);
    }
#pragma unroll
    for (int o = 8; o >= 1; o >>= 1) {
        const bool upper = (lane & o) != 0;
#pragma unroll
        for (int i = 0; i < o; ++i) {
            const float send = upper ? a[i] : a[i + o];
            const float keep = upper ? a[i + o] : a[i];
            a[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
        }
    }
}

// Same for one 16-value group: lanes l and l ^ 16 both end with column l & 15 in a[0].
__device__ __forceinline__ void transpose_sum16(float (&a)[16], int lane)
{
#pragma unroll
    for (int i = 0; i < 16; ++i)
        a[i] += __shfl_xor_sync(0xffffffffu, a[i], 16);
#pragma unroll
    for (int o = 8; o >= 1; o >>= 1) {
        const bool upper = (lane & o) != 0;
#pragma unroll
        for (int i = 0; i < o; ++i) {
            const float send = upper ? a[i] : a[i + o];
            const float keep = upper ? a[i + o] : a[i];
            a[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
        }
    }
}

// K of a paged cache as the tcgen05 producers see it (bt == nullptr: contiguous).
struct KPaging {
    const int32_t *bt;   // block table [b][pps]
    int page_size, pps, num_pages, n;
    int ps_shift;        // log2(page_size) for pages of 16, 32 or 64 slots
    // The pool's slots run on across pages (page stride = page_size * slot stride): a tile
    // whose pages are consecutive in the pool is one box of the merged map.
    int merged;
};

// Largest number of pages a 128-key tile spans (page sizes 16, 32, 64 or multiples of 128).
constexpr int kMaxTilePages = 8;
// Key tiles whose page ids are fetched together (kPageWindowTiles * kMaxTilePages ints of
// shared memory).
constexpr int kPageWindowTiles = 32;
constexpr int kPageWindow = kPageWindowTiles * kMaxTilePages;

// The page ids of positions [k0, min(k0 + tiles * 128, n)) of sequence bb (tiles <=
// kPageWindowTiles) into shared memory (`buf`, 16-byte aligned, kPageWindow + 4 ints) with
// asynchronous copies -- 16 bytes at a time where the table allows, 4 at its unaligned edges,
// never past the entries needed.  fetch_pages_issue only issues them (fetch_pages_wait waits
// for them); fetch_pages does both (one round trip a window).  Returns `ids`, with ids[i] the
// id of page k0 / page_size + i.  Invalid ids are clamped when read.
__device__ __forceinline__ const int *fetch_pages_issue(int *buf, const KPaging &pg, int bb,
                                                        int k0, int tiles = kPageWindowTiles)
{
    const int end = min(k0 + tiles * 128, pg.n);
    const int p0 = k0 / pg.page_size;
    const int count = (end - 1) / pg.page_size - p0 + 1;
    const int32_t *src = pg.bt + (int64_t)bb * pg.pps + p0;
    // The same offset within 16 bytes on both sides, so the middle moves in 16-byte pieces.
    int *ids = buf + (int)(((uintptr_t)src >> 2) & 3);
    int i = 0;
    for (; i < count && (((uintptr_t)(src + i)) & 15); ++i)
        asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(ptx::smem_addr(ids + i)),
                     "l"(src + i)
                     : "memory");
    for (; i + 4 <= count; i += 4)
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(ptx::smem_addr(ids + i)),
                     "l"(src + i)
                     : "memory");
    for (; i < count; ++i)
        asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(ptx::smem_addr(ids + i)),
                     "l"(src + i)
                     : "memory");
    return ids;
}

// fetch_pages_issue spread over a warp (every lane calls it): lane i copies entries i, i + 32,
// ... of the 16-byte-aligned middle (16 bytes each) and at most one 4-byte edge entry, so a
// window of 16-slot pages (256 ids) costs two copies a lane instead of 64 on one thread.
// Same destination layout as fetch_pages_issue; each lane then commits and waits for its own.
__device__ __forceinline__ void fetch_pages_issue_warp(int *buf, const KPaging &pg, int bb, int k0,
                                                       int tiles, int lane)
{
    const int end = min(k0 + tiles * 128, pg.n);
    const int p0 = k0 / pg.page_size;
    const int count = (end - 1) / pg.page_size - p0 + 1;
    const int32_t *src = pg.bt + (int64_t)bb * pg.pps + p0;
    const int off = (int)(((uintptr_t)src >> 2) & 3);
    int *ids = buf + off;
    const int head = min(count, (4 - off) & 3);            // entries before a 16-byte boundary
    const int nvec = (count - head) >> 2;
    const int done = head + 4 * nvec;
    if (lane < head)
        asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(ptx::smem_addr(ids + lane)),
                     "l"(src + lane)
                     : "memory");
    for (int v = lane; v < nvec; v += 32)
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(
                         ptx::smem_addr(ids + head + 4 * v)),
                     "l"(src + head + 4 * v)
                     : "memory");
    if (lane < count - done)
        asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(
                         ptx::smem_addr(ids + done + lane)),
                     "l"(src + done + lane)
                     : "memory");
}

__device__ __forceinline__ void fetch_pages_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }

// Waits for this thread's page-id copies except the newest `pending` groups (0 or 1).
template <int pending>
__device__ __forceinline__ void fetch_pages_wait_group()
{
    asm volatile("cp.async.wait_group %0;" ::"n"(pending) : "memory");
}

// For the window of kPageWindowTiles (= 32) tiles from key w0 (ids from fetch_pages): lane t
// returns the first page of tile t when that tile's pages are consecutive and the merged map
// can load it as one box a slab, else -1.  Every lane of the warp calls it once a window, so
// the per-tile path reads one register (a shuffle) instead of the tile's page ids.
__device__ __forceinline__ int tile_runs(const KPaging &pg, const int *ids, int w0, int tiles,
                                         int lane)
{
    static_assert(kPageWindowTiles == 32, "one lane per tile of the window");
    if (!pg.merged || pg.page_size >= 128 || lane >= tiles)
        return -1;
    const int npg = 128 >> pg.ps_shift;
    const int k0 = w0 + lane * 128;
    const int valid = (pg.n - k0 + pg.page_size - 1) >> pg.ps_shift;
    if (valid < npg)
        return -1;
    const int first = ids[lane * npg];
    bool run = (unsigned)first <= (unsigned)(pg.num_pages - npg);
    for (int j = 1; j < npg; ++j)
        run = run && ids[lane * npg + j] == first + j;
    return run ? first : -1;
}

// Where fetch_pages(buf, pg, bb, k0, ...) puts the page ids (any thread can compute it).
__device__ __forceinline__ const int *page_ids_at(int *buf, const KPaging &pg, int bb, int k0)
{
    const int32_t *src = pg.bt + (int64_t)bb * pg.pps + k0 / pg.page_size;
    return buf + (int)(((uintptr_t)src >> 2) & 3);
}

// Waits for every page-id copy this thread has issued.
__device__ __forceinline__ void fetch_pages_wait()
{
    asm volatile("cp.async.wait_all;" ::: "memory");
}

__device__ __forceinline__ const int *fetch_pages(int *buf, const KPaging &pg, int bb, int k0,
                                                  int tiles = kPageWindowTiles)
{
    const int *ids = fetch_pages_issue(buf, pg, bb, k0, tiles);
    fetch_pages_wait();
    return ids;
}

// One 128-key tile of K (nslab slabs of 64 columns, slab_bytes apart) into shared memory with
// TMA, completing on `bar`: one box per slab from a contiguous cache (map over
// [L][b][Hkv][n][d]), or one box of min(page_size, 128) slots per page from a paged one (map
// over [L][page][slot][Hkv][d]; `ids` from fetch_pages for the window starting at `w0`).
// Positions past the cache read page 0, whose rows the callers mask.
template <bool kPaged>
__device__ __forceinline__ void load_k_tile(uint8_t *dst, uint32_t slab_bytes, int nslab,
                                            const CUtensorMap *map, const CUtensorMap *merged,
                                            uint64_t *bar, int k0, int l, int bb, int h,
                                            const KPaging &pg, const int *ids, int w0,
                                            uint64_t policy)
{
    if constexpr (!kPaged) {
        for (int s = 0; s < nslab; ++s)
            ptx::tma_load_5d_hint(dst + s * slab_bytes, map, bar, s * 64, k0, h, bb, l, policy);
    } else if (pg.page_size >= 128) {
        // One page holds the whole tile.
        int page = 0, slot = 0;
        if (k0 < pg.n) {
            const int pi = k0 / pg.page_size;
            const int pid = ids[pi - w0 / pg.page_size];
            page = (unsigned)pid < (unsigned)pg.num_pages ? pid : 0;
            slot = k0 - pi * pg.page_size;
        }
        for (int s = 0; s < nslab; ++s)
            ptx::tma_load_5d_hint(dst + s * slab_bytes, map, bar, s * 64, h, slot, page, l,
                                  policy);
    } else {
        // 2..8 pages of 16, 32 or 64 slots; the tile and the window start on page boundaries.
        const int npg = 128 >> pg.ps_shift;
        const int i0 = (k0 - w0) >> pg.ps_shift;                            // first page in ids
        const int valid = (pg.n - k0 + pg.page_size - 1) >> pg.ps_shift;    // pages before n
        if (pg.merged && valid >= npg) {
            // Pages handed out in order: the tile's pages follow each other in the pool.
            const int first = ids[i0];
            bool run = (unsigned)first <= (unsigned)(pg.num_pages - npg);
            for (int j = 1; j < npg; ++j)
                run = run && ids[i0 + j] == first + j;
            if (run) {
                for (int s = 0; s < nslab; ++s)
                    ptx::tma_load_5d_hint(dst + s * slab_bytes, merged, bar, s * 64, h,
                                          first << pg.ps_shift, l, 0, policy);
                return;
            }
        }
        for (int j = 0; j < npg; ++j) {
            int page = 0;
            if (j < valid) {
                const int pid = ids[i0 + j];
                page = (unsigned)pid < (unsigned)pg.num_pages ? pid : 0;
            }
            for (int s = 0; s < nslab; ++s)
                ptx::tma_load_5d_hint(dst + s * slab_bytes + (j << pg.ps_shift) * 128, map, bar,
                                      s * 64, h, 0, page, l, policy);
        }
    }
}

// load_k_tile issued by a whole warp, one box per lane: box i of a tile is slab i % nslab of
// page i / nslab (nslab boxes for a contiguous cache, a page of 128 slots or more, or a run
// of consecutive pages).  The caller arms `bar` for the whole tile before any lane issues.
// Pages below 128 slots: run_first >= 0 says the tile's pages are consecutive from page
// run_first (the merged map applies; the caller decides, see tile_runs), else one box per
// page and slab.
template <bool kPaged>
__device__ __forceinline__ void load_k_tile_warp(uint8_t *dst, uint32_t slab_bytes, int nslab,
                                                 const CUtensorMap *map,
                                                 const CUtensorMap *merged, uint64_t *bar,
                                                 int k0, int l, int bb, int h, const KPaging &pg,
                                                 const int *ids, int w0, uint64_t policy,
                                                 int lane, int run_first = -1)
{
    if constexpr (!kPaged) {
        if (lane < nslab)
            ptx::tma_load_5d_hint(dst + lane * slab_bytes, map, bar, lane * 64, k0, h, bb, l,
                                  policy);
    } else if (pg.page_size >= 128) {
        int page = 0, slot = 0;
        if (k0 < pg.n) {
            // Power-of-two page sizes by shifts (off the producer's path), others by division.
            const bool pow2 = (1 << pg.ps_shift) == pg.page_size;
            const int pi = pow2 ? k0 >> pg.ps_shift : k0 / pg.page_size;
            const int pw = pow2 ? w0 >> pg.ps_shift : w0 / pg.page_size;
            const int pid = ids[pi - pw];
            page = (unsigned)pid < (unsigned)pg.num_pages ? pid : 0;
            slot = k0 - pi * pg.page_size;
        }
        if (lane < nslab)
            ptx::tma_load_5d_hint(dst + lane * slab_bytes, map, bar, lane * 64, h, slot, page, l,
                                  policy);
    } else {
        const int npg = 128 >> pg.ps_shift;
        const int i0 = (k0 - w0) >> pg.ps_shift;
        const int valid = (pg.n - k0 + pg.page_size - 1) >> pg.ps_shift;
        if (run_first >= 0) {   // the tile's pages are consecutive: one box a slab
            if (lane < nslab)
                ptx::tma_load_5d_hint(dst + lane * slab_bytes, merged, bar, lane * 64, h,
                                      run_first << pg.ps_shift, l, 0, policy);
            return;
        }
        // nslab is 1 or 2 (d = 64 or 128): a shift, not a division, on the producer's path.
        const int j = lane >> (nslab - 1), s = lane & (nslab - 1);
        if (j < npg) {
            int page = 0;
            if (j < valid) {
                const int pid = ids[i0 + j];
                page = (unsigned)pid < (unsigned)pg.num_pages ? pid : 0;
            }
            ptx::tma_load_5d_hint(dst + s * slab_bytes + (j << pg.ps_shift) * 128, map, bar,
                                  s * 64, h, 0, page, l, policy);
        }
    }
}

// Host: a 5-D TMA map over [L][b][heads][rows][d] (bf16, 128-byte swizzle) with box
// {64, box_rows, box_heads, 1, 1}; false when the driver entry point is missing or the strides
// are not 16-byte multiples.
bool encode_5d(CUtensorMap *map, const TensorDesc &t, int L, int b, int heads, int rows, int d,
               int box_rows, int box_heads);
bool have_tensor_maps();
// Host: the K maps of load_k_tile -- contiguous, or over a paged cache's pools (t.bt set);
// `merged` (paged caches) views the pool's slots as one run per layer, when the layout allows
// it (KPaging::merged, from k_paging).
bool encode_k_map(CUtensorMap *map, const TensorDesc &t, int L, int b, int Hkv, int n, int d);
bool encode_k_merged_map(CUtensorMap *map, const TensorDesc &t, int L, int Hkv, int d);
KPaging k_paging(const TensorDesc &t, int n);

}  // namespace tc
}  // namespace dge
