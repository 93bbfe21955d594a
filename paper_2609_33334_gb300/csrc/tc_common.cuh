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
};

// Largest number of pages a 128-key tile spans (page sizes 16, 32, 64 or multiples of 128).
constexpr int kMaxTilePages = 8;
// Key tiles whose page ids are fetched together (kPageWindowTiles * kMaxTilePages ints of
// shared memory).
constexpr int kPageWindowTiles = 32;
constexpr int kPageWindow = kPageWindowTiles * kMaxTilePages;

// The page ids of positions [k0, min(k0 + tiles * 128, n)) of sequence bb (tiles <=
// kPageWindowTiles) into shared memory with 4-byte asynchronous copies, waited for before
// returning (one round trip a window); ids[i] belongs to page k0 / page_size + i.  Invalid
// ids are clamped when read.
__device__ __forceinline__ void fetch_pages(int *ids, const KPaging &pg, int bb, int k0,
                                            int tiles = kPageWindowTiles)
{
    const int end = min(k0 + tiles * 128, pg.n);
    const int p0 = k0 / pg.page_size, p1 = (end - 1) / pg.page_size;
    const int32_t *src = pg.bt + (int64_t)bb * pg.pps;
    for (int p = p0; p <= p1; ++p)
        asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(ptx::smem_addr(ids + (p - p0))),
                     "l"(src + p)
                     : "memory");
    asm volatile("cp.async.wait_all;" ::: "memory");
}

// One 128-key tile of K (nslab slabs of 64 columns, slab_bytes apart) into shared memory with
// TMA, completing on `bar`: one box per slab from a contiguous cache (map over
// [L][b][Hkv][n][d]), or one box of min(page_size, 128) slots per page from a paged one (map
// over [L][page][slot][Hkv][d]; `ids` from fetch_pages for the window starting at `w0`).
// Positions past the cache read page 0, whose rows the callers mask.
template <bool kPaged>
__device__ __forceinline__ void load_k_tile(uint8_t *dst, uint32_t slab_bytes, int nslab,
                                            const CUtensorMap *map, uint64_t *bar, int k0, int l,
                                            int bb, int h, const KPaging &pg, const int *ids,
                                            int w0, uint64_t policy)
{
    if constexpr (!kPaged) {
        for (int s = 0; s < nslab; ++s)
            ptx::tma_load_5d_hint(dst + s * slab_bytes, map, bar, s * 64, k0, h, bb, l, policy);
    } else {
        const int rows = pg.page_size < 128 ? pg.page_size : 128;
        const int npg = 128 / rows;
        const int pbase = w0 / pg.page_size;
        for (int j = 0; j < npg; ++j) {
            const int pos = k0 + j * rows;
            int page = 0, slot = 0;
            if (pos < pg.n) {
                const int pid = ids[pos / pg.page_size - pbase];
                page = (pid >= 0 && pid < pg.num_pages) ? pid : 0;
                slot = pos % pg.page_size;
            }
            for (int s = 0; s < nslab; ++s)
                ptx::tma_load_5d_hint(dst + s * slab_bytes + j * rows * 128, map, bar, s * 64, h,
                                      slot, page, l, policy);
        }
    }
}

// Host: a 5-D TMA map over [L][b][heads][rows][d] (bf16, 128-byte swizzle) with box
// {64, box_rows, box_heads, 1, 1}; false when the driver entry point is missing or the strides
// are not 16-byte multiples.
bool encode_5d(CUtensorMap *map, const TensorDesc &t, int L, int b, int heads, int rows, int d,
               int box_rows, int box_heads);
bool have_tensor_maps();
// Host: the K map of load_k_tile -- contiguous, or over a paged cache's pools (t.bt set).
bool encode_k_map(CUtensorMap *map, const TensorDesc &t, int L, int b, int Hkv, int n, int d);
KPaging k_paging(const TensorDesc &t, int n);

}  // namespace tc
}  // namespace dge
