// common.cuh -- internal types and device helpers of libdge (not part of the ABI).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "dge.h"

namespace dge {

constexpr int kMaxLayers = 256;
constexpr int kMaxRows = 640;          // stacked observation rows per unit held on chip
constexpr int kMaxSelectBlock = 64;     // largest block of block-granular selection
constexpr int kMaxSelectBlocks = 16384; // blocks per unit it sorts in shared memory
constexpr int kStatusBytes = 256;      // status region at the start of every workspace

// Device status word values (same numbering as the ABI status codes).
constexpr uint32_t kStatusOk = 0;

// Per-layer budgets and the first packed row of each layer.
struct LayerTable {
    int32_t budget[kMaxLayers];
    int64_t row_base[kMaxLayers];
};

// A bf16 tensor [layer][batch][head][pos][d] with element strides, or a paged cache: each
// layer's pool of pages [page][slot][head][d] (s_page, s_pos = between slots, s_head), with
// position p of sequence b in slot p % page_size of page bt[b * pps + p / page_size].
struct TensorDesc {
    const __nv_bfloat16 *data;
    int64_t s_layer, s_batch, s_head, s_pos;
    const int32_t *bt = nullptr;   // block table [b][pps] (paged caches only)
    int page_size = 0, pps = 0, num_pages = 0;
    int64_t s_page = 0;
};

// Everything a kernel needs to know about one eviction problem.
struct Geometry {
    int L, b, Hq, Hkv, G, d;
    int m;          // SCORED observation rows per query head
    int R;          // stacked rows per unit (G*m, or G*n for H2O)
    int n;          // cache length
    int P;          // scored positions [0, P)
    int tail, sinks;
    int variant;
    int pool, pool_kernel;
    int select_block;  // 0: select positions; >= 2: select blocks of this many candidates
    float scale_log2;   // scale * log2(e): logits are kept in base-2 units
    int64_t U;          // units = L*b*Hkv
};

__host__ __device__ inline void unit_coords(const Geometry &g, int64_t u, int &l, int &bb, int &h)
{
    h = (int)(u % g.Hkv);
    const int64_t lb = u / g.Hkv;
    bb = (int)(lb % g.b);
    l = (int)(lb / g.b);
}

// Cache position of stacked row r (head-major stacking of the group's query heads).
__host__ __device__ inline int row_position(const Geometry &g, int r)
{
    if (g.variant == DGE_VARIANT_H2O)
        return r % g.n;
    return g.n - g.m + (r % g.m);
}

// Address of row `row` of query head (h*G + row / rows_per_head) for unit (l, bb, h).
__device__ inline const __nv_bfloat16 *q_row_ptr(const TensorDesc &Q, const Geometry &g, int l,
                                                 int bb, int h, int r, int rows_per_head)
{
    const int qh = h * g.G + r / rows_per_head;
    const int i = r % rows_per_head;
    return Q.data + l * Q.s_layer + bb * Q.s_batch + (int64_t)qh * Q.s_head + (int64_t)i * Q.s_pos;
}

__device__ inline const __nv_bfloat16 *kv_unit_ptr(const TensorDesc &T, int l, int bb, int h)
{
    return T.data + l * T.s_layer + bb * T.s_batch + (int64_t)h * T.s_head;
}

// Page of position `pos` of sequence bb in a paged cache; page 0 for a table entry outside
// the pool (the caller validated the table on the host side only when it was host-visible,
// so a bad device entry is clamped rather than followed).
__device__ inline int kv_page(const TensorDesc &T, int bb, int pos)
{
    const int page = __ldg(T.bt + (int64_t)bb * T.pps + pos / T.page_size);
    return (page >= 0 && page < T.num_pages) ? page : 0;
}

// Row `pos` of unit (l, bb, h) of K or V, contiguous or paged.
__device__ inline const __nv_bfloat16 *kv_row_ptr(const TensorDesc &T, int l, int bb, int h,
                                                  int pos)
{
    if (T.bt)
        return T.data + l * T.s_layer + (int64_t)kv_page(T, bb, pos) * T.s_page +
               (int64_t)(pos % T.page_size) * T.s_pos + (int64_t)h * T.s_head;
    return kv_unit_ptr(T, l, bb, h) + (int64_t)pos * T.s_pos;
}

// ---------------------------------------------------------------------------
// PTX wrappers (warp-level tensor core path and async copies).

__device__ __forceinline__ uint32_t smem_u32(const void *p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// 16-byte async copy global -> shared; bytes beyond src_bytes (0 or 16) are zero-filled.
__device__ __forceinline__ void cp_async_16(void *smem, const void *gmem, int src_bytes)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(smem_u32(smem)),
                 "l"(gmem), "r"(src_bytes));
}

__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }

template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N)); }

__device__ __forceinline__ void ldmatrix_x4(uint32_t (&r)[4], const void *smem)
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];\n"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(smem_u32(smem)));
}

// D = A(16x16 bf16, row) * B(16x8 bf16, col) + D, fp32 accumulate.
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                               uint32_t b1)
{
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
        "{%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};\n"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Hardware base-2 exponential (MUFU); ex2(-inf) = +0.
__device__ __forceinline__ float ex2(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;\n" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ void set_status(uint32_t *status, uint32_t code)
{
    if (status)
        atomicCAS(status, 0u, code);
}

// Order-preserving map of a float to uint32 (larger float -> larger key); -0.0 maps to the
// key of +0.0, since the two compare equal (a tie broken by position, like any other).
__device__ __forceinline__ uint32_t float_key(float f)
{
    const uint32_t u = __float_as_uint(f == 0.f ? 0.f : f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__device__ __forceinline__ float key_float(uint32_t k)
{
    return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}

}  // namespace dge
