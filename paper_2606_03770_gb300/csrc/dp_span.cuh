// dp_span.cuh -- the DP's column arithmetic on order keys, shared by the
// four-warp DP kernel (dp_eval.cu) and the warp-per-run kernel (dp_warp.cu):
// one cell and one span of a band-form column of Eq. 1 by the crossover
// bisection, the asynchronous row copies, and a warp sum.
#pragma once
#include "e2ga_internal.cuh"

namespace e2 {

namespace {

// D_k[r] for one cell (see the header comment), on order keys (the largest
// value is +inf).
template <typename Key>
__device__ __forceinline__ Key dp_cell(const Key *__restrict__ prev, const Key *__restrict__ row, Key tau, int r)
{
    int lo = 0, hi = r + 1;
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (prev[mid] >= row[r - mid]) hi = mid;
        else lo = mid + 1;
    }
    Key h = (Key)~(Key)0;
    if (lo <= r) h = prev[lo];
    if (lo >= 1) h = min(h, row[r - lo + 1]);
    return max(h, tau);
}

// D_k[r] for the cells r0 <= r < r1 of one column: the first crossover by
// bisection, then each next one from the last.  With both operands
// non-decreasing, the crossover of r + 1 is that of r or one more (if
// prev[s] >= row[r-s] then prev[s+1] >= row[(r+1)-(s+1)]), so every cell after
// the first costs one probe.
template <typename Key>
__device__ __forceinline__ void dp_span(const Key *__restrict__ prev, const Key *__restrict__ row, Key tau,
                                        Key *__restrict__ cur, int r0, int r1)
{
    if (r0 >= r1) return;
    int r = r0, lo = 0, hi = r0 + 1;
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (prev[mid] >= row[r - mid]) hi = mid;
        else lo = mid + 1;
    }
    for (;;) {
        Key h = (Key)~(Key)0;
        if (lo <= r) h = prev[lo];
        if (lo >= 1) h = min(h, row[r - lo + 1]);
        cur[r] = max(h, tau);
        if (++r >= r1) break;
        if (!(prev[lo] >= row[r - lo])) ++lo;                // lo <= r: the crossover moves by at most one
    }
}

__device__ __forceinline__ void cp_async4(void *smem_dst, const void *gmem_src)
{
    const unsigned sa = (unsigned)__cvta_generic_to_shared(smem_dst);
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(sa), "l"(gmem_src) : "memory");
}

__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;" ::: "memory"); }


__device__ __forceinline__ int warp_sum(int x)
{
#pragma unroll
    for (int o = 16; o; o >>= 1) x += __shfl_xor_sync(0xFFFFFFFFu, x, o);
    return x;
}

// A row of order keys from the rank table into shared memory, copied
// asynchronously.
__device__ __forceinline__ void stage_row(uint32_t *dst, const uint32_t *src, int W, int lane)
{
    for (int n = lane; n < W; n += 32) cp_async4(dst + n, src + n);
}

// The head row of a master, fetched asynchronously while the warp builds H.
template <typename Key> struct HeadRow;
template <> struct HeadRow<uint32_t> {
    __device__ __forceinline__ void start(uint32_t *dst, const uint32_t *src, int W, int lane)
    {
        for (int r = lane; r < W; r += 32) cp_async4(dst + r, src + r);
    }
    __device__ __forceinline__ void finish(uint32_t *, const uint32_t *, int, int) { cp_async_wait_all(); }
};

}  // namespace

}  // namespace e2
