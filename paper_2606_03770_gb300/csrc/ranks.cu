// ranks.cu -- 32-bit order keys for the DP.
//
// The DP of a variant v only ever compares values drawn from one finite set
// S_v: the stage times l_d(n, master) of every device, the link times
// tau_v(a, b), and 0 (the empty stage).  Replacing each value x by
//     rank_v(x) = #{ y in S_v : y < x }      (+inf -> 0xFFFFFFFF)
// keeps every comparison, every tie and every argmin exactly as in float64,
// while halving the shared memory of the DP and making each comparison a
// single 32-bit instruction.  The float64 times are kept for what the DP
// reports (the bottleneck T and the latency Lambda are recomputed from the
// chosen partition).
//
// rank_v(x) = (#stage times < x) + (#link times < x), each a binary search in
// a sorted list.  Stage times are sorted once per context; link times change
// with every congestion redraw, but tau_v(a,b) = A_v / Beff(a,b) falls as Beff
// rises for every v, so one ascending sort of the effective bandwidths gives
// every variant's sorted link times.  Sorting is a bitonic network (global
// passes for strides >= 1024 elements, the rest in shared memory).
#include "e2ga_internal.cuh"

namespace e2 {

namespace {

constexpr int kLocal = 2048;   // elements sorted per CTA in shared memory

__device__ __forceinline__ void cmpx(uint64_t &a, uint64_t &b, bool up)
{
    if ((a > b) == up) { const uint64_t t = a; a = b; b = t; }
}

// Bitonic stages (k, j) with j < kLocal for every k in [k_lo, k_hi], on
// chunks of kLocal elements in shared memory; blockIdx.y selects the array.
__global__ void __launch_bounds__(1024) bitonic_local(uint64_t *data, size_t stride_arrays, size_t k_lo,
                                                      size_t k_hi)
{
    __shared__ uint64_t s[kLocal];
    uint64_t *a = data + blockIdx.y * stride_arrays + (size_t)blockIdx.x * kLocal;
    const size_t base = (size_t)blockIdx.x * kLocal;
    for (int i = threadIdx.x; i < kLocal; i += blockDim.x) s[i] = a[i];
    __syncthreads();
    for (size_t k = k_lo; k <= k_hi; k <<= 1) {
        for (size_t j = (k >> 1) < (size_t)(kLocal >> 1) ? (k >> 1) : (size_t)(kLocal >> 1); j > 0; j >>= 1) {
            for (int t = threadIdx.x; t < kLocal / 2; t += blockDim.x) {
                const size_t i = 2 * j * (t / j) + (t % j);          // lower index of the pair
                const bool up = ((base + i) & k) == 0;
                cmpx(s[i], s[i + j], up);
            }
            __syncthreads();
        }
    }
    for (int i = threadIdx.x; i < kLocal; i += blockDim.x) a[i] = s[i];
}

// One bitonic stage (k, j) with j >= kLocal, in global memory.
__global__ void bitonic_global(uint64_t *data, size_t stride_arrays, size_t n, size_t k, size_t j)
{
    uint64_t *a = data + blockIdx.y * stride_arrays;
    for (size_t t = blockIdx.x * (size_t)blockDim.x + threadIdx.x; t < n / 2; t += (size_t)gridDim.x * blockDim.x) {
        const size_t i = 2 * j * (t / j) + (t % j);
        cmpx(a[i], a[i + j], (i & k) == 0);
    }
}

// Keys for the stage-time sort: every finite or infinite l_d(n, master) of
// variant v, padded with +inf up to the power of two.
__global__ void leaf_keys(Dims dm, const double *leaf, uint64_t *keys, size_t cap)
{
    const size_t per = (size_t)dm.M * 2 * dm.N;
    for (size_t idx = blockIdx.x * (size_t)blockDim.x + threadIdx.x; idx < (size_t)dm.V * cap;
         idx += (size_t)gridDim.x * blockDim.x) {
        const int v = (int)(idx / cap);
        const size_t i = idx - (size_t)v * cap;
        uint64_t key = ~0ull;
        if (i < per) {
            const size_t row = i / dm.N, n = i - row * dm.N;           // row = d * 2 + master
            key = dkey(leaf[((size_t)v * dm.M * 2 + row) * dm.LS + n]);
        }
        keys[idx] = key;
    }
}

// Keys for the link sort: effective bandwidth of every ordered pair (the
// diagonal, never a pipeline link, as +inf: a harmless extra 0 link time).
__global__ void beff_keys(int M, const double *link_bw, const double *cong, uint64_t *keys, size_t cap)
{
    const size_t MM = (size_t)M * M;
    for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < cap; i += (size_t)gridDim.x * blockDim.x) {
        uint64_t key = ~0ull;
        if (i < MM) {
            const int a = (int)(i / M), b = (int)(i - (size_t)a * M);
            key = a == b ? kInfKey : dkey(link_bw[i] * cong[i]);
        }
        keys[i] = key;
    }
}

// Sorted link times of variant v: tau_sorted[v][i] = A_v / Beff_desc[i].
__global__ void tau_sorted_kernel(Dims dm, const uint64_t *beff_sorted, const uint64_t *prof, double *tau_sorted)
{
    const size_t MM = (size_t)dm.M * dm.M;
    for (size_t idx = blockIdx.x * (size_t)blockDim.x + threadIdx.x; idx < (size_t)dm.V * MM;
         idx += (size_t)gridDim.x * blockDim.x) {
        const int v = (int)(idx / MM);
        const size_t i = idx - (size_t)v * MM;
        const double beff = keyd(beff_sorted[MM - 1 - i]);              // descending bandwidth
        tau_sorted[idx] = __ull2double_rn(prof[kAct * dm.V + v]) / beff;
    }
}

__device__ __forceinline__ size_t lower_bound_key(const uint64_t *a, size_t n, uint64_t x)
{
    size_t lo = 0, hi = n;
    while (lo < hi) {
        const size_t mid = (lo + hi) >> 1;
        if (a[mid] < x) lo = mid + 1;
        else hi = mid;
    }
    return lo;
}

__device__ __forceinline__ uint32_t rank_of(uint64_t x, const uint64_t *leaf_sorted, size_t nleaf,
                                            const uint64_t *tau_sorted, size_t ntau)
{
    if (x >= kInfKey) return 0xFFFFFFFFu;
    return (uint32_t)(lower_bound_key(leaf_sorted, nleaf, x) + lower_bound_key(tau_sorted, ntau, x));
}

// rank tables: leaf_rank[v][d][mf][n] and tau_rank[v][a][b]
__global__ void rank_kernel_tables(Dims dm, const double *leaf, const double *tau, const uint64_t *leaf_sorted,
                                   size_t leaf_cap, const double *tau_sorted, uint32_t *leaf_rank, uint32_t *tau_rank)
{
    const size_t nleaf = (size_t)dm.M * 2 * dm.N, MM = (size_t)dm.M * dm.M;
    const size_t L = (size_t)dm.V * dm.M * 2 * dm.LS, T = (size_t)dm.V * MM;
    for (size_t idx = blockIdx.x * (size_t)blockDim.x + threadIdx.x; idx < L + T;
         idx += (size_t)gridDim.x * blockDim.x) {
        int v;
        uint64_t x;
        if (idx < L) {
            v = (int)(idx / ((size_t)dm.M * 2 * dm.LS));
            x = dkey(leaf[idx]);
        } else {
            v = (int)((idx - L) / MM);
            x = dkey(tau[idx - L]);
        }
        const uint64_t *ls = leaf_sorted + (size_t)v * leaf_cap;
        const uint64_t *ts = reinterpret_cast<const uint64_t *>(tau_sorted) + (size_t)v * MM;
        const uint32_t r = rank_of(x, ls, nleaf, ts, MM);
        if (idx < L) leaf_rank[idx] = r;
        else tau_rank[idx - L] = r;
    }
}

inline unsigned grid_for(size_t n, int threads, size_t cap = 152 * 32)
{
    size_t b = (n + threads - 1) / threads;
    if (b > cap) b = cap;
    return (unsigned)(b ? b : 1);
}

// Adds its launches to *launches.
cudaError_t bitonic_sort(uint64_t *data, size_t n_pow2, int arrays, cudaStream_t st, unsigned long long *launches)
{
    // n_pow2 >= kLocal, a power of two
    bitonic_local<<<dim3((unsigned)(n_pow2 / kLocal), arrays), 1024, 0, st>>>(data, n_pow2, 2, kLocal);
    ++*launches;
    for (size_t k = 2 * kLocal; k <= n_pow2; k <<= 1) {
        for (size_t j = k >> 1; j >= (size_t)kLocal; j >>= 1) {
            bitonic_global<<<dim3(grid_for(n_pow2 / 2, 256), arrays), 256, 0, st>>>(data, n_pow2, n_pow2, k, j);
            ++*launches;
        }
        bitonic_local<<<dim3((unsigned)(n_pow2 / kLocal), arrays), 1024, 0, st>>>(data, n_pow2, k, k);
        ++*launches;
    }
    return cudaGetLastError();
}

}  // namespace

size_t rank_pow2(size_t n)
{
    size_t p = kLocal;
    while (p < n) p <<= 1;
    return p;
}

cudaError_t build_leaf_sorted(const e2_ctx *c)
{
    const size_t cap = rank_pow2((size_t)c->dm.M * 2 * c->dm.N);
    leaf_keys<<<grid_for((size_t)c->dm.V * cap, 256), 256, 0, c->stream>>>(c->dm, c->leaf, c->leaf_sorted, cap);
    ++c->launches;
    return bitonic_sort(c->leaf_sorted, cap, c->dm.V, c->stream, &c->launches);
}

cudaError_t build_ranks(const e2_ctx *c)
{
    const size_t MM = (size_t)c->dm.M * c->dm.M, bcap = rank_pow2(MM);
    beff_keys<<<grid_for(bcap, 256), 256, 0, c->stream>>>(c->dm.M, c->link_bw, c->cong, c->beff_sorted, bcap);
    ++c->launches;
    cudaError_t e = bitonic_sort(c->beff_sorted, bcap, 1, c->stream, &c->launches);
    if (e != cudaSuccess) return e;
    tau_sorted_kernel<<<grid_for((size_t)c->dm.V * MM, 256), 256, 0, c->stream>>>(c->dm, c->beff_sorted, c->prof,
                                                                                c->tau_sorted);
    const size_t leaf_cap = rank_pow2((size_t)c->dm.M * 2 * c->dm.N);
    const size_t total = (size_t)c->dm.V * c->dm.M * 2 * c->dm.LS + (size_t)c->dm.V * MM;
    rank_kernel_tables<<<grid_for(total, 256), 256, 0, c->stream>>>(c->dm, c->leaf, c->tau, c->leaf_sorted, leaf_cap,
                                                                    c->tau_sorted, c->leaf_rank, c->tau_rank);
    c->launches += 2;
    return cudaGetLastError();
}

}  // namespace e2
