// elites_noalloc.cu -- elite selection for callers that cannot allocate
// device memory.
//
// The regular path (e2_ga_step) keeps its scratch (genome fingerprints and
// duplicate flags) in the workspace the caller allocated for a context.  Some
// callers cannot allocate at all: code running while a CUDA graph is being
// captured (cudaMalloc is not capturable), plug-ins inside a host framework
// whose allocator already owns the device memory and hands none out, or
// latency-critical loops that must never hit cudaMalloc's implicit device
// synchronisation.  e2_select_elites_noalloc serves them: the caller passes
// only its inputs (population and fitness) and its output (elite indices);
// the scratch lives in the file-scope array below, sized for at most
// E2_NOALLOC_MAX_POP genomes.  The array is part of the library's device image:
// every GPU that loads the library holds it (1 MiB) until the process exits.
//
// Every call shares that one array and leaves its contents behind.  Nothing in
// it has to start at zero (each call writes every entry it reads), but two
// calls that overlap on the GPU -- on different streams, or from different
// host threads -- race on it and must be serialised by the caller.
//
// The duplicate test and the ranks follow the same order as e2_ga_step's
// elites: fitness keys compared as the bit patterns of w and phase (the order
// of the values for the non-negative and +inf results an evaluation produces,
// and a total order for any other input), staged tile by tile in shared
// memory with one warp per genome.
#include <mutex>

#include "e2ga_internal.cuh"

namespace {

constexpr int kNoallocMaxPop = E2_NOALLOC_MAX_POP;
constexpr int kMaxDeviceIds = 64;
constexpr int kTile = 1024;
constexpr int kWarps = 8;

// Scratch: [0, P) fingerprints (u64), then [P, 2P) duplicate flags (stored in
// the low word of a u64 slot so that the array stays one type).
static __device__ __align__(256) unsigned long long g_noalloc_scratch[2 * kNoallocMaxPop];

// Device address of g_noalloc_scratch per device id, with the CUDA context
// that was current when it was looked up (a reset device gets a new context,
// and the address is looked up again).
struct ScratchSlot {
    void *ctx = nullptr;
    unsigned long long *addr = nullptr;
};
ScratchSlot g_scratch[kMaxDeviceIds];
std::mutex g_scratch_mutex;

// cuCtxGetCurrent, reached through the runtime's entry-point table (no link
// against the driver library).
typedef int (*CtxGetCurrentFn)(void **);

void *current_context()
{
    static CtxGetCurrentFn fn = nullptr;
    static bool looked = false;
    if (!looked) {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<CtxGetCurrentFn>(p);
        else
            cudaGetLastError();
        looked = true;
    }
    void *ctx = nullptr;
    if (!fn || fn(&ctx) != 0) return nullptr;
    return ctx;
}

__device__ __forceinline__ uint64_t key_bits(const double *fit, size_t i, int q)
{
    return (uint64_t)__double_as_longlong(fit[i * 4 + q]);
}

__global__ void fingerprint_noalloc(e2::DevPop p, int P, int M, int K, unsigned long long *hash)
{
    const int g = blockIdx.x * blockDim.x + threadIdx.x;
    if (g >= P) return;
    uint64_t h = 0x9E3779B97F4A7C15ull;
    auto mix = [&](uint64_t x) { h = (h ^ x) * 0xBF58476D1CE4E5B9ull; h ^= h >> 31; };
    const int R = p.nclus[g];
    for (int i = 0; i < M; ++i) mix(p.perm[(size_t)g * M + i]);
    for (int i = 0; i < R && i < K; ++i) mix((uint64_t)p.sizes[(size_t)g * K + i] << 16);
    mix((uint64_t)R << 40);
    mix(p.roles[g]);
    hash[g] = h;
}

// Duplicate flag, one warp per genome: equal to a lower-indexed genome
// (compared in full only where the fitness keys and the fingerprint agree).
__global__ void __launch_bounds__(32 * kWarps) dup_noalloc(e2::DevPop p, int P, int M, int K, const double *fit,
                                                           const unsigned long long *hash, unsigned long long *dup)
{
    __shared__ uint64_t s_w[kTile], s_p[kTile], s_h[kTile];
    const int lane = threadIdx.x & 31, wl = threadIdx.x >> 5;
    const int g = blockIdx.x * kWarps + wl;
    const bool live = g < P;
    const uint64_t w = live ? key_bits(fit, g, 0) : 0, ph = live ? key_bits(fit, g, 1) : 0;
    const uint64_t h = live ? hash[g] : 0;
    const int gmax = min(P, (int)(blockIdx.x + 1) * kWarps);
    int d = 0;
    for (int base = 0; base < gmax - 1; base += kTile) {
        __syncthreads();
        for (int t = threadIdx.x; t < kTile && base + t < P; t += blockDim.x) {
            s_w[t] = key_bits(fit, base + t, 0);
            s_p[t] = key_bits(fit, base + t, 1);
            s_h[t] = hash[base + t];
        }
        __syncthreads();
        if (!live || d) continue;
        const int lim = min(kTile, g - base);
        for (int t0 = 0; t0 < lim && !d; t0 += 32) {
            const int t = t0 + lane;
            const bool cand = t < lim && s_h[t] == h && s_w[t] == w && s_p[t] == ph;
            unsigned b = __ballot_sync(0xFFFFFFFFu, cand);
            while (b && !d) {
                const int o = base + t0 + __ffs(b) - 1;
                b &= b - 1;
                bool diff = p.nclus[o] != p.nclus[g] || p.roles[o] != p.roles[g];
                for (int i = lane; i < M && !diff; i += 32) diff = p.perm[(size_t)o * M + i] != p.perm[(size_t)g * M + i];
                for (int i = lane; i < K && !diff; i += 32) diff = p.sizes[(size_t)o * K + i] != p.sizes[(size_t)g * K + i];
                d = __ballot_sync(0xFFFFFFFFu, diff) == 0u;
            }
        }
    }
    if (live && lane == 0) dup[g] = (unsigned long long)d;
}

// rank(g) in the order (duplicate, w bits, phase bits, index), one warp per
// genome over shared-memory tiles of the keys; ranks below Q are the elites.
__global__ void __launch_bounds__(32 * kWarps) rank_noalloc(int P, int Q, const double *fit,
                                                            const unsigned long long *dup, int32_t *elite)
{
    __shared__ uint64_t s_w[kTile], s_p[kTile];
    __shared__ int s_d[kTile];
    const int lane = threadIdx.x & 31, wl = threadIdx.x >> 5;
    const int g = blockIdx.x * kWarps + wl;
    const bool live = g < P;
    const uint64_t w = live ? key_bits(fit, g, 0) : 0, ph = live ? key_bits(fit, g, 1) : 0;
    const int dg = live ? (int)dup[g] : 0;
    int rank = 0;
    for (int base = 0; base < P; base += kTile) {
        __syncthreads();
        for (int t = threadIdx.x; t < kTile && base + t < P; t += blockDim.x) {
            s_w[t] = key_bits(fit, base + t, 0);
            s_p[t] = key_bits(fit, base + t, 1);
            s_d[t] = (int)dup[base + t];
        }
        __syncthreads();
        const int lim = min(kTile, P - base);
        if (live)
            for (int t = lane; t < lim; t += 32) {
                const int o = base + t;
                bool before;
                if (s_d[t] != dg) before = s_d[t] < dg;
                else if (s_w[t] != w) before = s_w[t] < w;
                else if (s_p[t] != ph) before = s_p[t] < ph;
                else before = o < g;
                rank += before;
            }
    }
#pragma unroll
    for (int x = 16; x; x >>= 1) rank += __shfl_xor_sync(0xFFFFFFFFu, rank, x);
    if (live && lane == 0 && rank < Q) elite[rank] = g;
}

// Device memory of device `dev` (or managed memory).
bool on_device(const void *p, int dev)
{
    cudaPointerAttributes a;
    if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    if (a.type == cudaMemoryTypeManaged) return true;
    return a.type == cudaMemoryTypeDevice && a.device == dev;
}

// Statuses only: this entry point keeps no error text.
int reject(int code, const char *) { return code; }

}  // namespace

extern "C" int e2_select_elites_noalloc(const e2_genomes *pop, const double *fitness, int32_t P, int32_t M,
                                        int32_t K_max, int32_t Q, int32_t *elite_idx, void *stream)
{
    if (!pop || !pop->perm || !pop->sizes || !pop->nclus || !pop->roles || !fitness)
        return reject(E2_EINVAL, "null input");
    if (P < 1 || P > kNoallocMaxPop) return reject(E2_EINVAL, "P must lie in [1, E2_NOALLOC_MAX_POP]");
    if (M < 1 || M > E2_MAX_DEVICES || K_max < 1 || K_max > E2_MAX_CLUSTERS || Q < 0 || Q > P)
        return reject(E2_EINVAL, "M, K_max or Q out of range");
    if (Q > 0 && !elite_idx) return reject(E2_EINVAL, "null output");
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return reject(E2_ECUDA, "cudaGetDevice failed");
    if (dev < 0 || dev >= kMaxDeviceIds) return reject(E2_EINVAL, "device id beyond the supported range");
    if (!on_device(pop->perm, dev) || !on_device(pop->sizes, dev) || !on_device(pop->nclus, dev) ||
        !on_device(pop->roles, dev) || !on_device(fitness, dev) || (Q > 0 && !on_device(elite_idx, dev)))
        return reject(E2_EINVAL, "inputs and output must be device memory of the current device");
    unsigned long long *hash = nullptr;
    {
        // set-up, once per device and context: the scratch array's device
        // address, looked up with that device current
        std::lock_guard<std::mutex> lock(g_scratch_mutex);
        void *ctx = current_context();
        ScratchSlot &sl = g_scratch[dev];
        if (!sl.addr || sl.ctx != ctx) {
            void *addr = nullptr;
            const cudaError_t e = cudaGetSymbolAddress(&addr, g_noalloc_scratch);
            if (e != cudaSuccess || !addr) {
                cudaGetLastError();
                return reject(E2_ECUDA, "cudaGetSymbolAddress of the scratch array failed");
            }
            sl.addr = static_cast<unsigned long long *>(addr);
            sl.ctx = ctx;
        }
        hash = sl.addr;
    }
    unsigned long long *dup = hash + P;
    const e2::DevPop p{pop->perm, pop->sizes, pop->nclus, pop->roles};
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const unsigned blocks = (unsigned)((P + 255) / 256);
    const unsigned wblocks = (unsigned)((P + kWarps - 1) / kWarps);
    fingerprint_noalloc<<<blocks, 256, 0, s>>>(p, P, M, K_max, hash);
    dup_noalloc<<<wblocks, 32 * kWarps, 0, s>>>(p, P, M, K_max, fitness, hash, dup);
    if (Q > 0) rank_noalloc<<<wblocks, 32 * kWarps, 0, s>>>(P, Q, fitness, dup, elite_idx);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return reject(E2_ECUDA, cudaGetErrorString(e));
    return E2_OK;
}
