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
#include "e2ga_internal.cuh"

namespace {

constexpr int kNoallocMaxPop = E2_NOALLOC_MAX_POP;
constexpr int kMaxDeviceIds = 64;

// Scratch: [0, P) fingerprints (u64), then [P, 2P) duplicate flags (stored in
// the low word of a u64 slot so that the array stays one type).
static __device__ __align__(256) unsigned long long g_noalloc_scratch[2 * kNoallocMaxPop];

// Device address of g_noalloc_scratch per device id, set up on the first call
// made with that device current.
unsigned long long *g_scratch_addr[kMaxDeviceIds] = {};

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

// Duplicate flag: equal to a lower-indexed genome (compared in full when the
// fitness and fingerprint agree).
__global__ void __launch_bounds__(256) dup_noalloc(e2::DevPop p, int P, int M, int K, const double *fit,
                                                   const unsigned long long *hash, unsigned long long *dup)
{
    const int g = blockIdx.x * blockDim.x + threadIdx.x;
    if (g >= P) return;
    const double w = fit[(size_t)g * 4], ph = fit[(size_t)g * 4 + 1];
    const unsigned long long h = hash[g];
    unsigned long long d = 0;
    for (int o = 0; o < g && !d; ++o) {
        if (hash[o] != h || fit[(size_t)o * 4] != w || fit[(size_t)o * 4 + 1] != ph) continue;
        bool eq = p.nclus[o] == p.nclus[g] && p.roles[o] == p.roles[g];
        for (int i = 0; i < M && eq; ++i) eq = p.perm[(size_t)o * M + i] == p.perm[(size_t)g * M + i];
        for (int i = 0; i < K && eq; ++i) eq = p.sizes[(size_t)o * K + i] == p.sizes[(size_t)g * K + i];
        d = eq;
    }
    dup[g] = d;
}

// rank(g) in the order (duplicate, w, phase, index); ranks below Q are elites.
__global__ void __launch_bounds__(256) rank_noalloc(int P, int Q, const double *fit,
                                                    const unsigned long long *dup, int32_t *elite)
{
    const int g = blockIdx.x * blockDim.x + threadIdx.x;
    if (g >= P) return;
    const unsigned long long dg = dup[g];
    const double w = fit[(size_t)g * 4], ph = fit[(size_t)g * 4 + 1];
    int rank = 0;
    for (int o = 0; o < P; ++o) {
        const unsigned long long d = dup[o];
        const double wo = fit[(size_t)o * 4], po = fit[(size_t)o * 4 + 1];
        bool before;
        if (d != dg) before = d < dg;
        else if (wo != w) before = wo < w;
        else if (po != ph) before = po < ph;
        else before = o < g;
        rank += before;
    }
    if (rank < Q) elite[rank] = g;
}

bool on_device(const void *p)
{
    cudaPointerAttributes a;
    if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
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
    if (!on_device(pop->perm) || !on_device(pop->sizes) || !on_device(pop->nclus) || !on_device(pop->roles) ||
        !on_device(fitness) || (Q > 0 && !on_device(elite_idx)))
        return reject(E2_EINVAL, "inputs and output must be device memory of the current device");
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return reject(E2_ECUDA, "cudaGetDevice failed");
    if (dev < 0 || dev >= kMaxDeviceIds) return reject(E2_EINVAL, "device id beyond the supported range");
    if (!g_scratch_addr[dev]) {
        void *addr = nullptr;
        const cudaError_t e = cudaGetSymbolAddress(&addr, g_noalloc_scratch);
        if (e != cudaSuccess || !addr) return reject(E2_ECUDA, "cudaGetSymbolAddress of the scratch array failed");
        g_scratch_addr[dev] = static_cast<unsigned long long *>(addr);
    }
    unsigned long long *hash = g_scratch_addr[dev];
    unsigned long long *dup = hash + P;
    const e2::DevPop p{pop->perm, pop->sizes, pop->nclus, pop->roles};
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const unsigned blocks = (unsigned)((P + 255) / 256);
    fingerprint_noalloc<<<blocks, 256, 0, s>>>(p, P, M, K_max, hash);
    dup_noalloc<<<blocks, 256, 0, s>>>(p, P, M, K_max, fitness, hash, dup);
    if (Q > 0) rank_noalloc<<<blocks, 256, 0, s>>>(P, Q, fitness, dup, elite_idx);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return reject(E2_ECUDA, cudaGetErrorString(e));
    return E2_OK;
}
