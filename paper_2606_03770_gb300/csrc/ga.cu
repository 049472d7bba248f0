// ga.cu -- cost tables, congestion redraw, population validation, the random
// initial population, elites and the generation step (Sec. 3.2 cost model,
// Sec. 3.4 and App. A genetic algorithm).  All randomness comes from
// Philox-4x32-10 streams keyed by (seed, generation, slot, purpose), so a
// generation replays bit for bit whatever the thread mapping.
#include "e2ga_internal.cuh"

namespace e2 {

namespace {

constexpr int kBitmapWords = E2_MAX_DEVICES / 32;

// Blocks of a stage that sit in device memory: as many as fit beside the LM
// head and output layer on the master (which never leave device memory); -1
// when the head alone does not fit.
__device__ __forceinline__ long long device_blocks(uint64_t nb, uint64_t bm, uint64_t hm, uint64_t mem)
{
    if (hm > mem) return -1;
    const uint64_t cap = bm ? (mem - hm) / bm : nb;
    return (long long)(nb < cap ? nb : cap);
}

// l_d(n, master): the larger of compute time and streaming time of n identical
// blocks (plus the LM head and output layer on the master), +inf when they do
// not fit in memory (Sec. 3.2).  With GPU-CPU offload (a device with host
// memory) the blocks beyond device memory sit in host memory, if they fit,
// and run there at the host's rate and bandwidth after the device's part:
// the two times add (the plans' G--C split, Sec. 4.3).
__global__ void tables_kernel(Dims dm, const double *rate, const double *bw, const uint64_t *mem,
                              const double *rate_cpu, const double *bw_cpu, const uint64_t *mem_cpu,
                              const uint64_t *prof, double *leaf)
{
    const size_t total = (size_t)dm.V * dm.M * 2 * dm.LS;
    for (size_t idx = blockIdx.x * (size_t)blockDim.x + threadIdx.x; idx < total;
         idx += (size_t)gridDim.x * blockDim.x) {
        const int n = (int)(idx % dm.LS);
        size_t rest = idx / dm.LS;
        const int mf = (int)(rest & 1);
        rest >>= 1;
        const int d = (int)(rest % dm.M);
        const int v = (int)(rest / dm.M);
        double out = keyd(kInfKey);
        if (n < dm.N) {
            const uint64_t nb = (uint64_t)n + 1;
            const int V = dm.V;
            const uint64_t bm = prof[kBlkMem * V + v];
            const long long g = device_blocks(nb, bm, mf ? prof[kHeadMem * V + v] : 0ull, mem[d]);
            const uint64_t c = g < 0 ? 0ull : nb - (uint64_t)g;        // offloaded blocks
            if (g >= 0 && (c == 0 || c * bm <= mem_cpu[d])) {
                const uint64_t gb = (uint64_t)g;
                const uint64_t fl = gb * prof[kBlkFlops * V + v] + (mf ? prof[kHeadFlops * V + v] : 0ull);
                const uint64_t by = gb * prof[kBlkBytes * V + v] + (mf ? prof[kHeadBytes * V + v] : 0ull);
                const double tc = __ull2double_rn(fl) / rate[d];
                const double tm = __ull2double_rn(by) / bw[d];
                out = tc >= tm ? tc : tm;
                if (c > 0) {
                    const double hc = __ull2double_rn(c * prof[kBlkFlops * V + v]) / rate_cpu[d];
                    const double hb = __ull2double_rn(c * prof[kBlkBytes * V + v]) / bw_cpu[d];
                    out = out + (hc >= hb ? hc : hb);
                }
            }
        }
        leaf[idx] = out;
    }
}

// Per-layer profiles (blocks of several types): the time of blocks j..j+n-1 on
// device d, with and without the head, from the prefix sums PF, PB, PM
// (psum[a][v][N+1]): the larger of compute and streaming time, +inf beyond
// device memory or past the last block.
__global__ void layered_tables_kernel(Dims dm, const double *rate, const double *bw, const uint64_t *mem,
                                      const uint64_t *prof, const uint64_t *psum, double *lcost)
{
    const size_t NN = (size_t)dm.N * dm.N, total = (size_t)dm.V * dm.M * 2 * NN;
    const size_t row = (size_t)dm.N + 1, plane = (size_t)dm.V * row;
    for (size_t idx = blockIdx.x * (size_t)blockDim.x + threadIdx.x; idx < total;
         idx += (size_t)gridDim.x * blockDim.x) {
        const int n = (int)(idx % dm.N) + 1;
        const int j = (int)((idx / dm.N) % dm.N);
        size_t rest = idx / NN;
        const int mf = (int)(rest & 1);
        rest >>= 1;
        const int d = (int)(rest % dm.M);
        const int v = (int)(rest / dm.M);
        double out = keyd(kInfKey);
        if (j + n <= dm.N) {
            const int V = dm.V;
            const uint64_t *pf = psum + (size_t)v * row, *pb = psum + plane + (size_t)v * row,
                           *pm = psum + 2 * plane + (size_t)v * row;
            const uint64_t need = pm[j + n] - pm[j] + (mf ? prof[kHeadMem * V + v] : 0ull);
            if (need <= mem[d]) {
                const uint64_t fl = pf[j + n] - pf[j] + (mf ? prof[kHeadFlops * V + v] : 0ull);
                const uint64_t by = pb[j + n] - pb[j] + (mf ? prof[kHeadBytes * V + v] : 0ull);
                const double tc = __ull2double_rn(fl) / rate[d];
                const double tm = __ull2double_rn(by) / bw[d];
                out = tc >= tm ? tc : tm;
            }
        }
        lcost[idx] = out;
    }
}

// Per (variant, device): the most blocks the device can hold in device and
// host memory together, without and with the LM head (the number of finite
// entries of its two cost rows), the most of them in device memory (the G of
// the G--C split; -1 where the head does not fit), and the per-block time
// rounded down to float, used by the latency bound: max(blk_flops/rate,
// blk_bytes/bw), or the host's per-block time where that is smaller and the
// device offloads (a lower bound on every block's time either way).
__global__ void captab_kernel(Dims dm, const double *rate, const double *bw, const uint64_t *mem,
                              const double *rate_cpu, const double *bw_cpu, const uint64_t *mem_cpu,
                              const uint64_t *prof, int32_t *cap, int32_t *capg, float *cpb)
{
    const size_t total = (size_t)dm.V * dm.M;
    for (size_t idx = blockIdx.x * (size_t)blockDim.x + threadIdx.x; idx < total;
         idx += (size_t)gridDim.x * blockDim.x) {
        const int v = (int)(idx / dm.M), d = (int)(idx - (size_t)v * dm.M);
        const int V = dm.V;
        const uint64_t N = (uint64_t)dm.N;
        const uint64_t bm = prof[kBlkMem * V + v], hm = prof[kHeadMem * V + v], mm = mem[d];
        const uint64_t hc = bm ? mem_cpu[d] / bm : N;                 // blocks host memory holds
        const uint64_t g0 = bm ? mm / bm : N;
        const uint64_t c0 = g0 + hc;
        const uint64_t g1 = mm < hm ? 0ull : (bm ? (mm - hm) / bm : N);
        const uint64_t c1 = mm < hm ? 0ull : g1 + hc;
        cap[idx * 2] = (int32_t)(c0 < N ? c0 : N);
        cap[idx * 2 + 1] = (int32_t)(c1 < N ? c1 : N);
        capg[idx * 2] = (int32_t)(g0 < N ? g0 : N);
        capg[idx * 2 + 1] = mm < hm ? -1 : (int32_t)(g1 < N ? g1 : N);
        const double tc = __ull2double_rn(prof[kBlkFlops * V + v]) / rate[d];
        const double tm = __ull2double_rn(prof[kBlkBytes * V + v]) / bw[d];
        double t = tc >= tm ? tc : tm;
        if (dm.offload && hc > 0) {
            const double hc_ = __ull2double_rn(prof[kBlkFlops * V + v]) / rate_cpu[d];
            const double hb = __ull2double_rn(prof[kBlkBytes * V + v]) / bw_cpu[d];
            const double th = hc_ >= hb ? hc_ : hb;
            t = th < t ? th : t;
        }
        cpb[idx] = __double2float_rd(t);
    }
}

// tau_v(a, b) = A_v / (B(a,b) * congestion(a,b)) (Sec. 3.2), and the same
// rounded down to float for the latency bound.
__global__ void tau_kernel(Dims dm, const double *link_bw, const double *cong, const uint64_t *prof,
                           double *tau, float *tau_lb)
{
    const size_t MM = (size_t)dm.M * dm.M, total = (size_t)dm.V * MM;
    for (size_t idx = blockIdx.x * (size_t)blockDim.x + threadIdx.x; idx < total;
         idx += (size_t)gridDim.x * blockDim.x) {
        const int v = (int)(idx / MM);
        const size_t ab = idx - (size_t)v * MM;
        const double beff = link_bw[ab] * cong[ab];
        const double t = __ull2double_rn(prof[kAct * dm.V + v]) / beff;
        tau[idx] = t;
        tau_lb[idx] = __double2float_rd(t);
    }
}

// Congestion factor of each unordered pair a < b: lo + (hi - lo) u, with u a
// 53-bit uniform from words 2(aM+b), 2(aM+b)+1 of the stream (seed, gen, 0, CONG).
__global__ void redraw_kernel(int M, uint64_t seed, uint32_t gen, double lo, double hi, double *cong)
{
    const size_t MM = (size_t)M * M;
    for (size_t idx = blockIdx.x * (size_t)blockDim.x + threadIdx.x; idx < MM;
         idx += (size_t)gridDim.x * blockDim.x) {
        const int a = (int)(idx / M), b = (int)(idx - (size_t)a * M);
        if (a == b) { cong[idx] = 1.0; continue; }
        if (a > b) continue;
        Stream st(seed, gen, 0, kCong);
        const uint32_t w0 = st.word(2u * (uint32_t)idx), w1 = st.word(2u * (uint32_t)idx + 1u);
        const uint64_t u53 = ((uint64_t)(w0 >> 5) << 26) | (uint64_t)(w1 >> 6);
        const double u = (double)u53 * (1.0 / 9007199254740992.0);
        const double span = hi - lo;
        const double t = span * u;
        const double f = lo + t;
        cong[idx] = f;
        cong[(size_t)b * M + a] = f;
    }
}

__global__ void validate_kernel(Dims dm, DevPop p, int32_t *err)
{
    const int g = blockIdx.x * blockDim.x + threadIdx.x;
    if (g >= dm.P) return;
    const int M = dm.M, K = dm.K;
    const int R = p.nclus[g];
    bool ok = R >= 1 && R <= K && R <= M;
    int sum = 0;
    for (int c = 0; c < K && ok; ++c) {
        const int s = p.sizes[(size_t)g * K + c];
        if (c < R) { ok = s >= 1; sum += s; }
        else ok = s == 0;
    }
    ok = ok && sum == M;
    if (ok && R < 64) ok = (p.roles[g] >> R) == 0ull;
    uint32_t seen[kBitmapWords];
    const int words = (M + 31) >> 5;
    for (int w = 0; w < words; ++w) seen[w] = 0;
    for (int i = 0; i < M && ok; ++i) {
        const int d = p.perm[(size_t)g * M + i];
        if (d >= M || ((seen[d >> 5] >> (d & 31)) & 1u)) ok = false;
        else seen[d >> 5] |= 1u << (d & 31);
    }
    if (!ok) {
        atomicMin(err, g);
        // replaced by a valid genome (the identity ordering as one prefill
        // replica), so that no later kernel reads an invalid one
        for (int i = 0; i < M; ++i) p.perm[(size_t)g * M + i] = (uint16_t)i;
        for (int c = 0; c < K; ++c) p.sizes[(size_t)g * K + c] = (uint16_t)(c ? 0 : M);
        p.nclus[g] = 1;
        p.roles[g] = 0;
    }
}

// Fisher-Yates shuffle of the identity ordering (word M-1-t draws position t);
// element i of the ordering lives at perm[i * stride].
template <typename T>
__device__ void random_perm(Stream &st, int M, T *perm, int stride = 1)
{
    for (int i = 0; i < M; ++i) perm[(size_t)i * stride] = (T)i;
    for (int t = M - 1; t >= 1; --t) {
        const uint32_t j = below(st.word((uint32_t)(M - 1 - t)), (uint32_t)t + 1);
        const T x = perm[(size_t)t * stride];
        perm[(size_t)t * stride] = perm[(size_t)j * stride];
        perm[(size_t)j * stride] = x;
    }
}

// Grouping of Mr devices: replica count 1 + uniform(min(Kr, Mr)) from word 0;
// the R-1 cut points by sequential selection sampling (candidate cut t taken
// with probability needed/remaining, word t); one role bit per replica from
// two words of the roles stream.  Returns R.
__device__ int random_grouping(Stream &sg, Stream &sr, int Mr, int Kr, uint16_t *sizes, uint64_t *roles)
{
    const int cap = Kr < Mr ? Kr : Mr;
    const int R = 1 + (int)below(sg.word(0), (uint32_t)cap);
    int need = R - 1, prev = 0, c = 0;
    for (int t = 1; t <= Mr - 1 && need > 0; ++t) {
        if (below(sg.word((uint32_t)t), (uint32_t)(Mr - t)) < (uint32_t)need) {
            sizes[c++] = (uint16_t)(t - prev);
            prev = t;
            --need;
        }
    }
    sizes[c] = (uint16_t)(Mr - prev);
    const uint64_t bits = (uint64_t)sr.word(0) | ((uint64_t)sr.word(1) << 32);
    *roles = R >= 64 ? bits : (bits & ((1ull << R) - 1ull));
    return R;
}

__global__ void init_kernel(Dims dm, DevPop p, uint64_t seed)
{
    const int s = blockIdx.x * blockDim.x + threadIdx.x;
    if (s >= dm.P) return;
    const int M = dm.M, K = dm.K;
    uint16_t *perm = p.perm + (size_t)s * M;
    uint16_t *sizes = p.sizes + (size_t)s * K;
    Stream sp(seed, 0, (uint32_t)s, kInitPerm);
    random_perm(sp, M, perm);
    for (int c = 0; c < K; ++c) sizes[c] = 0;
    Stream sg(seed, 0, (uint32_t)s, kInitGroup), sr(seed, 0, (uint32_t)s, kInitRoles);
    uint64_t roles;
    p.nclus[s] = (uint8_t)random_grouping(sg, sr, M, K, sizes, &roles);
    p.roles[s] = roles;
}

// Total order of the elites: distinct genomes before duplicates, then lower w,
// lower bottleneck phase, lower index.  w and phase are non-negative or +inf,
// so they are compared as their bit patterns (same order, integer pipe).
__device__ __forceinline__ bool elite_before(int da, uint64_t wa, uint64_t pa, int a, int db, uint64_t wb,
                                             uint64_t pb, int b)
{
    if (da != db) return da < db;
    if (wa != wb) return wa < wb;
    if (pa != pb) return pa < pb;
    return a < b;
}

// Fitness keys of the elites' comparisons are staged in shared memory, tile
// by tile, and shared by the block's warps (one warp per genome).
constexpr int kEliteTile = 1024;

// A genome equal to a lower-indexed one is a duplicate.  Equal genomes have
// equal fingerprints (the finaliser's hash of the ordering, the replica sizes,
// their count and the roles), so a genome is compared in full only with
// genomes of its fingerprint: first with the lowest-indexed one, found in an
// open-addressing table (dup_table_size(P) >= 2P slots, linear probing, so
// never full; a slot keeps its fingerprint and the smallest index that carries
// it); if the two differ -- a 64-bit collision, or genomes that differ only
// in sizes or role bits past their replica count, which the fingerprint does
// not cover -- with every lower-indexed genome of its fingerprint.
// From kDupTableFrom genomes on (below, the table's fill and extra launch cost
// more than the quadratic test: 1,024 genomes +2% per generation, 4,096 -1.8%).
constexpr int kDupTableFrom = 4096;
constexpr uint64_t kNoKey = ~0ull;                       // an empty slot
__device__ __forceinline__ uint64_t table_key(uint64_t h) { return h == kNoKey ? kNoKey - 1 : h; }
__device__ __forceinline__ unsigned table_start(uint64_t k, unsigned mask) { return (unsigned)(k ^ (k >> 32)) & mask; }

// (the table is filled with kNoKey and INT32_MAX beforehand)
__global__ void __launch_bounds__(256) dup_insert_kernel(int P, const uint64_t *hash, unsigned long long *tkey,
                                                         int32_t *tidx, unsigned mask)
{
    for (int g = blockIdx.x * blockDim.x + threadIdx.x; g < P; g += gridDim.x * blockDim.x) {
        const uint64_t k = table_key(hash[g]);
        unsigned s = table_start(k, mask);
        for (unsigned i = 0; i <= mask; ++i, s = (s + 1) & mask) {   // (a free slot is always found)
            const unsigned long long prev = atomicCAS(&tkey[s], (unsigned long long)kNoKey, (unsigned long long)k);
            if (prev == kNoKey || prev == k) {
                atomicMin(&tidx[s], g);
                break;
            }
        }
    }
}

// Whether genomes a and b are equal (ordering, sizes, replica count, roles); a warp.
__device__ __forceinline__ bool same_genome(const DevPop &p, int a, int b, int M, int K, int lane)
{
    bool diff = p.nclus[a] != p.nclus[b] || p.roles[a] != p.roles[b];
    for (int i = lane; i < M && !diff; i += 32) diff = p.perm[(size_t)a * M + i] != p.perm[(size_t)b * M + i];
    for (int i = lane; i < K && !diff; i += 32) diff = p.sizes[(size_t)a * K + i] != p.sizes[(size_t)b * K + i];
    return __ballot_sync(0xFFFFFFFFu, diff) == 0u;
}

// One warp per genome.
__global__ void __launch_bounds__(256) dup_lookup_kernel(Dims dm, DevPop p, const uint64_t *hash,
                                                         const unsigned long long *tkey, const int32_t *tidx,
                                                         unsigned mask, int32_t *dup)
{
    const int lane = threadIdx.x & 31;
    const int g = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (g >= dm.P) return;
    const uint64_t hr = hash[g], k = table_key(hr);
    int first = g;
    if (lane == 0) {                                              // (present: g itself was inserted)
        unsigned s = table_start(k, mask);
        for (unsigned i = 0; i < mask && tkey[s] != k; ++i) s = (s + 1) & mask;
        if (tkey[s] == k) first = tidx[s];
    }
    first = __shfl_sync(0xFFFFFFFFu, first, 0);
    bool d = false;
    if (first < g) {
        d = same_genome(p, first, g, dm.M, dm.K, lane);
        for (int base = first + 1; base < g && !d; base += 32) {  // a fingerprint shared by different genomes
            const int o = base + lane;
            unsigned b = __ballot_sync(0xFFFFFFFFu, o < g && hash[o] == hr);
            while (b && !d) {
                const int oo = base + __ffs(b) - 1;
                b &= b - 1;
                d = same_genome(p, oo, g, dm.M, dm.K, lane);
            }
        }
    }
    if (lane == 0) dup[g] = d;
}

// Below kDupTableFrom genomes, the duplicate test compares each genome with
// every lower-indexed one: equal genomes have equal fitness (the evaluation is
// deterministic) and equal fingerprints, so only those pairs are compared in
// full.
__global__ void __launch_bounds__(256) dup_kernel(Dims dm, DevPop p, const double *fit,
                                                  const uint64_t *hash, int32_t *dup)
{
    __shared__ uint64_t s_w[kEliteTile], s_p[kEliteTile], s_h[kEliteTile];
    const int lane = threadIdx.x & 31, wl = threadIdx.x >> 5;
    const int g = blockIdx.x * (blockDim.x >> 5) + wl;
    const bool live = g < dm.P;
    const uint64_t *fk = reinterpret_cast<const uint64_t *>(fit);
    const uint64_t w = live ? fk[(size_t)g * 4] : 0, ph = live ? fk[(size_t)g * 4 + 1] : 0, h = live ? hash[g] : 0;
    const int M = dm.M, K = dm.K;
    const int gmax = min(dm.P, (int)((blockIdx.x + 1) * (blockDim.x >> 5)));   // highest genome of the block
    int d = 0;
    for (int base = 0; base < gmax - 1; base += kEliteTile) {
        __syncthreads();
        for (int t = threadIdx.x; t < kEliteTile && base + t < dm.P; t += blockDim.x) {
            s_w[t] = fk[(size_t)(base + t) * 4];
            s_p[t] = fk[(size_t)(base + t) * 4 + 1];
            s_h[t] = hash[base + t];
        }
        __syncthreads();
        if (!live || d) continue;
        const int lim = min(kEliteTile, g - base);
        for (int t0 = 0; t0 < lim && !d; t0 += 32) {
            const int t = t0 + lane;
            const bool cand = t < lim && s_h[t] == h && s_w[t] == w && s_p[t] == ph;
            unsigned b = __ballot_sync(0xFFFFFFFFu, cand);
            while (b && !d) {
                const int oo = base + t0 + __ffs(b) - 1;
                b &= b - 1;
                bool diff = p.nclus[oo] != p.nclus[g] || p.roles[oo] != p.roles[g];
                for (int i = lane; i < M && !diff; i += 32) diff = p.perm[(size_t)oo * M + i] != p.perm[(size_t)g * M + i];
                for (int i = lane; i < K && !diff; i += 32) diff = p.sizes[(size_t)oo * K + i] != p.sizes[(size_t)g * K + i];
                d = __ballot_sync(0xFFFFFFFFu, diff) == 0u;
            }
        }
    }
    if (live && lane == 0) dup[g] = d;
}

// rank(g) = number of genomes before g in the elite order (duplicate flag,
// w, phase, index); the first Q ranks are the elites, and the warp of an elite
// copies it into slot rank(g) of the next population.
__global__ void __launch_bounds__(256) rank_kernel(Dims dm, const double *fit, const int32_t *dup,
                                                   int32_t *elite, double *elite_fit, DevPop src, DevPop dst,
                                                   const unsigned long long *ctl)
{
    __shared__ uint64_t s_w[kEliteTile], s_p[kEliteTile];
    __shared__ int s_d[kEliteTile];
    if (ctl[2] != 0) return;                       // the candidate ranking took the elites
    const int lane = threadIdx.x & 31, wl = threadIdx.x >> 5;
    const int g = blockIdx.x * (blockDim.x >> 5) + wl;
    const bool live = g < dm.P;
    const uint64_t *fk = reinterpret_cast<const uint64_t *>(fit);
    const uint64_t w = live ? fk[(size_t)g * 4] : 0, ph = live ? fk[(size_t)g * 4 + 1] : 0;
    const int dg = live ? dup[g] : 0;
    int rank = 0;
    for (int base = 0; base < dm.P; base += kEliteTile) {
        __syncthreads();
        for (int t = threadIdx.x; t < kEliteTile && base + t < dm.P; t += blockDim.x) {
            s_w[t] = fk[(size_t)(base + t) * 4];
            s_p[t] = fk[(size_t)(base + t) * 4 + 1];
            s_d[t] = dup[base + t];
        }
        __syncthreads();
        const int lim = min(kEliteTile, dm.P - base);
        if (live)
            for (int t = lane; t < lim; t += 32) rank += elite_before(s_d[t], s_w[t], s_p[t], base + t, dg, w, ph, g);
    }
#pragma unroll
    for (int x = 16; x; x >>= 1) rank += __shfl_xor_sync(0xFFFFFFFFu, rank, x);
    if (live && rank < dm.Q) {
        const int M = dm.M, K = dm.K;
        for (int i = lane; i < M; i += 32) dst.perm[(size_t)rank * M + i] = src.perm[(size_t)g * M + i];
        for (int i = lane; i < K; i += 32) dst.sizes[(size_t)rank * K + i] = src.sizes[(size_t)g * K + i];
        if (lane == 0) {
            dst.nclus[rank] = src.nclus[g];
            dst.roles[rank] = src.roles[g];
            elite[rank] = g;
            for (int q = 0; q < 4; ++q) elite_fit[(size_t)rank * 4 + q] = fit[(size_t)g * 4 + q];
        }
    }
}

// Elite selection without ranking every genome.  When at least Q genomes are
// distinct, the elites are the Q first distinct genomes in the order (w,
// phase, index), and each has w <= w_Q, the Q-th smallest w among the
// distinct genomes (a genome with a larger w has at least Q distinct genomes
// before it).  One CTA finds w_Q exactly by a radix select over the bit
// patterns of w (8 passes of 8 bits, highest first) and lists the distinct
// genomes with w <= w_Q; only they are ranked against the population.  When
// w_Q is +inf (fewer than Q genomes have a finite w, as early in a search on
// a large fleet) the finite ones are ranked and the rest of the elites are
// the first distinct genomes of the (+inf, +inf) group in index order.  With
// fewer than Q distinct genomes (duplicates then fill the elite slots) the
// full ranking runs instead.  ctl: [0] w_Q bits, [1] candidates to rank,
// [2] 1 = the selection applies (0: full ranking), [3] elites listed after
// the candidates whose rank is their place in the list.
constexpr int kSelThreads = 1024;

__global__ void __launch_bounds__(kSelThreads) elite_select_kernel(int P, int Q, const double *fit, const int32_t *dup,
                                                                   unsigned long long *ctl, int32_t *cand)
{
    __shared__ unsigned hist[256];
    __shared__ unsigned long long s_prefix;
    __shared__ unsigned s_need, s_distinct, s_ncand;
    const uint64_t *fk = reinterpret_cast<const uint64_t *>(fit);
    const int tid = threadIdx.x;
    if (tid == 0) { s_prefix = 0; s_need = (unsigned)Q; s_distinct = 0; s_ncand = 0; }
    __syncthreads();
    unsigned nd = 0;
    for (int g = tid; g < P; g += kSelThreads) nd += dup[g] == 0;
    atomicAdd(&s_distinct, nd);
    __syncthreads();
    const bool apply = Q > 0 && s_distinct >= (unsigned)Q;
    for (int pass = 0; apply && pass < 8; ++pass) {
        const int shift = 56 - 8 * pass;
        const uint64_t hi_mask = pass ? ~0ull << (shift + 8) : 0ull;
        for (int b = tid; b < 256; b += kSelThreads) hist[b] = 0;
        __syncthreads();
        const uint64_t prefix = s_prefix;
        for (int g = tid; g < P; g += kSelThreads) {
            if (dup[g]) continue;
            const uint64_t w = fk[(size_t)g * 4];
            if ((w & hi_mask) == prefix) atomicAdd(&hist[(w >> shift) & 0xFFu], 1u);
        }
        __syncthreads();
        if (tid < 32) {                                   // the bucket holding the need-th smallest:
            const unsigned need = s_need;                 // a warp scan of eight-bin sums, then the
            unsigned c = 0;                               // lane whose sums cross need scans its bins
#pragma unroll
            for (int j = 0; j < 8; ++j) c += hist[tid * 8 + j];
            unsigned incl = c;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const unsigned y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
                if (tid >= o) incl += y;
            }
            const unsigned crossed = __ballot_sync(0xFFFFFFFFu, incl >= need);
            if (tid == __ffs(crossed) - 1) {
                unsigned left = need - (incl - c), b = (unsigned)tid * 8;
                while (hist[b] < left) { left -= hist[b]; ++b; }
                s_need = left;
                s_prefix = prefix | ((uint64_t)b << shift);
            }
        }
        __syncthreads();
    }
    __shared__ unsigned s_bad, s_wsum[kSelThreads / 32], s_run;
    unsigned direct = 0;                                  // elites whose rank is their place in the list
    bool use = apply;
    if (apply) {
        const uint64_t wq = s_prefix;
        if (wq != kInfKey) {                              // rank every distinct genome with w <= w_Q
            for (int g = tid; g < P; g += kSelThreads)
                if (!dup[g] && fk[(size_t)g * 4] <= wq) cand[atomicAdd(&s_ncand, 1u)] = g;
            __syncthreads();
        } else {
            // fewer than Q distinct genomes with a finite w: those are ranked; the
            // rest of the elites are the first distinct genomes of the (+inf, +inf)
            // group, in index order (an infinite w comes with an infinite phase;
            // anything else takes the full ranking)
            if (tid == 0) s_bad = 0;
            __syncthreads();
            for (int g = tid; g < P; g += kSelThreads) {
                if (dup[g]) continue;
                if (fk[(size_t)g * 4] != kInfKey) cand[atomicAdd(&s_ncand, 1u)] = g;
                else if (fk[(size_t)g * 4 + 1] != kInfKey) s_bad = 1;
            }
            __syncthreads();
            use = s_bad == 0;
            const unsigned F = s_ncand, need = (unsigned)Q - F;
            if (use) {
                const int lane = tid & 31, wl = tid >> 5;
                if (tid == 0) s_run = 0;
                __syncthreads();
                for (int base = 0; base < P && s_run < need; base += kSelThreads) {
                    const int g = base + tid;
                    const bool f = g < P && !dup[g] && fk[(size_t)g * 4] == kInfKey;
                    const unsigned bal = __ballot_sync(0xFFFFFFFFu, f);
                    if (lane == 0) s_wsum[wl] = __popc(bal);
                    __syncthreads();
                    unsigned before = 0;
                    for (int w2 = 0; w2 < wl; ++w2) before += s_wsum[w2];
                    const unsigned ord = s_run + before + __popc(bal & ((1u << lane) - 1u));
                    if (f && ord < need) cand[F + ord] = g;
                    __syncthreads();
                    if (tid == 0) {
                        unsigned t = 0;
                        for (int w2 = 0; w2 < kSelThreads / 32; ++w2) t += s_wsum[w2];
                        s_run += t;
                    }
                    __syncthreads();
                }
                direct = need;
            }
        }
    }
    if (tid == 0) {
        ctl[0] = s_prefix;
        ctl[1] = use ? s_ncand : 0;
        ctl[2] = use ? 1ull : 0ull;
        ctl[3] = use ? direct : 0;
    }
}

// rank(g) for the candidates, one warp each.  Every genome before a candidate
// in the elite order is distinct with a w no larger, so it is a candidate
// itself: a candidate's rank is its count of candidates before it, taken
// over tiles of the candidate list staged in shared memory.  An elite (rank
// < Q) is copied into slot rank of the next population.
__global__ void __launch_bounds__(256) elite_cand_rank_kernel(Dims dm, const double *fit,
                                                              const unsigned long long *ctl, const int32_t *cand,
                                                              int32_t *elite, double *elite_fit, DevPop src, DevPop dst)
{
    __shared__ uint64_t s_w[kEliteTile], s_p[kEliteTile];
    __shared__ int s_g[kEliteTile];
    if (ctl[2] == 0) return;
    const unsigned ncand = (unsigned)ctl[1], total = ncand + (unsigned)ctl[3];
    const int lane = threadIdx.x & 31, NWB = blockDim.x >> 5;
    const uint64_t *fk = reinterpret_cast<const uint64_t *>(fit);
    for (unsigned i0 = blockIdx.x * NWB; i0 < total; i0 += gridDim.x * NWB) {   // uniform over the block
        const unsigned i = i0 + (threadIdx.x >> 5);
        const bool live = i < total, ranked = i < ncand;
        const int g = live ? cand[i] : 0;
        const uint64_t w = ranked ? fk[(size_t)g * 4] : 0, ph = ranked ? fk[(size_t)g * 4 + 1] : 0;
        int rank = (int)i;                               // entries past ncand: rank = place in the list
        if (i0 < ncand) {
            int cnt = 0;
            for (unsigned base = 0; base < ncand; base += kEliteTile) {
                __syncthreads();
                for (unsigned t = threadIdx.x; t < kEliteTile && base + t < ncand; t += blockDim.x) {
                    const int h = cand[base + t];
                    s_g[t] = h;
                    s_w[t] = fk[(size_t)h * 4];
                    s_p[t] = fk[(size_t)h * 4 + 1];
                }
                __syncthreads();
                if (ranked) {
                    const unsigned lim = min((unsigned)kEliteTile, ncand - base);
                    for (unsigned t = lane; t < lim; t += 32)
                        cnt += elite_before(0, s_w[t], s_p[t], s_g[t], 0, w, ph, g);
                }
            }
#pragma unroll
            for (int x = 16; x; x >>= 1) cnt += __shfl_xor_sync(0xFFFFFFFFu, cnt, x);
            if (ranked) rank = cnt;
        }
        if (live && rank < dm.Q) {
            const int M = dm.M, K = dm.K;
            for (int j = lane; j < M; j += 32) dst.perm[(size_t)rank * M + j] = src.perm[(size_t)g * M + j];
            for (int j = lane; j < K; j += 32) dst.sizes[(size_t)rank * K + j] = src.sizes[(size_t)g * K + j];
            if (lane == 0) {
                dst.nclus[rank] = src.nclus[g];
                dst.roles[rank] = src.roles[g];
                elite[rank] = g;
                for (int q = 0; q < 4; ++q) elite_fit[(size_t)rank * 4 + q] = fit[(size_t)g * 4 + q];
            }
        }
    }
}

struct GaThr {
    uint64_t cx, half, mut, k1, k2, k3;
};

__device__ __forceinline__ bool key_before(uint64_t wa, uint64_t pa, int a, uint64_t wb, uint64_t pb, int b)
{
    if (wa != wb) return wa < wb;
    if (pa != pb) return pa < pb;
    return a < b;
}

__device__ __forceinline__ unsigned lanemask_lt()
{
    unsigned m;
    asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
    return m;
}

// One child per warp (App. A).  Slots [0, Q) copy the elites.  Otherwise:
//  * tournaments: lanes draw the candidates, a warp reduction keeps the
//    fittest (the fitness order is strict, so this is the winner of the
//    sequential tournament);
//  * uniform crossover of the ordering chromosome, one position per lane;
//  * repair: first occurrence of each device by shared-memory atomicMin; a
//    later repeat is a hole; the h-th hole (by position) takes the h-th
//    missing device (by id), ranks from warp ballots;
//  * grouping and roles from one parent; then at most one mutation, its
//    random words drawn by the lanes and the sequential steps (Fisher-Yates,
//    selection sampling) taken by lane 0 in shared memory.
// Per warp, shared memory holds the child ordering, the first-occurrence
// table, the missing devices, the random words (M words each) and the sizes.
__global__ void __launch_bounds__(256) ga_kernel(Dims dm, DevPop src, DevPop dst, const double *fit,
                                                 uint64_t seed, uint32_t gen, GaThr thr)
{
    extern __shared__ uint32_t ga_smem[];
    const int lane = threadIdx.x & 31, wl = threadIdx.x >> 5, NWB = blockDim.x >> 5;
    const int M = dm.M, K = dm.K, P = dm.P;
    uint32_t *child = ga_smem + (size_t)wl * (4 * M + 64);
    int32_t *first = reinterpret_cast<int32_t *>(child + M);
    uint32_t *missing = reinterpret_cast<uint32_t *>(first + M);
    uint32_t *words = missing + M;
    uint32_t *ssz = words + M;                                    // [64] sizes
    const uint64_t *fk = reinterpret_cast<const uint64_t *>(fit);
    for (int s = dm.Q + blockIdx.x * NWB + wl; s < P; s += gridDim.x * NWB) {   // the children
        uint16_t *out_perm = dst.perm + (size_t)s * M;
        uint16_t *cs = dst.sizes + (size_t)s * K;
        // ---- two tournaments
        Stream sel(seed, gen, (uint32_t)s, kSelect);
        int par[2];
        for (int q = 0; q < 2; ++q) {
            uint64_t bw = ~0ull, bp = ~0ull;
            int bi = 0x7FFFFFFF;
            for (int t = lane; t < dm.tournament; t += 32) {
                const int cnd = (int)below(sel.word((uint32_t)(q * dm.tournament + t)), (uint32_t)P);
                const uint64_t cw = fk[(size_t)cnd * 4], cp = fk[(size_t)cnd * 4 + 1];
                if (key_before(cw, cp, cnd, bw, bp, bi)) { bw = cw; bp = cp; bi = cnd; }
            }
#pragma unroll
            for (int o = 16; o; o >>= 1) {
                const uint64_t w2 = __shfl_xor_sync(0xFFFFFFFFu, bw, o), p2 = __shfl_xor_sync(0xFFFFFFFFu, bp, o);
                const int i2 = __shfl_xor_sync(0xFFFFFFFFu, bi, o);
                if (key_before(w2, p2, i2, bw, bp, bi)) { bw = w2; bp = p2; bi = i2; }
            }
            par[q] = bi;
        }
        // ---- uniform crossover and repair
        const uint16_t *pa = src.perm + (size_t)par[0] * M, *pb = src.perm + (size_t)par[1] * M;
        Stream cx(seed, gen, (uint32_t)s, kCross);
        for (int q = lane; 4 * q < M; q += 32)                  // a lane takes the 4 positions of one
            for (int i = 4 * q; i < 4 * q + 4 && i < M; ++i) {  // block of the stream (one Philox call)
                child[i] = (uint64_t)cx.word((uint32_t)i) < thr.cx ? pb[i] : pa[i];
                first[i] = 0x7FFFFFFF;
            }
        __syncwarp();
        for (int i = lane; i < M; i += 32) atomicMin(&first[child[i]], i);
        __syncwarp();
        const unsigned lt = lanemask_lt();
        int nmiss = 0;
        for (int base = 0; base < M; base += 32) {
            const int d = base + lane;
            const bool pm = d < M && first[d] == 0x7FFFFFFF;
            const unsigned bm = __ballot_sync(0xFFFFFFFFu, pm);
            if (pm) missing[nmiss + __popc(bm & lt)] = (uint32_t)d;
            nmiss += __popc(bm);
        }
        __syncwarp();
        int nh = 0;
        for (int base = 0; base < M; base += 32) {
            const int i = base + lane;
            const bool hole = i < M && first[child[i]] != i;
            const unsigned bh = __ballot_sync(0xFFFFFFFFu, hole);
            if (hole) child[i] = missing[nh + __popc(bh & lt)];
            nh += __popc(bh);
        }
        // ---- grouping and roles from one parent
        const int from = (uint64_t)cx.word((uint32_t)M) < thr.half ? par[1] : par[0];
        for (int i = lane; i < K; i += 32) ssz[i] = src.sizes[(size_t)from * K + i];
        int R = src.nclus[from];
        uint64_t rl = src.roles[from];
        __syncwarp();
        // ---- mutation
        Stream mt(seed, gen, (uint32_t)s, kMutate);
        if ((uint64_t)mt.word(0) < thr.mut) {
            const uint64_t kind = mt.word(1);
            if (kind < thr.k1) {                                   // swap two positions
                const uint32_t x = below(mt.word(2), (uint32_t)M), y = below(mt.word(3), (uint32_t)M);
                if (lane == 0) { const uint32_t t = child[x]; child[x] = child[y]; child[y] = t; }
            } else {
                int r = 0;
                if (kind < thr.k2) {                               // regroup from a random replica
                    r = (int)below(mt.word(2), (uint32_t)R);
                } else if (kind >= thr.k3) {                       // regenerate both chromosomes
                    Stream sp(seed, gen, (uint32_t)s, kMutPerm);
                    for (int q = lane; 4 * q < M - 1; q += 32)
                        for (int t = 4 * q; t < 4 * q + 4 && t < M - 1; ++t) words[t] = sp.word((uint32_t)t);
                    for (int i = lane; i < M; i += 32) child[i] = (uint32_t)i;
                    __syncwarp();
                    if (lane == 0)
                        for (int t = M - 1; t >= 1; --t) {        // Fisher-Yates, word M-1-t for position t
                            const uint32_t j = below(words[M - 1 - t], (uint32_t)t + 1);
                            const uint32_t x = child[t];
                            child[t] = child[j];
                            child[j] = x;
                        }
                    __syncwarp();
                }
                int kept = 0;
                for (int c = 0; c < r; ++c) kept += (int)ssz[c];
                const int Mr = M - kept, Kr = K - r;
                Stream sg(seed, gen, (uint32_t)s, kMutGroup), sr(seed, gen, (uint32_t)s, kMutRoles);
                for (int q = lane; 4 * q < Mr; q += 32)
                    for (int t = 4 * q; t < 4 * q + 4 && t < Mr; ++t) words[t] = sg.word((uint32_t)t);
                const uint64_t bits = (uint64_t)sr.word(0) | ((uint64_t)sr.word(1) << 32);
                __syncwarp();
                if (lane == 0) {
                    // replica count from word 0, cut t taken with probability needed/remaining
                    const int cap = Kr < Mr ? Kr : Mr;
                    const int Rn = 1 + (int)below(words[0], (uint32_t)cap);
                    int need = Rn - 1, prev = 0, cc = r;
                    for (int t = 1; t <= Mr - 1 && need > 0; ++t) {
                        if (below(words[t], (uint32_t)(Mr - t)) < (uint32_t)need) {
                            ssz[cc++] = (uint32_t)(t - prev);
                            prev = t;
                            --need;
                        }
                    }
                    ssz[cc++] = (uint32_t)(Mr - prev);
                    for (; cc < K; ++cc) ssz[cc] = 0;
                    const uint64_t nr = Rn >= 64 ? bits : (bits & ((1ull << Rn) - 1ull));
                    const uint64_t keep = r >= 64 ? ~0ull : ((1ull << r) - 1ull);
                    rl = (rl & keep) | (r >= 64 ? 0ull : (nr << r));
                    R = r + Rn;
                }
                R = __shfl_sync(0xFFFFFFFFu, R, 0);
                rl = __shfl_sync(0xFFFFFFFFu, rl, 0);
            }
        }
        __syncwarp();
        for (int i = lane; i < M; i += 32) out_perm[i] = (uint16_t)child[i];
        for (int i = lane; i < K; i += 32) cs[i] = (uint16_t)ssz[i];
        if (lane == 0) { dst.nclus[s] = (uint8_t)R; dst.roles[s] = rl; }
        __syncwarp();
    }
}

// 1D launch helpers
inline unsigned grid_for(size_t n, int threads, size_t cap = 152 * 32)
{
    size_t b = (n + threads - 1) / threads;
    if (b > cap) b = cap;
    return (unsigned)(b ? b : 1);
}

}  // namespace

cudaError_t launch_tables(const e2_ctx *c)
{
    const size_t total = (size_t)c->dm.V * c->dm.M * 2 * c->dm.LS;
    tables_kernel<<<grid_for(total, 256), 256, 0, c->stream>>>(c->dm, c->rate, c->bw, c->mem, c->rate_cpu, c->bw_cpu,
                                                                c->mem_cpu, c->prof, c->leaf);
    const size_t vm = (size_t)c->dm.V * c->dm.M;
    captab_kernel<<<grid_for(vm, 256), 256, 0, c->stream>>>(c->dm, c->rate, c->bw, c->mem, c->rate_cpu, c->bw_cpu,
                                                             c->mem_cpu, c->prof, c->cap, c->capg, c->cpb);
    c->launches += 2;
    if (c->dm.layered) {
        const size_t lt = (size_t)c->dm.V * c->dm.M * 2 * c->dm.N * c->dm.N;
        layered_tables_kernel<<<grid_for(lt, 256), 256, 0, c->stream>>>(c->dm, c->rate, c->bw, c->mem, c->prof,
                                                                         c->psum, c->lcost);
        ++c->launches;
    }
    return cudaGetLastError();
}

cudaError_t launch_tau(const e2_ctx *c)
{
    const size_t total = (size_t)c->dm.V * c->dm.M * c->dm.M;
    tau_kernel<<<grid_for(total, 256), 256, 0, c->stream>>>(c->dm, c->link_bw, c->cong, c->prof, c->tau, c->tau_lb);
    ++c->launches;
    return cudaGetLastError();
}

cudaError_t launch_redraw(const e2_ctx *c, uint64_t seed, uint32_t gen)
{
    const size_t total = (size_t)c->dm.M * c->dm.M;
    redraw_kernel<<<grid_for(total, 256), 256, 0, c->stream>>>(c->dm.M, seed, gen, c->cong_lo, c->cong_hi, c->cong);
    ++c->launches;
    return cudaGetLastError();
}

cudaError_t launch_validate(const e2_ctx *c, const DevPop &p)
{
    validate_kernel<<<(c->dm.P + 127) / 128, 128, 0, c->stream>>>(c->dm, p, c->err);
    ++c->launches;
    return cudaGetLastError();
}

cudaError_t launch_init(const e2_ctx *c, const DevPop &p, uint64_t seed)
{
    init_kernel<<<(c->dm.P + 31) / 32, 32, 0, c->stream>>>(c->dm, p, seed);
    ++c->launches;
    return cudaGetLastError();
}

// Duplicate flags, then ranks; the elites go to slots [0, Q) of dst.
cudaError_t launch_elites(const e2_ctx *c, const DevPop &p, const DevPop &dst)
{
    const unsigned blocks = (unsigned)(((size_t)c->dm.P * 32 + 255) / 256);
    const bool table = c->dm.P >= kDupTableFrom;
    if (table) {
        const unsigned tsize = dup_table_size(c->dm.P);
        cudaError_t e = cudaMemsetAsync(c->dup_key, 0xFF, sizeof(uint64_t) * tsize, c->stream);
        if (e == cudaSuccess) e = cudaMemsetAsync(c->dup_idx, 0x7F, sizeof(int32_t) * tsize, c->stream);
        if (e != cudaSuccess) return e;
        dup_insert_kernel<<<(unsigned)((c->dm.P + 255) / 256), 256, 0, c->stream>>>(
            c->dm.P, c->hash, reinterpret_cast<unsigned long long *>(c->dup_key), c->dup_idx, tsize - 1);
        dup_lookup_kernel<<<blocks, 256, 0, c->stream>>>(c->dm, p, c->hash,
                                                         reinterpret_cast<const unsigned long long *>(c->dup_key),
                                                         c->dup_idx, tsize - 1, c->dup);
    } else {
        dup_kernel<<<blocks, 256, 0, c->stream>>>(c->dm, p, c->fit, c->hash, c->dup);
    }
    if (c->dm.Q > 0) {
        elite_select_kernel<<<1, kSelThreads, 0, c->stream>>>(c->dm.P, c->dm.Q, c->fit, c->dup, c->elite_ctl,
                                                              c->elite_cand);
        elite_cand_rank_kernel<<<152 * 4, 256, 0, c->stream>>>(c->dm, c->fit, c->elite_ctl, c->elite_cand,
                                                               c->elite, c->elite_fit, p, dst);
        rank_kernel<<<blocks, 256, 0, c->stream>>>(c->dm, c->fit, c->dup, c->elite, c->elite_fit, p, dst,
                                                   c->elite_ctl);
    }
    c->launches += (table ? 2 : 1) + (c->dm.Q > 0 ? 3 : 0);
    return cudaGetLastError();
}

cudaError_t launch_ga(const e2_ctx *c, const DevPop &src, const DevPop &dst, uint64_t seed, uint32_t gen,
                      cudaStream_t st)
{
    if (c->dm.P <= c->dm.Q) return cudaSuccess;              // no children
    GaThr thr{c->thr_cx, c->thr_half, c->thr_mut, c->thr_k1, c->thr_k2, c->thr_k3};
    const size_t per_warp = 4 * (4 * (size_t)c->dm.M + 64);
    int nw = 8;
    while (nw > 1 && (size_t)nw * per_warp > 48 * 1024) nw >>= 1;
    if ((size_t)nw * per_warp > 48 * 1024) {
        const cudaError_t e = cudaFuncSetAttribute(ga_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                   (int)((size_t)nw * per_warp));
        if (e != cudaSuccess) return e;
    }
    const long long blocks = ((long long)(c->dm.P - c->dm.Q) + nw - 1) / nw;
    ga_kernel<<<(unsigned)(blocks < 152 * 64 ? blocks : 152 * 64), 32 * nw, (size_t)nw * per_warp, st>>>(
        c->dm, src, dst, c->fit, seed, gen, thr);
    ++c->launches;
    return cudaGetLastError();
}

// The generation step: the children (which need only the fitness) on the side
// stream, concurrently with the duplicate test and the ranks (which copy the
// elites) on the context's stream; the context's stream then waits for the
// children.
cudaError_t launch_step(const e2_ctx *c, const DevPop &src, const DevPop &dst, uint64_t seed, uint32_t gen)
{
    cudaError_t e = cudaEventRecord(c->ev_fork, c->stream);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(c->side, c->ev_fork, 0);
    if (e == cudaSuccess) e = launch_ga(c, src, dst, seed, gen, c->side);
    if (e == cudaSuccess) e = cudaEventRecord(c->ev_join, c->side);
    if (e == cudaSuccess) e = launch_elites(c, src, dst);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(c->stream, c->ev_join, 0);
    return e;
}

cudaError_t find_ga_node(cudaGraph_t graph, cudaGraphNode_t *node)
{
    *node = nullptr;
    size_t n = 0;
    cudaError_t e = cudaGraphGetNodes(graph, nullptr, &n);
    if (e != cudaSuccess) return e;
    cudaGraphNode_t nodes[64];
    if (n > 64) return cudaErrorInvalidValue;
    e = cudaGraphGetNodes(graph, nodes, &n);
    if (e != cudaSuccess) return e;
    for (size_t i = 0; i < n; ++i) {
        cudaGraphNodeType t;
        if ((e = cudaGraphNodeGetType(nodes[i], &t)) != cudaSuccess) return e;
        if (t != cudaGraphNodeTypeKernel) continue;
        cudaKernelNodeParams p{};
        if ((e = cudaGraphKernelNodeGetParams(nodes[i], &p)) != cudaSuccess) return e;
        if (p.func == reinterpret_cast<void *>(ga_kernel)) {
            *node = nodes[i];
            return cudaSuccess;
        }
    }
    return cudaErrorInvalidValue;
}

cudaError_t set_ga_node(const e2_ctx *c, cudaGraphExec_t exec, cudaGraphNode_t node, const DevPop &src,
                        const DevPop &dst, uint64_t seed, uint32_t gen)
{
    cudaKernelNodeParams p{};
    cudaError_t e = cudaGraphKernelNodeGetParams(node, &p);     // launch shape as recorded
    if (e != cudaSuccess) return e;
    Dims dm = c->dm;
    DevPop s = src, d = dst;
    const double *fit = c->fit;
    GaThr thr{c->thr_cx, c->thr_half, c->thr_mut, c->thr_k1, c->thr_k2, c->thr_k3};
    void *args[] = {&dm, &s, &d, &fit, &seed, &gen, &thr};
    p.kernelParams = args;
    p.extra = nullptr;
    return cudaGraphExecKernelNodeSetParams(exec, node, &p);
}

}  // namespace e2
