// dp_eval.cu -- population fitness: DP_Pipe per replica (Alg. 1, Eq. 1-2),
// the decode batch sweep (Alg. 2), and the objective (Eq. 3-5).
//
// One CTA evaluates one (genome, replica slot).  With identical blocks
// (Sec. 3.2: the premise that lets the paper fix the node order) a stage's time
// depends only on its device, its block count n and whether it is the master,
// so the replica's costs fit in two rows per device, l_k(n) and l_k^head(n),
// staged in shared memory as 64-bit keys (non-negative doubles order like their
// bit patterns).
//
// Band form of Eq. 1.  Device k can take at most W = N - m + 1 blocks.  Let
// D_k[r] = DP(i = r + k - 1, k), r in [0, W).  Then
//     D_1[r] = l_1(r + 1)                                         (Eq. 2)
//     D_k[r] = min_{s in [0, r]} max(D_{k-1}[s], l_k(r - s + 1), tau_k)   (Eq. 1)
// where s = j - (k - 1) indexes the split.  D_{k-1}[s] is non-decreasing in s
// (one more block never lowers the best bottleneck when blocks are identical)
// and l_k(r - s + 1) is non-increasing in s, so max(D_{k-1}[s], l_k(.)) falls
// then rises: its minimum sits at the crossover s0 = first s with
// D_{k-1}[s] >= l_k(r - s + 1) and equals min(l_k(r - s0 + 2), D_{k-1}[s0]).
// A bisection over s finds s0, so a cell costs O(log W) probes instead of the
// O(W) scan, with bit-identical values (min and max are exact).
//
// Tie rule.  The oracle keeps the smallest split j attaining the minimum.  The
// set of minimisers is {s : D_{k-1}[s] <= D and l_k(r-s+1) <= D} (tau <= D
// always), an interval whose first element is the first s with
// l_k(r-s+1) <= D.  So the traceback needs only the cell value D and the cost
// row: n_k = largest n <= r + 1 with l_k(n) <= D.
//
// Masters.  Columns k < mu do not involve the master and are shared by every
// mu (computed once by the CTA).  Warps take masters mu = w+1, w+1+NW, ... and
// run columns mu..m in private ping-pong buffers; the last column needs only
// its final cell.  mu* = the smallest mu with the least bottleneck (the
// oracle's first-wins argmin).  The CTA then recomputes mu*'s columns into the
// shared column store for the traceback.
#include "e2ga_internal.cuh"

namespace e2 {

namespace {

// D_k[r] for one cell (see the header comment).
__device__ __forceinline__ uint64_t dp_cell(const uint64_t *__restrict__ prev,
                                            const uint64_t *__restrict__ row, uint64_t tau, int r)
{
    int lo = 0, hi = r + 1;
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (prev[mid] >= row[r - mid]) hi = mid;
        else lo = mid + 1;
    }
    uint64_t h = kInfKey;
    if (lo <= r) h = prev[lo];
    if (lo >= 1) h = umin64(h, row[r - lo + 1]);
    return umax64(h, tau);
}

__device__ __forceinline__ int warp_sum(int x)
{
#pragma unroll
    for (int o = 16; o; o >>= 1) x += __shfl_xor_sync(0xFFFFFFFFu, x, o);
    return x;
}

// Candidates (mu, k, i, j) the plain recurrence examines for one DP run:
// m * (N + sum_{k=2..m} (N-k+1)(N-k+2)/2).
__device__ __forceinline__ unsigned long long paper_candidates(int m, int N)
{
    const unsigned long long a = (unsigned long long)(N - m + 1), b = (unsigned long long)(N - 1);
    unsigned long long s = 0;
    if (m >= 2) s = (b * (b + 1) * (b + 2) - (a - 1) * a * (a + 1)) / 6;
    return (unsigned long long)m * ((unsigned long long)N + s);
}

// Bisection probes of one full column of W cells: sum_{n=1..W} (floor(log2 n) + 1).
__device__ __forceinline__ unsigned long long column_probes(int W)
{
    const int L = 31 - __clz(W);
    return (unsigned long long)W + (unsigned long long)(W + 1) * L - (2ull << L) + 2ull;
}

}  // namespace

// Shared-memory bytes for the largest replica the problem allows.
size_t dp_smem_bytes(int M, int N, int threads)
{
    const int NW = threads / 32;
    size_t best = 0;
    const int mmax = M < N ? M : N;
    for (int m = 1; m <= mmax; ++m) {
        const size_t W = (size_t)(N - m + 1);
        const size_t u64s = 4 * (size_t)m * W + (size_t)(NW + 1) * W + (size_t)m;
        const size_t bytes = u64s * 8 + (size_t)m * (3 * sizeof(int)) + (size_t)m * sizeof(uint16_t) + 16;
        if (bytes > best) best = bytes;
    }
    return (best + 15) & ~(size_t)15;
}

namespace {

__device__ __forceinline__ void bar_named(int id, int nthreads)
{
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

__device__ __forceinline__ double warp_sum_d(double x)
{
#pragma unroll
    for (int o = 16; o; o >>= 1) x += __shfl_xor_sync(0xFFFFFFFFu, x, o);
    return x;
}

}  // namespace

// Pre-pass, one warp per (genome, replica slot): the replica's offset in the
// ordering chromosome, and the set of variants worth a DP run (bit i = variant
// 0 for a prefill replica, variant i+1 for a decode replica):
//  * memory: with identical blocks a partition with master mu exists iff every
//    device holds >= 1 block and the capacities, capped at W = N - m + 1, add
//    up to N (exact);
//  * decode latency: Lambda >= sum of link times + sum_k n_k c_k (c_k the
//    per-block time, the head only adds), whose least value puts one block on
//    each device and the other N - m on the cheapest devices up to their
//    capacity.  A variant whose bound misses Min_TPS fails whatever partition
//    the DP returns; the 1e-9 margin exceeds the rounding of every sum here.
// Also a heavy-first ordering key: 0 empty slot, 1 nothing to run, else a
// log-scale bucket of m * W * (variants to run).
__global__ void __launch_bounds__(128) variant_kernel(Dims dm, Tables tb, DevPop pop, SlotInfo si, unsigned *bins,
                                                      unsigned long long *stats)
{
    __shared__ uint16_t s_dev[4][kMaxReplicaDevices];
    __shared__ int s_c0[4][kMaxReplicaDevices], s_c1[4][kMaxReplicaDevices];
    __shared__ uint64_t s_cb[4][kMaxReplicaDevices];
    const int slot = (int)((blockIdx.x * blockDim.x + threadIdx.x) >> 5), lane = threadIdx.x & 31;
    const int K = dm.K, M = dm.M, N = dm.N;
    if (slot >= dm.P * K) return;
    const int g = slot / K, c = slot - g * K;
    const int R = pop.nclus[g];
    int key = 0, off = 0, n_mem = 0, n_lat = 0;
    uint64_t mask = 0;
    if (c < R) {
        const uint16_t *sz = pop.sizes + (size_t)g * K;
        off = warp_sum(lane < c ? sz[lane] : 0) + warp_sum(lane + 32 < c ? sz[lane + 32] : 0);
        const int m = sz[c];
        const int role = (int)((pop.roles[g] >> c) & 1ull);
        key = 1;
        if (m <= N) {
            const int W = N - m + 1;
            const int wl = threadIdx.x >> 5;
            uint16_t *sdev = s_dev[wl];
            int *sc0 = s_c0[wl], *sc1 = s_c1[wl];
            uint64_t *scb = s_cb[wl];      // per-block times as order-preserving keys
            const uint16_t *devs = pop.perm + (size_t)g * M + off;
            for (int k = lane; k < m; k += 32) sdev[k] = devs[k];
            __syncwarp();
            const int nv = role ? dm.b_max : 1;
            for (int i = 0; i < nv; ++i) {
                const int v = role ? i + 1 : 0;
                const int32_t *cap = tb.cap + (size_t)v * M * 2;
                int s0 = 0, z = 0;
                for (int k = lane; k < m; k += 32) {
                    const int d = sdev[k];
                    const int c0 = min(cap[d * 2], W), c1 = min(cap[d * 2 + 1], W);
                    sc0[k] = c0;
                    sc1[k] = c1;
                    s0 += c0;
                    z += c0 == 0;
                }
                s0 = warp_sum(s0);
                z = warp_sum(z);
                __syncwarp();
                bool ok = false;
                for (int k = lane; k < m && !ok; k += 32)
                    ok = (z - (sc0[k] == 0)) == 0 && sc1[k] >= 1 && s0 - sc0[k] + sc1[k] >= N;
                if (!__any_sync(0xFFFFFFFFu, ok)) { ++n_mem; continue; }
                if (role && dm.min_tps > 0.0) {
                    const double *cpb = tb.cpb + (size_t)v * M;
                    const double *tau = tb.tau + (size_t)v * M * M;
                    for (int k = lane; k < m; k += 32) scb[k] = dkey(cpb[sdev[k]]);
                    __syncwarp();
                    double part = 0.0;
                    for (int k = lane; k < m; k += 32) {
                        const uint64_t ck = scb[k];
                        long long before = 0;            // capacity of the cheaper devices
                        for (int j = 0; j < m; ++j) {
                            const uint64_t cj = scb[j];
                            if (cj < ck || (cj == ck && j < k)) before += sc0[j] - 1;
                        }
                        const long long ek = sc0[k] - 1;
                        const long long room = (long long)(N - m) - before;
                        const long long take = room <= 0 ? 0 : (room < ek ? room : ek);
                        part += keyd(ck) * (double)(1 + take);
                        if (k >= 1) part += tau[(size_t)sdev[k - 1] * M + sdev[k]];
                    }
                    const double lb = warp_sum_d(part) * (1.0 - 1e-9);
                    if (lb > 0.0 && 1.0 / lb < dm.min_tps) { ++n_lat; continue; }
                }
                mask |= 1ull << i;
            }
            if (mask) {
                const float est = (float)m * (float)W * (float)__popcll(mask);
                const int k2 = 2 + (int)(8.0f * __log2f(1.0f + est));
                key = k2 < kOrderBins - 1 ? k2 : kOrderBins - 1;
            }
        }
    }
    if (lane == 0) {
        si.off[slot] = off;
        si.mask[slot] = mask;
        si.key[slot] = (uint8_t)key;
        atomicAdd(&bins[key], 1u);
        if (n_mem) atomicAdd(&stats[kStPrecheck], (unsigned long long)n_mem);
        if (n_lat) atomicAdd(&stats[kStTpsPruned], (unsigned long long)n_lat);
    }
}

// Exclusive scan of the bins in descending key order (heaviest first).
__global__ void order_scan_kernel(unsigned *bins)
{
    __shared__ unsigned s[kOrderBins];
    const int t = threadIdx.x;
    s[t] = bins[kOrderBins - 1 - t];
    __syncthreads();
    for (int o = 1; o < kOrderBins; o <<= 1) {
        const unsigned v = t >= o ? s[t - o] : 0u;
        __syncthreads();
        s[t] += v;
        __syncthreads();
    }
    const unsigned incl = s[t];
    const unsigned cnt = bins[kOrderBins - 1 - t];
    __syncthreads();
    bins[kOrderBins - 1 - t] = incl - cnt;
}

__global__ void order_scatter_kernel(int total, const uint8_t *keys, unsigned *cursor, int *order)
{
    for (int s = blockIdx.x * blockDim.x + threadIdx.x; s < total; s += gridDim.x * blockDim.x)
        order[atomicAdd(&cursor[keys[s]], 1u)] = s;
}

// One CTA per (genome, replica slot), heaviest first.  Per variant:
//  1. stage the cost rows l_k(n), l_k^head(n) and the link times;
//  2. exact memory check per master;
//  3. prefix columns F_k (no master, devices 1..k) on warps 0-1 and suffix
//     columns G_k (no master, devices k..m) on warps 2-3, concurrently:
//        F_k[r] = min_s max(F_{k-1}[s], l_k(r-s+1), tau_k)
//        G_k[r] = min_s max(G_{k+1}[s], l_k(r-s+1), tau_{k+1})
//  4. master mu: the prefix holds a extra blocks, the suffix b, the master
//     W - a - b, so with H_mu[c] = min_{a+b=c} max(F_{mu-1}[a], G_{mu+1}[b])
//        V_mu = max(tau_mu, tau_{mu+1}, min_c max(H_mu[c], l_mu^head(W - c)))
//     (F_0 and G_{m+1} are the empty stage: 0 at index 0, +inf after);
//  5. mu* = smallest mu with the least V_mu; its prefix columns D_k (master
//     at mu*) are recomputed for the traceback;
//  6. traceback with the smallest-split rule (n_k = number of n <= r+1 with
//     l_k(n) <= D, counted with warp ballots) and Lambda in pipeline order.
// Every value is a min/max of the same leaf and link times the oracle uses,
// so V, mu*, the partition and Lambda are bit-identical to Alg. 1.
__global__ void __launch_bounds__(128) dp_eval_kernel(Dims dm, Tables tb, DevPop pop, EvalOut out,
                                                      const int *order, SlotInfo si)
{
    extern __shared__ __align__(16) unsigned char smem[];
    __shared__ int s_off, s_m, s_role, s_S0, s_Z, s_mu, s_done;
    __shared__ uint64_t s_V;
    __shared__ double s_L;
    __shared__ uint64_t s_wV[4];
    __shared__ int s_wMu[4];

    const int K = dm.K, M = dm.M, N = dm.N;
    const int slot = order[blockIdx.x];
    const int g = slot / K, c = slot - g * K;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5, NW = blockDim.x >> 5;
    const size_t gk = (size_t)g * K + c;
    if (c >= pop.nclus[g]) {
        if (tid == 0) {
            out.master[gk] = -1; out.bsel[gk] = -1;
            out.T[gk] = keyd(kInfKey); out.L[gk] = keyd(kInfKey);
        }
        return;
    }
    const int off = si.off[slot], m = pop.sizes[gk];
    const int role = (int)((pop.roles[g] >> c) & 1ull);
    uint64_t vmask = si.mask[slot];
    int16_t *lay_out = out.layers + (size_t)g * M + off;

    unsigned long long st_runs = 0, st_cells = 0, st_probes = 0;
    bool served = false;
    int served_v = -1;

    if (m <= N && vmask) {
        const int W = N - m + 1;
        uint64_t *leaf0 = reinterpret_cast<uint64_t *>(smem);   // [m][W] l_k(n)
        uint64_t *leaf1 = leaf0 + (size_t)m * W;                // [m][W] l_k^head(n)
        uint64_t *Fst = leaf1 + (size_t)m * W;                  // [m][W] prefix / traceback columns
        uint64_t *Gst = Fst + (size_t)m * W;                    // [m][W] suffix columns
        uint64_t *Hb = Gst + (size_t)m * W;                     // [NW][W] per-warp convolution
        uint64_t *delta = Hb + (size_t)NW * W;                  // [W] the empty stage
        uint64_t *tauk = delta + W;                             // [m] tauk[k] = link (k-1) -> k
        int *cnt0 = reinterpret_cast<int *>(tauk + m);          // [m]
        int *cnt1 = cnt0 + m;                                   // [m]
        int *nk = cnt1 + m;                                     // [m]
        uint16_t *devs = reinterpret_cast<uint16_t *>(nk + m);  // [m]

        for (int k = tid; k < m; k += blockDim.x) devs[k] = pop.perm[(size_t)g * M + off + k];
        for (int r = tid; r < W; r += blockDim.x) delta[r] = r ? kInfKey : 0ull;
        __syncthreads();

        // column accessors (1-based device index k)
        auto colF = [&](int k) -> const uint64_t * {
            return k == 0 ? delta : k == 1 ? leaf0 : Fst + (size_t)(k - 1) * W;
        };
        auto colG = [&](int k) -> const uint64_t * {
            return k == m + 1 ? delta : k == m ? leaf0 + (size_t)(m - 1) * W : Gst + (size_t)(k - 1) * W;
        };

        const unsigned long long cprobe = column_probes(W);
        const unsigned long long lprobe = 32 - __clz(W);
        while (vmask && !served) {
            const int bit = 63 - __clzll((long long)vmask);          // highest batch first
            vmask &= ~(1ull << bit);
            const int v = role ? bit + 1 : 0;
            // ---- 1. capacities, link times and cost rows of this variant
            for (int k = tid; k < m; k += blockDim.x) {
                const size_t vd = (size_t)v * M + devs[k];
                const int c0 = tb.cap[vd * 2], c1 = tb.cap[vd * 2 + 1];
                cnt0[k] = c0 < W ? c0 : W;
                cnt1[k] = c1 < W ? c1 : W;
                tauk[k] = k ? dkey(tb.tau[((size_t)v * M + devs[k - 1]) * M + devs[k]]) : 0ull;
            }
            for (int e = tid; e < m * W; e += blockDim.x) {
                const int k = e / W, n = e - k * W;
                const double *base = tb.leaf + ((size_t)v * M + devs[k]) * 2 * dm.LS;
                leaf0[e] = dkey(base[n]);
                leaf1[e] = dkey(base[dm.LS + n]);
            }
            __syncthreads();
            // ---- 2. masters the memory allows (the pre-pass guarantees one)
            if (wid == 0) {
                int s = 0, z = 0;
                for (int k = lane; k < m; k += 32) { s += cnt0[k]; z += cnt0[k] == 0; }
                s = warp_sum(s); z = warp_sum(z);
                if (lane == 0) { s_S0 = s; s_Z = z; }
            }
            __syncthreads();
            const int S0 = s_S0, Z = s_Z;
            auto mu_ok = [&](int mu) {
                const int k = mu - 1;
                return (Z - (cnt0[k] == 0)) == 0 && cnt1[k] >= 1 && S0 - cnt0[k] + cnt1[k] >= N;
            };
            ++st_runs;
            // ---- 3. prefix columns (warps 0-1) and suffix columns (warps 2-3)
            if (wid < 2) {
                for (int k = 2; k <= m - 1; ++k) {
                    const uint64_t *prev = colF(k - 1), *row = leaf0 + (size_t)(k - 1) * W;
                    const uint64_t t = tauk[k - 1];
                    uint64_t *cur = Fst + (size_t)(k - 1) * W;
                    for (int r = tid; r < W; r += 64) cur[r] = dp_cell(prev, row, t, r);
                    bar_named(1, 64);
                }
            } else {
                for (int k = m - 1; k >= 2; --k) {
                    const uint64_t *prev = colG(k + 1), *row = leaf0 + (size_t)(k - 1) * W;
                    const uint64_t t = tauk[k];
                    uint64_t *cur = Gst + (size_t)(k - 1) * W;
                    for (int r = tid - 64; r < W; r += 64) cur[r] = dp_cell(prev, row, t, r);
                    bar_named(2, 64);
                }
            }
            if (tid == 0 && m >= 3) {
                st_cells += 2ull * (m - 2) * W;
                st_probes += 2ull * (m - 2) * cprobe;
            }
            __syncthreads();
            // ---- 4. one master per warp at a time
            uint64_t bestV = kInfKey;
            int bestMu = 0x7FFFFFFF;
            unsigned long long w_cells = 0, w_probes = 0;
            uint64_t *H = Hb + (size_t)wid * W;
            for (int mu = wid + 1; mu <= m; mu += NW) {
                if (!mu_ok(mu)) continue;
                const uint64_t *P = colF(mu - 1), *S = colG(mu + 1);
                for (int r = lane; r < W; r += 32) H[r] = dp_cell(P, S, 0ull, r);
                __syncwarp();
                uint64_t V = dp_cell(H, leaf1 + (size_t)(mu - 1) * W, 0ull, W - 1);
                if (mu >= 2) V = umax64(V, tauk[mu - 1]);
                if (mu <= m - 1) V = umax64(V, tauk[mu]);
                __syncwarp();
                w_cells += W + 1;
                w_probes += cprobe + lprobe;
                if (V < bestV) { bestV = V; bestMu = mu; }
            }
            if (lane == 0) { s_wV[wid] = bestV; s_wMu[wid] = bestMu; st_cells += w_cells; st_probes += w_probes; }
            __syncthreads();
            if (tid == 0) {
                uint64_t V = kInfKey;
                int mu = 0x7FFFFFFF;
                for (int w = 0; w < NW; ++w)
                    if (s_wV[w] < V || (s_wV[w] == V && s_wMu[w] < mu)) { V = s_wV[w]; mu = s_wMu[w]; }
                s_V = V; s_mu = mu;
            }
            __syncthreads();
            const uint64_t V = s_V;
            const int mus = s_mu;
            if (V >= kInfKey) continue;      // cannot happen after the exact memory check
            // ---- 5. mu*'s prefix columns, for the traceback
            auto rowk = [&](int k) -> const uint64_t * { return (k == mus ? leaf1 : leaf0) + (size_t)(k - 1) * W; };
            auto colD = [&](int k) -> const uint64_t * {
                if (k == 1) return mus == 1 ? leaf1 : leaf0;
                return Fst + (size_t)(k - 1) * W;
            };
            for (int k = (mus > 2 ? mus : 2); k <= m - 1; ++k) {
                const uint64_t *prev = colD(k - 1), *row = rowk(k);
                const uint64_t t = tauk[k - 1];
                uint64_t *cur = Fst + (size_t)(k - 1) * W;
                for (int r = tid; r < W; r += blockDim.x) cur[r] = dp_cell(prev, row, t, r);
                __syncthreads();
                if (tid == 0) { st_cells += W; st_probes += cprobe; }
            }
            // ---- 6. traceback (smallest split on ties) and Lambda in pipeline order
            if (wid == 0) {
                int r = W - 1;
                uint64_t D = V;
                for (int k = m; k >= 2; --k) {
                    const uint64_t *row = rowk(k);
                    int n = 0;                                    // #{n <= r+1 : l_k(n) <= D}
                    for (int base = 0; base <= r; base += 32) {
                        const int p = base + lane;
                        const unsigned b = __ballot_sync(0xFFFFFFFFu, p <= r && row[p] <= D);
                        n += __popc(b);
                        if (b != 0xFFFFFFFFu) break;
                    }
                    if (lane == 0) nk[k - 1] = n;
                    r = r + 1 - n;
                    D = colD(k - 1)[r];
                }
                if (lane == 0) {
                    nk[0] = r + 1;
                    double lam = keyd(rowk(1)[nk[0] - 1]);
                    for (int k = 2; k <= m; ++k) {
                        lam = lam + keyd(tauk[k - 1]);
                        lam = lam + keyd(rowk(k)[nk[k - 1] - 1]);
                    }
                    s_L = lam;
                    s_done = (!role) || (1.0 / lam >= dm.min_tps);
                }
            }
            __syncthreads();
            if (s_done) {
                for (int k = tid; k < m; k += blockDim.x) lay_out[k] = (int16_t)nk[k];
                if (tid == 0) {
                    out.master[gk] = (int16_t)(mus - 1);
                    out.bsel[gk] = (int16_t)v;
                    out.T[gk] = keyd(V);
                    out.L[gk] = s_L;
                }
                served = true;
                served_v = v;
            }
            __syncthreads();
        }
    }
    if (!served) {
        for (int k = tid; k < m; k += blockDim.x) lay_out[k] = -1;
        if (tid == 0) {
            out.master[gk] = -1; out.bsel[gk] = -1;
            out.T[gk] = keyd(kInfKey); out.L[gk] = keyd(kInfKey);
        }
    }
    // per-CTA tallies
    if (lane == 0 && (st_cells | st_probes)) {
        atomicAdd(&out.stats[kStCells], st_cells);
        atomicAdd(&out.stats[kStProbes], st_probes);
    }
    if (tid == 0) {
        // candidates the plain recurrence examines for the same sweep: every
        // variant from the top down to the accepted one (all of them if none)
        unsigned long long nrun = 0;
        if (m <= N) nrun = served ? (role ? (unsigned long long)(dm.b_max - served_v + 1) : 1ull)
                                  : (role ? (unsigned long long)dm.b_max : 1ull);
        atomicAdd(&out.stats[kStReplicas], 1ull);
        if (st_runs) atomicAdd(&out.stats[kStDpRuns], st_runs);
        if (nrun) atomicAdd(&out.stats[kStPaper], nrun * paper_candidates(m, N));
        if (served) atomicAdd(&out.stats[kStServed], 1ull);
    }
}

// Objective, one thread per genome (Sec. 3.3).  PS and DS are summed over the
// serving replicas of each role in ascending replica order, then Eq. 3
// (bottleneck phase), Eq. 4 (backlog) and Eq. 5 (waiting time).  Also a
// 64-bit fingerprint of the genome for the elites' duplicate test.
__global__ void __launch_bounds__(32) score_kernel(Dims dm, DevPop pop, EvalOut out)
{
    const int g = blockIdx.x * blockDim.x + threadIdx.x;
    if (g >= dm.P) return;
    const int K = dm.K, M = dm.M;
    const int R = pop.nclus[g];
    const uint64_t roles = pop.roles[g];
    double PS = 0.0, DS = 0.0;
    for (int c = 0; c < R; ++c) {
        const int b = out.bsel[(size_t)g * K + c];
        if (b < 0) continue;
        const double T = out.T[(size_t)g * K + c];
        if (((roles >> c) & 1ull) == 0) PS = PS + (double)dm.NP / T;
        else DS = DS + (double)b / T;
    }
    double w = keyd(kInfKey), phase = keyd(kInfKey);
    if (PS != 0.0 && DS != 0.0) {
        const double tp = (double)dm.NP / PS, td = (double)dm.ND / DS;
        phase = tp >= td ? tp : td;                 // Eq. 3
        const double x = phase - dm.t_a;
        const double bn = x > 0.0 ? x : 0.0;        // Eq. 4
        w = bn > 0.0 ? tp + bn : 0.0;               // Eq. 5
    }
    double *f = out.fit + (size_t)g * 4;
    f[0] = w; f[1] = phase; f[2] = PS; f[3] = DS;
    // fingerprint: ordering, grouping, replica count, roles
    uint64_t h = 0x9E3779B97F4A7C15ull;
    auto mix = [&](uint64_t x) { h = (h ^ x) * 0xBF58476D1CE4E5B9ull; h ^= h >> 31; };
    const uint16_t *pp = pop.perm + (size_t)g * M;
    for (int i = 0; i < M; ++i) mix(pp[i]);
    const uint16_t *ss = pop.sizes + (size_t)g * K;
    for (int i = 0; i < R; ++i) mix((uint64_t)ss[i] << 16);
    mix((uint64_t)R << 40);
    mix(roles);
    out.hash[g] = h;
    atomicAdd(&out.stats[kStGenomes], 1ull);
}

cudaError_t configure_eval(size_t smem)
{
    return cudaFuncSetAttribute(dp_eval_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
}

cudaError_t launch_eval(const e2_ctx *c, const DevPop &p)
{
    Tables tb{c->rate, c->bw, c->mem, c->prof, c->leaf, c->tau, c->cap, c->cpb};
    EvalOut out{c->fit, c->layers, c->master, c->bsel, c->T, c->L, c->hash, c->stats};
    const long long blocks = (long long)c->dm.P * c->dm.K;
    SlotInfo si{c->slot_off, c->slot_mask, c->slot_key};
    cudaError_t e = cudaMemsetAsync(c->order_bins, 0, sizeof(unsigned) * kOrderBins, c->stream);
    if (e != cudaSuccess) return e;
    const unsigned gb = (unsigned)((blocks + 255) / 256 < 1024 ? (blocks + 255) / 256 : 1024);
    variant_kernel<<<(unsigned)((blocks * 32 + 127) / 128), 128, 0, c->stream>>>(c->dm, tb, p, si, c->order_bins, c->stats);
    order_scan_kernel<<<1, kOrderBins, 0, c->stream>>>(c->order_bins);
    order_scatter_kernel<<<gb, 256, 0, c->stream>>>((int)blocks, c->slot_key, c->order_bins, c->order);
    dp_eval_kernel<<<(unsigned)blocks, c->dp_threads, c->dp_smem, c->stream>>>(c->dm, tb, p, out, c->order, si);
    score_kernel<<<(c->dm.P + 31) / 32, 32, 0, c->stream>>>(c->dm, p, out);
    return cudaGetLastError();
}

}  // namespace e2
