// dp_eval.cu -- population fitness: DP_Pipe per replica (Alg. 1, Eq. 1-2),
// the decode batch sweep (Alg. 2), and the objective (Eq. 3-5).
//
// Work is split over four or five kernels per evaluation: a pre-pass that
// decides, per (genome, replica slot, variant), whether a DP run can matter
// (memory and latency bounds) and counts and orders the surviving runs; a
// scatter that writes them into one work list; persistent DP CTAs that drain
// the list (two launches where the replica sizes fall into two shared-memory
// classes); and a warp per genome (a block per genome for a wide role search)
// that picks each replica's answer and scores the genome.
//
// With identical blocks (Sec. 3.2: the premise that lets the paper fix the
// node order) a stage's time depends only on its device, its block count n and
// whether it is the master, so the replica's costs fit in two rows per device,
// l_k(n) and l_k^head(n), staged in shared memory as 32-bit order keys (exact
// ranks of the float64 times, built in ranks.cu).
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
// O(W) scan, with bit-identical values (min and max are exact); and the
// crossover of cell r + 1 is that of cell r or one more, so a thread that owns
// a span of cells bisects only for the first (dp_span).
//
// Tie rule.  The oracle keeps the smallest split j attaining the minimum.  The
// set of minimisers is {s : D_{k-1}[s] <= D and l_k(r-s+1) <= D} (tau <= D
// always), an interval whose first element is the first s with
// l_k(r-s+1) <= D.  So the traceback needs only the cell value D and the cost
// row: n_k = largest n <= r + 1 with l_k(n) <= D.
//
// Masters.  Alg. 1 reruns the whole table for every master mu.  Here the
// master-free prefix columns F_k (devices 1..k) and suffix columns G_k
// (devices k..m) are computed once per run, and each master's bottleneck
// follows from F_{mu-1}, G_{mu+1} and the master's head row (dp_eval_body,
// step 4).  mu* = the smallest mu with the least bottleneck (the oracle's
// first-wins argmin); its columns are recomputed for the traceback.
#include "e2ga_internal.cuh"
#include "dp_span.cuh"

namespace e2 {

namespace {

// Candidates (mu, k, i, j) the plain recurrence examines for one DP run:
// m * (N + sum_{k=2..m} (N-k+1)(N-k+2)/2).
__device__ __forceinline__ unsigned long long paper_candidates(int m, int N)
{
    const unsigned long long a = (unsigned long long)(N - m + 1), b = (unsigned long long)(N - 1);
    unsigned long long s = 0;
    if (m >= 2) s = (b * (b + 1) * (b + 2) - (a - 1) * a * (a + 1)) / 6;
    return (unsigned long long)m * ((unsigned long long)N + s);
}

// Probes of one column of W cells split into contiguous spans over T = 32,
// 64 or 128 threads (index 0, 1, 2): per span the bisection of its first cell
// (floor(log2(r + 1)) + 1 probes for cell r), then one per further cell.
__constant__ uint16_t c_span_probes[3][E2_MAX_BLOCKS + 1];

}  // namespace

// Shared-memory bytes for the largest replica the problem allows, with keys of
// key_bytes bytes.
size_t dp_smem_bytes(int M, int N, int threads, int key_bytes, bool spill)
{
    size_t best = 0;
    const int mmax = M < N ? M : N;
    for (int m = 1; m <= mmax; ++m) {
        const size_t bytes = dp_item_bytes(m, N, threads / 32, key_bytes, spill);
        if (bytes > best) best = bytes;
    }
    return best;
}

namespace {

__device__ __forceinline__ void bar_named(int id, int nthreads)
{
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

}  // namespace

// Shared-memory bytes per warp of the pre-pass (18 bytes per device, rounded
// up to 16 so that every warp's arrays start aligned).
__host__ __device__ __forceinline__ size_t variant_stride(int mcap) { return ((size_t)mcap * 18 + 15) & ~(size_t)15; }

// Per slot: slots with nothing to run get their outputs here (empty slots,
// more devices than blocks, no variant left by the pre-pass).  Every other
// slot contributes one work item per variant to run; items are ordered by
// level (the variant's rank among its replica's variants, largest batch
// first), then by work size (m * W, log scale), largest first.  A replica's
// smaller batches thus come after every replica's larger ones, by which time
// the larger batch has usually been decided: a variant below an accepted one
// is skipped, as the sequential sweep of Alg. 2 would.  The items of DP class
// 0 (size bit 4 clear) take the upper half of the bins, which the descending
// scan places first; a replica's items all share its class.
__device__ __forceinline__ int item_bin(int level, int size)
{
    const int lv = level < 63 ? level : 63;
    return ((size >> 4) ? 0 : kOrderBins) + (63 - lv) * kSizeBins + (size & (kSizeBins - 1));
}

// Pre-pass and work count, one warp per (genome, replica slot).  For each
// variant of the replica (prefill: v = 0; decode: v = 1..b_max, bit v-1) the
// warp decides whether a DP run can matter:
//  * memory: with identical blocks a partition with master mu exists iff every
//    device holds >= 1 block and the capacities, capped at W = N - m + 1, add
//    up to N (exact);
//  * decode latency: Lambda >= sum of link times + sum_k n_k c_k (c_k the
//    per-block time, the head only adds), whose least value puts one block on
//    each device and the other N - m on the cheapest devices up to their
//    capacity.  It is summed in float from times rounded down, every operation
//    rounded toward -inf, so it never exceeds the exact bound; a variant whose
//    bound is above Lambda_max (rounded up to float) fails whatever partition
//    the DP returns.
// Both tests are monotone in the batch: the capacities shrink as b grows (more
// KV memory per block), and the bound is the least of a linear cost whose
// coefficients (per-block and link times) grow with b over a feasible set that
// shrinks with b, when the profile's costs grow with the batch (physical
// profiles do; checked at e2_create).  So the largest batch the memory allows
// is found by a search (the largest batch first, then the smallest, then
// bisection), and the largest the bound keeps by a second search below it;
// every smaller batch is kept.  A failed test is exact (memory) or a proof
// (the bound never exceeds the exact value), so every batch above it fails
// too; rounding can only keep a variant the exact bound would drop, which
// costs a DP run and changes no result.  Other profiles test every batch from
// the largest down, and the first that passes keeps the smaller ones.
// The surviving variants form the slot's mask.  A replica with nothing to run
// (more devices than blocks, no variant left) gets its outputs here, and the
// genome's last replica writes those of its empty slots (a warp on an empty
// slot does nothing else); the others count their work items into the
// ordering bins, which bins_kernel then scans into starting offsets, class 0
// first and heaviest first within a class.
__global__ void __launch_bounds__(64, 20) slot_kernel(Dims dm, Tables tb, DevPop pop, SlotInfo si, EvalOut out,
                                                  unsigned *ctrl)
{
    // per warp: device ids, capacities and per-block times of up to mcap devices
    extern __shared__ __align__(16) unsigned char vsm[];
    const int mcap = dm.M < dm.N ? dm.M : dm.N;
    const int lane = threadIdx.x & 31, wl = threadIdx.x >> 5;
    const int K = dm.K, M = dm.M, N = dm.N;
    const long long slot = (long long)blockIdx.x * (blockDim.x >> 5) + wl;
    if (slot < (long long)dm.P * K) {
        const int g = (int)(slot / K), c = (int)(slot - (long long)g * K);
        // the genome's replica count, sizes and roles, loaded together (all in bounds)
        const uint16_t *sz = pop.sizes + (size_t)g * K;
        const int R = pop.nclus[g];
        const int m_c = sz[c];
        const uint64_t roles = pop.roles[g];
        const int s_lo = lane < c ? sz[lane] : 0, s_hi = lane + 32 < c ? sz[lane + 32] : 0;
        uint64_t mask = 0;
        unsigned long long n_pre = 0, n_tps = 0;
        int m = 0, off = 0, role = 0;
        if (c < R) {
            m = m_c;
            role = (int)((roles >> c) & 1ull);
            off = warp_sum(s_lo) + warp_sum(s_hi);
            if (lane == 0) si.off[slot] = off;
        }
        if (c < R && m <= N) {
            const int W = N - m + 1;
            unsigned char *wbase = vsm + (size_t)wl * variant_stride(mcap);
            uint32_t *scb = reinterpret_cast<uint32_t *>(wbase);          // per-block times (float bits)
            float *stau = reinterpret_cast<float *>(scb + mcap);          // link (k-1) -> k
            int *sc0 = reinterpret_cast<int *>(stau + mcap), *sc1 = sc0 + mcap;
            uint16_t *sdev = reinterpret_cast<uint16_t *>(sc1 + mcap);
            for (int k = lane; k < m; k += 32) sdev[k] = pop.perm[(size_t)g * M + off + k];
            __syncwarp();
            // with the role search, the decode sweep and then the prefill variant
            // (its result goes to bit b_max); otherwise the genome's role only
            const int npass = dm.role_search ? 2 : 1;
            // Stage variant i (capacities, and the per-block and link times
            // when the latency bound applies) and return its memory verdict.
            auto stage = [&](int prole, int i, bool bound) -> bool {
                const int v = prole ? i + 1 : 0;
                const int32_t *cap = tb.cap + (size_t)v * M * 2;
                const float *cpb = tb.cpb + (size_t)v * M;
                const float *tau = tb.tau_lb + (size_t)v * M * M;
                int s0 = 0, z = 0;
                __syncwarp();
                for (int k = lane; k < m; k += 32) {                   // every load of the variant at once
                    const int d = sdev[k];
                    const int c0 = min(cap[d * 2], W), c1 = min(cap[d * 2 + 1], W);
                    if (bound) {
                        scb[k] = __float_as_uint(cpb[d]);               // non-negative: bits order as values
                        stau[k] = k ? tau[(size_t)sdev[k - 1] * M + d] : 0.0f;
                    }
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
                return __any_sync(0xFFFFFFFFu, ok);
            };
            // The latency bound of the staged variant, against Lambda_max.
            auto fast_enough = [&]() -> bool {
                float part = 0.0f;
                for (int k = lane; k < m; k += 32) {
                    const uint32_t ck = scb[k];
                    int before = 0;                  // capacity of the cheaper devices
                    for (int j = 0; j < m; ++j) {
                        const uint32_t cj = scb[j];
                        if (cj < ck || (cj == ck && j < k)) before += sc0[j] - 1;
                    }
                    const int ek = sc0[k] - 1;
                    const int room = (N - m) - before;
                    const int take = room <= 0 ? 0 : (room < ek ? room : ek);
                    part = __fadd_rd(part, __fmul_rd(__uint_as_float(ck), (float)(1 + take)));
                    if (k >= 1) part = __fadd_rd(part, stau[k]);
                }
#pragma unroll
                for (int o = 16; o; o >>= 1) part = __fadd_rd(part, __shfl_xor_sync(0xFFFFFFFFu, part, o));
                return !(part > dm.lam_max_up);                         // 1.0 / Lambda >= Min_TPS possible
            };
            for (int pass = 0; pass < npass; ++pass) {
                const int prole = dm.role_search ? (pass == 0) : role;
                const int nvar = prole ? dm.b_max : 1;
                if (dm.layered) {                           // per-layer profiles: every variant runs (the
                    if (dm.role_search && !prole) mask |= 1ull << dm.b_max;   // tests assume identical blocks)
                    else mask |= nvar >= 64 ? ~0ull : ((1ull << nvar) - 1ull);
                    continue;
                }
                const bool bound = prole && dm.min_tps > 0.0;
                // When the costs grow with the batch both verdicts are monotone,
                // so each is found by a search over the variants: the largest
                // first (it usually decides), then the smallest, then bisection
                // between the largest known pass (lo) and the smallest known
                // failure (hi).  The memory search comes first; the bound then
                // searches the variants the memory allows.  Otherwise each
                // variant is tested from the largest down, and the first that
                // passes both keeps the smaller ones.
                int lo = -1, hi = nvar, next = nvar - 1, staged = -1, bm = -1;
                bool tps = false;
                while (hi - lo > 1) {
                    bool pass = true;
                    if (staged != next) {
                        pass = stage(prole, next, bound);
                        staged = next;
                    }
                    if (tps && pass) pass = fast_enough();
                    if (pass) lo = next;
                    else hi = next;
                    if (!tps && hi - lo <= 1) {                 // the memory search is done
                        bm = lo;
                        if (!bound || bm < 0) break;
                        tps = true;
                        lo = -1;
                        hi = bm + 1;
                        next = bm;
                        continue;
                    }
                    next = !dm.grows ? hi - 1 : lo < 0 ? 0 : (lo + hi) >> 1;
                }
                const int bs = tps ? lo : bm;               // largest variant both tests keep
                n_pre += (unsigned long long)(nvar - 1 - bm);
                n_tps += (unsigned long long)(bm - bs);
                if (bs >= 0) {
                    if (dm.role_search && !prole) mask |= 1ull << dm.b_max;
                    else mask |= (2ull << bs) - 1ull;       // this variant and every smaller batch
                }
            }
        }
        // ---- the slot's outputs or its work count (the genome's last replica
        //      also writes those of its slots past R)
        if (c < R && !mask)                                          // a replica that cannot serve
            for (int k = lane; k < m; k += 32) out.layers[(size_t)g * M + off + k] = -1;
        if (c == R - 1)
            for (int e = R + lane; e < K; e += 32) {
                const size_t es = (size_t)g * K + e;
                out.master[es] = -1; out.bsel[es] = -1;
                out.T[es] = keyd(kInfKey); out.L[es] = keyd(kInfKey);
            }
        if (lane == 0 && c < R) {
            si.mask[slot] = mask;
            si.best[slot] = -1;
            if (n_pre) atomicAdd(&out.stats[kStPrecheck], n_pre);
            if (n_tps) atomicAdd(&out.stats[kStTpsPruned], n_tps);
            if (!mask) {
                out.master[slot] = -1; out.bsel[slot] = -1;
                out.T[slot] = keyd(kInfKey); out.L[slot] = keyd(kInfKey);
                if (c < R) {
                    atomicAdd(&out.stats[kStReplicas], 1ull);
                    const int runs = dm.role_search ? dm.b_max + 1 : (role ? dm.b_max : 1);
                    if (m <= N) atomicAdd(&out.stats[kStPaper], runs * paper_candidates(m, N));
                }
            } else {
                const int W = N - m + 1;
                const int lg = (int)(1.0f * __log2f(1.0f + (float)m * (float)W));
                const int cls = dp_item_bytes(m, N, dm.dp_warps, 4, false) <= dm.dp_small;   // class 1 never spills
                const int size = (lg < kSizeBins - 1 ? lg : kSizeBins - 1) | cls << 4;
                si.size[slot] = (uint8_t)size;
                const int nv = __popcll(mask);
                for (int lv = 0; lv < nv; ++lv) atomicAdd(&ctrl[item_bin(lv, size)], 1u);
            }
        }
    }
}

// The ordering bins' scan, after the pre-pass: with nb bins in use (class
// 1's only where that class exists), lane t owns positions [t nb/32,
// (t+1) nb/32) of the descending bin order (class 0's bins, then class 1's),
// read eight at a time.  One warp.
__global__ void bins_kernel(Dims dm, unsigned *ctrl)
{
    const int lane = threadIdx.x & 31;
    const int per = (dm.dp_small ? kAllBins : kOrderBins) / 32;
    unsigned *own = ctrl + kAllBins - 1 - lane * per;              // own[-j] = position per lane + j
    unsigned sum = 0;
    for (int j = 0; j < per; j += 8) {
        unsigned v[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) v[q] = __ldcg(own - j - q);
#pragma unroll
        for (int q = 0; q < 8; ++q) sum += v[q];
    }
    unsigned incl = sum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const unsigned x = __shfl_up_sync(0xFFFFFFFFu, incl, o);
        if (lane >= o) incl += x;
    }
    unsigned base = incl - sum;
    if (dm.dp_small && lane == kOrderBins / per) {               // class 0 holds the first kOrderBins positions
        ctrl[kCtrlEnd] = base;
        ctrl[kCtrlNext + 1] = base;
    }
    for (int j = 0; j < per; j += 8) {
        unsigned v[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) v[q] = __ldcg(own - j - q);
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            own[-j - q] = base;
            base += v[q];
        }
    }
    if (lane == 31) {
        ctrl[kCtrlEnd + 1] = base;
        if (!dm.dp_small) ctrl[kCtrlEnd] = ctrl[kCtrlNext + 1] = base;   // one class: class 1 is empty
    }
}

// Item lv of a slot (its variants from the largest batch down) goes to bin
// item_bin(lv, size) as (slot << 8) | role << 7 | sweep << 6 | bit: role 1 =
// decode; sweep 1 = an accepted result stops the smaller batches (every item
// but the prefill run of a searched role).  The lanes of a warp whose items
// share a bin take their positions with one atomic.
__global__ void order_scatter_kernel(Dims dm, DevPop pop, SlotInfo si, WorkList wl)
{
    const int total = dm.P * dm.K, lane = threadIdx.x & 31;
    const unsigned below = (1u << lane) - 1u;
    for (int base = blockIdx.x * blockDim.x + (threadIdx.x & ~31); base < total; base += gridDim.x * blockDim.x) {
        const int slot = base + lane;
        uint64_t mask = 0;
        int size = 0, grole = 0;
        if (slot < total) {
            const int g = slot / dm.K, c = slot - g * dm.K;
            if (c < pop.nclus[g]) mask = si.mask[slot];
            if (mask) {
                size = si.size[slot];
                grole = (int)((pop.roles[g] >> c) & 1ull);
            }
        }
        for (int lv = 0; __any_sync(0xFFFFFFFFu, mask != 0); ++lv) {
            int bit = 0, bin = -1;
            if (mask) {
                bit = 63 - __clzll((long long)mask);
                mask &= ~(1ull << bit);
                bin = item_bin(lv, size);
            }
            const unsigned peers = __match_any_sync(0xFFFFFFFFu, bin);
            if (bin >= 0) {
                const int leader = __ffs(peers) - 1;
                unsigned at = 0;
                if (lane == leader) at = atomicAdd(&wl.ctrl[bin], (unsigned)__popc(peers));
                at = __shfl_sync(peers, at, leader);
                const bool pre = dm.role_search ? bit == dm.b_max : !grole;
                const uint64_t flags = (pre ? 0u : 0x80u) | (dm.role_search && pre ? 0u : 0x40u);
                wl.items[at + __popc(peers & below)] = ((uint64_t)slot << 8) | flags | (uint64_t)bit;
            }
        }
    }
}

// Persistent CTAs; each work item is one (genome, replica slot, variant) the
// pre-pass kept, skipped if a larger batch of its replica was already
// accepted.  Per item:
//  1. stage the master-free cost rows l_k(n) and the link times as 32-bit
//     order keys (exact ranks, see ranks.cu);
//  2. masters the memory allows;
//  3. prefix columns F_k (no master, devices 1..k) on warps 0-1 and suffix
//     columns G_k (no master, devices k..m) on warps 2-3, concurrently, each
//     thread a span of a column:
//        F_k[r] = min_s max(F_{k-1}[s], l_k(r-s+1), tau_k)
//        G_k[r] = min_s max(G_{k+1}[s], l_k(r-s+1), tau_{k+1})
//  4. master mu: the prefix holds a extra blocks, the suffix b, the master
//     W - a - b, so with H_mu[c] = min_{a+b=c} max(F_{mu-1}[a], G_{mu+1}[b])
//        V_mu = max(tau_mu, tau_{mu+1}, min_c max(H_mu[c], l_mu^head(W - c)))
//     (F_0 and G_{m+1} are the empty stage: 0 at index 0, +inf after); the
//     warp fetches l_mu^head asynchronously while it builds H_mu;
//  5. mu* = smallest mu with the least V_mu; its prefix columns D_k (master at
//     mu*) are recomputed for the traceback;
//  6. traceback with the smallest-split rule (n_k = number of n <= r+1 with
//     l_k(n) <= D, counted with warp ballots); the bottleneck T (the largest
//     stage or link time of the partition, equal to V) and Lambda (summed in
//     pipeline order) in float64 from the stage and link tables; meanwhile
//     warp 1 claims the next item.
// Every comparison is between ranks of the same stage and link times the
// oracle compares, so V, mu*, the partition, T and Lambda are bit-identical to
// Alg. 1.
template <typename Key, bool SPILL>
__device__ __forceinline__ void dp_eval_body(const Dims &dm, const Tables &tb, const DevPop &pop, const EvalOut &out,
                                             const WorkList &wl, const SlotInfo &si, const SplitOut &so, int cls)
{
    extern __shared__ __align__(16) unsigned char smem[];
    __shared__ int s_S0, s_Z, s_mu, s_done;
    __shared__ uint32_t s_V;
    __shared__ double s_L, s_T;
    __shared__ unsigned s_item, s_next;           // s_next: an item claimed during the last traceback
    // (spilled layout) s_next's item word, replica size and offset, and where its device ids,
    // capacities and keys wait in shared memory (-1: not fetched)
    __shared__ unsigned long long s_pre_item;
    __shared__ int s_pre_m, s_pre_off, s_pre_at, s_pre_use;
    __shared__ unsigned long long s_bestkey;     // (V << 32) | mu of the best master so far
    __shared__ uint32_t s_V0, s_V1;
    __shared__ unsigned s_prb[3];                // probes of a column over 32, 64, 128 threads

    const int K = dm.K, M = dm.M, N = dm.N;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5, NW = blockDim.x >> 5;
    constexpr Key kInf = (Key)~(Key)0;
    const unsigned n_items = wl.ctrl[kCtrlEnd + cls];         // this class's items end here
    constexpr bool spill = SPILL;
    // this CTA's suffix-column scratch (only the first launch's CTAs spill)
    uint32_t *gsp = spill ? wl.gspill + (size_t)blockIdx.x * wl.spill_stride : nullptr;
    if (tid == 0) { s_next = ~0u; s_pre_at = -1; }
  for (;;) {
    // ---- next work item of the class (heaviest first); warp 1 claims it
    //      while warp 0 traces the last one back
    if (tid == 0) {
        const unsigned nx = s_next;
        s_next = ~0u;
        s_item = nx != ~0u ? nx : atomicAdd(&wl.ctrl[kCtrlNext + cls], 1u);
        s_pre_use = nx != ~0u ? s_pre_at : -1;
        s_pre_at = -1;
    }
    __syncthreads();
    const unsigned idx = s_item;
    const int pre_at = SPILL ? s_pre_use : -1;                  // the item's data fetched already
    __syncthreads();
    if (idx >= n_items) break;
    const uint64_t item = pre_at >= 0 ? s_pre_item : wl.items[idx];
    const int slot = (int)(item >> 8), code = (int)(item & 0x3Fu);
    if (tid == 0) s_done = *(volatile const int32_t *)&si.best[slot] > code;   // a larger batch won
    __syncthreads();
    if (s_done) continue;
    const int g = slot / K, c = slot - g * K;
    const size_t gk = (size_t)g * K + c;
    const int off = pre_at >= 0 ? s_pre_off : si.off[slot], m = pre_at >= 0 ? s_pre_m : pop.sizes[gk];
    const int role = (int)((item >> 7) & 1u);                   // decode
    const bool sweep = (item >> 6) & 1u;                        // the result advances the decode sweep
    uint64_t vmask = 1ull << code;
    int16_t *lay_out = so.layers + ((size_t)g * dm.V + code) * M + off;

    unsigned long long st_runs = 0, st_cells = 0, st_probes = 0;
    bool served = false;

    if (m <= N && vmask) {
        const int W = N - m + 1;
        int *cnt0 = reinterpret_cast<int *>(smem);              // [m]
        int *cnt1 = cnt0 + m;                                   // [m]
        int *nk = cnt1 + m;                                     // [m]
        Key *leaf0 = reinterpret_cast<Key *>(nk + m);           // [m][W] l_k(n)
        Key *Fst = leaf0 + (size_t)m * W;                       // [m][W] prefix / traceback columns
        Key *Gst = Fst + (size_t)m * W;                         // [m][W] suffix columns ([2][W] spilled)
        Key *Hb = Gst + (size_t)(spill ? 2 : m) * W;            // [NW][W] per-warp convolution
        Key *Lb = Hb + (size_t)NW * W;                          // [NW][W] per-warp head row
        Key *Sb = Lb + (size_t)NW * W;                          // [NW][W] per-warp suffix column (spilled)
        Key *row1s = Sb + (spill ? (size_t)NW * W : 0);         // [W] head row of mu*
        Key *delta = row1s + W;                                 // [W] the empty stage
        Key *tauk = delta + W;                                  // [m] tauk[k] = link (k-1) -> k
        Key *lbm = tauk + m;                                    // [m] l^head_k(1)
        uint16_t *devs = reinterpret_cast<uint16_t *>(lbm + m);   // [m]

        int p_c0 = 0, p_c1 = 0;                                 // this thread's device's fetched
        Key p_t = 0, p_l = 0;                                   // capacities and keys (pre_at >= 0)
        if (pre_at >= 0) {                                      // read them all before any is overwritten
            const int *q0 = reinterpret_cast<const int *>(smem + pre_at), *q1 = q0 + m;
            const Key *qt = reinterpret_cast<const Key *>(q1 + m), *ql = qt + m;
            const uint16_t *qd = reinterpret_cast<const uint16_t *>(ql + m);
            int d = 0;
            if (tid < m) { d = qd[tid]; p_c0 = q0[tid]; p_c1 = q1[tid]; p_t = qt[tid]; p_l = ql[tid]; }
            __syncthreads();
            if (tid < m) devs[tid] = (uint16_t)d;
        } else {
            for (int k = tid; k < m; k += blockDim.x) devs[k] = pop.perm[(size_t)g * M + off + k];
        }
        if (tid < 3) s_prb[tid] = c_span_probes[tid][W];
        for (int r = tid; r < W; r += blockDim.x) delta[r] = r ? kInf : (Key)0;
        __syncthreads();

        // column accessors (1-based device index k)
        auto colF = [&](int k) -> const Key * {
            return k == 0 ? delta : k == 1 ? leaf0 : Fst + (size_t)(k - 1) * W;
        };
        // suffix column G_k: in shared memory (two of them, alternating, when spilled;
        // the others then live in this CTA's global scratch, gsp)
        auto colG = [&](int k) -> const Key * {
            return k == m + 1 ? delta : k == m ? leaf0 + (size_t)(m - 1) * W
                                               : Gst + (size_t)(spill ? (k & 1) : k - 1) * W;
        };

        const unsigned long long lprobe = 32 - __clz(W);
        while (vmask && !served) {
            const int bit = 63 - __clzll((long long)vmask);          // highest batch first
            vmask &= ~(1ull << bit);
            const int v = role ? bit + 1 : 0;
            const size_t vM = (size_t)v * M;
            // ---- 1. capacities, link ranks and master-free cost rows
            if (pre_at >= 0) {
                if (tid < m) { cnt0[tid] = p_c0; cnt1[tid] = p_c1; tauk[tid] = p_t; lbm[tid] = p_l; }
            } else {
                for (int k = tid; k < m; k += blockDim.x) {
                    const size_t vd = vM + devs[k];
                    const int c0 = tb.cap[vd * 2], c1 = tb.cap[vd * 2 + 1];
                    cnt0[k] = c0 < W ? c0 : W;
                    cnt1[k] = c1 < W ? c1 : W;
                    tauk[k] = k ? (Key)tb.tau_rank[(vM + devs[k - 1]) * M + devs[k]] : (Key)0;
                    lbm[k] = (Key)tb.leaf_rank[((vM + devs[k]) * 2 + 1) * dm.LS];   // l^head_k(1)
                }
            }
            for (int k = wid; k < m; k += NW)                       // the loads of a row overlap
                stage_row(leaf0 + (size_t)k * W, tb.leaf_rank + (vM + devs[k]) * 2 * dm.LS, W, lane);
            if (SPILL && wid == NW - 1)                             // device 1's head row (step 3)
                stage_row(row1s, tb.leaf_rank + ((vM + devs[0]) * 2 + 1) * dm.LS, W, lane);
            cp_async_wait_all();
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
            // ---- 3. prefix columns (warps 0-1) and suffix columns (warps 2-3).
            //      With the spilled layout (the largest replicas) the prefix chain
            //      runs first with the head on device 1: if then V_1 (its last
            //      cell) equals V0 (the master-free optimum, from the suffix
            //      side), every V_mu >= V0 = V_1, so mu* = 1 and these are the
            //      columns step 5 would recompute; steps 4 and 5 are skipped.
            //      Otherwise the chain runs again without the head.
            auto prefix_chain = [&](bool head1) {
                for (int k = 2; k <= m - 1; ++k) {
                    const Key *prev = (head1 && k == 2) ? row1s : colF(k - 1), *row = leaf0 + (size_t)(k - 1) * W;
                    const Key t = tauk[k - 1];
                    Key *cur = Fst + (size_t)(k - 1) * W;
                    const int per = (W + 63) >> 6;                 // cells per thread
                    dp_span(prev, row, t, cur, tid * per, min(W, (tid + 1) * per));
                    bar_named(1, 64);
                }
            };
            // the last cell of a chain, its minimum over every split taken by a warp's lanes
            auto top_cell = [&](const Key *a, const Key *b, Key t) -> uint32_t {
                uint32_t x = kInf;
                for (int q = lane; q < W; q += 32) x = min(x, (uint32_t)max(a[q], b[W - 1 - q]));
#pragma unroll
                for (int o = 16; o; o >>= 1) x = min(x, __shfl_xor_sync(0xFFFFFFFFu, x, o));
                return max(x, (uint32_t)t);
            };
            if (wid < 2) {
                prefix_chain(SPILL);
                if (wid == 0) {                                   // V0 = F_m[W-1] (V_1 when spilled)
                    uint32_t v = 0;
                    if (m >= 2)
                        v = top_cell((SPILL && m == 2) ? row1s : colF(m - 1), leaf0 + (size_t)(m - 1) * W, tauk[m - 1]);
                    if (lane == 0) {
                        if (SPILL) {                              // (V_1, 1) seeds the best master
                            s_V1 = v;
                            s_bestkey = (m >= 2 && v != (uint32_t)kInf) ? ((unsigned long long)v << 32) | 1u : ~0ull;
                        } else {
                            s_V0 = v;
                            s_bestkey = ~0ull;
                        }
                    }
                }
            } else {
                for (int k = m - 1; k >= 2; --k) {
                    const Key *prev = colG(k + 1), *row = leaf0 + (size_t)(k - 1) * W;
                    const Key t = tauk[k];
                    Key *cur = Gst + (size_t)(spill ? (k & 1) : k - 1) * W;
                    const int per = (W + 63) >> 6;
                    const int r0 = (tid - 64) * per, r1 = min(W, (tid - 63) * per);
                    dp_span(prev, row, t, cur, r0, r1);
                    if (spill)                                      // the thread's own cells, to the scratch
                        for (int r = r0; r < r1; ++r) __stcg(gsp + (size_t)(k - 1) * W + r, (uint32_t)cur[r]);
                    bar_named(2, 64);
                }
                if (SPILL && wid == 2) {                          // V0 = G_1[W-1]
                    const uint32_t v = m >= 2 ? top_cell(leaf0, colG(2), tauk[1]) : 0u;
                    if (lane == 0) s_V0 = v;
                }
            }
            if (tid == 0 && m >= 3) {
                st_cells += 2ull * (m - 2) * W;
                st_probes += 2ull * (m - 2) * s_prb[1];
            }
            __syncthreads();
            // ---- 4. one master per warp at a time, skipping a master whose lower
            //      bound V_mu >= max(V0, l^head_mu(1)) (V0 the master-free
            //      optimum F_m[W-1]: the head only adds) exceeds the best V found
            //      so far, or ties it with a larger index
            const uint32_t V0 = s_V0;
            bool spec = false;                                    // mu* = 1 proved (the spilled layout)
            if (SPILL) {
                spec = m >= 2 && s_V1 == V0 && V0 != (uint32_t)kInf;
                if (tid == 0 && m >= 2) { st_cells += 1; st_probes += lprobe; }
                if (!spec && m >= 3) {                            // the combine needs the master-free columns
                    if (wid < 2) prefix_chain(false);
                    if (tid == 0) {
                        st_cells += (unsigned long long)(m - 2) * W;
                        st_probes += (unsigned long long)(m - 2) * s_prb[1];
                    }
                    __syncthreads();
                }
            }
            auto bound = [&](int k) -> uint32_t { return mu_ok(k + 1) ? max(V0, (uint32_t)lbm[k]) : (uint32_t)kInf; };

            unsigned long long w_cells = 0, w_probes = 0;
            Key *H = Hb + (size_t)wid * W, *L1 = Lb + (size_t)wid * W;
            for (int mu = wid + 1; mu <= m && !spec; mu += NW) {
                if (!mu_ok(mu) || (SPILL && m >= 2 && mu == 1)) continue;   // (V_1 is known when spilled)
                const uint32_t lb = bound(mu - 1);
                const unsigned long long bk = *reinterpret_cast<volatile unsigned long long *>(&s_bestkey);
                const uint32_t bv = (uint32_t)(bk >> 32);
                if (lb > bv || (lb == bv && (unsigned)mu > (unsigned)(bk & 0xFFFFFFFFu))) continue;
                const uint32_t *hrow = tb.leaf_rank + ((vM + devs[mu - 1]) * 2 + 1) * dm.LS;
                const Key *P = colF(mu - 1), *S = colG(mu + 1);
                HeadRow<Key> hr;
                hr.start(L1, hrow, W, lane);                          // in flight while H is built
                if (spill && mu + 1 <= m - 1) {                       // the suffix column from the scratch
                    Key *sb = Sb + (size_t)wid * W;                   // (L2: written by this CTA's other warps)
                    for (int r = lane; r < W; r += 32) sb[r] = (Key)__ldcg(gsp + (size_t)mu * W + r);
                    __syncwarp();
                    S = sb;
                }
                const int per = (W + 31) >> 5;
                dp_span(P, S, (Key)0, H, lane * per, min(W, (lane + 1) * per));
                hr.finish(L1, hrow, W, lane);
                __syncwarp();
                uint32_t V = dp_cell(H, L1, (Key)0, W - 1);
                if (mu >= 2) V = max(V, (uint32_t)tauk[mu - 1]);
                if (mu <= m - 1) V = max(V, (uint32_t)tauk[mu]);
                __syncwarp();
                w_cells += W + 1;
                w_probes += s_prb[0] + lprobe;
                if (lane == 0) atomicMin(&s_bestkey, ((unsigned long long)V << 32) | (unsigned)mu);
            }
            if (lane == 0) { st_cells += w_cells; st_probes += w_probes; }
            if (tid == 0 && m >= 2) { st_cells += 1; st_probes += lprobe; }
            __syncthreads();
            if (tid == 0) {
                s_V = (uint32_t)(s_bestkey >> 32);
                s_mu = (int)(s_bestkey & 0xFFFFFFFFu);
            }
            __syncthreads();
            const uint32_t V = s_V;
            const int mus = s_mu;
            if (V == kInf) {
                // the pre-pass tested this variant's memory exactly, unless the
                // profile's costs do not grow with the batch: then the batches
                // below the largest that passed run untested, and may have no
                // partition.  Otherwise this cannot happen.
                if (tid == 0 && (dm.grows || !role)) atomicAdd(&out.stats[kStDeviceErrors], 1ull);
                continue;
            }
            if (!spec) {
                for (int r = tid; r < W; r += blockDim.x)
                    row1s[r] = (Key)tb.leaf_rank[((vM + devs[mus - 1]) * 2 + 1) * dm.LS + r];
                __syncthreads();
            }
            // ---- 5. mu*'s prefix columns, for the traceback (already there when spec)
            auto rowk = [&](int k) -> const Key * { return k == mus ? row1s : leaf0 + (size_t)(k - 1) * W; };
            auto colD = [&](int k) -> const Key * {
                if (k == 1) return mus == 1 ? row1s : leaf0;
                return Fst + (size_t)(k - 1) * W;
            };
            for (int k = (mus > 2 ? mus : 2); k <= m - 1 && !spec; ++k) {
                const Key *prev = colD(k - 1), *row = rowk(k);
                const Key t = tauk[k - 1];
                Key *cur = Fst + (size_t)(k - 1) * W;
                const int per = (W + 127) >> 7;
                dp_span(prev, row, t, cur, tid * per, min(W, (tid + 1) * per));
                __syncthreads();
                if (tid == 0) { st_cells += W; st_probes += s_prb[2]; }
            }
            // ---- 6. traceback (smallest split on ties), T and Lambda
            if (wid == 0) {
                int r = W - 1;
                uint32_t D = V;
                for (int k = m; k >= 2; --k) {
                    const Key *row = rowk(k);
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
                if (lane == 0) nk[0] = r + 1;
                __syncwarp();
                // stage and link times of the partition, lane k holds device k
                const double *lrow = tb.leaf + vM * 2 * dm.LS;
                const double *trow = tb.tau + vM * M;
                double lam = 0.0;
                uint64_t tmax = 0;
                for (int base = 0; base < m; base += 32) {
                    const int k = base + lane;               // 0-based device
                    double lk = 0.0, tk = 0.0;
                    if (k < m) {
                        lk = lrow[((size_t)devs[k] * 2 + (k == mus - 1)) * dm.LS + nk[k] - 1];
                        if (k >= 1) tk = trow[(size_t)devs[k - 1] * M + devs[k]];
                        tmax = umax64(tmax, umax64(dkey(lk), dkey(tk)));
                    }
                    for (int q = 0; q < 32 && base + q < m; ++q) {
                        const double lq = __shfl_sync(0xFFFFFFFFu, lk, q);
                        const double tq = __shfl_sync(0xFFFFFFFFu, tk, q);
                        if (base + q == 0) lam = lq;
                        else { lam = lam + tq; lam = lam + lq; }
                    }
                }
#pragma unroll
                for (int o = 16; o; o >>= 1) tmax = umax64(tmax, __shfl_xor_sync(0xFFFFFFFFu, tmax, o));
                if (lane == 0) {
                    s_L = lam;
                    s_T = keyd(tmax);
                    s_done = (!role) || lam <= dm.lam_max;       // 1.0 / lam >= Min_TPS
                }
            } else if (wid == 1) {
                unsigned nx = 0;
                if (lane == 0) nx = atomicAdd(&wl.ctrl[kCtrlNext + cls], 1u);
                nx = __shfl_sync(0xFFFFFFFFu, nx, 0);
                if (lane == 0) s_next = nx;
                if (SPILL && nx < n_items) {
                    // (spilled layout) the next item's header, device ids, capacities
                    // and keys, into this run's suffix-column and per-warp buffers,
                    // which nothing reads from here to the next item
                    const uint64_t it2 = wl.items[nx];
                    const int slot2 = (int)(it2 >> 8), code2 = (int)(it2 & 0x3Fu);
                    const int g2 = slot2 / K, c2 = slot2 - g2 * K;
                    const int off2 = si.off[slot2], m2 = pop.sizes[(size_t)g2 * K + c2];
                    const int at = (int)(reinterpret_cast<unsigned char *>(Gst) - smem);
                    const long room = reinterpret_cast<unsigned char *>(row1s) - reinterpret_cast<unsigned char *>(Gst);
                    if (m2 <= N && m2 <= (int)blockDim.x && 18L * m2 <= room) {
                        const int W2 = N - m2 + 1;
                        const size_t vM2 = (size_t)(((it2 >> 7) & 1u) ? code2 + 1 : 0) * M;
                        int *q0 = reinterpret_cast<int *>(smem + at), *q1 = q0 + m2;
                        Key *qt = reinterpret_cast<Key *>(q1 + m2), *ql = qt + m2;
                        uint16_t *qd = reinterpret_cast<uint16_t *>(ql + m2);
                        for (int k = lane; k < m2; k += 32) {
                            const int d = pop.perm[(size_t)g2 * M + off2 + k];
                            qd[k] = (uint16_t)d;
                            const int a0 = tb.cap[(vM2 + d) * 2], a1 = tb.cap[(vM2 + d) * 2 + 1];
                            q0[k] = a0 < W2 ? a0 : W2;
                            q1[k] = a1 < W2 ? a1 : W2;
                            ql[k] = (Key)tb.leaf_rank[((vM2 + d) * 2 + 1) * dm.LS];
                        }
                        __syncwarp();
                        for (int k = lane; k < m2; k += 32)
                            qt[k] = k ? (Key)tb.tau_rank[(vM2 + qd[k - 1]) * M + qd[k]] : (Key)0;
                        if (lane == 0) { s_pre_item = it2; s_pre_m = m2; s_pre_off = off2; s_pre_at = at; }
                    }
                }
            }
            __syncthreads();
            if (s_done) {
                for (int k = tid; k < m; k += blockDim.x) lay_out[k] = (int16_t)nk[k];
                if (tid == 0) {
                    const size_t sv = gk * dm.V + code;
                    so.mu[sv] = (int16_t)(mus - 1);
                    so.T[sv] = s_T;
                    so.L[sv] = s_L;
                    __threadfence();
                    if (sweep) atomicMax(&si.best[slot], code);
                }
                served = true;
            }
            __syncthreads();
        }
    }
    __syncthreads();
    if (lane == 0 && (st_cells | st_probes)) {
        atomicAdd(&out.stats[kStCells], st_cells);
        atomicAdd(&out.stats[kStProbes], st_probes);
    }
    if (tid == 0 && st_runs) atomicAdd(&out.stats[cls ? kStDpRunsSmall : kStDpRuns], st_runs);
  }
}

// ---------------------------------------------------------------------------
// Blocks of several types (per-layer prefix sums): the plain-scan DP.
//
// A stage's cost now depends on where it starts, and the best bottleneck of a
// prefix is no longer monotone in its length (a heavy block can make fewer
// blocks cost more), so the crossover bisection of dp_eval_body does not
// apply.  Each cell takes the full minimum over its splits, as Eq. 1 writes
// it, on the float64 times themselves (their bit patterns, which order like
// the values), read from the per-layer cost table:
//   F_k[r] = min_s max(F_{k-1}[s], l_k(s+k-1 .. r+k-1), tau_k)     devices 1..k, no master
//   G_k[b] = min_t max(l_k(first t+1 of its range), G_{k+1}[b-t], tau_{k+1})   devices k..m
//   V_mu   = min_{a,b} max(F_{mu-1}[a], l^head_mu(the W-a-b blocks between), G_{mu+1}[b], tau_mu, tau_mu+1)
// mu* = the smallest mu with the least V_mu; its prefix columns (the head at
// mu*) are recomputed from column mu* on, and the traceback takes the smallest
// split attaining each cell's value.  Every value and tie is the oracle's.
// ---------------------------------------------------------------------------
__host__ __device__ __forceinline__ unsigned dp_layered_item_bytes(int m, int N)
{
    const unsigned W = (unsigned)(N - m + 1);
    const unsigned bytes = 8u * (2u * (unsigned)m * W + 2u * (unsigned)m) + 4u * (unsigned)m + 2u * (unsigned)m;
    return (bytes + 15u) & ~15u;
}

size_t dp_layered_smem_bytes(int M, int N)
{
    size_t best = 0;
    const int mmax = M < N ? M : N;
    for (int m = 1; m <= mmax; ++m) {
        const size_t b = dp_layered_item_bytes(m, N);
        if (b > best) best = b;
    }
    return best;
}

__global__ void __launch_bounds__(128) dp_layered_kernel(Dims dm, Tables tb, DevPop pop, EvalOut out, WorkList wl,
                                                         SlotInfo si, SplitOut so)
{
    extern __shared__ __align__(16) unsigned char lsm[];
    __shared__ unsigned s_item;
    __shared__ int s_done, s_mu;
    __shared__ double s_T, s_L;
    const int K = dm.K, M = dm.M, N = dm.N;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5, NW = blockDim.x >> 5;
    const uint64_t INF = kInfKey;
    const unsigned n_items = wl.ctrl[kCtrlEnd];
    const size_t NN = (size_t)N * N;
    for (;;) {
        if (tid == 0) s_item = atomicAdd(&wl.ctrl[kCtrlNext], 1u);
        __syncthreads();
        const unsigned idx = s_item;
        __syncthreads();
        if (idx >= n_items) break;
        const uint64_t item = wl.items[idx];
        const int slot = (int)(item >> 8), code = (int)(item & 0x3Fu);
        if (tid == 0) s_done = *(volatile const int32_t *)&si.best[slot] > code;   // a larger batch won
        __syncthreads();
        if (s_done) continue;
        const int g = slot / K, c = slot - g * K;
        const size_t gk = (size_t)g * K + c;
        const int off = si.off[slot], m = pop.sizes[gk];
        const int role = (int)((item >> 7) & 1u);
        const bool sweep = (item >> 6) & 1u;
        const int v = role ? code + 1 : 0;
        const int W = N - m + 1;
        uint64_t *F = reinterpret_cast<uint64_t *>(lsm);          // [m][W] prefix (then mu*'s) columns
        uint64_t *G = F + (size_t)m * W;                          // [m][W] suffix columns
        uint64_t *Vmu = G + (size_t)m * W;                        // [m]
        uint64_t *tk = Vmu + m;                                   // [m] tk[k] = link k-1 -> k (0-based)
        int *nk = reinterpret_cast<int *>(tk + m);                // [m]
        uint16_t *devs = reinterpret_cast<uint16_t *>(nk + m);    // [m]
        const double *lc = tb.lcost + (size_t)v * M * 2 * NN;
        for (int k = tid; k < m; k += blockDim.x) devs[k] = pop.perm[(size_t)g * M + off + k];
        __syncthreads();
        for (int k = tid; k < m; k += blockDim.x)
            tk[k] = k ? dkey(tb.tau[((size_t)v * M + devs[k - 1]) * M + devs[k]]) : 0ull;
        // l_k(j .. j+n-1) (k 0-based), with the head when mf
        auto cost = [&](int k, int j, int n, int mf) -> uint64_t {
            return dkey(lc[((size_t)devs[k] * 2 + mf) * NN + (size_t)j * N + (n - 1)]);
        };
        __syncthreads();
        unsigned long long probes = 0;
        // ---- prefix columns F_1..F_m (no master)
        for (int r = tid; r < W; r += blockDim.x) F[r] = cost(0, 0, r + 1, 0);
        __syncthreads();
        for (int k = 2; k <= m; ++k) {
            const uint64_t *prev = F + (size_t)(k - 2) * W;
            uint64_t *cur = F + (size_t)(k - 1) * W;
            const uint64_t t = tk[k - 1];
            for (int r = tid; r < W; r += blockDim.x) {
                uint64_t best = INF;
                for (int s2 = 0; s2 <= r; ++s2)
                    best = umin64(best, umax64(umax64(prev[s2], cost(k - 1, s2 + k - 1, r - s2 + 1, 0)), t));
                cur[r] = best;
                probes += (unsigned long long)(r + 1);
            }
            __syncthreads();
        }
        // ---- suffix columns G_m..G_2: devices k..m hold the last b + m - k + 1 blocks
        for (int b = tid; b < W; b += blockDim.x) G[(size_t)(m - 1) * W + b] = cost(m - 1, N - 1 - b, b + 1, 0);
        __syncthreads();
        for (int k = m - 1; k >= 2; --k) {
            const uint64_t *nxt = G + (size_t)k * W;
            uint64_t *cur = G + (size_t)(k - 1) * W;
            const uint64_t t = tk[k];
            for (int b = tid; b < W; b += blockDim.x) {
                const int j0 = N - (b + m - k + 1);
                uint64_t best = INF;
                for (int t2 = 0; t2 <= b; ++t2)
                    best = umin64(best, umax64(umax64(cost(k - 1, j0, t2 + 1, 0), nxt[b - t2]), t));
                cur[b] = best;
                probes += (unsigned long long)(b + 1);
            }
            __syncthreads();
        }
        // ---- masters: a warp per master, lanes over the (a, b) splits
        for (int mu = wid + 1; mu <= m; mu += NW) {
            const uint64_t *Fp = mu >= 2 ? F + (size_t)(mu - 2) * W : nullptr;
            const uint64_t *Gs = mu <= m - 1 ? G + (size_t)mu * W : nullptr;
            uint64_t lk = 0;
            if (mu >= 2) lk = umax64(lk, tk[mu - 1]);
            if (mu <= m - 1) lk = umax64(lk, tk[mu]);
            uint64_t best = INF;
            const int amax = mu >= 2 ? W - 1 : 0;
            for (int a = 0; a <= amax; ++a) {
                const uint64_t fa = Fp ? Fp[a] : 0ull;
                if (fa >= best) continue;                       // cannot lower the minimum
                const int bmax = mu <= m - 1 ? W - 1 - a : 0;
                for (int b = lane; b <= bmax; b += 32) {
                    const uint64_t gb = Gs ? Gs[b] : 0ull;
                    const uint64_t h = cost(mu - 1, (mu - 1) + a, W - a - b, 1);
                    best = umin64(best, umax64(umax64(fa, gb), umax64(h, lk)));
                }
                probes += (unsigned long long)((bmax + 1 + 31 - lane) / 32);
#pragma unroll
                for (int o = 16; o; o >>= 1) best = umin64(best, __shfl_xor_sync(0xFFFFFFFFu, best, o));
            }
            if (lane == 0) Vmu[mu - 1] = best;
        }
        __syncthreads();
        if (tid == 0) {                                           // the smallest master with the least value
            int mus = 1;
            for (int mu = 2; mu <= m; ++mu)
                if (Vmu[mu - 1] < Vmu[mus - 1]) mus = mu;
            s_mu = mus;
        }
        __syncthreads();
        const int mus = s_mu;
        const uint64_t V = Vmu[mus - 1];
        if (V == INF) {                                           // no partition (memory)
            if (tid == 0 && !role) {                              // a prefill result that does not exist
                const size_t sv = gk * dm.V + code;
                so.T[sv] = keyd(kInfKey);
                so.L[sv] = keyd(kInfKey);
            }
            if (lane == 0) atomicAdd(&out.stats[kStProbes], probes);
            if (tid == 0) atomicAdd(&out.stats[kStDpRuns], 1ull);
            __syncthreads();
            continue;
        }
        // ---- mu*'s prefix columns from column mu* on (the head at mu*)
        for (int k = mus; k <= m; ++k) {
            uint64_t *cur = F + (size_t)(k - 1) * W;
            const int mf = k == mus;
            if (k == 1) {
                for (int r = tid; r < W; r += blockDim.x) cur[r] = cost(0, 0, r + 1, 1);
            } else {
                const uint64_t *prev = F + (size_t)(k - 2) * W;
                const uint64_t t = tk[k - 1];
                for (int r = tid; r < W; r += blockDim.x) {
                    uint64_t best = INF;
                    for (int s2 = 0; s2 <= r; ++s2)
                        best = umin64(best, umax64(umax64(prev[s2], cost(k - 1, s2 + k - 1, r - s2 + 1, mf)), t));
                    cur[r] = best;
                    probes += (unsigned long long)(r + 1);
                }
            }
            __syncthreads();
        }
        // ---- traceback (warp 0): the smallest split attaining each cell's value
        if (wid == 0) {
            int r = W - 1;
            for (int k = m; k >= 2; --k) {
                const uint64_t D = F[(size_t)(k - 1) * W + r];
                const uint64_t *prev = F + (size_t)(k - 2) * W;
                const uint64_t t = tk[k - 1];
                const int mf = k == mus;
                int sp = -1;
                for (int base = 0; base <= r && sp < 0; base += 32) {
                    const int s2 = base + lane;
                    const bool hit = s2 <= r && umax64(umax64(prev[s2], cost(k - 1, s2 + k - 1, r - s2 + 1, mf)), t) == D;
                    const unsigned bal = __ballot_sync(0xFFFFFFFFu, hit);
                    if (bal) sp = base + __ffs(bal) - 1;
                }
                if (sp < 0) {                                     // cannot happen: D is attained
                    sp = 0;
                    if (lane == 0) atomicAdd(&out.stats[kStDeviceErrors], 1ull);
                }
                if (lane == 0) nk[k - 1] = r - sp + 1;
                r = sp;
            }
            if (lane == 0) nk[0] = r + 1;
            __syncwarp();
            // stage and link times of the partition in pipeline order
            if (lane == 0) {
                double lam = 0.0;
                uint64_t tmax = 0;
                int j = 0;
                for (int k = 0; k < m; ++k) {
                    const double lk = keyd(cost(k, j, nk[k], k == mus - 1));
                    const double tl = k ? keyd(tk[k]) : 0.0;
                    if (k == 0) lam = lk;
                    else { lam = lam + tl; lam = lam + lk; }
                    tmax = umax64(tmax, umax64(dkey(lk), dkey(tl)));
                    j += nk[k];
                }
                s_L = lam;
                s_T = keyd(tmax);
                s_done = (!role) || lam <= dm.lam_max;            // 1.0 / lam >= Min_TPS
            }
        }
        __syncthreads();
        const size_t sv = gk * dm.V + code;
        if (s_done) {
            int16_t *lay_out = so.layers + ((size_t)g * dm.V + code) * M + off;
            for (int k = tid; k < m; k += blockDim.x) lay_out[k] = (int16_t)nk[k];
            if (tid == 0) {
                so.mu[sv] = (int16_t)(mus - 1);
                so.T[sv] = s_T;
                so.L[sv] = s_L;
                __threadfence();
                if (sweep) atomicMax(&si.best[slot], code);
            }
        } else if (tid == 0 && !role) {
            so.T[sv] = keyd(kInfKey);
        }
        if (lane == 0) atomicAdd(&out.stats[kStProbes], probes);
        if (tid == 0) {
            atomicAdd(&out.stats[kStDpRuns], 1ull);
            atomicAdd(&out.stats[kStCells], (unsigned long long)(2 * m + (m - mus + 1)) * W + m);
        }
        __syncthreads();
    }
}

// One launch per DP class (cls): the same code over the class's items, with
// the class's shared-memory allocation.
// SPILL: the suffix columns live in the global scratch (dm.g_spill), a
// separate instance so that the other contexts keep their register count.
template <bool SPILL>
__global__ void __launch_bounds__(128, SPILL ? 6 : 0) dp_eval_kernel(Dims dm, Tables tb, DevPop pop, EvalOut out, WorkList wl,
                                                      SlotInfo si, SplitOut so, int cls)
{
    dp_eval_body<uint32_t, SPILL>(dm, tb, pop, out, wl, si, so, cls);
}

// The genome's objective from the role sums (PS, DS; PL, DL the rate-weighted
// latencies sum_P PS_c Lambda_c and sum_D DS_c Lambda_c, all summed in
// ascending replica order).  Objective 0: Eq. 3 bottleneck phase, Eq. 4
// backlog, Eq. 5 waiting time.  Objective 1: the per-request finishing time of
// the FT comparison, a request's prefill pass plus ND decode passes, each
// averaged over its role's replicas in proportion to their rates.  Either way
// the second key is Eq. 3's phase; no prefill or no decode capacity: +inf.
__device__ __forceinline__ void objective(const Dims &dm, double PS, double DS, double PL, double DL, double &w,
                                          double &phase)
{
    w = keyd(kInfKey);
    phase = keyd(kInfKey);
    if (PS != 0.0 && DS != 0.0) {
        const double tp = (double)dm.NP / PS, td = (double)dm.ND / DS;
        phase = tp >= td ? tp : td;                 // Eq. 3
        if (dm.objective == 1) {
            w = PL / PS + (double)dm.ND * (DL / DS);
        } else {
            const double x = phase - dm.t_a;
            const double bn = x > 0.0 ? x : 0.0;    // Eq. 4
            w = bn > 0.0 ? tp + bn : 0.0;           // Eq. 5
        }
    }
}

// One warp per genome.  Each replica that had work gets its outputs from its
// lane: the largest accepted variant is the sweep's answer (Alg. 2 keeps the
// highest feasible batch), with its master, batch and times, and the serving
// replica's rate (NP / T for prefill, b / T for decode).  The lanes then copy
// the partition, position by position, from the accepted variant's split
// results.  Lane 0 sums PS and DS in ascending replica order and applies
// Eq. 3 (bottleneck phase), Eq. 4 (backlog) and Eq. 5 (waiting time).  A
// 64-bit fingerprint of the genome, folded as a tree over the lanes, serves
// the elites' duplicate test.
__global__ void __launch_bounds__(128) finalize_score_kernel(Dims dm, DevPop pop, SlotInfo si, SplitOut so,
                                                             EvalOut out)
{
    __shared__ int s_off[4][E2_MAX_CLUSTERS + 1];     // replica start in the ordering
    __shared__ int s_best[4][E2_MAX_CLUSTERS];        // accepted variant bit, -1 none, -2 no work here
    const int wl = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int g = blockIdx.x * 4 + wl;
    if (g >= dm.P) return;
    const int K = dm.K, M = dm.M;
    const int R = pop.nclus[g];
    const uint64_t roles = pop.roles[g];
    // the fingerprint's inputs, loaded up front: replica sizes (lane c holds
    // sizes[c] and sizes[c + 32]) and the ordering folded by the lanes
    auto mix = [](uint64_t h, uint64_t x) { h = (h ^ x) * 0xBF58476D1CE4E5B9ull; return h ^ (h >> 31); };
    const int sz_lo = lane < K ? pop.sizes[(size_t)g * K + lane] : 0;
    const int sz_hi = lane + 32 < K ? pop.sizes[(size_t)g * K + lane + 32] : 0;
    uint64_t hl = 0x9E3779B97F4A7C15ull ^ (uint64_t)lane;
    {
        const uint16_t *pp = pop.perm + (size_t)g * M;
        for (int i = lane; i < M; i += 32) hl = mix(hl, pp[i]);
    }
    unsigned long long n_rep = 0, n_served = 0, n_paper = 0;
    double rate[2], lat[2];
    int kind[2];                                   // -1 none, 0 prefill, 1 decode
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int c = lane + 32 * h;
        kind[h] = -1;
        rate[h] = 0.0;
        lat[h] = 0.0;
        if (c < R) {
            const int slot = g * K + c;
            const uint64_t mask = si.mask[slot];
            s_off[wl][c] = si.off[slot];
            int best = -2;                         // no work: outputs written by the pre-pass
            if (mask) {
                const int m = h ? sz_hi : sz_lo;
                const int role = (int)((roles >> c) & 1ull);
                best = si.best[slot];
                unsigned long long nrun = role ? (unsigned long long)dm.b_max : 1ull;
                if (best < 0) {
                    out.master[slot] = -1; out.bsel[slot] = -1;
                    out.T[slot] = keyd(kInfKey); out.L[slot] = keyd(kInfKey);
                } else {
                    const size_t sv = (size_t)slot * dm.V + best;
                    const double T = so.T[sv];
                    out.master[slot] = so.mu[sv];
                    out.bsel[slot] = (int16_t)(role ? best + 1 : 0);
                    out.T[slot] = T;
                    lat[h] = so.L[sv];
                    out.L[slot] = lat[h];
                    if (role) nrun = (unsigned long long)(dm.b_max - best);   // variants b_max .. best+1
                    ++n_served;
                    kind[h] = role;
                    rate[h] = role ? (double)(best + 1) / T : (double)dm.NP / T;
                }
                ++n_rep;
                n_paper += nrun * paper_candidates(m, dm.N);
            }
            s_best[wl][c] = best;
        }
    }
    if (lane == 0) s_off[wl][R] = M;
    __syncwarp();
    // partition: position i belongs to the last replica c with off_c <= i
    const int16_t *split = so.layers + (size_t)g * dm.V * M;
    for (int i = lane; i < M; i += 32) {
        int lo = 0, hi = R - 1;
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (s_off[wl][mid] <= i) lo = mid;
            else hi = mid - 1;
        }
        const int best = s_best[wl][lo];
        if (best >= 0) out.layers[(size_t)g * M + i] = split[(size_t)best * M + i];
        else if (best == -1) out.layers[(size_t)g * M + i] = -1;
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) {
        n_rep += __shfl_xor_sync(0xFFFFFFFFu, n_rep, o);
        n_served += __shfl_xor_sync(0xFFFFFFFFu, n_served, o);
        n_paper += __shfl_xor_sync(0xFFFFFFFFu, n_paper, o);
    }
    if (lane == 0 && n_rep) {
        atomicAdd(&out.stats[kStReplicas], n_rep);
        atomicAdd(&out.stats[kStPaper], n_paper);
        if (n_served) atomicAdd(&out.stats[kStServed], n_served);
    }
    double PS = 0.0, DS = 0.0, PL = 0.0, DL = 0.0;   // PL, DL: rate-weighted latencies (finishing time)
    for (int c = 0; c < R; ++c) {
        const int h = c >> 5;
        const double x = __shfl_sync(0xFFFFFFFFu, h ? rate[1] : rate[0], c & 31);
        const double l = __shfl_sync(0xFFFFFFFFu, h ? lat[1] : lat[0], c & 31);
        const int k = __shfl_sync(0xFFFFFFFFu, h ? kind[1] : kind[0], c & 31);
        if (k == 0) { PS = PS + x; PL = PL + x * l; }
        else if (k == 1) { DS = DS + x; DL = DL + x * l; }
    }
    // fingerprint: lanes mixed interleaved slices of the ordering; a tree fold,
    // then the sizes in replica order (from the lanes that hold them)
#pragma unroll
    for (int o = 16; o; o >>= 1) {
        const uint64_t other = __shfl_down_sync(0xFFFFFFFFu, hl, o);
        if (lane < o) hl = mix(hl, other);
    }
    uint64_t h = hl;
    for (int i = 0; i < R; ++i) {
        const int si_ = __shfl_sync(0xFFFFFFFFu, i < 32 ? sz_lo : sz_hi, i & 31);
        h = mix(h, (uint64_t)si_ << 16);
    }
    if (lane != 0) return;
    double w, phase;
    objective(dm, PS, DS, PL, DL, w, phase);
    double *f = out.fit + (size_t)g * 4;
    f[0] = w; f[1] = phase; f[2] = PS; f[3] = DS;
    h = mix(h, (uint64_t)R << 40);
    h = mix(h, roles);
    out.hash[g] = h;
    atomicAdd(&out.stats[kStGenomes], 1ull);
}

// Alg. 2's role search, one warp per genome (or a block, below).  The lead
// warp reads every replica's two results (lane l: replicas l and l + 32): the
// prefill run (variant bit b_max, run when the memory allows) and the decode
// sweep's answer (the largest accepted batch).  Every role assignment r (bit
// c = 1: replica c decodes) is scored with the objective (PS and DS summed in
// ascending replica order over the replicas that serve their role); the least
// (objective, phase, r) wins.  Some replicas' roles are fixed in the winner:
// one that serves neither role has its bit clear (it adds nothing either way,
// and the smaller mask wins); under the waiting time, one that cannot decode
// prefills (clearing its bit keeps DS and can only raise PS, since
// round-to-nearest addition is monotone, so w and the phase do not grow and
// the mask shrinks; under the finishing time a slow prefill replica can raise
// the rate-weighted mean latency, so only the first rule applies).  The
// search therefore walks the F other ("free") replicas' roles, free replica j
// being replica fr(j): compact assignments r' over j, in the order of the
// full masks they stand for.  With more than E2_MAX_ROLE_SEARCH free replicas
// the search is not run: the genome keeps its own role bits for them (the
// fixed replicas' bits clear) and is counted in the stats.  The replicas'
// outputs are those of their chosen roles, the chosen roles are written into
// the genome, and the genome is scored.
template <int WPG, bool FT>
__global__ void __launch_bounds__(128) finalize_roles_kernel(Dims dm, DevPop pop, SlotInfo si, SplitOut so,
                                                             EvalOut out)
{
    constexpr int KC = E2_MAX_CLUSTERS, KF = E2_MAX_ROLE_SEARCH;
    __shared__ double s_ps[4][KC], s_ds[4][KC];
    __shared__ double s_pl[4][KC], s_dl[4][KC];        // rate x Lambda (finishing time)
    __shared__ int s_pv[4][KC], s_dv[4][KC];
    __shared__ int s_off[4][KC + 1], s_code[4][KC];
    __shared__ long long s_qp[4][KC], s_qd[4][KC];
    __shared__ int s_fr[4][KF];                        // full index of free replica j
    __shared__ uint64_t s_free[4];                     // mask of the free replicas
    __shared__ double s_bw[4], s_bph[4];
    __shared__ unsigned long long s_wmin[4];           // the least w a warp of the genome has scored (bits)
    __shared__ uint64_t s_br[4];
    const int wl = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // WPG warps per genome: 1 (four genomes per block), or 4 (one genome per
    // block, its assignments split over the block's 128 threads)
    const int g = WPG == 1 ? (int)blockIdx.x * 4 + wl : (int)blockIdx.x;
    const int gw = WPG == 1 ? wl : 0;                  // the genome's shared-memory row
    const int id = WPG == 1 ? lane : (int)threadIdx.x; // the thread's place in its genome's search
    const bool lead = WPG == 1 || wl == 0;              // the warp that reads and writes the genome
    if (g >= dm.P) return;
    const int K = dm.K, M = dm.M, V = dm.V, bp = dm.b_max;
    const int R = pop.nclus[g];
    const uint64_t roles0 = pop.roles[g];
    // the objective of full assignment r, PS and DS (and, for the finishing
    // time, the rate-weighted latencies) summed in ascending replica order from
    // replica c0 on, the sums over replicas 0..c0-1 given
    constexpr bool ft = FT;                            // objective 1: the finishing time
    auto score_from = [&](uint64_t r, int c0, const double *pre, double &PS, double &DS, double &w,
                          double &phase) {
        PS = pre[0]; DS = pre[1];
        double PL = pre[2], DL = pre[3];
        for (int c = c0; c < R; ++c) {
            if ((r >> c) & 1ull) {
                if (s_dv[gw][c]) { DS = DS + s_ds[gw][c]; if (ft) DL = DL + s_dl[gw][c]; }
            } else if (s_pv[gw][c]) {
                PS = PS + s_ps[gw][c];
                if (ft) PL = PL + s_pl[gw][c];
            }
        }
        objective(dm, PS, DS, PL, DL, w, phase);
    };
    const double zero4[4] = {0.0, 0.0, 0.0, 0.0};
    auto score = [&](uint64_t r, double &PS, double &DS, double &w, double &phase) {
        score_from(r, 0, zero4, PS, DS, w, phase);
    };
    // ---- each replica's two results (lane l: replicas l and l + 32)
    int best[2] = {-1, -1}, pok[2] = {0, 0}, m[2] = {0, 0};
    if (lead) {
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int c = lane + 32 * h;
            if (c >= R) continue;
            const int slot = g * K + c;
            const uint64_t mask = si.mask[slot];
            m[h] = pop.sizes[slot];
            pok[h] = (int)((mask >> bp) & 1ull);
            if (pok[h] && dm.layered) pok[h] = so.T[(size_t)slot * V + bp] < keyd(kInfKey);   // the run found none
            best[h] = mask ? si.best[slot] : -1;
            s_off[gw][c] = si.off[slot];
            s_pv[gw][c] = pok[h];
            s_dv[gw][c] = best[h] >= 0;
            s_ps[gw][c] = pok[h] ? (double)dm.NP / so.T[(size_t)slot * V + bp] : 0.0;
            s_ds[gw][c] = best[h] >= 0 ? (double)(best[h] + 1) / so.T[(size_t)slot * V + best[h]] : 0.0;
            s_pl[gw][c] = pok[h] ? s_ps[gw][c] * so.L[(size_t)slot * V + bp] : 0.0;
            s_dl[gw][c] = best[h] >= 0 ? s_ds[gw][c] * so.L[(size_t)slot * V + best[h]] : 0.0;
        }
        // the free replicas: those that can decode, and under the finishing
        // time also those that can only prefill
        const bool f0 = lane < R && (best[0] >= 0 || (ft && pok[0]));
        const bool f1 = lane + 32 < R && (best[1] >= 0 || (ft && pok[1]));
        const unsigned b0 = __ballot_sync(0xFFFFFFFFu, f0), b1 = __ballot_sync(0xFFFFFFFFu, f1);
        const uint64_t fm = (uint64_t)b0 | ((uint64_t)b1 << 32);
        const uint64_t below = (1ull << lane) - 1ull;
        if (f0) { const int j = __popcll(fm & below); if (j < KF) s_fr[gw][j] = lane; }
        if (f1) { const int j = __popcll(fm & (below << 32 | 0xFFFFFFFFull)); if (j < KF) s_fr[gw][j] = lane + 32; }
        if (lane == 0) { s_off[gw][R] = M; s_free[gw] = fm; }
    }
    if (WPG == 1) __syncwarp();
    else __syncthreads();
    const uint64_t freem = s_free[gw];
    const int F = __popcll(freem);
    // a compact assignment over the free replicas -> its full mask
    auto expand = [&](uint64_t r) -> uint64_t {
        uint64_t full = 0;
        for (int j = 0; j < F; ++j)
            if ((r >> j) & 1ull) full |= 1ull << s_fr[gw][j];
        return full;
    };
    double bw = keyd(kInfKey), bph = keyd(kInfKey);
    uint64_t br = ~0ull;                                // compact
    bool capped = F > KF;
    if (!capped) {
    // ---- the best assignment.  Thread id owns the compact assignments whose
    //      first low = min(F, 5) free replicas' roles (7 with a block per
    //      genome) are the bits of id, and walks the other H = F - low free
    //      replicas' roles in Gray-code order (one role flips per step).  Along
    //      the walk PS and DS are kept as exact fixed-point sums (each rate
    //      rounded to an integer multiple of 2^-s, s per genome so that the
    //      total stays below 2^62), with the counts of replicas serving each
    //      role; the fixed replicas add constant terms.  Two screens skip
    //      assignments that can only lose (waiting time only).  (1) Integer
    //      compares: a w no larger than the best w needs NP/PS <= max(w, T_a)
    //      and ND/DS <= T_a + w (the phase exceeds T_a by at most w, and
    //      w >= NP/PS once it does), i.e. PS and DS above thresholds derived
    //      from the best, with margins for the fixed-point rounding; with a
    //      best w of 0, both must stay within the best phase.  (2) A lower
    //      bound on w and the phase from the float values of the sums, without
    //      a division (relative error below 1e-6, against a 1e-5 margin),
    //      against the best.  The others are scored exactly: PS and DS summed
    //      in float64 in ascending replica order, then the objective, as the
    //      oracle does.  The best key is shared over the warp whenever a lane
    //      improves it, so that few steps of the warp take the exact path.
    //      With at most 8 free replicas every assignment is scored exactly.
    constexpr int kFixed = WPG == 1 ? 5 : 7;            // free replicas whose roles are the bits of id
    const int low = F < kFixed ? F : kFixed, H = F - low;
    // fixed-point scales: totals below 2^62; the screen needs every serving
    // rate to be at least 2^24 units (else every assignment is scored exactly)
    double totp = 0.0, totd = 0.0;
    for (int c = 0; c < R; ++c) { totp = totp + s_ps[gw][c]; totd = totd + s_ds[gw][c]; }
    const int sp_ = totp > 0.0 ? 61 - ilogb(totp) : 0, sd_ = totd > 0.0 ? 61 - ilogb(totd) : 0;
    // the screens bound the waiting time; the finishing time is scored exactly
    bool in_range = !ft && isfinite(totp) && isfinite(totd) && sp_ > -126 + 64 && sp_ < 126 && sd_ > -126 + 64 &&
                    sd_ < 126;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int c = lane + 32 * h;
        if (c >= R) continue;
        const long long qp = in_range && s_pv[gw][c] ? __double2ll_rn(ldexp(s_ps[gw][c], sp_)) : 0ll;
        const long long qd = in_range && s_dv[gw][c] ? __double2ll_rn(ldexp(s_ds[gw][c], sd_)) : 0ll;
        if (lead) {
            s_qp[gw][c] = qp;
            s_qd[gw][c] = qd;
        }
        if ((s_pv[gw][c] && qp < (1ll << 24)) || (s_dv[gw][c] && qd < (1ll << 24))) in_range = false;
    }
    in_range = __all_sync(0xFFFFFFFFu, in_range);
    if (lead && lane == 0) s_wmin[gw] = dkey(keyd(kInfKey));
    if (WPG == 1) __syncwarp();
    else __syncthreads();
    if (F <= 8) {                                               // at most 256 assignments: score them all
        for (uint64_t r = id; r < (1ull << F); r += 32 * WPG) {
            double PS, DS, w, ph;
            score(expand(r), PS, DS, w, ph);
            if (w < bw || (w == bw && (ph < bph || (ph == bph && r < br)))) { bw = w; bph = ph; br = r; }
        }
    } else {
        auto fr = [&](int j) { return s_fr[gw][j]; };
        long long P = 0, D = 0;                                 // fixed-point PS and DS
        int np = 0, nd = 0;                                     // replicas serving prefill / decode
        for (int c = 0; c < R; ++c)                             // the fixed replicas prefill
            if (!((freem >> c) & 1ull) && s_pv[gw][c]) { P += s_qp[gw][c]; ++np; }
        for (int j = 0; j < F; ++j) {                           // free replicas above low start as prefill
            const int c = fr(j);
            const bool dec = j < low && ((id >> j) & 1);
            if (dec) { if (s_dv[gw][c]) { D += s_qd[gw][c]; ++nd; } }
            else if (s_pv[gw][c]) { P += s_qp[gw][c]; ++np; }
        }
        // float value of a fixed-point sum (truncated to 24 bits, then scaled)
        auto to_float = [](long long x, int s) -> float {
            const int lz = __clzll(x), sh = lz < 40 ? 40 - lz : 0;
            return __uint2float_rn((unsigned)(x >> sh)) * __int_as_float((127 + sh - s) << 23);
        };
        const float npf = (float)dm.NP, ndf = (float)dm.ND;
        const float ta_up = (float)dm.t_a * (1.0f + 1e-6f);
        bool finite = false, zero = false;                      // the screen's w: finite / own best w of 0
        bool improved = false;                                  // this lane found a better one
        float bw_up = 0.0f, bph_up = 0.0f;                      // the screen's w and phase, rounded up to float
        long long pthr = 0, dthr = 0;                           // screen (1): P, D below these lose
        // the screens compare with we = min(own best w, the least w any warp of
        // the genome has scored); the phase screen only with the own best
        double wsh = keyd(kInfKey);                             // the shared least w last taken
        // start from the genome's own roles over the free replicas: a real
        // assignment, scored exactly
        bool own_fin;                                           // the lane's own best w is finite
        {
            uint64_t r0 = 0;
            for (int j = 0; j < F; ++j) r0 |= ((roles0 >> fr(j)) & 1ull) << j;
            double PS, DS, w, ph;
            score(expand(r0), PS, DS, w, ph);
            bw = w; bph = ph; br = r0;
            own_fin = w < keyd(kInfKey);
            improved = true;
        }
        // one assignment: the screens, then the exact score where they cannot
        // decide.  With a block per genome the roles of free replicas
        // 0..low+1 are fixed per thread and combination: the exact sums over
        // full replicas 0..fr(low+1) are taken once (prefix)
        double pre[4][4] = {{0.0, 0.0, 0.0, 0.0}, {0.0, 0.0, 0.0, 0.0}, {0.0, 0.0, 0.0, 0.0},
                            {0.0, 0.0, 0.0, 0.0}};     // [combination][PS, DS, PL, DL]
        const int c_pre = WPG > 1 ? fr(low + 1) + 1 : 0;       // first replica after the prefix
        auto consider = [&](long long P, long long D, int np, int nd, uint64_t r, int j) {
            if (np == 0 || nd == 0) {                              // PS or DS is 0: w = phase = +inf
                if (!own_fin && r < br) br = r;                    // ties the own best only while it is +inf
                return;
            }
            if (finite && in_range) {
                if (P < pthr || D < dthr) return;
                const float tp = npf * __frcp_rn(to_float(P, sp_)), td = ndf * __frcp_rn(to_float(D, sd_));
                const float ph_lo = fmaxf(tp, td) * (1.0f - 1e-5f);
                const float w_lo = ph_lo > ta_up ? (tp * (1.0f - 1e-5f) + ph_lo) - ta_up : 0.0f;
                if (w_lo > bw_up || (zero && ph_lo > bph_up)) return;
            }
            double PS, DS, w, ph;
            if (WPG > 1) score_from(expand(r), c_pre, pre[j], PS, DS, w, ph);
            else score(expand(r), PS, DS, w, ph);
            if (w < bw || (w == bw && (ph < bph || (ph == bph && r < br)))) {
                bw = w; bph = ph; br = r;
                own_fin = true;                                    // PS, DS > 0: w is finite
                improved = true;
            }
        };
        // the first U = min(H, 2) walked free replicas are taken in all 2^U
        // combinations at every step (independent work for the lane); the
        // Gray code walks the other H - U
        const int U = H < 2 ? H : 2;                            // 2 with a block per genome (F >= 9)
        if (WPG > 1)
            for (int j = 0; j < 4; ++j)
                for (int c = 0; c < c_pre; ++c) {
                    bool dec = false;                               // fixed replicas prefill
                    if ((freem >> c) & 1ull) {
                        const int jj = __popcll(freem & ((1ull << c) - 1ull));   // its free index (< low + 2)
                        dec = jj < low ? ((id >> jj) & 1) : ((j >> (jj - low)) & 1);
                    }
                    if (dec) {
                        if (s_dv[gw][c]) {
                            pre[j][1] = pre[j][1] + s_ds[gw][c];
                            if (ft) pre[j][3] = pre[j][3] + s_dl[gw][c];
                        }
                    } else if (s_pv[gw][c]) {
                        pre[j][0] = pre[j][0] + s_ps[gw][c];
                        if (ft) pre[j][2] = pre[j][2] + s_pl[gw][c];
                    }
                }
        long long dP[2] = {0, 0}, dD[2] = {0, 0};
        int dn[2] = {0, 0}, dm_[2] = {0, 0};
        for (int j = 0; j < U; ++j) {                           // free replica low + j: prefill -> decode
            const int c = fr(low + j);
            dP[j] = -s_qp[gw][c]; dD[j] = s_qd[gw][c];
            dn[j] = -s_pv[gw][c]; dm_[j] = s_dv[gw][c];
        }
        uint64_t gq = 0;                                        // Gray code of the outer step
        const uint64_t nq = 1ull << (H - U);
        for (uint64_t q = 0;; ) {
            const uint64_t rb = (uint64_t)id | (gq << (low + U));
            consider(P, D, np, nd, rb, 0);
            if (U >= 1) consider(P + dP[0], D + dD[0], np + dn[0], nd + dm_[0], rb | (1ull << low), 1);
            if (U >= 2) {
                consider(P + dP[1], D + dD[1], np + dn[1], nd + dm_[1], rb | (2ull << low), 2);
                consider(P + dP[0] + dP[1], D + dD[0] + dD[1], np + dn[0] + dn[1], nd + dm_[0] + dm_[1],
                         rb | (3ull << low), 3);
            }
            // every lane screens against the warp's best: when a lane improved
            // on its own, the best key (w, phase, r) is shared (all 32 lanes
            // run the same number of steps once F >= 5)
            if (H > 0 && __any_sync(0xFFFFFFFFu, improved)) {
#pragma unroll
                for (int o = 16; o; o >>= 1) {
                    const double ow = __shfl_xor_sync(0xFFFFFFFFu, bw, o), op = __shfl_xor_sync(0xFFFFFFFFu, bph, o);
                    const uint64_t orr = __shfl_xor_sync(0xFFFFFFFFu, br, o);
                    if (ow < bw || (ow == bw && (op < bph || (op == bph && orr < br)))) { bw = ow; bph = op; br = orr; }
                }
                improved = true;                                    // every lane's best may have changed
                own_fin = bw < keyd(kInfKey);
                if (lane == 0 && own_fin) atomicMin(&s_wmin[gw], (unsigned long long)dkey(bw));
            }
            {                                                       // another warp's better w
                const double ws = keyd(*reinterpret_cast<volatile unsigned long long *>(&s_wmin[gw]));
                if (ws < wsh) { wsh = ws; improved = true; }
            }
            if (improved) {                                         // the float copies of the screen's state
                improved = false;
                const double we = bw < wsh ? bw : wsh;
                if (we < keyd(kInfKey)) {
                    finite = true;
                    zero = bw == 0.0;
                    bw_up = (float)we;
                    if ((double)bw_up < we) bw_up = nextafterf(bw_up, HUGE_VALF);
                    bph_up = (float)bph;
                    if ((double)bph_up < bph) bph_up = nextafterf(bph_up, HUGE_VALF);
                    if (in_range) {
                        // PS >= NP / max(w, T_a) and DS >= ND / (T_a + w) for a w no larger than
                        // we (with an own best w of 0: both phases within its phase), less
                        // 1e-9 relative and R units
                        const double ptp = zero ? bph : (we > dm.t_a ? we : dm.t_a);
                        const double ptd = zero ? bph : dm.t_a + we;
                        const double pmin = ldexp((double)dm.NP / ptp, sp_) * (1.0 - 1e-9);
                        const double dmin = ldexp((double)dm.ND / ptd, sd_) * (1.0 - 1e-9);
                        pthr = pmin < 4e18 ? (long long)pmin - R : (long long)4e18;
                        dthr = dmin < 4e18 ? (long long)dmin - R : (long long)4e18;
                    }
                }
            }
            if (++q == nq) break;
            // the next Gray code flips bit t: free replica low + U + t changes role
            const int t = __ffsll((long long)q) - 1, c = fr(low + U + t);
            gq ^= 1ull << t;
            const long long qp = s_qp[gw][c], qd = s_qd[gw][c];     // 0 where the role is not served
            const int pv = s_pv[gw][c], dv = s_dv[gw][c];
            if ((gq >> t) & 1ull) { P -= qp; D += qd; np -= pv; nd += dv; }   // prefill -> decode
            else { P += qp; D -= qd; np += pv; nd -= dv; }                     // decode -> prefill
        }
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) {
        const double ow = __shfl_xor_sync(0xFFFFFFFFu, bw, o), op = __shfl_xor_sync(0xFFFFFFFFu, bph, o);
        const uint64_t orr = __shfl_xor_sync(0xFFFFFFFFu, br, o);
        if (ow < bw || (ow == bw && (op < bph || (op == bph && orr < br)))) { bw = ow; bph = op; br = orr; }
    }
    if (WPG > 1) {                                      // the best of the genome's warps
        if (lane == 0) { s_bw[wl] = bw; s_bph[wl] = bph; s_br[wl] = br; }
        __syncthreads();
        if (wl != 0) return;
        for (int o = 1; o < WPG; ++o) {
            const double ow = s_bw[o], op = s_bph[o];
            const uint64_t orr = s_br[o];
            if (ow < bw || (ow == bw && (op < bph || (op == bph && orr < br)))) { bw = ow; bph = op; br = orr; }
        }
    }
    }  // !capped
    else if (!lead) {
        return;
    }
    // ---- outputs of the chosen roles (the genome's first warp)
    const uint64_t brf = capped ? (roles0 & freem) : expand(br);
    unsigned long long n_rep = 0, n_served = 0, n_paper = 0;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int c = lane + 32 * h;
        if (c >= R) continue;
        const int slot = g * K + c;
        const int role = (int)((brf >> c) & 1ull);
        const int code = role ? best[h] : (pok[h] ? bp : -1);
        s_code[gw][c] = code;
        if (code < 0) {
            out.master[slot] = -1; out.bsel[slot] = -1;
            out.T[slot] = keyd(kInfKey); out.L[slot] = keyd(kInfKey);
        } else {
            const size_t sv = (size_t)slot * V + code;
            out.master[slot] = so.mu[sv];
            out.bsel[slot] = (int16_t)(role ? code + 1 : 0);
            out.T[slot] = so.T[sv];
            out.L[slot] = so.L[sv];
            ++n_served;
        }
        if (si.mask[slot]) {                         // replicas with no work were counted by the pre-pass
            const unsigned long long ndec = best[h] >= 0 ? (unsigned long long)(bp - best[h]) : (unsigned long long)bp;
            ++n_rep;
            n_paper += (1 + ndec) * paper_candidates(m[h], dm.N);
        }
    }
    __syncwarp();
    const int16_t *split = so.layers + (size_t)g * V * M;
    for (int i = lane; i < M; i += 32) {
        int lo = 0, hi = R - 1;
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (s_off[gw][mid] <= i) lo = mid;
            else hi = mid - 1;
        }
        const int code = s_code[gw][lo];
        out.layers[(size_t)g * M + i] = code >= 0 ? split[(size_t)code * M + i] : (int16_t)-1;
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) {
        n_rep += __shfl_xor_sync(0xFFFFFFFFu, n_rep, o);
        n_served += __shfl_xor_sync(0xFFFFFFFFu, n_served, o);
        n_paper += __shfl_xor_sync(0xFFFFFFFFu, n_paper, o);
    }
    // fingerprint of the genome with its chosen roles (a tree fold over the lanes)
    uint64_t hl = 0x9E3779B97F4A7C15ull ^ (uint64_t)lane;
    auto mix = [](uint64_t h, uint64_t x) { h = (h ^ x) * 0xBF58476D1CE4E5B9ull; return h ^ (h >> 31); };
    const uint16_t *pp = pop.perm + (size_t)g * M;
    for (int i = lane; i < M; i += 32) hl = mix(hl, pp[i]);
#pragma unroll
    for (int o = 16; o; o >>= 1) {
        const uint64_t other = __shfl_down_sync(0xFFFFFFFFu, hl, o);
        if (lane < o) hl = mix(hl, other);
    }
    if (lane != 0) return;
    if (n_rep) {
        atomicAdd(&out.stats[kStReplicas], n_rep);
        atomicAdd(&out.stats[kStPaper], n_paper);
    }
    if (n_served) atomicAdd(&out.stats[kStServed], n_served);
    if (capped) atomicAdd(&out.stats[kStRoleCapped], 1ull);
    double PS, DS, w, phase;
    score(brf, PS, DS, w, phase);
    double *f = out.fit + (size_t)g * 4;
    f[0] = w; f[1] = phase; f[2] = PS; f[3] = DS;
    pop.roles[g] = brf;
    uint64_t h = hl;
    const uint16_t *ss = pop.sizes + (size_t)g * K;
    for (int i = 0; i < R; ++i) h = mix(h, (uint64_t)ss[i] << 16);
    h = mix(h, (uint64_t)R << 40);
    h = mix(h, brf);
    out.hash[g] = h;
    atomicAdd(&out.stats[kStGenomes], 1ull);
}

// The adapted-SplitWise rule of the paper's comparison (Sec. 4.2, "Baseline
// chosen"), one warp per genome; lane l holds replicas l and l + 32.  Every
// replica was evaluated in both roles (as for the role search): its prefill
// run (variant bit b_max, present when the memory allows) and its decode
// sweep's answer (the largest accepted batch).  A replica's strength is its
// prefill throughput NP/T (-1 when it cannot prefill); the n_P strongest
// replicas prefill (ties to the lower index), the rest decode, with
// n_P = R NP / (NP + ND) rounded half up and clamped to [1, R-1] (R = 1: 1).
// The replicas' outputs are those of their roles, the roles are written into
// the genome, and the genome is scored.
__global__ void __launch_bounds__(128) finalize_splitwise_kernel(Dims dm, DevPop pop, SlotInfo si, SplitOut so,
                                                                 EvalOut out)
{
    __shared__ int s_off[4][E2_MAX_CLUSTERS + 1];     // replica start in the ordering
    __shared__ int s_code[4][E2_MAX_CLUSTERS];        // variant bit of the chosen role's result, -1 none
    const int wl = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int g = blockIdx.x * 4 + wl;
    if (g >= dm.P) return;
    const int K = dm.K, M = dm.M, V = dm.V, bp = dm.b_max;
    const int R = pop.nclus[g];
    double strength[2];
    int pok[2], best[2], m[2];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int c = lane + 32 * h;
        strength[h] = -1.0;
        pok[h] = 0;
        best[h] = -1;
        m[h] = 0;
        if (c < R) {
            const int slot = g * K + c;
            const uint64_t mask = si.mask[slot];
            m[h] = pop.sizes[slot];
            pok[h] = (int)((mask >> bp) & 1ull);
            if (pok[h] && dm.layered) pok[h] = so.T[(size_t)slot * V + bp] < keyd(kInfKey);   // the run found none
            best[h] = mask ? si.best[slot] : -1;
            s_off[wl][c] = si.off[slot];
            if (pok[h]) strength[h] = (double)dm.NP / so.T[(size_t)slot * V + bp];
        }
    }
    if (lane == 0) s_off[wl][R] = M;
    // prefill count from the token ratio, in integers
    int nP = R;
    if (R > 1) {
        const uint64_t den = dm.NP + dm.ND;
        nP = (int)((2ull * (uint64_t)R * dm.NP + den) / (2ull * den));
        nP = nP < 1 ? 1 : (nP > R - 1 ? R - 1 : nP);
    }
    // rank of each replica by strength (stronger first, ties to the lower index)
    int rank[2] = {0, 0};
    for (int o = 0; o < R; ++o) {
        const double so_ = __shfl_sync(0xFFFFFFFFu, o < 32 ? strength[0] : strength[1], o & 31);
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int c = lane + 32 * h;
            if (c < R && o != c && (so_ > strength[h] || (so_ == strength[h] && o < c))) ++rank[h];
        }
    }
    const unsigned dec_lo = __ballot_sync(0xFFFFFFFFu, lane < R && rank[0] >= nP);
    const unsigned dec_hi = __ballot_sync(0xFFFFFFFFu, lane + 32 < R && rank[1] >= nP);
    const uint64_t roles = (uint64_t)dec_lo | ((uint64_t)dec_hi << 32);
    // outputs of the chosen roles
    unsigned long long n_rep = 0, n_served = 0, n_paper = 0;
    double rate[2] = {0.0, 0.0}, lat[2] = {0.0, 0.0};
    int kind[2] = {-1, -1};
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int c = lane + 32 * h;
        if (c >= R) continue;
        const int slot = g * K + c;
        const int role = (int)((roles >> c) & 1ull);
        const int code = role ? best[h] : (pok[h] ? bp : -1);
        s_code[wl][c] = code;
        if (code < 0) {
            out.master[slot] = -1; out.bsel[slot] = -1;
            out.T[slot] = keyd(kInfKey); out.L[slot] = keyd(kInfKey);
        } else {
            const size_t sv = (size_t)slot * V + code;
            const double T = so.T[sv];
            out.master[slot] = so.mu[sv];
            out.bsel[slot] = (int16_t)(role ? code + 1 : 0);
            out.T[slot] = T;
            lat[h] = so.L[sv];
            out.L[slot] = lat[h];
            kind[h] = role;
            rate[h] = role ? (double)(code + 1) / T : (double)dm.NP / T;
            ++n_served;
        }
        if (si.mask[slot]) {                         // replicas with no work were counted by the pre-pass
            const unsigned long long ndec = best[h] >= 0 ? (unsigned long long)(bp - best[h]) : (unsigned long long)bp;
            ++n_rep;
            n_paper += (1 + ndec) * paper_candidates(m[h], dm.N);
        }
    }
    __syncwarp();
    const int16_t *split = so.layers + (size_t)g * V * M;
    for (int i = lane; i < M; i += 32) {
        int lo = 0, hi = R - 1;
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (s_off[wl][mid] <= i) lo = mid;
            else hi = mid - 1;
        }
        const int code = s_code[wl][lo];
        out.layers[(size_t)g * M + i] = code >= 0 ? split[(size_t)code * M + i] : (int16_t)-1;
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) {
        n_rep += __shfl_xor_sync(0xFFFFFFFFu, n_rep, o);
        n_served += __shfl_xor_sync(0xFFFFFFFFu, n_served, o);
        n_paper += __shfl_xor_sync(0xFFFFFFFFu, n_paper, o);
    }
    double PS = 0.0, DS = 0.0, PL = 0.0, DL = 0.0;
    for (int c = 0; c < R; ++c) {
        const int h = c >> 5;
        const double x = __shfl_sync(0xFFFFFFFFu, h ? rate[1] : rate[0], c & 31);
        const double l = __shfl_sync(0xFFFFFFFFu, h ? lat[1] : lat[0], c & 31);
        const int k = __shfl_sync(0xFFFFFFFFu, h ? kind[1] : kind[0], c & 31);
        if (k == 0) { PS = PS + x; PL = PL + x * l; }
        else if (k == 1) { DS = DS + x; DL = DL + x * l; }
    }
    // fingerprint of the genome with its roles (a tree fold over the lanes)
    auto mix = [](uint64_t h, uint64_t x) { h = (h ^ x) * 0xBF58476D1CE4E5B9ull; return h ^ (h >> 31); };
    uint64_t hl = 0x9E3779B97F4A7C15ull ^ (uint64_t)lane;
    const uint16_t *pp = pop.perm + (size_t)g * M;
    for (int i = lane; i < M; i += 32) hl = mix(hl, pp[i]);
#pragma unroll
    for (int o = 16; o; o >>= 1) {
        const uint64_t other = __shfl_down_sync(0xFFFFFFFFu, hl, o);
        if (lane < o) hl = mix(hl, other);
    }
    if (lane != 0) return;
    if (n_rep) {
        atomicAdd(&out.stats[kStReplicas], n_rep);
        atomicAdd(&out.stats[kStPaper], n_paper);
    }
    if (n_served) atomicAdd(&out.stats[kStServed], n_served);
    double w, phase;
    objective(dm, PS, DS, PL, DL, w, phase);
    double *f = out.fit + (size_t)g * 4;
    f[0] = w; f[1] = phase; f[2] = PS; f[3] = DS;
    pop.roles[g] = roles;
    uint64_t h = hl;
    const uint16_t *ss = pop.sizes + (size_t)g * K;
    for (int i = 0; i < R; ++i) h = mix(h, (uint64_t)ss[i] << 16);
    h = mix(h, (uint64_t)R << 40);
    h = mix(h, roles);
    out.hash[g] = h;
    atomicAdd(&out.stats[kStGenomes], 1ull);
}

// The G--C split of the plans (Sec. 4.3) under GPU-CPU offload, one warp per
// genome: of the n blocks at ordering position i, the ones in the device's own
// memory, min(n, capg), for the variant its replica serves (bsel: 0 prefill,
// b decode) and whether the device is the replica's master; -1 where the
// replica cannot serve.  Runs after the replicas' outputs are final.
__global__ void __launch_bounds__(128) gc_split_kernel(Dims dm, DevPop pop, const int32_t *capg, EvalOut out)
{
    __shared__ int s_off[4][E2_MAX_CLUSTERS + 1];
    const int wl = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int g = blockIdx.x * 4 + wl;
    if (g >= dm.P) return;
    const int K = dm.K, M = dm.M;
    const int R = pop.nclus[g];
    // replica offsets: an exclusive scan of the sizes (lane l: replicas l and l + 32)
    const int s_lo = lane < R ? pop.sizes[(size_t)g * K + lane] : 0;
    const int s_hi = lane + 32 < R ? pop.sizes[(size_t)g * K + lane + 32] : 0;
    int in_lo = s_lo, in_hi = s_hi;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int a = __shfl_up_sync(0xFFFFFFFFu, in_lo, o), b = __shfl_up_sync(0xFFFFFFFFu, in_hi, o);
        if (lane >= o) { in_lo += a; in_hi += b; }
    }
    const int total_lo = __shfl_sync(0xFFFFFFFFu, in_lo, 31);
    if (lane < R) s_off[wl][lane] = in_lo - s_lo;
    if (lane + 32 < R) s_off[wl][lane + 32] = total_lo + in_hi - s_hi;
    if (lane == 0) s_off[wl][R] = M;
    __syncwarp();
    for (int i = lane; i < M; i += 32) {
        int lo = 0, hi = R - 1;
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (s_off[wl][mid] <= i) lo = mid;
            else hi = mid - 1;
        }
        const size_t slot = (size_t)g * K + lo;
        const int n = out.layers[(size_t)g * M + i];
        int16_t gb = -1;
        if (n >= 0) {
            const int v = out.bsel[slot];
            const int mf = (i - s_off[wl][lo]) == out.master[slot];
            const int d = pop.perm[(size_t)g * M + i];
            const int c = capg[((size_t)v * M + d) * 2 + mf];
            gb = (int16_t)(n < c ? n : c);
        }
        out.gpu_layers[(size_t)g * M + i] = gb;
    }
}

// Persistent grids of the DP.  Shared memory is what limits CTAs per SM when
// the largest replica's DP is big (many blocks); the replica sizes whose DP
// fits in half of it then form class 1, launched with that smaller allocation
// and a grid of as many CTAs as fit, where this raises the CTAs per SM.
// The probe counts of c_span_probes (a function of W alone).
static cudaError_t load_span_probes()
{
    static uint16_t t[3][E2_MAX_BLOCKS + 1];
    for (int i = 0; i < 3; ++i) {
        const int T = 32 << i;
        t[i][0] = 0;
        for (int W = 1; W <= E2_MAX_BLOCKS; ++W) {
            const int per = (W + T - 1) / T, spans = (W + per - 1) / per;
            unsigned n = (unsigned)(W - spans);
            for (int j = 0; j < spans; ++j) {
                unsigned bits = 0;
                for (unsigned x = (unsigned)(j * per + 1); x; x >>= 1) ++bits;   // floor(log2(r + 1)) + 1
                n += bits;
            }
            t[i][W] = (uint16_t)n;
        }
    }
    return cudaMemcpyToSymbol(c_span_probes, t, sizeof t);
}

cudaError_t configure_eval(e2_ctx *c)
{
    cudaError_t e = load_span_probes();
    if (e != cudaSuccess) return e;
    if (c->dm.layered) {                         // the plain-scan path: one launch, one class
        const void *lk = reinterpret_cast<const void *>(dp_layered_kernel);
        e = cudaFuncSetAttribute(lk, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)c->dp_smem);
        if (e != cudaSuccess) return e;
        int per_sm = 0, sms = 0;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, lk, c->dp_threads, c->dp_smem);
        if (e != cudaSuccess) return e;
        e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, c->device);
        if (e != cudaSuccess) return e;
        c->dp_grid = (per_sm > 0 ? per_sm : 1) * (sms > 0 ? sms : 1);
        c->dm.dp_warps = c->dp_threads / 32;
        c->dm.dp_small = 0;
        c->dp_warp1 = 0;
        c->dp_grid1 = 0;
        c->dp_smem1 = 0;
        return cudaSuccess;
    }
    // class 0 runs every replica size (spilling its suffix columns where that
    // raises its occupancy); class 1, where it raises the occupancy of the
    // sizes it takes, runs the small ones without spilling
    const void *kernel = c->dm.g_spill ? reinterpret_cast<const void *>(dp_eval_kernel<true>)
                                       : reinterpret_cast<const void *>(dp_eval_kernel<false>);
    const void *kernel1 = reinterpret_cast<const void *>(dp_eval_kernel<false>);
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)c->dp_smem);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributePreferredSharedMemoryCarveout, cudaSharedmemCarveoutMaxShared);
    if (e != cudaSuccess) return e;
    int per_sm = 0, per_sm1 = 0, sms = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, c->dp_threads, c->dp_smem);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, c->device);
    if (e != cudaSuccess) return e;
    if (sms < 1) sms = 1;
    c->dp_grid = (per_sm > 0 ? per_sm : 1) * sms;
    const int warps = c->dp_threads / 32, mmax = c->dm.M < c->dm.N ? c->dm.M : c->dm.N;
    size_t small = 0;
    if (!c->dm.g_spill) {
        // the sizes whose run fits in half the largest one's shared memory
        for (int m = 1; m <= mmax; ++m) {
            const size_t b = dp_item_bytes(m, c->dm.N, warps, 4, false);
            if (2 * b <= c->dp_smem && b > small) small = b;
        }
    } else {
        // the non-spilling kernel's best occupancy (its registers' limit), and the
        // largest size that keeps it
        e = cudaFuncSetAttribute(kernel1, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)c->dp_smem);
        if (e != cudaSuccess) return e;
        e = cudaFuncSetAttribute(kernel1, cudaFuncAttributePreferredSharedMemoryCarveout,
                                 cudaSharedmemCarveoutMaxShared);
        if (e != cudaSuccess) return e;
        int best1 = 0;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&best1, kernel1, c->dp_threads, 16);
        if (e != cudaSuccess) return e;
        for (int m = 1; m <= mmax; ++m) {
            const size_t b = dp_item_bytes(m, c->dm.N, warps, 4, false);
            if (b <= small || b > c->dp_smem) continue;
            int occ = 0;
            e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, kernel1, c->dp_threads, b);
            if (e != cudaSuccess) return e;
            if (occ >= best1) small = b;
        }
    }
    c->dm.dp_warps = warps;
    c->dm.dp_small = 0;
    c->dp_grid1 = 0;
    c->dp_smem1 = 0;
    if (small > 0) {
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm1, kernel1, c->dp_threads, small);
        if (e != cudaSuccess) return e;
        if (per_sm1 > per_sm) {
            c->dm.dp_small = (unsigned)small;
            c->dp_grid1 = per_sm1 * sms;
            c->dp_smem1 = small;
        }
    }
    // without a four-warp class 1, the small sizes may run one per warp: the
    // largest per-warp slice whose runs in flight per SM are at least twice
    // class 0's (its CTAs per SM).  A warp's run takes longer than a CTA's, so
    // this pays only with many runs per warp: the population's slots at least
    // eight times the class's runs in flight on the GPU.
    c->dp_warp1 = 0;
    if (c->dm.dp_small == 0) {
        size_t wslice = 0;
        int wocc = 0;
        for (int m = 1; m <= mmax; ++m) {
            const size_t b = dp_item_bytes(m, c->dm.N, 1, 4, false);
            if (b <= wslice || b > c->dp_smem) continue;
            int occ = 0;
            e = dp_warp_occupancy((unsigned)b, &occ);
            if (e != cudaSuccess) return e;
            if (occ * kDpWarpRuns >= 2 * per_sm) { wslice = b; wocc = occ; }
        }
        const long long slots = (long long)c->dm.P * c->dm.K;
        if (wslice > 0 && slots < 8LL * kDpWarpRuns * wocc * sms) wslice = 0;
        if (wslice > 0) {
            e = dp_warp_occupancy((unsigned)wslice, &wocc);
            if (e != cudaSuccess) return e;
            c->dm.dp_small = (unsigned)wslice;
            c->dm.dp_warps = 1;
            c->dp_warp1 = 1;
            c->dp_grid1 = wocc * sms;
            c->dp_smem1 = wslice;
        }
    }
    if (c->dm.g_spill && c->dp_grid > kSpillCtas) c->dp_grid = kSpillCtas;   // the scratch holds kSpillCtas CTAs
    c->dm.dp_grid0 = c->dp_grid;
    return cudaSuccess;
}

cudaError_t launch_eval(const e2_ctx *c, const DevPop &p)
{
    Tables tb{c->rate, c->bw, c->mem, c->rate_cpu, c->bw_cpu, c->mem_cpu, c->prof, c->leaf, c->tau, c->cap,
              c->capg, c->cpb, c->tau_lb, c->leaf_rank, c->tau_rank, c->lcost};
    EvalOut out{c->fit, c->layers, c->master, c->bsel, c->T, c->L, c->hash, c->stats, c->gpu_layers};
    SlotInfo si{c->slot_off, c->slot_mask, c->slot_size, c->slot_best};
    WorkList wl{c->items, c->order_bins, c->gspill, (unsigned)c->spill_stride};
    SplitOut so{c->split_T, c->split_L, c->split_mu, c->split_layers};
    const long long slots = (long long)c->dm.P * c->dm.K;
    cudaError_t e = cudaMemsetAsync(c->order_bins, 0, sizeof(unsigned) * kCtrlWords, c->stream);
    if (e != cudaSuccess) return e;
    const unsigned gb = (unsigned)((slots + 255) / 256 < 1024 ? (slots + 255) / 256 : 1024);
    const int mcap = c->dm.M < c->dm.N ? c->dm.M : c->dm.N;
    slot_kernel<<<(unsigned)((slots + 1) / 2), 64, 2 * variant_stride(mcap), c->stream>>>(c->dm, tb, p, si, out,
                                                                                      c->order_bins);
    bins_kernel<<<1, 32, 0, c->stream>>>(c->dm, c->order_bins);
    order_scatter_kernel<<<gb, 256, 0, c->stream>>>(c->dm, p, si, wl);
    // while a launch sequence is being recorded, the timing events become
    // event-record nodes of the graph (an ordinary record would only mark a
    // dependency)
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (c->ev_dp_start && (e = cudaStreamIsCapturing(c->stream, &cs)) != cudaSuccess) return e;
    const unsigned rec = cs == cudaStreamCaptureStatusActive ? cudaEventRecordExternal : cudaEventRecordDefault;
    if (c->ev_dp_start && (e = cudaEventRecordWithFlags(c->ev_dp_start, c->stream, rec)) != cudaSuccess) return e;
    // a four-warp class 1 runs beside class 0, on the side stream; the
    // warp-per-run class runs after it on the context's stream (sharing the
    // SMs with class 0's CTAs was slower: DP +4.6% at c3, +2.3% at c5)
    const bool beside = c->dp_grid1 > 0 && !c->dp_warp1;
    if (beside) {
        if ((e = cudaEventRecord(c->ev_dp_fork, c->stream)) != cudaSuccess) return e;
        if ((e = cudaStreamWaitEvent(c->side, c->ev_dp_fork, 0)) != cudaSuccess) return e;
    }
    if (c->dm.layered)
        dp_layered_kernel<<<(unsigned)c->dp_grid, c->dp_threads, c->dp_smem, c->stream>>>(c->dm, tb, p, out, wl, si, so);
    else if (c->dm.g_spill)
        dp_eval_kernel<true><<<(unsigned)c->dp_grid, c->dp_threads, c->dp_smem, c->stream>>>(c->dm, tb, p, out, wl, si,
                                                                                           so, 0);
    else
        dp_eval_kernel<false><<<(unsigned)c->dp_grid, c->dp_threads, c->dp_smem, c->stream>>>(c->dm, tb, p, out, wl, si,
                                                                                            so, 0);
    if (c->dp_grid1 > 0) {                       // class 1: the small sizes, never spilling
        if (c->dp_warp1)
            e = dp_warp_launch(c->dp_grid1, (unsigned)c->dp_smem1, c->stream, c->dm, tb, p, out, wl, si, so);
        else
            dp_eval_kernel<false><<<(unsigned)c->dp_grid1, c->dp_threads, c->dp_smem1, c->side>>>(c->dm, tb, p, out,
                                                                                                wl, si, so, 1);
        if (e == cudaSuccess) e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    if (beside) {
        if ((e = cudaEventRecord(c->ev_dp_join, c->side)) != cudaSuccess) return e;
        if ((e = cudaStreamWaitEvent(c->stream, c->ev_dp_join, 0)) != cudaSuccess) return e;
    }
    if (c->ev_dp_stop && (e = cudaEventRecordWithFlags(c->ev_dp_stop, c->stream, rec)) != cudaSuccess) return e;
    const unsigned fb = (unsigned)(((size_t)c->dm.P * 32 + 127) / 128);
    if (c->dm.role_search == 2)
        finalize_splitwise_kernel<<<fb, 128, 0, c->stream>>>(c->dm, p, si, so, out);
    else if (c->dm.role_search && c->dm.K >= 12) {    // up to 2^K_max assignments: a block per genome
        if (c->dm.objective == 1) finalize_roles_kernel<4, true><<<(unsigned)c->dm.P, 128, 0, c->stream>>>(c->dm, p, si, so, out);
        else finalize_roles_kernel<4, false><<<(unsigned)c->dm.P, 128, 0, c->stream>>>(c->dm, p, si, so, out);
    } else if (c->dm.role_search) {
        if (c->dm.objective == 1) finalize_roles_kernel<1, true><<<fb, 128, 0, c->stream>>>(c->dm, p, si, so, out);
        else finalize_roles_kernel<1, false><<<fb, 128, 0, c->stream>>>(c->dm, p, si, so, out);
    }
    else finalize_score_kernel<<<fb, 128, 0, c->stream>>>(c->dm, p, si, so, out);
    c->launches += c->dp_grid1 > 0 ? 6 : 5;
    if (c->dm.offload) {
        gc_split_kernel<<<fb, 128, 0, c->stream>>>(c->dm, p, c->capg, out);
        ++c->launches;
    }
    return cudaGetLastError();
}

}  // namespace e2
