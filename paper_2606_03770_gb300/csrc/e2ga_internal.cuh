// e2ga_internal.cuh -- device-side layout and helpers shared by the library's
// translation units.  Not part of the public ABI (see include/e2ga.h).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <string>

#include "e2ga.h"

namespace e2 {

// +inf as a 64-bit key.  Every time in the planner is a non-negative float64
// (or +inf), and non-negative IEEE-754 doubles order exactly like their bit
// patterns read as unsigned integers, so the DP compares 64-bit integer keys.
constexpr uint64_t kInfKey = 0x7FF0000000000000ull;

// Philox stream purposes (counter word 3).
enum Purpose : uint32_t {
    kInitPerm = 0, kInitGroup = 1, kInitRoles = 2, kSelect = 3, kCross = 4, kMutate = 5,
    kMutPerm = 6, kMutGroup = 7, kMutRoles = 8, kCong = 9
};

// Profile arrays in the workspace: kProf* index the 7 arrays of length V.
enum ProfArray { kBlkFlops = 0, kBlkBytes, kBlkMem, kHeadFlops, kHeadBytes, kHeadMem, kAct, kNumProf };

struct DevPop {
    uint16_t *perm;    // [P][M]
    uint16_t *sizes;   // [P][K]
    uint8_t *nclus;    // [P]
    uint64_t *roles;   // [P]
};

// Largest replica (devices) a DP can receive: replicas with more devices than
// blocks are infeasible, and the evaluation pre-pass stages up to 256 devices
// of a replica per warp in shared memory.
constexpr int kMaxReplicaDevices = 256;

// Buckets of the work ordering of the evaluation: 64 levels (the rank of a
// variant among its replica's variants, largest batch first) x 16 work sizes,
// once per shared-memory class of the DP (class 0: every replica size; class
// 1, where it exists: the sizes whose DP fits in the smaller allocation that
// lets more CTAs share an SM).
constexpr int kOrderBins = 1024;
constexpr int kSizeBins = 16;
constexpr int kDpClasses = 2;
constexpr int kAllBins = kDpClasses * kOrderBins;
// Control words after the ordering bins: where each class's items end (class
// 1's follow class 0's), each class's DP cursor (starting where its items
// start), the pre-pass's warp ticket.
enum CtrlWord { kCtrlEnd = kAllBins, kCtrlNext = kCtrlEnd + kDpClasses, kCtrlTicket = kCtrlNext + kDpClasses,
                kCtrlWords };

// Shared memory of one DP run on a replica of m devices over N blocks, with
// `warps` warps per CTA and `key_bytes`-byte order keys: the per-device
// counters, the cost rows and the prefix and suffix columns ([m][W] each),
// the per-warp rows, the head row, the empty stage, the link and head keys and
// the device ids (rounded up to 16 bytes).  No slack: a few bytes more per CTA
// can cost a CTA per SM (the 80-block model's largest DP, 22,208 B, fits 10
// per SM; 16 B more fit 9).
//
// With `spill` the suffix columns live in a global scratch (L2) and shared
// memory keeps two of them (the chain's previous and current column) plus a
// per-warp buffer the master combine stages its suffix column into: about a
// third less shared memory for the large replicas, and more CTAs per SM.
__host__ __device__ __forceinline__ unsigned dp_item_bytes(int m, int N, int warps, int key_bytes, bool spill = false)
{
    const unsigned W = (unsigned)(N - m + 1);
    const unsigned gcols = spill ? 2u : (unsigned)m;
    const unsigned keys = 2u * (unsigned)m * W + gcols * W + (unsigned)((spill ? 3 : 2) * warps + 2) * W +
                          2u * (unsigned)m;
    const unsigned bytes = (unsigned)m * 12u + keys * (unsigned)key_bytes + (unsigned)m * 2u;
    return (bytes + 15u) & ~15u;
}

// Whether the DP spills its suffix columns (see dp_item_bytes): when the
// largest replica's run would otherwise need more than kSpillAbove bytes of
// shared memory (fewer than five CTAs per SM), as with the 126-block model.
// A function of the sizes alone, so that the workspace size can include the
// scratch: kSpillCtas persistent CTAs at most, each with room for the largest
// run's suffix columns.
constexpr unsigned kSpillAbove = 40u * 1024u;
// Slots of the duplicate test's fingerprint table: the power of two >= 2P.
__host__ __device__ __forceinline__ unsigned dup_table_size(int P)
{
    unsigned t = 2;
    while (t < 2u * (unsigned)P) t <<= 1;
    return t;
}
constexpr int kSpillCtas = 4096;
__host__ __forceinline__ bool dp_spills(int M, int N, int warps)
{
    const int mmax = M < N ? M : N;
    unsigned best = 0;
    for (int m = 1; m <= mmax; ++m) {
        const unsigned b = dp_item_bytes(m, N, warps, 4, false);
        if (b > best) best = b;
    }
    return best > kSpillAbove;
}
__host__ __forceinline__ size_t dp_spill_stride(int M, int N)   // keys per CTA: max over m of m * W
{
    const int mmax = M < N ? M : N;
    size_t best = 0;
    for (int m = 1; m <= mmax; ++m) {
        const size_t k = (size_t)m * (size_t)(N - m + 1);
        if (k > best) best = k;
    }
    return (best + 3) & ~(size_t)3;
}

// Stats slots (unsigned long long, atomically accumulated).
enum StatSlot { kStGenomes = 0, kStReplicas, kStDpRuns, kStCells, kStProbes, kStPaper, kStPrecheck,
                kStServed, kStTpsPruned, kStDpRunsSmall, kStRoleCapped, kStDeviceErrors, kNumStats };

// Everything a kernel needs, passed by value.
struct Dims {
    int M, N, V, b_max, P, Q, K;
    int LS;              // leaf row stride (>= N, even)
    int tournament;
    uint64_t NP, ND;
    double min_tps, t_a;
    double lam_max;      // largest latency Lambda with 1.0 / Lambda >= min_tps (see e2_create)
    int role_search;     // 1: both roles per replica, best assignment per genome (Alg. 2);
                         // 2: both roles per replica, the adapted-SplitWise rule picks the roles
    float lam_max_up;    // lam_max rounded up to float (the float latency bound is compared with it)
    unsigned dp_small;   // shared-memory bytes of DP class 1 (0: one class); m is in class 1 iff
                         // dp_item_bytes(m, N, dp_warps, 4, false) <= dp_small (class 1 never spills)
    int dp_warps;        // warps of a class-1 run's layout: 1 when class 1 runs one run per warp
    int grows;           // 1: block memory, head memory, block flops and bytes and activation bytes never
                         // shrink from one decode batch to the next (the pre-pass tests are then monotone)
    int objective;       // 0: waiting time w (Eq. 3-5); 1: per-request finishing time FT
    int offload;         // 1: some device has host memory for offloaded blocks
    int layered;         // 1: blocks of several types (per-layer prefix sums): the plain-scan DP path
    int g_spill;         // 1: the DP keeps its suffix columns in the global scratch (dp_item_bytes)
    int dp_grid0;        // CTAs of the first DP launch (the ones with a suffix-column scratch)
};

struct Tables {
    const double *rate, *bw;
    const uint64_t *mem;
    const double *rate_cpu, *bw_cpu;   // [M] host side of offloaded blocks (offload only)
    const uint64_t *mem_cpu;           // [M] host memory for blocks, bytes (offload only)
    const uint64_t *prof;      // [kNumProf][V]
    const double *leaf;        // [V][M][2][LS]: leaf[((v*M+d)*2+mf)*LS + n-1] = l_d(n blocks, master mf)
    const double *tau;         // [V][M][M]
    const int32_t *cap;        // [V][M][2]: most blocks device d holds (device + host memory), without / with
                               // the head
    const int32_t *capg;       // [V][M][2]: of those, the most in device memory (-1: the head does not fit)
    const float *cpb;          // [V][M]: per-block time max(blk_flops/rate, blk_bytes/bw), rounded down
    const float *tau_lb;       // [V][M][M]: tau rounded down
    const uint32_t *leaf_rank; // [V][M][2][LS]: order key of leaf within its variant's value set
    const uint32_t *tau_rank;  // [V][M][M]
    const double *lcost;       // [V][M][2][N][N] (per-layer profiles only): lcost[((v*M+d)*2+mf)*N*N + j*N + n-1]
                               // = time of blocks j..j+n-1 on device d (+inf beyond the model or memory)
};

// Per (genome, replica slot) results of the evaluation pre-pass.
struct SlotInfo {
    int32_t *off;              // [P*K] offset of the replica in the ordering chromosome
    uint64_t *mask;            // [P*K] variants to run (bit i: prefill v=0 / decode v=i+1)
    uint8_t *size;             // [P*K] log-scale work size of one DP run of the slot | DP class << 4
    int32_t *best;             // [P*K] largest variant bit accepted so far (-1: none)
};

// Work items of the DP: (slot << 8) | role << 7 | sweep << 6 | variant bit.
struct WorkList {
    uint64_t *items;           // [P*K*(b_max+1)] (slot << 8) | role << 7 | sweep << 6 | variant bit
    unsigned *ctrl;            // [kAllBins] bins/cursors, then the CtrlWord words
    uint32_t *gspill;          // [kSpillCtas][spill_stride] suffix columns of each persistent DP CTA
    unsigned spill_stride;     // keys per CTA
};

// Results of the DP runs, per (slot, variant bit).
struct SplitOut {
    double *T, *L;             // [P*K*b_max]
    int16_t *mu;               // [P*K*b_max]
    int16_t *layers;           // [P*b_max][M]
};

struct EvalOut {
    double *fit;               // [P][4]
    int16_t *layers;           // [P][M]
    int16_t *master, *bsel;    // [P][K]
    double *T, *L;             // [P][K]
    uint64_t *hash;            // [P]
    unsigned long long *stats; // [kNumStats]
    int16_t *gpu_layers;       // [P][M] blocks in device memory (offload only)
};

// ---------------------------------------------------------------------------
// Philox-4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11): ten rounds of two
// 32x32->64 multiplies of counter words 0 and 2, the high halves xored with
// the other words and the key, the key advanced by the Weyl increments
// between rounds.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint32_t k0, uint32_t k1)
{
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        if (r) { k0 += 0x9E3779B9u; k1 += 0xBB67AE85u; }
        const uint32_t lo0 = 0xD2511F53u * c.x, hi0 = __umulhi(0xD2511F53u, c.x);
        const uint32_t lo1 = 0xCD9E8D57u * c.z, hi1 = __umulhi(0xCD9E8D57u, c.z);
        c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
    }
    return c;
}

// A stream (seed, generation, slot, purpose) of 32-bit words; word t is
// component t%4 of the block with counter (t/4, slot, generation, purpose).
struct Stream {
    uint32_t k0, k1, gen, slot, purpose;
    uint32_t blk;
    uint4 cache;
    __device__ Stream(uint64_t seed, uint32_t g, uint32_t s, uint32_t p)
        : k0((uint32_t)seed), k1((uint32_t)(seed >> 32)), gen(g), slot(s), purpose(p), blk(0xFFFFFFFFu) {}
    __device__ __forceinline__ uint32_t word(uint32_t t)
    {
        const uint32_t b = t >> 2;
        if (b != blk) {
            cache = philox4x32_10(make_uint4(b, slot, gen, purpose), k0, k1);
            blk = b;
        }
        const uint32_t q = t & 3u;
        return q == 0 ? cache.x : q == 1 ? cache.y : q == 2 ? cache.z : cache.w;
    }
};

// Integer in [0, n): multiply-shift of one word (Lemire, no rejection).
__device__ __forceinline__ uint32_t below(uint32_t x, uint32_t n)
{
    return (uint32_t)(((uint64_t)x * n) >> 32);
}

__device__ __forceinline__ uint64_t dkey(double x) { return (uint64_t)__double_as_longlong(x); }
__device__ __forceinline__ double keyd(uint64_t k) { return __longlong_as_double((long long)k); }
__device__ __forceinline__ uint64_t umin64(uint64_t a, uint64_t b) { return a < b ? a : b; }
__device__ __forceinline__ uint64_t umax64(uint64_t a, uint64_t b) { return a > b ? a : b; }

}  // namespace e2

// Host-side context (opaque to callers).
struct e2_ctx {
    int device = 0;
    cudaStream_t stream = nullptr;
    cudaStream_t side = nullptr;                 // children of the generation step run here
    cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
    e2::Dims dm{};
    double cong_lo = 0, cong_hi = 0;
    uint64_t thr_cx = 0, thr_half = 0, thr_mut = 0, thr_k1 = 0, thr_k2 = 0, thr_k3 = 0;
    // device pointers (all inside the caller's workspace)
    double *rate = nullptr, *bw = nullptr;
    uint64_t *mem = nullptr;
    double *rate_cpu = nullptr, *bw_cpu = nullptr;   // host side of offload (zeros without it)
    uint64_t *mem_cpu = nullptr;
    int32_t *capg = nullptr;                          // [V][M][2] blocks in device memory
    uint64_t *psum = nullptr;                         // [3][V][N+1] per-layer prefix sums PF, PB, PM (layered)
    double *lcost = nullptr;                          // [V][M][2][N][N] per-layer stage times (layered)
    int16_t *gpu_layers = nullptr;                    // [P][M] G of the G--C split (offload only)
    double *link_bw = nullptr, *cong = nullptr;
    uint64_t *prof = nullptr;
    double *leaf = nullptr, *tau = nullptr;
    int32_t *cap = nullptr;
    float *cpb = nullptr;
    float *tau_lb = nullptr;
    uint64_t *leaf_sorted = nullptr;  // [V][pow2(2 M N)] sorted stage-time keys
    uint64_t *beff_sorted = nullptr;  // [pow2(M M)] sorted effective link bandwidths
    double *tau_sorted = nullptr;     // [V][M M] sorted link times
    uint32_t *leaf_rank = nullptr;    // [V][M][2][LS]
    uint32_t *tau_rank = nullptr;     // [V][M][M]
    e2::DevPop pop[2]{};
    int cur = 0;
    double *fit = nullptr;
    int16_t *layers = nullptr, *master = nullptr, *bsel = nullptr;
    double *T = nullptr, *L = nullptr;
    uint64_t *hash = nullptr;
    int32_t *dup = nullptr, *elite = nullptr;
    uint64_t *dup_key = nullptr;      // [dup_table_size(P)] fingerprint table of the duplicate test
    int32_t *dup_idx = nullptr;       //   and the smallest genome index of each fingerprint
    double *elite_fit = nullptr;
    unsigned long long *elite_ctl = nullptr;   // [8]: threshold key of the elite selection, counts, path flag
    int32_t *elite_cand = nullptr;             // [P] its candidates
    unsigned long long *stats = nullptr;
    int32_t *err = nullptr;
    unsigned *order_bins = nullptr;   // [kCtrlWords]
    uint64_t *items = nullptr;        // [P*K*b_max] DP work items, heaviest first
    uint32_t *gspill = nullptr;       // suffix-column scratch of the DP CTAs (dm.g_spill only)
    size_t spill_stride = 0;          // its keys per CTA
    int32_t *slot_off = nullptr;      // [P*K]
    uint64_t *slot_mask = nullptr;    // [P*K]
    uint8_t *slot_size = nullptr;     // [P*K]
    int32_t *slot_best = nullptr;     // [P*K]
    double *split_T = nullptr, *split_L = nullptr;   // [P*K*b_max]
    int16_t *split_mu = nullptr;                     // [P*K*b_max]
    int16_t *split_layers = nullptr;                 // [P*b_max*M]
    mutable unsigned long long launches = 0;   // kernels launched (a graph replay adds its kernel nodes)
    unsigned long long gen_kernels[2] = {0, 0}; // kernel nodes of each recorded generation
    int dp_grid = 0;                  // persistent DP CTAs of class 0
    int dp_grid1 = 0;                 // persistent DP CTAs of class 1 (0: one class)
    size_t dp_smem1 = 0;              // their shared memory (per warp with dp_warp1)
    int dp_warp1 = 0;                 // 1: class 1 runs one DP run per warp (dp_warp.cu)
    cudaEvent_t ev_dp_fork = nullptr, ev_dp_join = nullptr;   // class 1 runs on the side stream
    cudaEvent_t ev_dp_start = nullptr, ev_dp_stop = nullptr;   // optional timing hook
    // recorded generation (e2_run_generation), one per population buffer
    cudaStream_t cap_stream = nullptr;                          // private stream the graphs are recorded on
    cudaGraph_t gen_graph[2] = {nullptr, nullptr};
    cudaGraphExec_t gen_exec[2] = {nullptr, nullptr};
    cudaGraphNode_t gen_ga_node[2] = {nullptr, nullptr};        // the generation kernel's node
    cudaEvent_t gen_ev[2][2] = {{nullptr, nullptr}, {nullptr, nullptr}};   // timing events recorded in it
    bool gen_eager = false;                                     // recording failed: eager launches
    // launch shapes
    int dp_threads = 128;
    size_t dp_smem = 0;
    bool evaluated = false;
    bool have_elites = false;
    bool have_results = false;           // an evaluation has filled the result buffers
    std::string last_error;
};

namespace e2 {
// launchers (defined in the .cu files); return cudaGetLastError()
cudaError_t launch_tables(const e2_ctx *c);   // leaf, cap and cpb tables (and lcost for per-layer profiles)
cudaError_t launch_tau(const e2_ctx *c);
cudaError_t launch_redraw(const e2_ctx *c, uint64_t seed, uint32_t gen);
cudaError_t launch_validate(const e2_ctx *c, const DevPop &p);
cudaError_t launch_eval(const e2_ctx *c, const DevPop &p);
cudaError_t launch_init(const e2_ctx *c, const DevPop &p, uint64_t seed);
cudaError_t launch_elites(const e2_ctx *c, const DevPop &p, const DevPop &dst);
cudaError_t launch_ga(const e2_ctx *c, const DevPop &src, const DevPop &dst, uint64_t seed, uint32_t gen,
                      cudaStream_t st);
// elites and children of the next population (children on the side stream)
cudaError_t launch_step(const e2_ctx *c, const DevPop &src, const DevPop &dst, uint64_t seed, uint32_t gen);
// the generation kernel's node of a recorded graph, and new (seed, generation) for it
cudaError_t find_ga_node(cudaGraph_t graph, cudaGraphNode_t *node);
cudaError_t set_ga_node(const e2_ctx *c, cudaGraphExec_t exec, cudaGraphNode_t node, const DevPop &src,
                        const DevPop &dst, uint64_t seed, uint32_t gen);
size_t dp_smem_bytes(int M, int N, int threads, int key_bytes, bool spill = false);
// The warp-per-run DP kernel of the small replica sizes (dp_warp.cu): its CTA
// size, its CTAs per SM with `slice` bytes of shared memory per warp, and its
// launch on `stream` over class 1 of the work list.
constexpr int kDpWarpRuns = 4;
cudaError_t dp_warp_occupancy(unsigned slice, int *per_sm);
cudaError_t dp_warp_launch(int grid, unsigned slice, cudaStream_t stream, const Dims &dm, const Tables &tb,
                           const DevPop &pop, const EvalOut &out, const WorkList &wl, const SlotInfo &si,
                           const SplitOut &so);
size_t dp_layered_smem_bytes(int M, int N);   // the plain-scan DP's shared memory for the largest replica
cudaError_t configure_eval(e2_ctx *c);   // shared memory limit and persistent grid size
size_t rank_pow2(size_t n);
cudaError_t build_leaf_sorted(const e2_ctx *c);   // once per context
cudaError_t build_ranks(const e2_ctx *c);         // after every change of the link table
}  // namespace e2
