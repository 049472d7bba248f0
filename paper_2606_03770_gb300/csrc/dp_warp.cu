// dp_warp.cu -- DP_Pipe (Alg. 1, Eq. 1-2) for the small replica sizes, one
// run per warp.
//
// The four-warp kernel (dp_eval.cu) spreads a run over 128 threads and meets
// at a block barrier after every phase.  Its runs in flight per SM are bounded
// by registers and shared memory; for a small replica (a few devices) most of
// its threads idle, and its latency is the chain of columns, not their width.
// Here each warp of a CTA claims and runs its own work items from class 1 of
// the work list in its own slice of shared memory, with warp barriers only:
//  1. stage the master-free cost rows and the link keys (as dp_eval.cu);
//  2. the masters the memory allows;
//  3. prefix columns F_k on lanes 0-15 and suffix columns G_k on lanes 16-31,
//     one column of each per step (both chains have m - 2 columns);
//  4. the masters in index order, each from F_{mu-1}, G_{mu+1} and its head
//     row, skipping a master whose lower bound max(F_m[W-1], l^head_mu(1)) is
//     no better than the best so far (an equal bound loses the tie: its index
//     is larger);
//  5. mu*'s prefix columns, recomputed for the traceback;
//  6. the traceback with the smallest-split rule, T and Lambda.
// Every step computes what the four-warp kernel computes, on the same order
// keys and in the same float64 order, so the results are the same bits.
#include "e2ga_internal.cuh"
#include "dp_span.cuh"

namespace e2 {

namespace {

// Probes of the spans of one column of W cells split over T threads (the
// bisection of a span's first cell r, floor(log2(r + 1)) + 1 probes, then
// one per further cell), summed by the warp: the lanes' spans at `lanes`
// lanes of `per` cells each.
__device__ __forceinline__ int column_probes(int W, int per, int lanes, int lane)
{
    const int r0 = (lane % lanes) * per, r1 = min(W, r0 + per);
    int p = 0;
    if (lane < lanes && r0 < r1) p = (32 - __clz(r0 + 1)) + (r1 - r0 - 1);
    return warp_sum(p);
}

__global__ void __launch_bounds__(32 * kDpWarpRuns) dp_warp_kernel(Dims dm, Tables tb, DevPop pop, EvalOut out,
                                                                   WorkList wl, SlotInfo si, SplitOut so,
                                                                   unsigned slice)
{
    using Key = uint32_t;
    constexpr Key kInf = ~0u;
    constexpr unsigned kFull = 0xFFFFFFFFu;
    extern __shared__ __align__(16) unsigned char wsm[];
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    unsigned char *base = wsm + (size_t)wid * slice;
    const int K = dm.K, M = dm.M, N = dm.N;
    const unsigned n_items = wl.ctrl[kCtrlEnd + 1];
    for (;;) {
        // ---- next work item of class 1; skipped if a larger batch of its
        //      replica was accepted meanwhile (one lane reads, the warp follows)
        unsigned idx = 0;
        if (lane == 0) idx = atomicAdd(&wl.ctrl[kCtrlNext + 1], 1u);
        idx = __shfl_sync(kFull, idx, 0);
        if (idx >= n_items) break;
        const uint64_t item = wl.items[idx];
        const int slot = (int)(item >> 8), code = (int)(item & 0x3Fu);
        int done = 0;
        if (lane == 0) done = *(volatile const int32_t *)&si.best[slot] > code;
        if (__shfl_sync(kFull, done, 0)) continue;
        const int g = slot / K, c = slot - g * K;
        const size_t gk = (size_t)g * K + c;
        const int off = si.off[slot], m = pop.sizes[gk];
        const int role = (int)((item >> 7) & 1u);                 // decode
        const bool sweep = (item >> 6) & 1u;                      // the result advances the decode sweep
        int16_t *lay_out = so.layers + ((size_t)g * dm.V + code) * M + off;
        if (m > N) continue;                                      // (the pre-pass queues none)
        const int W = N - m + 1;
        // this warp's slice (the layout of dp_item_bytes(m, N, 1, 4, false))
        int *cnt0 = reinterpret_cast<int *>(base);                // [m]
        int *cnt1 = cnt0 + m;                                     // [m]
        int *nk = cnt1 + m;                                       // [m]
        Key *leaf0 = reinterpret_cast<Key *>(nk + m);             // [m][W] l_k(n)
        Key *Fst = leaf0 + (size_t)m * W;                         // [m][W] prefix / traceback columns
        Key *Gst = Fst + (size_t)m * W;                           // [m][W] suffix columns
        Key *H = Gst + (size_t)m * W;                             // [W] convolution of a master
        Key *L1 = H + W;                                          // [W] head row of a master
        Key *row1s = L1 + W;                                      // [W] head row of mu*
        Key *delta = row1s + W;                                   // [W] the empty stage
        Key *tauk = delta + W;                                    // [m] link (k-1) -> k
        Key *lbm = tauk + m;                                      // [m] l^head_k(1)
        uint16_t *devs = reinterpret_cast<uint16_t *>(lbm + m);   // [m]
        for (int k = lane; k < m; k += 32) devs[k] = pop.perm[(size_t)g * M + off + k];
        for (int r = lane; r < W; r += 32) delta[r] = r ? kInf : (Key)0;
        __syncwarp();

        auto colF = [&](int k) -> const Key * {
            return k == 0 ? delta : k == 1 ? leaf0 : Fst + (size_t)(k - 1) * W;
        };
        auto colG = [&](int k) -> const Key * {
            return k == m + 1 ? delta : k == m ? leaf0 + (size_t)(m - 1) * W : Gst + (size_t)(k - 1) * W;
        };
        const int per16 = (W + 15) >> 4, per32 = (W + 31) >> 5;
        const int chain_probes = column_probes(W, per16, 16, lane);   // one prefix + one suffix column
        const int warp_probes = column_probes(W, per32, 32, lane);
        const int lprobe = 32 - __clz(W);
        unsigned runs = 0, cells = 0, probes = 0;
        uint64_t vmask = 1ull << code;
        bool served = false;
        while (vmask && !served) {
            const int bit = 63 - __clzll((long long)vmask);           // highest batch first
            vmask &= ~(1ull << bit);
            const int v = role ? bit + 1 : 0;
            const size_t vM = (size_t)v * M;
            // ---- 1. capacities, link ranks and master-free cost rows
            for (int k = lane; k < m; k += 32) {
                const size_t vd = vM + devs[k];
                const int c0 = tb.cap[vd * 2], c1 = tb.cap[vd * 2 + 1];
                cnt0[k] = c0 < W ? c0 : W;
                cnt1[k] = c1 < W ? c1 : W;
                tauk[k] = k ? (Key)tb.tau_rank[(vM + devs[k - 1]) * M + devs[k]] : (Key)0;
                lbm[k] = (Key)tb.leaf_rank[((vM + devs[k]) * 2 + 1) * dm.LS];
            }
            for (int k = 0; k < m; ++k) stage_row(leaf0 + (size_t)k * W, tb.leaf_rank + (vM + devs[k]) * 2 * dm.LS, W, lane);
            cp_async_wait_all();
            __syncwarp();
            // ---- 2. masters the memory allows
            int S0 = 0, Z = 0;
            for (int k = lane; k < m; k += 32) { S0 += cnt0[k]; Z += cnt0[k] == 0; }
            S0 = warp_sum(S0);
            Z = warp_sum(Z);
            auto mu_ok = [&](int mu) {
                const int k = mu - 1;
                return (Z - (cnt0[k] == 0)) == 0 && cnt1[k] >= 1 && S0 - cnt0[k] + cnt1[k] >= N;
            };
            ++runs;
            // ---- 3. prefix columns on lanes 0-15, suffix columns on lanes 16-31
            {
                const int hl = lane & 15, r0 = hl * per16, r1 = min(W, r0 + per16);
                for (int i = 0; i < m - 2; ++i) {
                    if (lane < 16) {
                        const int k = i + 2;
                        dp_span(colF(k - 1), leaf0 + (size_t)(k - 1) * W, tauk[k - 1], Fst + (size_t)(k - 1) * W, r0, r1);
                    } else {
                        const int k = m - 1 - i;
                        dp_span(colG(k + 1), leaf0 + (size_t)(k - 1) * W, tauk[k], Gst + (size_t)(k - 1) * W, r0, r1);
                    }
                    __syncwarp();
                }
                if (m >= 3) {
                    cells += 2u * (unsigned)(m - 2) * (unsigned)W;
                    probes += (unsigned)(m - 2) * (unsigned)chain_probes;
                }
            }
            // V0 = F_m[W-1], the master-free optimum (the minimum over every split)
            uint32_t V0 = 0;
            if (m >= 2) {
                const Key *prev = colF(m - 1), *row = leaf0 + (size_t)(m - 1) * W;
                V0 = kInf;
                for (int q = lane; q < W; q += 32) V0 = min(V0, (uint32_t)max(prev[q], row[W - 1 - q]));
#pragma unroll
                for (int o = 16; o; o >>= 1) V0 = min(V0, __shfl_xor_sync(kFull, V0, o));
                V0 = max(V0, (uint32_t)tauk[m - 1]);
                cells += 1;
                probes += lprobe;
            }
            // ---- 4. the masters in index order; (bv, bmu) the least V so far
            uint32_t bv = kInf;
            int bmu = 0;
            for (int mu = 1; mu <= m; ++mu) {
                if (!mu_ok(mu)) continue;
                const uint32_t lb = max(V0, (uint32_t)lbm[mu - 1]);
                if (lb > bv || (lb == bv && bmu != 0)) continue;
                const uint32_t *hrow = tb.leaf_rank + ((vM + devs[mu - 1]) * 2 + 1) * dm.LS;
                HeadRow<Key> hr;
                hr.start(L1, hrow, W, lane);                          // in flight while H is built
                dp_span(colF(mu - 1), colG(mu + 1), (Key)0, H, lane * per32, min(W, (lane + 1) * per32));
                hr.finish(L1, hrow, W, lane);
                __syncwarp();
                uint32_t V = dp_cell(H, L1, (Key)0, W - 1);
                if (mu >= 2) V = max(V, (uint32_t)tauk[mu - 1]);
                if (mu <= m - 1) V = max(V, (uint32_t)tauk[mu]);
                __syncwarp();                                         // H and L1 are the next master's
                cells += W + 1;
                probes += warp_probes + lprobe;
                if (V < bv) { bv = V; bmu = mu; }                     // a tie keeps the smaller index
            }
            if (bv == kInf) {
                // as in dp_eval.cu: only a profile whose costs do not grow with
                // the batch can leave a queued run without a partition
                if (lane == 0 && (dm.grows || !role)) atomicAdd(&out.stats[kStDeviceErrors], 1ull);
                continue;
            }
            const uint32_t V = bv;
            const int mus = bmu;
            // ---- 5. mu*'s prefix columns, for the traceback
            for (int r = lane; r < W; r += 32) row1s[r] = (Key)tb.leaf_rank[((vM + devs[mus - 1]) * 2 + 1) * dm.LS + r];
            __syncwarp();
            auto rowk = [&](int k) -> const Key * { return k == mus ? row1s : leaf0 + (size_t)(k - 1) * W; };
            auto colD = [&](int k) -> const Key * {
                if (k == 1) return mus == 1 ? row1s : leaf0;
                return Fst + (size_t)(k - 1) * W;
            };
            const int k0 = mus > 2 ? mus : 2;
            for (int k = k0; k <= m - 1; ++k) {
                dp_span(colD(k - 1), rowk(k), tauk[k - 1], Fst + (size_t)(k - 1) * W, lane * per32,
                        min(W, (lane + 1) * per32));
                __syncwarp();
            }
            if (m - 1 >= k0) {
                cells += (unsigned)(m - k0) * (unsigned)W;
                probes += (unsigned)(m - k0) * (unsigned)warp_probes;
            }
            // ---- 6. traceback (smallest split on ties), T and Lambda
            int r = W - 1;
            uint32_t D = V;
            for (int k = m; k >= 2; --k) {
                const Key *row = rowk(k);
                int n = 0;                                            // #{n <= r+1 : l_k(n) <= D}
                for (int b0 = 0; b0 <= r; b0 += 32) {
                    const int p = b0 + lane;
                    const unsigned b = __ballot_sync(kFull, p <= r && row[p] <= D);
                    n += __popc(b);
                    if (b != kFull) break;
                }
                if (lane == 0) nk[k - 1] = n;
                r = r + 1 - n;
                D = colD(k - 1)[r];
            }
            if (lane == 0) nk[0] = r + 1;
            __syncwarp();
            // stage and link times of the partition (lane k holds device k),
            // Lambda summed in pipeline order
            const double *lrow = tb.leaf + vM * 2 * dm.LS;
            const double *trow = tb.tau + vM * M;
            double lam = 0.0;
            uint64_t tmax = 0;
            for (int b0 = 0; b0 < m; b0 += 32) {
                const int k = b0 + lane;
                double lk = 0.0, tk = 0.0;
                if (k < m) {
                    lk = lrow[((size_t)devs[k] * 2 + (k == mus - 1)) * dm.LS + nk[k] - 1];
                    if (k >= 1) tk = trow[(size_t)devs[k - 1] * M + devs[k]];
                    tmax = umax64(tmax, umax64(dkey(lk), dkey(tk)));
                }
                for (int q = 0; q < 32 && b0 + q < m; ++q) {
                    const double lq = __shfl_sync(kFull, lk, q);
                    const double tq = __shfl_sync(kFull, tk, q);
                    if (b0 + q == 0) lam = lq;
                    else { lam = lam + tq; lam = lam + lq; }
                }
            }
#pragma unroll
            for (int o = 16; o; o >>= 1) tmax = umax64(tmax, __shfl_xor_sync(kFull, tmax, o));
            if ((!role) || lam <= dm.lam_max) {                       // 1.0 / lam >= Min_TPS
                for (int k = lane; k < m; k += 32) lay_out[k] = (int16_t)nk[k];
                if (lane == 0) {
                    const size_t sv = gk * dm.V + code;
                    so.mu[sv] = (int16_t)(mus - 1);
                    so.T[sv] = keyd(tmax);
                    so.L[sv] = lam;
                    __threadfence();
                    if (sweep) atomicMax(&si.best[slot], code);
                }
                served = true;
            }
            __syncwarp();                                             // the next variant reuses the slice
        }
        if (lane == 0) {
            if (cells | probes) {
                atomicAdd(&out.stats[kStCells], (unsigned long long)cells);
                atomicAdd(&out.stats[kStProbes], (unsigned long long)probes);
            }
            if (runs) atomicAdd(&out.stats[kStDpRunsSmall], (unsigned long long)runs);
        }
    }
}

}  // namespace

cudaError_t dp_warp_occupancy(unsigned slice, int *per_sm)
{
    const void *k = reinterpret_cast<const void *>(dp_warp_kernel);
    const int smem = (int)(slice * kDpWarpRuns);
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(k, cudaFuncAttributePreferredSharedMemoryCarveout, cudaSharedmemCarveoutMaxShared);
    if (e != cudaSuccess) return e;
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(per_sm, k, 32 * kDpWarpRuns, (size_t)smem);
}

cudaError_t dp_warp_launch(int grid, unsigned slice, cudaStream_t stream, const Dims &dm, const Tables &tb,
                           const DevPop &pop, const EvalOut &out, const WorkList &wl, const SlotInfo &si,
                           const SplitOut &so)
{
    dp_warp_kernel<<<(unsigned)grid, 32 * kDpWarpRuns, (size_t)slice * kDpWarpRuns, stream>>>(dm, tb, pop, out, wl,
                                                                                            si, so, slice);
    return cudaGetLastError();
}

}  // namespace e2
