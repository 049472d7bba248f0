// e2ga_api.cu -- the C ABI (include/e2ga.h): input validation, workspace
// layout, table construction and the call sequence of a search.
#include <math.h>
#include <stdio.h>
#include <string.h>

#include <new>

#include "e2ga_internal.cuh"

using namespace e2;

namespace {

constexpr uint64_t kTwo53 = 1ull << 53;

// Message of the last failed e2_create on this thread (no context exists then).
thread_local char g_create_error[256] = "";

size_t align_up(size_t x, size_t a = 256) { return (x + a - 1) / a * a; }

struct Layout {
    size_t rate, bw, mem, rate_cpu, bw_cpu, mem_cpu, link_bw, cong, prof, leaf, tau, tau_lb, cap, capg, cpb,
        leaf_sorted, beff_sorted, tau_sorted, leaf_rank, tau_rank, gpu_layers, psum, lcost, gspill;
    size_t perm[2], sizes[2], nclus[2], roles[2];
    size_t fit, layers, master, bsel, T, L, hash, dup, dup_key, dup_idx, elite, elite_fit, elite_ctl, elite_cand, stats, err, order_bins, items, slot_off, slot_mask, slot_size, slot_best,
        split_T, split_L, split_mu, split_layers, total;
    int LS;
};

bool dims_ok(int32_t M, int32_t N, int32_t b_max, int32_t P, int32_t Q, int32_t K)
{
    // the evaluation's work items, P * K_max * (b_max + 1), are counted and
    // indexed in 32 bits
    return M >= 1 && M <= E2_MAX_DEVICES && N >= 1 && N <= E2_MAX_BLOCKS && b_max >= 1 &&
           b_max <= E2_MAX_BATCH && P >= 1 && P <= E2_MAX_POP && Q >= 0 && Q <= P && K >= 1 &&
           K <= E2_MAX_CLUSTERS && (uint64_t)P * (uint64_t)K * (uint64_t)(b_max + 1) < (1ull << 31);
}

Layout layout(int M, int N, int b_max, int P, int Q, int K, bool layered = false)
{
    Layout l{};
    const size_t V = (size_t)b_max + 1, MM = (size_t)M * M;
    l.LS = (N + 1) & ~1;
    size_t o = 0;
    auto take = [&](size_t bytes) { size_t at = o; o = align_up(o + bytes); return at; };
    l.rate = take(8 * (size_t)M);
    l.bw = take(8 * (size_t)M);
    l.mem = take(8 * (size_t)M);
    l.rate_cpu = take(8 * (size_t)M);
    l.bw_cpu = take(8 * (size_t)M);
    l.mem_cpu = take(8 * (size_t)M);
    l.link_bw = take(8 * MM);
    l.cong = take(8 * MM);
    l.prof = take(8 * kNumProf * V);
    l.leaf = take(8 * V * M * 2 * (size_t)l.LS);
    l.tau = take(8 * V * MM);
    l.cap = take(4 * V * M * 2);
    l.capg = take(4 * V * M * 2);
    l.cpb = take(4 * V * M);
    l.tau_lb = take(4 * V * MM);
    l.leaf_sorted = take(8 * V * rank_pow2((size_t)M * 2 * N));
    l.beff_sorted = take(8 * rank_pow2(MM));
    l.tau_sorted = take(8 * V * MM);
    l.leaf_rank = take(4 * V * M * 2 * (size_t)l.LS);
    l.tau_rank = take(4 * V * MM);
    for (int b = 0; b < 2; ++b) {
        l.perm[b] = take(2 * (size_t)P * M);
        l.sizes[b] = take(2 * (size_t)P * K);
        l.nclus[b] = take((size_t)P);
        l.roles[b] = take(8 * (size_t)P);
    }
    l.fit = take(32 * (size_t)P);
    l.layers = take(2 * (size_t)P * M);
    l.gpu_layers = take(2 * (size_t)P * M);
    l.master = take(2 * (size_t)P * K);
    l.bsel = take(2 * (size_t)P * K);
    l.T = take(8 * (size_t)P * K);
    l.L = take(8 * (size_t)P * K);
    l.hash = take(8 * (size_t)P);
    l.dup = take(4 * (size_t)P);
    l.dup_key = take(8 * (size_t)dup_table_size(P));         // fingerprint table of the duplicate test
    l.dup_idx = take(4 * (size_t)dup_table_size(P));
    l.elite = take(4 * (size_t)(Q > 0 ? Q : 1));
    l.elite_fit = take(32 * (size_t)(Q > 0 ? Q : 1));
    l.elite_ctl = take(64);                                   // the elite selection's threshold and counts
    l.elite_cand = take(4 * (size_t)P);                       // its candidate list
    l.stats = take(8 * kNumStats);
    l.err = take(4);
    l.order_bins = take(4 * (size_t)kCtrlWords);
    l.items = take(8 * (size_t)P * K * V);
    l.slot_off = take(4 * (size_t)P * K);
    l.slot_mask = take(8 * (size_t)P * K);
    l.slot_size = take((size_t)P * K);
    l.slot_best = take(4 * (size_t)P * K);
    l.split_T = take(8 * (size_t)P * K * V);                 // per (slot, variant bit): decode b = bit + 1,
    l.split_L = take(8 * (size_t)P * K * V);                 // and bit b_max = prefill when roles are searched
    l.split_mu = take(2 * (size_t)P * K * V);
    l.split_layers = take(2 * (size_t)P * V * M);
    if (layered) {
        l.psum = take(8 * 3 * V * ((size_t)N + 1));
        l.lcost = take(8 * V * M * 2 * (size_t)N * N);
    } else if (dp_spills(M, N, 4)) {
        l.gspill = take(4 * (size_t)kSpillCtas * dp_spill_stride(M, N));
    }
    l.total = o;
    return l;
}

uint64_t threshold(double p)
{
    if (!(p > 0.0)) return 0;
    if (p >= 1.0) return 4294967296ull;
    return (uint64_t)floor(p * 4294967296.0);
}

int fail(e2_ctx *c, int status, const char *msg)
{
    if (c) c->last_error = msg;
    return status;
}

int cuda_fail(e2_ctx *c, cudaError_t e, const char *where)
{
    char buf[256];
    snprintf(buf, sizeof buf, "%s: %s", where, cudaGetErrorString(e));
    if (c) c->last_error = buf;
    return E2_ECUDA;
}

#define E2_CUDA(ctx, call)                                   \
    do {                                                     \
        cudaError_t e2_err_ = (call);                        \
        if (e2_err_ != cudaSuccess) return cuda_fail((ctx), e2_err_, #call); \
    } while (0)

bool is_host(const void *p)
{
    cudaPointerAttributes a;
    if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
        cudaGetLastError();
        return true;
    }
    return a.type == cudaMemoryTypeHost || a.type == cudaMemoryTypeUnregistered;
}

bool finite_pos(double x) { return isfinite(x) && x > 0.0; }

// Host-side validation of everything e2_create receives (no CUDA call).
int validate_inputs(const e2_devices *d, const e2_links *l, const e2_layer_profile *pf, const e2_params *p,
                    char *msg, size_t n)
{
    if (!d || !l || !pf || !p) { snprintf(msg, n, "null descriptor"); return E2_EINVAL; }
    if (!dims_ok(d->M, pf->N, pf->b_max, p->P, p->Q, p->K_max)) {
        snprintf(msg, n, "sizes out of range (M=%d N=%d b_max=%d P=%d Q=%d K_max=%d)", d->M, pf->N,
                 pf->b_max, p->P, p->Q, p->K_max);
        return E2_EINVAL;
    }
    const int M = d->M, V = pf->b_max + 1;
    if (!d->rate || !d->bw || !d->mem || !l->bw || !l->cong) { snprintf(msg, n, "null array"); return E2_EINVAL; }
    const uint64_t *arr[kNumProf] = {pf->blk_flops, pf->blk_bytes, pf->blk_mem, pf->head_flops,
                                     pf->head_bytes, pf->head_mem, pf->act_bytes};
    for (int a = 0; a < kNumProf; ++a)
        if (!arr[a]) { snprintf(msg, n, "null profile array %d", a); return E2_EINVAL; }
    for (int i = 0; i < M; ++i) {
        if (!finite_pos(d->rate[i]) || !finite_pos(d->bw[i])) {
            snprintf(msg, n, "device %d: rate and bandwidth must be finite and > 0", i);
            return E2_EINVAL;
        }
    }
    if (d->mem_cpu) {
        if (!d->rate_cpu || !d->bw_cpu) { snprintf(msg, n, "mem_cpu given without rate_cpu and bw_cpu"); return E2_EINVAL; }
        for (int i = 0; i < M; ++i)
            if (d->mem_cpu[i] && (!finite_pos(d->rate_cpu[i]) || !finite_pos(d->bw_cpu[i]))) {
                snprintf(msg, n, "device %d: host rate and bandwidth must be finite and > 0 where mem_cpu > 0", i);
                return E2_EINVAL;
            }
    }
    for (int a = 0; a < M; ++a)
        for (int b = 0; b < M; ++b) {
            if (a == b) continue;
            const double bw = l->bw[(size_t)a * M + b], cg = l->cong[(size_t)a * M + b];
            if (!(bw > 0.0) || !finite_pos(cg)) {
                snprintf(msg, n, "link %d->%d: bandwidth must be > 0, congestion finite and > 0", a, b);
                return E2_EINVAL;
            }
        }
    if (!finite_pos(l->cong_lo) || !finite_pos(l->cong_hi) || l->cong_lo > l->cong_hi) {
        snprintf(msg, n, "congestion range must satisfy 0 < lo <= hi < inf");
        return E2_EINVAL;
    }
    for (int v = 0; v < V; ++v) {
        for (int a = 0; a < 3; ++a) {   // n * block + head must stay below 2^53
            const uint64_t blk = arr[a][v], head = arr[a + 3][v];
            if (head >= kTwo53 || blk > (kTwo53 - head) / (uint64_t)pf->N) {
                snprintf(msg, n, "profile variant %d: N*block + head reaches 2^53", v);
                return E2_EINVAL;
            }
        }
        if (pf->act_bytes[v] >= kTwo53) { snprintf(msg, n, "activation bytes reach 2^53"); return E2_EINVAL; }
    }
    if (pf->PF || pf->PB || pf->PM) {                 // blocks of several types: per-layer prefix sums
        if (!pf->PF || !pf->PB || !pf->PM) { snprintf(msg, n, "PF, PB and PM must be given together"); return E2_EINVAL; }
        if (pf->N > E2_MAX_LAYERED_BLOCKS) {
            snprintf(msg, n, "per-layer profiles take at most %d blocks", E2_MAX_LAYERED_BLOCKS);
            return E2_EINVAL;
        }
        const uint64_t *ps[3] = {pf->PF, pf->PB, pf->PM};
        for (int a = 0; a < 3; ++a)
            for (int v = 0; v < V; ++v) {
                const uint64_t *row = ps[a] + (size_t)v * (pf->N + 1);
                if (row[0] != 0) { snprintf(msg, n, "prefix sums must start at 0"); return E2_EINVAL; }
                for (int i = 0; i < pf->N; ++i)
                    if (row[i + 1] < row[i]) { snprintf(msg, n, "prefix sums must not decrease"); return E2_EINVAL; }
                if (row[pf->N] >= kTwo53 || arr[a + 3][v] >= kTwo53 - row[pf->N]) {
                    snprintf(msg, n, "profile variant %d: a stage's sum plus the head reaches 2^53", v);
                    return E2_EINVAL;
                }
            }
        if (d->mem_cpu)
            for (int i = 0; i < M; ++i)
                if (d->mem_cpu[i]) { snprintf(msg, n, "per-layer profiles do not take GPU-CPU offload"); return E2_EINVAL; }
    }
    if (pf->NP < 1 || pf->ND < 1 || pf->NP >= kTwo53 || pf->ND >= kTwo53) {
        snprintf(msg, n, "NP and ND must be in [1, 2^53)");
        return E2_EINVAL;
    }
    if (!(isfinite(p->min_tps) && p->min_tps >= 0) || !(isfinite(p->t_a) && p->t_a >= 0)) {
        snprintf(msg, n, "min_tps and t_a must be finite and >= 0");
        return E2_EINVAL;
    }
    const double probs[5] = {p->p_cx, p->p_mut, p->p_swap, p->p_regroup, p->p_regroup_all};
    for (double q : probs)
        if (!(q >= 0.0 && q <= 1.0)) { snprintf(msg, n, "probabilities must lie in [0, 1]"); return E2_EINVAL; }
    if (p->tournament < 1) { snprintf(msg, n, "tournament size must be >= 1"); return E2_EINVAL; }
    if (p->role_search < 0 || p->role_search > 2) { snprintf(msg, n, "role_search must be 0, 1 or 2"); return E2_EINVAL; }
    if (p->role_search && pf->b_max > 63) { snprintf(msg, n, "role_search 1 and 2 need b_max <= 63"); return E2_EINVAL; }
    if (p->objective != 0 && p->objective != 1) { snprintf(msg, n, "objective must be 0 or 1"); return E2_EINVAL; }
    return E2_OK;
}

DevPop pop_at(unsigned char *ws, const Layout &l, int b)
{
    return DevPop{reinterpret_cast<uint16_t *>(ws + l.perm[b]), reinterpret_cast<uint16_t *>(ws + l.sizes[b]),
                  ws + l.nclus[b], reinterpret_cast<uint64_t *>(ws + l.roles[b])};
}

int copy_pop(e2_ctx *c, const DevPop &dst, const e2_genomes *g, bool out)
{
    const size_t P = c->dm.P, M = c->dm.M, K = c->dm.K;
    if (!g || !g->perm || !g->sizes || !g->nclus || !g->roles) return fail(c, E2_EINVAL, "null genome array");
    const cudaMemcpyKind k = cudaMemcpyDefault;
    if (!out) {
        E2_CUDA(c, cudaMemcpyAsync(dst.perm, g->perm, 2 * P * M, k, c->stream));
        E2_CUDA(c, cudaMemcpyAsync(dst.sizes, g->sizes, 2 * P * K, k, c->stream));
        E2_CUDA(c, cudaMemcpyAsync(dst.nclus, g->nclus, P, k, c->stream));
        E2_CUDA(c, cudaMemcpyAsync(dst.roles, g->roles, 8 * P, k, c->stream));
    } else {
        E2_CUDA(c, cudaMemcpyAsync(g->perm, dst.perm, 2 * P * M, k, c->stream));
        E2_CUDA(c, cudaMemcpyAsync(g->sizes, dst.sizes, 2 * P * K, k, c->stream));
        E2_CUDA(c, cudaMemcpyAsync(g->nclus, dst.nclus, P, k, c->stream));
        E2_CUDA(c, cudaMemcpyAsync(g->roles, dst.roles, 8 * P, k, c->stream));
        if (is_host(g->perm) || is_host(g->sizes) || is_host(g->nclus) || is_host(g->roles))
            E2_CUDA(c, cudaStreamSynchronize(c->stream));
    }
    return E2_OK;
}

// Copy a population into the current buffer and validate it on the device
// (invalid genomes are replaced there by a valid one); the smallest invalid
// index lands in the error word, read back by check_validated.
constexpr int32_t kNoBadGenome = 0x7F7F7F7F;   // the error word's bytes all 0x7F

int upload_and_validate(e2_ctx *c, const e2_genomes *g)
{
    int st = copy_pop(c, c->pop[c->cur], g, false);
    if (st) return st;
    E2_CUDA(c, cudaMemsetAsync(c->err, 0x7F, 4, c->stream));
    E2_CUDA(c, launch_validate(c, c->pop[c->cur]));
    c->evaluated = false;
    return E2_OK;
}

int check_validated(e2_ctx *c, int32_t bad)
{
    if (bad == kNoBadGenome) return E2_OK;
    char buf[160];
    snprintf(buf, sizeof buf, "genome %d is not a valid gene (ordering, grouping or roles); replaced by the identity "
             "ordering as one replica", bad);
    return fail(c, E2_EINVAL, buf);
}

int set_and_validate(e2_ctx *c, const e2_genomes *g)
{
    int st = upload_and_validate(c, g);
    if (st) return st;
    int32_t bad = kNoBadGenome;
    E2_CUDA(c, cudaMemcpyAsync(&bad, c->err, 4, cudaMemcpyDeviceToHost, c->stream));
    E2_CUDA(c, cudaStreamSynchronize(c->stream));
    return check_validated(c, bad);
}

}  // namespace

extern "C" {

size_t e2_workspace_bytes(int32_t M, int32_t N, int32_t b_max, int32_t P, int32_t Q, int32_t K_max)
{
    return e2_workspace_bytes_ex(M, N, b_max, P, Q, K_max, 0u);
}

size_t e2_workspace_bytes_ex(int32_t M, int32_t N, int32_t b_max, int32_t P, int32_t Q, int32_t K_max,
                             uint32_t flags)
{
    if (!dims_ok(M, N, b_max, P, Q, K_max) || (flags & ~E2_WS_LAYERED)) return 0;
    const bool layered = (flags & E2_WS_LAYERED) != 0;
    if (layered && N > E2_MAX_LAYERED_BLOCKS) return 0;
    return layout(M, N, b_max, P, Q, K_max, layered).total;
}

// Whether the decode variants' costs never shrink as the batch grows: block
// and head memory (so capacities never grow), block flops and bytes (per-block
// times) and activation bytes (link times), over v = 1..b_max.  Physical
// profiles do; the evaluation pre-pass then searches its monotone tests
// instead of testing every batch.
static int costs_grow_with_batch(const e2_layer_profile *prof, int b_max)
{
    const uint64_t *rows[] = {prof->blk_mem, prof->head_mem, prof->blk_flops, prof->blk_bytes, prof->act_bytes};
    for (const uint64_t *r : rows)
        for (int v = 1; v < b_max; ++v)
            if (r[v + 1] < r[v]) return 0;
    return 1;
}

// The decode test of Alg. 2 keeps batch b when 1.0 / Lambda_b >= Min_TPS,
// the quotient rounded to nearest.  Correctly rounded division is monotone, so
// for Lambda >= 0 the test holds exactly when Lambda <= Lambda_max, the largest
// double that passes it; found here by bisection over the bit patterns of the
// non-negative doubles (which order like the values), so that the kernels
// compare instead of dividing (a float64 division costs hundreds of cycles).
static double latency_ceiling(double min_tps)
{
    auto pass = [&](uint64_t bits) {
        double x;
        memcpy(&x, &bits, sizeof x);
        return 1.0 / x >= min_tps;
    };
    const uint64_t inf_bits = 0x7FF0000000000000ull;
    if (pass(inf_bits)) return HUGE_VAL;            // min_tps <= 0: every latency passes
    uint64_t lo = 0, hi = inf_bits;                 // pass(lo) (1/0 = +inf), !pass(hi)
    while (hi - lo > 1) {
        const uint64_t mid = lo + (hi - lo) / 2;
        if (pass(mid)) lo = mid;
        else hi = mid;
    }
    double x;
    memcpy(&x, &lo, sizeof x);
    return x;
}

int e2_create(const e2_devices *devs, const e2_links *links, const e2_layer_profile *prof,
              const e2_params *prm, void *workspace, size_t workspace_bytes, void *stream, e2_ctx **out)
{
    g_create_error[0] = 0;
    auto reject = [&](int code, const char *why) {
        snprintf(g_create_error, sizeof g_create_error, "%s", why);
        return code;
    };
    if (!out) return reject(E2_EINVAL, "null output pointer");
    *out = nullptr;
    char msg[256];
    int st = validate_inputs(devs, links, prof, prm, msg, sizeof msg);
    if (st) return reject(st, msg);
    const int M = devs->M, N = prof->N, b_max = prof->b_max, P = prm->P, Q = prm->Q, K = prm->K_max;
    const bool layered = prof->PF != nullptr;
    const Layout l = layout(M, N, b_max, P, Q, K, layered);
    if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255))
        return reject(E2_EINVAL, "workspace must be non-null and 256-byte aligned");
    if (workspace_bytes < l.total) return reject(E2_ENOMEM, "workspace smaller than e2_workspace_bytes()");

    e2_ctx *c = new (std::nothrow) e2_ctx();
    if (!c) return E2_ENOMEM;
    c->stream = static_cast<cudaStream_t>(stream);
    c->dm = Dims{M, N, b_max + 1, b_max, P, Q, K, l.LS, prm->tournament, prof->NP, prof->ND,
                 prm->min_tps, prm->t_a, latency_ceiling(prm->min_tps), prm->role_search, 0.0f, 0u, 4,
                 costs_grow_with_batch(prof, b_max), prm->objective};
    c->dm.layered = layered ? 1 : 0;
    c->dm.offload = 0;
    if (devs->mem_cpu)
        for (int i = 0; i < M; ++i) c->dm.offload |= devs->mem_cpu[i] != 0;
    {
        const double lm = c->dm.lam_max;                       // rounded up to float
        float f = (float)lm;
        if ((double)f < lm) f = nextafterf(f, HUGE_VALF);
        c->dm.lam_max_up = f;
    }
    c->cong_lo = links->cong_lo;
    c->cong_hi = links->cong_hi;
    c->thr_cx = threshold(prm->p_cx);
    c->thr_half = threshold(0.5);
    c->thr_mut = threshold(prm->p_mut);
    const double s1 = prm->p_swap, s2 = s1 + prm->p_regroup, s3 = s2 + prm->p_regroup_all;
    c->thr_k1 = threshold(s1);
    c->thr_k2 = threshold(s2);
    c->thr_k3 = threshold(s3);

    auto fail_free = [&](int code, const char *why) {
        if (c->side) cudaStreamDestroy(c->side);
        if (c->ev_fork) cudaEventDestroy(c->ev_fork);
        if (c->ev_join) cudaEventDestroy(c->ev_join);
        if (c->ev_dp_fork) cudaEventDestroy(c->ev_dp_fork);
        if (c->ev_dp_join) cudaEventDestroy(c->ev_dp_join);
        delete c;
        return reject(code, why);
    };
    if (cudaGetDevice(&c->device) != cudaSuccess) return fail_free(E2_ECUDA, "no CUDA device");
    int smem_optin = 0;
    if (cudaDeviceGetAttribute(&smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, c->device) != cudaSuccess)
        return fail_free(E2_ECUDA, "cudaDeviceGetAttribute failed");
    c->dp_threads = 128;
    c->dm.g_spill = !layered && dp_spills(M, N, c->dp_threads / 32);
    c->dp_smem = layered ? dp_layered_smem_bytes(M, N) : dp_smem_bytes(M, N, c->dp_threads, 4, c->dm.g_spill);
    if ((M < N ? M : N) > kMaxReplicaDevices)
        return fail_free(E2_EINVAL, "replicas could exceed 256 devices (min(M, N) > 256)");
    if (c->dp_smem + 1024 > (size_t)smem_optin)
        return fail_free(E2_EINVAL, "the largest replica's DP does not fit in shared memory (N too large)");
    if (configure_eval(c) != cudaSuccess) return fail_free(E2_ECUDA, "configuring the DP kernel failed");
    if (cudaStreamCreateWithFlags(&c->side, cudaStreamNonBlocking) != cudaSuccess ||
        cudaEventCreateWithFlags(&c->ev_fork, cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&c->ev_join, cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&c->ev_dp_fork, cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&c->ev_dp_join, cudaEventDisableTiming) != cudaSuccess)
        return fail_free(E2_ECUDA, "creating the side stream failed");

    unsigned char *ws = static_cast<unsigned char *>(workspace);
    c->rate = reinterpret_cast<double *>(ws + l.rate);
    c->bw = reinterpret_cast<double *>(ws + l.bw);
    c->mem = reinterpret_cast<uint64_t *>(ws + l.mem);
    c->rate_cpu = reinterpret_cast<double *>(ws + l.rate_cpu);
    c->bw_cpu = reinterpret_cast<double *>(ws + l.bw_cpu);
    c->mem_cpu = reinterpret_cast<uint64_t *>(ws + l.mem_cpu);
    c->capg = reinterpret_cast<int32_t *>(ws + l.capg);
    c->gpu_layers = reinterpret_cast<int16_t *>(ws + l.gpu_layers);
    if (layered) {
        c->psum = reinterpret_cast<uint64_t *>(ws + l.psum);
        c->lcost = reinterpret_cast<double *>(ws + l.lcost);
    }
    if (c->dm.g_spill) {
        c->gspill = reinterpret_cast<uint32_t *>(ws + l.gspill);
        c->spill_stride = dp_spill_stride(M, N);
    }
    c->link_bw = reinterpret_cast<double *>(ws + l.link_bw);
    c->cong = reinterpret_cast<double *>(ws + l.cong);
    c->prof = reinterpret_cast<uint64_t *>(ws + l.prof);
    c->leaf = reinterpret_cast<double *>(ws + l.leaf);
    c->tau = reinterpret_cast<double *>(ws + l.tau);
    c->cap = reinterpret_cast<int32_t *>(ws + l.cap);
    c->cpb = reinterpret_cast<float *>(ws + l.cpb);
    c->tau_lb = reinterpret_cast<float *>(ws + l.tau_lb);
    c->leaf_sorted = reinterpret_cast<uint64_t *>(ws + l.leaf_sorted);
    c->beff_sorted = reinterpret_cast<uint64_t *>(ws + l.beff_sorted);
    c->tau_sorted = reinterpret_cast<double *>(ws + l.tau_sorted);
    c->leaf_rank = reinterpret_cast<uint32_t *>(ws + l.leaf_rank);
    c->tau_rank = reinterpret_cast<uint32_t *>(ws + l.tau_rank);
    for (int b = 0; b < 2; ++b) c->pop[b] = pop_at(ws, l, b);
    c->fit = reinterpret_cast<double *>(ws + l.fit);
    c->layers = reinterpret_cast<int16_t *>(ws + l.layers);
    c->master = reinterpret_cast<int16_t *>(ws + l.master);
    c->bsel = reinterpret_cast<int16_t *>(ws + l.bsel);
    c->T = reinterpret_cast<double *>(ws + l.T);
    c->L = reinterpret_cast<double *>(ws + l.L);
    c->hash = reinterpret_cast<uint64_t *>(ws + l.hash);
    c->dup = reinterpret_cast<int32_t *>(ws + l.dup);
    c->dup_key = reinterpret_cast<uint64_t *>(ws + l.dup_key);
    c->dup_idx = reinterpret_cast<int32_t *>(ws + l.dup_idx);
    c->elite = reinterpret_cast<int32_t *>(ws + l.elite);
    c->elite_fit = reinterpret_cast<double *>(ws + l.elite_fit);
    c->elite_ctl = reinterpret_cast<unsigned long long *>(ws + l.elite_ctl);
    c->elite_cand = reinterpret_cast<int32_t *>(ws + l.elite_cand);
    c->stats = reinterpret_cast<unsigned long long *>(ws + l.stats);
    c->err = reinterpret_cast<int32_t *>(ws + l.err);
    c->order_bins = reinterpret_cast<unsigned *>(ws + l.order_bins);
    c->items = reinterpret_cast<uint64_t *>(ws + l.items);
    c->slot_best = reinterpret_cast<int32_t *>(ws + l.slot_best);
    c->split_T = reinterpret_cast<double *>(ws + l.split_T);
    c->split_L = reinterpret_cast<double *>(ws + l.split_L);
    c->split_mu = reinterpret_cast<int16_t *>(ws + l.split_mu);
    c->split_layers = reinterpret_cast<int16_t *>(ws + l.split_layers);
    c->slot_off = reinterpret_cast<int32_t *>(ws + l.slot_off);
    c->slot_mask = reinterpret_cast<uint64_t *>(ws + l.slot_mask);
    c->slot_size = ws + l.slot_size;

    const size_t V = (size_t)b_max + 1, MM = (size_t)M * M;
    uint64_t *prof_h = new (std::nothrow) uint64_t[kNumProf * V];
    if (!prof_h) return fail_free(E2_ENOMEM, "host allocation failed");
    const uint64_t *arr[kNumProf] = {prof->blk_flops, prof->blk_bytes, prof->blk_mem, prof->head_flops,
                                     prof->head_bytes, prof->head_mem, prof->act_bytes};
    for (int a = 0; a < kNumProf; ++a) memcpy(prof_h + a * V, arr[a], 8 * V);
    cudaError_t e = cudaSuccess;
    auto chk = [&](cudaError_t x) { if (e == cudaSuccess) e = x; };
    chk(cudaMemsetAsync(ws, 0, l.total, c->stream));
    chk(cudaMemcpyAsync(c->rate, devs->rate, 8 * (size_t)M, cudaMemcpyHostToDevice, c->stream));
    chk(cudaMemcpyAsync(c->bw, devs->bw, 8 * (size_t)M, cudaMemcpyHostToDevice, c->stream));
    chk(cudaMemcpyAsync(c->mem, devs->mem, 8 * (size_t)M, cudaMemcpyHostToDevice, c->stream));
    if (c->dm.offload) {                       // otherwise the host side stays zero (no offload)
        chk(cudaMemcpyAsync(c->rate_cpu, devs->rate_cpu, 8 * (size_t)M, cudaMemcpyHostToDevice, c->stream));
        chk(cudaMemcpyAsync(c->bw_cpu, devs->bw_cpu, 8 * (size_t)M, cudaMemcpyHostToDevice, c->stream));
        chk(cudaMemcpyAsync(c->mem_cpu, devs->mem_cpu, 8 * (size_t)M, cudaMemcpyHostToDevice, c->stream));
    }
    chk(cudaMemcpyAsync(c->link_bw, links->bw, 8 * MM, cudaMemcpyHostToDevice, c->stream));
    chk(cudaMemcpyAsync(c->cong, links->cong, 8 * MM, cudaMemcpyHostToDevice, c->stream));
    chk(cudaMemcpyAsync(c->prof, prof_h, 8 * kNumProf * V, cudaMemcpyHostToDevice, c->stream));
    if (layered) {
        const size_t row = 8 * V * ((size_t)N + 1);
        chk(cudaMemcpyAsync(c->psum, prof->PF, row, cudaMemcpyHostToDevice, c->stream));
        chk(cudaMemcpyAsync(c->psum + V * ((size_t)N + 1), prof->PB, row, cudaMemcpyHostToDevice, c->stream));
        chk(cudaMemcpyAsync(c->psum + 2 * V * ((size_t)N + 1), prof->PM, row, cudaMemcpyHostToDevice, c->stream));
    }
    if (e == cudaSuccess) e = launch_tables(c);
    if (e == cudaSuccess) e = launch_tau(c);
    if (e == cudaSuccess) e = build_leaf_sorted(c);
    if (e == cudaSuccess) e = build_ranks(c);
    if (e == cudaSuccess) e = cudaStreamSynchronize(c->stream);
    delete[] prof_h;
    if (e != cudaSuccess) return fail_free(E2_ECUDA, cudaGetErrorString(e));
    *out = c;
    return E2_OK;
}

namespace {

void drop_generation_graph(e2_ctx *c, int b)
{
    if (c->gen_exec[b]) cudaGraphExecDestroy(c->gen_exec[b]);
    if (c->gen_graph[b]) cudaGraphDestroy(c->gen_graph[b]);
    c->gen_exec[b] = nullptr;
    c->gen_graph[b] = nullptr;
    c->gen_ga_node[b] = nullptr;
}

// Records the launches of one generation from population buffer b (the same
// sequence e2_eval_population and e2_ga_step issue) on the private stream.
cudaError_t record_generation(e2_ctx *c, int b)
{
    drop_generation_graph(c, b);
    cudaError_t e = cudaSuccess;
    if (!c->cap_stream) e = cudaStreamCreateWithFlags(&c->cap_stream, cudaStreamNonBlocking);
    if (e != cudaSuccess) return e;
    const cudaStream_t user = c->stream;
    const unsigned long long launched = c->launches;         // recording launches nothing
    c->stream = c->cap_stream;
    e = cudaStreamBeginCapture(c->cap_stream, cudaStreamCaptureModeThreadLocal);
    if (e == cudaSuccess) {
        cudaError_t le = cudaMemsetAsync(c->stats, 0, 8 * kNumStats, c->stream);
        if (le == cudaSuccess) le = launch_eval(c, c->pop[b]);
        if (le == cudaSuccess) le = launch_step(c, c->pop[b], c->pop[b ^ 1], 0, 0);
        cudaGraph_t g = nullptr;
        e = cudaStreamEndCapture(c->cap_stream, &g);
        if (le != cudaSuccess) e = le;
        if (e == cudaSuccess) {
            c->gen_graph[b] = g;
            e = cudaGraphInstantiate(&c->gen_exec[b], g, 0);
        } else if (g) {
            cudaGraphDestroy(g);
        }
    }
    c->stream = user;
    c->gen_kernels[b] = c->launches - launched;
    c->launches = launched;
    if (e == cudaSuccess) e = find_ga_node(c->gen_graph[b], &c->gen_ga_node[b]);
    if (e != cudaSuccess) {
        drop_generation_graph(c, b);
        cudaGetLastError();
        return e;
    }
    c->gen_ev[b][0] = c->ev_dp_start;
    c->gen_ev[b][1] = c->ev_dp_stop;
    return cudaSuccess;
}

}  // namespace

int e2_destroy(e2_ctx *c)
{
    if (!c) return E2_OK;
    cudaError_t e = cudaStreamSynchronize(c->stream);
    for (int b = 0; b < 2; ++b) drop_generation_graph(c, b);
    if (c->cap_stream) cudaStreamDestroy(c->cap_stream);
    if (c->side) cudaStreamDestroy(c->side);
    if (c->ev_fork) cudaEventDestroy(c->ev_fork);
    if (c->ev_join) cudaEventDestroy(c->ev_join);
    if (c->ev_dp_fork) cudaEventDestroy(c->ev_dp_fork);
    if (c->ev_dp_join) cudaEventDestroy(c->ev_dp_join);
    delete c;
    return e == cudaSuccess ? E2_OK : E2_ECUDA;
}

int e2_set_population(e2_ctx *c, const e2_genomes *g)
{
    if (!c) return E2_EINVAL;
    return set_and_validate(c, g);
}

int e2_get_population(e2_ctx *c, const e2_genomes *g)
{
    if (!c) return E2_EINVAL;
    return copy_pop(c, c->pop[c->cur], g, true);
}

int e2_init_population(e2_ctx *c, uint64_t seed)
{
    if (!c) return E2_EINVAL;
    E2_CUDA(c, launch_init(c, c->pop[c->cur], seed));
    c->evaluated = false;
    return E2_OK;
}

int e2_eval_population(e2_ctx *c, const e2_genomes *genomes, double *fitness_out, const e2_partitions *parts)
{
    if (!c) return E2_EINVAL;
    if (genomes) {
        int st = set_and_validate(c, genomes);
        if (st) return st;
    }
    E2_CUDA(c, cudaMemsetAsync(c->stats, 0, 8 * kNumStats, c->stream));
    E2_CUDA(c, launch_eval(c, c->pop[c->cur]));
    c->evaluated = true;
    c->have_results = true;
    return e2_get_results(c, fitness_out, parts);
}

int e2_get_results(e2_ctx *c, double *fitness_out, const e2_partitions *parts)
{
    if (!c) return E2_EINVAL;
    if (!c->have_results) return fail(c, E2_ESTATE, "no population has been evaluated");
    const size_t P = c->dm.P, M = c->dm.M, K = c->dm.K;
    bool host = false;
    auto out = [&](void *dst, const void *src, size_t bytes) -> cudaError_t {
        if (!dst) return cudaSuccess;
        host = host || is_host(dst);
        return cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDefault, c->stream);
    };
    E2_CUDA(c, out(fitness_out, c->fit, 32 * P));
    if (parts) {
        E2_CUDA(c, out(parts->layers, c->layers, 2 * P * M));
        E2_CUDA(c, out(parts->master, c->master, 2 * P * K));
        E2_CUDA(c, out(parts->bsel, c->bsel, 2 * P * K));
        E2_CUDA(c, out(parts->T, c->T, 8 * P * K));
        E2_CUDA(c, out(parts->lambda, c->L, 8 * P * K));
        // without offload every block sits in device memory: the split is the partition
        E2_CUDA(c, out(parts->gpu_layers, c->dm.offload ? c->gpu_layers : c->layers, 2 * P * M));
    }
    if (host) E2_CUDA(c, cudaStreamSynchronize(c->stream));
    return E2_OK;
}

int e2_ga_step(e2_ctx *c, uint64_t seed, uint32_t generation)
{
    if (!c) return E2_EINVAL;
    if (!c->evaluated) return fail(c, E2_ESTATE, "the current population has not been evaluated");
    E2_CUDA(c, launch_step(c, c->pop[c->cur], c->pop[c->cur ^ 1], seed, generation));
    c->cur ^= 1;
    c->evaluated = false;
    c->have_elites = true;
    return E2_OK;
}

int e2_run_generation(e2_ctx *c, uint64_t seed, uint32_t generation)
{
    if (!c) return E2_EINVAL;
    const int b = c->cur;
    if (!c->gen_eager && (!c->gen_exec[b] || c->gen_ev[b][0] != c->ev_dp_start || c->gen_ev[b][1] != c->ev_dp_stop))
        c->gen_eager = record_generation(c, b) != cudaSuccess;
    if (c->gen_eager) {                                         // the same work, launched one by one
        int st = e2_eval_population(c, nullptr, nullptr, nullptr);
        return st ? st : e2_ga_step(c, seed, generation);
    }
    E2_CUDA(c, set_ga_node(c, c->gen_exec[b], c->gen_ga_node[b], c->pop[b], c->pop[b ^ 1], seed, generation));
    E2_CUDA(c, cudaGraphLaunch(c->gen_exec[b], c->stream));
    c->launches += c->gen_kernels[b];
    c->have_results = true;
    c->cur ^= 1;
    c->evaluated = false;
    c->have_elites = true;
    return E2_OK;
}

int e2_run_generation_io(e2_ctx *c, const e2_genomes *population, uint64_t seed, uint32_t generation,
                         double *fitness_out, const e2_genomes *next_out)
{
    if (!c) return E2_EINVAL;
    if (next_out && (!next_out->perm || !next_out->sizes || !next_out->nclus || !next_out->roles))
        return fail(c, E2_EINVAL, "null genome array");
    if (population) {
        const int st = upload_and_validate(c, population);
        if (st) return st;
    }
    const int st = e2_run_generation(c, seed, generation);
    if (st) return st;
    const size_t P = c->dm.P, M = c->dm.M, K = c->dm.K;
    const DevPop &nx = c->pop[c->cur];
    const cudaMemcpyKind k = cudaMemcpyDefault;
    if (fitness_out) E2_CUDA(c, cudaMemcpyAsync(fitness_out, c->fit, 32 * P, k, c->stream));
    if (next_out) {
        E2_CUDA(c, cudaMemcpyAsync(next_out->perm, nx.perm, 2 * P * M, k, c->stream));
        E2_CUDA(c, cudaMemcpyAsync(next_out->sizes, nx.sizes, 2 * P * K, k, c->stream));
        E2_CUDA(c, cudaMemcpyAsync(next_out->nclus, nx.nclus, P, k, c->stream));
        E2_CUDA(c, cudaMemcpyAsync(next_out->roles, nx.roles, 8 * P, k, c->stream));
    }
    int32_t bad = kNoBadGenome;
    if (population) E2_CUDA(c, cudaMemcpyAsync(&bad, c->err, 4, cudaMemcpyDeviceToHost, c->stream));
    const bool host = population || (fitness_out && is_host(fitness_out)) ||
                      (next_out && (is_host(next_out->perm) || is_host(next_out->sizes) ||
                                    is_host(next_out->nclus) || is_host(next_out->roles)));
    if (host) E2_CUDA(c, cudaStreamSynchronize(c->stream));
    return check_validated(c, bad);
}

int e2_redraw_congestion(e2_ctx *c, uint64_t seed, uint32_t generation)
{
    if (!c) return E2_EINVAL;
    E2_CUDA(c, launch_redraw(c, seed, generation));
    E2_CUDA(c, launch_tau(c));
    E2_CUDA(c, build_ranks(c));
    c->evaluated = false;
    return E2_OK;
}

int e2_get_congestion(e2_ctx *c, double *cong_out)
{
    if (!c || !cong_out) return E2_EINVAL;
    E2_CUDA(c, cudaMemcpyAsync(cong_out, c->cong, 8 * (size_t)c->dm.M * c->dm.M, cudaMemcpyDefault, c->stream));
    if (is_host(cong_out)) E2_CUDA(c, cudaStreamSynchronize(c->stream));
    return E2_OK;
}

int e2_get_elites(e2_ctx *c, int32_t *idx_out, double *fitness_out)
{
    if (!c) return E2_EINVAL;
    if (!c->have_elites) return fail(c, E2_ESTATE, "no generation step has run");
    const size_t Q = c->dm.Q;
    bool host = false;
    if (idx_out && Q) {
        E2_CUDA(c, cudaMemcpyAsync(idx_out, c->elite, 4 * Q, cudaMemcpyDefault, c->stream));
        host = host || is_host(idx_out);
    }
    if (fitness_out && Q) {
        E2_CUDA(c, cudaMemcpyAsync(fitness_out, c->elite_fit, 32 * Q, cudaMemcpyDefault, c->stream));
        host = host || is_host(fitness_out);
    }
    if (host) E2_CUDA(c, cudaStreamSynchronize(c->stream));
    return E2_OK;
}

int e2_get_stats(e2_ctx *c, e2_stats *out)
{
    if (!c || !out) return E2_EINVAL;
    unsigned long long s[kNumStats];
    E2_CUDA(c, cudaMemcpyAsync(s, c->stats, sizeof s, cudaMemcpyDeviceToHost, c->stream));
    E2_CUDA(c, cudaStreamSynchronize(c->stream));
    out->genomes = s[kStGenomes];
    out->replicas = s[kStReplicas];
    out->dp_runs = s[kStDpRuns] + s[kStDpRunsSmall];   // the kernel counts each launch's runs apart
    out->dp_cells = s[kStCells];
    out->dp_probes = s[kStProbes];
    out->paper_candidates = s[kStPaper];
    out->prechecked = s[kStPrecheck];
    out->served = s[kStServed];
    out->tps_pruned = s[kStTpsPruned];
    out->dp_runs_small = s[kStDpRunsSmall];
    out->role_search_capped = s[kStRoleCapped];
    out->device_errors = s[kStDeviceErrors];
    out->dp_launches = c->dp_grid1 > 0 ? 2 : 1;
    out->dp_ctas = (uint64_t)c->dp_grid;
    out->dp_smem = c->dp_smem;
    out->dp_ctas_small = (uint64_t)c->dp_grid1;
    out->dp_smem_small = c->dp_smem1;
    out->dp_runs_per_cta_small = c->dp_grid1 > 0 ? (c->dp_warp1 ? (uint64_t)kDpWarpRuns : 1u) : 0u;
    out->launches = c->launches;
    if (out->device_errors)
        return fail(c, E2_EDEVICE, "a device-side consistency check of the last evaluation failed");
    return E2_OK;
}

int e2_set_timing_events(e2_ctx *c, void *dp_start, void *dp_stop)
{
    if (!c || (!dp_start) != (!dp_stop)) return E2_EINVAL;
    c->ev_dp_start = static_cast<cudaEvent_t>(dp_start);
    c->ev_dp_stop = static_cast<cudaEvent_t>(dp_stop);
    return E2_OK;
}

const char *e2_strerror(int s)
{
    switch (s) {
    case E2_OK: return "ok";
    case E2_EINVAL: return "invalid argument";
    case E2_ENOMEM: return "workspace too small";
    case E2_ECUDA: return "CUDA runtime error";
    case E2_EDEVICE: return "device-side check failed";
    case E2_ESTATE: return "call out of order";
    default: return "unknown status";
    }
}

const char *e2_last_error(const e2_ctx *c) { return c ? c->last_error.c_str() : g_create_error; }

}  // extern "C"
