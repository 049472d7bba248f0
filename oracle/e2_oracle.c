/*
 * e2_oracle.c -- plain, slow CPU oracle for the E2LLM deployment search
 * (arxiv 2606.03770).  TEST INFRASTRUCTURE ONLY: the test-suite, the smoke
 * check and the benchmark's CPU-baseline leg call it; the product path never
 * does.  It shares no source with the CUDA library.
 *
 * Everything is IEEE-754 binary64, round to nearest, compiled with
 * -ffp-contract=off so that no multiply-add is fused.
 *
 * What it computes, in the paper's order:
 *   stage cost l_k(j,i,m)         Sec. 3.2 (text after Eq. 2)
 *   link cost tau = A / B          Sec. 3.2 (text after Eq. 2)
 *   DP_Pipe: Eq. 1, Eq. 2, master enumeration, argmin over mu, traceback
 *                                  Alg. 1
 *   per-request latency Lambda     Sec. 3.2 (text after Alg. 1)
 *   prefill / decode evaluation    Alg. 2 (replica loop, b sweep)
 *   role assignment by brute force Alg. 2 (optional)
 *   role assignment by the adapted-SplitWise rule
 *                                  Sec. 4.2 "Baseline chosen" (optional)
 *   objective Eq. 3, 4, 5 and the multi-replica aggregation
 *                                  Sec. 3.3
 *   finishing-time objective (HexGen-2's, the FT baseline)
 *                                  Sec. 2, Sec. 4.2 (optional)
 *   GA: gene, crossover + repair, mutation mixture, elites
 *                                  Sec. 3.4, App. A
 *   Philox-4x32-10 counter-based generator
 *                                  Salmon et al., SC'11
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORC_INF (1.0 / 0.0)

/* ------------------------------------------------------------------------ */
/* Problem description (the oracle's own layout).                            */
/* ------------------------------------------------------------------------ */
typedef struct {
    int M, N, V;                 /* devices, blocks, variants = 1 + b_max     */
    const double *rate;          /* [M] FLOP/s                                */
    const double *bw;            /* [M] bytes/s                               */
    const uint64_t *mem;         /* [M] bytes                                 */
    const double *link_bw;       /* [M*M] bytes/s, row = sender               */
    const double *cong;          /* [M*M] congestion factor                   */
    const uint64_t *blk_flops, *blk_bytes, *blk_mem;      /* [V] per block    */
    const uint64_t *head_flops, *head_bytes, *head_mem;   /* [V] master extra */
    const uint64_t *act_bytes;   /* [V] activation bytes per microbatch       */
    uint64_t NP, ND;
    double min_tps, t_a;
    int role_search;             /* 0: roles from the genome; 1: Alg. 2's     */
                                 /* brute force over every role assignment;   */
                                 /* 2: adapted SplitWise (strongest prefill)  */
    int objective;               /* 0: waiting time w (Eq. 3-5); 1: per-      */
                                 /* request finishing time FT                 */
    const double *rate_cpu;      /* [M] host FLOP/s of offloaded blocks, or   */
    const double *bw_cpu;        /* [M] host bytes/s; mem_cpu [M] host bytes  */
    const uint64_t *mem_cpu;     /* for blocks; NULL: no offload anywhere     */
    const uint64_t *PF, *PB, *PM;/* [V][N+1] prefix sums of per-block flops,  */
                                 /* bytes, resident bytes (blocks of several  */
                                 /* types, Sec. 3.1); NULL: identical blocks  */
} orc_problem;

/* ------------------------------------------------------------------------ */
/* Cost model.                                                               */
/* ------------------------------------------------------------------------ */

/* Blocks of a stage of n blocks on device d that sit in the device's own
 * (GPU or unified) memory, the rest being offloaded to host memory: as many
 * as fit next to the LM head and output layer when d is the master (the head
 * itself never leaves device memory), the "G" of the plans' G--C column
 * (Sec. 4.3).  -1 when the head does not fit at all. */
int orc_gpu_blocks(const orc_problem *p, int v, int d, int n, int master)
{
    uint64_t hm = master ? p->head_mem[v] : 0;
    if (hm > p->mem[d]) return -1;
    uint64_t bm = p->blk_mem[v];
    uint64_t cap = bm ? (p->mem[d] - hm) / bm : (uint64_t)n;
    return (uint64_t)n < cap ? n : (int)cap;
}

/* l_k(j,i,m): time of n = i-j+1 identical blocks on device d, plus the LM head
 * and output layer when the device is the master (Sec. 3.1: both live on the
 * master).  A block's time is the larger of its compute time and its memory
 * streaming time; a stage that does not fit in memory costs +inf (Sec. 3.2:
 * memory-infeasible candidates take +inf).
 *
 * GPU--CPU offload (Sec. 1: offloading is a first-class part of the cost
 * model; the plans' G--C column, Sec. 4.3): the g = orc_gpu_blocks blocks in
 * device memory run at the device's rate and bandwidth, the other n - g in
 * host memory (mem_cpu) at the host's, one after the other, so their times
 * add.  Without host memory (mem_cpu NULL or 0: unified-memory devices) every
 * block must fit in device memory, as before. */
double orc_stage_cost(const orc_problem *p, int v, int d, int n, int master);

/* l_k(j,i,m) for blocks of several types (Sec. 3.1: blocks of the same type
 * share a latency, types such as sliding-window and full attention differ):
 * the stage of blocks j..j+n-1 costs the sums of its blocks' work, read off
 * the per-variant prefix sums PF, PB, PM (the head added on the master), the
 * larger of compute and streaming time, +inf beyond device memory.  Without
 * prefix sums every block is the same and only n matters. */
double orc_stage_cost_at(const orc_problem *p, int v, int d, int j, int n, int master)
{
    if (!p->PF) return orc_stage_cost(p, v, d, n, master);
    const uint64_t *pf = p->PF + (size_t)v * (p->N + 1), *pb = p->PB + (size_t)v * (p->N + 1),
                   *pm = p->PM + (size_t)v * (p->N + 1);
    uint64_t need = pm[j + n] - pm[j] + (master ? p->head_mem[v] : 0);
    if (need > p->mem[d]) return ORC_INF;
    uint64_t fl = pf[j + n] - pf[j] + (master ? p->head_flops[v] : 0);
    uint64_t by = pb[j + n] - pb[j] + (master ? p->head_bytes[v] : 0);
    double tc = (double)fl / p->rate[d];
    double tm = (double)by / p->bw[d];
    return tc >= tm ? tc : tm;
}

double orc_stage_cost(const orc_problem *p, int v, int d, int n, int master)
{
    int g = orc_gpu_blocks(p, v, d, n, master);
    if (g < 0) return ORC_INF;
    uint64_t c = (uint64_t)(n - g);                     /* offloaded blocks */
    if (c > 0) {
        uint64_t host = p->mem_cpu ? p->mem_cpu[d] : 0;
        if (c * p->blk_mem[v] > host) return ORC_INF;
    }
    uint64_t fl = (uint64_t)g * p->blk_flops[v] + (master ? p->head_flops[v] : 0);
    uint64_t by = (uint64_t)g * p->blk_bytes[v] + (master ? p->head_bytes[v] : 0);
    double tc = (double)fl / p->rate[d];
    double tm = (double)by / p->bw[d];
    double t = tc >= tm ? tc : tm;
    if (c > 0) {
        double hc = (double)(c * p->blk_flops[v]) / p->rate_cpu[d];
        double hmm = (double)(c * p->blk_bytes[v]) / p->bw_cpu[d];
        t = t + (hc >= hmm ? hc : hmm);
    }
    return t;
}

/* tau(k-1,k) = A / B(k-1,k): time to move one microbatch of activations over
 * the link, with the link's bandwidth scaled by its congestion factor. */
double orc_link_cost(const orc_problem *p, int v, int a, int b)
{
    double beff = p->link_bw[(size_t)a * p->M + b] * p->cong[(size_t)a * p->M + b];
    return (double)p->act_bytes[v] / beff;
}

static double dmax(double a, double b) { return a >= b ? a : b; }

/* ------------------------------------------------------------------------ */
/* DP_Pipe (Alg. 1).                                                         */
/* devs[0..m-1] are the cluster's devices in pipeline order o_1..o_m.        */
/* Returns 1 if a partition exists.  Outputs the bottleneck V, the master    */
/* slot mu* (0-based), and the number of blocks per device.                  */
/* cand counts the candidates (mu,k,i,j) the recurrence examines.            */
/* ------------------------------------------------------------------------ */
int orc_dp_pipe(const orc_problem *p, int v, const uint16_t *devs, int m,
                double *V_out, int *mu_out, int16_t *layers_out, uint64_t *cand)
{
    const int N = p->N;
    *V_out = ORC_INF;
    *mu_out = -1;
    for (int k = 0; k < m; ++k) layers_out[k] = -1;
    /* Every device of the replica holds at least one block (Eq. 1 with j >= k-1). */
    if (m < 1 || m > N) return 0;

    double *D = (double *)malloc(sizeof(double) * (size_t)N * m);   /* D[k][i]  */
    int *TB = (int *)malloc(sizeof(int) * (size_t)N * m);
    double *Dbest = (double *)malloc(sizeof(double) * (size_t)N * m);
    int *TBbest = (int *)malloc(sizeof(int) * (size_t)N * m);
    double best = ORC_INF;
    int mu_best = -1;
    uint64_t count = 0;

    for (int mu = 1; mu <= m; ++mu) {                    /* master enumeration */
        for (int i = 0; i < N; ++i) {                    /* Eq. 2 (k = 1)      */
            D[i] = orc_stage_cost_at(p, v, devs[0], 0, i + 1, mu == 1);
            TB[i] = -1;
            count += 1;
        }
        for (int k = 2; k <= m; ++k) {                   /* Eq. 1 (k >= 2)     */
            double tau = orc_link_cost(p, v, devs[k - 2], devs[k - 1]);
            double *Dk = D + (size_t)(k - 1) * N;
            const double *Dp = D + (size_t)(k - 2) * N;
            int *TBk = TB + (size_t)(k - 1) * N;
            for (int i = 0; i < N; ++i) {
                double bestc = ORC_INF;
                int bj = -1;
                for (int j = k - 1; j <= i; ++j) {
                    double c = dmax(dmax(Dp[j - 1], orc_stage_cost_at(p, v, devs[k - 1], j, i - j + 1, mu == k)), tau);
                    count += 1;
                    if (c < bestc) { bestc = c; bj = j; }
                }
                Dk[i] = bestc;
                TBk[i] = bj;
            }
        }
        double Vmu = D[(size_t)(m - 1) * N + (N - 1)];
        if (Vmu < best) {                                /* argmin, first wins */
            best = Vmu;
            mu_best = mu;
            memcpy(Dbest, D, sizeof(double) * (size_t)N * m);
            memcpy(TBbest, TB, sizeof(int) * (size_t)N * m);
        }
    }
    if (cand) *cand += count;
    int ok = 0;
    if (mu_best > 0 && best < ORC_INF) {
        /* Traceback: walk k = m..2 through TB, the first device takes the rest. */
        int i = N - 1;
        for (int k = m; k >= 2; --k) {
            int j = TBbest[(size_t)(k - 1) * N + i];
            layers_out[k - 1] = (int16_t)(i - j + 1);
            i = j - 1;
        }
        layers_out[0] = (int16_t)(i + 1);
        *V_out = best;
        *mu_out = mu_best - 1;
        ok = 1;
    }
    free(D); free(TB); free(Dbest); free(TBbest);
    return ok;
}

/* Lambda = sum_k l_k + sum_k tau(k-1,k), summed in pipeline order. */
double orc_latency(const orc_problem *p, int v, const uint16_t *devs, int m, int mu,
                   const int16_t *layers)
{
    double s = orc_stage_cost_at(p, v, devs[0], 0, layers[0], mu == 0);
    int j = layers[0];
    for (int k = 1; k < m; ++k) {
        s = s + orc_link_cost(p, v, devs[k - 1], devs[k]);
        s = s + orc_stage_cost_at(p, v, devs[k], j, layers[k], mu == k);
        j += layers[k];
    }
    return s;
}

/* One replica in its role (Alg. 2, replica loop).  Prefill: one DP with l_P.
 * Decode: the highest b whose DP is feasible and gives 1/Lambda >= Min_TPS.
 * Returns 1 if the replica can serve.  *b_out = 0 for prefill. */
int orc_eval_cluster(const orc_problem *p, const uint16_t *devs, int m, int decode,
                     double *T_out, double *L_out, int *mu_out, int *b_out,
                     int16_t *layers_out, uint64_t *cand)
{
    double Vv;
    int mu;
    *T_out = ORC_INF; *L_out = ORC_INF; *mu_out = -1; *b_out = -1;
    if (!decode) {
        if (orc_dp_pipe(p, 0, devs, m, &Vv, &mu, layers_out, cand)) {
            *T_out = Vv;
            *L_out = orc_latency(p, 0, devs, m, mu, layers_out);
            *mu_out = mu;
            *b_out = 0;
            return 1;
        }
        return 0;
    }
    for (int b = p->V - 1; b >= 1; --b) {
        if (orc_dp_pipe(p, b, devs, m, &Vv, &mu, layers_out, cand)) {
            double L = orc_latency(p, b, devs, m, mu, layers_out);
            if (1.0 / L >= p->min_tps) {
                *T_out = Vv; *L_out = L; *mu_out = mu; *b_out = b;
                return 1;
            }
        }
    }
    for (int k = 0; k < m; ++k) layers_out[k] = -1;
    return 0;
}

/* Objective (Sec. 3.3): PS and DS are summed over the replicas of each role
 * in ascending replica order; Eq. 3 bottleneck phase, Eq. 4 backlog, Eq. 5
 * per-request waiting time.  No prefill or no decode capacity: +inf.
 *
 * With objective 1 the first fitness entry is instead the per-request
 * finishing time that HexGen-2 minimises (Sec. 2: a sum of computation and
 * communication time; Sec. 4.2: the FT baseline keeps the planner and swaps
 * the objective).  A request spends Lambda_c, the end-to-end pass latency of
 * its prefill replica c (every stage and link time added), in prefill, and ND
 * passes of Lambda_c' on its decode replica c'.  Requests are routed in
 * proportion to the replicas' rates (PS_c = NP/T_c, DS_c = b_c/T_c), so the
 * expected finishing time is
 *     FT = (sum_P PS_c * Lambda_c) / PS + ND * ((sum_D DS_c * Lambda_c) / DS),
 * the sums in ascending replica order.  The phase of Eq. 3 stays the second
 * key. */
void orc_score(const orc_problem *p, int R, const uint64_t roles, const double *T, const double *L,
               const int16_t *bsel, double fit[4])
{
    double PS = 0.0, DS = 0.0, PL = 0.0, DL = 0.0;
    for (int c = 0; c < R; ++c) {
        if (bsel[c] < 0) continue;
        if (((roles >> c) & 1u) == 0) {
            double r = (double)p->NP / T[c];
            PS = PS + r;
            PL = PL + r * L[c];
        } else {
            double r = (double)bsel[c] / T[c];
            DS = DS + r;
            DL = DL + r * L[c];
        }
    }
    double w = ORC_INF, phase = ORC_INF;
    if (PS != 0.0 && DS != 0.0) {
        double tp = (double)p->NP / PS;
        double td = (double)p->ND / DS;
        phase = dmax(tp, td);                              /* Eq. 3 */
        if (p->objective == 1) {
            w = PL / PS + (double)p->ND * (DL / DS);       /* finishing time */
        } else {
            double x = phase - p->t_a;
            double bn = x > 0.0 ? x : 0.0;                 /* Eq. 4 */
            w = bn > 0.0 ? tp + bn : 0.0;                  /* Eq. 5 */
        }
    }
    fit[0] = w; fit[1] = phase; fit[2] = PS; fit[3] = DS;
}

/* Decode the two-chromosome gene (Sec. 3.4, App. A): the ordering chromosome
 * perm and the grouping chromosome sizes; replica c takes the next sizes[c]
 * devices of the ordering.  Evaluates every replica and scores the genome. */
void orc_eval_genome(const orc_problem *p, int K, const uint16_t *perm, const uint16_t *sizes,
                     int R, uint64_t roles, double fit[4], int16_t *layers, int16_t *master,
                     int16_t *bsel, double *T, double *L, uint64_t *cand)
{
    int off = 0;
    for (int c = 0; c < K; ++c) {
        master[c] = -1; bsel[c] = -1; T[c] = ORC_INF; L[c] = ORC_INF;
    }
    for (int c = 0; c < R; ++c) {
        int m = sizes[c];
        double Tc, Lc;
        int mu, b;
        orc_eval_cluster(p, perm + off, m, (int)((roles >> c) & 1u), &Tc, &Lc, &mu, &b,
                         layers + off, cand);
        T[c] = Tc; L[c] = Lc; master[c] = (int16_t)mu; bsel[c] = (int16_t)b;
        off += m;
    }
    orc_score(p, R, roles, T, L, bsel, fit);
}

/* Alg. 2 with its role search: every replica is evaluated in both roles
 * (the prefill DP and the decode sweep), then every role assignment (bit c =
 * 1: replica c decodes) is scored with the objective, masks in increasing
 * order; the first with the least (objective, phase) wins.  The replicas'
 * outputs are those of their chosen roles, and the chosen assignment goes to
 * *roles_out.  This is the plain enumeration over all 2^R masks; the search
 * the library runs (orc_eval_genome_roles) is pinned against it. */
void orc_eval_genome_roles_full(const orc_problem *p, int K, const uint16_t *perm, const uint16_t *sizes,
                                int R, double fit[4], int16_t *layers, int16_t *master, int16_t *bsel,
                                double *T, double *L, uint64_t *cand, uint64_t *roles_out)
{
    double Tr[2][64], Lr[2][64];
    int mur[2][64], br[2][64];
    int16_t *lay[2];
    lay[0] = (int16_t *)malloc(sizeof(int16_t) * (size_t)p->M);
    lay[1] = (int16_t *)malloc(sizeof(int16_t) * (size_t)p->M);
    int off = 0;
    for (int c = 0; c < K; ++c) {
        master[c] = -1; bsel[c] = -1; T[c] = ORC_INF; L[c] = ORC_INF;
    }
    for (int c = 0; c < R; ++c) {
        for (int role = 0; role < 2; ++role)
            orc_eval_cluster(p, perm + off, sizes[c], role, &Tr[role][c], &Lr[role][c], &mur[role][c],
                             &br[role][c], lay[role] + off, cand);
        off += sizes[c];
    }
    uint64_t best = 0;
    double bw = ORC_INF, bp = ORC_INF;
    int have = 0;
    for (uint64_t mask = 0; mask < ((uint64_t)1 << R); ++mask) {
        double Tm[64], Lm[64], f[4];
        int16_t bm[64];
        for (int c = 0; c < R; ++c) {
            const int role = (int)((mask >> c) & 1u);
            Tm[c] = Tr[role][c];
            Lm[c] = Lr[role][c];
            bm[c] = (int16_t)br[role][c];
        }
        orc_score(p, R, mask, Tm, Lm, bm, f);
        if (!have || f[0] < bw || (f[0] == bw && f[1] < bp)) {
            have = 1; bw = f[0]; bp = f[1]; best = mask;
        }
    }
    off = 0;
    for (int c = 0; c < R; ++c) {
        const int role = (int)((best >> c) & 1u);
        T[c] = Tr[role][c]; L[c] = Lr[role][c]; master[c] = (int16_t)mur[role][c]; bsel[c] = (int16_t)br[role][c];
        for (int k = 0; k < sizes[c]; ++k) layers[off + k] = lay[role][off + k];
        off += sizes[c];
    }
    orc_score(p, R, best, T, L, bsel, fit);
    *roles_out = best;
    free(lay[0]);
    free(lay[1]);
}

/* Most replicas that can decode whose roles orc_eval_genome_roles enumerates. */
#define ORC_MAX_FREE_ROLES 20

/* Alg. 2's role search as the library runs it, for up to 64 replicas.  Some
 * replicas' roles are fixed in the winning assignment:
 *  * a replica that serves neither role adds nothing in either, so its bit is
 *    clear (the smaller mask wins the tie);
 *  * under the waiting time (objective 0), a replica that cannot decode
 *    prefills: clearing its decode bit leaves DS as it is and adds its
 *    prefill rate (if any) to PS at its place in the ascending-order sum,
 *    which can only raise PS (round-to-nearest addition is monotone), so w
 *    and the phase do not grow, and the mask gets smaller.  (Under the
 *    finishing time a slow prefill replica can raise the rate-weighted mean
 *    latency, so there only the first rule applies.)
 * So only the F other replicas are enumerated: the 2^F assignments of their
 * roles, in increasing order of their masks (the order of the full masks),
 * the first with the least (objective, phase) winning; each is scored as the
 * full mask with the fixed replicas' bits clear, exactly as the plain
 * enumeration scores it.  With more than ORC_MAX_FREE_ROLES such replicas the
 * search is not run: the genome keeps its own role bits for them (the fixed
 * ones clear), and *capped is set. */
void orc_eval_genome_roles(const orc_problem *p, int K, const uint16_t *perm, const uint16_t *sizes,
                           int R, uint64_t roles_in, double fit[4], int16_t *layers, int16_t *master,
                           int16_t *bsel, double *T, double *L, uint64_t *cand, uint64_t *roles_out, int *capped)
{
    double Tr[2][64], Lr[2][64];
    int mur[2][64], br[2][64];
    int dok[64], pok[64];
    int16_t *lay[2];
    lay[0] = (int16_t *)malloc(sizeof(int16_t) * (size_t)p->M);
    lay[1] = (int16_t *)malloc(sizeof(int16_t) * (size_t)p->M);
    int off = 0;
    for (int c = 0; c < K; ++c) {
        master[c] = -1; bsel[c] = -1; T[c] = ORC_INF; L[c] = ORC_INF;
    }
    for (int c = 0; c < R; ++c) {
        pok[c] = orc_eval_cluster(p, perm + off, sizes[c], 0, &Tr[0][c], &Lr[0][c], &mur[0][c], &br[0][c],
                                  lay[0] + off, cand);
        dok[c] = orc_eval_cluster(p, perm + off, sizes[c], 1, &Tr[1][c], &Lr[1][c], &mur[1][c], &br[1][c],
                                  lay[1] + off, cand);
        off += sizes[c];
    }
    int free_idx[64], F = 0;
    uint64_t free_mask = 0;
    for (int c = 0; c < R; ++c)
        if (dok[c] || (p->objective == 1 && pok[c])) { free_idx[F++] = c; free_mask |= (uint64_t)1 << c; }
    uint64_t best = roles_in & free_mask;
    *capped = F > ORC_MAX_FREE_ROLES;
    if (!*capped) {
        double bw = ORC_INF, bp = ORC_INF;
        int have = 0;
        for (uint64_t sub = 0; sub < ((uint64_t)1 << F); ++sub) {
            uint64_t mask = 0;
            for (int j = 0; j < F; ++j)
                if ((sub >> j) & 1u) mask |= (uint64_t)1 << free_idx[j];
            double Tm[64], Lm[64], f[4];
            int16_t bm[64];
            for (int c = 0; c < R; ++c) {
                const int role = (int)((mask >> c) & 1u);
                Tm[c] = Tr[role][c];
                Lm[c] = Lr[role][c];
                bm[c] = (int16_t)br[role][c];
            }
            orc_score(p, R, mask, Tm, Lm, bm, f);
            if (!have || f[0] < bw || (f[0] == bw && f[1] < bp)) {
                have = 1; bw = f[0]; bp = f[1]; best = mask;
            }
        }
    }
    off = 0;
    for (int c = 0; c < R; ++c) {
        const int role = (int)((best >> c) & 1u);
        T[c] = Tr[role][c]; L[c] = Lr[role][c]; master[c] = (int16_t)mur[role][c]; bsel[c] = (int16_t)br[role][c];
        for (int k = 0; k < sizes[c]; ++k) layers[off + k] = lay[role][off + k];
        off += sizes[c];
    }
    orc_score(p, R, best, T, L, bsel, fit);
    *roles_out = best;
    free(lay[0]);
    free(lay[1]);
}

/* Number of prefill replicas of the adapted-SplitWise rule: SplitWise sizes
 * each phase's pool by the input-to-generated token ratio, so R replicas split
 * as NP : ND, rounded half up, with at least one replica in each role (one
 * replica: prefill). */
int orc_splitwise_prefill_count(uint64_t NP, uint64_t ND, int R)
{
    if (R <= 1) return R;
    uint64_t den = NP + ND;
    int n = (int)((2 * (uint64_t)R * NP + den) / (2 * den));
    if (n < 1) n = 1;
    if (n > R - 1) n = R - 1;
    return n;
}

/* Adapted SplitWise (Sec. 4.2, "Baseline chosen"): every replica is
 * evaluated in both roles; within the genome the strongest replicas take the
 * prefill role and the rest decode.  A replica's strength is its prefill
 * throughput NP/T from its prefill partition (the quantity that exists only
 * after partitioning, Sec. 2); a replica that cannot serve prefill is the
 * weakest.  Ties go to the lower replica index.  The prefill count is
 * orc_splitwise_prefill_count.  The chosen roles are written to *roles_out. */
void orc_eval_genome_splitwise(const orc_problem *p, int K, const uint16_t *perm, const uint16_t *sizes,
                               int R, double fit[4], int16_t *layers, int16_t *master, int16_t *bsel,
                               double *T, double *L, uint64_t *cand, uint64_t *roles_out)
{
    double Tr[2][64], Lr[2][64];
    int mur[2][64], br[2][64];
    int ok[2][64];
    int16_t *lay[2];
    lay[0] = (int16_t *)malloc(sizeof(int16_t) * (size_t)p->M);
    lay[1] = (int16_t *)malloc(sizeof(int16_t) * (size_t)p->M);
    int off = 0;
    for (int c = 0; c < K; ++c) {
        master[c] = -1; bsel[c] = -1; T[c] = ORC_INF; L[c] = ORC_INF;
    }
    for (int c = 0; c < R; ++c) {
        for (int role = 0; role < 2; ++role)
            ok[role][c] = orc_eval_cluster(p, perm + off, sizes[c], role, &Tr[role][c], &Lr[role][c],
                                           &mur[role][c], &br[role][c], lay[role] + off, cand);
        off += sizes[c];
    }
    const int nP = orc_splitwise_prefill_count(p->NP, p->ND, R);
    uint64_t roles = 0;
    for (int c = 0; c < R; ++c) {
        double sc = ok[0][c] ? (double)p->NP / Tr[0][c] : -1.0;
        int rank = 0;                          /* replicas stronger than c, ties to the lower index */
        for (int o = 0; o < R; ++o) {
            if (o == c) continue;
            double so = ok[0][o] ? (double)p->NP / Tr[0][o] : -1.0;
            if (so > sc || (so == sc && o < c)) ++rank;
        }
        if (rank >= nP) roles |= (uint64_t)1 << c;
    }
    off = 0;
    for (int c = 0; c < R; ++c) {
        const int role = (int)((roles >> c) & 1u);
        T[c] = Tr[role][c]; L[c] = Lr[role][c]; master[c] = (int16_t)mur[role][c]; bsel[c] = (int16_t)br[role][c];
        for (int k = 0; k < sizes[c]; ++k) layers[off + k] = lay[role][off + k];
        off += sizes[c];
    }
    orc_score(p, R, roles, T, L, bsel, fit);
    *roles_out = roles;
    free(lay[0]);
    free(lay[1]);
}

/* role_search 3 is the plain 2^R enumeration (test use only: the pin of the
 * search).  capped_out, if not NULL, receives the genomes whose search was not
 * run (more than ORC_MAX_FREE_ROLES replicas can decode). */
void orc_eval_population(const orc_problem *p, int P, int K, const uint16_t *perm,
                         const uint16_t *sizes, const uint8_t *nclus, const uint64_t *roles,
                         double *fitness, int16_t *layers, int16_t *master, int16_t *bsel,
                         double *T, double *L, uint64_t *cand, int nthreads, uint64_t *roles_out,
                         uint64_t *capped_out)
{
    uint64_t total = 0, capped_total = 0;
    const int M = p->M;
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1) num_threads(nthreads > 0 ? nthreads : 1) reduction(+ : total, capped_total)
#endif
    for (int g = 0; g < P; ++g) {
        uint64_t c = 0;
        int capped = 0;
        if (p->role_search == 3)
            orc_eval_genome_roles_full(p, K, perm + (size_t)g * M, sizes + (size_t)g * K, nclus[g],
                                       fitness + (size_t)g * 4, layers + (size_t)g * M, master + (size_t)g * K,
                                       bsel + (size_t)g * K, T + (size_t)g * K, L + (size_t)g * K, &c,
                                       roles_out + g);
        else if (p->role_search == 2)
            orc_eval_genome_splitwise(p, K, perm + (size_t)g * M, sizes + (size_t)g * K, nclus[g],
                                      fitness + (size_t)g * 4, layers + (size_t)g * M, master + (size_t)g * K,
                                      bsel + (size_t)g * K, T + (size_t)g * K, L + (size_t)g * K, &c,
                                      roles_out + g);
        else if (p->role_search)
            orc_eval_genome_roles(p, K, perm + (size_t)g * M, sizes + (size_t)g * K, nclus[g], roles[g],
                                  fitness + (size_t)g * 4, layers + (size_t)g * M, master + (size_t)g * K,
                                  bsel + (size_t)g * K, T + (size_t)g * K, L + (size_t)g * K, &c,
                                  roles_out + g, &capped);
        else {
            orc_eval_genome(p, K, perm + (size_t)g * M, sizes + (size_t)g * K, nclus[g], roles[g],
                            fitness + (size_t)g * 4, layers + (size_t)g * M, master + (size_t)g * K,
                            bsel + (size_t)g * K, T + (size_t)g * K, L + (size_t)g * K, &c);
            roles_out[g] = roles[g];
        }
        total += c;
        capped_total += (uint64_t)capped;
    }
    (void)nthreads;
    if (cand) *cand = total;
    if (capped_out) *capped_out = capped_total;
}

/* ------------------------------------------------------------------------ */
/* Philox-4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11, "Parallel random       */
/* numbers: as easy as 1, 2, 3").  Round: two 32x32->64 products of counter  */
/* words 0 and 2 with the round multipliers, the high halves xored with the  */
/* other counter words and the key; the key is bumped by the Weyl constants  */
/* between rounds.                                                            */
/* ------------------------------------------------------------------------ */
void orc_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4])
{
    uint32_t c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3];
    uint32_t k0 = key[0], k1 = key[1];
    for (int r = 0; r < 10; ++r) {
        if (r > 0) { k0 += 0x9E3779B9u; k1 += 0xBB67AE85u; }
        uint64_t p0 = (uint64_t)0xD2511F53u * c0;
        uint64_t p1 = (uint64_t)0xCD9E8D57u * c2;
        uint32_t n0 = (uint32_t)(p1 >> 32) ^ c1 ^ k0;
        uint32_t n1 = (uint32_t)p1;
        uint32_t n2 = (uint32_t)(p0 >> 32) ^ c3 ^ k1;
        uint32_t n3 = (uint32_t)p0;
        c0 = n0; c1 = n1; c2 = n2; c3 = n3;
    }
    out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

/* Word t of the stream (seed, generation, slot, purpose): counter =
 * (t / 4, slot, generation, purpose), key = (seed low, seed high). */
uint32_t orc_word(uint64_t seed, uint32_t gen, uint32_t slot, uint32_t purpose, uint32_t t)
{
    uint32_t ctr[4] = {t >> 2, slot, gen, purpose};
    uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
    uint32_t out[4];
    orc_philox4x32_10(ctr, key, out);
    return out[t & 3u];
}

/* Integer in [0, n) from one word: multiply-shift (Lemire) without rejection. */
static uint32_t below(uint32_t x, uint32_t n) { return (uint32_t)(((uint64_t)x * n) >> 32); }

/* Probability p as a threshold on a 32-bit word: event iff word < thr. */
uint64_t orc_threshold(double p)
{
    if (!(p > 0.0)) return 0;
    if (p >= 1.0) return 4294967296ull;
    return (uint64_t)floor(p * 4294967296.0);
}

enum {
    ORC_INIT_PERM = 0, ORC_INIT_GROUP = 1, ORC_INIT_ROLES = 2, ORC_SELECT = 3, ORC_CROSS = 4,
    ORC_MUTATE = 5, ORC_MUT_PERM = 6, ORC_MUT_GROUP = 7, ORC_MUT_ROLES = 8, ORC_CONG = 9
};

typedef struct {
    int P, M, K, Q, tournament;
    double p_cx, p_mut, p_swap, p_regroup, p_regroup_all;
} orc_ga;

/* Fisher-Yates shuffle of the identity ordering. */
static void orc_random_perm(uint64_t seed, uint32_t gen, uint32_t slot, uint32_t purpose, int M,
                            uint16_t *perm)
{
    for (int i = 0; i < M; ++i) perm[i] = (uint16_t)i;
    for (int t = M - 1; t >= 1; --t) {
        uint32_t j = below(orc_word(seed, gen, slot, purpose, (uint32_t)(M - 1 - t)), (uint32_t)t + 1);
        uint16_t x = perm[t]; perm[t] = perm[j]; perm[j] = x;
    }
}

/* New grouping of Mr devices into 1..min(Kr, Mr) replicas: the replica count
 * is uniform, the cut points a uniform subset drawn by sequential selection
 * sampling (each candidate cut taken with probability needed/remaining).
 * Writes the sizes and returns the replica count.  Role bits come from the
 * roles stream, one bit per replica. */
static int orc_random_grouping(uint64_t seed, uint32_t gen, uint32_t slot, uint32_t pgroup,
                               uint32_t proles, int Mr, int Kr, uint16_t *sizes_out,
                               uint64_t *roles_out)
{
    int cap = Kr < Mr ? Kr : Mr;
    int R = 1 + (int)below(orc_word(seed, gen, slot, pgroup, 0), (uint32_t)cap);
    int need = R - 1, prev = 0, c = 0;
    for (int t = 1; t <= Mr - 1 && need > 0; ++t) {
        if (below(orc_word(seed, gen, slot, pgroup, (uint32_t)t), (uint32_t)(Mr - t)) < (uint32_t)need) {
            sizes_out[c++] = (uint16_t)(t - prev);
            prev = t;
            --need;
        }
    }
    sizes_out[c++] = (uint16_t)(Mr - prev);
    uint64_t bits = (uint64_t)orc_word(seed, gen, slot, proles, 0) |
                    ((uint64_t)orc_word(seed, gen, slot, proles, 1) << 32);
    *roles_out = R >= 64 ? bits : (bits & ((1ull << R) - 1));
    return R;
}

void orc_init_population(const orc_ga *ga, uint64_t seed, uint16_t *perm, uint16_t *sizes,
                         uint8_t *nclus, uint64_t *roles)
{
    for (int s = 0; s < ga->P; ++s) {
        uint16_t *pp = perm + (size_t)s * ga->M;
        uint16_t *ss = sizes + (size_t)s * ga->K;
        orc_random_perm(seed, 0, (uint32_t)s, ORC_INIT_PERM, ga->M, pp);
        memset(ss, 0, sizeof(uint16_t) * ga->K);
        nclus[s] = (uint8_t)orc_random_grouping(seed, 0, (uint32_t)s, ORC_INIT_GROUP, ORC_INIT_ROLES,
                                                ga->M, ga->K, ss, &roles[s]);
    }
}

/* Fitness order: lower waiting time, then lower bottleneck phase, then lower index. */
static int key_less(const double *fit, int a, int b)
{
    double wa = fit[(size_t)a * 4], wb = fit[(size_t)b * 4];
    if (wa != wb) return wa < wb;
    double pa = fit[(size_t)a * 4 + 1], pb = fit[(size_t)b * 4 + 1];
    if (pa != pb) return pa < pb;
    return a < b;
}

static int genome_equal(const orc_ga *ga, const uint16_t *perm, const uint16_t *sizes,
                        const uint8_t *nclus, const uint64_t *roles, int a, int b)
{
    if (nclus[a] != nclus[b] || roles[a] != roles[b]) return 0;
    if (memcmp(perm + (size_t)a * ga->M, perm + (size_t)b * ga->M, sizeof(uint16_t) * ga->M)) return 0;
    if (memcmp(sizes + (size_t)a * ga->K, sizes + (size_t)b * ga->K, sizeof(uint16_t) * ga->K)) return 0;
    return 1;
}

/* Elite citizens (App. A): the Q best distinct genomes of the evaluated
 * population, which already carries the previous elites in its first Q
 * slots.  A genome equal to a lower-indexed one is a duplicate; duplicates
 * rank after every distinct genome.  Order: (duplicate, fitness key). */
void orc_elites(const orc_ga *ga, const uint16_t *perm, const uint16_t *sizes, const uint8_t *nclus,
                const uint64_t *roles, const double *fit, int32_t *elite_idx)
{
    const int P = ga->P;
    int *dup = (int *)calloc((size_t)P, sizeof(int));
    int *order = (int *)malloc(sizeof(int) * (size_t)P);
    for (int g = 0; g < P; ++g) {
        for (int h = 0; h < g; ++h)
            if (genome_equal(ga, perm, sizes, nclus, roles, h, g)) { dup[g] = 1; break; }
        order[g] = g;
    }
    /* insertion sort by (dup, key) -- plain and stable */
    for (int a = 1; a < P; ++a) {
        int x = order[a], b = a - 1;
        while (b >= 0) {
            int y = order[b];
            int before = dup[x] != dup[y] ? dup[x] < dup[y] : key_less(fit, x, y);
            if (!before) break;
            order[b + 1] = y;
            --b;
        }
        order[b + 1] = x;
    }
    for (int q = 0; q < ga->Q; ++q) elite_idx[q] = order[q];
    free(dup); free(order);
}

/* Repair after crossover (App. A): scanning positions in order, a device met
 * a second time leaves a hole; the holes, in position order, take the devices
 * that are missing, in ascending order.  seen is scratch of M bytes. */
void orc_repair(uint16_t *cp, int M, unsigned char *seen)
{
    memset(seen, 0, (size_t)M);
    for (int i = 0; i < M; ++i) {
        if (seen[cp[i]]) cp[i] = 0xFFFFu;
        else seen[cp[i]] = 1;
    }
    int miss = 0;
    for (int i = 0; i < M; ++i) {
        if (cp[i] != 0xFFFFu) continue;
        while (seen[miss]) ++miss;
        cp[i] = (uint16_t)miss;
        seen[miss] = 1;
    }
}

/* One generation (Alg. 2, population update; App. A): slots [0,Q) take the
 * elites, every other slot a child of two tournament winners.  Ordering
 * chromosome: uniform crossover, then repair (a repeated device leaves a hole;
 * holes are filled in position order with the missing devices in ascending
 * order).  Grouping chromosome and roles: taken whole from one parent.
 * Mutation (probability p_mut): swap two positions, regroup from a random
 * replica onward, regroup everything, or regenerate both chromosomes. */
void orc_ga_step(const orc_ga *ga, uint64_t seed, uint32_t gen, const uint16_t *perm,
                 const uint16_t *sizes, const uint8_t *nclus, const uint64_t *roles,
                 const double *fit, const int32_t *elite_idx, uint16_t *nperm, uint16_t *nsizes,
                 uint8_t *nclus_out, uint64_t *nroles)
{
    const int P = ga->P, M = ga->M, K = ga->K;
    const uint64_t thr_cx = orc_threshold(ga->p_cx), thr_half = orc_threshold(0.5);
    const uint64_t thr_mut = orc_threshold(ga->p_mut);
    const double s1 = ga->p_swap, s2 = s1 + ga->p_regroup, s3 = s2 + ga->p_regroup_all;
    const uint64_t t1 = orc_threshold(s1), t2 = orc_threshold(s2), t3 = orc_threshold(s3);
    unsigned char *seen = (unsigned char *)malloc((size_t)M);
    for (int s = 0; s < P; ++s) {
        uint16_t *cp = nperm + (size_t)s * M;
        uint16_t *cs = nsizes + (size_t)s * K;
        if (s < ga->Q) {
            int e = elite_idx[s];
            memcpy(cp, perm + (size_t)e * M, sizeof(uint16_t) * M);
            memcpy(cs, sizes + (size_t)e * K, sizeof(uint16_t) * K);
            nclus_out[s] = nclus[e];
            nroles[s] = roles[e];
            continue;
        }
        int par[2];
        for (int q = 0; q < 2; ++q) {                 /* tournament selection */
            int best = (int)below(orc_word(seed, gen, (uint32_t)s, ORC_SELECT, (uint32_t)(q * ga->tournament)), (uint32_t)P);
            for (int t = 1; t < ga->tournament; ++t) {
                int c = (int)below(orc_word(seed, gen, (uint32_t)s, ORC_SELECT, (uint32_t)(q * ga->tournament + t)), (uint32_t)P);
                if (key_less(fit, c, best)) best = c;
            }
            par[q] = best;
        }
        const uint16_t *pa = perm + (size_t)par[0] * M, *pb = perm + (size_t)par[1] * M;
        for (int i = 0; i < M; ++i)                   /* uniform crossover */
            cp[i] = (uint64_t)orc_word(seed, gen, (uint32_t)s, ORC_CROSS, (uint32_t)i) < thr_cx ? pb[i] : pa[i];
        orc_repair(cp, M, seen);
        int src = (uint64_t)orc_word(seed, gen, (uint32_t)s, ORC_CROSS, (uint32_t)M) < thr_half ? par[1] : par[0];
        memcpy(cs, sizes + (size_t)src * K, sizeof(uint16_t) * K);
        int R = nclus[src];
        uint64_t rl = roles[src];

        if ((uint64_t)orc_word(seed, gen, (uint32_t)s, ORC_MUTATE, 0) < thr_mut) {
            uint64_t kind = orc_word(seed, gen, (uint32_t)s, ORC_MUTATE, 1);
            if (kind < t1) {                          /* swap two positions */
                uint32_t x = below(orc_word(seed, gen, (uint32_t)s, ORC_MUTATE, 2), (uint32_t)M);
                uint32_t y = below(orc_word(seed, gen, (uint32_t)s, ORC_MUTATE, 3), (uint32_t)M);
                uint16_t tmp = cp[x]; cp[x] = cp[y]; cp[y] = tmp;
            } else {
                int r = 0;
                if (kind < t2)                        /* regroup from a random replica */
                    r = (int)below(orc_word(seed, gen, (uint32_t)s, ORC_MUTATE, 2), (uint32_t)R);
                else if (kind >= t3)                  /* regenerate both chromosomes */
                    orc_random_perm(seed, gen, (uint32_t)s, ORC_MUT_PERM, M, cp);
                int kept = 0;
                for (int c = 0; c < r; ++c) kept += cs[c];
                for (int c = r; c < K; ++c) cs[c] = 0;
                uint64_t nr;
                int Rn = orc_random_grouping(seed, gen, (uint32_t)s, ORC_MUT_GROUP, ORC_MUT_ROLES,
                                             M - kept, K - r, cs + r, &nr);
                uint64_t keep_mask = r >= 64 ? ~0ull : ((1ull << r) - 1);
                rl = (rl & keep_mask) | (r >= 64 ? 0 : (nr << r));
                R = r + Rn;
            }
        }
        nclus_out[s] = (uint8_t)R;
        nroles[s] = rl;
    }
    free(seen);
}

/* Congestion redraw: each unordered pair (a<b) gets a factor lo + (hi-lo) u,
 * u a 53-bit uniform in [0,1) from two words of the stream (seed, generation,
 * 0, CONG), word pair 2 (a M + b). */
void orc_redraw_congestion(int M, uint64_t seed, uint32_t gen, double lo, double hi, double *cong)
{
    for (int a = 0; a < M; ++a) {
        cong[(size_t)a * M + a] = 1.0;
        for (int b = a + 1; b < M; ++b) {
            uint32_t idx = (uint32_t)(a * M + b);
            uint32_t w0 = orc_word(seed, gen, 0, ORC_CONG, 2 * idx);
            uint32_t w1 = orc_word(seed, gen, 0, ORC_CONG, 2 * idx + 1);
            uint64_t u53 = ((uint64_t)(w0 >> 5) << 26) | (uint64_t)(w1 >> 6);
            double u = (double)u53 * (1.0 / 9007199254740992.0);
            double span = hi - lo;
            double t = span * u;
            double f = lo + t;
            cong[(size_t)a * M + b] = f;
            cong[(size_t)b * M + a] = f;
        }
    }
}

int orc_num_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
