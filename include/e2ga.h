/*
 * e2ga.h -- C ABI of the GB300 (sm_103a) batched fitness engine for the E2LLM
 * deployment search (arxiv 2606.03770).
 *
 * The library evaluates a whole genetic-algorithm population on one GPU.  A
 * genome (Sec. 3.4, App. A "Gene definition") is an ordering of the M devices
 * plus a grouping of that ordering into R <= K_max replicas, each replica
 * tagged prefill (role bit 0) or decode (role bit 1).  For every replica the
 * library runs DP_Pipe (Alg. 1, Eq. 1-2): the min-max partition of N identical
 * transformer blocks into contiguous stages on the replica's devices, in
 * genome order, with the master (the device holding the LM head and output
 * layer, Sec. 3.1) enumerated, links as pipeline stages and memory-infeasible
 * stages at +inf.  Prefill replicas use the prefill profile; decode replicas
 * take the largest batch b <= b_max whose partition exists and meets
 * 1/Lambda >= Min_TPS (Alg. 2).  The genome is scored with the bottleneck
 * phase, backlog and waiting time of Eq. 3-5.  Selection, crossover with
 * repair, mutation and elites (App. A) run on the device, driven by
 * Philox-4x32-10 streams keyed by (seed, generation, slot, purpose).
 *
 * Conventions
 *  - Every function returns an e2_status.  Nothing aborts, traps or throws.
 *  - Device work is enqueued on the stream given to e2_create and is
 *    asynchronous, except where a function says it synchronises.
 *  - Pointers marked "host or device" may point at host memory (pageable or
 *    pinned) or at device memory of the current device; the library copies
 *    with cudaMemcpyDefault.  When an OUTPUT pointer is host memory the call
 *    synchronises the stream before it returns, so the data is ready.
 *  - Device memory: the library allocates none.  The caller provides one
 *    device workspace of e2_workspace_bytes() bytes (for example a byte
 *    tensor from PyTorch's allocator), 256-byte aligned, that outlives the
 *    context.
 *  - Layouts are row-major.  Genome arrays: perm [P][M] u16, sizes [P][K_max]
 *    u16 (entries >= R are zero), nclus [P] u8, roles [P] u64 (bit c = role of
 *    replica c, no bits at or above R).
 *  - Times are seconds, rates FLOP/s or bytes/s, sizes bytes, all float64
 *    unless stated.  Integer inputs must stay below 2^53 after the library's
 *    sums (N blocks plus the head); e2_create checks this.
 */
#ifndef E2GA_H
#define E2GA_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    E2_OK = 0,
    E2_EINVAL = 1,    /* invalid argument (null pointer, size, value, genome) */
    E2_ENOMEM = 2,    /* workspace smaller than e2_workspace_bytes()          */
    E2_ECUDA = 3,     /* a CUDA runtime call failed                           */
                      /* (4 is not used: no kernel waits on the device)       */
    E2_EDEVICE = 5,   /* a device-side consistency check failed: an evaluation */
                      /* met a state its own pre-checks rule out (reported by  */
                      /* e2_get_stats; the results of that evaluation are not  */
                      /* to be trusted)                                        */
    E2_ESTATE = 6     /* call order: e.g. e2_ga_step before any evaluation    */
} e2_status;

/* Fleet (Sec. 3.1: profiled devices).  M >= 1, M <= E2_MAX_DEVICES.
 *
 * GPU-CPU offload (Sec. 1: offloading is part of the cost model; the plans'
 * G--C column, Sec. 4.3): a device with host memory mem_cpu[d] > 0 keeps as
 * many of a stage's blocks in its own memory as fit there (beside the LM head
 * and output layer on the master, which never leave it) and the rest in host
 * memory, if they fit, where they run at rate_cpu[d] and bw_cpu[d]; the two
 * parts run one after the other, so the stage time is
 *   max(g*F (+F_head)/rate, g*B (+B_head)/bw) + max(c*F/rate_cpu, c*B/bw_cpu)
 * for g blocks in device memory and c = n - g offloaded.  mem_cpu NULL (or 0
 * for a device, e.g. unified memory) means no offload there. */
typedef struct {
    int32_t M;
    const double *rate;     /* [M] compute rate, FLOP/s, finite > 0   (host)  */
    const double *bw;       /* [M] memory bandwidth, bytes/s, finite > 0      */
    const uint64_t *mem;    /* [M] memory available to the model, bytes       */
    const double *rate_cpu; /* [M] host FLOP/s for offloaded blocks, finite   */
                            /*     > 0 where mem_cpu > 0; NULL if mem_cpu is  */
    const double *bw_cpu;   /* [M] host bytes/s, likewise                     */
    const uint64_t *mem_cpu;/* [M] host memory for offloaded blocks, bytes,   */
                            /*     or NULL (no device offloads)               */
} e2_devices;

/* Links (Sec. 3.2: tau(k-1,k) = A / B(k-1,k)).  Row = sender.  The effective
 * bandwidth is bw[a][b] * cong[a][b]; bw may be +inf (a free link).  The
 * diagonal is never read. */
typedef struct {
    const double *bw;       /* [M][M] base link bandwidth, bytes/s, > 0 (host) */
    const double *cong;     /* [M][M] congestion factor, finite > 0     (host) */
    double cong_lo, cong_hi;/* range of e2_redraw_congestion's factors         */
} e2_links;

/* Layer profile of one model (Sec. 3.1, Alg. 2 inputs l_P, l_D(b)).  N
 * blocks; V = 1 + b_max variants: v = 0 prefill (one request of NP tokens),
 * v = b decode with b requests in flight.  With PF == NULL the blocks are
 * identical: the stage time of n blocks on device d is max(flops/rate_d,
 * bytes/bw_d) with flops = n*blk_flops[v] (+ head_flops[v] on the master),
 * likewise bytes; it is +inf when n*blk_mem[v] (+ head_mem[v]) exceeds mem_d.
 *
 * Blocks of several types (Sec. 3.1: blocks of one type, e.g. sliding-window
 * or full attention, share a latency): PF, PB, PM give per variant the prefix
 * sums [V][N+1] of the blocks' flops, bytes and resident bytes (PF[v][0] = 0,
 * non-decreasing).  The stage of blocks j..i then costs PF[v][i+1]-PF[v][j]
 * flops (+ the head on the master), likewise bytes and memory.  A stage's cost
 * depends on where it starts, and the best bottleneck of a prefix is no longer
 * monotone in its length, so these contexts run the plain scan over every
 * split (Alg. 1's recurrence, with the masters factored through prefix and
 * suffix tables) instead of the identical-block kernel.  Needs
 * e2_workspace_bytes_ex(..., E2_WS_LAYERED), N <= E2_MAX_LAYERED_BLOCKS, and
 * no GPU-CPU offload (mem_cpu NULL or all zero).  blk_* must still hold valid
 * values (they bound the range checks; the largest block's work is a good
 * choice). */
typedef struct {
    int32_t N;                      /* blocks, 1..E2_MAX_BLOCKS               */
    int32_t b_max;                  /* 1..E2_MAX_BATCH                        */
    const uint64_t *blk_flops;      /* [V] (host) */
    const uint64_t *blk_bytes;      /* [V] */
    const uint64_t *blk_mem;        /* [V] */
    const uint64_t *head_flops;     /* [V] LM head + output layer (master)    */
    const uint64_t *head_bytes;     /* [V] */
    const uint64_t *head_mem;       /* [V] */
    const uint64_t *act_bytes;      /* [V] activation bytes per link crossing */
    uint64_t NP;                    /* mean input tokens per request, >= 1    */
    uint64_t ND;                    /* mean generated tokens per request, >= 1*/
    const uint64_t *PF;             /* [V][N+1] prefix sums of block flops, or NULL */
    const uint64_t *PB;             /* [V][N+1] of block bytes (NULL iff PF is)     */
    const uint64_t *PM;             /* [V][N+1] of block resident bytes             */
} e2_layer_profile;

/* Search parameters (Alg. 2 inputs P, G, Q, Min_TPS; App. A mutation mix). */
typedef struct {
    int32_t P;              /* population, 1..E2_MAX_POP, with                  */
                            /* P * K_max * (b_max + 1) < 2^31                   */
    int32_t Q;              /* elites, 0..P                                     */
    int32_t K_max;          /* replicas per genome, 1..E2_MAX_CLUSTERS          */
    int32_t tournament;     /* tournament size, >= 1                            */
    double min_tps;         /* per-request tokens/s floor, >= 0 (Sec. 3.5)      */
    double t_a;             /* request inter-arrival time T_a, s, >= 0 (Eq. 4)  */
    double p_cx;            /* per-position probability of taking parent B      */
    double p_mut;           /* probability that a child mutates                 */
    double p_swap;          /* mutation kinds, App. A: swap two positions       */
    double p_regroup;       /*   regroup from a random replica onward           */
    double p_regroup_all;   /*   regroup everything; the rest: regenerate both  */
    int32_t role_search;    /* 0: each replica's role is a bit of the genome;   */
                            /* 1: Alg. 2's brute-force role assignment: every   */
                            /* replica is evaluated in both roles, the best of  */
                            /* the 2^R assignments (least objective, then       */
                            /* phase, then smallest mask) is taken and written  */
                            /* back into the genome's role bits.  Replicas      */
                            /* whose role is fixed in the winner are not        */
                            /* enumerated: one that serves neither role         */
                            /* (bit clear) and, under the waiting time, one     */
                            /* that cannot decode (it prefills).  A genome with */
                            /* more than E2_MAX_ROLE_SEARCH other replicas is   */
                            /* not searched: it keeps its own role bits for     */
                            /* them, the fixed ones clear, and is counted in    */
                            /* e2_stats.role_search_capped.  Needs b_max <= 63. */
                            /* 2: the adapted-SplitWise rule of the paper's     */
                            /* comparison (Sec. 4.2 "Baseline chosen"): both    */
                            /* roles evaluated; the n_P strongest replicas      */
                            /* (prefill throughput NP/T, ties to the lower      */
                            /* index; a replica that cannot prefill is the      */
                            /* weakest) prefill, the rest decode, with          */
                            /* n_P = R*NP/(NP+ND) rounded half up, clamped to   */
                            /* [1, R-1] (R = 1: 1); the roles are written back  */
                            /* into the genome.  Needs b_max <= 63.             */
    int32_t objective;      /* fitness[0] of a genome: 0 the waiting time w of  */
                            /* Eq. 3-5; 1 the per-request finishing time of the */
                            /* FT comparison (Sec. 2, Sec. 4.2: HexGen-2's      */
                            /* objective), FT = (sum_P PS_c Lambda_c) / PS +    */
                            /* ND (sum_D DS_c Lambda_c) / DS, the sums in       */
                            /* ascending replica order (+inf when PS or DS is   */
                            /* 0).  Either way fitness[1] is Eq. 3's phase and  */
                            /* the fitness order is (fitness[0], fitness[1],    */
                            /* index).                                          */
} e2_params;

/* A population in the layout above; "host or device" pointers. */
typedef struct {
    uint16_t *perm;
    uint16_t *sizes;
    uint8_t *nclus;
    uint64_t *roles;
} e2_genomes;

/* Per-replica results of an evaluation; "host or device" pointers, any may be
 * NULL (not returned).  Slot-aligned with the genome:
 *   layers [P][M]  blocks placed on the device at ordering position p, or -1
 *                  when its replica cannot serve;
 *   master [P][K_max]  master position inside the replica (0-based) or -1;
 *   bsel   [P][K_max]  0 prefill, b >= 1 chosen decode batch, -1 no service
 *                      (or replica index >= R);
 *   T      [P][K_max]  bottleneck stage time of the chosen variant (+inf if none);
 *   lambda [P][K_max]  per-request latency Lambda of the chosen variant (+inf);
 *   gpu_layers [P][M]  of layers[p], the blocks in the device's own memory
 *                      (the rest offloaded to host memory: the plans' G--C
 *                      split), -1 when the replica cannot serve. */
typedef struct {
    int16_t *layers;
    int16_t *master;
    int16_t *bsel;
    double *T;
    double *lambda;
    int16_t *gpu_layers;
} e2_partitions;

/* Counters of the last evaluation (device-side tallies), then host-side
 * figures of the context: its DP launch shapes and its kernel launches so
 * far. */
typedef struct {
    uint64_t genomes;           /* genomes evaluated                           */
    uint64_t replicas;          /* replicas evaluated (sum of R)                */
    uint64_t dp_runs;           /* DP_Pipe runs that reached the recurrence     */
    uint64_t dp_cells;          /* DP cells D_mu(i,k) computed                  */
    uint64_t dp_probes;         /* split-point probes made: a bisection for the
                                   first cell of each thread's span of a column,
                                   one probe for each further cell              */
    uint64_t paper_candidates;  /* (mu,k,i,j) candidates Alg. 1 would examine   */
    uint64_t prechecked;        /* variants rejected by the memory count check
                                   (over each replica's whole sweep)            */
    uint64_t served;            /* replicas that can serve                      */
    uint64_t tps_pruned;        /* decode variants a latency lower bound proved
                                   to miss Min_TPS (their DP is skipped)        */
    uint64_t dp_runs_small;     /* of dp_runs, those of the second DP launch:
                                   the small replica sizes, run with
                                   more runs in flight per SM, four warps per
                                   run or one (0 where that raises no occupancy
                                   and one launch runs them all)                */
    uint64_t dp_launches;       /* DP kernel launches per evaluation (1 or 2;
                                   fixed at e2_create)                          */
    uint64_t dp_ctas;           /* persistent CTAs of the first DP launch       */
    uint64_t dp_smem;           /* and its dynamic shared memory per CTA (B)    */
    uint64_t dp_ctas_small;     /* the same for the second launch (0: none)     */
    uint64_t dp_smem_small;     /* (per run: per warp when a warp runs one)     */
    uint64_t launches;          /* kernels this context has launched since
                                   e2_create, cumulative (a recorded generation
                                   counts its kernel nodes per replay)          */
    uint64_t role_search_capped;/* genomes of the last evaluation whose role
                                   search was not run (more than
                                   E2_MAX_ROLE_SEARCH replicas to enumerate)    */
    uint64_t device_errors;     /* consistency checks of the last evaluation
                                   that failed on the device (a DP run whose
                                   memory the pre-pass tested exactly found no
                                   partition, or a traceback found no split
                                   attaining its cell); nonzero makes
                                   e2_get_stats return E2_EDEVICE               */
    uint64_t dp_runs_per_cta_small; /* runs in flight per CTA of the second launch:
                                   1 (four warps per run) or 4 (a warp each; 0:
                                   no second launch)                            */
} e2_stats;

typedef struct e2_ctx e2_ctx;

#define E2_MAX_DEVICES 4096
#define E2_MAX_BLOCKS 1024
#define E2_MAX_BATCH 64
#define E2_MAX_CLUSTERS 64
#define E2_MAX_POP (1 << 22)
#define E2_MAX_ROLE_SEARCH 20   /* most replicas whose roles the role search enumerates */
#define E2_MAX_LAYERED_BLOCKS 180   /* most blocks of a profile with per-layer sums */
#define E2_WS_LAYERED 1u        /* e2_workspace_bytes_ex flag: per-layer profile (PF != NULL) */

/* Bytes of device workspace a context with these sizes needs.  Returns 0 on
 * invalid sizes (each within its E2_MAX_* bound, Q <= P, and
 * P * K_max * (b_max + 1) < 2^31).  Reads only M, N, b_max, P, Q, K_max. */
size_t e2_workspace_bytes(int32_t M, int32_t N, int32_t b_max, int32_t P, int32_t Q,
                          int32_t K_max);

/* The same with flags: E2_WS_LAYERED adds the per-layer stage-cost table of a
 * profile with prefix sums (V x M x 2 x N x N float64 times: 29 MB for 32
 * devices and 80 blocks, 1.2 GB for 512 devices and 126 blocks).  Returns 0
 * on invalid sizes or unknown flags (and with E2_WS_LAYERED for
 * N > E2_MAX_LAYERED_BLOCKS). */
size_t e2_workspace_bytes_ex(int32_t M, int32_t N, int32_t b_max, int32_t P, int32_t Q, int32_t K_max,
                             uint32_t flags);

/* Validate and copy the inputs (host pointers), lay out the workspace, build
 * the stage-cost and link-cost tables on the device (Sec. 3.2 cost model) and
 * return a context bound to `stream` (a cudaStream_t; NULL = legacy default)
 * and to the current device.  The caller keeps ownership of every input and
 * of the workspace.  Synchronises the stream.  Errors: E2_EINVAL for any
 * invalid value, for min(M, N) > 256 (a replica's DP holds at most 256
 * devices) or when the largest replica's DP exceeds shared memory;
 * E2_ENOMEM for a short workspace; E2_ECUDA. */
int e2_create(const e2_devices *devs, const e2_links *links, const e2_layer_profile *prof,
              const e2_params *prm, void *workspace, size_t workspace_bytes, void *stream,
              e2_ctx **out);

/* Release the context (host memory only; the workspace stays the caller's).
 * Synchronises the stream.  NULL is accepted. */
int e2_destroy(e2_ctx *ctx);

/* Copy a population (host or device pointers) into the context's current
 * population and validate it (each ordering a permutation, 1 <= R <= K_max,
 * sizes >= 1 summing to M, zero sizes beyond R, no role bits at or above R).
 * Synchronises.  E2_EINVAL names the first bad genome via e2_last_error; every
 * invalid genome is then replaced by the identity ordering as one prefill
 * replica, so that the context never holds an invalid population. */
int e2_set_population(e2_ctx *ctx, const e2_genomes *g);

/* Copy the context's current population out (host or device pointers). */
int e2_get_population(e2_ctx *ctx, const e2_genomes *g);

/* Random initial population (Alg. 2, first step) from Philox streams of
 * generation 0: Fisher-Yates orderings, a uniform replica count in
 * 1..min(K_max, M), uniform cut points, random roles. */
int e2_init_population(e2_ctx *ctx, uint64_t seed);

/* Evaluate a population: DP_Pipe per replica and variant, the decode batch
 * sweep, and the objective of Eq. 3-5.  `genomes` (host or device) replaces
 * the current population when not NULL (validated like e2_set_population);
 * NULL evaluates the current one.  fitness_out [P][4] = {w, phase, PS, DS}
 * (host or device, may be NULL; fitness[0] is the objective e2_params.objective
 * selects); `parts` may be NULL.  The results also stay in the context for
 * e2_ga_step. */
int e2_eval_population(e2_ctx *ctx, const e2_genomes *genomes, double *fitness_out,
                       const e2_partitions *parts);

/* One generation (Alg. 2 population update, App. A): elites = the Q best
 * distinct genomes of the evaluated population by (w, phase, index); slots
 * [0, Q) of the next population take them in that order, slots [Q, P) take
 * children (tournament selection, uniform crossover with repair, grouping and
 * roles from one parent, mutation), all drawn from the streams of
 * (seed, generation).  The next population becomes current.  E2_ESTATE if the
 * current population has not been evaluated. */
int e2_ga_step(e2_ctx *ctx, uint64_t seed, uint32_t generation);

/* Redraw every link's congestion factor uniformly in [cong_lo, cong_hi) from
 * the stream of (seed, generation) and rebuild the link-cost tables.  The
 * population's results are stale afterwards (E2_ESTATE for e2_ga_step until
 * the next evaluation). */
int e2_redraw_congestion(e2_ctx *ctx, uint64_t seed, uint32_t generation);

/* Copy the current congestion matrix [M][M] out (host or device pointer). */
int e2_get_congestion(e2_ctx *ctx, double *cong_out);

/* Elite indices [Q] (into the population that was evaluated before the last
 * e2_ga_step) and their fitness [Q][4]; either may be NULL. */
int e2_get_elites(e2_ctx *ctx, int32_t *idx_out, double *fitness_out);

/* Copies the results of the most recent evaluation (by e2_eval_population or
 * e2_run_generation): fitness P x 4 and, if parts is not NULL, the partitions;
 * host or device pointers, NULL ones skipped.  Synchronises when a
 * destination is host memory.  E2_ESTATE if nothing was evaluated yet. */
int e2_get_results(e2_ctx *ctx, double *fitness_out, const e2_partitions *parts);

/* One generation of Alg. 2 from the current population: its evaluation
 * (as e2_eval_population(ctx, NULL, NULL, NULL)) followed by the elites and the
 * next population (as e2_ga_step(ctx, seed, generation)), with the same
 * results.  The context records this launch sequence as a CUDA graph on first
 * use (one per population buffer, recorded on a private stream and again when
 * the timing events of e2_set_timing_events change) and afterwards replays it
 * on its stream, setting only the new seed and generation: one launch instead
 * of nine (two memsets and seven kernels).  If recording fails the calls are
 * issued one by one.
 * E2_EINVAL for a NULL context; E2_ECUDA on a CUDA failure. */
int e2_run_generation(e2_ctx *ctx, uint64_t seed, uint32_t generation);

/* One generation with the host in the loop, synchronising once (no
 * counterpart in the paper; the host-driven form of Alg. 2's loop).  If
 * `population` is not NULL it replaces the current population (host or device
 * arrays, validated on the device like e2_set_population, without a separate
 * synchronisation).  Then the work of e2_run_generation(ctx, seed,
 * generation); then, where not NULL, the evaluated population's fitness
 * [P][4] goes to fitness_out and the next population to next_out (host or
 * device).  Synchronises when `population` is given or a destination is host
 * memory.  E2_EINVAL when `population` holds an invalid genome (the smallest
 * such index in e2_last_error): the generation ran with each invalid genome
 * replaced by the identity ordering as one prefill replica, so the outputs
 * are of that population and the context stays usable.  E2_EINVAL also for a
 * NULL context or a NULL array in next_out; E2_ECUDA on a CUDA failure. */
int e2_run_generation_io(e2_ctx *ctx, const e2_genomes *population, uint64_t seed, uint32_t generation,
                         double *fitness_out, const e2_genomes *next_out);

/* Counters of the last evaluation.  Synchronises.  Fills *out and returns
 * E2_EDEVICE (with a message in e2_last_error) when device_errors is nonzero. */
int e2_get_stats(e2_ctx *ctx, e2_stats *out);

/* Timing hook (no counterpart in the paper; for measurement): two CUDA events
 * (cudaEvent_t, created with timing enabled on the context's device) that
 * every later e2_eval_population records on the context's stream immediately
 * before and after its DP_Pipe kernel, so that cudaEventElapsedTime gives that
 * kernel's duration.  NULL, NULL turns the hook off.  The caller owns the
 * events and must keep them alive while the hook is set. */
int e2_set_timing_events(e2_ctx *ctx, void *dp_start, void *dp_stop);

/* Elite selection that allocates nothing.  The paper has no counterpart: this
 * is a service of this library for callers that cannot allocate device memory
 * -- code recording a CUDA graph (allocation is not capturable), plug-ins whose
 * host framework's allocator owns all device memory, loops that must never
 * pay cudaMalloc's implicit synchronisation.  It computes what e2_ga_step's
 * elite step computes (the Q best distinct genomes of an evaluated
 * population by (w, phase, index)) without a context or workspace: its
 * scratch is a file-scope device array sized for E2_NOALLOC_MAX_POP genomes (1 MiB,
 * held by every GPU that loads the library until the process exits).
 *   pop       population [P] in the genome layout, DEVICE pointers
 *   fitness   [P][4] {w, phase, PS, DS} from e2_eval_population, DEVICE
 *   elite_idx [Q] output, DEVICE; may be NULL when Q == 0
 *   stream    cudaStream_t the work is enqueued on (asynchronous)
 * The order is e2_ga_step's: w and phase compared as their bit patterns.
 * Returns E2_EINVAL for P > E2_NOALLOC_MAX_POP, other out-of-range sizes, null or
 * host pointers, or device memory of another GPU than the current one; E2_ECUDA
 * if the scratch address cannot be obtained or a launch fails.  The first call
 * on each device (and again the first after a reset of that device, which gives
 * it a new context) looks up the scratch array's device address with that
 * device current; make that first call before any stream capture.  All calls
 * share the one scratch array and overwrite it; calls that overlap on the GPU
 * (other streams, other host threads) race and must be serialised by the
 * caller.  Cost: two O(P^2) passes over shared-memory tiles of the fitness
 * keys, one warp per genome (the same shape as e2_ga_step's elites). */
#define E2_NOALLOC_MAX_POP 65536
int e2_select_elites_noalloc(const e2_genomes *pop, const double *fitness, int32_t P, int32_t M,
                             int32_t K_max, int32_t Q, int32_t *elite_idx, void *stream);

/* Measurement hook (no counterpart in the paper): the integer issue rate of
 * the instruction mix the DP_Pipe kernel is bound by, on the current device.
 * One launch of a full-occupancy grid in which every thread runs 8
 * independent chains of `iters` steps:
 *   kind 0: unsigned 32-bit min and max (2 operations per chain and step);
 *   kind 1: 32-bit adds (2 per step);
 *   kind 2: the DP's mix -- min, max, compare, select, add (5 per step).
 * *ops_per_launch receives the operations the launch executes and *ms_out its
 * duration from CUDA events recorded on `stream` (a cudaStream_t; NULL = the
 * legacy default stream) around it; the call synchronises on the second
 * event.  Allocates no device memory.  E2_EINVAL for a kind outside 0..2,
 * iters outside 1..2^24 or null outputs; E2_ECUDA on a CUDA failure. */
int e2_probe_int_rate(int32_t kind, int32_t iters, void *stream, double *ops_per_launch, float *ms_out);

/* Text of a status code, and the context's last detailed error message.  With
 * ctx == NULL: the message of the calling thread's last failed e2_create ("" if
 * none). */
const char *e2_strerror(int status);
const char *e2_last_error(const e2_ctx *ctx);

#ifdef __cplusplus
}
#endif
#endif /* E2GA_H */
