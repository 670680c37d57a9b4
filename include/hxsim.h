/*
 * hxsim.h -- C ABI of the batched HexGen-Flow scheduler simulation on GB300.
 *
 * HexGen-Flow (arXiv 2505.05286) tunes its dispatcher weight alpha by
 * replaying a recent request trace through a simulator of its own two-level
 * scheduler and keeping the point with the lowest simulated P95 latency
 * (Sec. 4.3, Eq. alpha* = argmin T_0.95(alpha)).  This library runs that
 * simulation for many (hyper-parameter point x trace) pairs at once on one
 * GPU: one warp simulates one pair, event by event, and a final kernel picks
 * the best point.
 *
 * What one simulation computes (all times int64 microseconds; alpha, gamma
 * and the SLO multiplier fixed point with HX_SCALE = 1e6; every division
 * truncates toward zero):
 *  - the workflow of Sec. 2.1 / Sec. 3.3: a query issues schema linking (S),
 *    then k candidate generations (G_c) in parallel, each followed by its
 *    self-correction calls C_{c,1..r_c}, then evaluation (E) once every
 *    chain has finished; a call is dispatched the moment it is released;
 *  - Eq. (comp): t_comp = ceil(prompt * 1e6 / prefill_tok_s)
 *    + out_est * decode_us_tok on the instance's type (true `out` gives the
 *    service time);
 *  - the dispatch score of Eq. (score), in fixed point:
 *    S_m = (SCALE - A) * min(beta / max(t_queue_m, 1), 2^43 - 1) - A * t_comp_m,
 *    t_queue_m = sum of t_comp over the requests dispatched to m and not yet
 *    finished; the highest score wins, ties to the lowest instance index;
 *  - the SLO budget of Sec. 4.2 at dispatch:
 *    t_slo = (T_slo - elapsed) * tbar / (tbar + rest of this request's path),
 *    tbar = mean of t_comp over instances, the rest = stage reference costs
 *    of G, min(rho, R - u) corrections and E as applicable;
 *  - Eq. (priority) with ageing weight gamma: U = t_comp - t_slo + gamma*tau;
 *    at each batch boundary an instance starts its highest-U waiting request
 *    (ties to the lowest request id); alternatively FCFS, or LLF (the
 *    query's laxity: deadline - now - the same remaining-path cost);
 *  - events in the order (time, completions before arrivals, instance,
 *    request id / query id);
 *  - per simulation the nearest-rank P95 of query latencies
 *    (sorted L[ceil(0.95 n) - 1]), the number of queries with latency <= T_slo,
 *    T_slo = slo_mult * (S + slowest chain + E on the reference type);
 *  - Sec. 5's further settings: several tenants, each with its own SLO
 *    multiplier (the multi-tenant evaluation); single-shot requests, a query
 *    of one E call with k = 0 (the competing workloads), released on
 *    arrival, whose budget denominator is its own tbar; and instances that
 *    become slow or unavailable for a while, handled by timeout and re-issue
 *    (Sec. 3.3): an attempt that starts on an instance inside one of its
 *    fault windows runs slow_fp / SCALE times longer (rounded up; 0 = never
 *    finishes), and with a timeout factor it fails at start + timeout_mult *
 *    its t_comp on that instance if it would run longer; the failure frees
 *    its slot and t_queue like a completion, releases nothing, and the
 *    request is dispatched again at that time over the other instances
 *    (round robin steps past the failed one).  Attempts that start outside
 *    every window never time out.
 *
 * Errors: every function returns an HX_* status; nothing throws or aborts
 * across the ABI.  hx_last_error() returns the calling thread's last message.
 * Ownership: the caller keeps its host buffers (they may be freed once
 * hx_sim_create returns); the library owns all device memory of a handle.
 */
#ifndef HXSIM_H
#define HXSIM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define HX_SCALE 1000000LL

enum {
  HX_OK = 0,
  HX_ERR_INVALID = 1,    /* malformed or out-of-range input */
  HX_ERR_CUDA = 2,       /* a CUDA runtime call failed */
  HX_ERR_OOM = 3,        /* device or host allocation failed */
  HX_ERR_CAPACITY = 4,   /* a simulation outgrew its scratch (per-sim status) */
  HX_ERR_STEP_LIMIT = 5, /* a simulation exceeded its event bound (per-sim status) */
  HX_ERR_STATE = 6,      /* call out of order (e.g. results before run) */
  HX_ERR_INVARIANT = 7,  /* a simulation broke a scheduler invariant (per-sim status;
                            a library bug, never expected) */
  HX_SKIPPED = 8,        /* not in the run's subset (per-sim status) */
  HX_ERR_BOUNDS = 9      /* bounds-checked build only: an index the simulation formed was out
                            of range; the access was skipped (per-sim status; a library bug,
                            never expected) */
};

enum { HX_STAGE_S = 0, HX_STAGE_G = 1, HX_STAGE_C = 2, HX_STAGE_E = 3 };
enum { HX_LOCAL_PQ = 0, HX_LOCAL_FCFS = 1, HX_LOCAL_LLF = 2 };
enum { HX_DISPATCH_WB = 0, HX_DISPATCH_RR = 1 };
enum { HX_OBJ_P95 = 0, HX_OBJ_P95_SLO95 = 1 };

/* Limits checked by hx_sim_create. */
#define HX_MAX_INST 64
#define HX_MAX_TYPES 4
#define HX_MAX_SLOTS 16
#define HX_MAX_K 8
#define HX_MAX_RETRY 15
#define HX_MAX_TENANTS 4
#define HX_MAX_FAULTS 16

/* One request trace (host memory).  Calls of query i are
 * [call_base[i], call_base[i+1]) in the order S, G_0..G_{k-1}, the
 * corrections C_{c,r} by (c, r) ascending (r = 1..r_c), then E.
 * The request id of a call is its index within the trace. */
typedef struct hx_trace {
  int32_t n_queries;
  int32_t n_calls;              /* < 2^24 */
  const int64_t* arrival_us;    /* [n_queries] non-decreasing, >= 0 */
  const uint8_t* k;             /* [n_queries] 1..8, or 0 for a single-shot request (one E call) */
  const int32_t* call_base;     /* [n_queries + 1] */
  const int32_t* prompt;        /* [n_calls] >= 1 */
  const int32_t* out;           /* [n_calls] true output tokens >= 0 */
  const int32_t* out_est;       /* [n_calls] scheduler's believed output tokens >= 0 */
  const uint8_t* stage;         /* [n_calls] HX_STAGE_* */
  const uint8_t* cand;          /* [n_calls] candidate c (G and C calls) */
  const uint8_t* retry;         /* [n_calls] r for C calls, 0 otherwise */
  const uint8_t* tenant;        /* [n_queries] < cluster n_tenants; NULL = all tenant 0 */
} hx_trace;

/* A fault window of one instance: attempts that start on `inst` at a time in
 * [t0_us, t1_us) run slow_fp / SCALE times longer; slow_fp = 0 means they
 * never finish (only allowed with a timeout).  The first listed window that
 * covers a start applies. */
typedef struct hx_fault {
  int32_t inst;
  int32_t pad;
  int64_t t0_us;                    /* 0 <= t0_us <= t1_us <= 2^38 */
  int64_t t1_us;
  int64_t slow_fp;                  /* 0, or SCALE / 100 .. 100 * SCALE */
} hx_fault;

/* Heterogeneous instances (Sec. 3.3's empirical performance profiles). */
typedef struct hx_cluster {
  int32_t n_types;                  /* 1..4 */
  const int32_t* prefill_tok_s;     /* [n_types] >= 1 */
  const int32_t* decode_us_tok;     /* [n_types] >= 0 */
  const int32_t* slots;             /* [n_types] 1..16 concurrent requests */
  int32_t n_inst;                   /* 1..64 */
  const uint8_t* inst_type;         /* [n_inst] */
  int32_t ref_type;                 /* type whose exclusive latency defines T_slo */
  int64_t slo_mult_fp;              /* T_slo = slo_mult_fp * L0 / SCALE, <= 16 * SCALE */
  int32_t rmax;                     /* workflow's retry bound R, 0..15 */
  const int32_t* stage_ref_prompt;  /* [4] reference tokens per stage (S,G,C,E) */
  const int32_t* stage_ref_out;     /* [4] */
  int32_t n_tenants;                /* 0 or 1 = one tenant; up to HX_MAX_TENANTS */
  int32_t n_faults;                 /* 0..HX_MAX_FAULTS */
  const int64_t* tenant_slo_mult_fp;  /* [n_tenants] SLO multipliers (<= 16 * SCALE), NULL =
                                         slo_mult_fp for every tenant */
  int64_t timeout_mult_fp;          /* 0 = no timeout, else SCALE .. 100 * SCALE */
  const hx_fault* faults;           /* [n_faults] */
} hx_cluster;

/* Hyper-parameter points (host memory). */
typedef struct hx_grid {
  int32_t n_points;
  const int64_t* alpha_fp;          /* [n] 0..SCALE (Eq. score's alpha) */
  const int64_t* gamma_fp;          /* [n] 0..4*SCALE (urgency ageing weight) */
  const int32_t* rho;               /* [n] 0..15 corrections assumed by the budget */
  const int64_t* beta_us2;          /* [n] >= 0, beta = C_ref * Q_ref */
  const uint8_t* local_policy;      /* [n] HX_LOCAL_*: urgency queue (Sec. 4.2), FCFS, or the
                                       least-laxity-first baseline of Sec. 5.1 */
  const uint8_t* dispatch_policy;   /* [n] HX_DISPATCH_* */
} hx_grid;

typedef struct hx_options {
  int32_t n_record;                 /* >= 0 simulations whose per-call log is kept (runs
                                       the generic kernel) */
  const int32_t* record_sims;       /* [n_record] distinct sim indices (trace * P + point) */
  int32_t max_resident_warps;       /* 0 = fill the GPU */
  int32_t timing;                   /* 1 = time each kernel with CUDA events */
  int32_t force_generic;            /* 1 = always use the simulation kernel built for
                                       mixed policies and logging (testing) */
  int32_t n_subset;                 /* 0 = run every simulation */
  const int32_t* sim_subset;        /* [n_subset] distinct sim indices to run, any order; the
                                       others report HX_SKIPPED, and the best-point
                                       reduction counts them as failed */
  int32_t checked;                  /* 1 = also check the scheduler's invariants after every
                                       event (runs the generic kernel) */
  int32_t arena_entries;            /* testing: local-queue entries per resident warp
                                       (0 = enough for any run); a simulation whose
                                       queues outgrow it reports HX_ERR_CAPACITY */
} hx_options;

/* Per-simulation result, index sim = trace * n_points + point. */
typedef struct hx_result {
  int64_t p95_us;       /* nearest-rank P95 of query latency (-1 if failed) */
  int64_t makespan_us;  /* completion time of the last query */
  int64_t events;       /* completed LLM calls (= n_calls when ok) */
  uint64_t digest;      /* order-free checksum of every call's (id, instance, start)
                           and every query's (id, end) */
  int32_t slo_met;      /* queries with latency <= T_slo */
  int32_t n_done;       /* completed queries */
  int32_t status;       /* HX_OK, HX_ERR_CAPACITY, HX_ERR_STEP_LIMIT, HX_ERR_INVARIANT
                           or HX_SKIPPED */
  int32_t cycles_k;     /* diagnostic: SM clock cycles / 1024 the simulation took
                           (saturated; varies from run to run) */
} hx_result;

/* Best point (Sec. 4.3's argmin of P95; the constrained objective keeps
 * points whose SLO attainment is >= 95%, else the most SLO hits).
 * Ties go to the lowest point index; failed simulations never win. */
typedef struct hx_best {
  int32_t global_point;       /* argmin over points of the sum over traces */
  int32_t pad;
  int64_t global_sum_p95;     /* its summed P95 */
  int64_t global_slo_met;     /* its summed SLO count */
  int32_t* per_trace_point;   /* caller-owned [n_traces], may be NULL */
} hx_best;

/* Per-simulation counts beside hx_result (Sec. 5's multi-tenant
 * evaluation): SLO hits, completed queries and the nearest-rank P95 of query
 * latency per tenant, and the attempts that timed out and were re-issued. */
typedef struct hx_extra {
  int32_t slo_met[HX_MAX_TENANTS];
  int32_t n_done[HX_MAX_TENANTS];
  int32_t reissued;
  int32_t pad;
  int64_t p95_us[HX_MAX_TENANTS];  /* sorted L_t[ceil(0.95 n_t) - 1] over tenant t's queries;
                                      0 for a tenant without queries, -1 if the simulation
                                      failed or was skipped */
} hx_extra;

typedef struct hx_sim hx_sim;

/* Validate and copy traces, cluster and grid to library-owned device memory
 * and size the per-warp scratch.  On failure *out is NULL.
 *
 * Defines the simulations of Sec. 4.3's alpha tuning: every (trace, point)
 * pair replays the trace through the scheduler of Sec. 4.1 (Eq. comp for
 * t_comp, the queue cost t_queue, Eq. score) and Sec. 4.2 (the SLO budget at
 * send time, Eq. priority), over the workflow of Sec. 2.1 on the instance
 * profiles of Sec. 3.3.  `traces` [n_traces] and the cluster and grid arrays
 * are host memory the caller keeps; `opt` may be NULL.  Errors:
 * HX_ERR_INVALID (input outside the domain above, with a message),
 * HX_ERR_OOM, HX_ERR_CUDA. */
int hx_sim_create(const hx_trace* traces, int32_t n_traces, const hx_cluster* cluster,
                  const hx_grid* grid, const hx_options* opt, hx_sim** out);

/* Replace the trace contents of an existing handle with traces of the same
 * shapes (n_queries and n_calls per trace), copying host -> device on
 * `stream`; no device allocation.  The traces are validated as at create
 * (on up to 16 host threads; the lowest-numbered bad trace is reported)
 * before anything is copied, and the call returns once the copies are done.
 * A trace whose tenant pointer is NULL puts every query in tenant 0, as at
 * create.  Errors: HX_ERR_INVALID, HX_ERR_OOM (host staging), HX_ERR_CUDA. */
int hx_sim_upload(hx_sim* h, const hx_trace* traces, int32_t n_traces, void* stream);

/* Enqueue the whole path on `stream` (a cudaStream_t, NULL = legacy default):
 * per-call preparation (Eq. comp per call and instance type, the mean cost
 * tbar of Sec. 4.2, the query deadline of Sec. 5.1's SLO), every
 * simulation (Sec. 4.1 dispatch and Sec. 4.2 local queues, event by event,
 * reduced to Sec. 4.3's T_0.95 and the SLO count), and the best-point
 * reduction (Sec. 4.3's argmin over the grid).  Asynchronous; may be called
 * repeatedly.  Errors: HX_ERR_INVALID (NULL handle), HX_ERR_CUDA (a launch
 * failed); per-simulation problems are reported in hx_result.status. */
int hx_sim_run(hx_sim* h, void* stream);

/* Wait for the last run and copy n <= n_sims results to host memory
 * (`host_out` [n], caller-owned): per simulation Sec. 4.3's objective T_0.95
 * (the nearest-rank P95 of query latency), the number of queries within
 * their SLO (Sec. 5.1: latency <= slo_mult times the exclusive latency),
 * makespan, completed calls, the digest and the status.  Errors:
 * HX_ERR_STATE before a run, HX_ERR_INVALID (n too large), HX_ERR_CUDA. */
int hx_sim_results(hx_sim* h, hx_result* host_out, size_t n);

/* Wait for the last run and copy n <= n_sims per-tenant counts (see
 * hx_extra; Sec. 5's multi-tenant SLO attainment); same indexing as
 * hx_sim_results. */
int hx_sim_extras(hx_sim* h, hx_extra* host_out, size_t n);

/* Wait for the last run and return the best point for `objective`:
 * Sec. 4.3's alpha* = argmin T_0.95 per trace and over the grid (sum over
 * traces), or the same among points with >= 95% SLO attainment.
 * out->per_trace_point, if not NULL, is caller memory of n_traces. */
int hx_sim_best(hx_sim* h, int32_t objective, hx_best* out);

/* Per-point sums over the handle's traces from the last run (the partial
 * sums a rank contributes when traces are spread over several GPUs): summed
 * P95, summed SLO hits, and the number of failed simulations, each
 * [n_points] host arrays.  Waits for the run. */
int hx_sim_point_sums(hx_sim* h, int64_t* sum_p95, int64_t* sum_slo_met, int32_t* n_failed, size_t n_points);

/* The grid's best point (Sec. 4.3) from per-point sums added up over every
 * rank's traces, with the same rules as hx_sim_best; n_queries_total is the
 * number of queries behind the sums.  Runs the best-point kernel on the
 * current device (allocating a small temporary buffer); synchronous. */
int hx_best_of_sums(const int64_t* sum_p95, const int64_t* sum_slo_met, const int32_t* n_failed, int32_t n_points,
                    int64_t n_queries_total, int32_t objective, hx_best* out);

/* Per-call log of recorded simulation `rec_index` (position in
 * opt.record_sims): instance, dispatch time, SLO budget, start and end time
 * of every call of its trace (its last attempt when attempts were
 * re-issued).  Arrays are [n_calls] of that trace; any may be NULL. */
int hx_sim_records(hx_sim* h, int32_t rec_index, int32_t* inst, int64_t* enq_us,
                   int64_t* budget_us, int64_t* start_us, int64_t* end_us, size_t n_calls);

/* Per-call preparation output of trace `trace_index` after a run: Eq. (comp)
 * per type (est with the believed output, svc with the true output),
 * [n_calls * 4] type-minor (unused types 0); the mean over instances tbar
 * [n_calls]; and the query deadline (arrival + T_slo) of each call
 * [n_calls].  Any pointer may be NULL. */
int hx_sim_prep(hx_sim* h, int32_t trace_index, int32_t* est, int32_t* svc, int32_t* tbar,
                int64_t* deadline_us, size_t n_calls);

/* Milliseconds of the last run's kernels (prep, simulate, best); needs
 * opt.timing = 1.  Waits for the run. */
int hx_sim_timings(hx_sim* h, float* prep_ms, float* sim_ms, float* best_ms);

/* The same for an earlier run: back = 0 is the last run, 1 the one before,
 * up to min(runs, 64) - 1 (the handle keeps the events of its last 64
 * runs).  Waits for that run.  HX_ERR_INVALID for `back` out of range. */
int hx_sim_timings_back(hx_sim* h, int32_t back, float* prep_ms, float* sim_ms, float* best_ms);

/* Size of the device array behind hx_sim_run_static. */
#define HX_STATIC_SCRATCH_BYTES (64u << 20)

/* The whole path (preparation, every simulation of one trace, best point)
 * without allocating any memory, for callers that cannot allocate device
 * memory: code that runs where cudaMalloc is not allowed or not available (a
 * plugin or service whose host process owns every allocation, a real-time
 * loop that must not enter the allocator), or that cannot keep a handle.
 * It has no counterpart in the paper.
 *
 * Inputs (one trace, the cluster, the grid) and outputs (`results`, host
 * [n_points], and optionally `best` for `objective`) are the caller's host
 * memory, validated exactly as hx_sim_create validates them.  Every
 * intermediate buffer -- the copied inputs, the per-call records, the
 * per-warp local-queue arenas, the results -- is carved from one file-scope
 * device array of HX_STATIC_SCRATCH_BYTES (64 MiB), which every GPU that
 * loads the library holds until the process exits; a trace whose scratch
 * does not fit is rejected with HX_ERR_INVALID and a message giving the
 * bytes it would need.  Fewer warps run when the trace is large, so results
 * are the same as hx_sim_run's but throughput is lower.
 *
 * A call made while `stream` is not capturing looks up the current device's
 * address of the array (cudaGetSymbolAddress, with that device current), so
 * a device reset between calls is harmless; a call made during stream
 * capture reuses the address of the last earlier call on that device, so
 * the first call on a device must come before any stream capture
 * (HX_ERR_STATE otherwise).  Runs on `stream` and returns when the results
 * are in `results`.  Every call on a device shares the one array, whose
 * contents the next call overwrites: calls that overlap on the GPU (other
 * threads, other streams) race and corrupt each other. */
int hx_sim_run_static(const hx_trace* trace, const hx_cluster* cluster, const hx_grid* grid,
                      int32_t objective, hx_result* results, hx_best* best, void* stream);

/* Self-test of the library's device integer division (the reward and budget
 * quotients): divides count pairs (host arrays, n < 2^63, 1 <= d < 2^54) on
 * the current device with the library's routine into q and with the
 * compiler's 64-bit division into q_ref.  Allocates and frees its own device
 * buffers; synchronous. */
int hx_selftest_div(const uint64_t* n, const uint64_t* d, uint64_t* q, uint64_t* q_ref, size_t count);

typedef struct hx_info {
  int64_t n_sims;
  int64_t n_calls_total;
  int64_t n_queries_total;
  int64_t scratch_bytes;        /* per-warp scratch, all resident warps */
  int64_t device_bytes;         /* everything the handle holds on the device */
  int32_t resident_warps;
  int32_t warps_per_block;
  int32_t blocks;
  int32_t smem_per_block;
  int32_t generic_kernel;       /* 1: the kernel with logging and every policy; 0: the
                                   PQ + workload-balanced instantiation without logging */
  int32_t work_order;           /* order the simulations are taken in: 0 trace-major, highest
                                   point first; 1 the caller's subset (likewise ordered);
                                   2 every trace's workload-balanced alpha = 1 points first
                                   (their long local queues make them the costliest), chosen
                                   when the run is 1-4 waves of warps deep and every trace's
                                   records fit in L2; 3 trace-major, but the traces of about
                                   the last two waves take their alpha = 1 points first
                                   (deeper runs).  Results never depend on it. */
} hx_info;

int hx_sim_info(hx_sim* h, hx_info* out);

/* Wait for the handle's last run and free everything it holds (the end of
 * the tuning pass of Sec. 4.3); NULL is allowed.  Always HX_OK. */
int hx_sim_destroy(hx_sim* h);

/* The calling thread's last error message ("" if none). */
const char* hx_last_error(void);

#ifdef __cplusplus
}
#endif
#endif
