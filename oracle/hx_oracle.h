/*
 * hx_oracle.h -- reference CPU simulator of the HexGen-Flow scheduler.
 *
 * TEST INFRASTRUCTURE ONLY.  This is the slow, single-threaded, plain-C
 * statement of what the batched simulation computes, used to check the CUDA
 * library bit for bit.  Only the tests, the smoke check and the CPU-baseline
 * leg of the benchmark may load it; the library never does.
 *
 * It shares no code, header, table or helper with the CUDA library.
 */
#ifndef HX_ORACLE_H
#define HX_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct {
  int32_t n_queries;
  int32_t n_calls;
  const int64_t* arrival_us;  /* [n_queries], non-decreasing */
  const uint8_t* k;           /* [n_queries] candidates per query */
  const int32_t* call_base;   /* [n_queries + 1] */
  const int32_t* prompt;      /* [n_calls] input tokens */
  const int32_t* out;         /* [n_calls] true output tokens */
  const int32_t* out_est;     /* [n_calls] believed output tokens */
  const uint8_t* stage;       /* [n_calls] 0=S 1=G 2=C 3=E */
  const uint8_t* cand;        /* [n_calls] */
  const uint8_t* retry;       /* [n_calls] */
  const uint8_t* tenant;      /* [n_queries] tenant of each query, NULL = all tenant 0 */
} hxo_trace;

/* A fault window of one instance: attempts that start on it in [t0, t1)
 * run slow_fp / SCALE times longer; slow_fp = 0 means they never finish. */
typedef struct {
  int32_t inst;
  int32_t pad;
  int64_t t0_us;
  int64_t t1_us;
  int64_t slow_fp;
} hxo_fault;

#define HXO_MAX_TENANTS 4

typedef struct {
  int32_t n_types;
  const int32_t* prefill_tok_s;  /* [n_types] */
  const int32_t* decode_us_tok;  /* [n_types] */
  const int32_t* slots;          /* [n_types] */
  int32_t n_inst;
  const uint8_t* inst_type;      /* [n_inst] */
  int32_t ref_type;
  int64_t slo_mult_fp;
  int32_t rmax;
  const int32_t* stage_ref_prompt;  /* [4] */
  const int32_t* stage_ref_out;     /* [4] */
  int32_t n_tenants;                /* 1..HXO_MAX_TENANTS */
  int32_t n_faults;
  const int64_t* tenant_slo_mult_fp;  /* [n_tenants], NULL = slo_mult_fp for every tenant */
  int64_t timeout_mult_fp;          /* 0 = no timeout, else >= SCALE */
  const hxo_fault* faults;          /* [n_faults] */
} hxo_cluster;

typedef struct {
  int64_t alpha_fp;
  int64_t gamma_fp;
  int64_t beta_us2;
  int32_t rho;
  int32_t local_policy;     /* 0 = urgency PQ, 1 = FCFS, 2 = least laxity first */
  int32_t dispatch_policy;  /* 0 = workload balanced, 1 = round robin */
} hxo_point;

typedef struct {
  int64_t p95_us;
  int64_t makespan_us;
  int64_t events;       /* completed LLM calls */
  uint64_t digest;
  int32_t slo_met;
  int32_t n_done;
  int32_t status;       /* 0 ok, otherwise an HXO_ERR_* code */
  int32_t pad;
} hxo_result;

enum { HXO_OK = 0, HXO_ERR_INVALID = 1, HXO_ERR_OOM = 3, HXO_ERR_INVARIANT = 7 };

/* Per-tenant SLO counts and the number of timed-out attempts re-issued. */
typedef struct {
  int32_t slo_met[HXO_MAX_TENANTS];
  int32_t n_done[HXO_MAX_TENANTS];
  int32_t reissued;
  int32_t pad;
  int64_t p95_us[HXO_MAX_TENANTS]; /* nearest-rank P95 of each tenant's query latencies
                                      (0 for a tenant without queries, -1 if failed) */
} hxo_extra;

/* Per-call estimates of Eq. (comp) and the mean over instances, and the
 * per-query SLO.  est/svc are [n_calls * n_types] (type-minor). */
int hxo_prep(const hxo_trace* tr, const hxo_cluster* cl, int64_t* est, int64_t* svc,
             int64_t* tbar, int64_t* t_slo, int64_t* stage_ref_cost);

/* Optional per-call log; any pointer may be NULL, otherwise [n_calls]. */
typedef struct {
  int32_t* inst;    /* instance the call was dispatched to */
  int64_t* enq;     /* dispatch (= enqueue) time */
  int64_t* budget;  /* SLO budget t_slo assigned at dispatch */
  int64_t* start;
  int64_t* end;
} hxo_log;

/* One simulation.  log and ext may be NULL.  check != 0 re-verifies the
 * scheduler invariants after every event (slow). */
int hxo_simulate(const hxo_trace* tr, const hxo_cluster* cl, const hxo_point* pt,
                 int check, hxo_result* res, const hxo_log* log, hxo_extra* ext);

/* SLO budget of Sec. 4.2: (T_slo - elapsed) * tbar / remaining, truncated. */
int64_t hxo_budget(int64_t t_slo, int64_t elapsed, int64_t tbar, int64_t remaining);

/* Workload-balanced score of Eq. (score) in fixed point. */
int64_t hxo_score(int64_t alpha_fp, int64_t beta_us2, int64_t t_queue, int64_t t_comp);

/* Local-queue choice at a batch boundary: index of the request to start.
 * policy 0: argmax urgency_fp, ties to the lowest request id;
 * policy 1: earliest enqueue time, ties to the lowest request id. */
int32_t hxo_pick(int32_t policy, int32_t n, const int32_t* rid, const int64_t* urgency_fp,
                 const int64_t* enq_us);

/* Best point over a [n_traces * n_points] result table (Sec. 4.3). */
int hxo_best(const hxo_result* res, int32_t n_traces, int32_t n_points, const int32_t* n_queries,
             int32_t objective, int32_t* global_point, int64_t* global_sum_p95,
             int32_t* per_trace_point);

#ifdef __cplusplus
}
#endif
#endif
