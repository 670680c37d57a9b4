// hx_device.cuh -- device-side data layout and kernels of the batched
// HexGen-Flow scheduler simulation (arXiv 2505.05286, Sec. 4) for sm_103a.
//
//   hx_prep_kernel  : per query, Eq. (comp) per call and instance type, the
//                     mean cost tbar of Sec. 4.2, workflow successor links
//                     (Sec. 2.1) and the query deadline (SLO of Sec. 5.1);
//                     writes one 64-byte record per call.
//   hx_sim_kernel   : persistent; one warp runs one (trace, point) discrete
//                     event simulation of the workload-balanced dispatcher
//                     (Sec. 4.1) and the urgency queues (Sec. 4.2), and
//                     reduces it to P95 / SLO count / digest (Sec. 4.3).
//   hx_best_kernel  : argmin of the P95 objective per trace and over the grid.
#pragma once

#include <stdint.h>

#include "hxsim.h"

namespace hx {

constexpr int64_t kScale = 1000000;       // fixed point of alpha, gamma, slo_mult
constexpr int64_t kUsPerS = 1000000;      // prefill throughput is per second
constexpr int64_t kRewardCap = (int64_t(1) << 43) - 1;
constexpr uint64_t kKeyInf = ~0ull;
// Event keys (time << 7 | instance) stay below 2^46: every time is below 2^39.
constexpr uint64_t kNoEvent = 1ull << 46;
constexpr int64_t kTimeInf = INT64_MAX;
constexpr int kWarpsPerBlock = 4;
constexpr unsigned kFull = 0xffffffffu;
constexpr uint64_t kArrivalTag = 64;      // event-key tag: after every instance
constexpr int kFRows = 18;                // S, G/C with 0..15 corrections done, E

// One call as the simulator reads it: 64 bytes, 16-byte aligned.
struct __align__(16) CallRec {
  int2 ev[4];         // per type: Eq. (comp) with the believed output length, and the
                      // same with the true output length (service time)
  int64_t deadline;   // query arrival + T_slo
  int64_t arrival;    // query arrival
  int32_t tbar;       // mean of est over the instances
  int32_t next;       // S: unused; G/C: next correction's id, or ~(E's id) at chain end
  int32_t qid;        // query index within the trace
  uint8_t stage, u, k, fcode;  // stage, corrections done incl. this call (E: the query's
                               // tenant), k of the query, row of the rest-of-path table:
                               // S 0, G/C 1 + u, E 17
};
static_assert(sizeof(CallRec) == 64, "CallRec is one 64-byte unit");

// Local-queue entry: priority key (higher first) and request id (lower first).
struct __align__(16) HeapEnt {
  long long key;
  int rid;
  int svc;   // service time on the queue's instance
};

// A fault window of one instance (see hx_fault).
struct FaultK {
  int64_t t0, t1, slow;
  int32_t inst, pad;
};

// Cluster description passed by value (kernel parameter space).
struct ClusterK {
  int32_t n_inst, n_types, ref_type, rmax;
  int64_t slo_mult_fp;
  int32_t prefill[HX_MAX_TYPES], decode[HX_MAX_TYPES], slots[HX_MAX_TYPES], cnt[HX_MAX_TYPES];
  int32_t ref_prompt[4], ref_out[4];
  int32_t total_slots;
  int32_t smem_per_warp;
  uint8_t inst_type[HX_MAX_INST];
  uint8_t inst_slots[HX_MAX_INST];
  uint16_t slot_base[HX_MAX_INST];
  // tenants and faults (only the generic simulation kernel handles faults)
  int32_t n_tenants, n_faults;
  int64_t tenant_mult[HX_MAX_TENANTS];
  int64_t timeout_mult_fp;
  FaultK faults[HX_MAX_FAULTS];
};

struct PrepArgs {
  const int64_t* arrival;   // [Q]
  const uint8_t* kq;        // [Q]
  const int64_t* qcall;     // [Q + 1] first call (global index) of each query
  const int64_t* q_off;     // [T + 1]
  const int64_t* c_off;     // [T + 1]
  const int32_t* prompt;
  const int32_t* out;
  const int32_t* out_est;
  const uint8_t* stage;
  const uint8_t* cand;
  const uint8_t* retry;
  const uint8_t* tenant;    // [Q] or NULL
  int64_t n_queries;
  int32_t n_traces;
  CallRec* rec;             // [C]
  unsigned long long* work_counter;
  hx_result* skip_results;  // with a subset: every result starts as HX_SKIPPED
  hx_extra* skip_extras;    // and its per-tenant counts at zero (NULL: none kept)
  int64_t n_skip;           // n_sims with a subset, else 0
};

struct SimArgs {
  const CallRec* rec;
  const int64_t* arrival;
  const int64_t* qcall;
  const int64_t* q_off;
  const int64_t* c_off;
  const int64_t* alpha;
  const int64_t* gamma;
  const int32_t* rho;
  const int64_t* beta;
  const uint8_t* lpol;
  const uint8_t* dpol;
  int32_t n_points;
  int32_t n_traces;
  int64_t n_sims;
  hx_result* results;
  unsigned long long* work_counter;
  HeapEnt* arena;           // per resident warp: arena_per_warp entries
  int64_t arena_per_warp;
  uint8_t* chains;          // per resident warp: chains_per_warp bytes
  int64_t chains_per_warp;
  int64_t* topk;            // per resident warp: topk_per_warp latencies
  int64_t topk_per_warp;
  const int32_t* rec_map;   // [n_sims] record slot or -1; NULL when not recording
  int32_t* rec_inst;
  int64_t* rec_enq;
  int64_t* rec_budget;
  int64_t* rec_start;
  int64_t* rec_end;
  int64_t rec_stride;
  hx_extra* extras;         // [n_sims] per-tenant counts and re-issues (generic kernel), or NULL
  const int32_t* tenant_kcap;  // [n_traces * 4] top-K size per (trace, tenant) (0: no queries), or
                               // NULL: one tenant
  int64_t tenant_topk_off[HX_MAX_TENANTS];  // tenant t's top-K heap within the warp's topk slice
  const int64_t* subset;    // [n_work] sims to run in work order, or NULL: all n_sims
  int64_t n_work;
  int32_t checked;          // check the scheduler's invariants after every event (generic kernel)
};

// Per-warp shared memory of one simulation: per-instance local-queue and
// slot state, per-simulation constants and lane-0 accumulators, then one
// 64-bit (end << 24 | request id) key per batch slot of the cluster.  An
// instance's running calls occupy the first cnt of its slots in ascending key
// order, so the next completion on it is always its first slot.
struct WarpShared {
  int64_t q[HX_MAX_INST];       // t_queue: Eq. comp summed over requests dispatched and unfinished
  uint64_t ekey[HX_MAX_INST];   // next completion event key per instance
  int32_t erid[HX_MAX_INST];    // its request id
  int64_t orew[HX_MAX_INST];    // cached (1 - alpha) * reward per instance (its owner lane's)
  int32_t hoff[HX_MAX_INST];    // local queue: heap offset in the arena
  int32_t hsize[HX_MAX_INST];   //              heap size
  uint8_t cnt[HX_MAX_INST];     // running calls (the first cnt of the instance's slot keys)
  uint8_t hcl[HX_MAX_INST];     // local queue: heap capacity 8 << hcl (0: none yet)
  // this event's dispatches in order: (request id, service time), Eq. (comp) on the winner
  int2 prs[HX_MAX_K];
  int32_t pest[HX_MAX_K];
  // per-simulation constants
  int32_t A, one_minus_a;        // alpha and 1 - alpha, fixed point
  int32_t rewards, oob;          // 1 when dispatch scores need the reward term; an index check
                                // failed (bounds-checked build)
  int64_t G, beta;
  float betaf, pad3;            // beta as a float (the reward quotient's numerator)
  int64_t frest[kFRows];        // rest-of-path cost of the budget denominator by fcode
  int32_t lpol, dpol, recj, kcap, rr, bump;
  // this warp's scratch slices and the current trace's offsets
  HeapEnt* arena;
  uint8_t* chains;
  int64_t* topk;
  int64_t qb, cb;
  int32_t nq, nc;
  int64_t sim, clk0;            // result index and start clock of the simulation
  uint64_t akey;                // next arrival's event key (written alike by every lane)
  int32_t qa, trace;            // arrivals taken so far (likewise); the simulation's trace
  // lane-0 accumulators
  uint64_t digest;
  int64_t makespan;
  int32_t n_done, slo_met, events, tk;
  int64_t tkmin;                // root of the full top-K heap (written alike by every lane)
  longlong2 dterm[16];          // digest terms waiting to be hashed: (time, id tag)
  int32_t tslo[HX_MAX_TENANTS], tdone[HX_MAX_TENANTS];  // per-tenant counts (generic kernel)
  int32_t ttk[HX_MAX_TENANTS];  // per-tenant top-K heaps: entries (generic kernel with tenants)
  int64_t ttkmin[HX_MAX_TENANTS];  //                 and roots once full
  int32_t reissued, excl;       // timed-out attempts; the instance a re-issue avoids (-1: none)
  uint64_t slot[1];             // [total_slots], then with faults one fail flag byte per slot
};

struct BestCand {
  int64_t p95;
  int64_t slo;
  int32_t p;
  int32_t flags;  // bit0 valid, bit1 feasible
};

struct BestArgs {
  const hx_result* results;
  const int64_t* q_off;
  int32_t n_traces;
  int32_t n_points;
  BestCand* per_trace;      // [T * 2]
  BestCand* global;         // [2]
  int64_t* point_sums;      // [P * 3] (sum P95, sum SLO hits, failed sims) or NULL
};

__global__ void hx_prep_kernel(PrepArgs a, ClusterK c);
// hx_sim_kernel: any mix of dispatch and local-queue policies and per-call
// logs; hx_sim_kernel_lean: every point workload-balanced with the urgency
// queue, nothing logged (the same simulation with those branches removed).
__global__ void hx_sim_kernel(SimArgs a, ClusterK c);
__global__ void hx_sim_kernel_lean(SimArgs a, ClusterK c);
__global__ void hx_best_kernel(BestArgs a);
__global__ void hx_selftest_div_kernel(const uint64_t* n, const uint64_t* d, uint64_t* q, uint64_t* q_ref,
                                       int64_t count);

}  // namespace hx
