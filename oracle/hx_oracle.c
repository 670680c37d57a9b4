/*
 * hx_oracle.c -- reference CPU simulator of the HexGen-Flow scheduler
 * (arXiv 2505.05286, Sec. 4).
 *
 * TEST INFRASTRUCTURE ONLY.  A plain, slow, single-threaded statement of the
 * discrete-event simulation that the alpha-tuning of Sec. 4.3 runs for every
 * hyper-parameter point: workload-balanced dispatch (Sec. 4.1, Eq. comp and
 * Eq. score), the per-instance urgency queue (Sec. 4.2, the SLO budget and
 * Eq. priority), the workflow dependencies of Sec. 2.1 / Sec. 3.3, and the
 * P95 objective of Sec. 4.3.  Every quantity is recomputed from its
 * definition where it is used (scores over every instance, urgency of every
 * waiting request at every batch boundary, linear scans for the next event);
 * nothing is cached, blocked or reordered.  Only the tests, the smoke check
 * and the CPU-baseline leg of the benchmark use it.
 *
 * Readings of the paper (stated once here, used below):
 *  - time is int64 microseconds; alpha, gamma and the SLO multiplier are
 *    fixed point with SCALE = 1e6; every division truncates toward zero;
 *  - the queue Theta^m of the dispatcher is every request dispatched to m
 *    and not yet finished (waiting or running); the max(., 1) guard keeps
 *    beta / t_queue finite for an empty instance and the reward is capped at
 *    2^43 - 1;
 *  - the remaining work in the budget denominator is this request's own
 *    mean cost plus the stage reference costs of the rest of its own path
 *    (S -> G -> up to min(rho, R - u) corrections -> E);
 *  - urgency ages with weight gamma: U = t_comp - t_slo + gamma * tau;
 *  - the LLF baseline of Sec. 5.1 orders waiting requests by the query's
 *    laxity, deadline - now - remaining work, where the remaining work is
 *    the same remaining-path cost as the budget denominator;
 *  - events are taken one at a time ordered by (time, completions before
 *    arrivals, instance, request id / query id); after each event the
 *    released successors are dispatched in request-id order, then every
 *    instance with a free slot starts its most urgent waiting request;
 *  - P95 is the nearest-rank percentile: sorted latencies L[ceil(.95 n) - 1];
 *  - several tenants (the multi-tenant evaluation of Sec. 5): each query
 *    belongs to one, whose SLO multiplier replaces the cluster's in T_slo;
 *    SLO attainment is also counted per tenant;
 *  - a single-shot request (the competing workloads of Sec. 5) is a query
 *    with k = 0 made of one evaluation-stage call E: it is dispatched on
 *    arrival, its budget denominator is its own mean cost and its exclusive
 *    latency is that call on the reference type;
 *  - timeout and re-issue (Sec. 3.3, for an instance that becomes slow or
 *    unavailable): an attempt that starts on an instance inside one of its
 *    fault windows runs slow_fp / SCALE times longer (rounded up; slow_fp =
 *    0: it never finishes; the first listed window that covers the start
 *    applies).  With a timeout factor, such an attempt whose running time
 *    would exceed timeout_mult * its Eq. (comp) estimate on that instance
 *    fails at start + that timeout (attempts started outside every window
 *    never time out, so re-issues end with the windows): like a completion it
 *    frees its slot and its estimate from Theta^m, releases nothing, and
 *    the request is dispatched again at that time by the same policy over
 *    the other instances (over all of them when there is one); round robin
 *    steps past the failed instance.  Per-call logs keep the last attempt.
 */
#include "hx_oracle.h"

#include <stdlib.h>
#include <string.h>

#define US_PER_S 1000000LL
#define FP_ONE 1000000LL
#define REWARD_CAP ((((int64_t)1) << 43) - 1)

enum { ST_S = 0, ST_G = 1, ST_C = 2, ST_E = 3 };
enum { C_PENDING = 0, C_WAITING = 1, C_RUNNING = 2, C_DONE = 3 };

typedef __int128 i128;

/* ---------------------------------------------------------------- helpers */
static int64_t ceil_div_pos(int64_t a, int64_t b) { return (a + b - 1) / b; }

/* Eq. (comp): prefill time of the input plus decode time of the output. */
static int64_t cost_on_type(const hxo_cluster* cl, int type, int64_t prompt, int64_t out_tokens) {
  return ceil_div_pos(prompt * US_PER_S, cl->prefill_tok_s[type]) +
         out_tokens * (int64_t)cl->decode_us_tok[type];
}

static int64_t est_on(const hxo_trace* tr, const hxo_cluster* cl, int m, int32_t c) {
  return cost_on_type(cl, cl->inst_type[m], tr->prompt[c], tr->out_est[c]);
}

static int64_t svc_on(const hxo_trace* tr, const hxo_cluster* cl, int m, int32_t c) {
  return cost_on_type(cl, cl->inst_type[m], tr->prompt[c], tr->out[c]);
}

/* Mean over instances of Eq. (comp) (the t-bar of Sec. 4.2). */
static int64_t mean_est(const hxo_trace* tr, const hxo_cluster* cl, int32_t c) {
  int64_t s = 0;
  for (int m = 0; m < cl->n_inst; ++m) s += est_on(tr, cl, m, c);
  return s / cl->n_inst;
}

static int64_t stage_ref(const hxo_cluster* cl, int s) {
  int64_t sum = 0;
  for (int m = 0; m < cl->n_inst; ++m)
    sum += cost_on_type(cl, cl->inst_type[m], cl->stage_ref_prompt[s], cl->stage_ref_out[s]);
  return sum / cl->n_inst;
}

/* The splitmix64 output function (Steele, Lea & Flood, "Fast splittable
 * pseudorandom number generators", OOPSLA 2014): two xor-shift-multiply
 * rounds and a final xor-shift, each a bijection of 64-bit words. */
static uint64_t splitmix64_mix(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

/* Digest term of a (time, id << 8 | tag) pair: the splitmix64 output
 * function of (time * 0x9E3779B97F4A7C15) xor idtag. */
static uint64_t digest_term(uint64_t t, uint64_t idtag) {
  return splitmix64_mix((t * 0x9E3779B97F4A7C15ULL) ^ idtag);
}

static uint64_t call_term(int32_t rid, int inst, int64_t start) {
  return digest_term((uint64_t)start, ((uint64_t)(uint32_t)rid << 8) | (uint64_t)inst);
}

static uint64_t query_term(int32_t qid, int64_t end) {
  return digest_term((uint64_t)end, ((uint64_t)(uint32_t)qid << 8) | 0xFFu);
}

static int cmp_i64(const void* a, const void* b) {
  int64_t x = *(const int64_t*)a, y = *(const int64_t*)b;
  return (x > y) - (x < y);
}

/* ------------------------------------------------------------ validation */
static int validate(const hxo_trace* tr, const hxo_cluster* cl) {
  if (cl->n_types < 1 || cl->n_inst < 1) return 0;
  for (int t = 0; t < cl->n_types; ++t)
    if (cl->prefill_tok_s[t] < 1 || cl->decode_us_tok[t] < 0 || cl->slots[t] < 1) return 0;
  for (int m = 0; m < cl->n_inst; ++m)
    if (cl->inst_type[m] >= cl->n_types) return 0;
  if (cl->ref_type < 0 || cl->ref_type >= cl->n_types || cl->rmax < 0) return 0;
  if (cl->n_tenants < 1 || cl->n_tenants > HXO_MAX_TENANTS || cl->n_faults < 0) return 0;
  if (cl->timeout_mult_fp != 0 && cl->timeout_mult_fp < FP_ONE) return 0;
  for (int f = 0; f < cl->n_faults; ++f) {
    const hxo_fault* F = &cl->faults[f];
    if (F->inst < 0 || F->inst >= cl->n_inst || F->t0_us < 0 || F->t1_us < F->t0_us || F->slow_fp < 0) return 0;
    if (F->slow_fp == 0 && cl->timeout_mult_fp == 0) return 0; /* would never finish */
  }
  if (tr->n_queries < 0 || tr->call_base[0] != 0 || tr->call_base[tr->n_queries] != tr->n_calls) return 0;
  for (int32_t i = 0; i < tr->n_queries; ++i) {
    if (i > 0 && tr->arrival_us[i] < tr->arrival_us[i - 1]) return 0;
    if (tr->arrival_us[i] < 0) return 0;
    if (tr->tenant && tr->tenant[i] >= cl->n_tenants) return 0;
    int32_t b = tr->call_base[i], e = tr->call_base[i + 1], k = tr->k[i];
    if (k == 0) {
      /* a single-shot request: one evaluation-stage call */
      if (e - b != 1 || tr->stage[b] != ST_E || tr->prompt[b] < 1 || tr->out[b] < 0 || tr->out_est[b] < 0) return 0;
      continue;
    }
    if (k < 1 || e - b < 2 + k) return 0;
    if (tr->stage[b] != ST_S || tr->stage[e - 1] != ST_E) return 0;
    for (int c = 0; c < k; ++c)
      if (tr->stage[b + 1 + c] != ST_G || tr->cand[b + 1 + c] != c) return 0;
    int prev_c = -1, prev_r = 0;
    for (int32_t j = b + 1 + k; j < e - 1; ++j) {
      int c = tr->cand[j], r = tr->retry[j];
      if (tr->stage[j] != ST_C || c >= k || r < 1 || r > cl->rmax) return 0;
      if (c == prev_c) {
        if (r != prev_r + 1) return 0;
      } else {
        if (c < prev_c || r != 1) return 0;
      }
      prev_c = c;
      prev_r = r;
    }
    for (int32_t j = b; j < e; ++j)
      if (tr->prompt[j] < 1 || tr->out[j] < 0 || tr->out_est[j] < 0) return 0;
  }
  return 1;
}

/* ------------------------------------------------------------ public bits */
int64_t hxo_budget(int64_t t_slo, int64_t elapsed, int64_t tbar, int64_t remaining) {
  i128 num = (i128)(t_slo - elapsed) * (i128)tbar;
  return (int64_t)(num / remaining);
}

int64_t hxo_score(int64_t alpha_fp, int64_t beta_us2, int64_t t_queue, int64_t t_comp) {
  int64_t q = t_queue > 1 ? t_queue : 1;
  int64_t reward = beta_us2 / q;
  if (reward > REWARD_CAP) reward = REWARD_CAP;
  i128 s = (i128)(FP_ONE - alpha_fp) * reward - (i128)alpha_fp * t_comp;
  return (int64_t)s;
}

int32_t hxo_pick(int32_t policy, int32_t n, const int32_t* rid, const int64_t* urgency_fp,
                 const int64_t* enq_us) {
  int32_t best = -1;
  for (int32_t j = 0; j < n; ++j) {
    if (best < 0) { best = j; continue; }
    int better;
    if (policy == 0) {
      better = urgency_fp[j] > urgency_fp[best] ||
               (urgency_fp[j] == urgency_fp[best] && rid[j] < rid[best]);
    } else {
      better = enq_us[j] < enq_us[best] || (enq_us[j] == enq_us[best] && rid[j] < rid[best]);
    }
    if (better) best = j;
  }
  return best;
}

int hxo_prep(const hxo_trace* tr, const hxo_cluster* cl, int64_t* est, int64_t* svc, int64_t* tbar,
             int64_t* t_slo, int64_t* stage_ref_cost) {
  if (!validate(tr, cl)) return HXO_ERR_INVALID;
  const int T = cl->n_types;
  for (int32_t c = 0; c < tr->n_calls; ++c) {
    for (int t = 0; t < T; ++t) {
      est[(int64_t)c * T + t] = cost_on_type(cl, t, tr->prompt[c], tr->out_est[c]);
      svc[(int64_t)c * T + t] = cost_on_type(cl, t, tr->prompt[c], tr->out[c]);
    }
    tbar[c] = mean_est(tr, cl, c);
  }
  for (int s = 0; s < 4; ++s) stage_ref_cost[s] = stage_ref(cl, s);
  /* SLO: multiple of the exclusive latency on the reference type (Sec. 5.1):
   * S, then the slowest candidate chain (G plus its corrections), then E. */
  for (int32_t i = 0; i < tr->n_queries; ++i) {
    int32_t b = tr->call_base[i], e = tr->call_base[i + 1];
    int64_t chain[8] = {0, 0, 0, 0, 0, 0, 0, 0};
    int64_t l_s = 0, l_e = 0;
    for (int32_t j = b; j < e; ++j) {
      int64_t s = cost_on_type(cl, cl->ref_type, tr->prompt[j], tr->out[j]);
      if (tr->stage[j] == ST_S) l_s += s;
      else if (tr->stage[j] == ST_E) l_e += s;
      else chain[tr->cand[j]] += s;
    }
    int64_t longest = 0;
    for (int c = 0; c < tr->k[i]; ++c)
      if (chain[c] > longest) longest = chain[c];
    int64_t l0 = l_s + longest + l_e;
    int64_t mult = cl->slo_mult_fp;
    if (cl->tenant_slo_mult_fp) mult = cl->tenant_slo_mult_fp[tr->tenant ? tr->tenant[i] : 0];
    t_slo[i] = (int64_t)(((i128)mult * l0) / FP_ONE);
  }
  return HXO_OK;
}

/* ------------------------------------------------------------- simulator */
typedef struct {
  int32_t* v;
  int32_t n, cap;
} ivec;

static int ivec_push(ivec* a, int32_t x) {
  if (a->n == a->cap) {
    int32_t nc = a->cap ? 2 * a->cap : 16;
    int32_t* nv = (int32_t*)realloc(a->v, (size_t)nc * sizeof(int32_t));
    if (!nv) return 0;
    a->v = nv;
    a->cap = nc;
  }
  a->v[a->n++] = x;
  return 1;
}

static void ivec_remove_at(ivec* a, int32_t j) {
  memmove(a->v + j, a->v + j + 1, (size_t)(a->n - j - 1) * sizeof(int32_t));
  a->n--;
}

typedef struct {
  const hxo_trace* tr;
  const hxo_cluster* cl;
  const hxo_point* pt;
  int64_t* t_slo;       /* per query */
  int64_t cref[4];      /* stage reference costs */
  int32_t* qid;         /* per call */
  uint8_t* state;       /* per call */
  int32_t* inst;        /* per call */
  int64_t* enq;         /* per call */
  int64_t* budget;      /* per call */
  int64_t* remaining;   /* per call: remaining-path cost at dispatch */
  int64_t* start;       /* per call */
  int64_t* end;         /* per call */
  int32_t* chains_left; /* per query */
  int64_t* q;           /* per instance: sum of Eq. (comp) over Theta^m */
  ivec* waiting;        /* per instance */
  ivec* running;        /* per instance */
  uint8_t* failed;      /* per call: the running attempt times out */
  int64_t rr_next;
  uint64_t digest;
  int32_t reissued;
  int bad;
} sim_t;

/* Remaining mean cost of the request's own path (denominator of the budget). */
static int64_t remaining_cost(const sim_t* s, int32_t c, int64_t tb) {
  const int64_t R = s->cl->rmax;
  const int64_t rho = s->pt->rho;
  int st = s->tr->stage[c];
  int64_t corr_left;
  switch (st) {
    case ST_S:
      corr_left = rho < R ? rho : R;
      return tb + s->cref[ST_G] + corr_left * s->cref[ST_C] + s->cref[ST_E];
    case ST_G:
    case ST_C: {
      int64_t u = (st == ST_G) ? 0 : s->tr->retry[c];
      int64_t left = R - u;
      corr_left = rho < left ? rho : left;
      return tb + corr_left * s->cref[ST_C] + s->cref[ST_E];
    }
    default:
      return tb;
  }
}

/* Global coordinator (Sec. 4.1): budget at send time, score every instance
 * but `excl` (a re-issue's failed instance, -1 for none), dispatch to the
 * highest score (lowest index on ties), enqueue there. */
static void dispatch(sim_t* s, int32_t c, int64_t now, int excl) {
  const hxo_trace* tr = s->tr;
  const hxo_cluster* cl = s->cl;
  int32_t i = s->qid[c];
  int64_t tb = mean_est(tr, cl, c);
  int64_t elapsed = now - tr->arrival_us[i];
  s->remaining[c] = remaining_cost(s, c, tb);
  s->budget[c] = hxo_budget(s->t_slo[i], elapsed, tb, s->remaining[c]);
  int best = -1;
  if (cl->n_inst == 1) excl = -1;
  if (s->pt->dispatch_policy == 1) {
    best = (int)(s->rr_next % cl->n_inst);
    s->rr_next++;
    if (best == excl) {
      best = (int)(s->rr_next % cl->n_inst);
      s->rr_next++;
    }
  } else {
    int64_t best_score = 0;
    for (int m = 0; m < cl->n_inst; ++m) {
      if (m == excl) continue;
      int64_t sc = hxo_score(s->pt->alpha_fp, s->pt->beta_us2, s->q[m], est_on(tr, cl, m, c));
      if (best < 0 || sc > best_score) {
        best = m;
        best_score = sc;
      }
    }
  }
  s->inst[c] = best;
  s->enq[c] = now;
  s->state[c] = C_WAITING;
  s->q[best] += est_on(tr, cl, best, c);
  if (!ivec_push(&s->waiting[best], c)) s->bad = HXO_ERR_OOM;
}

/* Running time of an attempt of call c started on m at `now` under the
 * cluster's fault windows and timeout; *fail says the attempt times out. */
static int64_t attempt_time(const sim_t* s, int m, int32_t c, int64_t now, int* fail) {
  const hxo_cluster* cl = s->cl;
  int64_t run = svc_on(s->tr, cl, m, c);
  int in_window = 0, down = 0;
  for (int f = 0; f < cl->n_faults; ++f) {
    const hxo_fault* F = &cl->faults[f];
    if (F->inst == m && now >= F->t0_us && now < F->t1_us) {
      in_window = 1;
      if (F->slow_fp == 0) down = 1;
      else run = (int64_t)(((i128)run * F->slow_fp + FP_ONE - 1) / FP_ONE);
      break;
    }
  }
  *fail = 0;
  if (in_window && cl->timeout_mult_fp > 0) {
    int64_t timeout = (int64_t)(((i128)est_on(s->tr, cl, m, c) * cl->timeout_mult_fp) / FP_ONE);
    if (down || run > timeout) {
      *fail = 1;
      return timeout;
    }
  }
  return run;
}

/* Local queues (Sec. 4.2): at a batch boundary each instance with a free slot
 * starts its most urgent waiting request, re-evaluating urgency now. */
static void fill_slots(sim_t* s, int64_t now, int64_t** ubuf, int64_t** ebuf, int32_t** rbuf, int32_t* bufcap) {
  const hxo_trace* tr = s->tr;
  const hxo_cluster* cl = s->cl;
  for (int m = 0; m < cl->n_inst; ++m) {
    int slots = cl->slots[cl->inst_type[m]];
    while (s->running[m].n < slots && s->waiting[m].n > 0) {
      ivec* w = &s->waiting[m];
      if (w->n > *bufcap) {
        *bufcap = w->cap;
        *ubuf = (int64_t*)realloc(*ubuf, (size_t)*bufcap * sizeof(int64_t));
        *ebuf = (int64_t*)realloc(*ebuf, (size_t)*bufcap * sizeof(int64_t));
        *rbuf = (int32_t*)realloc(*rbuf, (size_t)*bufcap * sizeof(int32_t));
        if (!*ubuf || !*ebuf || !*rbuf) { s->bad = HXO_ERR_OOM; return; }
      }
      for (int32_t j = 0; j < w->n; ++j) {
        int32_t c = w->v[j];
        i128 u;
        if (s->pt->local_policy == 2) {
          /* LLF (Sec. 5.1): least laxity first, as an urgency to maximise */
          int32_t i = s->qid[c];
          int64_t laxity = tr->arrival_us[i] + s->t_slo[i] - now - s->remaining[c];
          u = -(i128)laxity;
        } else {
          /* Eq. (priority) with ageing weight gamma, in fixed point */
          u = (i128)FP_ONE * (est_on(tr, cl, m, c) - s->budget[c]) + (i128)s->pt->gamma_fp * (now - s->enq[c]);
        }
        if (u > (i128)INT64_MAX || u < (i128)INT64_MIN) s->bad = HXO_ERR_INVALID;
        (*ubuf)[j] = (int64_t)u;
        (*ebuf)[j] = s->enq[c];
        (*rbuf)[j] = c;
      }
      int32_t j = hxo_pick(s->pt->local_policy == 1 ? 1 : 0, w->n, *rbuf, *ubuf, *ebuf);
      int32_t c = w->v[j];
      ivec_remove_at(w, j);
      if (!ivec_push(&s->running[m], c)) { s->bad = HXO_ERR_OOM; return; }
      s->state[c] = C_RUNNING;
      s->start[c] = now;
      int fail;
      s->end[c] = now + attempt_time(s, m, c, now, &fail);
      s->failed[c] = (uint8_t)fail;
      s->digest += call_term(c, m, now);
    }
  }
}

static int check_invariants(const sim_t* s) {
  const hxo_cluster* cl = s->cl;
  for (int m = 0; m < cl->n_inst; ++m) {
    int slots = cl->slots[cl->inst_type[m]];
    if (s->running[m].n > slots) return 0;
    if (s->running[m].n < slots && s->waiting[m].n > 0) return 0; /* work conserving */
    int64_t sum = 0;
    for (int32_t j = 0; j < s->waiting[m].n; ++j) sum += est_on(s->tr, cl, m, s->waiting[m].v[j]);
    for (int32_t j = 0; j < s->running[m].n; ++j) sum += est_on(s->tr, cl, m, s->running[m].v[j]);
    if (sum != s->q[m]) return 0;
  }
  return 1;
}

int hxo_simulate(const hxo_trace* tr, const hxo_cluster* cl, const hxo_point* pt, int check,
                 hxo_result* res, const hxo_log* log, hxo_extra* ext) {
  memset(res, 0, sizeof(*res));
  if (ext) {
    memset(ext, 0, sizeof(*ext));
    for (int t = 0; t < HXO_MAX_TENANTS; ++t) ext->p95_us[t] = -1;
  }
  res->p95_us = -1;
  if (!validate(tr, cl) || pt->alpha_fp < 0 || pt->alpha_fp > FP_ONE || pt->beta_us2 < 0 ||
      pt->gamma_fp < 0 || pt->rho < 0 || pt->local_policy < 0 || pt->local_policy > 2 ||
      pt->dispatch_policy < 0 || pt->dispatch_policy > 1) {
    res->status = HXO_ERR_INVALID;
    return HXO_ERR_INVALID;
  }
  const int32_t nq = tr->n_queries, nc = tr->n_calls, N = cl->n_inst;
  sim_t s;
  memset(&s, 0, sizeof(s));
  s.tr = tr;
  s.cl = cl;
  s.pt = pt;
  size_t nc1 = (size_t)(nc > 0 ? nc : 1), nq1 = (size_t)(nq > 0 ? nq : 1);
  s.t_slo = (int64_t*)calloc(nq1, sizeof(int64_t));
  s.chains_left = (int32_t*)calloc(nq1, sizeof(int32_t));
  s.qid = (int32_t*)calloc(nc1, sizeof(int32_t));
  s.state = (uint8_t*)calloc(nc1, 1);
  s.inst = (int32_t*)calloc(nc1, sizeof(int32_t));
  s.enq = (int64_t*)calloc(nc1, sizeof(int64_t));
  s.budget = (int64_t*)calloc(nc1, sizeof(int64_t));
  s.remaining = (int64_t*)calloc(nc1, sizeof(int64_t));
  s.start = (int64_t*)calloc(nc1, sizeof(int64_t));
  s.end = (int64_t*)calloc(nc1, sizeof(int64_t));
  s.failed = (uint8_t*)calloc(nc1, 1);
  s.q = (int64_t*)calloc((size_t)N, sizeof(int64_t));
  s.waiting = (ivec*)calloc((size_t)N, sizeof(ivec));
  s.running = (ivec*)calloc((size_t)N, sizeof(ivec));
  int64_t* lat = (int64_t*)calloc(nq1, sizeof(int64_t));
  uint8_t* lat_tenant = (uint8_t*)calloc(nq1, 1);  /* tenant of lat[j] */
  int64_t* tlat = (int64_t*)calloc(nq1, sizeof(int64_t));
  int64_t* est_tmp = (int64_t*)calloc(nc1 * (size_t)cl->n_types, sizeof(int64_t));
  int64_t* svc_tmp = (int64_t*)calloc(nc1 * (size_t)cl->n_types, sizeof(int64_t));
  int64_t* tbar_tmp = (int64_t*)calloc(nc1, sizeof(int64_t));
  int64_t *ubuf = NULL, *ebuf = NULL;
  int32_t* rbuf = NULL;
  int32_t bufcap = 0;
  int status = HXO_OK;
  if (!s.t_slo || !s.chains_left || !s.qid || !s.state || !s.inst || !s.enq || !s.budget || !s.remaining || !s.start ||
      !s.end || !s.failed || !s.q || !s.waiting || !s.running || !lat || !lat_tenant || !tlat || !est_tmp ||
      !svc_tmp || !tbar_tmp) {
    status = HXO_ERR_OOM;
    goto done;
  }
  hxo_prep(tr, cl, est_tmp, svc_tmp, tbar_tmp, s.t_slo, s.cref);
  for (int32_t i = 0; i < nq; ++i)
    for (int32_t j = tr->call_base[i]; j < tr->call_base[i + 1]; ++j) s.qid[j] = i;

  int32_t next_q = 0, n_done = 0, slo_met = 0;
  int32_t t_slo_met[HXO_MAX_TENANTS] = {0, 0, 0, 0}, t_done[HXO_MAX_TENANTS] = {0, 0, 0, 0};
  int64_t makespan = 0, events = 0;
  for (;;) {
    /* next event: earliest completion by (end, instance, rid), else arrival */
    int best_m = -1;
    int32_t best_c = -1;
    for (int m = 0; m < N; ++m) {
      for (int32_t j = 0; j < s.running[m].n; ++j) {
        int32_t c = s.running[m].v[j];
        if (best_c < 0 || s.end[c] < s.end[best_c] ||
            (s.end[c] == s.end[best_c] && (m < best_m || (m == best_m && c < best_c)))) {
          best_m = m;
          best_c = c;
        }
      }
    }
    int has_arrival = next_q < nq;
    if (best_c < 0 && !has_arrival) break;
    int64_t now;
    if (best_c >= 0 && (!has_arrival || s.end[best_c] <= tr->arrival_us[next_q])) {
      /* completion of best_c on best_m */
      int32_t c = best_c, m = best_m;
      now = s.end[c];
      for (int32_t j = 0; j < s.running[m].n; ++j)
        if (s.running[m].v[j] == c) { ivec_remove_at(&s.running[m], j); break; }
      s.q[m] -= est_on(tr, cl, m, c);
      if (s.failed[c]) {
        /* the attempt timed out: the request goes out again, not to m */
        s.failed[c] = 0;
        s.reissued++;
        dispatch(&s, c, now, m);
        fill_slots(&s, now, &ubuf, &ebuf, &rbuf, &bufcap);
        if (s.bad) { status = s.bad; goto done; }
        if (check && !check_invariants(&s)) { status = HXO_ERR_INVARIANT; goto done; }
        continue;
      }
      s.state[c] = C_DONE;
      events++;
      int32_t i = s.qid[c];
      int32_t b = tr->call_base[i], e = tr->call_base[i + 1];
      int st = tr->stage[c];
      if (st == ST_S) {
        s.chains_left[i] = tr->k[i];
        for (int32_t j = b; j < e; ++j)
          if (tr->stage[j] == ST_G) dispatch(&s, j, now, -1);
      } else if (st == ST_G || st == ST_C) {
        int cand = tr->cand[c], r_next = (st == ST_G ? 0 : tr->retry[c]) + 1;
        int32_t nxt = -1;
        for (int32_t j = b; j < e; ++j)
          if (tr->stage[j] == ST_C && tr->cand[j] == cand && tr->retry[j] == r_next) nxt = j;
        if (nxt >= 0) {
          dispatch(&s, nxt, now, -1);
        } else if (--s.chains_left[i] == 0) {
          for (int32_t j = b; j < e; ++j)
            if (tr->stage[j] == ST_E) dispatch(&s, j, now, -1);
        }
      } else {
        int64_t l = now - tr->arrival_us[i];
        int ten = tr->tenant ? tr->tenant[i] : 0;
        lat_tenant[n_done] = (uint8_t)ten;
        lat[n_done++] = l;
        t_done[ten]++;
        if (l <= s.t_slo[i]) {
          slo_met++;
          t_slo_met[ten]++;
        }
        if (now > makespan) makespan = now;
        s.digest += query_term(i, now);
      }
    } else {
      now = tr->arrival_us[next_q];
      dispatch(&s, tr->call_base[next_q], now, -1);
      next_q++;
    }
    fill_slots(&s, now, &ubuf, &ebuf, &rbuf, &bufcap);
    if (s.bad) { status = s.bad; goto done; }
    if (check && !check_invariants(&s)) { status = HXO_ERR_INVARIANT; goto done; }
  }
  for (int m = 0; m < N; ++m)
    if (s.q[m] != 0) status = HXO_ERR_INVARIANT;
  for (int32_t c = 0; c < nc; ++c)
    if (s.state[c] != C_DONE) status = HXO_ERR_INVARIANT;
  if (n_done != nq) status = HXO_ERR_INVARIANT;

  res->n_done = n_done;
  res->slo_met = slo_met;
  if (ext) {
    for (int t = 0; t < HXO_MAX_TENANTS; ++t) {
      ext->slo_met[t] = t_slo_met[t];
      ext->n_done[t] = t_done[t];
    }
    ext->reissued = s.reissued;
    /* per tenant, the nearest-rank P95 of its own queries' latencies */
    for (int t = 0; t < HXO_MAX_TENANTS; ++t) {
      int32_t n = 0;
      for (int32_t j = 0; j < n_done; ++j)
        if (lat_tenant[j] == t) tlat[n++] = lat[j];
      if (status != HXO_OK) {
        ext->p95_us[t] = -1;
      } else if (n == 0) {
        ext->p95_us[t] = 0;
      } else {
        qsort(tlat, (size_t)n, sizeof(int64_t), cmp_i64);
        ext->p95_us[t] = tlat[(95 * (int64_t)n + 99) / 100 - 1];
      }
    }
  }
  res->makespan_us = makespan;
  res->events = events;
  res->digest = s.digest;
  if (status == HXO_OK) {
    if (nq > 0) {
      qsort(lat, (size_t)nq, sizeof(int64_t), cmp_i64);
      int64_t rank = (95 * (int64_t)nq + 99) / 100; /* ceil(0.95 n) */
      res->p95_us = lat[rank - 1];
    } else {
      res->p95_us = 0;
    }
  }
  if (log) {
    for (int32_t c = 0; c < nc; ++c) {
      if (log->inst) log->inst[c] = s.inst[c];
      if (log->enq) log->enq[c] = s.enq[c];
      if (log->budget) log->budget[c] = s.budget[c];
      if (log->start) log->start[c] = s.start[c];
      if (log->end) log->end[c] = s.end[c];
    }
  }
done:
  res->status = status;
  if (s.waiting)
    for (int m = 0; m < N; ++m) free(s.waiting[m].v);
  if (s.running)
    for (int m = 0; m < N; ++m) free(s.running[m].v);
  free(s.t_slo); free(s.chains_left); free(s.qid); free(s.state); free(s.inst); free(s.enq);
  free(s.budget); free(s.remaining); free(s.start); free(s.end); free(s.failed); free(s.q); free(s.waiting); free(s.running);
  free(lat); free(lat_tenant); free(tlat); free(est_tmp); free(svc_tmp); free(tbar_tmp); free(ubuf); free(ebuf); free(rbuf);
  return status;
}

/* ------------------------------------------------------------ best point */
typedef struct {
  int feasible;
  int64_t slo;
  int64_t p95;
  int32_t p;
  int valid;
} cand_t;

/* Lexicographic preference: valid, feasible, (more SLO hits if infeasible),
 * lower P95, lower point index. */
static int better(const cand_t* a, const cand_t* b, int objective) {
  if (!b->valid) return a->valid;
  if (!a->valid) return 0;
  if (objective == 1) {
    if (a->feasible != b->feasible) return a->feasible > b->feasible;
    if (!a->feasible && a->slo != b->slo) return a->slo > b->slo;
  }
  if (a->p95 != b->p95) return a->p95 < b->p95;
  return a->p < b->p;
}

int hxo_best(const hxo_result* res, int32_t n_traces, int32_t n_points, const int32_t* n_queries,
             int32_t objective, int32_t* global_point, int64_t* global_sum_p95,
             int32_t* per_trace_point) {
  if (n_traces < 0 || n_points < 1 || objective < 0 || objective > 1) return HXO_ERR_INVALID;
  for (int32_t t = 0; t < n_traces; ++t) {
    cand_t best = {0, 0, 0, -1, 0};
    for (int32_t p = 0; p < n_points; ++p) {
      const hxo_result* r = &res[(int64_t)t * n_points + p];
      cand_t c = {r->slo_met * 100LL >= 95LL * n_queries[t], r->slo_met, r->p95_us, p, r->status == 0};
      if (better(&c, &best, objective)) best = c;
    }
    if (per_trace_point) per_trace_point[t] = best.valid ? best.p : -1;
  }
  cand_t gbest = {0, 0, 0, -1, 0};
  int64_t nsum = 0;
  for (int32_t t = 0; t < n_traces; ++t) nsum += n_queries[t];
  for (int32_t p = 0; p < n_points; ++p) {
    cand_t c = {0, 0, 0, p, 1};
    for (int32_t t = 0; t < n_traces; ++t) {
      const hxo_result* r = &res[(int64_t)t * n_points + p];
      if (r->status != 0) c.valid = 0;
      c.slo += r->slo_met;
      c.p95 += r->p95_us;
    }
    c.feasible = c.slo * 100 >= 95 * nsum;
    if (better(&c, &gbest, objective)) gbest = c;
  }
  *global_point = gbest.valid ? gbest.p : -1;
  *global_sum_p95 = gbest.valid ? gbest.p95 : -1;
  return HXO_OK;
}
