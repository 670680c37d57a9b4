// hx_kernels.cu -- the three kernels of the batched HexGen-Flow scheduler
// simulation (arXiv 2505.05286, Sec. 4.1-4.3) for sm_103a.
//
// Integer-only: every time is int64 microseconds, every score and key int64
// fixed point; every division is the compiler's truncating `/`.  Nothing here
// is a dense contraction, so there are no tensor-core paths; the simulation
// kernel is bound by the SM issue rate, the preparation kernel by HBM.
#include <climits>

#include "hx_device.cuh"

namespace hx {

// ------------------------------------------------------------------ helpers
__device__ __forceinline__ int64_t ceil_div_pos(int64_t a, int64_t b) { return (a + b - 1) / b; }

constexpr uint64_t kDigestMul = 0x9E3779B97F4A7C15ull;  // golden-ratio increment of splitmix64
constexpr uint64_t kMixA = 0xBF58476D1CE4E5B9ull;       // splitmix64 output-function multipliers
constexpr uint64_t kMixB = 0x94D049BB133111EBull;       // (Steele, Lea & Flood, OOPSLA 2014)

// Digest terms: the splitmix64 output function (two xor-shift-multiply rounds
// and a final xor-shift) of (time * phi) xor (id << 8 | tag); every step is a
// bijection, so a change of any one call's instance or start (or any query's
// end) changes the sum.
__device__ __forceinline__ uint64_t digest_term(uint64_t t, uint64_t idtag) {
  uint64_t z = (t * kDigestMul) ^ idtag;
  z = (z ^ (z >> 30)) * kMixA;
  z = (z ^ (z >> 27)) * kMixB;
  return z ^ (z >> 31);
}

// Id tags: a call's start is (rid << 8 | instance), a query's end (qid << 8 | 0xFF).
__device__ __forceinline__ uint32_t call_tag(int32_t rid, int inst) { return ((uint32_t)rid << 8) | (uint32_t)inst; }
__device__ __forceinline__ uint32_t query_tag(int32_t qid) { return ((uint32_t)qid << 8) | 0xFFu; }

__device__ __forceinline__ uint64_t warp_min_u64(uint64_t v) {
  uint32_t hi = (uint32_t)(v >> 32), lo = (uint32_t)v;
  uint32_t mh = __reduce_min_sync(kFull, hi);
  uint32_t ml = __reduce_min_sync(kFull, hi == mh ? lo : 0xffffffffu);
  return ((uint64_t)mh << 32) | ml;
}

// Highest signed score, ties to the lowest index; every lane gets the index.
__device__ __forceinline__ int warp_argmax_s64(int64_t s, int idx) {
  uint64_t u = (uint64_t)s ^ 0x8000000000000000ull;
  uint32_t hi = (uint32_t)(u >> 32), lo = (uint32_t)u;
  uint32_t mh = __reduce_max_sync(kFull, hi);
  bool c1 = hi == mh;
  uint32_t ml = __reduce_max_sync(kFull, c1 ? lo : 0u);
  bool c2 = c1 && lo == ml;
  return (int)__reduce_min_sync(kFull, c2 ? (uint32_t)idx : 0xffffffffu);
}

// floor(n / d) for 0 <= n < 2^63 and 1 <= d < 2^54.  Trial-quotient method
// (Knuth, TAOCP vol. 2, 4.3.1): a quotient estimate from a single-precision
// reciprocal, refined once on the exact int64 remainder when it is 2^21 or
// more, then corrected by at most one step each way.  Operands reach float
// through two 32-bit halves.  The estimate's relative error is below
// 3.5 * 2^-23 (two conversions, the approximate reciprocal, one product), so
// below 2^21 it is within one of n/d, and below 2^30 the refined one is.
// Quotients of 2^30 or more (and d = 1) take the exact integer paths.
__device__ __forceinline__ float u64_to_float(uint64_t x) {
  return __fmaf_rn((float)(uint32_t)(x >> 32), 4294967296.0f, (float)(uint32_t)x);
}

__device__ __forceinline__ float s64_to_float(int64_t x) {
  return x < 0 ? -u64_to_float((uint64_t)(-x)) : u64_to_float((uint64_t)x);
}

// nf = u64_to_float(n), given by a caller that divides one n many times.
__device__ __forceinline__ uint64_t udiv_trial_f(uint64_t n, float nf, uint64_t d) {
  if (d == 1) return n;
  float rd;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(rd) : "f"(u64_to_float(d)));
  const float qf = nf * rd;
  if (qf >= 1073741824.0f) return n / d;
  uint64_t q = (uint32_t)qf;
  int64_t r = (int64_t)(n - q * d);
  if (qf >= 2097152.0f) {
    q += (int64_t)(int32_t)(s64_to_float(r) * rd);
    r = (int64_t)(n - q * d);
  }
  if (r < 0) {
    q--;
    r += (int64_t)d;
  } else if (r >= (int64_t)d) {
    q++;
    r -= (int64_t)d;
  }
  return q;
}

__device__ __forceinline__ uint64_t udiv_trial(uint64_t n, uint64_t d) { return udiv_trial_f(n, u64_to_float(n), d); }

// Workload-balanced reward term of Eq. (score): beta / max(t_queue, 1), capped.
__device__ __forceinline__ int64_t reward_of(int64_t beta, int64_t q) {
  int64_t r = beta / (q > 1 ? q : 1);
  return r < kRewardCap ? r : kRewardCap;
}

// (num * tb) / d truncated toward zero, for |num| < 2^41 and 1 <= tb <= d < 2^33:
// splitting num = q1 * d + r1 keeps every product below 2^63.
__device__ __forceinline__ int64_t scaled_div(int64_t num, int64_t tb, int64_t d) {
  if (num < (int64_t(1) << 32) && num > -(int64_t(1) << 32)) return (num * tb) / d;
  int64_t q1 = num / d, r1 = num % d;
  return q1 * tb + (r1 * tb) / d;
}

__device__ __forceinline__ int64_t cost_on_type(const ClusterK& c, int t, int64_t prompt, int64_t out) {
  return ceil_div_pos(prompt * kUsPerS, c.prefill[t]) + out * (int64_t)c.decode[t];
}

// ------------------------------------------------------------- prep kernel
// One thread per query: Eq. (comp) per call and type, tbar, chain successor
// links and the deadline arrival + slo_mult * L0 (L0 = S + slowest
// candidate chain + E on the reference type).
__global__ void __launch_bounds__(256) hx_prep_kernel(PrepArgs a, ClusterK c) {
  int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (g == 0) *a.work_counter = 0ull;
  // a run over a subset: the simulations outside it report HX_SKIPPED
  for (int64_t i = g; i < a.n_skip; i += (int64_t)gridDim.x * blockDim.x) {
    hx_result r;
    r.p95_us = -1;
    r.makespan_us = 0;
    r.events = 0;
    r.digest = 0;
    r.slo_met = 0;
    r.n_done = 0;
    r.status = HX_SKIPPED;
    r.cycles_k = 0;
    a.skip_results[i] = r;
    if (a.skip_extras) {
      hx_extra x;
      for (int t = 0; t < HX_MAX_TENANTS; ++t) {
        x.slo_met[t] = 0;
        x.n_done[t] = 0;
        x.p95_us[t] = -1;
      }
      x.reissued = 0;
      x.pad = 0;
      a.skip_extras[i] = x;
    }
  }
  if (g >= a.n_queries) return;
  int lo = 0, hi = a.n_traces;  // trace of query g: q_off[t] <= g < q_off[t+1]
  while (hi - lo > 1) {
    int mid = (lo + hi) >> 1;
    if (a.q_off[mid] <= g) lo = mid; else hi = mid;
  }
  const int t = lo;
  const int64_t cbase = a.c_off[t];
  const int32_t qid = (int32_t)(g - a.q_off[t]);
  const int64_t b = a.qcall[g], e = a.qcall[g + 1];
  const int k = a.kq[g];
  const int64_t arr = a.arrival[g];
  const int T = c.n_types;

  // pass 1: first correction of every chain and the exclusive latency L0
  int32_t first_corr[HX_MAX_K];
  int64_t chain[HX_MAX_K];
#pragma unroll
  for (int i = 0; i < HX_MAX_K; ++i) { first_corr[i] = -1; chain[i] = 0; }
  int64_t l_s = 0, l_e = 0;
  for (int64_t j = b; j < e; ++j) {
    const int st = a.stage[j];
    const int64_t s_ref = cost_on_type(c, c.ref_type, a.prompt[j], a.out[j]);
    if (st == HX_STAGE_S) {
      l_s += s_ref;
    } else if (st == HX_STAGE_E) {
      l_e += s_ref;
    } else {
      const int cd = a.cand[j];
      chain[cd] += s_ref;
      if (st == HX_STAGE_C && a.retry[j] == 1) first_corr[cd] = (int32_t)(j - cbase);
    }
  }
  int64_t longest = 0;
  for (int i = 0; i < k; ++i) longest = chain[i] > longest ? chain[i] : longest;
  const int tenant = a.tenant ? a.tenant[g] : 0;
  const int64_t mult = c.n_tenants > 1 ? c.tenant_mult[tenant] : c.slo_mult_fp;
  const int64_t t_slo = (mult * (l_s + longest + l_e)) / kScale;
  const int64_t deadline = arr + t_slo;
  const int32_t e_rid = (int32_t)(e - 1 - cbase);

  // pass 2: one 64-byte record per call
  for (int64_t j = b; j < e; ++j) {
    const int64_t p = a.prompt[j], o = a.out[j], oe = a.out_est[j];
    const int st = a.stage[j];
    CallRec r;
    int64_t sum = 0;
#pragma unroll
    for (int ty = 0; ty < HX_MAX_TYPES; ++ty) {
      if (ty < T) {
        const int64_t pre = ceil_div_pos(p * kUsPerS, c.prefill[ty]);
        const int64_t es = pre + oe * (int64_t)c.decode[ty];
        r.ev[ty] = make_int2((int32_t)es, (int32_t)(pre + o * (int64_t)c.decode[ty]));
        sum += es * c.cnt[ty];
      } else {
        r.ev[ty] = make_int2(0, 0);
      }
    }
    r.tbar = (int32_t)(sum / c.n_inst);
    r.deadline = deadline;
    r.arrival = arr;
    r.qid = qid;
    r.stage = (uint8_t)st;
    r.k = (uint8_t)k;
    if (st == HX_STAGE_S) {
      r.u = 0;
      r.fcode = 0;
      r.next = -1;
    } else if (st == HX_STAGE_E) {
      r.u = (uint8_t)tenant;
      r.fcode = kFRows - 1;
      r.next = -1;
    } else {
      const int cd = a.cand[j];
      int32_t nx;
      if (st == HX_STAGE_G) {
        r.u = 0;
        nx = first_corr[cd];
      } else {
        r.u = a.retry[j];
        nx = (j + 1 < e - 1 && a.stage[j + 1] == HX_STAGE_C && a.cand[j + 1] == cd) ? (int32_t)(j + 1 - cbase) : -1;
      }
      r.next = nx >= 0 ? nx : ~e_rid;
      r.fcode = (uint8_t)(1 + r.u);
    }
    const int4* src = reinterpret_cast<const int4*>(&r);
    int4* dst = reinterpret_cast<int4*>(a.rec + j);
    dst[0] = src[0];
    dst[1] = src[1];
    dst[2] = src[2];
    dst[3] = src[3];
  }
}

// -------------------------------------------------------- simulation kernel
namespace {

// The digest is a sum of terms, so they are hashed 16 at a time: every lane
// calls with the same (t, tag); lane 0 appends it, and a full batch is hashed
// one term per lane and summed into W->digest.
__device__ __noinline__ void digest_flush(WarpShared* W, int n, int lane) {
  __syncwarp();
  const longlong2 e = W->dterm[lane < n ? lane : 0];
  uint64_t y = lane < n ? digest_term((uint64_t)e.x, (uint64_t)e.y) : 0ull;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) y += __shfl_xor_sync(kFull, y, o);
  if (lane == 0) W->digest += y;
  __syncwarp();
}

__device__ __forceinline__ void digest_push(WarpShared* W, int& dn, int64_t t, uint32_t tag, int lane) {
  W->dterm[dn] = make_longlong2(t, (long long)tag);  // every lane writes the same pair
  if (++dn == 16) {
    digest_flush(W, 16, lane);
    dn = 0;
  }
}

__device__ __forceinline__ bool ent_better(long long ka, int ra, long long kb, int rb) {
  return ka > kb || (ka == kb && ra < rb);
}

// Local queues are 32-ary max-heaps on (key desc, rid asc) in the warp's
// arena: node i has children 32 i + 1 .. 32 i + 32, so 40k waiting requests
// sit four levels deep.  Push sifts up on one lane (new requests rarely
// climb); pop and replace sift down with the whole warp, one lane per child.
__device__ __forceinline__ void heap_push(HeapEnt* h, int n, long long key, int rid, int svc) {
  int i = n;
  while (i > 0) {
    const int par = (i - 1) >> 5;
    const HeapEnt pe = h[par];
    if (!ent_better(key, rid, pe.key, pe.rid)) break;
    h[i] = pe;
    i = par;
  }
  HeapEnt e;
  e.key = key;
  e.rid = rid;
  e.svc = svc;
  h[i] = e;
}

// All lanes call with the same arguments.  The top entry leaves the heap and
// `sink` takes its place, sinking to its level; the heap then holds m
// entries (m = n - 1 and sink = the last entry: a pop; m = n and sink = a new
// entry: a replace).  Every lane gets the old top.
__device__ __forceinline__ HeapEnt heap_sift_warp(HeapEnt* h, int m, HeapEnt sink, int lane) {
  const HeapEnt top = h[0];
  int i = 0;
  for (;;) {
    const int first = 32 * i + 1;
    if (first >= m) break;
    const int child = first + lane;
    long long ck = LLONG_MIN;
    int cr = INT_MAX, cs = 0;
    if (child < m) {
      const HeapEnt e = h[child];
      ck = e.key;
      cr = e.rid;
      cs = e.svc;
    }
    // warp argmax of (key desc, rid asc): the rids decide only among equal keys
    const uint64_t uk = (uint64_t)ck ^ 0x8000000000000000ull;
    const uint32_t hi = (uint32_t)(uk >> 32), lo = (uint32_t)uk;
    const uint32_t mh = __reduce_max_sync(kFull, hi);
    const bool c1 = hi == mh;
    const uint32_t ml = __reduce_max_sync(kFull, c1 ? lo : 0u);
    unsigned best = __ballot_sync(kFull, c1 && lo == ml);
    if (best & (best - 1)) {
      const bool tie = (best >> lane) & 1u;
      const uint32_t mr = __reduce_min_sync(kFull, tie ? (uint32_t)cr : 0xffffffffu);
      best = __ballot_sync(kFull, tie && (uint32_t)cr == mr);
    }
    const int b = __ffs(best) - 1;
    // the best child moves up unless the sinking entry goes before it
    if (!__shfl_sync(kFull, (int)ent_better(ck, cr, sink.key, sink.rid), b)) break;
    if (lane == b) {
      HeapEnt e;
      e.key = ck;
      e.rid = cr;
      e.svc = cs;
      h[i] = e;
    }
    i = first + b;
  }
  if (lane == 0 && m > 0) h[i] = sink;
  __syncwarp();
  return top;
}

// Min-heap of the K largest latencies seen so far, 32-ary like the local
// queues; its root is the K-th largest latency, i.e. the nearest-rank P95
// when K = n - ceil(0.95 n) + 1.  All lanes call with the same v: lane 0
// writes the heap, every lane writes the same size (*size) and root (*root)
// copies in shared memory.
__device__ __noinline__ void topk_insert_warp(int64_t* h, int32_t* size, int kcap, int64_t* root_out, int64_t v,
                                              int lane) {
  const int n = *size;
  if (n < kcap) {
    // filling: sift up on lane 0 (few levels)
    if (lane == 0) {
      int i = n;
      while (i > 0) {
        const int par = (i - 1) >> 5;
        const int64_t pv = h[par];
        if (pv <= v) break;
        h[i] = pv;
        i = par;
      }
      h[i] = v;
    }
    __syncwarp();
    *size = n + 1;
    if (n + 1 == kcap) *root_out = h[0];
  } else if (v > *root_out) {
    // v replaces the root and sinks; one lane per child (latencies are >= 0)
    int i = 0;
    int64_t root = v;
    for (;;) {
      const int first = 32 * i + 1;
      if (first >= n) break;
      const int ch = first + lane;
      const uint64_t cv = ch < n ? (uint64_t)h[ch] : ~0ull;
      const uint64_t mn = warp_min_u64(cv);
      if (mn >= (uint64_t)v) break;
      const int b = __ffs(__ballot_sync(kFull, cv == mn)) - 1;
      if (i == 0) root = (int64_t)mn;
      if (lane == 0) h[i] = (int64_t)mn;
      i = first + b;
    }
    if (lane == 0) h[i] = v;
    __syncwarp();
    *root_out = root;
  }
}

// Queue this event's dispatches to instance m (pending entries on the lanes of
// mask pm) in m's heap, re-homing the heap in the arena when it is full.
// All lanes call.  Returns HX_OK or HX_ERR_CAPACITY.
__device__ __noinline__ int64_t budget_wide(int64_t num, int64_t tb, int64_t d) { return scaled_div(num, tb, d); }

// t_slo of Eq. (budget): (deadline - now) * tbar / (tbar + F), truncated
// toward zero; |num| < 2^34 keeps |num| * tbar below 2^63.
__device__ __forceinline__ int64_t slo_budget(int64_t num, int64_t tb, int64_t dd) {
  if (num > -(int64_t(1) << 34) && num < (int64_t(1) << 34)) {
    const uint64_t res = udiv_trial((uint64_t)(num < 0 ? -num : num) * (uint64_t)tb, (uint64_t)dd);
    return num < 0 ? -(int64_t)res : (int64_t)res;
  }
  return budget_wide(num, tb, dd);
}

// Local-queue key, higher first, of pending entry j: Eq. (priority) with
// the budget at send time (now) and the common now dropped; FCFS: earliest
// enqueue; LLF: least deadline - now - remaining work, again with the common
// now dropped.
__device__ __forceinline__ long long pending_key(const WarpShared* W, const CallRec* rec, int64_t now, int lpol,
                                                 int j) {
  const CallRec* r = rec + W->prs[j].x;
  const int64_t dl = r->deadline;
  const int4 tail = *reinterpret_cast<const int4*>(&r->tbar);
  const int64_t tb = tail.x;
  const int64_t dd = tb + W->frest[(uint32_t)tail.w >> 24];
  return lpol == HX_LOCAL_PQ     ? (long long)(kScale * ((int64_t)W->pest[j] - slo_budget(dl - now, tb, dd)) - W->G * now)
         : lpol == HX_LOCAL_FCFS ? (long long)(-now)
                                 : (long long)(dd - dl);
}

// The instance's new requests (pending entries, bits of pm) join its local
// queue, their keys formed one per lane.
__device__ __forceinline__ int push_pending(WarpShared* W, const CallRec* rec, int64_t now, int lpol,
                                        int64_t arena_per_warp, int m, unsigned pm, int lane) {
  const long long key = ((pm >> lane) & 1u) ? pending_key(W, rec, now, lpol, lane) : 0;
  HeapEnt* const arena = W->arena;
  while (pm) {
    const int j = __ffs(pm) - 1;
    pm &= pm - 1;
    const long long kj = __shfl_sync(kFull, key, j);
    const int2 rs = W->prs[j];
    const int rid = rs.x, svc = rs.y;
    const int size = W->hsize[m], hcl = W->hcl[m], off = W->hoff[m], bump = W->bump;
    const int cap = hcl ? 8 << hcl : 0;
    __syncwarp();
    int hoff = off;
    if (size == cap) {
      const int ncap = cap ? 2 * cap : 16;
      if ((int64_t)bump + ncap > arena_per_warp) return HX_ERR_CAPACITY;
      hoff = bump;
      for (int i = lane; i < size; i += 32) arena[hoff + i] = arena[off + i];
      __syncwarp();
      if (lane == 0) {
        W->bump = bump + ncap;
        W->hoff[m] = hoff;
        W->hcl[m] = (uint8_t)(hcl + 1);
      }
    }
    if (lane == 0) {
      heap_push(arena + hoff, size, kj, rid, svc);
      W->hsize[m] = size + 1;
    }
    __syncwarp();
  }
  return HX_OK;
}

// One new request (the single bit of pm) meets an instance with one free slot
// and a non-empty local queue: the more urgent of it and the queue's top
// starts and the other waits, i.e. a push and a pop in one sift (the new
// request replaces the top).  Returns the started (request id, service time).
__device__ __forceinline__ int2 push_pop(WarpShared* W, const CallRec* rec, int64_t now, int lpol, int m, unsigned pm,
                                     int lane) {
  const int j = __ffs(pm) - 1;
  const long long key = pending_key(W, rec, now, lpol, j);  // the same on every lane
  const int2 rs = W->prs[j];
  HeapEnt* const h = W->arena + W->hoff[m];
  const HeapEnt top = h[0];
  if (ent_better(key, rs.x, top.key, top.rid)) return rs;
  HeapEnt e;
  e.key = key;
  e.rid = rs.x;
  e.svc = rs.y;
  heap_sift_warp(h, W->hsize[m], e, lane);
  return make_int2(top.rid, top.svc);
}

// All lanes: a query's evaluation call finished at `now` (Sec. 4.3's metrics).
__device__ __forceinline__ void finish_query(WarpShared* W, int& dn, int32_t qid, int64_t now, int64_t arrival,
                                            int64_t deadline, int lane) {
  {
    // every lane reads the counters, then every lane writes the same new values
    const int32_t slo = W->slo_met + (now <= deadline ? 1 : 0), nd = W->n_done + 1;
    __syncwarp();
    W->slo_met = slo;
    W->n_done = nd;
    W->makespan = now;
  }
  digest_push(W, dn, now, query_tag(qid), lane);
  // most latencies of a full heap fall below its root and change nothing
  const int64_t v = now - arrival;
  if (W->tk < W->kcap || v > W->tkmin) topk_insert_warp(W->topk, &W->tk, W->kcap, &W->tkmin, v, lane);
}

__device__ __noinline__ void log_dispatch(const SimArgs& a, int recj, int rid, int m, int64_t now, int64_t budget) {
  const int64_t o = (int64_t)recj * a.rec_stride + rid;
  a.rec_inst[o] = m;
  a.rec_enq[o] = now;
  a.rec_budget[o] = budget;
}


}  // namespace

// Resident blocks per SM the register allocation aims for (4 warps each).
#ifndef HX_SIM_MIN_BLOCKS
#define HX_SIM_MIN_BLOCKS 8
#endif

// Bounds-checked build (-DHX_CHECKED): before every shared- or global-memory
// access whose index the simulation forms from its own state (instance,
// request id, query id, slot count, heap offset and size, top-K size), the
// index is range-checked; a failed check sets the simulation's status to
// HX_ERR_BOUNDS and leaves the loop it is in instead of making the access,
// and the simulation stops after that event.  Every checked value is the
// same on all lanes, so the exit is warp-uniform.  In the normal build the
// checks compile to nothing.
#ifdef HX_CHECKED
#define HX_BOUND(cond)          \
  if (!(cond)) {                \
    status = HX_ERR_BOUNDS;     \
    break;                      \
  }
#define HX_STOP_IF_FAILED() \
  if (status != HX_OK) break;
#else
#define HX_BOUND(cond)
#define HX_STOP_IF_FAILED()
#endif

template <bool kGeneric>
__device__ __forceinline__ void sim_body(const SimArgs& a, const ClusterK& c) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  WarpShared* const W = reinterpret_cast<WarpShared*>(smem_raw + warp * c.smem_per_warp);
  if (lane == 0) {
    // this warp's slices of the scratch arrays (kept in shared memory to spare registers)
    const int64_t gw = (int64_t)blockIdx.x * kWarpsPerBlock + warp;
    W->arena = a.arena + gw * a.arena_per_warp;
    W->chains = a.chains + gw * a.chains_per_warp;
    W->topk = a.topk + gw * a.topk_per_warp;
  }
  const int N = c.n_inst;
  const int m0 = lane, m1 = lane + 32;
  const bool valid0 = m0 < N, valid1 = m1 < N;
  const int ty0 = valid0 ? c.inst_type[m0] : 0;
  const int ty1 = valid1 ? c.inst_type[m1] : 0;

  for (;;) {
    unsigned long long work = 0;
    if (lane == 0) work = atomicAdd(a.work_counter, 1ull);
    const int64_t w = (int64_t)__shfl_sync(kFull, work, 0);
    if (w >= a.n_work) break;
    // trace-major, so that concurrent simulations share a trace in L2; within a
    // trace the highest point index (highest alpha, the longest queues) first
    // (a subset comes sorted in the same order)
    int t, p;
    if (a.subset) {
      const int64_t s = a.subset[w];
      t = (int)(s / a.n_points);
      p = (int)(s - (int64_t)t * a.n_points);
    } else {
      t = (int)(w / a.n_points);
      p = a.n_points - 1 - (int)(w - (int64_t)t * a.n_points);
    }
    const int64_t sim = (int64_t)t * a.n_points + p;
    const long long clk0 = clock64();
    const int64_t qb = a.q_off[t];
    const int32_t nq = (int32_t)(a.q_off[t + 1] - qb);
    const int64_t cb = a.c_off[t];
    const int32_t nc = (int32_t)(a.c_off[t + 1] - cb);
    const CallRec* const rec = a.rec + cb;
    if (lane == 0) {
      W->qb = qb;
      W->cb = cb;
      W->nq = nq;
      W->nc = nc;
      W->sim = sim;
      W->trace = t;
      W->clk0 = clk0;
    }

    // per-instance state that every lane reads later: written before the
    // barrier below
    for (int m = lane; m < 64; m += 32) {
      W->q[m] = 0;
      W->hoff[m] = 0;
      W->hcl[m] = 0;
      W->hsize[m] = 0;
      W->cnt[m] = 0;
    }
    for (int j = lane; j < c.total_slots; j += 32) W->slot[j] = kKeyInf;
    if (lane < kFRows) {
      // rest of the request's own path after it (the budget denominator minus
      // its own mean cost): stage reference costs, i.e. means over instances of
      // Eq. (comp) at the stage's reference tokens, for G, min(rho, R - u)
      // corrections and E
      int64_t cref[4];
      for (int s = 0; s < 4; ++s) {
        int64_t sum = 0;
        for (int ty = 0; ty < c.n_types; ++ty) sum += cost_on_type(c, ty, c.ref_prompt[s], c.ref_out[s]) * c.cnt[ty];
        cref[s] = sum / N;
      }
      const int64_t rho = a.rho[p], rmax = c.rmax;
      int64_t f;
      if (lane == 0) {
        f = cref[HX_STAGE_G] + (rho < rmax ? rho : rmax) * cref[HX_STAGE_C] + cref[HX_STAGE_E];
      } else if (lane == kFRows - 1) {
        f = 0;
      } else {
        const int64_t left = rmax - (lane - 1);
        f = (rho < left ? rho : left) * cref[HX_STAGE_C] + cref[HX_STAGE_E];
      }
      W->frest[lane] = f;
    }
    if (lane == 0) {
      const int64_t A = a.alpha[p];
      W->A = (int32_t)A;
      W->one_minus_a = (int32_t)(kScale - A);
      // rewards carry no weight at alpha = 1 and are unused by round robin
      W->rewards = (A != kScale && !(kGeneric && a.dpol[p] == HX_DISPATCH_RR)) ? 1 : 0;
      W->G = a.gamma[p];
      W->beta = a.beta[p];
      W->betaf = u64_to_float((uint64_t)a.beta[p]);
      W->lpol = a.lpol[p];
      W->dpol = a.dpol[p];
      W->recj = a.rec_map ? a.rec_map[sim] : -1;
      W->kcap = nq - (95 * nq + 99) / 100 + 1;
      W->rr = 0;
      W->bump = 0;
      W->digest = 0;
      W->makespan = 0;
      W->n_done = 0;
      W->slo_met = 0;
      W->events = 0;
      W->tk = 0;
      W->tkmin = 0;
      for (int t = 0; t < HX_MAX_TENANTS; ++t) {
        W->tslo[t] = 0;
        W->tdone[t] = 0;
        W->ttk[t] = 0;
        W->ttkmin[t] = 0;
      }
      W->reissued = 0;
      W->excl = -1;
    }
    __syncwarp();

    // this lane's instances m0 = lane and m1 = lane + 32: t_queue in W->q[m]
    // and the next completion's event key and request id in W->ekey[m] and
    // W->erid[m] (every change stored alike by every lane; the owner reads
    // the keys at the loop top), the cached (1 - alpha) * reward in
    // W->orew[m] (the owner lane alone) and its staleness in dirty0 / dirty1;
    // shared memory rather than registers leaves the allocator room.
    // Instances past N start with a reward far below any real score
    // (|alpha * est| < 2^52), so the argmax needs no validity test.
    const int32_t oma32 = W->one_minus_a;
    // rewards carry weight (alpha < 1 with workload-balanced dispatch): kept in
    // a predicate register rather than re-read at every queue-cost change
    const bool rewards_on = W->rewards != 0;
    const int64_t orew_idle = (int64_t)oma32 * reward_of(W->beta, 0);
    W->orew[m0] = valid0 ? orew_idle : -(int64_t(1) << 62);
    W->orew[m1] = valid1 ? orew_idle : -(int64_t(1) << 62);
    bool dirty0 = false, dirty1 = false;
    W->ekey[m0] = kKeyInf;
    W->ekey[m1] = kKeyInf;
    // this event's dispatches, entry j on lane j
    int pend_m = -1;

    W->qa = 0;
    W->akey = nq > 0 ? (((uint64_t)a.arrival[qb] << 7) | kArrivalTag) : kKeyInf;
    int64_t now = 0;
    int32_t status = HX_OK, npend = 0;
    uint64_t touched = 0;
    // event bound; re-issued attempts add events while fault windows last
    const bool faults = kGeneric && c.n_faults > 0;
    int32_t steps_left = nc + nq + 8 + (faults ? 16 * nc + 4096 : 0);
#ifdef HX_CHECKED
    // the warp's scratch slices must hold this trace's chain counters and top-K
    if (!(nq <= a.chains_per_warp && W->kcap <= a.topk_per_warp && (a.tenant_kcap == nullptr ||
          (int64_t)(HX_MAX_TENANTS + 1) * a.tenant_topk_off[0] <= a.topk_per_warp)))
      status = HX_ERR_BOUNDS;
#endif

    // Request rid starts on instance m now and runs until now + svc: its key
    // joins the cn sorted keys of m's running calls at sl.
    int dn = 0;  // digest terms waiting in W->dterm
    auto start_call = [&](uint64_t* sl, int m, int cn, int rid, int svc) {
      int64_t run = svc;
      bool fail = false;
      if (faults) {
        // the first fault window of m that covers now, and the timeout (Sec. 3.3)
        bool in_window = false, down = false;
        for (int f = 0; f < c.n_faults; ++f) {
          const FaultK& F = c.faults[f];
          if (F.inst == m && now >= F.t0 && now < F.t1) {
            in_window = true;
            if (F.slow == 0) down = true;
            else run = (run * F.slow + kScale - 1) / kScale;
            break;
          }
        }
        if (in_window && c.timeout_mult_fp > 0) {
          const int64_t timeout = ((int64_t)rec[rid].ev[c.inst_type[m]].x * c.timeout_mult_fp) / kScale;
          if (down || run > timeout) {
            fail = true;
            run = timeout;
          }
        }
      }
      const uint64_t nk = ((uint64_t)(now + run) << 24) | (uint64_t)(uint32_t)rid;
      const uint64_t cur = lane < cn ? sl[lane] : kKeyInf;
      uint8_t* const fl = faults ? reinterpret_cast<uint8_t*>(W->slot + c.total_slots) + (sl - W->slot) : nullptr;
      const uint8_t fcur = (faults && lane < cn) ? fl[lane] : 0;
      const int pos = __popc(__ballot_sync(kFull, cur < nk));
      if (lane >= pos && lane < cn) sl[lane + 1] = cur;
      if (lane == pos) sl[pos] = nk;
      if (faults) {
        if (lane >= pos && lane < cn) fl[lane + 1] = fcur;
        if (lane == pos) fl[pos] = fail ? 1 : 0;
      }
      digest_push(W, dn, now, call_tag(rid, m), lane);
      if (kGeneric && lane == 0) {
        const int recj = W->recj;
        if (recj >= 0) {
          a.rec_start[(int64_t)recj * a.rec_stride + rid] = now;
          a.rec_end[(int64_t)recj * a.rec_stride + rid] = now + run;
        }
      }
      __syncwarp();
    };

    auto set_key = [&](int m, uint64_t nk) {
      // an empty instance (nk all ones) maps to a key at or above kNoEvent
      W->ekey[m] = ((nk >> 24) << 7) | (uint64_t)m;  // every lane stores the same key
      W->erid[m] = (int32_t)(nk & 0xffffffull);
    };

    for (;;) {
      HX_STOP_IF_FAILED()
      const uint64_t k0 = W->ekey[m0], k1 = W->ekey[m1];
      const uint64_t ck = warp_min_u64(k0 < k1 ? k0 : k1);
      const uint64_t akey = W->akey;
      if (ck >= kNoEvent && akey == kKeyInf) break;
      if (--steps_left < 0) {
        status = HX_ERR_STEP_LIMIT;
        break;
      }
      touched = 0;
      npend = 0;
      // requests released by this event: rel_first .. rel_first + rel_count - 1
      int32_t rel_first = 0, rel_count = 0;
      if (ck < akey) {
        // completion on instance m
        const int m = (int)(ck & 127ull);
        now = (int64_t)(ck >> 7);
        HX_BOUND(m < N)
        uint64_t* const sl = W->slot + c.slot_base[m];
        const int cn = W->cnt[m];
        HX_BOUND(cn >= 1 && cn <= c.inst_slots[m] && c.slot_base[m] + cn <= c.total_slots)
        // the finishing call heads m's sorted slots; its id is kept beside
        // m's event key, so that its record load need not wait for the slot
        const int32_t rid = W->erid[m];
        HX_BOUND(rid < nc)
        // the finished call's record: issued now, used after the slot shift
        const CallRec* r = rec + rid;
        const int4 tail = *reinterpret_cast<const int4*>(&r->tbar);
        const int64_t est_m = r->ev[c.inst_type[m]].x;
        const int hs_m = W->hsize[m];
        // remove it: the remaining keys move down one slot
        const uint64_t nxt = lane + 1 < cn ? sl[lane + 1] : kKeyInf;
        const uint64_t head = cn > 1 ? sl[1] : kKeyInf;
        uint8_t* const fl = faults ? reinterpret_cast<uint8_t*>(W->slot + c.total_slots) + (sl - W->slot) : nullptr;
        const bool failed = faults && fl[0] != 0;
        const uint8_t fnxt = (faults && lane + 1 < cn) ? fl[lane + 1] : 0;
        __syncwarp();
        if (lane < cn) sl[lane] = nxt;
        if (faults && lane < cn) fl[lane] = fnxt;
        W->cnt[m] = cn - 1;  // every lane writes the same count
        set_key(m, head);
        {
          W->q[m] = W->q[m] - est_m;  // every lane stores the same value
          const bool stale = rewards_on;
          dirty0 = lane == m ? stale : dirty0;
          dirty1 = lane + 32 == m ? stale : dirty1;
        }
        // the freed slot needs a batch boundary only if requests wait for it
        if (hs_m > 0) touched |= 1ull << m;
        const int stg = tail.w & 0xff;
        const int32_t qid = tail.z;
        HX_BOUND(qid >= 0 && qid < nq)
        if (faults && failed) {
          // the attempt timed out: the request goes out again, avoiding m
          if (lane == 0) W->reissued++;
          W->excl = c.n_inst > 1 ? m : -1;
          rel_first = rid;
          rel_count = 1;
        } else if (stg == HX_STAGE_S) {
          const int k = (tail.w >> 16) & 0xff;
          HX_BOUND(k >= 1 && k <= HX_MAX_K && rid + k < nc)
          W->chains[qid] = (uint8_t)k;  // every lane writes the same byte
          rel_first = rid + 1;
          rel_count = k;
        } else if (stg == HX_STAGE_E) {
          const int64_t dl = r->deadline;
          const int64_t arr = r->arrival;
          if (kGeneric) {
            const int ten = (tail.w >> 8) & 0xff;
            HX_BOUND(ten < HX_MAX_TENANTS)
            if (lane == 0) {
              W->tdone[ten]++;
              W->tslo[ten] += now <= dl ? 1 : 0;
            }
            if (a.tenant_kcap) {
              // this tenant's own top-K, for its P95 (Sec. 5's per-tenant tail latency)
              const int kc = a.tenant_kcap[(int64_t)W->trace * HX_MAX_TENANTS + ten];
              HX_BOUND(W->trace < a.n_traces && kc <= a.tenant_topk_off[0])
              const int64_t v = now - arr;
              __syncwarp();
              if (W->ttk[ten] < kc || v > W->ttkmin[ten])
                topk_insert_warp(W->topk + a.tenant_topk_off[ten], &W->ttk[ten], kc, &W->ttkmin[ten], v, lane);
            }
          }
          finish_query(W, dn, qid, now, arr, dl, lane);
        } else {
          const int32_t nx = tail.y;
          HX_BOUND(nx >= 0 ? nx < nc : ~nx < nc)
          if (nx >= 0) {
            rel_first = nx;
            rel_count = 1;
          } else {
            uint8_t* const chains = W->chains;
            const int left = chains[qid] - 1;
            __syncwarp();
            chains[qid] = (uint8_t)left;  // every lane writes the same byte
            rel_first = ~nx;
            rel_count = left == 0 ? 1 : 0;
          }
        }
      } else {
        now = (int64_t)(akey >> 7);
        const int64_t qbase = W->qb;
        const int32_t qa = W->qa;
        HX_BOUND(qa < W->nq)
        rel_first = (int32_t)(a.qcall[qbase + qa] - W->cb);
        HX_BOUND(rel_first >= 0 && rel_first < nc)
        rel_count = 1;
        W->qa = qa + 1;
        W->akey = qa + 1 < W->nq ? (((uint64_t)a.arrival[qbase + qa + 1] << 7) | kArrivalTag) : kKeyInf;
      }

      // Sec. 4.1 for each released request, in request-id order: score every
      // instance and send it to the winner (its Sec. 4.2 key is formed at the
      // batch boundary below, and only if it has to wait).
      for (int32_t jr = 0; jr < rel_count; ++jr) {
        const int32_t rid = rel_first + jr;
        HX_BOUND(rid < nc)
        const CallRec* r = rec + rid;
        // Eq. (comp) and the service time on this lane's two instances
        const int2 ev0 = r->ev[ty0], ev1 = r->ev[ty1];
        const int e0 = ev0.x, e1 = ev1.x, v0 = ev0.y, v1 = ev1.y;
        // SIMT division passes: each lane refreshes one stale reward of its
        // instances per pass (two passes at most)
        const uint64_t beta = (uint64_t)W->beta;
        while (__any_sync(kFull, dirty0 || dirty1)) {
          const bool rj = dirty0 || dirty1;
          const int64_t q = W->q[dirty0 ? m0 : m1];
          const uint64_t res = udiv_trial_f(rj ? beta : 0ull, rj ? W->betaf : 0.0f, (rj && q > 1) ? (uint64_t)q : 1ull);
          const int64_t orew =
              (int64_t)W->one_minus_a * (res < (uint64_t)kRewardCap ? (int64_t)res : kRewardCap);
          if (rj) W->orew[dirty0 ? m0 : m1] = orew;
          if (dirty0) dirty0 = false;
          else dirty1 = false;
        }
        int m;
        // a re-issued request avoids the instance it timed out on
        const int excl = kGeneric ? W->excl : -1;
        if (kGeneric && W->dpol == HX_DISPATCH_RR) {
          m = W->rr;
          if (m == excl) m = (m + 1 == N) ? 0 : m + 1;
          __syncwarp();
          if (lane == 0) W->rr = (m + 1 == N) ? 0 : m + 1;
        } else {
          const int32_t A = W->A;
          int64_t s0 = W->orew[m0] - (int64_t)A * e0;
          int64_t s1 = W->orew[m1] - (int64_t)A * e1;
          if (kGeneric && excl >= 0) {
            if (m0 == excl) s0 = INT64_MIN;
            if (m1 == excl) s1 = INT64_MIN;
          }
          const bool take1 = s1 > s0;
          m = warp_argmax_s64(take1 ? s1 : s0, take1 ? m1 : m0);
        }
        if (kGeneric) W->excl = -1;
        HX_BOUND(m >= 0 && m < N)
        // the winner's costs, from the lane that owns it
        const int64_t est_m = __shfl_sync(kFull, m < 32 ? e0 : e1, m & 31);
        const int svc_m = __shfl_sync(kFull, m < 32 ? v0 : v1, m & 31);
        {
          W->q[m] = W->q[m] + est_m;  // every lane stores the same value
          const bool stale = rewards_on;
          dirty0 = lane == m ? stale : dirty0;
          dirty1 = lane + 32 == m ? stale : dirty1;
        }
        if (kGeneric) {
          const int recj = W->recj;
          if (recj >= 0) {
            HX_BOUND(rid < a.rec_stride)
            const int4 tail = *reinterpret_cast<const int4*>(&r->tbar);
            const int64_t budget = slo_budget(r->deadline - now, tail.x, tail.x + W->frest[(uint32_t)tail.w >> 24]);
            if (lane == 0) log_dispatch(a, recj, rid, m, now, budget);
          }
        }
        if (npend == 0) {
          // nothing of this event waits yet, m's queue is empty and m has a
          // free slot for this request and every one still to be dispatched in
          // this event: the batch boundary below would start it now whatever
          // the others do, so it starts at once
          uint64_t* const sl = W->slot + c.slot_base[m];
          __syncwarp();
          const int cn = W->cnt[m];
          if (W->hsize[m] == 0 && cn + (rel_count - jr) <= c.inst_slots[m]) {
            start_call(sl, m, cn, rid, svc_m);
            W->cnt[m] = cn + 1;  // every lane writes the same count
            set_key(m, sl[0]);
            continue;
          }
        }
        // the local-queue key is formed only if the request has to wait
        HX_BOUND(npend < HX_MAX_K)
        pend_m = lane == npend ? m : pend_m;
        W->prs[npend] = make_int2(rid, svc_m);  // every lane writes the same entry
        W->pest[npend] = (int32_t)est_m;
        npend++;
        touched |= 1ull << m;
      }
      HX_STOP_IF_FAILED()

      // Batch boundary on every touched instance: its free slots go to the most
      // urgent of the waiting requests and this event's new ones.
      uint64_t tm = touched;
      while (tm) {
        const int m = __ffsll((long long)tm) - 1;
        tm &= tm - 1;
        HX_BOUND(m < N)
#ifdef HX_CHECKED
        {
          // m's heap lies inside the warp's arena and holds at most its capacity
          const int64_t cap = W->hcl[m] ? (int64_t)8 << W->hcl[m] : 0;
          HX_BOUND(W->hoff[m] >= 0 && W->hoff[m] + cap <= a.arena_per_warp && W->hsize[m] <= cap &&
                   W->cnt[m] <= c.inst_slots[m])
        }
#endif
        uint64_t* const sl = W->slot + c.slot_base[m];
        const int ns = c.inst_slots[m];
        const unsigned pm = __ballot_sync(kFull, lane < npend && pend_m == m);
        __syncwarp();
        int cn = W->cnt[m];
        const int hs = W->hsize[m];
        // fast paths: an empty queue with room for all of this event's arrivals;
        // one arrival, one free slot and a waiting queue (one sift)
        const int npm = __popc(pm);
        const bool direct = hs == 0 && npm <= ns - cn;
        const bool fused = !direct && npm == 1 && ns - cn == 1;
        const int lpol = kGeneric ? W->lpol : HX_LOCAL_PQ;
        unsigned bits = direct ? pm : 0u;
        int2 fst = make_int2(0, 0);
        if (fused) {
          fst = push_pop(W, rec, now, lpol, m, pm, lane);
          bits = 1u;
        } else if (!direct && pm) {
          status = push_pending(W, rec, now, lpol, a.arena_per_warp, m, pm, lane);
          if (status != HX_OK) break;
        }
        for (;;) {
          int rid, svc;
          if (direct || fused) {
            if (!bits) break;
            const int j = __ffs(bits) - 1;
            bits &= bits - 1;
            const int2 rs = fused ? fst : W->prs[j];
            rid = rs.x;
            svc = rs.y;
          } else {
            const int n = W->hsize[m];
            __syncwarp();
            if (cn >= ns || n == 0) break;
            const HeapEnt top = heap_sift_warp(W->arena + W->hoff[m], n - 1, W->arena[W->hoff[m] + n - 1], lane);
            W->hsize[m] = n - 1;  // every lane writes the same size
            rid = top.rid;
            svc = top.svc;
          }
          HX_BOUND(rid >= 0 && rid < nc && cn < ns)
          start_call(sl, m, cn, rid, svc);
          ++cn;
        }
        HX_STOP_IF_FAILED()
        W->cnt[m] = cn;  // every lane writes the same count
        set_key(m, cn ? sl[0] : kKeyInf);
      }
      if (kGeneric && a.checked && status == HX_OK) {
        // after every event: no instance runs more calls than it has slots or
        // keeps a slot free while requests wait in its queue (Sec. 4.2: free
        // slots take waiting requests at every batch boundary), and t_queue
        // stays non-negative
        __syncwarp();
        bool bad = false;
        for (int m = lane; m < N; m += 32) {
          const int cn = W->cnt[m], ns = c.inst_slots[m];
          bad |= cn > ns || (cn < ns && W->hsize[m] > 0) || W->q[m] < 0;
        }
        if (__any_sync(kFull, bad)) status = HX_ERR_INVARIANT;
      }
      if (status != HX_OK) break;
    }

    digest_flush(W, dn, lane);
    // conservation at the end: every dispatched request finished (t_queue back
    // to zero, no running call, no waiting request)
    bool left = false;
    for (int m = lane; m < N; m += 32) left |= W->q[m] != 0 || W->cnt[m] != 0 || W->hsize[m] != 0;
    const bool leftover = __any_sync(kFull, left);
    if (lane == 0) {
      int st = status;
      const int32_t n_done = W->n_done;
      const int32_t steps0 = W->nc + nq + 8 + (kGeneric && c.n_faults > 0 ? 16 * W->nc + 4096 : 0);
      const int64_t events = (steps0 - steps_left) - W->qa - (kGeneric ? W->reissued : 0);
      // every query and every call completed exactly once
      if (st == HX_OK && (leftover || n_done != nq || events != W->nc)) st = HX_ERR_INVARIANT;
      hx_result res;
      res.p95_us = st == HX_OK ? (nq > 0 ? W->topk[0] : 0) : -1;
      res.makespan_us = W->makespan;
      res.events = events;
      res.digest = W->digest;
      res.slo_met = W->slo_met;
      res.n_done = n_done;
      res.status = st;
      const long long dc = (clock64() - W->clk0) >> 10;
      res.cycles_k = dc < INT32_MAX ? (int32_t)dc : INT32_MAX;
      a.results[W->sim] = res;
      if (kGeneric && a.extras) {
        hx_extra ex;
        for (int t = 0; t < HX_MAX_TENANTS; ++t) {
          ex.slo_met[t] = W->tslo[t];
          ex.n_done[t] = W->tdone[t];
          if (st != HX_OK) ex.p95_us[t] = -1;
          else if (!a.tenant_kcap) ex.p95_us[t] = t == 0 ? res.p95_us : 0;
          else ex.p95_us[t] = W->ttk[t] > 0 ? W->topk[a.tenant_topk_off[t]] : 0;
        }
        ex.reissued = W->reissued;
        ex.pad = 0;
        a.extras[W->sim] = ex;
      }
    }
    __syncwarp();
  }
}

__global__ void __launch_bounds__(kWarpsPerBlock * 32, HX_SIM_MIN_BLOCKS) hx_sim_kernel(SimArgs a, ClusterK c) {
  sim_body<true>(a, c);
}

__global__ void __launch_bounds__(kWarpsPerBlock * 32, HX_SIM_MIN_BLOCKS) hx_sim_kernel_lean(SimArgs a, ClusterK c) {
  sim_body<false>(a, c);
}

// ---------------------------------------------------------- best kernel
namespace {

__device__ __forceinline__ bool cand_better(const BestCand& x, const BestCand& y, int obj) {
  const bool xv = x.flags & 1, yv = y.flags & 1;
  if (xv != yv) return xv;
  if (!xv) return x.p < y.p;
  if (obj == HX_OBJ_P95_SLO95) {
    const bool xf = (x.flags >> 1) & 1, yf = (y.flags >> 1) & 1;
    if (xf != yf) return xf;
    if (!xf && x.slo != y.slo) return x.slo > y.slo;
  }
  if (x.p95 != y.p95) return x.p95 < y.p95;
  return x.p < y.p;
}

__device__ void block_reduce_best(BestCand mine[2], BestCand* out) {
  __shared__ BestCand red[2][256];
  for (int o = 0; o < 2; ++o) red[o][threadIdx.x] = mine[o];
  __syncthreads();
  for (int w = blockDim.x / 2; w > 0; w >>= 1) {
    if ((int)threadIdx.x < w) {
      for (int o = 0; o < 2; ++o)
        if (cand_better(red[o][threadIdx.x + w], red[o][threadIdx.x], o)) red[o][threadIdx.x] = red[o][threadIdx.x + w];
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    out[0] = red[0][0];
    out[1] = red[1][0];
  }
}

}  // namespace

// Blocks 0..T-1: best point of trace t; block T: best point of the sums over traces.
__global__ void __launch_bounds__(256) hx_best_kernel(BestArgs a) {
  const int P = a.n_points;
  BestCand mine[2];
  for (int o = 0; o < 2; ++o) {
    mine[o].p95 = 0;
    mine[o].slo = 0;
    mine[o].p = INT32_MAX;
    mine[o].flags = 0;
  }
  if ((int)blockIdx.x < a.n_traces) {
    const int t = blockIdx.x;
    const int64_t nq = a.q_off[t + 1] - a.q_off[t];
    for (int p = threadIdx.x; p < P; p += blockDim.x) {
      const hx_result r = a.results[(int64_t)t * P + p];
      BestCand x;
      x.p95 = r.p95_us;
      x.slo = r.slo_met;
      x.p = p;
      x.flags = (r.status == HX_OK ? 1 : 0) | ((int64_t)r.slo_met * 100 >= 95 * nq ? 2 : 0);
      for (int o = 0; o < 2; ++o)
        if (cand_better(x, mine[o], o)) mine[o] = x;
    }
    block_reduce_best(mine, a.per_trace + 2 * t);
  } else {
    const int64_t nsum = a.q_off[a.n_traces] - a.q_off[0];
    for (int p = threadIdx.x; p < P; p += blockDim.x) {
      BestCand x;
      x.p95 = 0;
      x.slo = 0;
      x.p = p;
      int valid = 1;
      for (int t = 0; t < a.n_traces; ++t) {
        const hx_result r = a.results[(int64_t)t * P + p];
        x.p95 += r.p95_us;
        x.slo += r.slo_met;
        valid &= r.status == HX_OK ? 1 : 0;
      }
      x.flags = valid | (x.slo * 100 >= 95 * nsum ? 2 : 0);
      if (a.point_sums) {
        a.point_sums[3 * p] = x.p95;
        a.point_sums[3 * p + 1] = x.slo;
        a.point_sums[3 * p + 2] = valid ? 0 : 1;
      }
      for (int o = 0; o < 2; ++o)
        if (cand_better(x, mine[o], o)) mine[o] = x;
    }
    block_reduce_best(mine, a.global);
  }
}

// Self-test of udiv_trial against the compiler's division.
__global__ void hx_selftest_div_kernel(const uint64_t* n, const uint64_t* d, uint64_t* q, uint64_t* q_ref,
                                       int64_t count) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < count) {
    q[i] = udiv_trial(n[i], d[i]);
    q_ref[i] = n[i] / d[i];
  }
}

}  // namespace hx
