// hx_kernels.cu -- the three kernels of the batched HexGen-Flow scheduler
// simulation (arXiv 2505.05286, Sec. 4.1-4.3) for sm_103a.
//
// Integer-only: every time is int64 microseconds, every score and key int64
// fixed point; every division is the compiler's truncating `/`.  Nothing here
// is a dense contraction, so there are no tensor-core paths; the simulation
// kernel is bound by the SM issue rate, the preparation kernel by HBM.
#include "hx_device.cuh"

namespace hx {

// ------------------------------------------------------------------ helpers
__device__ __forceinline__ int64_t ceil_div_pos(int64_t a, int64_t b) { return (a + b - 1) / b; }

// splitmix64 finalizer (Steele, Lea & Flood 2014), used for the digest.
__device__ __forceinline__ uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

__device__ __forceinline__ uint64_t call_term(int32_t rid, int inst, int64_t start) {
  return mix64((uint64_t)start ^ mix64(((uint64_t)(uint32_t)rid << 8) | (uint64_t)inst));
}

__device__ __forceinline__ uint64_t query_term(int32_t qid, int64_t end) {
  return mix64((uint64_t)end ^ mix64(((uint64_t)(uint32_t)qid << 8) | 0xFFull));
}

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
  const int64_t t_slo = (c.slo_mult_fp * (l_s + longest + l_e)) / kScale;
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
        r.est[ty] = (int32_t)es;
        r.svc[ty] = (int32_t)(pre + o * (int64_t)c.decode[ty]);
        sum += es * c.cnt[ty];
      } else {
        r.est[ty] = 0;
        r.svc[ty] = 0;
      }
    }
    r.tbar = (int32_t)(sum / c.n_inst);
    r.deadline = deadline;
    r.arrival = arr;
    r.qid = qid;
    r.stage = (uint8_t)st;
    r.k = (uint8_t)k;
    r.pad = 0;
    if (st == HX_STAGE_S) {
      r.u = 0;
      r.next = -1;
    } else if (st == HX_STAGE_E) {
      r.u = 0;
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

// Per-warp shared state of one simulation.
struct Smem {
  int64_t* q;          // [64] sum of est over requests dispatched and unfinished
  int64_t* rew;        // [64] reward_of(beta, q)
  uint64_t* nkey;      // [64] earliest running (end << 24 | rid), or kKeyInf
  int64_t* slot_end;   // [total_slots] end time or kTimeInf when free
  int32_t* slot_rid;   // [total_slots]
  int32_t* hoff;       // [64] local queue: offset of the heap in the arena
  int32_t* hcap;       // [64] capacity
  int32_t* hsize;      // [64] size
  uint32_t* freem;     // [64] free-slot mask
  int32_t* nslot;      // [64] slot of nkey
};

__device__ __forceinline__ Smem carve(unsigned char* base, int ts) {
  Smem s;
  s.q = reinterpret_cast<int64_t*>(base);
  s.rew = s.q + 64;
  s.nkey = reinterpret_cast<uint64_t*>(s.rew + 64);
  s.slot_end = reinterpret_cast<int64_t*>(s.nkey + 64);
  s.slot_rid = reinterpret_cast<int32_t*>(s.slot_end + ts);
  s.hoff = s.slot_rid + ts;
  s.hcap = s.hoff + 64;
  s.hsize = s.hcap + 64;
  s.freem = reinterpret_cast<uint32_t*>(s.hsize + 64);
  s.nslot = reinterpret_cast<int32_t*>(s.freem + 64);
  return s;
}

__device__ __forceinline__ bool ent_better(long long ka, int ra, long long kb, int rb) {
  return ka > kb || (ka == kb && ra < rb);
}

// Binary max-heap on (key desc, rid asc); single lane.
__device__ void heap_push(HeapEnt* h, int n, long long key, int rid) {
  int i = n;
  while (i > 0) {
    int par = (i - 1) >> 1;
    HeapEnt pe = h[par];
    if (!ent_better(key, rid, pe.key, pe.rid)) break;
    h[i] = pe;
    i = par;
  }
  HeapEnt e;
  e.key = key;
  e.rid = rid;
  e.pad = 0;
  h[i] = e;
}

__device__ HeapEnt heap_pop(HeapEnt* h, int n) {
  HeapEnt top = h[0];
  HeapEnt last = h[n - 1];
  int m = n - 1;
  int i = 0;
  for (;;) {
    int l = 2 * i + 1;
    if (l >= m) break;
    int r = l + 1;
    HeapEnt cl = h[l];
    int cidx = l;
    if (r < m) {
      HeapEnt cr = h[r];
      if (ent_better(cr.key, cr.rid, cl.key, cl.rid)) { cl = cr; cidx = r; }
    }
    if (!ent_better(cl.key, cl.rid, last.key, last.rid)) break;
    h[i] = cl;
    i = cidx;
  }
  if (m > 0) h[i] = last;
  return top;
}

// Min-heap of the K largest latencies seen so far; single lane.
__device__ void topk_insert(int64_t* h, int& n, int kcap, int64_t v) {
  if (n < kcap) {
    int i = n++;
    while (i > 0) {
      int par = (i - 1) >> 1;
      int64_t pv = h[par];
      if (pv <= v) break;
      h[i] = pv;
      i = par;
    }
    h[i] = v;
  } else if (v > h[0]) {
    int i = 0;
    for (;;) {
      int l = 2 * i + 1;
      if (l >= n) break;
      int r = l + 1;
      int cidx = l;
      int64_t cv = h[l];
      if (r < n && h[r] < cv) { cv = h[r]; cidx = r; }
      if (cv >= v) break;
      h[i] = cv;
      i = cidx;
    }
    h[i] = v;
  }
}

struct SimState {
  int64_t now;
  uint64_t touched;
  int32_t rr;
  int32_t bump;
  int32_t status;
};

}  // namespace

__global__ void __launch_bounds__(kWarpsPerBlock * 32) hx_sim_kernel(SimArgs a, ClusterK c) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int ts = c.total_slots;
  Smem S = carve(smem_raw + warp * c.smem_per_warp, ts);
  const int64_t gw = (int64_t)blockIdx.x * kWarpsPerBlock + warp;
  HeapEnt* arena = a.arena + gw * a.arena_per_warp;
  uint8_t* chains = a.chains + gw * a.chains_per_warp;
  int64_t* topk = a.topk + gw * a.topk_per_warp;
  const int N = c.n_inst;
  const int m0 = lane, m1 = lane + 32;
  const int ty0 = m0 < N ? c.inst_type[m0] : 0;
  const int ty1 = m1 < N ? c.inst_type[m1] : 0;

  // stage reference costs: mean over instances of Eq. (comp) at the stage's reference tokens
  int64_t cref[4];
#pragma unroll
  for (int s = 0; s < 4; ++s) {
    int64_t sum = 0;
    for (int ty = 0; ty < c.n_types; ++ty)
      sum += cost_on_type(c, ty, c.ref_prompt[s], c.ref_out[s]) * c.cnt[ty];
    cref[s] = sum / N;
  }

  for (;;) {
    unsigned long long simu = 0;
    if (lane == 0) simu = atomicAdd(a.work_counter, 1ull);
    const int64_t sim = (int64_t)__shfl_sync(kFull, simu, 0);
    if (sim >= a.n_sims) break;

    const int t = (int)(sim / a.n_points);
    const int p = (int)(sim - (int64_t)t * a.n_points);
    const int64_t qb = a.q_off[t];
    const int32_t nq = (int32_t)(a.q_off[t + 1] - qb);
    const int64_t cb = a.c_off[t];
    const int32_t nc = (int32_t)(a.c_off[t + 1] - cb);
    const CallRec* rec = a.rec + cb;
    const int64_t* arr = a.arrival + qb;
    const int64_t* qcall = a.qcall + qb;
    const int64_t A = a.alpha[p], G = a.gamma[p], beta = a.beta[p];
    const int rho = a.rho[p];
    const int lpol = a.lpol[p], dpol = a.dpol[p];
    const int recj = a.rec_map ? a.rec_map[sim] : -1;
    const int64_t one_minus_a = kScale - A;
    const int64_t rmax = c.rmax;
    const int64_t corr_plan = rho < rmax ? rho : rmax;
    const int64_t f_s = cref[HX_STAGE_G] + corr_plan * cref[HX_STAGE_C] + cref[HX_STAGE_E];
    const int64_t f_g = corr_plan * cref[HX_STAGE_C] + cref[HX_STAGE_E];
    const int64_t rew0 = reward_of(beta, 0);

    for (int m = lane; m < 64; m += 32) {
      S.q[m] = 0;
      S.rew[m] = rew0;
      S.nkey[m] = kKeyInf;
      S.hoff[m] = 0;
      S.hcap[m] = 0;
      S.hsize[m] = 0;
      S.freem[m] = m < N ? ((1u << c.inst_slots[m]) - 1u) : 0u;
      S.nslot[m] = -1;
    }
    for (int j = lane; j < ts; j += 32) {
      S.slot_end[j] = kTimeInf;
      S.slot_rid[j] = -1;
    }
    __syncwarp();

    uint64_t k0 = kKeyInf, k1 = kKeyInf;  // this lane's instances' next-completion event keys
    const int kcap = nq - (95 * nq + 99) / 100 + 1;
    int tk = 0;
    int32_t qa = 0;
    uint64_t akey = nq > 0 ? (((uint64_t)arr[0] << 7) | kArrivalTag) : kKeyInf;
    int32_t n_done = 0, slo_met = 0;
    int64_t makespan = 0, events = 0;
    uint64_t digest = 0;
    SimState st;
    st.now = 0;
    st.touched = 0;
    st.rr = 0;
    st.bump = 0;
    st.status = HX_OK;
    const int64_t max_steps = (int64_t)nc + nq + 8;
    int64_t steps = 0;

    // refresh this lane's event key for instance m from S.nkey
    auto refresh_key = [&](int m) {
      if (lane == (m & 31)) {
        const uint64_t nk = S.nkey[m];
        const uint64_t kk = nk == kKeyInf ? kKeyInf : (((nk >> 24) << 7) | (uint64_t)m);
        if (m < 32) k0 = kk; else k1 = kk;
      }
    };

    // Sec. 4.1 + 4.2: budget at send time, score every instance, enqueue.
    auto dispatch = [&](int32_t rid) {
      const CallRec* r = rec + rid;
      const int stg = r->stage;
      const int64_t tb = r->tbar;
      int64_t f;
      if (stg == HX_STAGE_S) f = f_s;
      else if (stg == HX_STAGE_G) f = f_g;
      else if (stg == HX_STAGE_C) {
        const int64_t left = rmax - (int64_t)r->u;
        f = (rho < left ? rho : left) * cref[HX_STAGE_C] + cref[HX_STAGE_E];
      } else f = 0;
      const int64_t budget = scaled_div(r->deadline - st.now, tb, tb + f);
      int m;
      if (dpol == HX_DISPATCH_RR) {
        m = st.rr;
        st.rr = (st.rr + 1 == N) ? 0 : st.rr + 1;
      } else {
        int64_t s0 = INT64_MIN, s1 = INT64_MIN;
        if (m0 < N) s0 = one_minus_a * S.rew[m0] - A * (int64_t)r->est[ty0];
        if (m1 < N) s1 = one_minus_a * S.rew[m1] - A * (int64_t)r->est[ty1];
        const bool take1 = s1 > s0;
        m = warp_argmax_s64(take1 ? s1 : s0, take1 ? m1 : m0);
      }
      const int64_t est_m = r->est[c.inst_type[m]];
      if (lane == (m & 31)) {
        const int64_t q = S.q[m] + est_m;
        S.q[m] = q;
        S.rew[m] = reward_of(beta, q);
      }
      const long long key = lpol == HX_LOCAL_PQ ? (long long)(kScale * (est_m - budget) - G * st.now)
                                                : (long long)(-st.now);
      // local queue push, growing the heap inside the arena when full
      const int size = S.hsize[m], cap = S.hcap[m], off = S.hoff[m];
      __syncwarp();
      int hoff = off;
      if (size == cap) {
        const int ncap = cap ? 2 * cap : 16;
        if ((int64_t)st.bump + ncap > a.arena_per_warp) {
          st.status = HX_ERR_CAPACITY;
          return;
        }
        hoff = st.bump;
        st.bump += ncap;
        for (int j = lane; j < size; j += 32) arena[hoff + j] = arena[off + j];
        __syncwarp();
        if (lane == 0) {
          S.hoff[m] = hoff;
          S.hcap[m] = ncap;
        }
      }
      if (lane == 0) {
        heap_push(arena + hoff, size, key, rid);
        S.hsize[m] = size + 1;
        if (recj >= 0) {
          const int64_t o = (int64_t)recj * a.rec_stride + rid;
          a.rec_inst[o] = m;
          a.rec_enq[o] = st.now;
          a.rec_budget[o] = budget;
        }
      }
      __syncwarp();
      st.touched |= 1ull << m;
    };

    // Batch boundary on instance m: start the best waiting requests on free slots.
    auto fill = [&](int m) {
      const int sb = c.slot_base[m];
      const int ty = c.inst_type[m];
      for (;;) {
        const bool go = S.freem[m] != 0u && S.hsize[m] > 0;
        __syncwarp();
        if (!go) break;
        int rid = 0;
        if (lane == 0) {
          const int n = S.hsize[m];
          HeapEnt top = heap_pop(arena + S.hoff[m], n);
          S.hsize[m] = n - 1;
          rid = top.rid;
          const int64_t end = st.now + rec[rid].svc[ty];
          const uint32_t fm = S.freem[m];
          const int sl = __ffs(fm) - 1;
          S.freem[m] = fm & ~(1u << sl);
          S.slot_end[sb + sl] = end;
          S.slot_rid[sb + sl] = rid;
          const uint64_t nk = ((uint64_t)end << 24) | (uint64_t)rid;
          if (nk < S.nkey[m]) {
            S.nkey[m] = nk;
            S.nslot[m] = sl;
          }
          if (recj >= 0) a.rec_start[(int64_t)recj * a.rec_stride + rid] = st.now;
        }
        rid = __shfl_sync(kFull, rid, 0);
        __syncwarp();
        refresh_key(m);
        digest += call_term(rid, m, st.now);
      }
    };

    for (;;) {
      const uint64_t ck = warp_min_u64(k0 < k1 ? k0 : k1);
      if (ck == kKeyInf && akey == kKeyInf) break;
      if (++steps > max_steps) {
        st.status = HX_ERR_STEP_LIMIT;
        break;
      }
      st.touched = 0;
      if (ck < akey) {
        // completion on instance m
        const int m = (int)(ck & 127ull);
        st.now = (int64_t)(ck >> 7);
        const int sb = c.slot_base[m];
        const int sl = S.nslot[m];
        const int32_t rid = S.slot_rid[sb + sl];
        __syncwarp();
        if (lane == 0) {
          S.slot_end[sb + sl] = kTimeInf;
          S.slot_rid[sb + sl] = -1;
          S.freem[m] |= 1u << sl;
        }
        __syncwarp();
        // earliest remaining (end, rid) on m: lanes over its slots
        uint64_t sk = kKeyInf;
        if (lane < c.inst_slots[m]) {
          const int64_t e = S.slot_end[sb + lane];
          if (e != kTimeInf) sk = ((uint64_t)e << 24) | (uint64_t)(uint32_t)S.slot_rid[sb + lane];
        }
        const uint64_t mk = warp_min_u64(sk);
        const unsigned who = __ballot_sync(kFull, sk == mk && mk != kKeyInf);
        __syncwarp();
        if (lane == 0) {
          S.nkey[m] = mk;
          S.nslot[m] = who ? __ffs(who) - 1 : -1;
        }
        const CallRec* r = rec + rid;
        const int64_t est_m = r->est[c.inst_type[m]];
        if (lane == (m & 31)) {
          const int64_t q = S.q[m] - est_m;
          S.q[m] = q;
          S.rew[m] = reward_of(beta, q);
        }
        __syncwarp();
        refresh_key(m);
        st.touched |= 1ull << m;
        events++;
        const int stg = r->stage;
        if (stg == HX_STAGE_S) {
          const int k = r->k;
          if (lane == 0) chains[r->qid] = (uint8_t)k;
          for (int j = 1; j <= k && st.status == HX_OK; ++j) dispatch(rid + j);
        } else if (stg == HX_STAGE_E) {
          const int64_t lat = st.now - r->arrival;
          slo_met += st.now <= r->deadline ? 1 : 0;
          n_done++;
          makespan = st.now > makespan ? st.now : makespan;
          digest += query_term(r->qid, st.now);
          if (lane == 0) topk_insert(topk, tk, kcap, lat);
          tk = __shfl_sync(kFull, tk, 0);
        } else {
          const int32_t nx = r->next;
          if (nx >= 0) {
            dispatch(nx);
          } else {
            int left = 0;
            if (lane == 0) {
              left = chains[r->qid] - 1;
              chains[r->qid] = (uint8_t)left;
            }
            left = __shfl_sync(kFull, left, 0);
            if (left == 0) dispatch(~nx);
          }
        }
      } else {
        st.now = (int64_t)(akey >> 7);
        const int32_t srid = (int32_t)(qcall[qa] - cb);
        qa++;
        akey = qa < nq ? (((uint64_t)arr[qa] << 7) | kArrivalTag) : kKeyInf;
        dispatch(srid);
      }
      if (st.status != HX_OK) break;
      uint64_t tm = st.touched;
      while (tm) {
        const int m = __ffsll((long long)tm) - 1;
        tm &= tm - 1;
        fill(m);
      }
    }

    if (lane == 0) {
      int status = st.status;
      if (status == HX_OK && n_done != nq) status = HX_ERR_STEP_LIMIT;
      hx_result res;
      res.p95_us = status == HX_OK ? (nq > 0 ? topk[0] : 0) : -1;
      res.makespan_us = makespan;
      res.events = events;
      res.digest = digest;
      res.slo_met = slo_met;
      res.n_done = n_done;
      res.status = status;
      res.pad = 0;
      a.results[sim] = res;
    }
    __syncwarp();
  }
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
      for (int o = 0; o < 2; ++o)
        if (cand_better(x, mine[o], o)) mine[o] = x;
    }
    block_reduce_best(mine, a.global);
  }
}

}  // namespace hx
