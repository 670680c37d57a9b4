// hx_api.cu -- the C ABI (include/hxsim.h): input validation, flattening of
// the traces into device arrays, per-warp scratch sizing and the launches of
// the preparation, simulation and best-point kernels on the caller's stream.
#include <cuda_runtime.h>
#include <nvtx3/nvToolsExt.h>

#include <algorithm>
#include <atomic>
#include <cstdio>
#include <cstddef>
#include <cstring>
#include <exception>
#include <memory>
#include <mutex>
#include <stdexcept>
#include <system_error>
#include <new>
#include <string>
#include <thread>
#include <vector>

#include "hx_device.cuh"

namespace {

thread_local std::string g_err;

// NVTX range over one ABI call (host side: validation, copies, launches), for
// profilers that group kernels by range (e.g. ncu --nvtx).
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

int fail(int code, const std::string& msg) {
  g_err = msg;
  return code;
}

// Host-side C++ exceptions (an allocation that fails) become a status
// here instead of crossing the C ABI.
template <class F>
int guarded(F&& f) noexcept {
  const char* msg = "unexpected host exception";
  int code = HX_ERR_STATE;
  try {
    return f();
  } catch (const std::bad_alloc&) {
    msg = "host allocation failed";
    code = HX_ERR_OOM;
  } catch (const std::length_error&) {
    msg = "host allocation failed";
    code = HX_ERR_OOM;
  } catch (...) {
  }
  try {
    g_err = msg;
  } catch (...) {
  }
  return code;
}

#define HX_CUDA(x)                                                                   \
  do {                                                                               \
    cudaError_t e_ = (x);                                                            \
    if (e_ != cudaSuccess)                                                           \
      return fail(e_ == cudaErrorMemoryAllocation ? HX_ERR_OOM : HX_ERR_CUDA,        \
                  std::string(#x) + ": " + cudaGetErrorString(e_));                  \
  } while (0)

constexpr int64_t kTokMax = int64_t(1) << 20;     // prompt / output tokens per call
constexpr int64_t kCostMax = int64_t(1) << 28;    // any per-call cost bound, us
constexpr int64_t kHorizonMax = int64_t(1) << 39; // last arrival + all service, us

int64_t align_up(int64_t x, int64_t a) { return (x + a - 1) / a * a; }

// The dynamic shared-memory limit of a kernel (cudaFuncAttributeMax-
// DynamicSharedMemorySize) is one setting per function and device, shared by
// every handle in the process.  It is set, under a mutex, to the largest size
// any launch of that kernel on that device has asked for, so a later handle
// or static call with a smaller cluster never lowers it below what an earlier
// handle launches with.  Called before every launch; it sets the attribute
// each time (a host-side call), so a device reset cannot leave it lower than
// the record says.
constexpr int kMaxDevices = 64;
std::mutex g_smem_mu;
int g_smem_limit[kMaxDevices][2] = {};  // [device][0: hx_sim_kernel, 1: hx_sim_kernel_lean]

int ensure_dyn_smem(bool generic, int bytes) {
  int dev = 0;
  HX_CUDA(cudaGetDevice(&dev));
  if (dev < 0 || dev >= kMaxDevices) return fail(HX_ERR_INVALID, "device index out of range");
  std::lock_guard<std::mutex> lock(g_smem_mu);
  int& cur = g_smem_limit[dev][generic ? 0 : 1];
  const int want = std::max(cur, bytes);
  const void* kfn = generic ? (const void*)hx::hx_sim_kernel : (const void*)hx::hx_sim_kernel_lean;
  if (cudaFuncSetAttribute(kfn, cudaFuncAttributeMaxDynamicSharedMemorySize, want) != cudaSuccess) {
    cudaGetLastError();
    return fail(HX_ERR_CUDA, "cannot reserve " + std::to_string(want) +
                                 " bytes of shared memory for the simulation kernel");
  }
  cur = want;
  return HX_OK;
}

// The lean instantiation serves grids that are all workload-balanced dispatch
// with the urgency queue, log nothing, check nothing, count one tenant and
// have no fault windows.
bool needs_generic(const hx_grid* grid, const hx::ClusterK& ck, bool record, bool force, bool checked) {
  if (record || force || checked || ck.n_tenants > 1 || ck.n_faults > 0) return true;
  for (int p = 0; p < grid->n_points; ++p)
    if (grid->local_policy[p] != HX_LOCAL_PQ || grid->dispatch_policy[p] != HX_DISPATCH_WB) return true;
  return false;
}

}  // namespace

struct hx_sim {
  int32_t n_traces = 0, n_points = 0;
  int64_t n_sims = 0, n_q = 0, n_c = 0;
  int32_t max_nq = 0, max_nc = 0, max_kcap = 1;
  hx::ClusterK ck{};
  int32_t n_tenants = 0;          // as given in hx_cluster (validation of later uploads)
  std::vector<hx_fault> faults;
  std::vector<int32_t> h_nq, h_nc;
  // device: inputs
  int64_t* d_arrival = nullptr;
  int64_t* d_qcall = nullptr;
  int64_t* d_q_off = nullptr;
  int64_t* d_c_off = nullptr;
  uint8_t* d_k = nullptr;
  uint8_t* d_tenant = nullptr;
  int32_t* d_prompt = nullptr;
  int32_t* d_out = nullptr;
  int32_t* d_out_est = nullptr;
  uint8_t* d_stage = nullptr;
  uint8_t* d_cand = nullptr;
  uint8_t* d_retry = nullptr;
  int64_t* d_alpha = nullptr;
  int64_t* d_gamma = nullptr;
  int64_t* d_beta = nullptr;
  int32_t* d_rho = nullptr;
  uint8_t* d_lp = nullptr;
  uint8_t* d_dp = nullptr;
  // device: derived and outputs
  hx::CallRec* d_rec = nullptr;
  hx_result* d_results = nullptr;
  hx_extra* d_extras = nullptr;  // generic kernel only
  unsigned long long* d_counter = nullptr;
  hx::BestCand* d_best_trace = nullptr;
  hx::BestCand* d_best_global = nullptr;
  int64_t* d_point_sums = nullptr;
  // per-tenant top-K heaps (generic kernel with several tenants)
  int32_t* d_tenant_kcap = nullptr;
  int64_t tenant_topk_off[HX_MAX_TENANTS] = {0, 0, 0, 0};
  // device: scratch
  hx::HeapEnt* d_arena = nullptr;
  uint8_t* d_chains = nullptr;
  int64_t* d_topk = nullptr;
  int64_t arena_per_warp = 0, chains_per_warp = 0, topk_per_warp = 0;
  // device: records
  int32_t n_record = 0;
  int64_t rec_stride = 0;
  int32_t* d_rec_map = nullptr;
  // run only these simulations, in work order (NULL: all of them)
  int64_t* d_subset = nullptr;  // the work order when not the kernel's own (see work_order)
  int64_t n_work = 0;
  int32_t work_order = 0;       // hx_info.work_order
  bool checked = false;
  int32_t* d_rec_inst = nullptr;
  int64_t* d_rec_enq = nullptr;
  int64_t* d_rec_budget = nullptr;
  int64_t* d_rec_start = nullptr;
  int64_t* d_rec_end = nullptr;
  std::vector<int32_t> record_sims;
  // launch shape
  int blocks = 0, resident_warps = 0, smem_per_block = 0;
  bool generic = true;  // which instantiation of the simulation kernel runs
  int64_t scratch_bytes = 0, device_bytes = 0;
  cudaStream_t last_stream = nullptr;
  bool ran = false;
  bool timing = false;
  // with timing: four events per run (before prep, before and after the
  // simulations, after the best point) for the last kTimedRuns runs
  static constexpr int kTimedRuns = 64;
  std::vector<cudaEvent_t> ev;
  int64_t runs = 0;
  cudaEvent_t* run_ev(int64_t r) { return ev.data() + 4 * (r % kTimedRuns); }
  std::vector<void*> allocs;

  template <class T>
  int alloc(T** p, int64_t count) {
    size_t bytes = (size_t)std::max<int64_t>(count, 1) * sizeof(T);
    void* q = nullptr;
    cudaError_t e = cudaMalloc(&q, bytes);
    if (e != cudaSuccess) {
      cudaGetLastError();
      return fail(HX_ERR_OOM, "cudaMalloc of " + std::to_string(bytes) + " bytes: " + cudaGetErrorString(e));
    }
    allocs.push_back(q);
    device_bytes += (int64_t)bytes;
    *p = static_cast<T*>(q);
    return HX_OK;
  }

  ~hx_sim() {
    for (void* p : allocs) cudaFree(p);
    for (auto e : ev)
      if (e) cudaEventDestroy(e);
  }
};

namespace {

int validate_cluster(const hx_cluster* c, int64_t* min_prefill, int64_t* max_decode) {
  if (!c) return fail(HX_ERR_INVALID, "cluster is NULL");
  if (c->n_types < 1 || c->n_types > HX_MAX_TYPES) return fail(HX_ERR_INVALID, "n_types must be 1..4");
  if (c->n_inst < 1 || c->n_inst > HX_MAX_INST) return fail(HX_ERR_INVALID, "n_inst must be 1..64");
  if (!c->prefill_tok_s || !c->decode_us_tok || !c->slots || !c->inst_type || !c->stage_ref_prompt ||
      !c->stage_ref_out)
    return fail(HX_ERR_INVALID, "cluster array is NULL");
  int64_t mp = INT64_MAX, md = 0;
  for (int t = 0; t < c->n_types; ++t) {
    if (c->prefill_tok_s[t] < 1) return fail(HX_ERR_INVALID, "prefill_tok_s must be >= 1");
    if (c->decode_us_tok[t] < 0) return fail(HX_ERR_INVALID, "decode_us_tok must be >= 0");
    if (c->slots[t] < 1 || c->slots[t] > HX_MAX_SLOTS) return fail(HX_ERR_INVALID, "slots must be 1..16");
    mp = std::min<int64_t>(mp, c->prefill_tok_s[t]);
    md = std::max<int64_t>(md, c->decode_us_tok[t]);
  }
  for (int m = 0; m < c->n_inst; ++m)
    if (c->inst_type[m] >= c->n_types) return fail(HX_ERR_INVALID, "inst_type out of range");
  if (c->ref_type < 0 || c->ref_type >= c->n_types) return fail(HX_ERR_INVALID, "ref_type out of range");
  if (c->slo_mult_fp < 0 || c->slo_mult_fp > 16 * HX_SCALE) return fail(HX_ERR_INVALID, "slo_mult_fp must be 0..16*SCALE");
  if (c->rmax < 0 || c->rmax > HX_MAX_RETRY) return fail(HX_ERR_INVALID, "rmax must be 0..15");
  for (int s = 0; s < 4; ++s) {
    const int64_t p = c->stage_ref_prompt[s], o = c->stage_ref_out[s];
    if (p < 0 || p > kTokMax || o < 0 || o > kTokMax) return fail(HX_ERR_INVALID, "stage reference tokens out of range");
    if ((p * 1000000 + mp - 1) / mp + o * md >= kCostMax) return fail(HX_ERR_INVALID, "stage reference cost too large");
  }
  if (c->n_tenants < 0 || c->n_tenants > HX_MAX_TENANTS) return fail(HX_ERR_INVALID, "n_tenants must be 0..4");
  if (c->tenant_slo_mult_fp)
    for (int t = 0; t < std::max(c->n_tenants, 1); ++t)
      if (c->tenant_slo_mult_fp[t] < 0 || c->tenant_slo_mult_fp[t] > 16 * HX_SCALE)
        return fail(HX_ERR_INVALID, "tenant_slo_mult_fp must be 0..16*SCALE");
  if (c->timeout_mult_fp != 0 && (c->timeout_mult_fp < HX_SCALE || c->timeout_mult_fp > 100 * HX_SCALE))
    return fail(HX_ERR_INVALID, "timeout_mult_fp must be 0 or SCALE..100*SCALE");
  if (c->n_faults < 0 || c->n_faults > HX_MAX_FAULTS) return fail(HX_ERR_INVALID, "n_faults must be 0..16");
  if (c->n_faults > 0 && !c->faults) return fail(HX_ERR_INVALID, "faults is NULL");
  for (int f = 0; f < c->n_faults; ++f) {
    const hx_fault& F = c->faults[f];
    if (F.inst < 0 || F.inst >= c->n_inst) return fail(HX_ERR_INVALID, "fault instance out of range");
    if (F.t0_us < 0 || F.t1_us < F.t0_us || F.t1_us > (int64_t(1) << 38))
      return fail(HX_ERR_INVALID, "fault window must satisfy 0 <= t0 <= t1 <= 2^38");
    if (F.slow_fp != 0 && (F.slow_fp < HX_SCALE / 100 || F.slow_fp > 100 * HX_SCALE))
      return fail(HX_ERR_INVALID, "fault slow_fp must be 0 or SCALE/100..100*SCALE");
    if (F.slow_fp == 0 && c->timeout_mult_fp == 0)
      return fail(HX_ERR_INVALID, "a stopped instance (slow_fp = 0) needs a timeout");
  }
  *min_prefill = mp;
  *max_decode = md;
  return HX_OK;
}

int validate_grid(const hx_grid* g) {
  if (!g) return fail(HX_ERR_INVALID, "grid is NULL");
  if (g->n_points < 1) return fail(HX_ERR_INVALID, "n_points must be >= 1");
  if (!g->alpha_fp || !g->gamma_fp || !g->rho || !g->beta_us2 || !g->local_policy || !g->dispatch_policy)
    return fail(HX_ERR_INVALID, "grid array is NULL");
  for (int p = 0; p < g->n_points; ++p) {
    if (g->alpha_fp[p] < 0 || g->alpha_fp[p] > HX_SCALE) return fail(HX_ERR_INVALID, "alpha_fp must be 0..SCALE");
    if (g->gamma_fp[p] < 0 || g->gamma_fp[p] > 4 * HX_SCALE) return fail(HX_ERR_INVALID, "gamma_fp must be 0..4*SCALE");
    if (g->rho[p] < 0 || g->rho[p] > HX_MAX_RETRY) return fail(HX_ERR_INVALID, "rho must be 0..15");
    if (g->beta_us2[p] < 0 || g->beta_us2[p] > (int64_t(1) << 62)) return fail(HX_ERR_INVALID, "beta_us2 out of range");
    if (g->local_policy[p] > 2 || g->dispatch_policy[p] > 1) return fail(HX_ERR_INVALID, "unknown policy");
  }
  return HX_OK;
}

int validate_trace(const hx_trace* tr, int ti, const hx_cluster* c, int64_t min_prefill, int64_t max_decode) {
  const std::string where = "trace " + std::to_string(ti) + ": ";
  if (tr->n_queries < 0 || tr->n_calls < 0 || tr->n_calls >= (1 << 24))
    return fail(HX_ERR_INVALID, where + "n_queries/n_calls out of range");
  if (tr->n_queries > 0 && (!tr->arrival_us || !tr->k || !tr->prompt || !tr->out || !tr->out_est || !tr->stage ||
                            !tr->cand || !tr->retry))
    return fail(HX_ERR_INVALID, where + "array is NULL");
  if (!tr->call_base) return fail(HX_ERR_INVALID, where + "call_base is NULL");
  if (tr->call_base[0] != 0 || tr->call_base[tr->n_queries] != tr->n_calls)
    return fail(HX_ERR_INVALID, where + "call_base must run from 0 to n_calls");
  // the time horizon: the last arrival plus every call's cost bound
  // ceil(prompt * 10^6 / min_prefill) + max(out, out_est) * max_decode;
  // summed here as sum(prompt) and sum(decode part), the sum of the ceilings
  // lying within n_calls above the ceiling of the sum
  int64_t tok_sum = 0, dec_sum = 0;
  for (int32_t i = 0; i < tr->n_queries; ++i) {
    if (tr->arrival_us[i] < 0 || (i > 0 && tr->arrival_us[i] < tr->arrival_us[i - 1]))
      return fail(HX_ERR_INVALID, where + "arrivals must be non-negative and sorted");
    const int32_t b = tr->call_base[i], e = tr->call_base[i + 1];
    const int k = tr->k[i];
    if (tr->tenant && tr->tenant[i] >= std::max(c->n_tenants, 1))
      return fail(HX_ERR_INVALID, where + "tenant out of range");
    if (k == 0) {
      // a single-shot request: one evaluation-stage call
      if (e - b != 1 || b < 0 || e > tr->n_calls || tr->stage[b] != HX_STAGE_E)
        return fail(HX_ERR_INVALID, where + "a k = 0 query must be a single E call");
    } else {
      if (k > HX_MAX_K) return fail(HX_ERR_INVALID, where + "k must be 0..8");
      if (e - b < 2 + k || b < 0 || e > tr->n_calls) return fail(HX_ERR_INVALID, where + "bad call_base");
      if (tr->stage[b] != HX_STAGE_S || tr->stage[e - 1] != HX_STAGE_E)
        return fail(HX_ERR_INVALID, where + "a query must start with S and end with E");
      for (int cd = 0; cd < k; ++cd)
        if (tr->stage[b + 1 + cd] != HX_STAGE_G || tr->cand[b + 1 + cd] != cd)
          return fail(HX_ERR_INVALID, where + "S must be followed by G_0..G_{k-1}");
      int prev_c = -1, prev_r = 0;
      for (int32_t j = b + 1 + k; j < e - 1; ++j) {
        const int cd = tr->cand[j], r = tr->retry[j];
        if (tr->stage[j] != HX_STAGE_C || cd >= k || r < 1 || r > c->rmax)
          return fail(HX_ERR_INVALID, where + "corrections must be C calls of a candidate with 1 <= retry <= rmax");
        if (cd == prev_c ? r != prev_r + 1 : (cd < prev_c || r != 1))
          return fail(HX_ERR_INVALID, where + "corrections must be ordered by (candidate, retry)");
        prev_c = cd;
        prev_r = r;
      }
    }
    for (int32_t j = b; j < e; ++j) {
      const int64_t p = tr->prompt[j], o = tr->out[j], oe = tr->out_est[j];
      if (p < 1 || p > kTokMax || o < 0 || o > kTokMax || oe < 0 || oe > kTokMax)
        return fail(HX_ERR_INVALID, where + "token counts out of range");
      // ceil(p * 10^6 / min_prefill) + dec >= 2^28, decided without a division:
      // ceil(x / d) >= m exactly when x > (m - 1) * d
      const int64_t dec = std::max(o, oe) * max_decode;
      if (dec >= kCostMax || p * 1000000 > (kCostMax - 1 - dec) * min_prefill)
        return fail(HX_ERR_INVALID, where + "a call's cost exceeds 2^28 us");
      tok_sum += p;
      dec_sum += dec;
    }
  }
  // fault windows stretch attempts (slow-down or timeout) and delay the rest
  int64_t stretch = HX_SCALE, last = tr->n_queries > 0 ? tr->arrival_us[tr->n_queries - 1] : 0;
  for (int f = 0; f < c->n_faults; ++f) {
    stretch = std::max(stretch, std::max<int64_t>(c->faults[f].slow_fp, c->timeout_mult_fp));
    last = std::max(last, c->faults[f].t1_us);
  }
  const int64_t widen = 1 + (stretch + HX_SCALE - 1) / HX_SCALE, halve = c->n_faults > 0 ? 1 : 2;
  const __int128 tok_us = (__int128)tok_sum * 1000000;
  const int64_t lower = (int64_t)((tok_us + min_prefill - 1) / min_prefill) + dec_sum;
  const int64_t upper = lower + tr->n_calls;
  if (upper <= kHorizonMax && upper * widen / halve + last <= kHorizonMax) return HX_OK;
  // near the limit: the exact sum of the per-call bounds decides
  int64_t horizon = 0;
  for (int32_t j = 0; j < tr->n_calls; ++j)
    horizon += (tr->prompt[j] * int64_t(1000000) + min_prefill - 1) / min_prefill +
               std::max<int64_t>(tr->out[j], tr->out_est[j]) * max_decode;
  if (horizon > kHorizonMax) return fail(HX_ERR_INVALID, where + "time horizon exceeds 2^39 us");
  horizon = horizon * widen / halve + last;
  if (horizon > kHorizonMax) return fail(HX_ERR_INVALID, where + "time horizon exceeds 2^39 us");
  return HX_OK;
}

// fn(t) for t = 0 .. n_traces - 1 on up to 16 host threads, one trace at a
// time each, when the traces hold enough calls to pay for the threads.
template <class F>
void for_each_trace(const hx_trace* traces, int32_t n_traces, F fn) {
  int64_t calls = 0;
  for (int32_t t = 0; t < n_traces; ++t) calls += traces[t].n_calls;
  const int64_t hw = std::max<int64_t>(1, std::thread::hardware_concurrency());
  const int nt = (int)std::min<int64_t>({16, hw, (int64_t)n_traces, calls / 200000 + 1});
  if (nt <= 1) {
    for (int32_t t = 0; t < n_traces; ++t) fn(t);
    return;
  }
  std::atomic<int32_t> next{0};
  std::mutex m;
  std::exception_ptr first;  // the first exception a worker met, thrown again below
  auto work = [&]() {
    try {
      for (int32_t t; (t = next.fetch_add(1)) < n_traces;) fn(t);
    } catch (...) {
      std::lock_guard<std::mutex> lock(m);
      if (!first) first = std::current_exception();
      next = n_traces;  // the others stop at their next trace
    }
  };
  std::vector<std::thread> pool;
  pool.reserve((size_t)nt - 1);  // any allocation failure comes before a thread starts
  for (int i = 1; i < nt; ++i) {
    try {
      pool.emplace_back(work);
    } catch (const std::system_error&) {
      break;  // fewer threads than asked for: those started and this one share the traces
    }
  }
  work();
  for (std::thread& th : pool) th.join();
  if (first) std::rethrow_exception(first);
}

// validate_trace over every trace, in parallel; the lowest-numbered failing
// trace's status and message are reported, as a loop in order would.
int validate_traces(const hx_trace* traces, int32_t n_traces, const hx_cluster* c, int64_t min_prefill,
                    int64_t max_decode) {
  std::vector<int> rc((size_t)n_traces, HX_OK);
  std::vector<std::string> msg((size_t)n_traces);
  for_each_trace(traces, n_traces, [&](int32_t t) {
    rc[t] = validate_trace(&traces[t], t, c, min_prefill, max_decode);
    if (rc[t] != HX_OK) msg[t] = g_err;  // this thread's message
  });
  for (int32_t t = 0; t < n_traces; ++t)
    if (rc[t] != HX_OK) return fail(rc[t], msg[t]);
  return HX_OK;
}

template <class T>
int upload(T* dst, const T* src, int64_t count, cudaStream_t s) {
  if (count <= 0) return HX_OK;
  HX_CUDA(cudaMemcpyAsync(dst, src, (size_t)count * sizeof(T), cudaMemcpyHostToDevice, s));
  return HX_OK;
}

// Top-K size of each (trace, tenant) for the per-tenant P95: n_t - ceil(0.95 n_t) + 1
// over the tenant's n_t queries (0 without queries); at most the trace's own K.
std::vector<int32_t> tenant_kcaps(const hx_trace* traces, int32_t n_traces) {
  std::vector<int32_t> k((size_t)n_traces * HX_MAX_TENANTS, 0);
  for (int t = 0; t < n_traces; ++t) {
    int32_t n[HX_MAX_TENANTS] = {0, 0, 0, 0};
    for (int32_t i = 0; i < traces[t].n_queries; ++i) n[traces[t].tenant ? traces[t].tenant[i] : 0]++;
    for (int u = 0; u < HX_MAX_TENANTS; ++u)
      k[(size_t)t * HX_MAX_TENANTS + u] = n[u] ? n[u] - (95 * n[u] + 99) / 100 + 1 : 0;
  }
  return k;
}

// Copies the per-call and per-query trace arrays of all traces to the device.
int upload_traces(hx_sim* h, const hx_trace* traces, cudaStream_t s) {
  std::vector<int64_t> arrival((size_t)h->n_q), qcall((size_t)h->n_q + 1);
  std::vector<uint8_t> kq((size_t)h->n_q), tenant((size_t)h->n_q, 0);
  std::vector<int64_t> q0((size_t)h->n_traces + 1, 0), c0((size_t)h->n_traces + 1, 0);
  for (int t = 0; t < h->n_traces; ++t) {
    q0[t + 1] = q0[t] + traces[t].n_queries;
    c0[t + 1] = c0[t] + traces[t].n_calls;
  }
  for_each_trace(traces, h->n_traces, [&](int32_t t) {
    const hx_trace& tr = traces[t];
    const int64_t qo = q0[t], co = c0[t];
    for (int32_t i = 0; i < tr.n_queries; ++i) {
      arrival[qo + i] = tr.arrival_us[i];
      kq[qo + i] = tr.k[i];
      qcall[qo + i] = co + tr.call_base[i];
      if (tr.tenant) tenant[qo + i] = tr.tenant[i];
    }
  });
  int64_t co = c0[h->n_traces];
  qcall[h->n_q] = co;
  int rc;
  if ((rc = upload(h->d_arrival, arrival.data(), h->n_q, s)) || (rc = upload(h->d_k, kq.data(), h->n_q, s)) ||
      (rc = upload(h->d_tenant, tenant.data(), h->n_q, s)) || (rc = upload(h->d_qcall, qcall.data(), h->n_q + 1, s)))
    return rc;
  co = 0;
  for (int t = 0; t < h->n_traces; ++t) {
    const hx_trace& tr = traces[t];
    if ((rc = upload(h->d_prompt + co, tr.prompt, tr.n_calls, s)) || (rc = upload(h->d_out + co, tr.out, tr.n_calls, s)) ||
        (rc = upload(h->d_out_est + co, tr.out_est, tr.n_calls, s)) ||
        (rc = upload(h->d_stage + co, tr.stage, tr.n_calls, s)) || (rc = upload(h->d_cand + co, tr.cand, tr.n_calls, s)) ||
        (rc = upload(h->d_retry + co, tr.retry, tr.n_calls, s)))
      return rc;
    co += tr.n_calls;
  }
  std::vector<int32_t> kcap;
  if (h->d_tenant_kcap) {
    kcap = tenant_kcaps(traces, h->n_traces);
    if ((rc = upload(h->d_tenant_kcap, kcap.data(), (int64_t)kcap.size(), s))) return rc;
  }
  // the host staging vectors die here: the copies must finish first
  HX_CUDA(cudaStreamSynchronize(s));
  return HX_OK;
}

// WarpShared with its trailing slot array sized for the cluster (and one
// fail flag per slot when the cluster has fault windows)
int per_warp_smem(int total_slots, bool faults) {
  const int64_t ts = std::max(total_slots, 1);
  return (int)align_up((int64_t)offsetof(hx::WarpShared, slot) + 8 * ts + (faults ? ts : 0), 16);
}

// Kernel-parameter copy of a validated cluster.
void fill_cluster(const hx_cluster* cluster, hx::ClusterK& ck) {
  ck = hx::ClusterK{};
  ck.n_inst = cluster->n_inst;
  ck.n_types = cluster->n_types;
  ck.ref_type = cluster->ref_type;
  ck.rmax = cluster->rmax;
  ck.slo_mult_fp = cluster->slo_mult_fp;
  for (int t = 0; t < HX_MAX_TYPES; ++t) {
    const bool on = t < cluster->n_types;
    ck.prefill[t] = on ? cluster->prefill_tok_s[t] : 1;
    ck.decode[t] = on ? cluster->decode_us_tok[t] : 0;
    ck.slots[t] = on ? cluster->slots[t] : 0;
    ck.cnt[t] = 0;
  }
  for (int s = 0; s < 4; ++s) {
    ck.ref_prompt[s] = cluster->stage_ref_prompt[s];
    ck.ref_out[s] = cluster->stage_ref_out[s];
  }
  int base = 0;
  for (int m = 0; m < HX_MAX_INST; ++m) {
    const bool on = m < cluster->n_inst;
    const int ty = on ? cluster->inst_type[m] : 0;
    ck.inst_type[m] = (uint8_t)ty;
    ck.inst_slots[m] = on ? (uint8_t)cluster->slots[ty] : 0;
    ck.slot_base[m] = (uint16_t)base;
    if (on) {
      base += cluster->slots[ty];
      ck.cnt[ty]++;
    }
  }
  ck.total_slots = base;
  // per-tenant SLO multipliers replace slo_mult_fp when given
  ck.n_tenants = std::max(cluster->n_tenants, 1);
  for (int t = 0; t < HX_MAX_TENANTS; ++t)
    ck.tenant_mult[t] = (cluster->tenant_slo_mult_fp && t < ck.n_tenants) ? cluster->tenant_slo_mult_fp[t]
                                                                          : cluster->slo_mult_fp;
  ck.timeout_mult_fp = cluster->timeout_mult_fp;
  ck.n_faults = cluster->n_faults;
  for (int f = 0; f < cluster->n_faults; ++f) {
    const hx_fault& F = cluster->faults[f];
    ck.faults[f].t0 = F.t0_us;
    ck.faults[f].t1 = F.t1_us;
    ck.faults[f].slow = F.slow_fp;
    ck.faults[f].inst = F.inst;
    ck.faults[f].pad = 0;
  }
  ck.smem_per_warp = per_warp_smem(base, cluster->n_faults > 0);
}

// The simulations of opt->sim_subset, checked (in range, distinct) and sorted
// into the kernel's work order: trace-major, highest point first.
int order_subset(const hx_options* opt, int32_t n_traces, int32_t n_points, std::vector<int64_t>* out) {
  out->clear();
  if (!opt || opt->n_subset == 0) return HX_OK;
  if (opt->n_subset < 0) return fail(HX_ERR_INVALID, "n_subset < 0");
  if (!opt->sim_subset) return fail(HX_ERR_INVALID, "sim_subset is NULL");
  const int64_t n_sims = (int64_t)n_traces * n_points;
  std::vector<int64_t> w((size_t)opt->n_subset);
  for (int32_t i = 0; i < opt->n_subset; ++i) {
    const int64_t s = opt->sim_subset[i];
    if (s < 0 || s >= n_sims)
      return fail(HX_ERR_INVALID, "sim_subset[" + std::to_string(i) + "] = " + std::to_string(s) + " is out of range");
    const int64_t t = s / n_points, p = s - t * n_points;
    w[i] = t * n_points + (n_points - 1 - p);
  }
  std::sort(w.begin(), w.end());
  for (size_t i = 1; i < w.size(); ++i)
    if (w[i] == w[i - 1]) return fail(HX_ERR_INVALID, "sim_subset lists a simulation twice");
  out->resize(w.size());
  for (size_t i = 0; i < w.size(); ++i) {
    const int64_t t = w[i] / n_points;
    (*out)[i] = t * n_points + (n_points - 1 - (w[i] - t * n_points));
  }
  return HX_OK;
}

// Work order for a whole grid when it pays to change the default one.  The
// kernel takes simulations trace-major (the warps on one trace share its
// records in L2), highest point first within a trace.  A simulation whose
// points dispatch workload-balanced at alpha = 1 sends every request to the
// fastest instance and builds the longest local queue, so it costs more per
// event than any other point, and trace-major order starts the last traces'
// such simulations in the last wave, where they set the end of the run.  If
// the run is at most four waves of warps deep and every trace's records fit
// in L2 together, all traces' alpha = 1 points go first (hx_info.work_order
// 2); otherwise the traces of about the last two waves take theirs first,
// the others staying trace-major (3).  *order is left empty, and 0 returned,
// when the default stands.  Results do not depend on the order.
int costliest_first(const hx_grid* grid, int32_t n_traces, int64_t n_calls, int64_t l2_bytes,
                    int64_t resident_warps, std::vector<int64_t>* order) {
  order->clear();
  const int32_t P = grid->n_points;
  const int64_t n_sims = (int64_t)n_traces * P;
  // a list longer than 2^24 entries (128 MiB) is not worth its device memory
  if (n_sims <= resident_warps || n_sims > (int64_t(1) << 24)) return 0;
  std::vector<int32_t> hot, cold;
  for (int32_t p = P - 1; p >= 0; --p)
    (grid->alpha_fp[p] == hx::kScale && grid->dispatch_policy[p] == HX_DISPATCH_WB ? hot : cold).push_back(p);
  if (hot.empty() || cold.empty()) return 0;
  int32_t t0 = 0;  // traces before t0 keep the default order
  if (n_sims > 4 * resident_warps || n_calls * (int64_t)sizeof(hx::CallRec) > l2_bytes) {
    const int64_t k = (2 * resident_warps + P - 1) / P;
    if (k >= n_traces) return 0;
    t0 = n_traces - (int32_t)k;
  }
  order->reserve((size_t)n_sims);
  for (int32_t t = 0; t < t0; ++t)
    for (int32_t p = P - 1; p >= 0; --p) order->push_back((int64_t)t * P + p);
  for (const std::vector<int32_t>* part : {&hot, &cold})
    for (int32_t t = t0; t < n_traces; ++t)
      for (int32_t p : *part) order->push_back((int64_t)t * P + p);
  return t0 == 0 ? 2 : 3;
}

}  // namespace

extern "C" {

const char* hx_last_error(void) { return g_err.c_str(); }

static int hx_sim_create_impl(const hx_trace* traces, int32_t n_traces, const hx_cluster* cluster, const hx_grid* grid,
                              const hx_options* opt, hx_sim** out) {
  NvtxRange range("hx_sim_create");
  if (!out) return fail(HX_ERR_INVALID, "out is NULL");
  *out = nullptr;
  g_err.clear();
  if (!traces || n_traces < 1) return fail(HX_ERR_INVALID, "need at least one trace");
  int64_t min_prefill = 0, max_decode = 0;
  int rc;
  if ((rc = validate_cluster(cluster, &min_prefill, &max_decode))) return rc;
  if ((rc = validate_grid(grid))) return rc;
  if ((rc = validate_traces(traces, n_traces, cluster, min_prefill, max_decode))) return rc;
  if (opt && opt->n_record < 0) return fail(HX_ERR_INVALID, "n_record < 0");
  if (opt && opt->n_record > 0) {
    if (!opt->record_sims) return fail(HX_ERR_INVALID, "record_sims is NULL");
    std::vector<int32_t> sorted(opt->record_sims, opt->record_sims + opt->n_record);
    std::sort(sorted.begin(), sorted.end());
    const int64_t n_sims = (int64_t)n_traces * grid->n_points;
    for (size_t j = 0; j < sorted.size(); ++j)
      if (sorted[j] < 0 || sorted[j] >= n_sims || (j > 0 && sorted[j] == sorted[j - 1]))
        return fail(HX_ERR_INVALID, "record_sims must be distinct valid sim indices");
  }
  if (opt && opt->checked != 0 && opt->checked != 1) return fail(HX_ERR_INVALID, "checked must be 0 or 1");
  if (opt && opt->arena_entries < 0) return fail(HX_ERR_INVALID, "arena_entries < 0");
  std::vector<int64_t> subset;
  if ((rc = order_subset(opt, n_traces, grid->n_points, &subset))) return rc;

  // the handle is freed on every early return (and exception) until it is handed out
  std::unique_ptr<hx_sim> owner(new (std::nothrow) hx_sim());
  hx_sim* h = owner.get();
  if (!h) return fail(HX_ERR_OOM, "host allocation failed");
  auto bail = [](int code) { return code; };
  h->n_traces = n_traces;
  h->n_points = grid->n_points;
  h->n_sims = (int64_t)n_traces * grid->n_points;
  std::vector<int64_t> q_off(n_traces + 1, 0), c_off(n_traces + 1, 0);
  for (int t = 0; t < n_traces; ++t) {
    const int32_t nq = traces[t].n_queries, nc = traces[t].n_calls;
    h->h_nq.push_back(nq);
    h->h_nc.push_back(nc);
    q_off[t + 1] = q_off[t] + nq;
    c_off[t + 1] = c_off[t] + nc;
    h->max_nq = std::max(h->max_nq, nq);
    h->max_nc = std::max(h->max_nc, nc);
    h->max_kcap = std::max(h->max_kcap, nq - (95 * nq + 99) / 100 + 1);
  }
  h->n_q = q_off[n_traces];
  h->n_c = c_off[n_traces];
  h->n_work = subset.empty() ? h->n_sims : (int64_t)subset.size();
  h->checked = opt && opt->checked == 1;
  if (h->n_c >= (int64_t(1) << 31)) return bail(fail(HX_ERR_INVALID, "more than 2^31 calls in total"));

  // cluster constants (kernel parameter)
  hx::ClusterK& ck = h->ck;
  fill_cluster(cluster, ck);
  h->n_tenants = cluster->n_tenants;
  h->faults.assign(cluster->faults, cluster->faults + cluster->n_faults);

  int dev = 0;
  cudaDeviceProp prop;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaGetDeviceProperties(&prop, dev) != cudaSuccess) {
    cudaGetLastError();
    return bail(fail(HX_ERR_CUDA, "no CUDA device"));
  }
  // device inputs
  if ((rc = h->alloc(&h->d_arrival, h->n_q)) || (rc = h->alloc(&h->d_k, h->n_q)) ||
      (rc = h->alloc(&h->d_tenant, h->n_q)) ||
      (rc = h->alloc(&h->d_qcall, h->n_q + 1)) || (rc = h->alloc(&h->d_q_off, n_traces + 1)) ||
      (rc = h->alloc(&h->d_c_off, n_traces + 1)) || (rc = h->alloc(&h->d_prompt, h->n_c)) ||
      (rc = h->alloc(&h->d_out, h->n_c)) || (rc = h->alloc(&h->d_out_est, h->n_c)) ||
      (rc = h->alloc(&h->d_stage, h->n_c)) || (rc = h->alloc(&h->d_cand, h->n_c)) ||
      (rc = h->alloc(&h->d_retry, h->n_c)) || (rc = h->alloc(&h->d_alpha, h->n_points)) ||
      (rc = h->alloc(&h->d_gamma, h->n_points)) || (rc = h->alloc(&h->d_beta, h->n_points)) ||
      (rc = h->alloc(&h->d_rho, h->n_points)) || (rc = h->alloc(&h->d_lp, h->n_points)) ||
      (rc = h->alloc(&h->d_dp, h->n_points)) || (rc = h->alloc(&h->d_rec, h->n_c)) ||
      (rc = h->alloc(&h->d_results, h->n_sims)) || (rc = h->alloc(&h->d_counter, 1)) ||
      (rc = h->alloc(&h->d_best_trace, 2 * (int64_t)n_traces)) || (rc = h->alloc(&h->d_best_global, 2)) ||
      (rc = h->alloc(&h->d_point_sums, 3 * (int64_t)h->n_points)))
    return bail(rc);
  cudaStream_t s0 = nullptr;
  if ((rc = upload_traces(h, traces, s0)) || (rc = upload(h->d_q_off, q_off.data(), n_traces + 1, s0)) ||
      (rc = upload(h->d_c_off, c_off.data(), n_traces + 1, s0)) ||
      (rc = upload(h->d_alpha, grid->alpha_fp, h->n_points, s0)) ||
      (rc = upload(h->d_gamma, grid->gamma_fp, h->n_points, s0)) ||
      (rc = upload(h->d_beta, grid->beta_us2, h->n_points, s0)) || (rc = upload(h->d_rho, grid->rho, h->n_points, s0)) ||
      (rc = upload(h->d_lp, grid->local_policy, h->n_points, s0)) ||
      (rc = upload(h->d_dp, grid->dispatch_policy, h->n_points, s0)))
    return bail(rc);

  h->generic = needs_generic(grid, ck, opt && opt->n_record > 0, opt && opt->force_generic, h->checked);
  const void* kfn = h->generic ? (const void*)hx::hx_sim_kernel : (const void*)hx::hx_sim_kernel_lean;
  // launch shape of the simulation kernel and its per-warp scratch
  h->smem_per_block = hx::kWarpsPerBlock * ck.smem_per_warp;
  if ((rc = ensure_dyn_smem(h->generic, h->smem_per_block))) return bail(rc);
  int bps = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&bps, kfn, hx::kWarpsPerBlock * 32, h->smem_per_block) !=
          cudaSuccess ||
      bps < 1) {
    cudaGetLastError();
    return bail(fail(HX_ERR_CUDA, "simulation kernel does not fit on an SM"));
  }
  int64_t blocks = (int64_t)bps * prop.multiProcessorCount;
  if (opt && opt->max_resident_warps > 0)
    blocks = std::min<int64_t>(blocks, std::max<int64_t>(1, opt->max_resident_warps / hx::kWarpsPerBlock));
  blocks = std::min<int64_t>(blocks, (h->n_sims + hx::kWarpsPerBlock - 1) / hx::kWarpsPerBlock);
  h->blocks = (int)std::max<int64_t>(blocks, 1);
  h->resident_warps = h->blocks * hx::kWarpsPerBlock;
  // the simulations' order: the caller's subset, else possibly the costliest first
  h->work_order = subset.empty()
                      ? costliest_first(grid, n_traces, h->n_c, (int64_t)prop.l2CacheSize, h->resident_warps, &subset)
                      : 1;
  if (!subset.empty() && ((rc = h->alloc(&h->d_subset, (int64_t)subset.size())) ||
                          (rc = upload(h->d_subset, subset.data(), (int64_t)subset.size(), s0))))
    return bail(rc);
  // heap arena: doubling regions of 16, 32, ... entries per instance total at
  // most 4 * (requests ever queued) + 16 * instances
  h->arena_per_warp = 4 * (int64_t)h->max_nc + 16 * HX_MAX_INST;
  if (opt && opt->arena_entries > 0) h->arena_per_warp = opt->arena_entries;
  h->chains_per_warp = align_up(std::max(h->max_nq, 1), 256);
  h->topk_per_warp = align_up(h->max_kcap, 32);
  if (h->generic && ck.n_tenants > 1) {
    // one more heap per tenant after the simulation's own, each sized for a
    // whole trace (a tenant's K never exceeds its trace's), so uploads of new
    // tenant assignments need no reallocation
    for (int t = 0; t < HX_MAX_TENANTS; ++t) h->tenant_topk_off[t] = h->topk_per_warp * (1 + t);
    h->topk_per_warp *= 1 + HX_MAX_TENANTS;
    if ((rc = h->alloc(&h->d_tenant_kcap, (int64_t)n_traces * HX_MAX_TENANTS))) return bail(rc);
    const std::vector<int32_t> kcap = tenant_kcaps(traces, n_traces);
    if ((rc = upload(h->d_tenant_kcap, kcap.data(), (int64_t)kcap.size(), s0))) return bail(rc);
    if (cudaStreamSynchronize(s0) != cudaSuccess) return bail(fail(HX_ERR_CUDA, "tenant upload failed"));
  }
  const int64_t w = h->resident_warps;
  if ((rc = h->alloc(&h->d_arena, w * h->arena_per_warp)) || (rc = h->alloc(&h->d_chains, w * h->chains_per_warp)) ||
      (rc = h->alloc(&h->d_topk, w * h->topk_per_warp)))
    return bail(rc);
  if (h->generic && (rc = h->alloc(&h->d_extras, h->n_sims))) return bail(rc);
  h->scratch_bytes = w * (h->arena_per_warp * (int64_t)sizeof(hx::HeapEnt) + h->chains_per_warp +
                          h->topk_per_warp * (int64_t)sizeof(int64_t));

  // per-call logs of selected simulations
  if (opt && opt->n_record > 0) {
    h->n_record = opt->n_record;
    h->rec_stride = std::max(h->max_nc, 1);
    std::vector<int32_t> map((size_t)h->n_sims, -1);
    for (int j = 0; j < opt->n_record; ++j) {
      const int32_t sim = opt->record_sims[j];  // checked above: distinct, in range
      map[sim] = j;
      h->record_sims.push_back(sim);
    }
    const int64_t n = (int64_t)h->n_record * h->rec_stride;
    if ((rc = h->alloc(&h->d_rec_map, h->n_sims)) || (rc = h->alloc(&h->d_rec_inst, n)) ||
        (rc = h->alloc(&h->d_rec_enq, n)) || (rc = h->alloc(&h->d_rec_budget, n)) ||
        (rc = h->alloc(&h->d_rec_start, n)) || (rc = h->alloc(&h->d_rec_end, n)) ||
        (rc = upload(h->d_rec_map, map.data(), h->n_sims, s0)))
      return bail(rc);
    if (cudaStreamSynchronize(s0) != cudaSuccess) return bail(fail(HX_ERR_CUDA, "record map upload failed"));
  }
  if (opt && opt->timing) {
    h->timing = true;
    h->ev.assign(4 * hx_sim::kTimedRuns, nullptr);
    for (auto& e : h->ev)
      if (cudaEventCreate(&e) != cudaSuccess) return bail(fail(HX_ERR_CUDA, "cudaEventCreate failed"));
  }
  if (cudaDeviceSynchronize() != cudaSuccess) return bail(fail(HX_ERR_CUDA, "upload failed"));
  *out = owner.release();
  return HX_OK;
}

static int hx_sim_upload_impl(hx_sim* h, const hx_trace* traces, int32_t n_traces, void* stream) {
  NvtxRange range("hx_sim_upload");
  if (!h || !traces) return fail(HX_ERR_INVALID, "NULL argument");
  if (n_traces != h->n_traces) return fail(HX_ERR_INVALID, "trace count differs from the handle's");
  for (int t = 0; t < n_traces; ++t)
    if (traces[t].n_queries != h->h_nq[t] || traces[t].n_calls != h->h_nc[t])
      return fail(HX_ERR_INVALID, "trace shapes differ from the handle's");
  // same validation as create, against the handle's cluster bounds
  int64_t min_prefill = INT64_MAX, max_decode = 0;
  for (int t = 0; t < h->ck.n_types; ++t) {
    min_prefill = std::min<int64_t>(min_prefill, h->ck.prefill[t]);
    max_decode = std::max<int64_t>(max_decode, h->ck.decode[t]);
  }
  hx_cluster c{};
  c.rmax = h->ck.rmax;
  c.n_inst = h->ck.n_inst;
  c.n_tenants = h->n_tenants;
  c.timeout_mult_fp = h->ck.timeout_mult_fp;
  c.n_faults = (int32_t)h->faults.size();
  c.faults = h->faults.data();
  int rc = validate_traces(traces, n_traces, &c, min_prefill, max_decode);
  if (rc) return rc;
  return upload_traces(h, traces, static_cast<cudaStream_t>(stream));
}

static int hx_sim_run_impl(hx_sim* h, void* stream) {
  NvtxRange range("hx_sim_run");
  if (!h) return fail(HX_ERR_INVALID, "handle is NULL");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  hx::PrepArgs pa;
  pa.arrival = h->d_arrival;
  pa.kq = h->d_k;
  pa.qcall = h->d_qcall;
  pa.q_off = h->d_q_off;
  pa.c_off = h->d_c_off;
  pa.prompt = h->d_prompt;
  pa.out = h->d_out;
  pa.out_est = h->d_out_est;
  pa.stage = h->d_stage;
  pa.cand = h->d_cand;
  pa.retry = h->d_retry;
  pa.tenant = h->d_tenant;
  pa.n_queries = h->n_q;
  pa.n_traces = h->n_traces;
  pa.rec = h->d_rec;
  pa.work_counter = h->d_counter;
  pa.skip_results = h->d_results;
  pa.skip_extras = h->d_extras;
  pa.n_skip = h->n_work < h->n_sims ? h->n_sims : 0;

  hx::SimArgs sa;
  sa.rec = h->d_rec;
  sa.arrival = h->d_arrival;
  sa.qcall = h->d_qcall;
  sa.q_off = h->d_q_off;
  sa.c_off = h->d_c_off;
  sa.alpha = h->d_alpha;
  sa.gamma = h->d_gamma;
  sa.rho = h->d_rho;
  sa.beta = h->d_beta;
  sa.lpol = h->d_lp;
  sa.dpol = h->d_dp;
  sa.n_points = h->n_points;
  sa.n_traces = h->n_traces;
  sa.n_sims = h->n_sims;
  sa.results = h->d_results;
  sa.work_counter = h->d_counter;
  sa.arena = h->d_arena;
  sa.arena_per_warp = h->arena_per_warp;
  sa.chains = h->d_chains;
  sa.chains_per_warp = h->chains_per_warp;
  sa.topk = h->d_topk;
  sa.topk_per_warp = h->topk_per_warp;
  sa.rec_map = h->d_rec_map;
  sa.rec_inst = h->d_rec_inst;
  sa.rec_enq = h->d_rec_enq;
  sa.rec_budget = h->d_rec_budget;
  sa.rec_start = h->d_rec_start;
  sa.rec_end = h->d_rec_end;
  sa.rec_stride = h->rec_stride;
  sa.extras = h->d_extras;
  sa.tenant_kcap = h->d_tenant_kcap;
  for (int t = 0; t < HX_MAX_TENANTS; ++t) sa.tenant_topk_off[t] = h->tenant_topk_off[t];
  sa.subset = h->d_subset;
  sa.n_work = h->n_work;
  sa.checked = h->checked ? 1 : 0;

  hx::BestArgs ba;
  ba.results = h->d_results;
  ba.q_off = h->d_q_off;
  ba.n_traces = h->n_traces;
  ba.n_points = h->n_points;
  ba.per_trace = h->d_best_trace;
  ba.global = h->d_best_global;
  ba.point_sums = h->d_point_sums;

  const int prep_blocks = (int)std::max<int64_t>(1, (h->n_q + 255) / 256);
  if (int rc = ensure_dyn_smem(h->generic, h->smem_per_block)) return rc;
  cudaEvent_t* ev = h->timing ? h->run_ev(h->runs) : nullptr;
  if (ev) HX_CUDA(cudaEventRecord(ev[0], s));
  hx::hx_prep_kernel<<<prep_blocks, 256, 0, s>>>(pa, h->ck);
  HX_CUDA(cudaGetLastError());
  if (ev) HX_CUDA(cudaEventRecord(ev[1], s));
  if (h->generic)
    hx::hx_sim_kernel<<<h->blocks, hx::kWarpsPerBlock * 32, h->smem_per_block, s>>>(sa, h->ck);
  else
    hx::hx_sim_kernel_lean<<<h->blocks, hx::kWarpsPerBlock * 32, h->smem_per_block, s>>>(sa, h->ck);
  HX_CUDA(cudaGetLastError());
  if (ev) HX_CUDA(cudaEventRecord(ev[2], s));
  hx::hx_best_kernel<<<h->n_traces + 1, 256, 0, s>>>(ba);
  HX_CUDA(cudaGetLastError());
  if (ev) HX_CUDA(cudaEventRecord(ev[3], s));
  h->last_stream = s;
  h->ran = true;
  h->runs++;
  return HX_OK;
}

static int hx_sim_results_impl(hx_sim* h, hx_result* host_out, size_t n) {
  NvtxRange range("hx_sim_results");
  if (!h || !host_out) return fail(HX_ERR_INVALID, "NULL argument");
  if (!h->ran) return fail(HX_ERR_STATE, "hx_sim_run has not been called");
  if ((int64_t)n > h->n_sims) return fail(HX_ERR_INVALID, "n exceeds the number of simulations");
  HX_CUDA(cudaStreamSynchronize(h->last_stream));
  HX_CUDA(cudaMemcpy(host_out, h->d_results, n * sizeof(hx_result), cudaMemcpyDeviceToHost));
  return HX_OK;
}

static int hx_sim_extras_impl(hx_sim* h, hx_extra* host_out, size_t n) {
  if (!h || !host_out) return fail(HX_ERR_INVALID, "NULL argument");
  if (!h->ran) return fail(HX_ERR_STATE, "hx_sim_run has not been called");
  if ((int64_t)n > h->n_sims) return fail(HX_ERR_INVALID, "n exceeds the number of simulations");
  HX_CUDA(cudaStreamSynchronize(h->last_stream));
  if (n == 0) return HX_OK;
  if (h->d_extras) {
    HX_CUDA(cudaMemcpy(host_out, h->d_extras, n * sizeof(hx_extra), cudaMemcpyDeviceToHost));
    return HX_OK;
  }
  // the lean kernel serves one tenant without faults: everything is tenant 0
  std::vector<hx_result> res(n);
  HX_CUDA(cudaMemcpy(res.data(), h->d_results, n * sizeof(hx_result), cudaMemcpyDeviceToHost));
  for (size_t i = 0; i < n; ++i) {
    hx_extra e{};
    e.slo_met[0] = res[i].slo_met;
    e.n_done[0] = res[i].n_done;
    for (int t = 0; t < HX_MAX_TENANTS; ++t) e.p95_us[t] = res[i].status != HX_OK ? -1 : t == 0 ? res[i].p95_us : 0;
    host_out[i] = e;
  }
  return HX_OK;
}

static int hx_sim_best_impl(hx_sim* h, int32_t objective, hx_best* out) {
  if (!h || !out) return fail(HX_ERR_INVALID, "NULL argument");
  if (objective != HX_OBJ_P95 && objective != HX_OBJ_P95_SLO95) return fail(HX_ERR_INVALID, "unknown objective");
  if (!h->ran) return fail(HX_ERR_STATE, "hx_sim_run has not been called");
  HX_CUDA(cudaStreamSynchronize(h->last_stream));
  hx::BestCand g[2];
  HX_CUDA(cudaMemcpy(g, h->d_best_global, sizeof(g), cudaMemcpyDeviceToHost));
  const bool gv = g[objective].flags & 1;
  out->global_point = gv ? g[objective].p : -1;
  out->pad = 0;
  out->global_sum_p95 = gv ? g[objective].p95 : -1;
  out->global_slo_met = gv ? g[objective].slo : -1;
  if (out->per_trace_point) {
    std::vector<hx::BestCand> pt((size_t)2 * h->n_traces);
    HX_CUDA(cudaMemcpy(pt.data(), h->d_best_trace, pt.size() * sizeof(hx::BestCand), cudaMemcpyDeviceToHost));
    for (int t = 0; t < h->n_traces; ++t) {
      const hx::BestCand& b = pt[(size_t)2 * t + objective];
      out->per_trace_point[t] = (b.flags & 1) ? b.p : -1;
    }
  }
  return HX_OK;
}

static int hx_sim_point_sums_impl(hx_sim* h, int64_t* sum_p95, int64_t* sum_slo_met, int32_t* n_failed,
                                  size_t n_points) {
  if (!h || !sum_p95 || !sum_slo_met || !n_failed) return fail(HX_ERR_INVALID, "NULL argument");
  if (!h->ran) return fail(HX_ERR_STATE, "hx_sim_run has not been called");
  if ((int64_t)n_points != h->n_points) return fail(HX_ERR_INVALID, "n_points differs from the handle's");
  HX_CUDA(cudaStreamSynchronize(h->last_stream));
  std::vector<int64_t> v(3 * n_points);
  HX_CUDA(cudaMemcpy(v.data(), h->d_point_sums, v.size() * sizeof(int64_t), cudaMemcpyDeviceToHost));
  for (size_t p = 0; p < n_points; ++p) {
    sum_p95[p] = v[3 * p];
    sum_slo_met[p] = v[3 * p + 1];
    n_failed[p] = (int32_t)v[3 * p + 2];
  }
  return HX_OK;
}

static int hx_best_of_sums_impl(const int64_t* sum_p95, const int64_t* sum_slo_met, const int32_t* n_failed,
                                int32_t n_points, int64_t n_queries_total, int32_t objective, hx_best* out) {
  if (!sum_p95 || !sum_slo_met || !n_failed || !out) return fail(HX_ERR_INVALID, "NULL argument");
  if (n_points < 1 || n_queries_total < 0) return fail(HX_ERR_INVALID, "bad sizes");
  if (objective != HX_OBJ_P95 && objective != HX_OBJ_P95_SLO95) return fail(HX_ERR_INVALID, "unknown objective");
  // the summed table as one pseudo-trace, reduced by the same best-point kernel
  std::vector<hx_result> table((size_t)n_points);
  for (int32_t p = 0; p < n_points; ++p) {
    if (sum_slo_met[p] < 0 || sum_slo_met[p] > INT32_MAX) return fail(HX_ERR_INVALID, "SLO sums out of range");
    hx_result r{};
    r.p95_us = sum_p95[p];
    r.slo_met = (int32_t)sum_slo_met[p];
    r.status = n_failed[p] ? HX_ERR_CAPACITY : HX_OK;
    table[p] = r;
  }
  const int64_t qoff[2] = {0, n_queries_total};
  void* buf = nullptr;
  const size_t bytes = table.size() * sizeof(hx_result) + 2 * sizeof(int64_t) + 4 * sizeof(hx::BestCand);
  HX_CUDA(cudaMalloc(&buf, bytes));
  auto run = [&]() -> int {
    unsigned char* b = static_cast<unsigned char*>(buf);
    hx_result* d_res = reinterpret_cast<hx_result*>(b);
    int64_t* d_qoff = reinterpret_cast<int64_t*>(b + table.size() * sizeof(hx_result));
    hx::BestCand* d_cand = reinterpret_cast<hx::BestCand*>(d_qoff + 2);
    HX_CUDA(cudaMemcpy(d_res, table.data(), table.size() * sizeof(hx_result), cudaMemcpyHostToDevice));
    HX_CUDA(cudaMemcpy(d_qoff, qoff, sizeof(qoff), cudaMemcpyHostToDevice));
    hx::BestArgs ba;
    ba.results = d_res;
    ba.q_off = d_qoff;
    ba.n_traces = 1;
    ba.n_points = n_points;
    ba.per_trace = d_cand;
    ba.global = d_cand + 2;
    ba.point_sums = nullptr;
    hx::hx_best_kernel<<<2, 256>>>(ba);
    HX_CUDA(cudaGetLastError());
    hx::BestCand g[2];
    HX_CUDA(cudaMemcpy(g, d_cand + 2, sizeof(g), cudaMemcpyDeviceToHost));
    const bool v = g[objective].flags & 1;
    out->global_point = v ? g[objective].p : -1;
    out->pad = 0;
    out->global_sum_p95 = v ? g[objective].p95 : -1;
    out->global_slo_met = v ? g[objective].slo : -1;
    return HX_OK;
  };
  const int rc = run();
  cudaFree(buf);
  return rc;
}

static int hx_sim_records_impl(hx_sim* h, int32_t rec_index, int32_t* inst, int64_t* enq_us, int64_t* budget_us,
                               int64_t* start_us, int64_t* end_us, size_t n_calls) {
  if (!h) return fail(HX_ERR_INVALID, "handle is NULL");
  if (!h->ran) return fail(HX_ERR_STATE, "hx_sim_run has not been called");
  if (rec_index < 0 || rec_index >= h->n_record) return fail(HX_ERR_INVALID, "rec_index out of range");
  const int t = (int)(h->record_sims[rec_index] / h->n_points);
  if ((int64_t)n_calls != h->h_nc[t]) return fail(HX_ERR_INVALID, "n_calls differs from the trace's");
  HX_CUDA(cudaStreamSynchronize(h->last_stream));
  const int64_t o = (int64_t)rec_index * h->rec_stride;
  if (n_calls == 0) return HX_OK;
  if (inst) HX_CUDA(cudaMemcpy(inst, h->d_rec_inst + o, n_calls * sizeof(int32_t), cudaMemcpyDeviceToHost));
  if (enq_us) HX_CUDA(cudaMemcpy(enq_us, h->d_rec_enq + o, n_calls * sizeof(int64_t), cudaMemcpyDeviceToHost));
  if (budget_us) HX_CUDA(cudaMemcpy(budget_us, h->d_rec_budget + o, n_calls * sizeof(int64_t), cudaMemcpyDeviceToHost));
  if (start_us) HX_CUDA(cudaMemcpy(start_us, h->d_rec_start + o, n_calls * sizeof(int64_t), cudaMemcpyDeviceToHost));
  if (end_us) HX_CUDA(cudaMemcpy(end_us, h->d_rec_end + o, n_calls * sizeof(int64_t), cudaMemcpyDeviceToHost));
  return HX_OK;
}

static int hx_sim_prep_impl(hx_sim* h, int32_t trace_index, int32_t* est, int32_t* svc, int32_t* tbar,
                            int64_t* deadline_us, size_t n_calls) {
  if (!h) return fail(HX_ERR_INVALID, "handle is NULL");
  if (!h->ran) return fail(HX_ERR_STATE, "hx_sim_run has not been called");
  if (trace_index < 0 || trace_index >= h->n_traces) return fail(HX_ERR_INVALID, "trace_index out of range");
  if ((int64_t)n_calls != h->h_nc[trace_index]) return fail(HX_ERR_INVALID, "n_calls differs from the trace's");
  HX_CUDA(cudaStreamSynchronize(h->last_stream));
  if (n_calls == 0) return HX_OK;
  int64_t off = 0;
  for (int t = 0; t < trace_index; ++t) off += h->h_nc[t];
  std::vector<hx::CallRec> recs(n_calls);
  HX_CUDA(cudaMemcpy(recs.data(), h->d_rec + off, n_calls * sizeof(hx::CallRec), cudaMemcpyDeviceToHost));
  for (size_t j = 0; j < n_calls; ++j) {
    for (int ty = 0; ty < 4; ++ty) {
      if (est) est[4 * j + ty] = recs[j].ev[ty].x;
      if (svc) svc[4 * j + ty] = recs[j].ev[ty].y;
    }
    if (tbar) tbar[j] = recs[j].tbar;
    if (deadline_us) deadline_us[j] = recs[j].deadline;
  }
  return HX_OK;
}

int hx_sim_timings(hx_sim* h, float* prep_ms, float* sim_ms, float* best_ms) {
  return hx_sim_timings_back(h, 0, prep_ms, sim_ms, best_ms);
}

int hx_sim_timings_back(hx_sim* h, int32_t back, float* prep_ms, float* sim_ms, float* best_ms) {
  if (!h) return fail(HX_ERR_INVALID, "handle is NULL");
  if (!h->timing) return fail(HX_ERR_STATE, "created without opt.timing");
  if (!h->ran) return fail(HX_ERR_STATE, "hx_sim_run has not been called");
  if (back < 0 || back >= hx_sim::kTimedRuns || back >= h->runs)
    return fail(HX_ERR_INVALID, "back must be 0 .. min(runs, " + std::to_string(hx_sim::kTimedRuns) + ") - 1");
  cudaEvent_t* ev = h->run_ev(h->runs - 1 - back);
  HX_CUDA(cudaEventSynchronize(ev[3]));
  float a = 0, b = 0, c = 0;
  HX_CUDA(cudaEventElapsedTime(&a, ev[0], ev[1]));
  HX_CUDA(cudaEventElapsedTime(&b, ev[1], ev[2]));
  HX_CUDA(cudaEventElapsedTime(&c, ev[2], ev[3]));
  if (prep_ms) *prep_ms = a;
  if (sim_ms) *sim_ms = b;
  if (best_ms) *best_ms = c;
  return HX_OK;
}

int hx_selftest_div(const uint64_t* n, const uint64_t* d, uint64_t* q, uint64_t* q_ref, size_t count) {
  if (!n || !d || !q || !q_ref) return fail(HX_ERR_INVALID, "NULL argument");
  for (size_t i = 0; i < count; ++i)
    if (n[i] >= (uint64_t(1) << 63) || d[i] < 1 || d[i] >= (uint64_t(1) << 54))
      return fail(HX_ERR_INVALID, "operands must satisfy n < 2^63 and 1 <= d < 2^54");
  if (count == 0) return HX_OK;
  uint64_t* buf = nullptr;
  HX_CUDA(cudaMalloc(&buf, 4 * count * sizeof(uint64_t)));
  auto run = [&]() -> int {
    HX_CUDA(cudaMemcpy(buf, n, count * 8, cudaMemcpyHostToDevice));
    HX_CUDA(cudaMemcpy(buf + count, d, count * 8, cudaMemcpyHostToDevice));
    hx::hx_selftest_div_kernel<<<(unsigned)((count + 255) / 256), 256>>>(buf, buf + count, buf + 2 * count,
                                                                         buf + 3 * count, (int64_t)count);
    HX_CUDA(cudaGetLastError());
    HX_CUDA(cudaMemcpy(q, buf + 2 * count, count * 8, cudaMemcpyDeviceToHost));
    HX_CUDA(cudaMemcpy(q_ref, buf + 3 * count, count * 8, cudaMemcpyDeviceToHost));
    return HX_OK;
  };
  const int rc = run();
  cudaFree(buf);
  return rc;
}

int hx_sim_info(hx_sim* h, hx_info* out) {
  if (!h || !out) return fail(HX_ERR_INVALID, "NULL argument");
  out->n_sims = h->n_sims;
  out->n_calls_total = h->n_c;
  out->n_queries_total = h->n_q;
  out->scratch_bytes = h->scratch_bytes;
  out->device_bytes = h->device_bytes;
  out->resident_warps = h->resident_warps;
  out->warps_per_block = hx::kWarpsPerBlock;
  out->blocks = h->blocks;
  out->smem_per_block = h->smem_per_block;
  out->generic_kernel = h->generic ? 1 : 0;
  out->work_order = h->work_order;
  return HX_OK;
}

int hx_sim_destroy(hx_sim* h) {
  if (!h) return HX_OK;
  if (h->ran && h->last_stream) cudaStreamSynchronize(h->last_stream);
  cudaDeviceSynchronize();
  delete h;
  return HX_OK;
}

}  // extern "C"

// ---------------------------------------------------------------------------
// hx_sim_run_static: the whole path for one trace without allocating memory.
//
// For callers that may not allocate device memory -- code running where
// cudaMalloc is forbidden or unavailable (a host process that only owns
// pre-arranged memory, a plugin whose host application controls every
// allocation, a latency-critical loop that must not hit the allocator) -- this
// entry point runs the same preparation, simulation and best-point kernels as
// hx_sim_run, but every intermediate buffer (the copied inputs, the per-call
// records, the per-warp heap arenas, the results) is carved from one
// file-scope device array of HX_STATIC_SCRATCH_BYTES.  That array exists on
// every GPU that loads this library, for as long as the library stays loaded.
namespace {

__device__ __align__(256) unsigned char hx_static_scratch[HX_STATIC_SCRATCH_BYTES];

std::mutex g_static_mu;
unsigned char* g_static_base[kMaxDevices] = {};

// Device address of hx_static_scratch on the current device (the host-side
// symbol is only a stand-in and must never be passed to a kernel).  It is
// looked up again on every call made while `s` is not capturing, so a
// device reset between calls cannot leave a stale address behind; a call
// made during stream capture uses the address of the last earlier call on
// this device, and fails if there was none.
int static_base(cudaStream_t s, unsigned char** out) {
  int dev = 0;
  HX_CUDA(cudaGetDevice(&dev));
  if (dev < 0 || dev >= kMaxDevices) return fail(HX_ERR_INVALID, "device index out of range");
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  HX_CUDA(cudaStreamIsCapturing(s, &cap));
  std::lock_guard<std::mutex> lock(g_static_mu);
  if (cap == cudaStreamCaptureStatusNone) {
    void* p = nullptr;
    HX_CUDA(cudaGetSymbolAddress(&p, hx_static_scratch));
    g_static_base[dev] = static_cast<unsigned char*>(p);
  } else if (!g_static_base[dev]) {
    return fail(HX_ERR_STATE, "the first hx_sim_run_static call on a device must come before any stream capture");
  }
  *out = g_static_base[dev];
  return HX_OK;
}

__global__ void hx_widen_kernel(const int32_t* src, int64_t* dst, int64_t n) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) dst[i] = src[i];
}

// Bump carving of the static array; offsets are 256-byte aligned.
struct Carve {
  int64_t used = 0;
  template <class T>
  int64_t take(int64_t count) {
    const int64_t off = used;
    used = align_up(used + std::max<int64_t>(count, 1) * (int64_t)sizeof(T), 256);
    return off;
  }
};

}  // namespace

static int hx_sim_run_static_impl(const hx_trace* trace, const hx_cluster* cluster, const hx_grid* grid,
                                  int32_t objective, hx_result* results, hx_best* best, void* stream) {
  g_err.clear();
  if (!trace || !results) return fail(HX_ERR_INVALID, "trace and results must not be NULL");
  if (objective != HX_OBJ_P95 && objective != HX_OBJ_P95_SLO95) return fail(HX_ERR_INVALID, "unknown objective");
  int64_t min_prefill = 0, max_decode = 0;
  int rc;
  if ((rc = validate_cluster(cluster, &min_prefill, &max_decode))) return rc;
  if ((rc = validate_grid(grid))) return rc;
  if ((rc = validate_trace(trace, 0, cluster, min_prefill, max_decode))) return rc;
  const int64_t nq = trace->n_queries, nc = trace->n_calls, P = grid->n_points;
  cudaStream_t s = static_cast<cudaStream_t>(stream);

  hx::ClusterK ck;
  fill_cluster(cluster, ck);

  // layout of the static array: inputs, records, results, then per-warp scratch
  Carve cv;
  const int64_t o_qoff = cv.take<int64_t>(2), o_coff = cv.take<int64_t>(2), o_ctr = cv.take<unsigned long long>(1);
  const int64_t o_arr = cv.take<int64_t>(nq), o_k = cv.take<uint8_t>(nq), o_cb32 = cv.take<int32_t>(nq + 1);
  const int64_t o_ten = cv.take<uint8_t>(nq);
  const int64_t o_qcall = cv.take<int64_t>(nq + 1);
  const int64_t o_prompt = cv.take<int32_t>(nc), o_out = cv.take<int32_t>(nc), o_oest = cv.take<int32_t>(nc);
  const int64_t o_stage = cv.take<uint8_t>(nc), o_cand = cv.take<uint8_t>(nc), o_retry = cv.take<uint8_t>(nc);
  const int64_t o_alpha = cv.take<int64_t>(P), o_gamma = cv.take<int64_t>(P), o_beta = cv.take<int64_t>(P);
  const int64_t o_rho = cv.take<int32_t>(P), o_lp = cv.take<uint8_t>(P), o_dp = cv.take<uint8_t>(P);
  const int64_t o_rec = cv.take<hx::CallRec>(nc), o_res = cv.take<hx_result>(P);
  const int64_t o_bt = cv.take<hx::BestCand>(2), o_bg = cv.take<hx::BestCand>(2);
  const int64_t fixed = cv.used;
  const int32_t kcap = (int32_t)(nq - (95 * nq + 99) / 100 + 1);
  const int64_t arena_per_warp = 4 * nc + 16 * HX_MAX_INST;
  const int64_t chains_per_warp = align_up(std::max<int64_t>(nq, 1), 256);
  const int64_t topk_per_warp = align_up(std::max<int32_t>(kcap, 1), 32);
  const int64_t per_warp = align_up(arena_per_warp * (int64_t)sizeof(hx::HeapEnt), 256) + chains_per_warp +
                           align_up(topk_per_warp * 8, 256);
  const int64_t room = (int64_t)HX_STATIC_SCRATCH_BYTES - fixed;
  const int64_t fit_warps = room > 0 ? room / per_warp : 0;
  if (fit_warps < hx::kWarpsPerBlock)
    return fail(HX_ERR_INVALID, "trace too large for the static scratch: it needs " +
                                    std::to_string(fixed + hx::kWarpsPerBlock * per_warp) + " bytes, the array holds " +
                                    std::to_string((int64_t)HX_STATIC_SCRATCH_BYTES));

  int dev = 0;
  cudaDeviceProp prop;
  HX_CUDA(cudaGetDevice(&dev));
  HX_CUDA(cudaGetDeviceProperties(&prop, dev));
  const int smem_per_block = hx::kWarpsPerBlock * ck.smem_per_warp;
  const bool generic = needs_generic(grid, ck, false, false, false);
  const void* kfn = generic ? (const void*)hx::hx_sim_kernel : (const void*)hx::hx_sim_kernel_lean;
  if ((rc = ensure_dyn_smem(generic, smem_per_block))) return rc;
  int bps = 0;
  HX_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&bps, kfn, hx::kWarpsPerBlock * 32, smem_per_block));
  if (bps < 1) return fail(HX_ERR_CUDA, "simulation kernel does not fit on an SM");
  int64_t blocks = std::min<int64_t>((int64_t)bps * prop.multiProcessorCount, fit_warps / hx::kWarpsPerBlock);
  blocks = std::max<int64_t>(1, std::min<int64_t>(blocks, (P + hx::kWarpsPerBlock - 1) / hx::kWarpsPerBlock));
  const int64_t warps = blocks * hx::kWarpsPerBlock;
  const int64_t o_arena = fixed;
  const int64_t o_chains = o_arena + warps * align_up(arena_per_warp * (int64_t)sizeof(hx::HeapEnt), 256);
  const int64_t o_topk = o_chains + warps * chains_per_warp;

  unsigned char* sb = nullptr;
  if ((rc = static_base(s, &sb))) return rc;
  auto at = [&](int64_t off) { return static_cast<void*>(sb + off); };
  const int64_t offs[4] = {0, nq, 0, nc};
  HX_CUDA(cudaMemcpyAsync(at(o_qoff), offs, 2 * sizeof(int64_t), cudaMemcpyHostToDevice, s));
  HX_CUDA(cudaMemcpyAsync(at(o_coff), offs + 2, 2 * sizeof(int64_t), cudaMemcpyHostToDevice, s));
  struct Up {
    int64_t off;
    const void* src;
    int64_t bytes;
  } ups[] = {{o_arr, trace->arrival_us, nq * 8},     {o_k, trace->k, nq},
             {o_ten, trace->tenant, trace->tenant ? nq : 0},
             {o_cb32, trace->call_base, (nq + 1) * 4}, {o_prompt, trace->prompt, nc * 4},
             {o_out, trace->out, nc * 4},             {o_oest, trace->out_est, nc * 4},
             {o_stage, trace->stage, nc},             {o_cand, trace->cand, nc},
             {o_retry, trace->retry, nc},             {o_alpha, grid->alpha_fp, P * 8},
             {o_gamma, grid->gamma_fp, P * 8},        {o_beta, grid->beta_us2, P * 8},
             {o_rho, grid->rho, P * 4},               {o_lp, grid->local_policy, P},
             {o_dp, grid->dispatch_policy, P}};
  for (const Up& u : ups)
    if (u.bytes > 0) HX_CUDA(cudaMemcpyAsync(at(u.off), u.src, (size_t)u.bytes, cudaMemcpyHostToDevice, s));
  hx_widen_kernel<<<(unsigned)std::max<int64_t>(1, (nq + 1 + 255) / 256), 256, 0, s>>>(
      static_cast<const int32_t*>(at(o_cb32)), static_cast<int64_t*>(at(o_qcall)), nq + 1);
  HX_CUDA(cudaGetLastError());

  hx::PrepArgs pa;
  pa.arrival = static_cast<const int64_t*>(at(o_arr));
  pa.kq = static_cast<const uint8_t*>(at(o_k));
  pa.qcall = static_cast<const int64_t*>(at(o_qcall));
  pa.q_off = static_cast<const int64_t*>(at(o_qoff));
  pa.c_off = static_cast<const int64_t*>(at(o_coff));
  pa.prompt = static_cast<const int32_t*>(at(o_prompt));
  pa.out = static_cast<const int32_t*>(at(o_out));
  pa.out_est = static_cast<const int32_t*>(at(o_oest));
  pa.stage = static_cast<const uint8_t*>(at(o_stage));
  pa.cand = static_cast<const uint8_t*>(at(o_cand));
  pa.retry = static_cast<const uint8_t*>(at(o_retry));
  pa.tenant = trace->tenant ? static_cast<const uint8_t*>(at(o_ten)) : nullptr;
  pa.n_queries = nq;
  pa.n_traces = 1;
  pa.rec = static_cast<hx::CallRec*>(at(o_rec));
  pa.work_counter = static_cast<unsigned long long*>(at(o_ctr));  // zeroed by the prep kernel
  pa.skip_results = nullptr;
  pa.skip_extras = nullptr;
  pa.n_skip = 0;

  hx::SimArgs sa;
  sa.rec = pa.rec;
  sa.arrival = pa.arrival;
  sa.qcall = pa.qcall;
  sa.q_off = pa.q_off;
  sa.c_off = pa.c_off;
  sa.alpha = static_cast<const int64_t*>(at(o_alpha));
  sa.gamma = static_cast<const int64_t*>(at(o_gamma));
  sa.rho = static_cast<const int32_t*>(at(o_rho));
  sa.beta = static_cast<const int64_t*>(at(o_beta));
  sa.lpol = static_cast<const uint8_t*>(at(o_lp));
  sa.dpol = static_cast<const uint8_t*>(at(o_dp));
  sa.n_points = (int32_t)P;
  sa.n_traces = 1;
  sa.n_sims = P;
  sa.results = static_cast<hx_result*>(at(o_res));
  sa.work_counter = pa.work_counter;
  sa.arena = static_cast<hx::HeapEnt*>(at(o_arena));
  sa.arena_per_warp = align_up(arena_per_warp * (int64_t)sizeof(hx::HeapEnt), 256) / (int64_t)sizeof(hx::HeapEnt);
  sa.chains = static_cast<uint8_t*>(at(o_chains));
  sa.chains_per_warp = chains_per_warp;
  sa.topk = static_cast<int64_t*>(at(o_topk));
  sa.topk_per_warp = align_up(topk_per_warp * 8, 256) / 8;
  sa.rec_map = nullptr;
  sa.rec_inst = nullptr;
  sa.rec_enq = nullptr;
  sa.rec_budget = nullptr;
  sa.rec_start = nullptr;
  sa.rec_end = nullptr;
  sa.rec_stride = 0;
  sa.extras = nullptr;
  sa.tenant_kcap = nullptr;
  for (int t = 0; t < HX_MAX_TENANTS; ++t) sa.tenant_topk_off[t] = 0;
  sa.subset = nullptr;
  sa.n_work = P;
  sa.checked = 0;

  hx::BestArgs ba;
  ba.results = sa.results;
  ba.q_off = pa.q_off;
  ba.n_traces = 1;
  ba.n_points = (int32_t)P;
  ba.per_trace = static_cast<hx::BestCand*>(at(o_bt));
  ba.global = static_cast<hx::BestCand*>(at(o_bg));
  ba.point_sums = nullptr;

  hx::hx_prep_kernel<<<(unsigned)std::max<int64_t>(1, (nq + 255) / 256), 256, 0, s>>>(pa, ck);
  HX_CUDA(cudaGetLastError());
  if (generic)
    hx::hx_sim_kernel<<<(unsigned)blocks, hx::kWarpsPerBlock * 32, smem_per_block, s>>>(sa, ck);
  else
    hx::hx_sim_kernel_lean<<<(unsigned)blocks, hx::kWarpsPerBlock * 32, smem_per_block, s>>>(sa, ck);
  HX_CUDA(cudaGetLastError());
  hx::hx_best_kernel<<<2, 256, 0, s>>>(ba);
  HX_CUDA(cudaGetLastError());
  HX_CUDA(cudaMemcpyAsync(results, at(o_res), (size_t)P * sizeof(hx_result), cudaMemcpyDeviceToHost, s));
  hx::BestCand bg[2];
  HX_CUDA(cudaMemcpyAsync(bg, at(o_bg), sizeof(bg), cudaMemcpyDeviceToHost, s));
  HX_CUDA(cudaStreamSynchronize(s));
  if (best) {
    const bool v = bg[objective].flags & 1;
    best->global_point = v ? bg[objective].p : -1;
    best->pad = 0;
    best->global_sum_p95 = v ? bg[objective].p95 : -1;
    best->global_slo_met = v ? bg[objective].slo : -1;
    if (best->per_trace_point) best->per_trace_point[0] = best->global_point;
  }
  return HX_OK;
}

// The C entry points: each runs its implementation above under guarded(), so
// that no C++ exception crosses the ABI.
extern "C" {

int hx_sim_create(const hx_trace* traces, int32_t n_traces, const hx_cluster* cluster, const hx_grid* grid,
                  const hx_options* opt, hx_sim** out) {
  return guarded([&] { return hx_sim_create_impl(traces, n_traces, cluster, grid, opt, out); });
}

int hx_sim_upload(hx_sim* h, const hx_trace* traces, int32_t n_traces, void* stream) {
  return guarded([&] { return hx_sim_upload_impl(h, traces, n_traces, stream); });
}

int hx_sim_run(hx_sim* h, void* stream) {
  return guarded([&] { return hx_sim_run_impl(h, stream); });
}

int hx_sim_results(hx_sim* h, hx_result* host_out, size_t n) {
  return guarded([&] { return hx_sim_results_impl(h, host_out, n); });
}

int hx_sim_extras(hx_sim* h, hx_extra* host_out, size_t n) {
  return guarded([&] { return hx_sim_extras_impl(h, host_out, n); });
}

int hx_sim_best(hx_sim* h, int32_t objective, hx_best* out) {
  return guarded([&] { return hx_sim_best_impl(h, objective, out); });
}

int hx_sim_point_sums(hx_sim* h, int64_t* sum_p95, int64_t* sum_slo_met, int32_t* n_failed, size_t n_points) {
  return guarded([&] { return hx_sim_point_sums_impl(h, sum_p95, sum_slo_met, n_failed, n_points); });
}

int hx_best_of_sums(const int64_t* sum_p95, const int64_t* sum_slo_met, const int32_t* n_failed, int32_t n_points,
                    int64_t n_queries_total, int32_t objective, hx_best* out) {
  return guarded(
      [&] { return hx_best_of_sums_impl(sum_p95, sum_slo_met, n_failed, n_points, n_queries_total, objective, out); });
}

int hx_sim_records(hx_sim* h, int32_t rec_index, int32_t* inst, int64_t* enq_us, int64_t* budget_us,
                   int64_t* start_us, int64_t* end_us, size_t n_calls) {
  return guarded(
      [&] { return hx_sim_records_impl(h, rec_index, inst, enq_us, budget_us, start_us, end_us, n_calls); });
}

int hx_sim_prep(hx_sim* h, int32_t trace_index, int32_t* est, int32_t* svc, int32_t* tbar, int64_t* deadline_us,
                size_t n_calls) {
  return guarded([&] { return hx_sim_prep_impl(h, trace_index, est, svc, tbar, deadline_us, n_calls); });
}

int hx_sim_run_static(const hx_trace* trace, const hx_cluster* cluster, const hx_grid* grid,
                      int32_t objective, hx_result* results, hx_best* best, void* stream) {
  return guarded([&] { return hx_sim_run_static_impl(trace, cluster, grid, objective, results, best, stream); });
}

}  // extern "C"
