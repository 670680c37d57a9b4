"""Kernel variants: source edits of the simulation kernel, built beside the
library and timed against it on the same workload, each required to give
bit-identical results.  This is how the alternatives the design notes
mention were measured (GPU only).

    python -m tests.kernel_variants FAMILY [--traces 64] [--reps 3] [--out FILE]

Family `state`: the instance of each pending dispatch kept in shared memory
instead of on the entry's lane; the lane's instance types re-read at each
dispatch from the kernel parameters or from a shared copy.

Family `misc`: the next arrival in the next-event minimum; the digest
flush, or the top-K insert, inlined.

Family `layout`: a lane's two event keys and two cached rewards adjacent in
shared memory.

Family `heap`: the heap sift's move-up test taken from the reduced maximum
key.

Family `div`: the reward pass's division without its divergent early
return; a warp barrier after each simulation's per-lane initial state.

Family `cache`: the call-record loads with an L2 evict-last policy; the
heap sift's deeper child loads not allocated in L1, or evicted from it first.

Family `micro`: the event key formed with one shift and a mask; the
simulation's beta, beta as a float and 1 - alpha, or its alpha, kept in
registers instead of re-read from shared memory.

Family `occupancy`: 7 or 6 resident 4-warp blocks per SM instead of 8 (the
register budget follows), and the digest summed per lane in a register.

Family `prefetch`:
  arrival_l1 / arrival_l2  at a query's arrival, prefetch its call records
                           (up to 10 records, 5 lines of 128 bytes) into L1 / L2;
  start_l1 / start_l2      when a request is dispatched, prefetch the records
                           that follow its own (its successors) into L1 / L2.
Every prefetch stays inside the trace's records.
"""
from __future__ import annotations

import argparse
import json
import os
import shutil
import subprocess
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

CSRC = os.path.join(ROOT, "paper_2505_05286_gb300", "csrc")
OUT = os.path.join(ROOT, "paper_2505_05286_gb300", "_variants")
NVCC = ["nvcc", "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-lineinfo", "-std=c++17", "-Xcompiler",
        "-fPIC", "-I", os.path.join(ROOT, "include")]

_ARRIVAL = ("""        rel_first = (int32_t)(a.qcall[qbase + qa] - W->cb);""",
            """        rel_first = (int32_t)(a.qcall[qbase + qa] - W->cb);
        {
          const char* pa = reinterpret_cast<const char*>(rec + rel_first) + 128 * lane;
          if (lane < 5 && (int64_t)rel_first * 64 + 128 * lane < (int64_t)nc * 64)
            asm volatile("prefetch.global.LVL [%0];" ::"l"(pa));
        }""")
_START = ("""        HX_BOUND(rid < nc)
        const CallRec* r = rec + rid;""",
          """        HX_BOUND(rid < nc)
        const CallRec* r = rec + rid;
        {
          const char* pa = reinterpret_cast<const char*>(r + 1) + 128 * lane;
          if (lane < 4 && (int64_t)(rid + 1) * 64 + 128 * lane < (int64_t)nc * 64)
            asm volatile("prefetch.global.LVL [%0];" ::"l"(pa));
        }""")

# Each lane keeps the sum of the digest terms it hashes in a register; the
# warp adds the 32 partial sums once, when the simulation ends, instead of a
# shuffle reduction at every 16-term flush.
_DIGEST_LANES = [
    ("""__device__ __noinline__ void digest_flush(WarpShared* W, int n, int lane) {
  __syncwarp();
  const longlong2 e = W->dterm[lane < n ? lane : 0];
  uint64_t y = lane < n ? digest_term((uint64_t)e.x, (uint64_t)e.y) : 0ull;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) y += __shfl_xor_sync(kFull, y, o);
  if (lane == 0) W->digest += y;
  __syncwarp();
}""", """__device__ __noinline__ uint64_t digest_flush(WarpShared* W, int n, int lane) {
  __syncwarp();
  const longlong2 e = W->dterm[lane < n ? lane : 0];
  const uint64_t y = lane < n ? digest_term((uint64_t)e.x, (uint64_t)e.y) : 0ull;
  __syncwarp();
  return y;
}"""),
    ("""__device__ __forceinline__ void digest_push(WarpShared* W, int& dn, int64_t t, uint32_t tag, int lane) {""",
     """__device__ __forceinline__ void digest_push(WarpShared* W, int& dn, uint64_t& dacc, int64_t t, uint32_t tag,
                                            int lane) {"""),
    ("""    digest_flush(W, 16, lane);
    dn = 0;""", """    dacc += digest_flush(W, 16, lane);
    dn = 0;"""),
    ("""__device__ __forceinline__ void finish_query(WarpShared* W, int& dn, int32_t qid,""",
     """__device__ __forceinline__ void finish_query(WarpShared* W, int& dn, uint64_t& dacc, int32_t qid,"""),
    ("""  digest_push(W, dn, now, query_tag(qid), lane);""", """  digest_push(W, dn, dacc, now, query_tag(qid), lane);"""),
    ("""    int dn = 0;  // digest terms waiting in W->dterm""",
     """    int dn = 0;  // digest terms waiting in W->dterm
    uint64_t dacc = 0;  // this lane's share of the digest"""),
    ("""      digest_push(W, dn, now, call_tag(rid, m), lane);""", """      digest_push(W, dn, dacc, now, call_tag(rid, m), lane);"""),
    ("""          finish_query(W, dn, qid, now, arr, dl, lane);""", """          finish_query(W, dn, dacc, qid, now, arr, dl, lane);"""),
    ("""    digest_flush(W, dn, lane);
""", """    dacc += digest_flush(W, dn, lane);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) dacc += __shfl_xor_sync(kFull, dacc, o);
    W->digest = dacc;
    __syncwarp();
"""),
]

# Micro changes of the hot loop.
_KEY_SHIFT = [("""      W->ekey[m] = ((nk >> 24) << 7) | (uint64_t)m;  // every lane stores the same key""",
               """      W->ekey[m] = ((nk >> 17) & ~0x7Full) | (uint64_t)m;  // every lane stores the same key""")]
_REWARDS_REG = [("""    const int32_t oma32 = W->one_minus_a;""",
                 """    const int32_t oma32 = W->one_minus_a;
    const bool rewards_on = W->rewards != 0;"""),
                ("""          const bool stale = W->rewards != 0;
          dirty0 = lane == m ? stale : dirty0;
          dirty1 = lane + 32 == m ? stale : dirty1;
        }
        // the freed slot""", """          const bool stale = rewards_on;
          dirty0 = lane == m ? stale : dirty0;
          dirty1 = lane + 32 == m ? stale : dirty1;
        }
        // the freed slot"""),
                ("""          const bool stale = W->rewards != 0;
          dirty0 = lane == m ? stale : dirty0;
          dirty1 = lane + 32 == m ? stale : dirty1;
        }
        if (kGeneric) {""", """          const bool stale = rewards_on;
          dirty0 = lane == m ? stale : dirty0;
          dirty1 = lane + 32 == m ? stale : dirty1;
        }
        if (kGeneric) {""")]
_BETA_REGS = [("""    const int32_t oma32 = W->one_minus_a;""",
               """    const int32_t oma32 = W->one_minus_a;
    const uint64_t beta_r = (uint64_t)W->beta;
    const float betaf_r = W->betaf;"""),
              ("""        const uint64_t beta = (uint64_t)W->beta;""", """        const uint64_t beta = beta_r;"""),
              ("""rj ? W->betaf : 0.0f""", """rj ? betaf_r : 0.0f"""),
              ("""              (int64_t)W->one_minus_a * (res < (uint64_t)kRewardCap""",
               """              (int64_t)oma32 * (res < (uint64_t)kRewardCap""")]

_A_REG = [("""    const bool rewards_on = W->rewards != 0;""",
           """    const bool rewards_on = W->rewards != 0;
    const int32_t alpha_r = W->A;"""),
          ("""          const int32_t A = W->A;""", """          const int32_t A = alpha_r;""")]

_HDR = "hx_device.cuh"
# The instance each of this event's dispatches went to, in shared memory
# beside the entry instead of on the entry's lane; the lane's two instance
# types read from the kernel's parameters at each dispatch.
_PEND_SMEM = [(_HDR, """  int32_t pest[HX_MAX_K];""", """  int32_t pest[HX_MAX_K];
  int32_t pendm[HX_MAX_K];"""),
              ("""    // this event's dispatches, entry j on lane j
    int pend_m = -1;
""", ""),
              ("""        pend_m = lane == npend ? m : pend_m;""",
               """        W->pendm[npend] = m;  // every lane writes the same entry"""),
              ("""        const unsigned pm = __ballot_sync(kFull, lane < npend && pend_m == m);""",
               """        const unsigned pm = __ballot_sync(kFull, lane < npend && W->pendm[lane < npend ? lane : 0] == m);""")]
_TY_PARAM = [("""  const int ty0 = valid0 ? c.inst_type[m0] : 0;
  const int ty1 = valid1 ? c.inst_type[m1] : 0;
""", ""),
             ("""        const int2 ev0 = r->ev[ty0], ev1 = r->ev[ty1];""",
              """        const int ty0 = c.inst_type[m0], ty1 = c.inst_type[m1];  // 0 past the cluster's instances
        const int2 ev0 = r->ev[ty0], ev1 = r->ev[ty1];""")]
# ... or from a per-warp shared copy filled once per kernel.
_TY_SMEM = [(_HDR, """  uint8_t hcl[HX_MAX_INST];""", """  uint8_t hcl[HX_MAX_INST];
  uint8_t ity[HX_MAX_INST];      // instance types (0 past the cluster's instances)"""),
            ("""  const int ty0 = valid0 ? c.inst_type[m0] : 0;
  const int ty1 = valid1 ? c.inst_type[m1] : 0;
""", """  W->ity[m0] = c.inst_type[m0];
  W->ity[m1] = c.inst_type[m1];
"""),
            ("""        const int2 ev0 = r->ev[ty0], ev1 = r->ev[ty1];""",
             """        const int ty0 = W->ity[m0], ty1 = W->ity[m1];
        const int2 ev0 = r->ev[ty0], ev1 = r->ev[ty1];""")]

# The next arrival joins the next-event minimum on lane 0 (at equal times a
# completion, tag < 64, still goes first).
_ARR_IN_MIN = [("""      const uint64_t ck = warp_min_u64(k0 < k1 ? k0 : k1);
      const uint64_t akey = W->akey;
      if (ck >= kNoEvent && akey == kKeyInf) break;""", """      const uint64_t akey = W->akey;
      const uint64_t k01 = k0 < k1 ? k0 : k1;
      const uint64_t ck = warp_min_u64(lane == 0 && akey < k01 ? akey : k01);
      if (ck >= kNoEvent) break;"""),
               ("""      if (ck < akey) {
        // completion on instance m""", """      if ((ck & 127ull) != kArrivalTag) {
        // completion on instance m""")]
# A lane's two event keys, and its two cached rewards, adjacent in shared
# memory: one 16-byte load each at the loop top and at the argmax.
_PAIRS = [("""      W->ekey[m] = ((nk >> 24) << 7) | (uint64_t)m;  // every lane stores the same key""",
           """      W->ekey[((m & 31) << 1) | (m >> 5)] = ((nk >> 24) << 7) | (uint64_t)m;  // every lane stores the same key"""),
          ("""    W->ekey[m0] = kKeyInf;
    W->ekey[m1] = kKeyInf;""", """    W->ekey[2 * lane] = kKeyInf;
    W->ekey[2 * lane + 1] = kKeyInf;"""),
          ("""      const uint64_t k0 = W->ekey[m0], k1 = W->ekey[m1];""",
           """      const ulonglong2 kp = *reinterpret_cast<const ulonglong2*>(&W->ekey[2 * lane]);
      const uint64_t k0 = kp.x, k1 = kp.y;"""),
          ("""    W->orew[m0] = valid0 ? orew_idle : -(int64_t(1) << 62);
    W->orew[m1] = valid1 ? orew_idle : -(int64_t(1) << 62);""",
           """    W->orew[2 * lane] = valid0 ? orew_idle : -(int64_t(1) << 62);
    W->orew[2 * lane + 1] = valid1 ? orew_idle : -(int64_t(1) << 62);"""),
          ("""          if (rj) W->orew[dirty0 ? m0 : m1] = orew;""", """          if (rj) W->orew[2 * lane + (dirty0 ? 0 : 1)] = orew;"""),
          ("""          int64_t s0 = W->orew[m0] - (int64_t)A * e0;
          int64_t s1 = W->orew[m1] - (int64_t)A * e1;""",
           """          const longlong2 op = *reinterpret_cast<const longlong2*>(&W->orew[2 * lane]);
          int64_t s0 = op.x - (int64_t)A * e0;
          int64_t s1 = op.y - (int64_t)A * e1;""")]

# Heap sift: whether the best child moves up is decided from the reduced
# maximum key itself (the child's rid is shuffled only on a key tie).
_SIFT_NOSHFL = [("""    if (!__shfl_sync(kFull, (int)ent_better(ck, cr, sink.key, sink.rid), b)) break;""",
                 """    const long long kb = (long long)((((uint64_t)mh << 32) | ml) ^ 0x8000000000000000ull);
    if (kb < sink.key || (kb == sink.key && __shfl_sync(kFull, cr, b) >= sink.rid)) break;""")]

# The reward pass without the divergent early return of the division: an
# idle instance (t_queue <= 1) divides by 2^62 like an inactive lane and
# takes beta by a select.
_DIV_UNIFORM = [("""          const uint64_t res = udiv_trial_f(rj ? beta : 0ull, rj ? W->betaf : 0.0f, (rj && q > 1) ? (uint64_t)q : 1ull);""",
                 """          const uint64_t res0 =
              udiv_trial_f(rj ? beta : 0ull, rj ? W->betaf : 0.0f, (rj && q > 1) ? (uint64_t)q : (1ull << 62));
          const uint64_t res = (rj && q <= 1) ? beta : res0;""")]
# A warp barrier after each simulation's per-lane initial state.
_SYNC_INIT = [("""    W->akey = nq > 0 ? (((uint64_t)a.arrival[qb] << 7) | kArrivalTag) : kKeyInf;
""", """    W->akey = nq > 0 ? (((uint64_t)a.arrival[qb] << 7) | kArrivalTag) : kKeyInf;
    __syncwarp();  // every lane's initial instance state is read by the others
""")]

# Call-record loads (read-only in the simulation kernel) with an L2
# evict-last policy, so that the alpha = 1 heaps streaming through L2 evict
# them last.
_LDG_LAST = """__device__ __forceinline__ int4 ldg_last4(const void* a) {
  int4 v;
  asm("{\\n .reg .b64 pol;\\n createpolicy.fractional.L2::evict_last.b64 pol, 1.0;\\n"
      " ld.global.L2::cache_hint.v4.s32 {%0, %1, %2, %3}, [%4], pol;\\n}"
      : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(a));
  return v;
}
__device__ __forceinline__ int2 ldg_last2(const void* a) {
  int2 v;
  asm("{\\n .reg .b64 pol;\\n createpolicy.fractional.L2::evict_last.b64 pol, 1.0;\\n"
      " ld.global.L2::cache_hint.v2.s32 {%0, %1}, [%2], pol;\\n}"
      : "=r"(v.x), "=r"(v.y) : "l"(a));
  return v;
}
__device__ __forceinline__ int64_t ldg_last8(const void* a) {
  int64_t v;
  asm("{\\n .reg .b64 pol;\\n createpolicy.fractional.L2::evict_last.b64 pol, 1.0;\\n"
      " ld.global.L2::cache_hint.s64 %0, [%1], pol;\\n}"
      : "=l"(v) : "l"(a));
  return v;
}

__device__ __forceinline__ bool ent_better("""
_REC_L2LAST = [("""__device__ __forceinline__ bool ent_better(""", _LDG_LAST),
               ("""  const int64_t dl = r->deadline;
  const int4 tail = *reinterpret_cast<const int4*>(&r->tbar);""",
                """  const int64_t dl = ldg_last8(&r->deadline);
  const int4 tail = ldg_last4(&r->tbar);"""),
               ("""        const CallRec* r = rec + rid;
        const int4 tail = *reinterpret_cast<const int4*>(&r->tbar);
        const int64_t est_m = r->ev[c.inst_type[m]].x;""",
                """        const CallRec* r = rec + rid;
        const int4 tail = ldg_last4(&r->tbar);
        const int64_t est_m = ldg_last2(&r->ev[c.inst_type[m]]).x;"""),
               ("""        const int2 ev0 = r->ev[ty0], ev1 = r->ev[ty1];""",
                """        const int2 ev0 = ldg_last2(&r->ev[ty0]), ev1 = ldg_last2(&r->ev[ty1]);""")]

# The heap sift's child loads below the top two levels with an L1 policy:
# not allocated in L1, or allocated to be evicted first (they are rarely
# read again), so that the 28 KB L1 keeps the call records.
def _sift_l1(policy):
    return [("""    if (child < m) {
      const HeapEnt e = h[child];
      ck = e.key;
      cr = e.rid;
      cs = e.svc;
    }""", """    if (child < m) {
      HeapEnt e;
      if (first >= 33) {
        int4 v;
        asm volatile("ld.global.L1::POLICY.v4.s32 {%0, %1, %2, %3}, [%4];"
                     : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(h + child) : "memory");
        e.key = (long long)(((unsigned long long)(unsigned)v.y << 32) | (unsigned)v.x);
        e.rid = v.z;
        e.svc = v.w;
      } else {
        e = h[child];
      }
      ck = e.key;
      cr = e.rid;
      cs = e.svc;
    }""".replace("POLICY", policy))]


_INLINE_DIGEST = [("""__device__ __noinline__ void digest_flush(""", """__device__ __forceinline__ void digest_flush(""")]
_INLINE_TOPK = [("""__device__ __noinline__ void topk_insert_warp(""", """__device__ __forceinline__ void topk_insert_warp(""")]

VARIANTS = {
    # measured on 64 ceiling traces: against the library that kept the event
    # keys and rewards in registers, both in shared memory 1.0135 (keys alone
    # 1.002, rewards alone 0.996); against that, t_queue stored by every lane
    # 1.0097 (both now in the library), pend_smem 0.990, ty_param 0.914,
    # ty_smem 0.993, both 0.993, 8 blocks per SM 0.958 (64 registers, spills);
    # with the heap helpers inlined (no spills left at 72 registers): 8 blocks
    # per SM 1.028 (no spills at 64; now the library's), pend_smem 0.998,
    # ty_param 0.920, ty_smem 0.994, both 0.997
    "state": {"pend_smem": (_PEND_SMEM, []), "ty_param": (_TY_PARAM, []), "ty_smem": (_TY_SMEM, []),
              "pend_ty_smem": (_PEND_SMEM + _TY_SMEM, [])},
    # measured on 64 ceiling traces: key_shift 1.000, beta_regs 0.992 (the
    # "rewards used" flag in a predicate register gave 1.013 and is now in the
    # library); alpha_reg is measured against the library that includes it
    # measured on 64 ceiling traces: arr_in_min 0.988, erid 1.004, the heap
    # sift inlined 1.005, the queue push helpers 1.007, both 1.014 (now in
    # the library), arr_in_min with erid 1.000; on the library with the
    # inlined helpers: arr_in_min 0.997, erid 1.005, inline_digest 0.998,
    # inline_topk 0.996, erid_topk 1.011; at 8 blocks per SM: arr_in_min
    # 0.996, erid 1.006 (now in the library), inline_digest 0.998,
    # inline_topk 1.006, erid_topk 1.006
    "misc": {"arr_in_min": (_ARR_IN_MIN, []), "inline_digest": (_INLINE_DIGEST, []),
             "inline_topk": (_INLINE_TOPK, [])},
    # measured on 64 ceiling traces: (est, svc) side by side in the call
    # record 1.009 (now in the library), pairs 0.991, both 0.994
    "layout": {"pairs": (_PAIRS, [])},
    # measured on 64 ceiling traces: sift_noshfl 0.992, push_pop's key formed
    # on every lane rather than on the entry's lane and shuffled 1.006 (now in
    # the library), both 0.998, pend_smem 0.994
    "heap": {"sift_noshfl": (_SIFT_NOSHFL, [])},
    # measured on 64 ceiling traces (library 3975 / 3980 ms): rec_l2last
    # 0.965; again (library 3985 / 3976 ms) 0.969, sift_noalloc 0.996,
    # sift_evict_first 0.997
    "cache": {"rec_l2last": (_REC_L2LAST, []), "sift_noalloc": (_sift_l1("no_allocate"), []),
              "sift_evict_first": (_sift_l1("evict_first"), [])},
    # measured on 64 ceiling traces (3 runs each, library 4127 / 4131 ms):
    # sync_init 0.997, div_uniform 0.998, both 0.997 -- within the run-to-run
    # spread; t_queue is now zeroed before the existing barrier instead
    "div": {"sync_init": (_SYNC_INIT, []), "div_uniform": (_DIV_UNIFORM, []),
            "div_sync": (_DIV_UNIFORM + _SYNC_INIT, [])},
    "micro": {"key_shift": _KEY_SHIFT, "beta_regs": _BETA_REGS, "alpha_reg": _A_REG},
    "prefetch": {f"{w}_{lvl.lower()}": [(e[0], e[1].replace("LVL", lvl))]
                 for w, e in (("arrival", _ARRIVAL), ("start", _START)) for lvl in ("L1", "L2")},
    # resident blocks per SM the register allocation aims at (8 by default), and the digest in registers
    "occupancy": {"blocks7": ([], ["-DHX_SIM_MIN_BLOCKS=7"]), "blocks6": ([], ["-DHX_SIM_MIN_BLOCKS=6"]),
                  "digest_lanes": (_DIGEST_LANES, [])},
}


def make_variant(name, edits, flags=()):
    """Copy the library sources, apply the edits ((anchor, replacement) in
    hx_kernels.cu, or (file, anchor, replacement)), build a .so (extra nvcc
    flags for hx_kernels.cu)."""
    d = os.path.join(OUT, name)
    shutil.rmtree(d, ignore_errors=True)
    shutil.copytree(CSRC, os.path.join(d, "csrc"))
    for e in edits:
        f, a, b = e if len(e) == 3 else ("hx_kernels.cu", *e)
        p = os.path.join(d, "csrc", f)
        s = open(p).read()
        if a not in s:
            raise RuntimeError(f"variant {name}: anchor not found in {f}: {a[:60]!r}")
        open(p, "w").write(s.replace(a, b))
    objs = []
    for src in ("hx_kernels.cu", "hx_api.cu"):
        o = os.path.join(d, src.replace(".cu", ".o"))
        extra = list(flags) if src == "hx_kernels.cu" else []
        subprocess.check_call(NVCC + ["-I", os.path.join(d, "csrc"), *extra, "-c", os.path.join(d, "csrc", src),
                                      "-o", o])
        objs.append(o)
    lib = os.path.join(d, "libhxsim.so")
    subprocess.check_call(NVCC[:3] + ["-shared", "-o", lib] + objs)
    return lib


def time_lib(lib_path, wl, reps, **sim_options):
    """Median simulation-kernel milliseconds over `reps` runs after one
    warm-up, and the results, with the library at lib_path (Sim options
    passed through)."""
    from paper_2505_05286_gb300 import hxsim as H
    saved = H._lib
    H._lib = H.load(lib_path)
    try:
        sim = H.Sim(wl.traces, wl.cluster, wl.grid, timing=True, **sim_options)
        sim.run()
        ms = []
        for _ in range(reps):
            sim.run()
            ms.append(sim.timings()[1])
        r = sim.results()
        sim.close()
    finally:
        H._lib = saved
    return float(np.median(ms)), ms, r


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("family", choices=sorted(VARIANTS))
    ap.add_argument("--traces", type=int, default=64)
    ap.add_argument("--reps", type=int, default=3)
    ap.add_argument("--out", default=None)
    args = ap.parse_args(argv)
    import torch

    from paper_2505_05286_gb300 import build as B
    from paper_2505_05286_gb300 import hxsim as H
    from paper_2505_05286_gb300 import workloads as W
    B.build()
    torch.cuda.set_device(0)
    wl = W.make_workload(4, n_traces=args.traces)
    fields = ("p95_us", "makespan_us", "events", "digest", "slo_met", "n_done", "status")
    base_ms, base_all, base = time_lib(H.LIB_PATH, wl, args.reps)
    out = {"workload": f"{wl.name} cut to {args.traces} traces", "sims": wl.n_sims, "library_ms": base_ms,
           "library_all_ms": base_all, "variants": {}}
    print("library", base_ms, base_all, flush=True)
    for name, spec in VARIANTS[args.family].items():
        edits, flags = spec if isinstance(spec, tuple) else (spec, [])
        ms, all_ms, r = time_lib(make_variant(name, edits, flags), wl, args.reps)
        same = all(np.array_equal(r[f], base[f]) for f in fields)
        out["variants"][name] = {"ms": ms, "all_ms": all_ms, "same_results": same, "speedup": base_ms / ms}
        print(name, ms, all_ms, same, round(base_ms / ms, 4), flush=True)
    again, again_all, _ = time_lib(H.LIB_PATH, wl, args.reps)
    out["library_again_ms"] = again
    print("library again", again, again_all, flush=True)
    if args.out:
        with open(args.out, "w") as f:
            json.dump(out, f, indent=1)
    return 0 if all(v["same_results"] for v in out["variants"].values()) else 1


if __name__ == "__main__":
    sys.exit(main())
