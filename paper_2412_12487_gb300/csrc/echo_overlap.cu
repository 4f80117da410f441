// echo_overlap.cu -- the validator's overlap test (Sec. 3: compose, then adjust the
// kernels that overlap communication; Sec. 2.3: their slowdown factor).  This file
// is compiled once for each (ECHO_OV_LAUNCH, ECHO_OV_PROP) pair, so that the four
// families of variants build in parallel; each object defines one entry point.
#include <cuda_runtime.h>

#include <cstdint>

#include "echo_internal.h"
#include "echo_bounds.h"
#include "echo_slowdown.cuh"

#if !defined(ECHO_OV_LAUNCH) || !defined(ECHO_OV_PROP)
#error "compile with -DECHO_OV_LAUNCH=0|1 -DECHO_OV_PROP=0|1"
#endif

namespace echo {
namespace {

using dev::slowed;

// Blocks per SM the register budget allows (4 warps each); wide cursor sets keep
// their registers instead of spilling.
constexpr int overlap_min_blocks(int ncmax) { return ncmax <= 6 ? 4 : ncmax <= 8 ? 3 : 1; }

__device__ __forceinline__ void cp_async8(void *dst, const void *src) {
  const uint32_t d = (uint32_t)__cvta_generic_to_shared(dst);
  asm volatile("cp.async.ca.shared.global [%0], [%1], 8;\n" ::"r"(d), "l"(src) : "memory");
}

// When rank r launched the comm op of cq entry e: the latest finish among its
// launch conditions on r (out of line: the cursor loads are unrolled many times).
// debug bounds: the launch conditions of cq entry e are nodes of the graph
__device__ __noinline__ bool lq_ok(const OverlapArgs &a, int32_t e) {
  bool ok = true;
  for (int32_t k = a.lq_off[e]; k < a.lq_off[e + 1]; ++k) ok &= in_range(a.lq_ops[k], a.lay.V);
  return ok;
}

__device__ __noinline__ int64_t launch_time(const int32_t *__restrict__ lq_off, const int32_t *__restrict__ lq_ops,
                                            const int64_t *__restrict__ f, int sh, int32_t e) {
  int64_t t = 0;
  for (int32_t k = lq_off[e]; k < lq_off[e + 1]; ++k) t = max(t, f[(int64_t)lq_ops[k] << sh]);
  return t;
}

// The validator's overlap test, as a walk over each rank's candidates.  Warp w
// takes piece p of rank r's candidate list (in issue order) for 32 scenarios
// (one per lane).  Every timeline of a rank runs its ops one after the other, so
// on each comm timeline the intervals are sorted and the candidates' starts only
// grow: the lane keeps, per comm timeline, a cursor at the first comm op of
// positive length that finishes after the current candidate starts, with that
// op's interval in registers.  The candidate overlaps this timeline iff that
// interval starts before the candidate finishes (later comm ops start after the
// cursor op ends).  A piece that starts mid-list places its cursors by binary
// search; the first piece starts them at the list heads.  The cursor lists hold
// only the comm ops that can overlap a compute op of the rank, so moves are rare,
// and the smallest cursor end and start decide most candidates with two
// comparisons.  The finish times and durations of the candidates come through a
// ring of kOvDepth batches of 8 (cp.async), so each warp keeps several batches of
// loads in flight.  An overlapped compute op of positive length gets
// rint(d * slowdown) (or the proportional form, both in fp64: on this part the
// multiply costs fewer issue slots than an exact integer form) for the next composition
// (cd_next, compact); the decisions themselves are stored only when `ov` is given.
// LAUNCH: a comm op's interval on the rank opens at the rank's launch of it
// (a.lq_off), else at its start.  PROP: the proportional slowdown model.
template <int NCMAX, bool LAUNCH, bool PROP>
__global__ void __launch_bounds__(kOvWarps * 32, overlap_min_blocks(NCMAX)) overlap_kernel(OverlapArgs a) {
  extern __shared__ int64_t ov_ring[];
  const int32_t S = a.S;
  const int lane = threadIdx.x & 31;
  const int64_t wid = (int64_t)blockIdx.x * kOvWarps + (threadIdx.x >> 5);
  const int64_t G = (S + 31) / 32;
  if (wid >= (int64_t)a.n_ranks * G * a.parts) return;  // uniform over the warp
  const int32_t part = (int32_t)(wid % a.parts);
  const int32_t r = (int32_t)(wid / a.parts % a.n_ranks);
  const int32_t s = (int32_t)(wid / a.parts / a.n_ranks) * 32 + lane;
  const bool act = s < S;  // inactive lanes still take part in the shuffles and copies
  const int32_t sl = act ? s : 0;
  const int nc = a.n_cq;
  // this piece of the rank's list, cut at multiples of the batch
  const int64_t r0 = a.cand_off[r], r1 = a.cand_off[r + 1];
  const int64_t nb = (r1 - r0 + kOvBatch - 1) / kOvBatch;
  const int64_t c0 = min(r1, r0 + nb * part / a.parts * kOvBatch);
  const int64_t c1 = min(r1, r0 + nb * (part + 1) / a.parts * kOvBatch);
  if (c0 >= c1) return;
  // element (i, s) of a matrix sits at base + (i << sh)
  const int sh = a.lay.slog2;
  const int64_t base = a.lay.at(0, sl);
  const int64_t *__restrict__ f = a.f + base;
  const int64_t *__restrict__ du = a.dur + base;  // comm ops' durations (never slowed)
  // the candidates' durations in the pass that produced f: the original ones, or the
  // previous validator pass's (compact [candidate][scenario] rows)
  const int64_t *__restrict__ cu = a.cd_used ? a.cd_used + a.lay_c.at(0, sl) : nullptr;
  int64_t *__restrict__ cn = a.cd_next ? a.cd_next + a.lay_c.at(0, sl) : nullptr;
  int64_t *ring = ov_ring + (int64_t)(threadIdx.x >> 5) * (kOvDepth * kOvBatch * 2 * 32) + lane;
  // per comm timeline: position, end, and interval of the cursor op; the cursor op
  // always has positive length and finishes after the current op's start (or the
  // cursor is at the end, with an interval that never overlaps)
  // (nid: the node of the cursor's next position, loaded one move ahead so that a
  // move waits for the interval's loads only)
  int32_t cur[NCMAX] = {}, end[NCMAX] = {}, nid[NCMAX] = {};
  int64_t sw[NCMAX], fw[NCMAX];
  auto fetch = [&](int j, int64_t w) {  // node w's interval as cursor j's op
    if (a.dbg && !(in_range(w, a.lay.V) && (!LAUNCH || lq_ok(a, cur[j])))) {  // debug bounds
      atomicCAS(a.status, 0, (int32_t)kDevBounds);
      sw[j] = fw[j] = INT64_MAX;
      return;
    }
    fw[j] = f[w << sh];
    if (LAUNCH) {  // from the rank's launch: its launch conditions' latest finish
      sw[j] = launch_time(a.lq_off, a.lq_ops, f, sh, cur[j]);
    } else {
      sw[j] = fw[j] - du[w << sh];
    }
  };
  auto seek = [&](int j) {  // cursor j at position cur[j]
    if (cur[j] < end[j]) {
      fetch(j, a.cq_ops[cur[j]]);
      nid[j] = cur[j] + 1 < end[j] ? a.cq_ops[cur[j] + 1] : 0;
    } else {
      sw[j] = fw[j] = INT64_MAX;
    }
  };
  auto advance = [&](int j) {  // cursor j one position on
    ++cur[j];
    if (cur[j] < end[j]) {
      const int64_t w = nid[j];
      nid[j] = cur[j] + 1 < end[j] ? a.cq_ops[cur[j] + 1] : 0;
      fetch(j, w);
    } else {
      sw[j] = fw[j] = INT64_MAX;
    }
  };
  {
    int64_t sv0 = 0;  // the piece's first candidate's start (only for a search)
    if (part > 0) {
      const int64_t v = a.cand_ops[c0], ci = a.cand_cidx[c0];
      if (a.dbg && !(in_range(v, a.lay.V) && in_range(ci, a.lay_c.V))) {  // debug bounds
        if (lane == 0) atomicCAS(a.status, 0, (int32_t)kDevBounds);
        return;
      }
      sv0 = f[v << sh] - (cu ? cu[ci << sh] : du[v << sh]);
    }
#pragma unroll
    for (int j = 0; j < NCMAX; ++j) {
      cur[j] = end[j] = 0;
      sw[j] = fw[j] = INT64_MAX;
      if (j < nc) {
        int32_t lo = (int32_t)a.cq_off[r * nc + j], hi = (int32_t)a.cq_off[r * nc + j + 1];
        end[j] = hi;
        if (part > 0) {
          while (lo < hi) {  // first comm op finishing after sv0 (finishes are sorted)
            const int32_t mid = (lo + hi) >> 1;
            if (a.dbg && !in_range(a.cq_ops[mid], a.lay.V)) {  // debug bounds: stop searching
              atomicCAS(a.status, 0, (int32_t)kDevBounds);
              break;
            }
            if (f[(int64_t)a.cq_ops[mid] << sh] > sv0)
              hi = mid;
            else
              lo = mid + 1;
          }
        }
        cur[j] = lo;
        seek(j);
        while (cur[j] < end[j] && sw[j] >= fw[j]) advance(j);  // zero-length ops never overlap
      }
    }
  }
  // The smallest cursor end and start over the timelines: while every cursor op
  // ends after a candidate starts (fmin > sv), no cursor moves, and the candidate
  // overlaps iff some cursor op starts before it ends (smin < fv).
  int64_t fmin, smin;
  auto bounds = [&]() {
    fmin = smin = INT64_MAX;
#pragma unroll
    for (int j = 0; j < NCMAX; ++j)
      if (j < nc) {
        fmin = min(fmin, fw[j]);
        smin = min(smin, sw[j]);
      }
  };
  bounds();
  // candidate ids of a batch: lanes 0..7 hold node, level-order index and class
  auto ids = [&](int64_t i0, int32_t &q, int32_t &cx, int32_t &kc) {
    const int64_t i = i0 + (lane & (kOvBatch - 1));
    const bool in = i < c1;
    q = in ? a.cand_ops[i] : 0;
    cx = in ? a.cand_cidx[i] : 0;
    kc = in ? a.cand_kcl[i] : 0;
  };
  // the batch's finish times and durations (those of the pass that produced f)
  // debug bounds: a batch's nodes, compact rows and kernel classes, before its copies
  auto batch_ok = [&](int64_t i0, int32_t q, int32_t cx, int32_t kc) {
    const int64_t i = i0 + (lane & (kOvBatch - 1));
    const bool ok = i >= c1 || (in_range(q, a.lay.V) && in_range(cx, a.lay_c.V) && in_range(kc, a.n_kclass));
    return __all_sync(0xffffffffu, ok);
  };
  auto issue = [&](int64_t i0, int32_t q, int32_t cx) {
    int64_t *slot = ring + ((i0 - c0) / kOvBatch % kOvDepth) * (kOvBatch * 2 * 32);
#pragma unroll
    for (int u = 0; u < kOvBatch; ++u) {
      const int64_t v = __shfl_sync(0xffffffffu, q, u), ci = __shfl_sync(0xffffffffu, cx, u);
      if (i0 + u < c1) {
        cp_async8(slot + (2 * u) * 32, f + (v << sh));
        cp_async8(slot + (2 * u + 1) * 32, cu ? cu + (ci << sh) : du + (v << sh));
      }
    }
    asm volatile("cp.async.commit_group;\n" ::: "memory");
  };
  static_assert(kOvDepth == 3, "the id registers below hold kOvDepth batches");
  int32_t q0, x0, k0, q1, x1, k1, q2, x2, k2, q3, x3, k3;
  ids(c0, q0, x0, k0);
  ids(c0 + kOvBatch, q1, x1, k1);
  ids(c0 + 2 * kOvBatch, q2, x2, k2);
  const bool dbg_bad = a.dbg && !(batch_ok(c0, q0, x0, k0) && batch_ok(c0 + kOvBatch, q1, x1, k1));
  if (dbg_bad) {
    if (lane == 0) atomicCAS(a.status, 0, (int32_t)kDevBounds);
    return;
  }
  issue(c0, q0, x0);
  issue(c0 + kOvBatch, q1, x1);
  for (int64_t i0 = c0; i0 < c1; i0 += kOvBatch) {
    ids(i0 + 3 * kOvBatch, q3, x3, k3);
    if (a.dbg && !batch_ok(i0 + 2 * kOvBatch, q2, x2, k2)) {
      if (lane == 0) atomicCAS(a.status, 0, (int32_t)kDevBounds);
      break;  // (the copies in flight land below)
    }
    issue(i0 + 2 * kOvBatch, q2, x2);
    asm volatile("cp.async.wait_group 2;\n" ::: "memory");  // this batch's copies landed
    int64_t *slot = ring + ((i0 - c0) / kOvBatch % kOvDepth) * (kOvBatch * 2 * 32);
    const int n_here = c1 - i0 < kOvBatch ? (int)(c1 - i0) : kOvBatch;
    // 1) the cursor walk, candidate after candidate: a bit per overlapped candidate
    //    (and, proportional model, its covered length in place of its finish)
    uint32_t hits = 0;
    if (act) {
      // (the next candidate's finish and duration load while this one is tested)
      int64_t fn = slot[0], dn = slot[32];
#pragma unroll 1
      for (int u = 0; u < n_here; ++u) {
        const int64_t fv = fn, dv = dn;
        if (u + 1 < n_here) {
          fn = slot[(2 * u + 2) * 32];
          dn = slot[(2 * u + 3) * 32];
        }
        const int64_t sv = fv - dv;
        if (fmin <= sv) {
#pragma unroll
          for (int j = 0; j < NCMAX; ++j) {
            if (j < nc && fw[j] <= sv) {  // the cursor op ended before this op starts: move on
              do {
                advance(j);
              } while (cur[j] < end[j] && (fw[j] <= sv || sw[j] >= fw[j]));
            }
          }
          bounds();
        }
        const bool hit = smin < fv && sv < fv;
        hits |= (uint32_t)hit << u;
        if (PROP && hit && cn) {
          // proportional model: the length of [sv, fv) covered by the union of the
          // comm intervals, swept in start order across the timelines.  Later
          // candidates start no earlier than fv, so a cursor moves past every
          // interval that ends by fv; one reaching beyond fv stays.
          int64_t len = 0, covered = sv;
          uint32_t held = 0;  // timelines whose cursor interval reaches beyond fv
          while (true) {
            int jb = -1;
            int64_t first = fv;
#pragma unroll
            for (int j = 0; j < NCMAX; ++j)
              if (j < nc && !((held >> j) & 1) && sw[j] < first) {
                first = sw[j];
                jb = j;
              }
            if (jb < 0) break;
#pragma unroll
            for (int j = 0; j < NCMAX; ++j) {  // (j == jb, in registers)
              if (j != jb) continue;
              const int64_t lo = max(sw[j], covered), hi = min(fw[j], fv);
              if (hi > lo) {
                len += hi - lo;
                covered = hi;
              }
              if (fw[j] > fv) {
                held |= 1u << j;
              } else {
                do {
                  advance(j);
                } while (cur[j] < end[j] && sw[j] >= fw[j]);
              }
            }
          }
          bounds();
          slot[(2 * u) * 32] = len;
        }
      }
    }
    // 2) the outputs, the batch's candidates independently of each other
#pragma unroll
    for (int u = 0; u < kOvBatch; ++u) {
      const int64_t v = __shfl_sync(0xffffffffu, q0, u);
      const int64_t kc = __shfl_sync(0xffffffffu, k0, u);
      const int64_t ci = __shfl_sync(0xffffffffu, x0, u);
      if (!act || u >= n_here) continue;
      const bool hit = (hits >> u) & 1;
      if (a.ov) a.ov[base + (v << sh)] = hit;
      if (cn) {
        const int64_t d0 = cu ? du[v << sh] : slot[(2 * u + 1) * 32];  // the original duration
        int64_t dn = d0;
        if (hit) {
          if (PROP)
            dn = dev::slowed_proportional(d0, a.sf[kc * S + sl], slot[(2 * u) * 32]);
          else
            dn = slowed(d0, a.sf[kc * S + sl]);
        }
        cn[ci << sh] = dn;
      }
    }
    q0 = q1, x0 = x1, k0 = k1;
    q1 = q2, x1 = x2, k1 = k2;
    q2 = q3, x2 = x3, k2 = k3;
  }
  asm volatile("cp.async.wait_all;\n" ::: "memory");
}

}  // namespace

#define ECHO_OV_CAT(l, p) launch_overlap_l##l##_p##p
#define ECHO_OV_NAME(l, p) ECHO_OV_CAT(l, p)

cudaError_t ECHO_OV_NAME(ECHO_OV_LAUNCH, ECHO_OV_PROP)(const OverlapArgs &a, dim3 grid, int tx, cudaStream_t st) {
  constexpr bool L = ECHO_OV_LAUNCH != 0, P = ECHO_OV_PROP != 0;
  const size_t smem = overlap_smem_bytes();
  // (the 3-cursor variant serves 1 and 2 comm timelines too: every cursor loop
  // stops at the actual count)
  if (a.n_cq <= 3)
    overlap_kernel<3, L, P><<<grid, tx, smem, st>>>(a);
  else if (a.n_cq <= 4)
    overlap_kernel<4, L, P><<<grid, tx, smem, st>>>(a);
  else if (a.n_cq <= 6)
    overlap_kernel<6, L, P><<<grid, tx, smem, st>>>(a);
  else if (a.n_cq <= 8)
    overlap_kernel<8, L, P><<<grid, tx, smem, st>>>(a);
  else
    overlap_kernel<kMaxStreams, L, P><<<grid, tx, smem, st>>>(a);
  return cudaGetLastError();
}

}  // namespace echo
