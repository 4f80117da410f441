// echo_overlap.cu -- the validator's overlap test (Sec. 3: compose, then adjust the
// kernels that overlap communication; Sec. 2.3: their slowdown factor).  This file
// is compiled once for each (ECHO_OV_LAUNCH, ECHO_OV_PROP) pair, so that the four
// families of variants build in parallel; each object defines one entry point.
#include <cuda_runtime.h>

#include <cstdint>

#include "echo_internal.h"

#if !defined(ECHO_OV_LAUNCH) || !defined(ECHO_OV_PROP)
#error "compile with -DECHO_OV_LAUNCH=0|1 -DECHO_OV_PROP=0|1"
#endif

namespace echo {
namespace {

// rint(p * 2^e) with ties to even, for p < 2^63 and a result below 2^63.
__device__ __forceinline__ int64_t rint_scaled(uint64_t p, int e) {
  if (e >= 0) return (int64_t)(p << e);
  const int k = -e;
  if (k >= 64) return 0;  // p * 2^e < 2^63 * 2^-64 = 1/2
  const uint64_t q = p >> k, rem = p & ((1ull << k) - 1), half = 1ull << (k - 1);
  return (int64_t)(q + ((rem > half || (rem == half && (q & 1))) ? 1 : 0));
}

// Slowed duration rint(fl(fl(d) * f)) (Sec. 2.3: a kernel's time grows by its
// slowdown factor), evaluated exactly in integers so that the fp64 pipe, which is
// slow on this part, stays idle.  f = M * 2^E is passed packed as (M << 11) |
// (E + 1075), M < 2^53 its significand.  Each rounding is IEEE 754
// roundTiesToEven: d to 53 significant bits (the int64 -> double conversion), the
// exact product d * M (< 2^106) to 53 significant bits (the double product), then
// to an integer (rint).  Products below 2^-1022, where the double product would be
// subnormal, round to 0 either way.
__device__ __forceinline__ int64_t slowed(int64_t d, uint64_t packed) {
  const uint64_t M = packed >> 11;
  int e = (int)(packed & 0x7FF) - 1075;
  uint64_t x = (uint64_t)d;
  if (x >> 53) {
    const int s = 11 - __clzll((long long)x);  // bit length - 53
    const uint64_t q = x >> s, rem = x & ((1ull << s) - 1), half = 1ull << (s - 1);
    x = q + ((rem > half || (rem == half && (q & 1))) ? 1 : 0);
    e += s;
  }
  const uint64_t lo = x * M, hi = __umul64hi(x, M);
  const int nb = hi ? 128 - __clzll((long long)hi) : 64 - __clzll((long long)lo);
  uint64_t p = lo;
  if (nb > 53) {  // nb <= 106, so 1 <= s <= 53 and every dropped bit is in lo
    const int s = nb - 53;
    p = (lo >> s) | (hi << (64 - s));
    const uint64_t rem = lo & ((1ull << s) - 1), half = 1ull << (s - 1);
    p += (rem > half || (rem == half && (p & 1))) ? 1 : 0;
    e += s;
  }
  return rint_scaled(p, e);
}

constexpr int kOverlapBatch = 8;  // divides 32 (the shuffled op list's width)
// Blocks per SM the register budget allows.  Occupancy hides the row-load latency
// (at 3 comm timelines, 64 registers beat 108 by 12%); wide cursor sets keep their
// registers instead of spilling.
constexpr int overlap_min_blocks(int ncmax) { return ncmax <= 3 ? 8 : ncmax <= 4 ? 6 : 1; }

// When rank r launched the comm op of cq entry e: the latest finish among its
// launch conditions on r (out of line: the cursor loads are unrolled many times).
__device__ __noinline__ int64_t launch_time(const int32_t *__restrict__ lq_off, const int32_t *__restrict__ lq_ops,
                                            const int64_t *__restrict__ f, int sh, int32_t e) {
  int64_t t = 0;
  for (int32_t k = lq_off[e]; k < lq_off[e + 1]; ++k) t = max(t, f[(int64_t)lq_ops[k] << sh]);
  return t;
}

// LAUNCH: a comm op's interval on the rank opens at the rank's launch of it
// (a.lq_off), else at its start.  PROP: the proportional slowdown model (a.model 1)
template <int NCMAX, bool LAUNCH, bool PROP>
__global__ void __launch_bounds__(kOverlapThreads, overlap_min_blocks(NCMAX)) overlap_kernel(OverlapArgs a) {
  const int32_t S = a.S;
  const int32_t s = blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t c = blockIdx.y + (int64_t)gridDim.y * blockIdx.z;
  if (c >= a.n_chunks) return;  // uniform over the block
  const bool act = s < S;       // inactive lanes still take part in the warp shuffles
  const int32_t sl = act ? s : 0;
  const int lane = threadIdx.x & 31;
  const int nc = a.n_cq;
  const int64_t r = a.chunks[2 * c];
  const int64_t c0 = a.chunks[2 * c + 1];
  const int64_t c1 = min(a.cand_off[r + 1], c0 + kOverlapChunk);
  // element (i, s) of a matrix sits at base + (i << sh)
  const int sh = a.lay.slog2;
  const int64_t base = a.lay.at(0, sl);
  const int64_t *__restrict__ f = a.f + base;
  const int64_t *__restrict__ du = a.dur + base;  // comm ops' durations (never slowed)
  // the candidates' durations in the pass that produced f: the original ones, or the
  // previous validator pass's (compact [candidate][scenario] rows)
  const int64_t *__restrict__ cu = a.cd_used ? a.cd_used + a.lay_c.at(0, sl) : nullptr;
  int64_t *__restrict__ cn = a.cd_next ? a.cd_next + a.lay_c.at(0, sl) : nullptr;
  int32_t qreg = c0 + lane < c1 ? a.cand_ops[c0 + lane] : 0;   // ops c0 .. c0+31 of the chunk
  int32_t creg = c0 + lane < c1 ? a.cand_cidx[c0 + lane] : 0;  // and their level-order indices
  auto cand_d = [&](int64_t v, int64_t ci) { return cu ? cu[ci << sh] : du[v << sh]; };
  // per comm timeline: position, end, and interval of the cursor op; the cursor op
  // always has positive length and finishes after the current op's start (or the
  // cursor is at the end, with an interval that never overlaps)
  int32_t cur[NCMAX] = {}, end[NCMAX] = {};
  int64_t sw[NCMAX], fw[NCMAX];
  auto load = [&](int j) {
    if (cur[j] < end[j]) {
      const int64_t w = a.cq_ops[cur[j]];
      fw[j] = f[w << sh];
      if (LAUNCH) {  // from the rank's launch: its launch conditions' latest finish
        sw[j] = launch_time(a.lq_off, a.lq_ops, f, sh, cur[j]);
      } else {
        sw[j] = fw[j] - du[w << sh];
      }
    } else {
      sw[j] = fw[j] = INT64_MAX;
    }
  };
  {
    const int64_t v = __shfl_sync(0xffffffffu, qreg, 0), ci = __shfl_sync(0xffffffffu, creg, 0);
    const int64_t sv = act ? f[v << sh] - cand_d(v, ci) : 0;
#pragma unroll
    for (int j = 0; j < NCMAX; ++j) {
      cur[j] = end[j] = 0;
      sw[j] = fw[j] = INT64_MAX;
      if (j < nc && act) {
        int32_t lo = (int32_t)a.cq_off[r * nc + j], hi = (int32_t)a.cq_off[r * nc + j + 1];
        end[j] = hi;
        while (lo < hi) {  // first comm op finishing after sv (finishes are sorted)
          const int32_t mid = (lo + hi) >> 1;
          if (f[(int64_t)a.cq_ops[mid] << sh] > sv)
            hi = mid;
          else
            lo = mid + 1;
        }
        cur[j] = lo;
        load(j);
        while (cur[j] < end[j] && sw[j] >= fw[j]) {  // zero-length ops never overlap
          ++cur[j];
          load(j);
        }
      }
    }
  }
  // groups of kOverlapBatch ops: their finish times and durations are loaded together
  for (int64_t i0 = c0; i0 < c1; i0 += kOverlapBatch) {
    if (i0 > c0 && ((i0 - c0) & 31) == 0) {
      qreg = i0 + lane < c1 ? a.cand_ops[i0 + lane] : 0;
      creg = i0 + lane < c1 ? a.cand_cidx[i0 + lane] : 0;
    }
    int64_t vb[kOverlapBatch], cb[kOverlapBatch], fb[kOverlapBatch], db[kOverlapBatch];
#pragma unroll
    for (int u = 0; u < kOverlapBatch; ++u) {
      vb[u] = __shfl_sync(0xffffffffu, qreg, (int)((i0 - c0 + u) & 31));
      cb[u] = __shfl_sync(0xffffffffu, creg, (int)((i0 - c0 + u) & 31));
      fb[u] = db[u] = 0;
      if (act && i0 + u < c1) {
        fb[u] = f[vb[u] << sh];
        db[u] = cand_d(vb[u], cb[u]);
      }
    }
    if (!act) continue;
#pragma unroll
    for (int u = 0; u < kOverlapBatch; ++u) {
      if (i0 + u < c1) {
        const int64_t v = vb[u], fv = fb[u], dv = db[u];
        const int64_t sv = fv - dv;
        bool hit = false;
#pragma unroll
        for (int j = 0; j < NCMAX; ++j) {
          if (j < nc) {
            if (fw[j] <= sv) {  // the cursor op ended before this op starts: move on
              do {
                ++cur[j];
                load(j);
              } while (cur[j] < end[j] && (fw[j] <= sv || sw[j] >= fw[j]));
            }
            hit |= sw[j] < fv;
          }
        }
        hit = hit && sv < fv;
        if (a.ov) a.ov[base + (v << sh)] = hit;
        if (cn) {
          const int64_t d0 = cu ? du[v << sh] : dv;  // the original duration
          int64_t dn = d0;
          if (PROP && hit) {
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
                    ++cur[j];
                    load(j);
                  } while (cur[j] < end[j] && sw[j] >= fw[j]);
                }
              }
            }
            const double f = a.sf[(int64_t)a.kcl[v] * S + sl];
            dn = __double2ll_rn(__dadd_rn((double)d0, __dmul_rn(__dsub_rn(f, 1.0), (double)len)));
          } else if (hit) {
            dn = slowed(d0, a.sfx[(int64_t)a.kcl[v] * S + sl]);
          }
          cn[cb[u] << sh] = dn;
        }
      }
    }
  }
}

}  // namespace

#define ECHO_OV_CAT(l, p) launch_overlap_l##l##_p##p
#define ECHO_OV_NAME(l, p) ECHO_OV_CAT(l, p)

cudaError_t ECHO_OV_NAME(ECHO_OV_LAUNCH, ECHO_OV_PROP)(const OverlapArgs &a, dim3 grid, int tx, cudaStream_t st) {
  constexpr bool L = ECHO_OV_LAUNCH != 0, P = ECHO_OV_PROP != 0;
  // (the 3-cursor variant serves 1 and 2 comm timelines too: every cursor loop
  // stops at the actual count)
  if (a.n_cq <= 3)
    overlap_kernel<3, L, P><<<grid, tx, 0, st>>>(a);
  else if (a.n_cq <= 4)
    overlap_kernel<4, L, P><<<grid, tx, 0, st>>>(a);
  else if (a.n_cq <= 6)
    overlap_kernel<6, L, P><<<grid, tx, 0, st>>>(a);
  else if (a.n_cq <= 8)
    overlap_kernel<8, L, P><<<grid, tx, 0, st>>>(a);
  else
    overlap_kernel<kMaxStreams, L, P><<<grid, tx, 0, st>>>(a);
  return cudaGetLastError();
}

}  // namespace echo
