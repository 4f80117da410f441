// echo_kernels.cu -- sm_103a kernels of the timeline composer, CC estimator and
// validator.  All floating point that decides an integer is written with explicit
// round-to-nearest intrinsics (no contraction), so results do not depend on -fmad.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>
#include <cstring>
#include <functional>
#include <mutex>
#include <vector>

#include "echo.h"
#include "echo_internal.h"

namespace echo {

namespace {

constexpr int kAR = 0, kAG = 1, kSR = 3;  // reduce-scatter (2) takes the generic ring path
constexpr int kRing = 0, kTree = 1;

__device__ __forceinline__ int64_t cdiv64(int64_t a, int64_t b) { return (a + b - 1) / b; }

__device__ __forceinline__ int64_t chunk_for(int64_t nbytes, const ChunkTable &t) {
  for (int i = 0; i < t.n; ++i)
    if (nbytes <= t.max_bytes[i]) return t.chunk[i];
  return t.chunk[t.n - 1];
}

// Eqs. 2-4 (Sec. 5.3): eta chunk rounds, eta*(N-1) ring steps (twice that for
// all-reduce), each L + p/B with p = S/(N*eta); inter-node link once M > 1.
__device__ double ring_ns(int type, int64_t S, int N, int M, double alpha, double Ba, double La,
                          double Be, double Le, double delta, int64_t C) {
  int64_t eta = cdiv64(S, (int64_t)N * C);
  if (eta < 1) eta = 1;
  double p = __ddiv_rn((double)S, __dmul_rn((double)N, (double)eta));
  double L = M > 1 ? Le : La;
  double B = M > 1 ? Be : Ba;
  double t = __dadd_rn(L, __ddiv_rn(p, B));
  int64_t steps = (type == kAR ? 2 : 1) * eta * (int64_t)(N - 1);
  double T = __dadd_rn(alpha, __dmul_rn((double)steps, t));
  if (type != kAG) T = __dadd_rn(T, __dmul_rn(delta, (double)S));
  return T;
}

// Eq. 5 (Sec. 5.3): tree all-reduce; eta chunks, K-1 intra-node hops (beta) and
// log2(M) inter-node levels (gamma) up and down.
__device__ double tree_ns(int64_t S, int M, int K, double lg, double alpha, double Ba, double La,
                          double Be, double Le, double delta, int64_t C) {
  int64_t eta = cdiv64(S, C);
  if (eta < 1) eta = 1;
  double pt = __ddiv_rn((double)S, (double)eta);
  double beta = __dadd_rn(La, __ddiv_rn(pt, Ba));
  double gamma = M > 1 ? __dadd_rn(Le, __ddiv_rn(pt, Be)) : beta;
  double T = __dadd_rn(alpha, __dmul_rn(gamma, (double)(eta - 1)));
  T = __dadd_rn(T, __dmul_rn(__dmul_rn(2.0, beta), (double)(K - 1)));
  T = __dadd_rn(T, __dmul_rn(__dmul_rn(2.0, gamma), lg));
  T = __dadd_rn(T, __dmul_rn(delta, (double)S));
  return T;
}

__device__ double cc_ns_of(int type, int algo, int64_t S, int N, int M, int K, double lg,
                           double alpha, double Ba, double La, double Be, double Le, double delta,
                           const ChunkTable &tbl) {
  if (N <= 1 || S <= 0) return 0.0;
  int64_t C = chunk_for(S, tbl);
  if (type == kSR) {  // send/recv: eta chunk transfers over the pair's link
    int64_t eta = cdiv64(S, C);
    if (eta < 1) eta = 1;
    double L = M > 1 ? Le : La;
    double B = M > 1 ? Be : Ba;
    double per = __dadd_rn(L, __ddiv_rn(__ddiv_rn((double)S, (double)eta), B));
    return __dadd_rn(alpha, __dmul_rn((double)eta, per));
  }
  if (type != kAR || algo == kRing) return ring_ns(type, S, N, M, alpha, Ba, La, Be, Le, delta, C);
  if (algo == kTree) return tree_ns(S, M, K, lg, alpha, Ba, La, Be, Le, delta, C);
  double r = ring_ns(kAR, S, N, M, alpha, Ba, La, Be, Le, delta, C);
  double t = tree_ns(S, M, K, lg, alpha, Ba, La, Be, Le, delta, C);
  return t < r ? t : r;
}

__device__ __forceinline__ int64_t slowed(int64_t d, double factor) {
  return __double2ll_rn(__dmul_rn((double)d, factor));
}

__device__ __forceinline__ void set_status(int32_t *status, int32_t code) {
  atomicCAS(status, 0, code);
}

// ---------------------------------------------------------------------------------
// B1: CC estimate over [signature x scenario]
// ---------------------------------------------------------------------------------
__global__ void cc_estimate_kernel(const CcSig *__restrict__ sig, int32_t G, ScenParams p, int32_t S,
                                   ChunkTable tbl, const int32_t *__restrict__ sig_count,
                                   double *__restrict__ cc_ns, int64_t *__restrict__ cc_dur,
                                   double *__restrict__ comm_sum, int32_t *status) {
  int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (int64_t)G * S) return;
  int32_t g = (int32_t)(idx / S), s = (int32_t)(idx % S);
  CcSig q = sig[g];
  double T = cc_ns_of(q.type, q.algo, q.nbytes, q.N, q.M, q.K, q.lg, p.alpha[s], p.bwa[s], p.lata[s],
                      p.bwe[s], p.late[s], p.delta[s], tbl);
  int64_t d = 0;
  if (T >= 0.0 && T < 2305843009213693952.0) {  // 2^61
    d = __double2ll_rn(T);
  } else {
    set_status(status, kDevCcOverflow);
  }
  cc_ns[idx] = T;
  cc_dur[idx] = d;
  atomicAdd(&comm_sum[s], (double)d * (double)sig_count[g]);
}

// every comm node takes its signature's duration row
__global__ void cc_scatter_kernel(const int32_t *__restrict__ comm_node, const int32_t *__restrict__ comm_sig,
                                  int64_t n_comm, const int64_t *__restrict__ cc_dur, int32_t S, MatLayout lay,
                                  int64_t *__restrict__ dur) {
  int64_t total = n_comm * S;
  for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
       idx += (int64_t)gridDim.x * blockDim.x) {
    int64_t c = idx / S;
    int32_t s = (int32_t)(idx - c * S);
    dur[lay.at(comm_node[c], s)] = cc_dur[(int64_t)comm_sig[c] * S + s];
  }
}

__global__ void cc_query_kernel(int64_t n, const uint8_t *__restrict__ type, const uint8_t *__restrict__ algo,
                                const int64_t *__restrict__ nbytes, const int32_t *__restrict__ N,
                                const int32_t *__restrict__ M, const double *__restrict__ lg, ScenParams p,
                                ChunkTable tbl, double *__restrict__ out) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    int n_r = N[i], m = M[i];
    int K = (n_r + m - 1) / m;
    out[i] = cc_ns_of(type[i], algo[i], nbytes[i], n_r, m, K, lg[i], p.alpha[i], p.bwa[i], p.lata[i],
                      p.bwe[i], p.late[i], p.delta[i], tbl);
  }
}

// ---------------------------------------------------------------------------------
// load: caller-order rows -> internal order and blocked layout, with validation
// and per-scenario sums
// ---------------------------------------------------------------------------------
__global__ void permute_rows_kernel(const int64_t *__restrict__ raw, const int32_t *__restrict__ int2ext,
                                    const uint8_t *__restrict__ local, int64_t V, int32_t S, MatLayout lay,
                                    int64_t *__restrict__ dur, double *__restrict__ sums, int32_t *status) {
  int32_t s = blockIdx.x * blockDim.x + threadIdx.x;
  if (s >= S) return;
  double acc = 0.0;
  bool neg = false;
  for (int64_t i = blockIdx.y; i < V; i += gridDim.y) {
    int64_t e = int2ext[i];
    int64_t d = 0;
    if (local[i]) {
      d = raw[e * S + s];
      neg |= d < 0;
      acc += (double)d;
    }
    dur[lay.at(i, s)] = d;
  }
  if (neg) set_status(status, kDevNegativeDuration);
  atomicAdd(&sums[s], acc);
}

// ---------------------------------------------------------------------------------
// B2: compose pass.  One thread block owns a block of SIGMA scenarios and walks
// the graph segment level by segment level; scenarios never interact, so only
// block-level synchronization is needed.  A segment is a serial chain of ops
// (each op's only input is the previous one, which feeds nothing else), so along
// it every op starts when the previous ends: finish = running sum.  The head of a
// segment starts at max(0, finish of the op issued before it on each of its
// timelines, finish of each data predecessor) (Sec. 4.2, 5.2); the first term
// comes from a per-(timeline, scenario) frontier holding the finish of the last
// op placed on that timeline, which the segment's tail advances.  The
// per-scenario makespan is fused in.
//
// compose_direct_kernel reads the graph and the durations from global memory and
// fits any graph; the staged and pipelined kernels are the fast paths.
// ---------------------------------------------------------------------------------
template <int SIGMA, bool SMEM_FRONTIER>
__global__ void __launch_bounds__(kComposeThreads)
compose_direct_kernel(ComposeArgs a) {
  extern __shared__ __align__(16) int64_t smem[];
  const int32_t S = a.S;
  const int32_t s0 = blockIdx.x * SIGMA;
  int64_t *mk_s = smem;  // [SIGMA]
  int64_t *fr = SMEM_FRONTIER ? smem + SIGMA
                              : a.gfrontier + (int64_t)blockIdx.x * a.n_queues * SIGMA;
  for (int64_t k = threadIdx.x; k < (int64_t)a.n_queues * SIGMA; k += blockDim.x) fr[k] = 0;
  if (threadIdx.x < SIGMA) mk_s[threadIdx.x] = 0;
  __syncthreads();

  const int j = threadIdx.x % SIGMA;
  const int sub = threadIdx.x / SIGMA;
  const int stride = blockDim.x / SIGMA;
  const int32_t s = s0 + j;
  const bool active = s < S;
  const int64_t *__restrict__ dur = a.dur;
  int64_t *f = a.f;
  int64_t mk = 0;
  for (int32_t l = 0; l < a.L; ++l) {
    const int64_t t0 = a.seg_lvl_off[l], t1 = a.seg_lvl_off[l + 1];
    if (active) {
      for (int64_t t = t0 + sub; t < t1; t += stride) {
        const int64_t h = a.seg_node_off[t], z = a.seg_node_off[t + 1] - 1;
        int64_t fv = 0;  // the head starts after its timelines and data predecessors
        for (int64_t k = a.nq_off[h]; k < a.nq_off[h + 1]; ++k) fv = max(fv, fr[(int64_t)a.nq[k] * SIGMA + j]);
        for (int64_t k = a.dp_off[h]; k < a.dp_off[h + 1]; ++k) fv = max(fv, f[a.lay.at(a.dp[k], s)]);
        for (int64_t i = h; i <= z; ++i) {  // along the chain every op starts when the previous ends
          fv += dur[a.lay.at(i, s)];
          f[a.lay.at(i, s)] = fv;
        }
        for (int64_t k = a.nq_off[z]; k < a.nq_off[z + 1]; ++k) fr[(int64_t)a.nq[k] * SIGMA + j] = fv;
        mk = max(mk, fv);
      }
    }
    __syncthreads();
  }
  if (active) atomicMax((unsigned long long *)&mk_s[j], (unsigned long long)mk);
  __syncthreads();
  if (threadIdx.x < SIGMA && s0 + (int32_t)threadIdx.x < S && a.makespan)
    a.makespan[s0 + threadIdx.x] = mk_s[threadIdx.x];
}

// -- asynchronous global->shared copies (cp.async; completion by wait_group) ----------
__device__ __forceinline__ void cp_async16(void *dst, const void *src) {
  unsigned d = (unsigned)__cvta_generic_to_shared(dst);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(d), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async8(void *dst, const void *src) {
  unsigned d = (unsigned)__cvta_generic_to_shared(dst);
  asm volatile("cp.async.ca.shared.global [%0], [%1], 8;\n" ::"r"(d), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory");
}
__device__ __forceinline__ void cp_async_wait_dyn(int n) {
  switch (n) {
    case 0: cp_async_wait<0>(); break;
    case 1: cp_async_wait<1>(); break;
    case 2: cp_async_wait<2>(); break;
    case 3: cp_async_wait<3>(); break;
    case 4: cp_async_wait<4>(); break;
    case 5: cp_async_wait<5>(); break;
    case 6: cp_async_wait<6>(); break;
    case 7: cp_async_wait<7>(); break;
    case 8: cp_async_wait<8>(); break;
    case 9: cp_async_wait<9>(); break;
    case 10: cp_async_wait<10>(); break;
    case 11: cp_async_wait<11>(); break;
    case 12: cp_async_wait<12>(); break;
    case 13: cp_async_wait<13>(); break;
    default: cp_async_wait<14>(); break;
  }
}

// A thread moves LANES consecutive int64 values of a row (a 16-byte vector when
// LANES == 2; rows are 16-byte aligned whenever SIGMA is even).  The s_* forms
// address shared memory explicitly (32-bit shared addresses).
__device__ __forceinline__ uint32_t saddr(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }
template <int LANES>
__device__ __forceinline__ void s_load(uint32_t a, int64_t (&v)[LANES]) {
  if constexpr (LANES == 2)
    asm volatile("ld.shared.v2.s64 {%0, %1}, [%2];\n" : "=l"(v[0]), "=l"(v[1]) : "r"(a));
  else
    asm volatile("ld.shared.s64 %0, [%1];\n" : "=l"(v[0]) : "r"(a));
}
template <int LANES>
__device__ __forceinline__ void s_store(uint32_t a, const int64_t (&v)[LANES]) {
  if constexpr (LANES == 2)
    asm volatile("st.shared.v2.s64 [%0], {%1, %2};\n" ::"r"(a), "l"(v[0]), "l"(v[1]) : "memory");
  else
    asm volatile("st.shared.s64 [%0], %1;\n" ::"r"(a), "l"(v[0]) : "memory");
}
template <int LANES>
__device__ __forceinline__ void s_max(int64_t (&m)[LANES], uint32_t a) {
  int64_t v[LANES];
  s_load<LANES>(a, v);
#pragma unroll
  for (int k = 0; k < LANES; ++k) m[k] = max(m[k], v[k]);
}
__device__ __forceinline__ uint32_t s_ld32(uint32_t a) {
  uint32_t v;
  asm volatile("ld.shared.u32 %0, [%1];\n" : "=r"(v) : "r"(a));
  return v;
}
__device__ __forceinline__ uint4 s_ld128(uint32_t a) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];\n" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a));
  return v;
}
template <int LANES>
__device__ __forceinline__ void g_max(int64_t (&m)[LANES], const int64_t *p) {
  if constexpr (LANES == 2) {
    const longlong2 t = *reinterpret_cast<const longlong2 *>(p);
    m[0] = max(m[0], (int64_t)t.x);
    m[1] = max(m[1], (int64_t)t.y);
  } else {
    m[0] = max(m[0], *p);
  }
}
template <int LANES>
__device__ __forceinline__ void g_store(int64_t *p, const int64_t (&v)[LANES]) {
  if constexpr (LANES == 2)
    *reinterpret_cast<longlong2 *>(p) = make_longlong2(v[0], v[1]);
  else
    *p = v[0];
}

// Compose the segments of one segment level (shared by the staged and the
// pipelined kernels).  Segment k's header and entries are in the record ring at
// word `ro`; its rows are i0 + header.z ... in the duration ring.  Thread `sub`
// handles segments sub, sub + step, ... for scenario lanes j0 .. j0+LANES-1.  This
// block's finish rows are a contiguous [V][SIGMA] array (padding lanes included),
// so every row moves as whole vectors.
template <int SIGMA, int LANES>
__device__ __forceinline__ void compose_segments(const StagedArgs &a, uint32_t ro, uint32_t i0, uint32_t seg0,
                                                 int32_t nseg, int sub, int step, int j0, int64_t *fr, int64_t *vr,
                                                 const int64_t *dr, const uint32_t *rr, uint32_t vmask,
                                                 uint32_t dmask, uint32_t rmask, int64_t (&mk)[LANES]) {
  int64_t *fb = a.f + ((int64_t)blockIdx.x * a.n_rows) * SIGMA;
  const uint32_t fr_a = saddr(fr) + j0 * 8, vr_a = saddr(vr) + j0 * 8, dr_a = saddr(dr) + j0 * 8;
  const uint32_t rr_a = saddr(rr);
  constexpr uint32_t kRowBytes = SIGMA * 8;
  for (int32_t k = sub; k < nseg; k += step) {
    const uint4 hd = s_ld128(rr_a + ((ro + 4 * k) & rmask) * 4);
    const uint32_t nqf = hd.y & 0xFFFFu, ndp = hd.y >> 16;
    const uint32_t len = hd.w & 0xFFFFu, nql = hd.w >> 16;
    const uint32_t e = ro + hd.x;
    const uint32_t first = i0 + hd.z;
    int64_t fv[LANES];
#pragma unroll
    for (int j = 0; j < LANES; ++j) fv[j] = 0;
    for (uint32_t q = 0; q < nqf; ++q) s_max<LANES>(fv, fr_a + s_ld32(rr_a + ((e + q) & rmask) * 4) * kRowBytes);
    for (uint32_t q = 0; q < ndp; ++q) {
      const uint32_t ref = s_ld32(rr_a + ((e + nqf + q) & rmask) * 4);
      if (ref & kFarRef)
        g_max<LANES>(fv, fb + (int64_t)(ref & ~kFarRef) * SIGMA + j0);
      else
        s_max<LANES>(fv, vr_a + (ref & vmask) * kRowBytes);
    }
    int64_t *gp = fb + (int64_t)first * SIGMA + j0;
#pragma unroll 4
    for (uint32_t t = 0; t < len; ++t, gp += SIGMA) {  // along the chain every op starts when the previous ends
      int64_t d[LANES];
      s_load<LANES>(dr_a + ((first + t) & dmask) * kRowBytes, d);
#pragma unroll
      for (int j = 0; j < LANES; ++j) fv[j] += d[j];
      g_store<LANES>(gp, fv);
    }
#pragma unroll
    for (int j = 0; j < LANES; ++j) mk[j] = max(mk[j], fv[j]);
    s_store<LANES>(vr_a + ((seg0 + k) & vmask) * kRowBytes, fv);
    for (uint32_t q = 0; q < nql; ++q)
      s_store<LANES>(fr_a + s_ld32(rr_a + ((e + nqf + ndp + q) & rmask) * 4) * kRowBytes, fv);
  }
}

// Staged compose (all threads copy and compose).  Shared memory holds the
// per-scenario makespans, the extents of the last 16 copy groups, two metadata
// buffers (kMetaChunk segment levels each), the frontier, a value ring with the
// finish times of the tails of the most recent 2^vlog2 segments (read by near
// predecessors), a ring of duration rows and a ring of record words.  Before
// composing segment level l, every thread copies into the rings all rows and
// record words that fit without touching level l-1 (which slower threads may still
// read); it then waits only for the copy groups that hold level l.  Predecessors
// too old for the value ring are read from global memory, where this block wrote
// them at an earlier level.  SIGMA/LANES threads share a segment.
template <int SIGMA, int THREADS>
__global__ void __launch_bounds__(THREADS)
compose_staged_kernel(StagedArgs a) {
  constexpr int LANES = (SIGMA % 2 == 0) ? 2 : 1;
  constexpr int TPN = SIGMA / LANES;  // threads per segment
  extern __shared__ __align__(16) unsigned char sbuf[];
  const int32_t S = a.S;
  const int32_t s0 = blockIdx.x * SIGMA;
  const int tid = threadIdx.x;
  const StagedLayout lay = staged_layout(a.n_queues, SIGMA, a.vlog2, a.dlog2, a.rlog2);
  const uint32_t vmask = (1u << a.vlog2) - 1, dmask = (1u << a.dlog2) - 1, rmask = (1u << a.rlog2) - 1;
  const uint32_t RR = dmask + 1, RB = rmask + 1;
  int64_t *mk_s = reinterpret_cast<int64_t *>(sbuf);                  // [SIGMA]
  uint2 *hist = reinterpret_cast<uint2 *>(sbuf + lay.hist);           // [16] (rows, words) copied by group
  uint32_t *meta_s = reinterpret_cast<uint32_t *>(sbuf + lay.meta);   // [2][kMetaCap][4]
  int64_t *fr = reinterpret_cast<int64_t *>(sbuf + lay.fr);           // [n_queues][SIGMA]
  int64_t *vr = reinterpret_cast<int64_t *>(sbuf + lay.vr);           // [value ring][SIGMA]
  int64_t *dr = reinterpret_cast<int64_t *>(sbuf + lay.dr);           // [duration ring][SIGMA]
  uint32_t *rr = reinterpret_cast<uint32_t *>(sbuf + lay.rr);         // [record ring]

  for (int k = tid; k < a.n_queues * SIGMA; k += blockDim.x) fr[k] = 0;
  if (tid < SIGMA) mk_s[tid] = 0;
  auto load_meta = [&](int32_t chunk) {  // segment levels [chunk*kMetaChunk, +kMetaChunk] (inclusive)
    uint32_t *dst = meta_s + (chunk & 1) * kMetaCap * 4;
    const int32_t base = chunk * kMetaChunk;
    for (int k = tid; k <= kMetaChunk; k += blockDim.x)
      if (base + k <= a.L) cp_async16(&dst[4 * k], &a.meta[4 * (base + k)]);
  };
  // this block's rows are contiguous: element e of the block lands in ring element
  // e mod (RR*SIGMA), and a 16-byte piece never straddles the ring's end
  const int64_t *durb = a.dur + ((int64_t)blockIdx.x * a.n_rows) * SIGMA;
  const uint32_t emask = RR * SIGMA - 1;
  uint32_t rows_done = 0, words_done = 0;
  auto issue_to = [&](uint32_t row_lim, uint32_t word_lim) {  // copy rows and words up to the limits
    if constexpr (SIGMA % 2 == 0) {
      const uint32_t e0 = rows_done * SIGMA, n16 = (row_lim - rows_done) * (SIGMA / 2);
      for (uint32_t t = tid; t < n16; t += blockDim.x) {
        const uint32_t e = e0 + 2 * t;
        cp_async16(dr + (e & emask), durb + e);
      }
    } else {
      for (uint32_t e = rows_done + tid; e < row_lim; e += blockDim.x) cp_async8(dr + (e & emask), durb + e);
    }
    for (uint32_t t = words_done + tid * 4; t < word_lim; t += blockDim.x * 4)
      cp_async16(&rr[t & rmask], &a.recs[t]);
    rows_done = row_lim;
    words_done = word_lim;
  };
  // group 0: the first metadata chunk and as many rows and words as the rings hold
  load_meta(0);
  issue_to(min(RR, a.n_rows), min(RB, a.n_words));
  cp_async_commit();
  int32_t g = 0;  // index of the last committed copy group
  if (tid == 0) hist[0] = make_uint2(rows_done, words_done);
  cp_async_wait<0>();
  __syncthreads();  // metadata and hist[0] visible to every thread

  const int j0 = (tid % TPN) * LANES;  // first scenario lane of this thread
  const int sub = tid / TPN;
  constexpr int kSegsPerStep = THREADS / TPN;
  int64_t mk[LANES];
#pragma unroll
  for (int k = 0; k < LANES; ++k) mk[k] = 0;
  uint32_t prev_i0 = 0, prev_ro = 0;  // level l-1 (still readable by slower threads)
  for (int32_t l = 0; l < a.L; ++l) {
    const int32_t kc = l / kMetaChunk;
    const int32_t cbase = kc * kMetaChunk;
    const bool new_chunk = l > 0 && l == cbase;
    if (new_chunk) load_meta(kc);  // its buffer was last used by chunk kc-2
    issue_to(min(prev_i0 + RR, a.n_rows), min(prev_ro + RB, a.n_words));
    cp_async_commit();
    ++g;
    if (tid == 0) hist[g & 15] = make_uint2(rows_done, words_done);
    const uint32_t *mb = meta_s + (kc & 1) * kMetaCap * 4 + 4 * (l - cbase);
    if (new_chunk) {
      cp_async_wait<0>();
    } else {
      // the oldest copy group that completes level l (look back at most 14 groups;
      // the slot of group g-16 is the one being rewritten now)
      const uint32_t need_rows = mb[4 + 1], need_words = mb[4];
      int32_t x = g;
      while (x > 0 && g - x < 14) {
        const uint2 ext = hist[(x - 1) & 15];
        if (ext.x >= need_rows && ext.y >= need_words)
          --x;
        else
          break;
      }
      cp_async_wait_dyn(g - x);
    }
    __syncthreads();

    const uint32_t ro = mb[0], i0 = mb[1], seg0 = mb[2];
    const int32_t nseg = (int32_t)(mb[4 + 2] - seg0);
    compose_segments<SIGMA, LANES>(a, ro, i0, seg0, nseg, sub, kSegsPerStep, j0, fr, vr, dr, rr, vmask, dmask,
                                   rmask, mk);
    prev_i0 = i0;
    prev_ro = ro;
  }
  cp_async_wait<0>();
#pragma unroll
  for (int j = 0; j < LANES; ++j) atomicMax((unsigned long long *)&mk_s[j0 + j], (unsigned long long)mk[j]);
  __syncthreads();
  if (tid < SIGMA && s0 + tid < S && a.makespan) a.makespan[s0 + tid] = mk_s[tid];
}

// -- mbarriers and 1-D bulk copies (TMA engine) ----------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;\n" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];\n" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok) : "r"(smem_u32(bar)), "r"(parity) : "memory");
  return ok != 0;
}
// wait for the phase of `parity` to complete; false once `limit` clock cycles pass
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity, long long limit) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity))
    if (clock64() - t0 > limit) return false;
  return true;
}
// addresses 16-byte aligned, size a multiple of 16; completes `bytes` on the mbarrier
__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes, uint64_t *bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];\n"
               ::"r"(smem_u32(dst)), "l"(src), "r"(bytes), "r"(smem_u32(bar)) : "memory");
}
// barrier over `threads` threads that also returns whether any of them passed `flag`
__device__ __forceinline__ bool named_barrier_or(int id, int threads, bool flag) {
  uint32_t any;
  asm volatile(
      "{\n .reg .pred pin, pout;\n setp.ne.u32 pin, %1, 0;\n bar.red.or.pred pout, %2, %3, pin;\n"
      " selp.u32 %0, 1, 0, pout;\n}\n"
      : "=r"(any) : "r"((uint32_t)flag), "r"(id), "r"(threads) : "memory");
  return any != 0;
}

// Pipelined compose (even SIGMA): the last warp is a producer that copies each
// segment level's duration rows, record block and metadata into the rings with the
// TMA engine (at most five 1-D bulk copies per level: this block's rows of a level
// are contiguous), as far ahead as the rings allow; kPipeConsumerWarps warps
// compose.  Stage l % kPipeStages has a "full" mbarrier (armed with the level's
// byte count) and an "empty" mbarrier (one arrival per consumer warp once the
// level is composed).  Every wait is bounded: on expiry the block records
// kDevTimeout, stops, and lets its copies in flight land first.
template <int SIGMA>
__global__ void __launch_bounds__((kPipeConsumerWarps + 1) * 32)
compose_pipelined_kernel(StagedArgs a) {
  constexpr int LANES = 2;
  constexpr int TPN = SIGMA / LANES;  // threads per segment
  constexpr int NB = kPipeStages;
  constexpr int NCT = kPipeConsumerWarps * 32;
  extern __shared__ __align__(16) unsigned char sbuf[];
  const int32_t S = a.S;
  const int32_t s0 = blockIdx.x * SIGMA;
  const int tid = threadIdx.x;
  const StagedLayout lay = staged_layout(a.n_queues, SIGMA, a.vlog2, a.dlog2, a.rlog2);
  const uint32_t vmask = (1u << a.vlog2) - 1, dmask = (1u << a.dlog2) - 1, rmask = (1u << a.rlog2) - 1;
  const uint32_t RR = dmask + 1, RB = rmask + 1;
  int64_t *mk_s = reinterpret_cast<int64_t *>(sbuf);                       // [SIGMA]
  uint64_t *full = reinterpret_cast<uint64_t *>(sbuf + lay.meta);          // [NB]
  uint64_t *empty = full + NB;                                              // [NB]
  uint32_t *hist = reinterpret_cast<uint32_t *>(sbuf + lay.meta + 256);    // [NB][2] producer only
  uint32_t *metas = reinterpret_cast<uint32_t *>(sbuf + lay.meta + 384);   // [NB][8]
  int64_t *fr = reinterpret_cast<int64_t *>(sbuf + lay.fr);
  int64_t *vr = reinterpret_cast<int64_t *>(sbuf + lay.vr);
  int64_t *dr = reinterpret_cast<int64_t *>(sbuf + lay.dr);
  uint32_t *rr = reinterpret_cast<uint32_t *>(sbuf + lay.rr);

  for (int k = tid; k < a.n_queues * SIGMA; k += blockDim.x) fr[k] = 0;
  if (tid < SIGMA) mk_s[tid] = 0;
  if (tid == 0) {
    for (int b = 0; b < NB; ++b) {
      mbar_init(&full[b], 1);  // the producer's arrive.expect_tx
      mbar_init(&empty[b], kPipeConsumerWarps);
    }
    asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
  }
  asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
  __syncthreads();

  if (tid >= NCT) {
    // ---------------- producer warp (one lane issues) ----------------
    const int lane = tid - NCT;
    if (lane == 0) {
      const int64_t *durb = a.dur + ((int64_t)blockIdx.x * a.n_rows) * SIGMA;
      const uint32_t emask = RR * SIGMA - 1;
      int32_t c_known = 0;  // every level < c_known has been composed
      int32_t issued = 0;   // levels [0, issued) have been armed
      bool fail = false;
      for (int32_t l = 0; l < a.L; ++l) {
        if (l == a.skip_level) break;  // failure injection: level l never arrives
        const uint4 m0 = *reinterpret_cast<const uint4 *>(a.meta + 4 * l);
        const uint4 m1 = *reinterpret_cast<const uint4 *>(a.meta + 4 * (l + 1));
        const uint32_t ro = m0.x, i0 = m0.y, ro1 = m1.x, i1 = m1.y;
        // ring space: level l overwrites rows and words of levels below c_known only
        while (c_known < l && (l - c_known >= NB || i1 > hist[2 * (c_known % NB)] + RR ||
                               ro1 > hist[2 * (c_known % NB) + 1] + RB)) {
          if (!mbar_wait(&empty[c_known % NB], (c_known / NB) & 1, a.wait_limit_cycles)) {
            fail = true;
            break;
          }
          ++c_known;
        }
        if (fail) break;
        hist[2 * (l % NB)] = i0;
        hist[2 * (l % NB) + 1] = ro;
        uint64_t *bar = &full[l % NB];
        const uint32_t e0 = i0 * SIGMA, ne = (i1 - i0) * SIGMA, w0 = ro & rmask, nw = ro1 - ro;
        mbar_arrive_expect_tx(bar, ne * 8 + nw * 4 + 32);
        const uint32_t ne1 = min(ne, emask + 1 - (e0 & emask));
        bulk_g2s(dr + (e0 & emask), durb + e0, ne1 * 8, bar);
        if (ne1 < ne) bulk_g2s(dr, durb + e0 + ne1, (ne - ne1) * 8, bar);
        const uint32_t nw1 = min(nw, RB - w0);
        bulk_g2s(rr + w0, a.recs + ro, nw1 * 4, bar);
        if (nw1 < nw) bulk_g2s(rr, a.recs + ro + nw1, (nw - nw1) * 4, bar);
        bulk_g2s(metas + 8 * (l % NB), a.meta + 4 * l, 32, bar);
        issued = l + 1;
      }
      if (fail) atomicCAS(a.status, 0, kDevTimeout);
      // let every copy this block started land before it exits
      for (int32_t x = max(c_known, issued - NB); x < issued; ++x)
        if (!mbar_wait(&full[x % NB], (x / NB) & 1, a.wait_limit_cycles)) atomicCAS(a.status, 0, kDevTimeout);
    }
    __syncwarp();
  } else {
    // ---------------- consumer warps ----------------
    const int j0 = (tid % TPN) * LANES;
    const int sub = tid / TPN;
    constexpr int kSegsPerStep = NCT / TPN;
    int64_t mk[LANES] = {0, 0};
    for (int32_t l = 0; l < a.L; ++l) {
      const bool ok = mbar_wait(&full[l % NB], (l / NB) & 1, a.wait_limit_cycles);
      if (ok) {
        const uint32_t *mb = metas + 8 * (l % NB);
        const uint32_t ro = mb[0], i0 = mb[1], seg0 = mb[2];
        const int32_t nseg = (int32_t)(mb[4 + 2] - seg0);
        compose_segments<SIGMA, LANES>(a, ro, i0, seg0, nseg, sub, kSegsPerStep, j0, fr, vr, dr, rr, vmask, dmask,
                                       rmask, mk);
      }
      // every consumer learns, in the same barrier, whether any of them gave up
      if (named_barrier_or(1, NCT, !ok)) {
        if (tid == 0) atomicCAS(a.status, 0, kDevTimeout);
        break;
      }
      if ((tid & 31) == 0) mbar_arrive(&empty[l % NB]);
    }
#pragma unroll
    for (int j = 0; j < LANES; ++j) atomicMax((unsigned long long *)&mk_s[j0 + j], (unsigned long long)mk[j]);
  }
  __syncthreads();
  if (tid < SIGMA && s0 + tid < S && a.makespan) a.makespan[s0 + tid] = mk_s[tid];
}

// ---------------------------------------------------------------------------------
// B3: validator overlap test.  One thread per (chunk of a rank's compute timeline,
// scenario); a warp covers 32 scenarios of one chunk and shares its op list.
// Every timeline of a rank runs its ops one after the other, so on each of the
// rank's comm timelines the intervals are sorted and the compute ops' starts only
// grow.  The thread keeps, per comm timeline, a cursor at the first comm op of
// positive length that finishes after the current compute op starts, with that
// op's interval in registers: the compute op overlaps this timeline iff that
// interval starts before the compute op finishes (any later comm op starts after
// the cursor op ends).  A binary search places the cursors at the chunk's first
// op; from there they only move forward, and only then touch memory.  A compute
// op of positive length that overlaps gets rint(d * slowdown) for the next
// composition (d_next), others keep d; the decisions themselves are stored only
// when `ov` is given.  The finish times and durations of 8 consecutive ops are
// loaded together before they are tested.
// ---------------------------------------------------------------------------------
constexpr int kOverlapThreads = 128;
constexpr int kOverlapBatch = 8;  // divides 32 (the shuffled op list's width)
template <int NCMAX>
__global__ void __launch_bounds__(kOverlapThreads) overlap_kernel(OverlapArgs a) {
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
  const int64_t c1 = min(a.q_off[r * a.n_streams + 1], c0 + kOverlapChunk);
  // element (i, s) of a matrix sits at base + (i << sh)
  const int sh = a.lay.slog2;
  const int64_t base = a.lay.at(0, sl);
  const int64_t *__restrict__ f = a.f + base;
  const int64_t *__restrict__ du = a.d_used + base;
  const bool same = a.d_orig == a.d_used;
  int32_t qreg = c0 + lane < c1 ? a.q_ops[c0 + lane] : 0;  // ops c0 .. c0+31 of the chunk
  int64_t cur[NCMAX], end[NCMAX], sw[NCMAX], fw[NCMAX];
  {
    const int64_t v = __shfl_sync(0xffffffffu, qreg, 0);
    const int64_t sv = act ? f[v << sh] - du[v << sh] : 0;
#pragma unroll
    for (int j = 0; j < NCMAX; ++j) {
      cur[j] = end[j] = 0;
      sw[j] = fw[j] = INT64_MAX;
      if (j < nc && act) {
        int64_t lo = a.cq_off[r * nc + j], hi = a.cq_off[r * nc + j + 1];
        end[j] = hi;
        while (lo < hi) {  // first comm op finishing after sv (finishes are sorted)
          const int64_t mid = (lo + hi) >> 1;
          if (f[(int64_t)a.cq_ops[mid] << sh] > sv)
            hi = mid;
          else
            lo = mid + 1;
        }
        cur[j] = lo;
        if (lo < end[j]) {
          const int64_t w = a.cq_ops[lo];
          fw[j] = f[w << sh];
          sw[j] = fw[j] - du[w << sh];
        }
      }
    }
  }
  // groups of kOverlapBatch ops: their finish times and durations are loaded together
  for (int64_t i0 = c0; i0 < c1; i0 += kOverlapBatch) {
    if (i0 > c0 && ((i0 - c0) & 31) == 0) qreg = i0 + lane < c1 ? a.q_ops[i0 + lane] : 0;
    int64_t vb[kOverlapBatch], fb[kOverlapBatch], db[kOverlapBatch];
#pragma unroll
    for (int u = 0; u < kOverlapBatch; ++u) {
      vb[u] = __shfl_sync(0xffffffffu, qreg, (int)((i0 - c0 + u) & 31));
      fb[u] = db[u] = 0;
      if (act && i0 + u < c1) {
        fb[u] = f[vb[u] << sh];
        db[u] = du[vb[u] << sh];
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
            // skip comm ops that ended by sv or have zero length
            while (cur[j] < end[j] && (fw[j] <= sv || sw[j] >= fw[j])) {
              if (++cur[j] < end[j]) {
                const int64_t w = a.cq_ops[cur[j]];
                fw[j] = f[w << sh];
                sw[j] = fw[j] - du[w << sh];
              } else {
                sw[j] = fw[j] = INT64_MAX;
              }
            }
            hit |= sw[j] < fv;
          }
        }
        hit = hit && sv < fv;
        const int64_t at = base + (v << sh);
        if (a.ov) a.ov[at] = hit;
        if (a.d_next) {
          const int64_t d0 = same ? dv : a.d_orig[at];
          a.d_next[at] = hit ? slowed(d0, a.sf[(int64_t)a.kcl[v] * S + sl]) : d0;
        }
      }
    }
  }
}

__global__ void copy_rows_kernel(const int32_t *__restrict__ rows, int64_t n_rows, int32_t S, MatLayout lay,
                                 const int64_t *__restrict__ src, int64_t *__restrict__ dst) {
  int64_t total = n_rows * S;
  for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
       idx += (int64_t)gridDim.x * blockDim.x) {
    int64_t k = idx / S;
    int64_t at = lay.at(rows[k], (int32_t)(idx - k * S));
    dst[at] = src[at];
  }
}

// ---------------------------------------------------------------------------------
// readback: internal order and blocked layout -> caller order, [op][scenario]
// ---------------------------------------------------------------------------------
__global__ void readback_kernel(const int32_t *__restrict__ ext2int, int64_t op0, int64_t op1, int32_t S,
                                MatLayout lay, const int64_t *__restrict__ f, const int64_t *__restrict__ d,
                                int64_t *__restrict__ start, int64_t *__restrict__ finish) {
  int64_t total = (op1 - op0) * S;
  for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
       idx += (int64_t)gridDim.x * blockDim.x) {
    int64_t o = idx / S;
    int32_t s = (int32_t)(idx - o * S);
    int64_t at = lay.at(ext2int[op0 + o], s);
    int64_t fv = f[at];
    if (start) start[idx] = fv - d[at];
    if (finish) finish[idx] = fv;
  }
}

__global__ void read_cc_kernel(const int32_t *__restrict__ ext2int, int64_t op0, int64_t op1, int32_t S,
                               const int32_t *__restrict__ node_sig, const double *__restrict__ cc_ns,
                               double *__restrict__ out) {
  int64_t total = (op1 - op0) * S;
  for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
       idx += (int64_t)gridDim.x * blockDim.x) {
    int64_t o = idx / S;
    int32_t s = (int32_t)(idx - o * S);
    int32_t g = node_sig[ext2int[op0 + o]];
    out[idx] = g >= 0 ? cc_ns[(int64_t)g * S + s] : __longlong_as_double(0x7ff8000000000000LL);
  }
}

__global__ void read_ov_kernel(const int32_t *__restrict__ ext2int, int64_t op0, int64_t op1, int32_t S,
                               MatLayout lay, const uint8_t *__restrict__ ov, const uint8_t *__restrict__ kcl,
                               uint8_t *__restrict__ out) {
  int64_t total = (op1 - op0) * S;
  for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
       idx += (int64_t)gridDim.x * blockDim.x) {
    int64_t o = idx / S;
    int32_t s = (int32_t)(idx - o * S);
    int64_t i = ext2int[op0 + o];
    out[idx] = (ov && kcl[i] != kNotSlowable) ? ov[lay.at(i, s)] : 0;  // only compute ops are tested
  }
}

int grid_for(int64_t n, int threads) {
  int64_t b = (n + threads - 1) / threads;
  if (b < 1) b = 1;
  if (b > 152 * 32) b = 152 * 32;
  return (int)b;
}

template <int SIGMA>
cudaError_t launch_compose_t(const ComposeArgs &a, cudaStream_t st) {
  bool in_smem = false;
  size_t smem = compose_smem_bytes(a.n_queues, SIGMA, &in_smem);
  dim3 grid((a.S + SIGMA - 1) / SIGMA);
  if (in_smem) {
    auto k = compose_direct_kernel<SIGMA, true>;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    k<<<grid, kComposeThreads, smem, st>>>(a);
  } else {
    auto k = compose_direct_kernel<SIGMA, false>;
    k<<<grid, kComposeThreads, smem, st>>>(a);
  }
  return cudaGetLastError();
}

template <int SIGMA, int THREADS>
cudaError_t launch_staged_t(const StagedArgs &a, const StagedPlan &plan, cudaStream_t st) {
  auto k = compose_staged_kernel<SIGMA, THREADS>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)plan.smem);
  if (e != cudaSuccess) return e;
  dim3 grid((a.S + SIGMA - 1) / SIGMA);
  k<<<grid, THREADS, plan.smem, st>>>(a);
  return cudaGetLastError();
}

template <int SIGMA>
cudaError_t launch_pipelined_t(const StagedArgs &a, const StagedPlan &plan, cudaStream_t st) {
  auto k = compose_pipelined_kernel<SIGMA>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)plan.smem);
  if (e != cudaSuccess) return e;
  dim3 grid((a.S + SIGMA - 1) / SIGMA);
  k<<<grid, (kPipeConsumerWarps + 1) * 32, plan.smem, st>>>(a);
  return cudaGetLastError();
}

}  // namespace

size_t compose_smem_bytes(int32_t n_queues, int sigma, bool *frontier_in_smem) {
  size_t fr = (size_t)n_queues * sigma * sizeof(int64_t);
  size_t base = (size_t)sigma * sizeof(int64_t);
  bool in = fr + base <= (size_t)200 * 1024;
  if (frontier_in_smem) *frontier_in_smem = in;
  return in ? fr + base : base;
}

cudaError_t launch_cc_estimate(const CcSig *sig, int32_t G, ScenParams p, int32_t S, const ChunkTable &tbl,
                               const int32_t *sig_count, double *cc_ns, int64_t *cc_dur, double *comm_sum,
                               int32_t *status, cudaStream_t st) {
  int64_t n = (int64_t)G * S;
  if (n == 0) return cudaSuccess;
  int threads = 256;
  int64_t blocks = (n + threads - 1) / threads;
  cc_estimate_kernel<<<(unsigned)blocks, threads, 0, st>>>(sig, G, p, S, tbl, sig_count, cc_ns, cc_dur,
                                                          comm_sum, status);
  return cudaGetLastError();
}

cudaError_t launch_cc_scatter(const int32_t *comm_node, const int32_t *comm_sig, int64_t n_comm,
                              const int64_t *cc_dur, int32_t S, MatLayout lay, int64_t *dur, cudaStream_t st) {
  if (n_comm == 0) return cudaSuccess;
  cc_scatter_kernel<<<grid_for(n_comm * S, 256), 256, 0, st>>>(comm_node, comm_sig, n_comm, cc_dur, S, lay, dur);
  return cudaGetLastError();
}

cudaError_t launch_cc_query(int64_t n, const uint8_t *type, const uint8_t *algo, const int64_t *nbytes,
                            const int32_t *N, const int32_t *M, const double *lg, ScenParams p,
                            const ChunkTable &tbl, double *out, cudaStream_t st) {
  if (n == 0) return cudaSuccess;
  cc_query_kernel<<<grid_for(n, 256), 256, 0, st>>>(n, type, algo, nbytes, N, M, lg, p, tbl, out);
  return cudaGetLastError();
}

cudaError_t launch_permute_rows(const int64_t *raw, const int32_t *int2ext, const uint8_t *local, int64_t V,
                                int32_t S, MatLayout lay, int64_t *dur, double *sums, int32_t *status,
                                cudaStream_t st) {
  if (V == 0 || S == 0) return cudaSuccess;
  int tx = S >= 128 ? 128 : ((S + 31) / 32) * 32;
  dim3 block(tx);
  int64_t gy = V < 8192 ? V : 8192;
  dim3 grid((S + tx - 1) / tx, (unsigned)gy);
  permute_rows_kernel<<<grid, block, 0, st>>>(raw, int2ext, local, V, S, lay, dur, sums, status);
  return cudaGetLastError();
}

cudaError_t launch_compose(const ComposeArgs &a, int sigma, cudaStream_t st) {
  if (a.S == 0) return cudaSuccess;
  switch (sigma) {
    case 1: return launch_compose_t<1>(a, st);
    case 2: return launch_compose_t<2>(a, st);
    case 4: return launch_compose_t<4>(a, st);
    case 8: return launch_compose_t<8>(a, st);
    case 16: return launch_compose_t<16>(a, st);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_compose_staged(const StagedArgs &a, int sigma, const StagedPlan &plan, cudaStream_t st) {
  if (a.S == 0) return cudaSuccess;
  switch (sigma * 10000 + plan.threads) {
    case 1 * 10000 + 256: return launch_staged_t<1, 256>(a, plan, st);
    case 1 * 10000 + 512: return launch_staged_t<1, 512>(a, plan, st);
    case 1 * 10000 + 1024: return launch_staged_t<1, 1024>(a, plan, st);
    case 2 * 10000 + 256: return launch_staged_t<2, 256>(a, plan, st);
    case 2 * 10000 + 512: return launch_staged_t<2, 512>(a, plan, st);
    case 4 * 10000 + 256: return launch_staged_t<4, 256>(a, plan, st);
    case 4 * 10000 + 512: return launch_staged_t<4, 512>(a, plan, st);
    case 8 * 10000 + 512: return launch_staged_t<8, 512>(a, plan, st);
    case 16 * 10000 + 1024: return launch_staged_t<16, 1024>(a, plan, st);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_compose_pipelined(const StagedArgs &a, int sigma, const StagedPlan &plan, cudaStream_t st) {
  if (a.S == 0) return cudaSuccess;
  switch (sigma) {
    case 2: return launch_pipelined_t<2>(a, plan, st);
    case 4: return launch_pipelined_t<4>(a, plan, st);
    case 8: return launch_pipelined_t<8>(a, plan, st);
    case 16: return launch_pipelined_t<16>(a, plan, st);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_overlap(const OverlapArgs &a, cudaStream_t st) {
  if (a.S == 0 || a.n_chunks == 0) return cudaSuccess;
  if (a.n_cq < 0 || a.n_cq > kMaxStreams) return cudaErrorInvalidValue;
  const int tx = a.S >= kOverlapThreads ? kOverlapThreads : ((a.S + 31) / 32) * 32;
  int64_t gy = a.n_chunks < 65535 ? a.n_chunks : 65535;
  int64_t gz = (a.n_chunks + gy - 1) / gy;
  dim3 grid((a.S + tx - 1) / tx, (unsigned)gy, (unsigned)gz);
  if (a.n_cq <= 1)
    overlap_kernel<1><<<grid, tx, 0, st>>>(a);
  else if (a.n_cq <= 2)
    overlap_kernel<2><<<grid, tx, 0, st>>>(a);
  else if (a.n_cq <= 3)
    overlap_kernel<3><<<grid, tx, 0, st>>>(a);
  else if (a.n_cq <= 4)
    overlap_kernel<4><<<grid, tx, 0, st>>>(a);
  else if (a.n_cq <= 8)
    overlap_kernel<8><<<grid, tx, 0, st>>>(a);
  else
    overlap_kernel<kMaxStreams><<<grid, tx, 0, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_copy_rows(const int32_t *rows, int64_t n_rows, int32_t S, MatLayout lay, const int64_t *src,
                             int64_t *dst, cudaStream_t st) {
  if (n_rows == 0 || S == 0) return cudaSuccess;
  copy_rows_kernel<<<grid_for(n_rows * S, 256), 256, 0, st>>>(rows, n_rows, S, lay, src, dst);
  return cudaGetLastError();
}

cudaError_t launch_readback(const int32_t *ext2int, int64_t op0, int64_t op1, int32_t S, MatLayout lay,
                            const int64_t *f, const int64_t *d, int64_t *start, int64_t *finish, cudaStream_t st) {
  int64_t n = (op1 - op0) * S;
  if (n <= 0) return cudaSuccess;
  readback_kernel<<<grid_for(n, 256), 256, 0, st>>>(ext2int, op0, op1, S, lay, f, d, start, finish);
  return cudaGetLastError();
}

cudaError_t launch_read_cc(const int32_t *ext2int, int64_t op0, int64_t op1, int32_t S, const int32_t *node_sig,
                           const double *cc_ns, double *out, cudaStream_t st) {
  int64_t n = (op1 - op0) * S;
  if (n <= 0) return cudaSuccess;
  read_cc_kernel<<<grid_for(n, 256), 256, 0, st>>>(ext2int, op0, op1, S, node_sig, cc_ns, out);
  return cudaGetLastError();
}

cudaError_t launch_read_ov(const int32_t *ext2int, int64_t op0, int64_t op1, int32_t S, MatLayout lay,
                           const uint8_t *ov, const uint8_t *kcl, uint8_t *out, cudaStream_t st) {
  int64_t n = (op1 - op0) * S;
  if (n <= 0) return cudaSuccess;
  read_ov_kernel<<<grid_for(n, 256), 256, 0, st>>>(ext2int, op0, op1, S, lay, ov, kcl, out);
  return cudaGetLastError();
}

}  // namespace echo

// ---------------------------------------------------------------------------------
// Allocation-free CC queries.
//
// Some callers cannot call cudaMalloc: a process whose device memory is owned by a
// framework's memory pool (a stray allocation would fail or fragment that pool), or
// one that runs under a fixed per-process memory budget.  echo_cc_query_noalloc
// serves them: the caller passes device arrays in and out, and the only other
// device memory the kernel touches is the file-scope array below, which every GPU
// that loads this library holds until the process exits.
//
// Layout of the array: bytes [0, 4) hold a status word, cleared at the start of
// every call; from byte 256 on, log2(m) for m = 0..kNoallocMaxNodes, computed on
// the host with the same libm log2 the allocating path uses, so both paths give
// identical estimates.  Node counts above kNoallocMaxNodes are rejected.
// ---------------------------------------------------------------------------------
namespace echo {
namespace {
constexpr int32_t kNoallocMaxNodes = 65536;
constexpr size_t kNoallocLgOffset = 256;
constexpr size_t kNoallocScratchBytes = kNoallocLgOffset + sizeof(double) * (kNoallocMaxNodes + 1);
constexpr int kNoallocMaxDevices = 64;
enum : int32_t { kNoallocOk = 0, kNoallocTooManyNodes = 1, kNoallocBadQuery = 2 };
}  // namespace
}  // namespace echo

static __device__ __align__(256) unsigned char g_noalloc_scratch[echo::kNoallocScratchBytes];

namespace echo {
namespace {

struct NoallocDevice {
  std::once_flag once;
  unsigned char *ptr = nullptr;  // device address of g_noalloc_scratch on this device
  cudaError_t err = cudaSuccess;
};
NoallocDevice g_noalloc_devices[kNoallocMaxDevices];

// Once per device, with that device current: look up the array's device address
// (host code cannot use the symbol itself) and fill the log2 table.
void noalloc_setup(NoallocDevice &d) {
  void *p = nullptr;
  d.err = cudaGetSymbolAddress(&p, g_noalloc_scratch);
  if (d.err != cudaSuccess) return;
  std::vector<double> lg(kNoallocMaxNodes + 1, 0.0);
  for (int32_t m = 1; m <= kNoallocMaxNodes; ++m) lg[m] = std::log2((double)m);
  unsigned char *base = static_cast<unsigned char *>(p);
  d.err = cudaMemcpy(base + kNoallocLgOffset, lg.data(), lg.size() * sizeof(double), cudaMemcpyHostToDevice);
  if (d.err != cudaSuccess) return;
  d.ptr = base;
}

__device__ __forceinline__ bool nonneg_finite(double x) { return isfinite(x) && x >= 0.0; }

// Same estimate as cc_query_kernel; log2(M) comes from the table in the static
// array and each query is checked on the device, since its fields live there.
__global__ void cc_query_noalloc_kernel(int64_t n, const uint8_t *__restrict__ type,
                                        const uint8_t *__restrict__ algo, const int64_t *__restrict__ nbytes,
                                        const int32_t *__restrict__ N, const int32_t *__restrict__ M,
                                        ScenParams p, ChunkTable tbl, unsigned char *scratch,
                                        double *__restrict__ out) {
  int32_t *status = reinterpret_cast<int32_t *>(scratch);
  const double *lg = reinterpret_cast<const double *>(scratch + kNoallocLgOffset);
  const double nan = __longlong_as_double(0x7ff8000000000000LL);
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int t = type[i], a = algo[i];
    const int n_r = N[i], m = M[i];
    const int64_t nb = nbytes[i];
    const bool ok = t <= kSR && (t != kAR || a <= 2) && nb >= 0 && n_r >= 1 && m >= 1 && m <= n_r &&
                    nonneg_finite(p.alpha[i]) && nonneg_finite(p.lata[i]) && nonneg_finite(p.late[i]) &&
                    nonneg_finite(p.delta[i]) && isfinite(p.bwa[i]) && p.bwa[i] > 0.0 &&
                    isfinite(p.bwe[i]) && p.bwe[i] > 0.0;
    if (!ok) {
      out[i] = nan;
      set_status(status, kNoallocBadQuery);
      continue;
    }
    if (m > kNoallocMaxNodes) {
      out[i] = nan;
      set_status(status, kNoallocTooManyNodes);
      continue;
    }
    const int K = (n_r + m - 1) / m;
    out[i] = cc_ns_of(t, a, nb, n_r, m, K, lg[m], p.alpha[i], p.bwa[i], p.lata[i], p.bwe[i], p.late[i],
                      p.delta[i], tbl);
  }
}

}  // namespace
}  // namespace echo

extern "C" int echo_cc_query_noalloc(const echo_cc_query_desc *q, double *out_ns, void *cuda_stream) {
  using namespace echo;
  if (!q || q->n < 0) return ECHO_E_INVALID_ARG;
  if (q->n == 0) return ECHO_OK;
  if (!out_ns || !q->cc_type || !q->cc_algo || !q->nbytes || !q->n_ranks || !q->n_nodes || !q->alpha_ns ||
      !q->bw_intra || !q->lat_intra || !q->bw_inter || !q->lat_inter || !q->delta)
    return ECHO_E_INVALID_ARG;
  // the chunk table is a few host values passed by value to the kernel
  ChunkTable tbl;
  std::memset(&tbl, 0, sizeof tbl);
  if (q->n_chunk == 0) {
    const int64_t mx[5] = {4LL << 20, 8LL << 20, 64LL << 20, 128LL << 20, INT64_MAX};
    const int64_t cb[5] = {18000, 36000, 72000, 144000, 288000};
    tbl.n = 5;
    for (int i = 0; i < 5; ++i) {
      tbl.max_bytes[i] = mx[i];
      tbl.chunk[i] = cb[i];
    }
  } else {
    if (q->n_chunk < 0 || q->n_chunk > kMaxChunk) return ECHO_E_UNSUPPORTED;
    if (!q->chunk_max_bytes || !q->chunk_bytes) return ECHO_E_INVALID_ARG;
    tbl.n = q->n_chunk;
    for (int i = 0; i < q->n_chunk; ++i) {
      if (q->chunk_bytes[i] <= 0 || (i > 0 && q->chunk_max_bytes[i] < q->chunk_max_bytes[i - 1]))
        return ECHO_E_INVALID_ARG;
      tbl.max_bytes[i] = q->chunk_max_bytes[i];
      tbl.chunk[i] = q->chunk_bytes[i];
    }
  }
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kNoallocMaxDevices) return ECHO_E_CUDA;
  NoallocDevice &d = g_noalloc_devices[dev];
  std::call_once(d.once, noalloc_setup, std::ref(d));
  if (d.err != cudaSuccess || !d.ptr) return ECHO_E_CUDA;
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  if (cudaMemsetAsync(d.ptr, 0, sizeof(int32_t), st) != cudaSuccess) return ECHO_E_CUDA;
  ScenParams p{q->alpha_ns, q->bw_intra, q->lat_intra, q->bw_inter, q->lat_inter, q->delta};
  cc_query_noalloc_kernel<<<grid_for(q->n, 256), 256, 0, st>>>(q->n, q->cc_type, q->cc_algo, q->nbytes,
                                                                q->n_ranks, q->n_nodes, p, tbl, d.ptr, out_ns);
  if (cudaGetLastError() != cudaSuccess) return ECHO_E_CUDA;
  int32_t status = 0;
  if (cudaMemcpyAsync(&status, d.ptr, sizeof(int32_t), cudaMemcpyDeviceToHost, st) != cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess)
    return ECHO_E_CUDA;
  if (status == kNoallocTooManyNodes) return ECHO_E_UNSUPPORTED;
  if (status == kNoallocBadQuery) return ECHO_E_INVALID_ARG;
  return ECHO_OK;
}
