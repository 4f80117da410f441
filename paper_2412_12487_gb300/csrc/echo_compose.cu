// echo_compose.cu -- sm_103a composition kernels (Sec. 4.2, 5.2): the levelled
// max-plus pass over the multi-rank execution graph, batched over scenario blocks.
#include <cuda_runtime.h>

#include <cstdint>

#include "echo_internal.h"

namespace echo {

namespace {

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
        if (a.dbg && !(range_ok(h, z + 1, a.V) && h <= z)) {  // debug bounds: skip a bad segment
          atomicCAS(a.status, 0, (int32_t)kDevBounds);
          continue;
        }
        int64_t fv = 0;  // the head starts after its timelines and data predecessors
        for (int64_t k = a.nq_off[h]; k < a.nq_off[h + 1]; ++k) {
          const int64_t q = a.nq[k];
          if (a.dbg && !in_range(q, a.n_queues)) {
            atomicCAS(a.status, 0, (int32_t)kDevBounds);
            continue;
          }
          fv = max(fv, fr[q * SIGMA + j]);
        }
        for (int64_t k = a.dp_off[h]; k < a.dp_off[h + 1]; ++k) {
          const int64_t u = a.dp[k];
          if (a.dbg && !in_range(u, a.V)) {
            atomicCAS(a.status, 0, (int32_t)kDevBounds);
            continue;
          }
          fv = max(fv, f[a.lay.at(u, s)]);
        }
        for (int64_t i = h; i <= z; ++i) {  // along the chain every op starts when the previous ends
          fv += dur[a.lay.at(i, s)];
          f[a.lay.at(i, s)] = fv;
        }
        for (int64_t k = a.nq_off[z]; k < a.nq_off[z + 1]; ++k) {
          const int64_t q = a.nq[k];
          if (a.dbg && !in_range(q, a.n_queues)) {
            atomicCAS(a.status, 0, (int32_t)kDevBounds);
            continue;
          }
          fr[q * SIGMA + j] = fv;
        }
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

// Debug bounds (out of line, off the hot path): the segment's chain rows, its
// candidates' compact rows, every input's value-ring slot and far row.  A failed
// check records kDevBounds.
__device__ __noinline__ bool segment_ok(const StagedArgs &a, uint32_t first, uint32_t len, uint64_t cmask,
                                        uint32_t c_first, uint32_t rr_a, uint32_t rmask, uint32_t e, uint32_t nin,
                                        uint32_t nfar, uint32_t ring_bytes, uint32_t row_bytes) {
  bool ok = len > 0 && range_ok(first, (int64_t)first + len, a.n_rows) && masked_row_ok(c_first, cmask, a.n_cand);
  for (uint32_t x = 0; ok && x < nin + nfar; ++x) {
    uint32_t w;
    asm volatile("ld.shared.u32 %0, [%1];\n" : "=r"(w) : "r"(rr_a + ((e + x) & rmask) * 4));
    ok = x < nin ? (w < ring_bytes && w % row_bytes == 0) : in_range(w, a.n_rows);
  }
  if (!ok) atomicCAS(a.status, 0, (int32_t)kDevBounds);
  return ok;
}

// Compose the segments of one segment level (shared by the staged and the
// pipelined kernels).  Segment k's header and entries are in the record ring at
// word `ro`; its rows are i0 + header.z ... (global rows), held in the duration
// ring of RR rows from ring row dpos0 + header.z on (wrapping).  Candidate rows of
// the level start at level-order index c0, in ring row cpos0 of the CRR-row
// candidate ring.  Thread `sub` handles segments sub, sub + step, ... for scenario
// lanes j0 .. j0+LANES-1; the segments of a level come heaviest first, so a warp's
// lanes hold segments of similar weight.  Every input of a head is the tail of an earlier segment: the
// recent ones are read from the value ring (entries are byte offsets of their
// slots), older ones from global memory (entries are node ids).  Inputs and
// durations are loaded four at a time so that their latencies overlap.  This
// block's finish rows are a contiguous [V][SIGMA] array (padding lanes included),
// so every row moves as whole vectors.
template <int SIGMA, int LANES, bool STORE_ALL, bool DBG>
__device__ __forceinline__ void compose_segments(const StagedArgs &a, uint32_t ro, uint32_t i0, uint32_t seg0,
                                                 int32_t nseg, int sub, int step, int j0, int64_t *vr,
                                                 const int64_t *dr, const uint32_t *rr, uint32_t vmask,
                                                 uint32_t dpos0, uint32_t RR, uint32_t rmask, int64_t (&mk)[LANES],
                                                 const int64_t *cr = nullptr, uint32_t cpos0 = 0, uint32_t c0 = 0,
                                                 uint32_t CRR = 0) {
  int64_t *fb = a.f + ((int64_t)blockIdx.x * a.n_rows) * SIGMA;
  const uint32_t vr_a = saddr(vr) + j0 * 8, dr_a = saddr(dr) + j0 * 8;
  const uint32_t rr_a = saddr(rr);
  const uint32_t cr_a = cr ? saddr(cr) + j0 * 8 : 0;
  constexpr uint32_t kRowBytes = SIGMA * 8;
  auto word = [&](uint32_t w) { return s_ld32(rr_a + (w & rmask) * 4); };
  for (int32_t k = sub; k < nseg; k += step) {
    const uint4 hd = s_ld128(rr_a + ((ro + 4 * k) & rmask) * 4);
    const uint32_t nin = hd.y & 0xFFFFu, nfar = hd.y >> 16;
    const uint32_t len = hd.w & 0xFFFFu;
    // chain positions whose duration the validator rewrote (second and later passes)
    const bool has_c = (hd.w >> 16) & 1, has_k = (hd.w >> 17) & 1;
    const uint32_t ec = ro + hd.x + nin + nfar;
    uint64_t cmask_bits = 0;
    uint32_t c_first = 0;
    if (cr && has_c) {
      cmask_bits = (uint64_t)word(ec) | ((uint64_t)word(ec + 1) << 32);
      c_first = word(ec + 2);
    }
    // chain positions whose finish is stored: all in the final composition; else
    // the tail (later heads read it) and those a later step reads (kept mask)
    uint64_t smask = ~0ull;
    if (!STORE_ALL) {
      smask = 1ull << (len - 1);
      if (has_k) {
        const uint32_t ek = ec + (has_c ? 3 : 0);
        smask |= (uint64_t)word(ek) | ((uint64_t)word(ek + 1) << 32);
      }
    }
    // a candidate's duration comes from the candidate ring instead of the duration ring
    // (the level's candidates span at most CRR rows, so one wrap suffices)
    auto patch = [&](uint32_t t, int64_t (&d)[LANES]) {
      if ((cmask_bits >> t) & 1) {
        uint32_t x = cpos0 + (c_first - c0) + (uint32_t)__popcll(cmask_bits & ((1ull << t) - 1));
        if (x >= CRR) x -= CRR;
        s_load<LANES>(cr_a + x * kRowBytes, d);
      }
    };
    const uint32_t e = ro + hd.x;
    const uint32_t first = i0 + hd.z;
    if (DBG && !segment_ok(a, first, len, cmask_bits, c_first, rr_a, rmask, e, nin, nfar, (vmask + 1) * kRowBytes,
                             kRowBytes))
      continue;  // debug bounds: a bad index skips the segment
    int64_t fv[LANES];
#pragma unroll
    for (int j = 0; j < LANES; ++j) fv[j] = 0;
    uint32_t q = 0;
    for (; q + 4 <= nin; q += 4) {
      const uint32_t o0 = word(e + q), o1 = word(e + q + 1), o2 = word(e + q + 2), o3 = word(e + q + 3);
      int64_t v0[LANES], v1[LANES], v2[LANES], v3[LANES];
      s_load<LANES>(vr_a + o0, v0);
      s_load<LANES>(vr_a + o1, v1);
      s_load<LANES>(vr_a + o2, v2);
      s_load<LANES>(vr_a + o3, v3);
#pragma unroll
      for (int j = 0; j < LANES; ++j) fv[j] = max(max(fv[j], max(v0[j], v1[j])), max(v2[j], v3[j]));
    }
    for (; q < nin; ++q) s_max<LANES>(fv, vr_a + word(e + q));
    for (uint32_t t = 0; t < nfar; t += 2) {
      const uint32_t u0 = word(e + nin + t), u1 = t + 1 < nfar ? word(e + nin + t + 1) : u0;
      g_max<LANES>(fv, fb + (int64_t)u0 * SIGMA + j0);
      g_max<LANES>(fv, fb + (int64_t)u1 * SIGMA + j0);
    }
    // along the chain every op starts when the previous one ends; p is the ring
    // row of chain position t (a level's rows span at most RR rows)
    int64_t *gp = fb + (int64_t)first * SIGMA + j0;
    uint32_t p = dpos0 + hd.z;
    if (p >= RR) p -= RR;
    auto next = [&](uint32_t x) { return x + 1 == RR ? 0u : x + 1; };
    uint32_t t = 0;
    for (; t + 4 <= len; t += 4, gp += 4 * SIGMA) {
      int64_t d0[LANES], d1[LANES], d2[LANES], d3[LANES];
      const uint32_t p1 = next(p), p2 = next(p1), p3 = next(p2);
      s_load<LANES>(dr_a + p * kRowBytes, d0);
      s_load<LANES>(dr_a + p1 * kRowBytes, d1);
      s_load<LANES>(dr_a + p2 * kRowBytes, d2);
      s_load<LANES>(dr_a + p3 * kRowBytes, d3);
      p = next(p3);
      if (cmask_bits) {
        patch(t, d0);
        patch(t + 1, d1);
        patch(t + 2, d2);
        patch(t + 3, d3);
      }
      const uint32_t sb = (uint32_t)(smask >> t);
#pragma unroll
      for (int j = 0; j < LANES; ++j) fv[j] += d0[j];
      if (STORE_ALL || (sb & 1)) g_store<LANES>(gp, fv);
#pragma unroll
      for (int j = 0; j < LANES; ++j) fv[j] += d1[j];
      if (STORE_ALL || (sb & 2)) g_store<LANES>(gp + SIGMA, fv);
#pragma unroll
      for (int j = 0; j < LANES; ++j) fv[j] += d2[j];
      if (STORE_ALL || (sb & 4)) g_store<LANES>(gp + 2 * SIGMA, fv);
#pragma unroll
      for (int j = 0; j < LANES; ++j) fv[j] += d3[j];
      if (STORE_ALL || (sb & 8)) g_store<LANES>(gp + 3 * SIGMA, fv);
    }
    for (; t < len; ++t, gp += SIGMA, p = next(p)) {
      int64_t d[LANES];
      s_load<LANES>(dr_a + p * kRowBytes, d);
      if (cmask_bits) patch(t, d);
#pragma unroll
      for (int j = 0; j < LANES; ++j) fv[j] += d[j];
      if (STORE_ALL || ((smask >> t) & 1)) g_store<LANES>(gp, fv);
    }
#pragma unroll
    for (int j = 0; j < LANES; ++j) mk[j] = max(mk[j], fv[j]);
    s_store<LANES>(vr_a + ((seg0 + k) & vmask) * kRowBytes, fv);
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
  const uint32_t vmask = (1u << a.vlog2) - 1, dmask = (1u << a.dlog2) - 1, rmask = (1u << a.rlog2) - 1;
  const uint32_t RR = dmask + 1, RB = rmask + 1;
  const StagedLayout lay = staged_layout(SIGMA, a.vlog2, RR, a.rlog2, (size_t)1 << a.clog2);
  int64_t *mk_s = reinterpret_cast<int64_t *>(sbuf);                  // [SIGMA]
  uint2 *hist = reinterpret_cast<uint2 *>(sbuf + lay.hist);           // [16] (rows, words) copied by group
  uint32_t *meta_s = reinterpret_cast<uint32_t *>(sbuf + lay.meta);   // [2][kMetaCap][4]
  int64_t *vr = reinterpret_cast<int64_t *>(sbuf + lay.vr);           // [value ring][SIGMA]
  int64_t *dr = reinterpret_cast<int64_t *>(sbuf + lay.dr);           // [duration ring][SIGMA]
  uint32_t *rr = reinterpret_cast<uint32_t *>(sbuf + lay.rr);         // [record ring]

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
    if (a.dbg)
      compose_segments<SIGMA, LANES, true, true>(a, ro, i0, seg0, nseg, tid / TPN, THREADS / TPN, j0, vr, dr, rr,
                                                 vmask, i0 & dmask, RR, rmask, mk);
    else if (a.store_all)
      compose_segments<SIGMA, LANES, true, false>(a, ro, i0, seg0, nseg, tid / TPN, THREADS / TPN, j0, vr, dr, rr,
                                                  vmask, i0 & dmask, RR, rmask, mk);
    else
      compose_segments<SIGMA, LANES, false, false>(a, ro, i0, seg0, nseg, tid / TPN, THREADS / TPN, j0, vr, dr, rr,
                                                   vmask, i0 & dmask, RR, rmask, mk);
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
// compose, one scenario per thread up to SIGMA 8 (a segment's SIGMA threads
// share its walk), two above.  The duration and candidate rings hold any number
// of rows (a.d_rows, a.c_rows: all the shared memory the rest leaves), so the
// producer writes each level's first ring rows beside its metadata.  Stage
// l % kPipeStages has a "full" mbarrier (armed with the level's byte count) and
// an "empty" mbarrier (one arrival per consumer warp once the level is composed).  Every wait is bounded: on expiry the block records
// kDevTimeout, stops, and lets its copies in flight land first.
template <int SIGMA, bool STORE_ALL, bool DBG>
__global__ void __launch_bounds__((kPipeConsumerWarps + 1) * 32)
compose_pipelined_kernel(StagedArgs a) {
  constexpr int LANES = SIGMA <= 8 ? 1 : 2;
  constexpr int TPN = SIGMA / LANES;  // threads per segment
  constexpr int NB = kPipeStages;
  constexpr int NCT = kPipeConsumerWarps * 32;
  extern __shared__ __align__(16) unsigned char sbuf[];
  const int32_t S = a.S;
  const int32_t s0 = blockIdx.x * SIGMA;
  const int tid = threadIdx.x;
  const StagedLayout lay = staged_layout(SIGMA, a.vlog2, a.d_rows, a.rlog2, a.c_rows);
  const uint32_t vmask = (1u << a.vlog2) - 1, rmask = (1u << a.rlog2) - 1;
  const uint32_t RR = a.d_rows, RB = rmask + 1, CRR = a.c_rows;
  int64_t *mk_s = reinterpret_cast<int64_t *>(sbuf);                       // [SIGMA]
  uint64_t *full = reinterpret_cast<uint64_t *>(sbuf + lay.meta);          // [NB]
  uint64_t *empty = full + NB;                                              // [NB]
  uint32_t *hist = reinterpret_cast<uint32_t *>(sbuf + lay.meta + 256);    // [NB][4] producer only
  uint32_t *metas = reinterpret_cast<uint32_t *>(sbuf + lay.meta + 512);   // [NB][8]
  uint32_t *pos = reinterpret_cast<uint32_t *>(sbuf + lay.meta + 1024);    // [NB][2] first ring rows
  int64_t *vr = reinterpret_cast<int64_t *>(sbuf + lay.vr);
  int64_t *dr = reinterpret_cast<int64_t *>(sbuf + lay.dr);
  uint32_t *rr = reinterpret_cast<uint32_t *>(sbuf + lay.rr);
  int64_t *cr = reinterpret_cast<int64_t *>(sbuf + lay.cr);

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
      const int64_t *cdb = a.cdur ? a.cdur + ((int64_t)blockIdx.x * a.n_cand) * SIGMA : nullptr;
      int32_t c_known = 0;  // every level < c_known has been composed
      int32_t issued = 0;   // levels [0, issued) have been armed
      bool fail = false;
      // metadata of levels l and l+1, and l+2 in flight (its load latency overlaps a level)
      uint4 m_cur = *reinterpret_cast<const uint4 *>(a.meta);
      uint4 m_nxt = *reinterpret_cast<const uint4 *>(a.meta + 4 * min(1, a.L));
      for (int32_t l = 0; l < a.L; ++l) {
        if (l == a.skip_level) break;  // failure injection: level l never arrives
        const uint4 m_fut = *reinterpret_cast<const uint4 *>(a.meta + 4 * min(l + 2, a.L));
        const uint4 m0 = m_cur, m1 = m_nxt;
        m_cur = m_nxt;
        m_nxt = m_fut;
        uint32_t ro = m0.x, i0 = m0.y, ro1 = m1.x, i1 = m1.y;
        uint32_t c0 = cdb ? m0.w : 0, c1 = cdb ? m1.w : 0;  // the level's candidate rows
        if (DBG && !(range_ok(i0, i1, a.n_rows) && range_ok(ro, ro1, a.n_words) && range_ok(c0, c1, a.n_cand))) {
          atomicCAS(a.status, 0, (int32_t)kDevBounds);  // debug bounds: copy nothing for this level
          i1 = i0 = min(i0, a.n_rows);
          ro1 = ro = min(ro, a.n_words);
          c1 = c0 = min(c0, a.n_cand);
        }
        // ring space: level l overwrites rows and words of levels below c_known only
        while (c_known < l && (l - c_known >= NB || i1 > hist[4 * (c_known % NB)] + RR ||
                               ro1 > hist[4 * (c_known % NB) + 1] + RB || c1 > hist[4 * (c_known % NB) + 2] + CRR)) {
          if (!mbar_wait(&empty[c_known % NB], (c_known / NB) & 1, a.wait_limit_cycles)) {
            fail = true;
            break;
          }
          ++c_known;
        }
        if (fail) break;
        hist[4 * (l % NB)] = i0;
        hist[4 * (l % NB) + 1] = ro;
        hist[4 * (l % NB) + 2] = c0;
        // ring rows of the level's first row and first candidate (read by the
        // consumers after the level's full barrier, which this arrival releases)
        const uint32_t dp = i0 % RR, cp = CRR ? c0 % CRR : 0;
        pos[2 * (l % NB)] = dp;
        pos[2 * (l % NB) + 1] = cp;
        uint64_t *bar = &full[l % NB];
        const uint32_t e0 = i0 * SIGMA, ne = (i1 - i0) * SIGMA, w0 = ro & rmask, nw = ro1 - ro;
        const uint32_t ce0 = c0 * SIGMA, nce = (c1 - c0) * SIGMA;
        mbar_arrive_expect_tx(bar, ne * 8 + nw * 4 + 32 + nce * 8);
        if (nce) {
          const uint32_t nce1 = min(nce, (CRR - cp) * SIGMA);
          bulk_g2s(cr + cp * SIGMA, cdb + ce0, nce1 * 8, bar);
          if (nce1 < nce) bulk_g2s(cr, cdb + ce0 + nce1, (nce - nce1) * 8, bar);
        }
        const uint32_t ne1 = min(ne, (RR - dp) * SIGMA);
        bulk_g2s(dr + dp * SIGMA, durb + e0, ne1 * 8, bar);
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
    int64_t mk[LANES];
#pragma unroll
    for (int j = 0; j < LANES; ++j) mk[j] = 0;
    for (int32_t l = 0; l < a.L; ++l) {
      const bool ok = mbar_wait(&full[l % NB], (l / NB) & 1, a.wait_limit_cycles);
      if (ok) {
        const uint32_t *mb = metas + 8 * (l % NB);
        const uint32_t ro = mb[0], i0 = mb[1], seg0 = mb[2], c0 = mb[3];
        const int32_t nseg = (int32_t)(mb[4 + 2] - seg0);
        const uint32_t dp = pos[2 * (l % NB)], cp = pos[2 * (l % NB) + 1];
        compose_segments<SIGMA, LANES, STORE_ALL, DBG>(a, ro, i0, seg0, nseg, tid / TPN, NCT / TPN, j0, vr, dr,
                                                       rr, vmask, dp, RR, rmask, mk, a.cdur ? cr : nullptr, cp,
                                                       c0, CRR);
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
  // debug bounds runs the checking variant, which stores every finish
  auto k = a.dbg ? compose_pipelined_kernel<SIGMA, true, true>
                 : a.store_all ? compose_pipelined_kernel<SIGMA, true, false> : compose_pipelined_kernel<SIGMA, false, false>;
  (void)plan;
  const size_t smem = staged_layout(SIGMA, a.vlog2, a.d_rows, a.rlog2, a.c_rows).total;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  dim3 grid((a.S + SIGMA - 1) / SIGMA);
  k<<<grid, (kPipeConsumerWarps + 1) * 32, smem, st>>>(a);
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

}  // namespace echo
