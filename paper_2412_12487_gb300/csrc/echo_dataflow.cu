// echo_dataflow.cu -- the dataflow composer: the max-plus pass of Sec. 4.2 with one
// warp per (rank, group of 32 scenarios) instead of one block per scenario block.
//
// The levelled kernels synchronize a whole scenario block at every segment level,
// so a graph with many levels and few scenarios leaves most SMs idle and pays one
// synchronization per level.  Here every warp walks its rank's ops in the internal
// (topological) order on its own, with the latest finish of each of the rank's
// timelines in shared memory, and waits only where a value comes from another
// warp:
//   - a collective or P2P op (Sec. 5.2: it starts when its last member has
//     launched it): each member warp publishes its partial launch time (the
//     latest finish among the op's inputs on its rank) and reads the others'.
//     Groups of more than 8 members gather at one member, which publishes the
//     finish;
//   - a data input produced on another rank: its producer publishes its finish.
// A published value is one 64-bit word per scenario: the time (below 2^61, which
// the host guarantees) with the launch's tag (1-7) in the top 3 bits, written by
// one relaxed store and polled by relaxed loads, so neither flags nor fences are
// needed; the host zeroes the words whenever the tags start over.  Every
// warp is resident (cooperative launch) and waits only for ops earlier in the
// topological order, so the earliest unfinished op can always proceed.  Every
// wait is bounded: a warp that gives up sets the abort flag and the timeout
// status, and every other warp leaves at its next wait.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>

#include "echo_internal.h"
#include "echo_bounds.h"

namespace echo {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr uint64_t kValueMask = (1ull << 61) - 1;

__device__ __forceinline__ uint64_t ld_relaxed_u64(const uint64_t *p) {
  uint64_t v;
  asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void st_relaxed_u64(uint64_t *p, uint64_t v) {
  asm volatile("st.relaxed.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

__device__ __forceinline__ int32_t ld_relaxed_s32(const int32_t *p) {
  int32_t v;
  asm volatile("ld.relaxed.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Waits until every lane sees the tag in the words p[i << 5] for i < n but
// `skip` (n <= 8: one round's loads are in flight together), and folds their
// values into t.  False when this wait or another warp's gave up.
__device__ bool df_gather(const uint64_t *p, uint32_t n, uint32_t skip, uint64_t tag, int64_t &t,
                          const DataflowArgs &a) {
  const long long t0 = clock64();
  unsigned ns = 32;
  uint64_t x[8];
  for (uint32_t round = 0;; ++round) {
    bool ok = true;
#pragma unroll
    for (uint32_t i = 0; i < 8; ++i) {
      x[i] = i < n && i != skip ? ld_relaxed_u64(p + ((int64_t)i << 5)) : tag;
      ok &= (x[i] & ~kValueMask) == tag;
    }
    if (__all_sync(kFull, ok)) break;
    const bool give_up = ((round & 15) == 15 && ld_relaxed_s32(a.abort_flag) != 0) ||
                         clock64() - t0 > a.wait_limit_cycles;
    if (__any_sync(kFull, give_up)) {
      if ((threadIdx.x & 31) == 0) {
        atomicExch(a.abort_flag, 1);
        atomicCAS(a.status, (int32_t)kDevOk, (int32_t)kDevTimeout);
      }
      return false;
    }
    if (round >= 32) {  // spin first: most waits end within a few L2 round trips
      __nanosleep(ns);
      if (ns < 256) ns <<= 1;
    }
  }
#pragma unroll
  for (uint32_t i = 0; i < 8; ++i) t = max(t, (int64_t)(x[i] & kValueMask));
  return true;
}

// Debug bounds: every index the batch of program entries [b, b + 8) will use (its
// nodes, candidate rows, other-input words and their payloads, partial slots,
// export ids, timelines) lies in its buffer (echo_bounds.h).  w holds the batch's
// record words as loaded by the warp (lane l: words 2(l % 4), 2(l % 4) + 1 of
// entry l / 4).  Uniform over the warp.
__device__ __noinline__ bool df_batch_ok(uint2 w, int64_t b, int64_t e1, bool cand, const DataflowArgs &a) {
  bool ok = true;
  for (int j = 0; j < kDfBatch; ++j) {
    const uint32_t v = __shfl_sync(0xffffffffu, w.x, 4 * j), ci = __shfl_sync(0xffffffffu, w.y, 4 * j);
    const uint32_t hdr = __shfl_sync(0xffffffffu, w.x, 4 * j + 1), oo = __shfl_sync(0xffffffffu, w.y, 4 * j + 1);
    const uint32_t slot = __shfl_sync(0xffffffffu, w.x, 4 * j + 2), nmme = __shfl_sync(0xffffffffu, w.y, 4 * j + 2);
    const uint32_t xid = __shfl_sync(0xffffffffu, w.x, 4 * j + 3);
    if (b + j >= e1) break;
    ok &= in_range(v, a.V) && (!cand || ci == ~0u || in_range(ci, a.n_cand));
    ok &= in_range(hdr & 15, a.n_streams) && ((hdr >> 16) >> a.n_streams) == 0;
    const uint32_t n_extra = (hdr >> 8) & 0xFF;
    ok &= range_ok(oo, (int64_t)oo + n_extra, a.n_opnd);
    for (uint32_t i = 0; ok && i < n_extra; ++i) {
      const uint32_t x = __ldg(&a.opnd[oo + i]), p = x & kDfPayload;
      ok &= (x >> 30) == kDfInLocal ? in_range(p, a.V) : (x >> 30) == kDfInRemote && in_range(p, a.n_exports);
    }
    if (hdr & kDfComm) {
      const uint32_t nm = nmme & 0xFFFF, me = nmme >> 16;
      if (slot & kDfBlockJoin)  // a block join: its members are this block's warps
        ok &= nm == (uint32_t)a.wpb && me < nm;
      else
        ok &= nm <= 1 || (me < nm && range_ok(slot, (int64_t)slot + nm, a.n_slots));
    }
    if (hdr & (kDfExport | kDfTwoHop)) ok &= in_range(xid, a.n_exports);
  }
  return ok;
}

// Join of a comm op whose nm members are the warps of this block (member me is this
// warp): each member stores its partial launch time, tagged with the join's
// sequence number, into slot seq % 2, and waits until every member's word of that
// slot carries the tag.  Members reach the block's joins in the same (internal)
// order and a member can only start join n + 2 once every member has finished
// reading join n, so two slots suffice; the tag ((seq / 2) mod 7) + 1 tells join n
// from n - 2.  Bounded like df_gather; false when this wait or another warp's
// gave up.
__device__ bool block_join(uint64_t *bjoin, uint32_t seq, uint32_t me, uint32_t nm, int64_t &t,
                           const DataflowArgs &a) {
  uint64_t *row = bjoin + (size_t)(seq & 1) * nm * 32 + (threadIdx.x & 31);
  const uint64_t tag = (uint64_t)((seq >> 1) % 7 + 1) << 61;
  asm volatile("st.volatile.shared.u64 [%0], %1;" ::"r"((uint32_t)__cvta_generic_to_shared(row + me * 32)),
               "l"(tag | (uint64_t)t)
               : "memory");
  const long long t0 = clock64();
  for (uint32_t round = 0;; ++round) {
    bool ok = true;
    int64_t m = t;
    for (uint32_t k = 0; k < nm; ++k) {
      uint64_t x;
      asm volatile("ld.volatile.shared.u64 %0, [%1];" : "=l"(x) : "r"((uint32_t)__cvta_generic_to_shared(row + k * 32))
                   : "memory");
      ok &= (x & ~kValueMask) == tag;
      m = max(m, (int64_t)(x & kValueMask));
    }
    if (__all_sync(kFull, ok)) {
      t = m;
      return true;
    }
    const bool give_up = ((round & 15) == 15 && ld_relaxed_s32(a.abort_flag) != 0) ||
                         clock64() - t0 > a.wait_limit_cycles;
    if (__any_sync(kFull, give_up)) {
      if ((threadIdx.x & 31) == 0) {
        atomicExch(a.abort_flag, 1);
        atomicCAS(a.status, (int32_t)kDevOk, (int32_t)kDevTimeout);
      }
      return false;
    }
    if (round >= 64) __nanosleep(64);
  }
}

__device__ __forceinline__ void cp_async_16(void *smem, const void *gmem) {
  const uint32_t sa = (uint32_t)__cvta_generic_to_shared(smem);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(sa), "l"(gmem) : "memory");
}

template <bool CAND>
__global__ void __launch_bounds__(kDfMaxWarpsPerBlock * 32, 2) compose_dataflow_kernel(DataflowArgs a) {
  // block: [2][wpb][32] tagged partial launch times of the block joins; then per
  // warp the duration ring [kDfDepth + 1][kDfBatch][32] and [n_streams][32] latest
  // finishes of the rank's timelines
  extern __shared__ int64_t df_smem[];
  uint64_t *bjoin = reinterpret_cast<uint64_t *>(df_smem);
  int64_t *dring = df_smem + 2 * a.wpb * 32 +
                   (int64_t)(threadIdx.x >> 5) * ((kDfDepth + 1) * kDfBatch * 32 + a.n_streams * 32);
  int64_t *df_last = dring + (kDfDepth + 1) * kDfBatch * 32;
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  for (int k = threadIdx.x; k < 2 * a.wpb * 32; k += blockDim.x) bjoin[k] = 0;  // tag 0: never written
  __syncthreads();
  const int64_t wid = (int64_t)blockIdx.x * a.wpb + wib;
  if (wid >= (int64_t)a.R * a.G) return;  // uniform over the warp
  const int32_t r = (int32_t)(wid % a.R), g = (int32_t)(wid / a.R);
  const int32_t s = g * 32 + lane;
  int64_t *last = df_last + lane;
  for (int k = 0; k < a.n_streams; ++k) last[k * 32] = 0;
  // rows of 32 scenarios: element (i, s) of an [n][S] matrix at ((g * n + i) << 5) + lane
  const int64_t *dur = a.dur + (((int64_t)g * a.V) << 5);
  const int64_t *cdu = CAND ? a.cdur + (((int64_t)g * a.n_cand) << 5) : nullptr;
  int64_t *f = a.f + (((int64_t)g * a.V) << 5) + lane;
  uint64_t *part = a.part + (((int64_t)g * a.n_slots) << 5) + lane;
  uint64_t *xval = a.xval + (((int64_t)g * a.n_exports) << 5) + lane;
  const uint64_t tag = (uint64_t)a.epoch << 61;
  const int64_t e0 = a.off[r], e1 = a.off[r + 1];
  int64_t mx = 0;
  // batches of 8 entries of 8 words: lane l holds words 2(l % 4) and 2(l % 4) + 1
  // of entry l / 4.  Records are loaded kDfDepth + 1 batches ahead of their use,
  // durations kDfDepth batches ahead into the ring (cp.async, one commit group per
  // batch): lane l copies 16 bytes, the scenarios 2(l % 16) and 2(l % 16) + 1, of
  // entries 2k + l / 16.  A lane reads elements other lanes copied, so the warp
  // synchronizes after its wait for a batch's group, and before it overwrites the
  // slot the previous batch was read from.
  auto rec = [&](int64_t b) -> uint2 {
    return b + lane / 4 < e1 ? __ldg(reinterpret_cast<const uint2 *>(a.rec) + 4 * b + lane) : make_uint2(0, 0);
  };
  auto durs = [&](int64_t b, uint2 w) {  // copies batch b's durations into its ring slot
    int64_t *slot = dring + ((b - e0) / kDfBatch % (kDfDepth + 1)) * (kDfBatch * 32) + (lane & 15) * 2;
    __syncwarp();
#pragma unroll
    for (int k = 0; k < kDfBatch / 2; ++k) {
      const int j = 2 * k + (lane >> 4);
      const uint32_t v = __shfl_sync(kFull, w.x, 4 * j), ci = CAND ? __shfl_sync(kFull, w.y, 4 * j) : ~0u;
      if (b + j < e1)
        cp_async_16(slot + j * 32, ((CAND && ci != ~0u) ? cdu + ((int64_t)ci << 5) : dur + ((int64_t)v << 5)) +
                                       (lane & 15) * 2);
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };
  static_assert(kDfDepth == 3, "the record registers below hold kDfDepth + 1 batches");
  uint2 w0 = rec(e0), w1 = rec(e0 + kDfBatch), w2 = rec(e0 + 2 * kDfBatch), w3 = rec(e0 + 3 * kDfBatch);
  // debug bounds: a batch is checked before its durations are copied; a bad index
  // stops this warp (its copies land first) and, through the abort flag, the others
  auto bad_batch = [&](int64_t bb, uint2 w) {
    if (!a.dbg || df_batch_ok(w, bb, e1, CAND, a)) return false;
    if (lane == 0) {
      atomicCAS(a.status, (int32_t)kDevOk, (int32_t)kDevBounds);
      atomicExch(a.abort_flag, 1);
    }
    asm volatile("cp.async.wait_all;" ::: "memory");
    return true;
  };
  if (bad_batch(e0, w0) || bad_batch(e0 + kDfBatch, w1) || bad_batch(e0 + 2 * kDfBatch, w2)) return;
  durs(e0, w0);
  durs(e0 + kDfBatch, w1);
  durs(e0 + 2 * kDfBatch, w2);
  int64_t cur = 0;  // finish of the previous op of the program
  for (int64_t b = e0; b < e1; b += kDfBatch) {
    const uint2 w4 = rec(b + 4 * kDfBatch);
    if (bad_batch(b + 3 * kDfBatch, w3)) return;
    durs(b + 3 * kDfBatch, w3);
    asm volatile("cp.async.wait_group 3;" ::: "memory");  // this lane's copies of the batch are complete
    __syncwarp();                                          // and so are the other lanes'
    const int64_t *d0 = dring + ((b - e0) / kDfBatch % (kDfDepth + 1)) * (kDfBatch * 32) + lane;
    const int n_here = e1 - b < kDfBatch ? (int)(e1 - b) : kDfBatch;
    // the batch's node ids, headers and durations in registers: their shuffles and
    // loads issue together, before any of the batch's stores (entries past the
    // program's end read zero words and an unused ring slot)
    uint32_t ev[kDfBatch], eh[kDfBatch];
    int64_t ed[kDfBatch];
#pragma unroll
    for (int j = 0; j < kDfBatch; ++j) {
      ev[j] = __shfl_sync(kFull, w0.x, 4 * j);
      eh[j] = __shfl_sync(kFull, w0.x, 4 * j + 1);
      ed[j] = d0[j * 32];
    }
    // a full batch of common ops (inputs: the previous op at most) runs branch-free
    bool plain = n_here == kDfBatch;
#pragma unroll
    for (int j = 0; j < kDfBatch; ++j) plain &= (eh[j] & kDfSlowMask) == 0;
    if (plain) {
#pragma unroll
      for (int j = 0; j < kDfBatch; ++j) {
        cur = ((eh[j] & kDfPrev) ? cur : 0) + ed[j];
        f[(int64_t)ev[j] << 5] = cur;
        last[(eh[j] & 15) * 32] = cur;
        mx = max(mx, cur);
      }
    } else {
#pragma unroll
    for (int j = 0; j < kDfBatch; ++j) {
      if (j >= n_here) break;
      const uint32_t v = ev[j];
      const uint32_t hdr = eh[j];
      int64_t t = (hdr & kDfPrev) ? cur : 0;
      if ((hdr & kDfSlowMask) == 0) {  // the common op: its inputs are the previous op at most
        cur = t + ed[j];
        f[(int64_t)v << 5] = cur;
        last[(hdr & 15) * 32] = cur;
        mx = max(mx, cur);
        continue;
      }
      // the latest finish among the op's inputs on this rank: the previous op, the
      // timelines' latest ops (mask), then the other inputs
      const uint32_t oo = __shfl_sync(kFull, w0.y, 4 * j + 1);
      for (uint32_t m = hdr >> 16; m; m &= m - 1) t = max(t, last[(__ffs(m) - 1) * 32]);
      const uint32_t n_extra = (hdr >> 8) & 0xFF;
      for (uint32_t i = 0; i < n_extra; ++i) {
        const uint32_t x = __ldg(&a.opnd[oo + i]), p = x & kDfPayload;
        if ((x >> 30) == kDfInLocal) {
          t = max(t, f[(int64_t)p << 5]);
        } else if (!df_gather(xval + ((int64_t)p << 5), 1, ~0u, tag, t, a)) {  // another warp's
          asm volatile("cp.async.wait_all;" ::: "memory");  // (its own copies land before it leaves)
          return;
        }
      }
      int64_t fv = t + ed[j];
      if (hdr & kDfComm) {
        const uint32_t slot = __shfl_sync(kFull, w0.x, 4 * j + 2), nmme = __shfl_sync(kFull, w0.y, 4 * j + 2);
        const uint32_t nm = nmme & 0xFFFF, me = nmme >> 16;
        if (slot & kDfBlockJoin) {  // the members are this block's warps: join in shared memory
          if (!block_join(bjoin, slot & ~kDfBlockJoin, me, nm, t, a)) {
            asm volatile("cp.async.wait_all;" ::: "memory");
            return;
          }
          fv = t + ed[j];
        } else if (nm > 1) {
          if (a.skip_slot != (int64_t)slot + me) st_relaxed_u64(part + ((int64_t)(slot + me) << 5), tag | (uint64_t)t);
          if (!(hdr & kDfTwoHop) || me == 0) {
            for (uint32_t m0 = 0; m0 < nm; m0 += 8)  // the other members, 8 at a time
              if (!df_gather(part + ((int64_t)(slot + m0) << 5), min(nm - m0, 8u), me - m0, tag, t, a)) {
                asm volatile("cp.async.wait_all;" ::: "memory");
                return;
              }
            fv = t + ed[j];
          } else {  // the first member gathers and publishes the finish
            int64_t u = 0;
            if (!df_gather(xval + ((int64_t)__shfl_sync(kFull, w0.x, 4 * j + 3) << 5), 1, ~0u, tag, u, a)) {
              asm volatile("cp.async.wait_all;" ::: "memory");
              return;
            }
            fv = u;
          }
        }
      }
      f[(int64_t)v << 5] = fv;  // (every member of a comm op stores the same finish)
      if (hdr & kDfExport)
        st_relaxed_u64(xval + ((int64_t)__shfl_sync(kFull, w0.x, 4 * j + 3) << 5), tag | (uint64_t)fv);
      last[(hdr & 15) * 32] = fv;
      cur = fv;
      mx = max(mx, fv);
    }
    }
    w0 = w1;
    w1 = w2;
    w2 = w3;
    w3 = w4;
  }
  asm volatile("cp.async.wait_all;" ::: "memory");
  if (s < a.S) atomicMax(reinterpret_cast<unsigned long long *>(a.makespan + s), (unsigned long long)mx);
}

}  // namespace

size_t dataflow_smem_bytes(int32_t n_streams, int32_t wpb) {
  return ((size_t)2 * wpb * 32 + (size_t)wpb * ((kDfDepth + 1) * kDfBatch * 32 + n_streams * 32)) * sizeof(int64_t);
}

bool dataflow_fits(int64_t n_warps, int32_t n_streams, int32_t wpb, int device) {
  int sms = 0, coop = 0, per_sm0 = 0, per_sm1 = 0;
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device);
  cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, device);
  const size_t smem = dataflow_smem_bytes(n_streams, wpb);
  if (cudaFuncSetAttribute(compose_dataflow_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
          cudaSuccess ||
      cudaFuncSetAttribute(compose_dataflow_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
          cudaSuccess ||
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm0, compose_dataflow_kernel<false>, 32 * wpb, smem) !=
          cudaSuccess ||
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm1, compose_dataflow_kernel<true>, 32 * wpb, smem) !=
          cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  const int64_t blocks = (n_warps + wpb - 1) / wpb;
  return coop && blocks <= (int64_t)std::min(per_sm0, per_sm1) * sms;
}

cudaError_t launch_compose_dataflow(const DataflowArgs &a, cudaStream_t st) {
  const int64_t warps = (int64_t)a.R * a.G;
  if (warps == 0) return cudaSuccess;
  if (a.wpb < 1 || a.wpb > kDfMaxWarpsPerBlock || a.R % a.wpb) return cudaErrorInvalidValue;
  const dim3 grid((unsigned)((warps + a.wpb - 1) / a.wpb)), block(32 * a.wpb);
  DataflowArgs args = a;
  void *params[] = {&args};
  const size_t smem = dataflow_smem_bytes(a.n_streams, a.wpb);
  if (a.cdur)
    return cudaLaunchCooperativeKernel((const void *)compose_dataflow_kernel<true>, grid, block, params, smem, st);
  return cudaLaunchCooperativeKernel((const void *)compose_dataflow_kernel<false>, grid, block, params, smem, st);
}

}  // namespace echo
