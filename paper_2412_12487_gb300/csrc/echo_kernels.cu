// echo_kernels.cu -- sm_103a kernels of the CC estimator, the validator and the
// readbacks.  All floating point that decides an integer is written with explicit
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

__device__ __forceinline__ void set_status(int32_t *status, int32_t code) {
  atomicCAS(status, 0, code);
}

// ---------------------------------------------------------------------------------
// B1: CC estimate over [signature x scenario]
// ---------------------------------------------------------------------------------
__global__ void cc_estimate_kernel(const CcSig *__restrict__ sig, int32_t G, ScenParams p, int32_t S,
                                   ChunkTable tbl, const int32_t *__restrict__ sig_count,
                                   double *__restrict__ cc_ns, int64_t *__restrict__ cc_dur,
                                   double *__restrict__ comm_sum, int32_t *status, int model, int ar_policy) {
  int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (int64_t)G * S) return;
  int32_t g = (int32_t)(idx / S), s = (int32_t)(idx % S);
  CcSig q = sig[g];
  double T;
  if (model == 1) {
    // alpha-beta comparison model (Sec. 2.3): size over bandwidth plus latency on
    // the bottleneck link
    T = (q.N <= 1 || q.nbytes <= 0)
            ? 0.0
            : __dadd_rn(q.M > 1 ? p.late[s] : p.lata[s], __ddiv_rn((double)q.nbytes, q.M > 1 ? p.bwe[s] : p.bwa[s]));
  } else {
    const int algo = q.type == kAR && ar_policy > 0 ? ar_policy - 1 : q.algo;  // a policy for every all-reduce
    T = cc_ns_of(q.type, algo, q.nbytes, q.N, q.M, q.K, q.lg, p.alpha[s], p.bwa[s], p.lata[s], p.bwe[s],
                 p.late[s], p.delta[s], tbl);
  }
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
template <typename T>
__global__ void permute_rows_kernel(const T *__restrict__ raw, const int32_t *__restrict__ int2ext,
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
      d = (int64_t)raw[e * S + s];
      neg |= d < 0;
      acc += (double)d;
    }
    dur[lay.at(i, s)] = d;
  }
  if (neg) set_status(status, kDevNegativeDuration);
  atomicAdd(&sums[s], acc);
}

// ---------------------------------------------------------------------------------
// B3: validator overlap test over the overlap candidates: the compute ops that
// some comm op of their rank is neither an ancestor nor a descendant of (the
// others can never overlap; their durations are copied unchanged).  One thread
// per (chunk of a rank's candidates, which run in issue order, scenario); a warp
// covers 32 scenarios of one chunk and shares its op list.
// Every timeline of a rank runs its ops one after the other, so on each of the
// rank's comm timelines the intervals are sorted and the compute ops' starts only
// grow.  The thread keeps, per comm timeline, a cursor at the first comm op of
// positive length that finishes after the current candidate starts, with that
// op's interval in registers: the compute op overlaps this timeline iff that
// interval starts before the compute op finishes (any later comm op starts after
// the cursor op ends).  A binary search places the cursors at the chunk's first
// op; from there they only move forward, and only then touch memory.  A compute
// op of positive length that overlaps gets rint(d * slowdown) for the next
// composition (cd_next, compact), others keep d; the decisions themselves are stored only
// when `ov` is given.  The finish times and durations of 8 consecutive ops are
// loaded together before they are tested.
// ---------------------------------------------------------------------------------
// ---------------------------------------------------------------------------------
// readback: internal order and blocked layout -> caller order, [op][scenario]
// ---------------------------------------------------------------------------------
// start = finish - the duration the op had in the last composition: d, or for an
// overlap candidate its row of the compact cd when given
__global__ void readback_kernel(const int32_t *__restrict__ ext2int, int64_t op0, int64_t op1, int32_t s0,
                                int32_t s1, MatLayout lay, const int64_t *__restrict__ f,
                                const int64_t *__restrict__ d, const int32_t *__restrict__ cidx, MatLayout lay_c,
                                const int64_t *__restrict__ cd, int64_t *__restrict__ start,
                                int64_t *__restrict__ finish) {
  const int32_t Sr = s1 - s0;
  int64_t total = (op1 - op0) * Sr;
  for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
       idx += (int64_t)gridDim.x * blockDim.x) {
    int64_t o = idx / Sr;
    int32_t s = s0 + (int32_t)(idx - o * Sr);
    const int32_t i = ext2int[op0 + o];
    int64_t at = lay.at(i, s);
    int64_t fv = f[at];
    if (start) {
      const int32_t ci = cd ? cidx[i] : -1;
      start[idx] = fv - (ci >= 0 ? cd[lay_c.at(ci, s)] : d[at]);
    }
    if (finish) finish[idx] = fv;
  }
}

// Full validator durations for the kernels without a candidate ring: the
// candidates' rows of the compact cd into dst (which holds the original durations).
__global__ void scatter_candidates_kernel(const int32_t *__restrict__ cand_node, int64_t n_cand, int32_t S,
                                          MatLayout lay, MatLayout lay_c, const int64_t *__restrict__ cd,
                                          int64_t *__restrict__ dst) {
  const int64_t total = n_cand * S;
  for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
       idx += (int64_t)gridDim.x * blockDim.x) {
    const int64_t k = idx / S;
    const int32_t s = (int32_t)(idx - k * S);
    dst[lay.at(cand_node[k], s)] = cd[lay_c.at(k, s)];
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
                               MatLayout lay, const uint8_t *__restrict__ ov, const uint8_t *__restrict__ cand,
                               uint8_t *__restrict__ out) {
  int64_t total = (op1 - op0) * S;
  for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
       idx += (int64_t)gridDim.x * blockDim.x) {
    int64_t o = idx / S;
    int32_t s = (int32_t)(idx - o * S);
    int64_t i = ext2int[op0 + o];
    out[idx] = (ov && cand[i]) ? ov[lay.at(i, s)] : 0;  // only the candidates are tested
  }
}

int grid_for(int64_t n, int threads) {
  int64_t b = (n + threads - 1) / threads;
  if (b < 1) b = 1;
  if (b > 152 * 32) b = 152 * 32;
  return (int)b;
}

}  // namespace

cudaError_t launch_cc_estimate(const CcSig *sig, int32_t G, ScenParams p, int32_t S, const ChunkTable &tbl,
                               const int32_t *sig_count, double *cc_ns, int64_t *cc_dur, double *comm_sum,
                               int32_t *status, int model, int ar_policy, cudaStream_t st) {
  int64_t n = (int64_t)G * S;
  if (n == 0) return cudaSuccess;
  int threads = 256;
  int64_t blocks = (n + threads - 1) / threads;
  cc_estimate_kernel<<<(unsigned)blocks, threads, 0, st>>>(sig, G, p, S, tbl, sig_count, cc_ns, cc_dur,
                                                          comm_sum, status, model, ar_policy);
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

cudaError_t launch_permute_rows(const void *raw, int bits, const int32_t *int2ext, const uint8_t *local, int64_t V,
                                int32_t S, MatLayout lay, int64_t *dur, double *sums, int32_t *status,
                                cudaStream_t st) {
  if (V == 0 || S == 0) return cudaSuccess;
  int tx = S >= 128 ? 128 : ((S + 31) / 32) * 32;
  dim3 block(tx);
  int64_t gy = V < 8192 ? V : 8192;
  dim3 grid((S + tx - 1) / tx, (unsigned)gy);
  if (bits == 32)
    permute_rows_kernel<int32_t><<<grid, block, 0, st>>>(static_cast<const int32_t *>(raw), int2ext, local, V, S,
                                                         lay, dur, sums, status);
  else
    permute_rows_kernel<int64_t><<<grid, block, 0, st>>>(static_cast<const int64_t *>(raw), int2ext, local, V, S,
                                                         lay, dur, sums, status);
  return cudaGetLastError();
}

template <typename T>
__global__ void replica_check_kernel(const T *__restrict__ raw, const int32_t *__restrict__ pairs, int64_t n_pairs,
                                     int32_t S, int32_t *flag) {
  const int64_t total = n_pairs * S;
  bool diff = false;
  for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
       idx += (int64_t)gridDim.x * blockDim.x) {
    const int64_t p = idx / S, s = idx - p * S;
    diff |= raw[(int64_t)pairs[2 * p] * S + s] != raw[(int64_t)pairs[2 * p + 1] * S + s];
  }
  if (__any_sync(0xffffffffu, diff) && (threadIdx.x & 31) == 0) *flag = 1;
}

cudaError_t launch_replica_check(const void *raw, int bits, const int32_t *pairs, int64_t n_pairs, int32_t S,
                                 int32_t *flag, cudaStream_t st) {
  if (n_pairs == 0 || S == 0) return cudaSuccess;
  const int64_t total = n_pairs * S;
  const int threads = 256;
  const int64_t blocks = std::min<int64_t>((total + threads - 1) / threads, 152 * 16);
  if (bits == 32)
    replica_check_kernel<int32_t><<<(unsigned)blocks, threads, 0, st>>>(static_cast<const int32_t *>(raw), pairs,
                                                                         n_pairs, S, flag);
  else
    replica_check_kernel<int64_t><<<(unsigned)blocks, threads, 0, st>>>(static_cast<const int64_t *>(raw), pairs,
                                                                         n_pairs, S, flag);
  return cudaGetLastError();
}

cudaError_t launch_overlap(const OverlapArgs &a, cudaStream_t st) {
  const int64_t warps = (int64_t)a.n_ranks * ((a.S + 31) / 32) * a.parts;
  if (a.S == 0 || warps == 0) return cudaSuccess;
  if (a.n_cq < 0 || a.n_cq > kMaxStreams || a.parts < 1) return cudaErrorInvalidValue;
  const dim3 grid((unsigned)((warps + kOvWarps - 1) / kOvWarps));
  const int tx = kOvWarps * 32;
  // the variants are compiled in four translation units (echo_overlap.cu)
  const bool prop = a.model == 1 && a.cd_next;
  if (a.lq_off)
    return prop ? launch_overlap_l1_p1(a, grid, tx, st) : launch_overlap_l1_p0(a, grid, tx, st);
  return prop ? launch_overlap_l0_p1(a, grid, tx, st) : launch_overlap_l0_p0(a, grid, tx, st);
}

cudaError_t launch_readback(const int32_t *ext2int, int64_t op0, int64_t op1, int32_t s0, int32_t s1, MatLayout lay,
                            const int64_t *f, const int64_t *d, const int32_t *cidx, MatLayout lay_c,
                            const int64_t *cd, int64_t *start, int64_t *finish, cudaStream_t st) {
  int64_t n = (op1 - op0) * (s1 - s0);
  if (n <= 0) return cudaSuccess;
  readback_kernel<<<grid_for(n, 256), 256, 0, st>>>(ext2int, op0, op1, s0, s1, lay, f, d, cidx, lay_c, cd, start,
                                                    finish);
  return cudaGetLastError();
}

cudaError_t launch_scatter_candidates(const int32_t *cand_node, int64_t n_cand, int32_t S, MatLayout lay,
                                      MatLayout lay_c, const int64_t *cd, int64_t *dst, cudaStream_t st) {
  if (n_cand == 0 || S == 0) return cudaSuccess;
  scatter_candidates_kernel<<<grid_for(n_cand * S, 256), 256, 0, st>>>(cand_node, n_cand, S, lay, lay_c, cd, dst);
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
                           const uint8_t *ov, const uint8_t *cand, uint8_t *out, cudaStream_t st) {
  int64_t n = (op1 - op0) * S;
  if (n <= 0) return cudaSuccess;
  read_ov_kernel<<<grid_for(n, 256), 256, 0, st>>>(ext2int, op0, op1, S, lay, ov, cand, out);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------------
// fp64 rates of this device (measurement support): each thread keeps 8 independent
// chains of one operation (add, multiply or divide with round-to-nearest, as the
// CC estimator uses them), so the pipe, not the dependence latency, sets the rate.
// The result feeds a kernel in the sink so nothing is optimized away.
// ---------------------------------------------------------------------------------
constexpr int kFp64Chains = 8;
template <int OP>
__global__ void fp64_rate_kernel(int iters, double y, double *sink) {
  double x[kFp64Chains];
#pragma unroll
  for (int k = 0; k < kFp64Chains; ++k) x[k] = 1.0 + (threadIdx.x + k) * 1e-9;
  for (int i = 0; i < iters; ++i) {
#pragma unroll
    for (int k = 0; k < kFp64Chains; ++k)
      x[k] = OP == 0 ? __dadd_rn(x[k], y) : OP == 1 ? __dmul_rn(x[k], y) : __ddiv_rn(x[k], y);
  }
  double t = 0.0;
#pragma unroll
  for (int k = 0; k < kFp64Chains; ++k) t = __dadd_rn(t, x[k]);
  if (t == 12345.0) sink[0] = t;  // never true for these inputs
}

}  // namespace echo

extern "C" int echo_measure_fp64(int device, double *rates) {
  using namespace echo;
  if (!rates) return ECHO_E_INVALID_ARG;
  int prev = 0;
  if (cudaGetDevice(&prev) != cudaSuccess || cudaSetDevice(device) != cudaSuccess) return ECHO_E_CUDA;
  struct Restore {
    int dev;
    ~Restore() { cudaSetDevice(dev); }
  } restore{prev};
  int sms = 0;
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device);
  double *sink = nullptr;
  if (cudaMalloc(&sink, sizeof(double)) != cudaSuccess) return ECHO_E_OOM;
  cudaEvent_t a, b;
  cudaEventCreate(&a);
  cudaEventCreate(&b);
  const int threads = 256, blocks = sms * 8;
  int rc = ECHO_OK;
  for (int op = 0; op < 3 && rc == ECHO_OK; ++op) {
    const int iters = op == 2 ? 256 : 4096;
    const double y = op == 1 ? 1.0000000001 : op == 2 ? 0.9999999999 : 1e-12;
    auto launch = [&]() {
      if (op == 0) fp64_rate_kernel<0><<<blocks, threads>>>(iters, y, sink);
      else if (op == 1) fp64_rate_kernel<1><<<blocks, threads>>>(iters, y, sink);
      else fp64_rate_kernel<2><<<blocks, threads>>>(iters, y, sink);
    };
    launch();  // warm-up
    float best = 0.f;
    for (int rep = 0; rep < 5; ++rep) {
      cudaEventRecord(a);
      launch();
      cudaEventRecord(b);
      if (cudaEventSynchronize(b) != cudaSuccess) {
        rc = ECHO_E_CUDA;
        break;
      }
      float ms = 0.f;
      cudaEventElapsedTime(&ms, a, b);
      if (rep == 0 || ms < best) best = ms;
    }
    rates[op] = (double)blocks * threads * iters * kFp64Chains / (best * 1e-3);
  }
  if (cudaGetLastError() != cudaSuccess && rc == ECHO_OK) rc = ECHO_E_CUDA;
  cudaEventDestroy(a);
  cudaEventDestroy(b);
  cudaFree(sink);
  return rc;
}

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
// Layout of the array: bytes [0, 4) hold a status word (one bit per kind of bad
// query), cleared at the start of every call; from byte 256 on, log2(m) for m = 0..kNoallocMaxNodes, computed on
// the host with the same libm log2 the allocating path uses, so both paths give
// identical estimates.  Node counts above kNoallocMaxNodes are rejected.
// ---------------------------------------------------------------------------------
namespace echo {
namespace {
constexpr int32_t kNoallocMaxNodes = 65536;
constexpr size_t kNoallocLgOffset = 256;
constexpr size_t kNoallocScratchBytes = kNoallocLgOffset + sizeof(double) * (kNoallocMaxNodes + 1);
constexpr int kNoallocMaxDevices = 64;
// status bits: a batch may hold both kinds of bad query, so each sets its own bit
// and the host ranks them (a malformed query before an unsupported size)
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
      atomicOr(status, kNoallocBadQuery);
      continue;
    }
    if (m > kNoallocMaxNodes) {
      out[i] = nan;
      atomicOr(status, kNoallocTooManyNodes);
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
  if (status & kNoallocBadQuery) return ECHO_E_INVALID_ARG;
  if (status & kNoallocTooManyNodes) return ECHO_E_UNSUPPORTED;
  return ECHO_OK;
}
