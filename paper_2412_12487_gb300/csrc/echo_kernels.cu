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

constexpr int kAR = 0, kAG = 1, kRS = 2, kSR = 3;
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
                                  int64_t n_comm, const int64_t *__restrict__ cc_dur, int32_t S,
                                  int64_t *__restrict__ dur) {
  int64_t total = n_comm * S;
  for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
       idx += (int64_t)gridDim.x * blockDim.x) {
    int64_t c = idx / S;
    int32_t s = (int32_t)(idx - c * S);
    dur[(int64_t)comm_node[c] * S + s] = cc_dur[(int64_t)comm_sig[c] * S + s];
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
// load: caller-order rows -> level order, with validation and per-scenario sums
// ---------------------------------------------------------------------------------
__global__ void permute_rows_kernel(const int64_t *__restrict__ raw, const int32_t *__restrict__ int2ext,
                                    const uint8_t *__restrict__ local, int64_t V, int32_t S,
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
    dur[i * S + s] = d;
  }
  if (neg) set_status(status, kDevNegativeDuration);
  atomicAdd(&sums[s], acc);
}

// ---------------------------------------------------------------------------------
// B2: compose pass.  One thread block owns SIGMA scenarios and walks every level
// of the level-ordered graph; scenarios never interact, so only block barriers
// are needed.  f(v) = max(0, finish of the op issued before v on each of its
// timelines, finish of each data predecessor) + d(v).  The first term comes from
// a per-(timeline, scenario) frontier that holds the finish of the last op placed
// on that timeline (Sec. 4.2); the per-scenario makespan is fused in.
// ---------------------------------------------------------------------------------
template <int SIGMA, bool SMEM_FRONTIER>
__global__ void __launch_bounds__(kComposeThreads)
compose_kernel(ComposeArgs a) {
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
    const int64_t i0 = a.lvl_off[l], i1 = a.lvl_off[l + 1];
    if (active) {
      for (int64_t i = i0 + sub; i < i1; i += stride) {
        int64_t m = 0;
        const int64_t q0 = a.nq_off[i], q1 = a.nq_off[i + 1];
        for (int64_t k = q0; k < q1; ++k) m = max(m, fr[(int64_t)a.nq[k] * SIGMA + j]);
        for (int64_t k = a.dp_off[i]; k < a.dp_off[i + 1]; ++k)
          m = max(m, f[(int64_t)a.dp[k] * S + s]);
        int64_t d = dur[i * S + s];
        if (a.ov) {
          const uint8_t c = a.kcl[i];
          if (c != kNotSlowable && a.ov[i * S + s]) d = slowed(d, a.sf[(int64_t)c * S + s]);
        }
        const int64_t fv = m + d;
        f[i * S + s] = fv;
        for (int64_t k = q0; k < q1; ++k) fr[(int64_t)a.nq[k] * SIGMA + j] = fv;
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

// ---------------------------------------------------------------------------------
// B3: validator overlap test.  One thread per (rank, scenario) walks the rank's
// compute timeline in time order with one monotone cursor per comm/memcpy
// timeline: ops on a timeline run one after the other, so their intervals are
// sorted and the first comm op finishing after a kernel's start is the only
// place a search has to resume from.
// ---------------------------------------------------------------------------------
__global__ void overlap_kernel(OverlapArgs a) {
  const int32_t S = a.S;
  const int32_t s = blockIdx.x * blockDim.x + threadIdx.x;
  const int32_t r = blockIdx.y;
  if (s >= S) return;
  const int ns = a.n_streams;
  const int64_t qbase = (int64_t)r * ns;
  int64_t cur[kMaxStreams];
  for (int k = 1; k < ns; ++k) cur[k] = a.q_off[qbase + k];
  const int64_t c0 = a.q_off[qbase], c1 = a.q_off[qbase + 1];
  for (int64_t i = c0; i < c1; ++i) {
    const int64_t v = a.q_ops[i];
    int64_t dv = a.dur[v * S + s];
    if (a.ov_prev && a.ov_prev[v * S + s]) dv = slowed(dv, a.sf[(int64_t)a.kcl[v] * S + s]);
    const int64_t fv = a.f[v * S + s];
    const int64_t sv = fv - dv;
    uint8_t hit = 0;
    if (sv < fv) {
      for (int k = 1; k < ns && !hit; ++k) {
        const int64_t e = a.q_off[qbase + k + 1];
        int64_t c = cur[k];
        while (c < e) {
          const int64_t w = a.q_ops[c];
          if (a.is_comm[w] && a.f[w * S + s] > sv) break;
          ++c;
        }
        cur[k] = c;
        for (int64_t jj = c; jj < e; ++jj) {
          const int64_t w = a.q_ops[jj];
          const int64_t fw = a.f[w * S + s];
          const int64_t sw = fw - a.dur[w * S + s];
          if (sw >= fv) break;
          if (a.is_comm[w] && sw < fw) {
            hit = 1;
            break;
          }
        }
      }
    }
    a.ov[v * S + s] = hit;
  }
}

// ---------------------------------------------------------------------------------
// readback: internal order -> caller order
// ---------------------------------------------------------------------------------
__global__ void readback_kernel(const int32_t *__restrict__ ext2int, int64_t op0, int64_t op1, int32_t S,
                                const int64_t *__restrict__ f, const int64_t *__restrict__ dur,
                                const uint8_t *__restrict__ ov, const uint8_t *__restrict__ kcl,
                                const double *__restrict__ sf, int64_t *__restrict__ start,
                                int64_t *__restrict__ finish) {
  int64_t total = (op1 - op0) * S;
  for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
       idx += (int64_t)gridDim.x * blockDim.x) {
    int64_t o = idx / S;
    int32_t s = (int32_t)(idx - o * S);
    int64_t i = ext2int[op0 + o];
    int64_t fv = f[i * S + s];
    int64_t d = dur[i * S + s];
    if (ov && kcl[i] != kNotSlowable && ov[i * S + s]) d = slowed(d, sf[(int64_t)kcl[i] * S + s]);
    if (start) start[idx] = fv - d;
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
                               const uint8_t *__restrict__ ov, const uint8_t *__restrict__ kcl,
                               uint8_t *__restrict__ out) {
  int64_t total = (op1 - op0) * S;
  for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
       idx += (int64_t)gridDim.x * blockDim.x) {
    int64_t o = idx / S;
    int32_t s = (int32_t)(idx - o * S);
    int64_t i = ext2int[op0 + o];
    out[idx] = (ov && kcl[i] != kNotSlowable) ? ov[i * S + s] : 0;  // only compute ops are tested
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
    auto k = compose_kernel<SIGMA, true>;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    k<<<grid, kComposeThreads, smem, st>>>(a);
  } else {
    auto k = compose_kernel<SIGMA, false>;
    k<<<grid, kComposeThreads, smem, st>>>(a);
  }
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
                              const int64_t *cc_dur, int32_t S, int64_t *dur, cudaStream_t st) {
  if (n_comm == 0) return cudaSuccess;
  cc_scatter_kernel<<<grid_for(n_comm * S, 256), 256, 0, st>>>(comm_node, comm_sig, n_comm, cc_dur, S, dur);
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
                                int32_t S, int64_t *dur, double *sums, int32_t *status, cudaStream_t st) {
  if (V == 0 || S == 0) return cudaSuccess;
  int tx = S >= 128 ? 128 : ((S + 31) / 32) * 32;
  dim3 block(tx);
  int64_t gy = V < 8192 ? V : 8192;
  dim3 grid((S + tx - 1) / tx, (unsigned)gy);
  permute_rows_kernel<<<grid, block, 0, st>>>(raw, int2ext, local, V, S, dur, sums, status);
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

cudaError_t launch_overlap(const OverlapArgs &a, cudaStream_t st) {
  if (a.S == 0 || a.n_ranks == 0) return cudaSuccess;
  int tx = a.S >= 128 ? 128 : ((a.S + 31) / 32) * 32;
  dim3 grid((a.S + tx - 1) / tx, a.n_ranks);
  overlap_kernel<<<grid, tx, 0, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_readback(const int32_t *ext2int, int64_t op0, int64_t op1, int32_t S, const int64_t *f,
                            const int64_t *dur, const uint8_t *ov, const uint8_t *kcl, const double *sf,
                            int64_t *start, int64_t *finish, cudaStream_t st) {
  int64_t n = (op1 - op0) * S;
  if (n <= 0) return cudaSuccess;
  readback_kernel<<<grid_for(n, 256), 256, 0, st>>>(ext2int, op0, op1, S, f, dur, ov, kcl, sf, start, finish);
  return cudaGetLastError();
}

cudaError_t launch_read_cc(const int32_t *ext2int, int64_t op0, int64_t op1, int32_t S, const int32_t *node_sig,
                           const double *cc_ns, double *out, cudaStream_t st) {
  int64_t n = (op1 - op0) * S;
  if (n <= 0) return cudaSuccess;
  read_cc_kernel<<<grid_for(n, 256), 256, 0, st>>>(ext2int, op0, op1, S, node_sig, cc_ns, out);
  return cudaGetLastError();
}

cudaError_t launch_read_ov(const int32_t *ext2int, int64_t op0, int64_t op1, int32_t S, const uint8_t *ov,
                           const uint8_t *kcl, uint8_t *out, cudaStream_t st) {
  int64_t n = (op1 - op0) * S;
  if (n <= 0) return cudaSuccess;
  read_ov_kernel<<<grid_for(n, 256), 256, 0, st>>>(ext2int, op0, op1, S, ov, kcl, out);
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
