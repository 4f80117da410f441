// echo_internal.h -- declarations shared by the host library and the kernels.
#pragma once

#include <cuda_runtime.h>

#include <cstdint>

namespace echo {

constexpr int kMaxStreams = 16;
constexpr int kMaxChunk = 16;
constexpr uint8_t kNotSlowable = 0xFF;
constexpr int kComposeThreads = 512;

// device status word: first error wins
enum DeviceStatus : int32_t { kDevOk = 0, kDevNegativeDuration = 1, kDevCcOverflow = 2 };

struct ChunkTable {
  int32_t n;
  int64_t max_bytes[kMaxChunk];
  int64_t chunk[kMaxChunk];
};

// one deduplicated collective signature (type, algorithm, bytes, group shape)
struct CcSig {
  int64_t nbytes;
  int32_t type, algo, N, M, K, pad;
  double lg;  // log2(M), computed on the host
};

struct ScenParams {  // device arrays [S]
  const double *alpha, *bwa, *lata, *bwe, *late, *delta;
};

struct ComposeArgs {
  int64_t V;
  int32_t S, L;
  int32_t n_queues;
  const int64_t *lvl_off;                     // [L+1]
  const int64_t *nq_off; const int32_t *nq;   // timelines of each node
  const int64_t *dp_off; const int32_t *dp;   // data predecessors (internal ids)
  const uint8_t *kcl;                         // kernel class or kNotSlowable
  const int64_t *dur;                         // [V][S]
  const uint8_t *ov;                          // [V][S] slow this op? (nullptr: raw durations)
  const double *sf;                           // [C][S]
  int64_t *f;                                 // [V][S] finish times (out)
  int64_t *makespan;                          // [S] (out)
  int64_t *gfrontier;                         // [grid][n_queues][sigma] when not in smem
};

struct OverlapArgs {
  int32_t S, n_ranks, n_streams;
  const int64_t *q_off; const int32_t *q_ops;  // timelines in internal ids
  const uint8_t *is_comm;                      // [V]
  const uint8_t *kcl;                          // [V]
  const int64_t *dur;                          // [V][S]
  const uint8_t *ov_prev;                      // durations of the pass that produced f
  const double *sf;
  const int64_t *f;                            // [V][S]
  uint8_t *ov;                                 // [V][S] (out)
};

// kernels.cu
cudaError_t launch_cc_estimate(const CcSig *sig, int32_t G, ScenParams p, int32_t S,
                               const ChunkTable &tbl, const int32_t *sig_count, double *cc_ns,
                               int64_t *cc_dur, double *comm_sum, int32_t *status, cudaStream_t st);
cudaError_t launch_cc_scatter(const int32_t *comm_node, const int32_t *comm_sig, int64_t n_comm,
                              const int64_t *cc_dur, int32_t S, int64_t *dur, cudaStream_t st);
cudaError_t launch_cc_query(int64_t n, const uint8_t *type, const uint8_t *algo, const int64_t *nbytes,
                            const int32_t *N, const int32_t *M, const double *lg, ScenParams p,
                            const ChunkTable &tbl, double *out, cudaStream_t st);
cudaError_t launch_permute_rows(const int64_t *raw, const int32_t *int2ext, const uint8_t *local,
                                int64_t V, int32_t S, int64_t *dur, double *sums, int32_t *status,
                                cudaStream_t st);
cudaError_t launch_compose(const ComposeArgs &a, int sigma, cudaStream_t st);
cudaError_t launch_overlap(const OverlapArgs &a, cudaStream_t st);
cudaError_t launch_readback(const int32_t *ext2int, int64_t op0, int64_t op1, int32_t S,
                            const int64_t *f, const int64_t *dur, const uint8_t *ov,
                            const uint8_t *kcl, const double *sf, int64_t *start, int64_t *finish,
                            cudaStream_t st);
cudaError_t launch_read_cc(const int32_t *ext2int, int64_t op0, int64_t op1, int32_t S,
                           const int32_t *node_sig, const double *cc_ns, double *out, cudaStream_t st);
cudaError_t launch_read_ov(const int32_t *ext2int, int64_t op0, int64_t op1, int32_t S,
                           const uint8_t *ov, const uint8_t *kcl, uint8_t *out, cudaStream_t st);
size_t compose_smem_bytes(int32_t n_queues, int sigma, bool *frontier_in_smem);

}  // namespace echo
