// echo_internal.h -- declarations shared by the host library and the kernels.
#pragma once

#include <cuda_runtime.h>

#include <cstdint>

#include "echo_bounds.h"

namespace echo {

constexpr int kMaxStreams = 16;
constexpr int kMaxChunk = 16;
constexpr uint8_t kNotSlowable = 0xFF;
constexpr int kComposeThreads = 512;       // direct compose kernel
constexpr int kMetaChunk = 128;            // segment levels of metadata staged at a time
constexpr int kMetaCap = 136;              // metadata entries per staging buffer (>= kMetaChunk + 1)
constexpr uint32_t kFarRef = 0x80000000u;  // predecessor reference read from global memory
constexpr int kOvBatch = 8;                // candidates per batch of the overlap test
constexpr int kOvDepth = 3;                // batches of candidate rows in flight per warp
constexpr int kOvWarps = 4;                // warps per block of the overlap test
constexpr int kMaxSegment = 64;            // longest serial chain composed as one segment
constexpr int kPipeStages = 16;            // stages (mbarrier pairs) of the pipelined compose
constexpr int kPipeConsumerWarps = 16;     // composing warps of the pipelined compose

// device status word: first error wins
enum DeviceStatus : int32_t {
  kDevOk = 0, kDevNegativeDuration = 1, kDevCcOverflow = 2, kDevTimeout = 3,
  kDevBounds = 4  // a debug-bounds index check failed (echo_bounds.h)
};

// Device layout of every [op][scenario] matrix (durations, finish times, validator
// outputs): scenario blocks of 2^slog2 scenarios, block b holding a contiguous
// [V][2^slog2] array, so one thread block's rows of consecutive ops form one
// contiguous range.  Lanes of a partial last block are padding (kept at zero in
// the duration matrices).
struct MatLayout {
  int64_t V;
  int32_t slog2;
  __host__ __device__ int64_t at(int64_t i, int32_t s) const {
    return (((int64_t)(s >> slog2) * V + i) << slog2) + (s & ((1 << slog2) - 1));
  }
  __host__ __device__ int64_t block(int32_t b) const { return ((int64_t)b * V) << slog2; }
};

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

// Direct compose: graph structure and durations read from global memory.  The
// graph is composed segment level by segment level; a segment is a serial chain
// whose nodes are numbered consecutively.
struct ComposeArgs {
  int64_t V;
  MatLayout lay;
  int32_t S, L;                               // L: segment levels
  int32_t n_queues;
  const int64_t *seg_lvl_off;                 // [L+1] segments of each level
  const int64_t *seg_node_off;                // [n_seg+1] nodes of each segment
  const int64_t *nq_off; const int32_t *nq;   // timelines of each node
  const int64_t *dp_off; const int32_t *dp;   // data predecessors (internal ids)
  const int64_t *dur;                         // durations of this pass (MatLayout)
  int64_t *f;                                 // finish times (MatLayout, out)
  int64_t *makespan;                          // [S] (out)
  int64_t *gfrontier;                         // [grid][n_queues][sigma] when not in smem
  int32_t dbg;                                // debug bounds: check every index (echo_bounds.h)
  int32_t *status;
};

// Staged and pipelined compose: per-segment-level records and duration rows are
// copied into shared-memory rings ahead of use.  Record block of a level (32-bit
// words): for each segment, 4 header words {offset of its entries in the block,
// nin | nfar << 16, first node - level's first node, length}; entries = the
// head's nin inputs held in the value ring (byte offsets of their slots), then its
// nfar inputs too old for the ring (node ids, read from global memory).  Every
// input is the tail of an earlier segment.  A segment whose chain holds overlap
// candidates has bit 16 of its length word set and 3 more entries: a 64-bit mask
// of those chain positions and the level-order index of the first.  A segment with
// chain positions before its tail whose finish a later step reads (validator
// inputs) has bit 17 set and 2 more entries: the 64-bit mask of those positions.
// Blocks are padded to 4 words.  Metadata of a level: record word offset, first node, first
// segment, first level-order candidate.
struct StagedArgs {
  int32_t S, L;                  // L: segment levels
  uint32_t n_rows, n_words;      // nodes; words of all record blocks
  int32_t vlog2, dlog2, rlog2;   // log2 sizes: value ring (segments), duration ring (rows), record ring (words)
  uint32_t d_rows, c_rows;       // ring sizes in rows (any size): duration and candidate rings
  const uint32_t *meta;          // [4*(L+1)]: record word offset, first node, first segment, first candidate
  const uint32_t *recs;          // record blocks
  const int64_t *dur;            // durations (MatLayout)
  int64_t *f;                    // finish times (MatLayout, out)
  int64_t *makespan;             // [S] (out)
  // pipelined kernel only
  const int64_t *cdur;           // validator durations of the candidates ([n_cand] rows per block), or null
  uint32_t n_cand;               // overlap candidates
  int32_t clog2;                 // log2 rows of the candidate ring (staged kernel)
  int32_t *status;               // device status word (kDevTimeout when a bounded wait gives up)
  long long wait_limit_cycles;   // bound of every mbarrier wait, in SM clock cycles
  int32_t skip_level;            // failure injection for tests: this level is never filled (-1: none)
  int32_t store_all;             // final composition: store every finish; else only those read again
  int32_t dbg;                   // debug bounds: check every index (echo_bounds.h)
};

// Plan of the staged kernels for one (graph, sigma); see plan_staged().
struct StagedPlan {
  bool ok = false;
  bool pipelined = false;  // bulk-copy producer warp (even sigma)
  int threads = 512;       // threads per block of the staged kernel
  int vring_log2 = 0, dring_log2 = 0, rring_log2 = 0;  // sizes (segments, rows, words)
  int cring_log2 = 0;  // candidate ring (rows of the validator's durations, pipelined kernel)
  size_t smem = 0;
  // the pipelined kernel's rings take rows of any count, so they fill the shared
  // memory left: without a candidate ring (a composition with the original
  // durations) and with one (a composition that reads the validator's)
  uint32_t pipe_drows = 0, pipe_drows_c = 0, pipe_crows = 0;
};

// Shared-memory layout of the staged kernels (byte offsets).  Every region starts
// on a 16-byte boundary, as 16-byte copy destinations require.
struct StagedLayout {
  size_t hist, meta, vr, dr, rr, cr, total;
};
__host__ __device__ inline size_t round16(size_t x) { return (x + 15) & ~(size_t)15; }
// d_rows, c_rows: rows of the duration and candidate rings.
__host__ __device__ inline StagedLayout staged_layout(int sigma, int vlog2, size_t d_rows, int rlog2, size_t c_rows) {
  StagedLayout L;
  L.hist = 128;                        // [0, 128): per-scenario makespans
  L.meta = L.hist + 16 * 8;            // 16 copy-group extents
  L.vr = L.meta + round16((size_t)2 * kMetaCap * 16);
  L.dr = L.vr + round16(((size_t)1 << vlog2) * sigma * 8);
  L.rr = L.dr + round16(d_rows * sigma * 8);
  L.cr = L.rr + round16(((size_t)1 << rlog2) * 4);
  L.total = L.cr + round16(c_rows * sigma * 8);
  return L;
}

// Validator: for each overlap candidate (a compute op), whether its interval
// overlaps a comm op of its rank, and the duration to use in the next composition.
struct OverlapArgs {
  MatLayout lay;           // [V][S] matrices
  MatLayout lay_c;         // [n_cand][S] compact matrices (rows in level order)
  int32_t S, n_streams;
  int32_t n_cq;            // comm timelines per rank (lists of a rank with fewer are empty)
  int32_t n_ranks;
  int32_t parts;           // pieces of each rank's candidate list (one warp per piece and 32 scenarios)
  const int64_t *cand_off; const int32_t *cand_ops;  // [R+1]: each rank's overlap candidates, in issue order
  const int32_t *cand_cidx;                          // level-order index of each entry of cand_ops
  const uint8_t *cand_kcl;                           // kernel class of each entry of cand_ops
  const int64_t *cq_off; const int32_t *cq_ops;  // [R*n_cq+1]: comm ops of each (rank, comm timeline)
  // launch conditions of each entry of cq_ops on its rank (CSR); null: a comm op's
  // interval is its execution [start, finish), else [latest of them, finish)
  const int32_t *lq_off, *lq_ops;
  const uint8_t *kcl;      // [V]
  const int64_t *f;        // finish times of the last pass
  const int64_t *dur;      // original durations
  const int64_t *cd_used;  // candidates' durations in the last pass (compact), or null: the original ones
  const double *sf;        // [C][S] slowdown factors
  int32_t model;           // 0: d * factor; 1: d + (factor - 1) * overlapped length
  int64_t *cd_next;        // (out, compact; may be null) candidates' durations for the next pass
  uint8_t *ov;             // (out, [V][S] rows of the candidates; may be null)
  int32_t n_kclass;        // rows of sf
  int32_t dbg;             // debug bounds: check every index (echo_bounds.h)
  int32_t *status;
};

// Dataflow composer (echo_dataflow.cu): one warp per (rank, group of 32
// scenarios), matrices in rows of 32 scenarios.  A rank's program lists its ops in
// internal order, 8 words each: node, level-order candidate index (~0u: none),
// header, offset of its other inputs in `opnd`, first partial slot (comm ops),
// member count | own member index << 16 (comm ops), export id (an op whose finish
// other warps read, or a two-hop join's), 0.  Header: bits 0-3 the op's timeline
// on the rank, kDf* flags (kDfPrev: the op before it in the program is an input),
// bits 8-15 the number of other inputs, bits 16-31 the rank's timelines whose
// latest op is another input.  Other inputs: top 2 bits the
// kind, an earlier op of the rank (node id) or another warp's op (export id).
// Published values are times (below 2^61) tagged with the launch's epoch (1-7)
// in the top 3 bits.
constexpr int kDfBatch = 8;
constexpr int kDfDepth = 3;       // batches of durations in flight ahead of the one in use
constexpr uint32_t kDfPayload = 0x3FFFFFFFu;
enum : uint32_t { kDfInLocal = 1, kDfInRemote = 2 };
enum : uint32_t { kDfComm = 1u << 4, kDfPrev = 1u << 5, kDfExport = 1u << 6, kDfTwoHop = 1u << 7 };
// anything beyond "the previous op of the program is the only input"
constexpr uint32_t kDfSlowMask = 0xFFFFFF00u | kDfComm | kDfExport | kDfTwoHop;
constexpr uint32_t kDfDirectMembers = 8;  // larger groups gather at their first member
// a comm op whose members are the ranks of one block: its slot word holds this
// flag and the op's sequence number among the block's joins (shared-memory join)
constexpr uint32_t kDfBlockJoin = 0x80000000u;
constexpr int kDfMaxWarpsPerBlock = 8;

struct DataflowArgs {
  int32_t S, G, R, n_streams;  // scenarios, groups of 32 scenarios, ranks, timelines per rank
  int64_t V, n_cand, n_slots, n_exports;  // rows of dur / f, of cdur, of part, of xval
  const int64_t *off;          // [R+1] program entries of each rank
  const uint32_t *rec;         // [entries][8]
  const uint32_t *opnd;
  const int64_t *dur;          // durations (comm rows: the CC durations)
  const int64_t *cdur;         // candidates' durations (compact), or null: dur
  int64_t *f;                  // finish times
  uint64_t *part;              // [n_slots][S] tagged partial launch times of comm ops
  uint64_t *xval;              // [n_exports][S] tagged finishes read by other warps
  uint32_t epoch;              // this launch's tag, 1-7 (0 marks a word never written)
  int32_t *abort_flag;         // set by a warp whose wait gave up (zeroed before the launch)
  int64_t *makespan;           // [S] (zeroed before the launch)
  int32_t *status;
  long long wait_limit_cycles;
  int64_t skip_slot;           // failure injection for tests: this partial is never published (-1: none)
  int64_t n_opnd;              // words of opnd
  int32_t dbg;                 // debug bounds: check every index (echo_bounds.h)
  int32_t wpb;                 // warps per block (consecutive ranks of one scenario group)
};
cudaError_t launch_compose_dataflow(const DataflowArgs &a, cudaStream_t st);
size_t dataflow_smem_bytes(int32_t n_streams, int32_t wpb);
// whether every warp of R * G warps can be resident at once (cooperative launch)
bool dataflow_fits(int64_t n_warps, int32_t n_streams, int32_t wpb, int device);

// shared memory of an overlap-test block: each warp's ring of candidate rows
inline size_t overlap_smem_bytes() { return (size_t)kOvWarps * kOvDepth * kOvBatch * 2 * 32 * sizeof(int64_t); }

// overlap.cu: the overlap test, one entry point per (launch interval, proportional
// model) pair, each dispatching on the number of comm timelines
cudaError_t launch_overlap_l0_p0(const OverlapArgs &a, dim3 grid, int tx, cudaStream_t st);
cudaError_t launch_overlap_l0_p1(const OverlapArgs &a, dim3 grid, int tx, cudaStream_t st);
cudaError_t launch_overlap_l1_p0(const OverlapArgs &a, dim3 grid, int tx, cudaStream_t st);
cudaError_t launch_overlap_l1_p1(const OverlapArgs &a, dim3 grid, int tx, cudaStream_t st);

// kernels.cu
// ar_policy: 0 each signature's own all-reduce algorithm, else 1 + the algorithm for all
cudaError_t launch_cc_estimate(const CcSig *sig, int32_t G, ScenParams p, int32_t S,
                               const ChunkTable &tbl, const int32_t *sig_count, double *cc_ns,
                               int64_t *cc_dur, double *comm_sum, int32_t *status, int model, int ar_policy,
                               cudaStream_t st);
cudaError_t launch_cc_scatter(const int32_t *comm_node, const int32_t *comm_sig, int64_t n_comm,
                              const int64_t *cc_dur, int32_t S, MatLayout lay, int64_t *dur, cudaStream_t st);
cudaError_t launch_cc_query(int64_t n, const uint8_t *type, const uint8_t *algo, const int64_t *nbytes,
                            const int32_t *N, const int32_t *M, const double *lg, ScenParams p,
                            const ChunkTable &tbl, double *out, cudaStream_t st);
// sets *flag when row pairs[2p] of the [V][S] matrix `raw` (int32 or int64) differs
// from row pairs[2p+1] in some scenario
cudaError_t launch_replica_check(const void *raw, int bits, const int32_t *pairs, int64_t n_pairs, int32_t S,
                                 int32_t *flag, cudaStream_t st);
cudaError_t launch_permute_rows(const void *raw, int bits, const int32_t *int2ext, const uint8_t *local,
                                int64_t V, int32_t S, MatLayout lay, int64_t *dur, double *sums, int32_t *status,
                                cudaStream_t st);
cudaError_t launch_compose(const ComposeArgs &a, int sigma, cudaStream_t st);
cudaError_t launch_compose_staged(const StagedArgs &a, int sigma, const StagedPlan &plan, cudaStream_t st);
cudaError_t launch_compose_pipelined(const StagedArgs &a, int sigma, const StagedPlan &plan, cudaStream_t st);
cudaError_t launch_overlap(const OverlapArgs &a, cudaStream_t st);
cudaError_t launch_readback(const int32_t *ext2int, int64_t op0, int64_t op1, int32_t s0, int32_t s1, MatLayout lay,
                            const int64_t *f, const int64_t *d, const int32_t *cidx, MatLayout lay_c,
                            const int64_t *cd, int64_t *start, int64_t *finish, cudaStream_t st);
cudaError_t launch_scatter_candidates(const int32_t *cand_node, int64_t n_cand, int32_t S, MatLayout lay,
                                      MatLayout lay_c, const int64_t *cd, int64_t *dst, cudaStream_t st);
cudaError_t launch_read_cc(const int32_t *ext2int, int64_t op0, int64_t op1, int32_t S,
                           const int32_t *node_sig, const double *cc_ns, double *out, cudaStream_t st);
cudaError_t launch_read_ov(const int32_t *ext2int, int64_t op0, int64_t op1, int32_t S, MatLayout lay,
                           const uint8_t *ov, const uint8_t *cand, uint8_t *out, cudaStream_t st);
size_t compose_smem_bytes(int32_t n_queues, int sigma, bool *frontier_in_smem);

}  // namespace echo
