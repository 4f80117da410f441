/*
 * echo.h -- C ABI of the GB300 (sm_103a) timeline composer for Echo-style
 * distributed-training simulation (arXiv 2412.12487).
 *
 * One context owns one device, one CUDA stream and all device memory it uses.
 * The calls follow the paper's statement of the problem:
 *
 *   echo_load_graph            per-rank execution graphs merged into one graph (Sec. 4.1-4.2)
 *   echo_load_scenarios        what-if parameters: kernel durations, link parameters,
 *                              slowdown factors (Sec. 3 inputs, Sec. 5.3 parameters)
 *   echo_estimate_collectives  CC estimator: sync join + execution closed forms (Sec. 5.2-5.3)
 *   echo_compose               timeline composer (Sec. 4.2) + validator adjustment (Sec. 3, 6)
 *   echo_read_*                per-op start/finish, step makespan, CC estimates
 *
 * Conventions for every call:
 *   - The return value is an echo_status; ECHO_OK (0) on success.  On failure the
 *     context keeps its previous state and echo_last_error() describes the cause.
 *   - Array arguments are caller-owned HOST memory unless stated otherwise.  They
 *     are read (or written) during the call only; nothing keeps a pointer to them.
 *     Pinned (page-locked) host memory makes the copies faster but is not required.
 *   - Op ids are the caller's ids 0..n_ops-1.  The library renumbers internally
 *     and never exposes its own numbering.
 *   - Times are int64 nanoseconds; the first op of every timeline may start at 0.
 *   - A context is not thread-safe.  Different contexts are independent.
 *   - Calls must come in order: graph -> scenarios -> estimate -> compose -> read.
 *     Loading a new graph invalidates the scenarios; loading new scenarios
 *     invalidates the estimates and the composition.  Out of order: ECHO_E_STATE.
 *   - Work is enqueued on the context's stream.  echo_load_*, echo_estimate_collectives
 *     and echo_read_* synchronize with that stream before returning (they report
 *     input errors found on the device); echo_compose only enqueues.
 */
#ifndef ECHO_H
#define ECHO_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define ECHO_ABI_VERSION 2

typedef enum {
  ECHO_OK = 0,
  ECHO_E_INVALID_ARG = 1, /* null pointer, bad size, negative duration, bad parameter */
  ECHO_E_BAD_GRAPH = 2,   /* index out of range, inconsistent timelines or groups     */
  ECHO_E_CYCLE = 3,       /* the dependencies (data + issue order) form a cycle        */
  ECHO_E_STATE = 4,       /* call made out of order                                    */
  ECHO_E_OOM = 5,         /* device or host allocation failed                          */
  ECHO_E_CUDA = 6,        /* a CUDA runtime call failed                                */
  ECHO_E_TIMEOUT = 7,     /* a bounded device-side wait gave up                        */
  ECHO_E_OVERFLOW = 8,    /* a finish time could exceed the int64 range                */
  ECHO_E_UNSUPPORTED = 9, /* a size beyond what the library supports                   */
  ECHO_E_BOUNDS = 10      /* a device-side index check failed (debug_bounds)           */
} echo_status;

/* op kinds (Sec. 4.2 timelines: computation, communication, memcpy) */
enum { ECHO_OP_COMPUTE = 0, ECHO_OP_MEMCPY = 1, ECHO_OP_COLL = 2, ECHO_OP_P2P = 3 };
/* collective types of Sec. 5.3 (send/recv is the P2P primitive of Sec. 5.2) */
enum { ECHO_CC_ALLREDUCE = 0, ECHO_CC_ALLGATHER = 1, ECHO_CC_REDUCESCATTER = 2, ECHO_CC_SENDRECV = 3 };
/* all-reduce algorithm (Sec. 5.1: NCCL runs ring or tree all-reduce; AUTO = the faster) */
enum { ECHO_ALGO_RING = 0, ECHO_ALGO_TREE = 1, ECHO_ALGO_AUTO = 2 };
/* collective cost models (echo_set_cc_model) */
enum { ECHO_CC_MODEL_WHITEBOX = 0, ECHO_CC_MODEL_ALPHA_BETA = 1 };

typedef struct echo_ctx echo_ctx;

/*
 * Multi-rank execution graph (Sec. 4.1: per-rank graphs of compute and comm ops;
 * Sec. 4.2: inter-rank dependency and matching rules, given here as shared comm
 * nodes and explicit data edges).
 *
 * Timelines: every rank r has n_streams serial timelines ("streams").  Queue
 * q = r * n_streams + k lists, in issue order, the ops rank r runs on its stream k.
 *   - stream 0 is the rank's compute timeline: it holds exactly the rank's
 *     ECHO_OP_COMPUTE ops and nothing else;
 *   - streams 1..n_streams-1 are communication / memcpy timelines;
 *   - a COMPUTE or MEMCPY op appears in exactly one queue;
 *   - a COLL or P2P op appears exactly once on every member rank of its group
 *     (in any stream >= 1 of that rank) and on no other rank.
 * An op starts when, on each of its timelines, the op issued before it has
 * finished, and all its data predecessors have finished (Sec. 5.2: a collective
 * starts when its last member launches; a P2P op waits for its peer).  Its finish
 * is start + duration.
 */
typedef struct {
  int64_t n_ops;           /* V >= 0                                                   */
  int32_t n_ranks;         /* >= 1                                                      */
  int32_t n_streams;       /* timelines per rank, 1..16                                 */
  int32_t gpus_per_node;   /* ranks r and r' share a node iff r/gpus_per_node equal     */
  int32_t n_groups;        /* communicator groups                                      */
  const uint8_t *kind;     /* [V] ECHO_OP_*                                             */
  const uint8_t *kclass;   /* [V] compute ops: kernel class = row of the slowdown table */
  const int32_t *group;    /* [V] COLL/P2P ops: group index; ignored for other kinds    */
  const uint8_t *cc_type;  /* [V] COLL: ALLREDUCE/ALLGATHER/REDUCESCATTER; P2P: SENDRECV */
  const uint8_t *cc_algo;  /* [V] all-reduce ops: ECHO_ALGO_*; ignored otherwise        */
  const int64_t *cc_bytes; /* [V] comm ops: message size in bytes (>= 0)                */
  const int64_t *pred_off; /* [V+1] CSR of data dependencies, pred_off[0] = 0           */
  const int32_t *pred_idx; /* [pred_off[V]] predecessor op ids                          */
  const int64_t *q_off;    /* [n_ranks*n_streams+1] CSR of the timelines, q_off[0] = 0  */
  const int32_t *q_ops;    /* [q_off[n_ranks*n_streams]] op ids in issue order          */
  const int64_t *grp_off;  /* [n_groups+1] CSR of group members, grp_off[0] = 0         */
  const int32_t *grp_rank; /* [grp_off[n_groups]] member ranks, no repeats; P2P: 1 or 2 */
  const int32_t *replica_of; /* [n_ranks] or NULL: replica folding, see below         */
} echo_graph_desc;

/*
 * Replica folding (Sec. 8.5: in DDP mode Echo simulates one copy of the workload
 * per DP group).  replica_of[b] = a marks rank b as a replica of rank a, and
 * replica_of[a] = a marks a representative.  A replica runs the same ops as its
 * representative, timeline by timeline and position by position: the op at
 * position i of b's timeline k is either an op that a representative also runs
 * (then it is the same op, e.g. a DP all-reduce shared by the replicas) or a copy
 * of the op at position i of a's timeline k with the same kind, kernel class,
 * message, group shape, data producers (up to the same mapping) and launch
 * conditions.  echo_load_graph checks this (ECHO_E_BAD_GRAPH otherwise) and
 * composes only the representatives' ops while every scenario batch gives each
 * copied compute or memcpy op the durations of its original (checked on the
 * device by echo_load_scenarios; a batch that does not runs the full graph).  The
 * times are exactly those of the full graph: a copy reports its original's.
 */

/*
 * S what-if scenarios.  All arrays are host memory; dur is row-major [V][S]
 * (scenario index innermost).  Link parameters feed the CC estimator of Sec. 5.3:
 * bandwidths in bytes/ns (= GB/s), latencies and alpha (connection setup) in ns,
 * delta (reduction cost) in ns per byte.  slowdown[c][s] is the factor of
 * Sec. 2.3 for a compute op of kernel class c that overlaps communication in
 * scenario s; it stands in for the XGBoost predictor of Sec. 6.
 */
typedef struct {
  int32_t n_scen;                  /* S >= 1                                          */
  int32_t n_kclass;                /* rows of slowdown; > every compute op's kclass   */
  int32_t n_chunk;                 /* entries of the chunk table, 0 = Table 6 default */
  const void *dur;                 /* [V][S] ns >= 0 (int64, or int32 when dur_bits is
                                      32); entries of COLL/P2P ops ignored            */
  const double *alpha_ns;          /* [S] >= 0                                        */
  const double *bw_intra;          /* [S] > 0, intra-node link                        */
  const double *lat_intra;         /* [S] >= 0                                        */
  const double *bw_inter;          /* [S] > 0, inter-node link                        */
  const double *lat_inter;         /* [S] >= 0                                        */
  const double *delta;             /* [S] >= 0                                        */
  const double *slowdown;          /* [n_kclass][S], each in (0, 1e6]                  */
  const int64_t *chunk_max_bytes;  /* [n_chunk] ascending: messages <= max use ...    */
  const int64_t *chunk_bytes;      /* [n_chunk] ... this chunk size (> 0); larger
                                      messages use the last entry                     */
  int32_t dur_bits;                /* width of the dur entries: 64 (0 means 64) or 32;
                                      32 halves the upload when every duration fits;
                                      the composition computes in int64 either way    */
} echo_scen_desc;

typedef struct {
  /* validator passes after the first composition (Sec. 3: compose, then adjust the
   * overlapped ops).  0 = compose only; 1 = the paper's flow (default); k > 1
   * recomputes the overlap from pass k's times and always slows the ORIGINAL
   * durations.  At most 8. */
  int32_t refine_passes;
  /* how an overlapped kernel is slowed: ECHO_OVERLAP_WHOLE (default) multiplies its
   * duration by its factor (Sec. 2.3: the factor is the ratio of its times with and
   * without overlapping communication); ECHO_OVERLAP_PROPORTIONAL adds (factor - 1)
   * times the length of its interval covered by its rank's comm intervals. */
  int32_t overlap_model;
  /* the interval of a comm op on a member rank r that the validator tests:
   * ECHO_COMM_EXECUTION (default) its execution [start, finish), the same on every
   * member (Sec. 5.2: it starts once the last member has launched it);
   * ECHO_COMM_LAUNCH [launch on r, finish), where r has launched it once the op
   * before it on r's timeline and its data producers that run on r have finished:
   * the comm kernel is resident on r while it waits for the other members. */
  int32_t comm_interval;
  /* all-reduce algorithm (Sec. 5.1: NCCL runs an all-reduce as a ring or a tree):
   * ECHO_AR_PER_OP (0, default) keeps each op's cc_algo; ECHO_AR_RING, ECHO_AR_TREE
   * and ECHO_AR_AUTO (the faster of the two) apply to every all-reduce of the
   * graph.  When it differs from the policy of the current estimates, echo_compose
   * runs the CC estimator again first (ECHO_E_OVERFLOW as there), and echo_read_cc
   * then reports those estimates. */
  int32_t ar_algo_policy;
  /* nonzero: every index the composition and validator kernels gather through (from
   * the graph's records, programs and candidate and comm lists) is checked on the
   * device against the bounds of the buffer it indexes before the access; a failed
   * check skips the access, stops the kernel's walk and makes the next echo_read_*
   * return ECHO_E_BOUNDS.  Never traps.  For debugging; slower.  The environment
   * variable ECHO_DEBUG_BOUNDS=1 turns it on for every composition. */
  int32_t debug_bounds;
} echo_compose_opts;
enum { ECHO_OVERLAP_WHOLE = 0, ECHO_OVERLAP_PROPORTIONAL = 1 };
enum { ECHO_COMM_EXECUTION = 0, ECHO_COMM_LAUNCH = 1 };
enum { ECHO_AR_PER_OP = 0, ECHO_AR_RING = 1, ECHO_AR_TREE = 2, ECHO_AR_AUTO = 3 };

/* Create a context on `device`, enqueuing on `cuda_stream` (a cudaStream_t; NULL =
 * a new non-blocking stream owned by the context; the legacy default stream is
 * passed as cudaStreamLegacy).  The caller's stream must outlive the context. */
int echo_create(echo_ctx **out, int device, void *cuda_stream);
/* Free everything the context owns.  NULL is accepted. */
int echo_destroy(echo_ctx *ctx);

/* Host-only check of a graph: the validation and topological levelling that
 * echo_load_graph performs, without a device.  Writes the number of levels and
 * the widest level (either pointer may be NULL). */
int echo_check_graph(const echo_graph_desc *g, int64_t *n_levels, int64_t *max_width);

/* Host-only overlap candidates: the compute ops that the validator pass (Sec. 3, 6)
 * tests.  This pruning is a static analysis of this library, not a step of the
 * paper, and never changes a result: flags[v] = 1
 * for every compute op v (caller ids) that can overlap a comm op of its rank in
 * some scenario, judged from the issue order and data edges among the rank's own
 * ops (an op that must finish before the comm op starts, or start after it ends,
 * never overlaps it).  flags: [n_ops] host buffer, or NULL; *n_candidates their
 * count, or NULL.  Errors as echo_check_graph. */
int echo_overlap_candidates(const echo_graph_desc *g, uint8_t *flags, int64_t *n_candidates);

/* Host-only check of a graph with replica_of: the validation echo_load_graph
 * performs, and the number of ops the folded graph composes (n_ops when
 * replica_of is NULL or marks no replica).  Errors as echo_load_graph. */
int echo_check_replicas(const echo_graph_desc *g, int64_t *n_ops_folded);

/* Validate, level (ASAP depth over data + issue-order dependencies), renumber in
 * level order and upload the graph.  Errors: ECHO_E_INVALID_ARG, ECHO_E_BAD_GRAPH,
 * ECHO_E_CYCLE, ECHO_E_UNSUPPORTED, ECHO_E_OOM, ECHO_E_CUDA. */
int echo_load_graph(echo_ctx *ctx, const echo_graph_desc *g);

/* Copy the scenarios to the device (durations permuted into the internal order)
 * and check them: negative durations -> ECHO_E_INVALID_ARG. */
int echo_load_scenarios(echo_ctx *ctx, const echo_scen_desc *sc);

/* CC estimator (Sec. 5.2-5.3): for every comm op and scenario, the execution time
 * of Eqs. 2-5 (ring all-gather, ring reduce-scatter, ring/tree/auto all-reduce,
 * send/recv, each all-reduce with its own cc_algo) in fp64 ns; the op's duration
 * is that value rounded to the nearest integer (ties to even).  Group shape: N members, M distinct nodes, K = the
 * largest member count on one node, log2(M) computed on the host.  A time that
 * could overflow the composition -> ECHO_E_OVERFLOW. */
int echo_estimate_collectives(echo_ctx *ctx);

/* Cost model of the next echo_estimate_collectives.  ECHO_CC_MODEL_WHITEBOX (the
 * default) is Eqs. 2-5 above.  ECHO_CC_MODEL_ALPHA_BETA is the model Sec. 2.3
 * describes for the simulators Echo is compared with (NCCL-Predictor, Sec. 8.3):
 * message size over bandwidth plus latency, here on the group's bottleneck link
 * (inter-node when the group spans nodes), 0 for N = 1 or 0 bytes, every
 * collective type alike; comparing the two shows how the makespan depends on the
 * estimator.  A context that had estimated must estimate again before composing.
 * An unknown model -> ECHO_E_INVALID_ARG. */
int echo_set_cc_model(echo_ctx *ctx, int model);

/* Timeline composer (Sec. 4.2) over all scenarios, then `refine_passes` validator
 * passes (Sec. 3, 2.3): a compute op whose [start, finish) interval overlaps, with
 * positive length, the interval of a comm op its rank takes part in gets duration
 * rint(d * slowdown[kclass][s]) and the timeline is composed again.  Only
 * enqueues work; opts may be NULL (refine_passes = 1). */
int echo_compose(echo_ctx *ctx, const echo_compose_opts *opts);

/* Final start and finish (Sec. 4.2: every op's place on its timelines) of ops
 * [op0, op1) (caller ids) in scenarios [s0, s1), into caller buffers of
 * (op1-op0)*(s1-s0) int64 each, row-major [op][s - s0]: host memory (pageable or
 * pinned) or device memory of the context's device.  Either may be NULL.  A range
 * outside [0, n_ops) x [0, n_scen) or an empty scenario range with ops:
 * ECHO_E_INVALID_ARG.  Large ranges are read back in chunks through a staging
 * buffer of the context. */
int echo_read_times(echo_ctx *ctx, int64_t op0, int64_t op1, int32_t s0, int32_t s1, int64_t *start,
                    int64_t *finish);
/* Step time per scenario: the largest finish time (0 for an empty graph). [S] */
int echo_read_makespan(echo_ctx *ctx, int64_t *makespan);
/* CC estimates (fp64 ns) of ops [op0, op1), [op][s]; NaN for non-comm ops. */
int echo_read_cc(echo_ctx *ctx, int64_t op0, int64_t op1, double *cc_ns);
/* Validator decisions of the last pass for ops [op0, op1), [op][s]: 1 = slowed. */
int echo_read_overlap(echo_ctx *ctx, int64_t op0, int64_t op1, uint8_t *overlapped);

/* Standalone CC estimator queries (Sec. 5.3), one fp64 time per query. */
typedef struct {
  int64_t n;                /* number of queries                                    */
  const uint8_t *cc_type;   /* [n] ECHO_CC_*                                        */
  const uint8_t *cc_algo;   /* [n] all-reduce: ECHO_ALGO_*                          */
  const int64_t *nbytes;    /* [n] >= 0                                             */
  const int32_t *n_ranks;   /* [n] N >= 1                                           */
  const int32_t *n_nodes;   /* [n] 1 <= M <= N; K = ceil(N/M) (most even layout)    */
  const double *alpha_ns, *bw_intra, *lat_intra, *bw_inter, *lat_inter, *delta; /* [n] */
  int32_t n_chunk;          /* chunk table as in echo_scen_desc (0 = Table 6)       */
  const int64_t *chunk_max_bytes, *chunk_bytes;
} echo_cc_query_desc;
int echo_cc_query(echo_ctx *ctx, const echo_cc_query_desc *q, double *out_ns);

/* Allocation-free variant of echo_cc_query.  The paper has no counterpart: this
 * entry point exists for callers that cannot call cudaMalloc, such as a process
 * whose device memory belongs to a framework's memory pool or one that runs under
 * a fixed device-memory budget.  It needs no context and allocates nothing.
 *   - The per-query arrays of *q and out_ns are DEVICE memory owned by the caller
 *     (out_ns: n doubles); the chunk table fields of *q are host memory.
 *   - Work runs on `cuda_stream` (a cudaStream_t; NULL = the default stream) of the
 *     current device, and the call waits for that stream before returning.
 *   - Besides the caller's arrays it uses one static device array of about 520 KB
 *     (a status word and log2(m) for m = 1..65536), which every GPU that loads the
 *     library holds until the process exits.  The first call on a device fills
 *     that table with a synchronous copy, so make the first call on each device
 *     before any stream capture.
 *   - Every call shares the array and clears its status word: calls that overlap
 *     on the GPU race.
 *   - A query whose node count M exceeds 65536 gets NaN, and so does a malformed
 *     query (the checks of echo_cc_query); other queries are still estimated.  The
 *     call returns ECHO_E_INVALID_ARG if any query was malformed, else
 *     ECHO_E_UNSUPPORTED if any node count was too large, whatever the mix. */
int echo_cc_query_noalloc(const echo_cc_query_desc *q, double *out_ns, void *cuda_stream);

/* Shape of the loaded graph (after echo_load_graph).  n_ops counts the caller's
 * ops; every other count describes the graph being composed, the folded one while
 * replicas are folded (replicas_folded = 1, see replica_of). */
typedef struct {
  int64_t n_ops, n_edges, n_levels, max_width, n_queue_entries, n_comm_ops, n_signatures;
  int64_t n_segments;        /* serial chains the composer contracts into one step each */
  int64_t n_segment_levels;  /* synchronized steps of one composition                   */
  int64_t n_overlap_candidates; /* compute ops the validator tests (the others can never
                                   overlap a comm op of their rank, whatever the durations) */
  int64_t n_ops_composed;    /* ops of the graph being composed                       */
  int32_t n_ranks, n_streams, sigma; /* sigma: scenarios per thread block of the composer;
                                        32: the dataflow composer (a warp per rank and 32
                                        scenarios), chosen for graphs with many levels and
                                        few scenarios */
  int32_t replicas_folded;
  int64_t n_validator_comm_entries; /* (comm op, member rank) pairs the validator's cursors
                                       visit: those that can overlap a compute op of the rank */
  int64_t n_kept_finishes;  /* ops whose finish a composition before the last stores (the
                               others are read by no later step); n_ops_composed for the
                               dataflow composer, which stores every finish */
} echo_graph_info;
int echo_graph_info_get(echo_ctx *ctx, echo_graph_info *info);

/* Kernel timing with CUDA events on the context's stream.  While enabled, every
 * kernel the library launches is bracketed by two events.  echo_read_profile
 * synchronizes, reports per kernel name the launches and total milliseconds
 * since the last read (up to `cap` entries, count in *n) and clears the record. */
typedef struct {
  char name[48];
  int64_t launches;
  double total_ms;
} echo_kernel_stat;
int echo_set_profiling(echo_ctx *ctx, int enable);
int echo_read_profile(echo_ctx *ctx, echo_kernel_stat *out, int cap, int *n);

/* Measurement support (the paper has no counterpart): the fp64 rates of `device`,
 * in operations per second, of round-to-nearest add, multiply and divide
 * (rates[0..2]), from CUDA-event timing of independent chains of each.  The
 * roofline of the CC estimator's fp64 arithmetic uses them.  Changes no clock or
 * setting of the device; the calling thread's current device is restored.
 * Allocates and frees 8 bytes. */
int echo_measure_fp64(int device, double *rates);

const char *echo_strerror(int status);
/* Copies the context's last error message (NUL-terminated) into buf. */
int echo_last_error(echo_ctx *ctx, char *buf, size_t n);

#ifdef __cplusplus
}
#endif
#endif /* ECHO_H */
