/*
 * echo_oracle.h -- TEST INFRASTRUCTURE ONLY: the CPU oracle's own declarations.
 * Nothing in the product library includes this file.
 */
#ifndef ECHO_ORACLE_H
#define ECHO_ORACLE_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum { ORACLE_OK = 0, ORACLE_E_INVALID = 1, ORACLE_E_DEADLOCK = 2, ORACLE_E_NOMEM = 3 };

typedef struct {
  int64_t n_ops;
  int32_t n_ranks, n_streams, gpus_per_node, n_groups;
  const uint8_t *kind, *kclass, *cc_type, *cc_algo;
  const int32_t *group;
  const int64_t *cc_bytes;
  const int64_t *pred_off;
  const int32_t *pred_idx;
  const int64_t *q_off; /* [n_ranks*n_streams+1]; queue r*n_streams+k */
  const int32_t *q_ops;
  const int64_t *grp_off;
  const int32_t *grp_rank;
} oracle_graph;

typedef struct {
  int32_t n_scen, n_kclass, n_chunk;
  const int64_t *dur; /* [n_ops][n_scen] */
  const double *alpha_ns, *bw_intra, *lat_intra, *bw_inter, *lat_inter, *delta; /* [n_scen] */
  const double *slowdown;                                                      /* [n_kclass][n_scen] */
  const int64_t *chunk_max_bytes, *chunk_bytes; /* [n_chunk]; n_chunk = 0 -> Table 6 */
  int32_t cc_model; /* 0: Eqs. 2-5 (white box), 1: alpha-beta */
  int32_t overlap_model; /* 0: an overlapped kernel takes d * factor;
                            1: d + (factor - 1) * (length of its overlap) */
  int32_t comm_interval; /* what counts as a comm op's interval on a member rank r:
                            0: its execution [start, finish);
                            1: [launch on r, finish), launch = when r's own launch
                               conditions of it hold */
  int32_t ar_algo_policy; /* all-reduce algorithm (Sec. 5.1: NCCL runs ring or tree):
                             0: each op's own cc_algo; 1: ring, 2: tree, 3: the
                             faster of the two, for every all-reduce */
} oracle_scen;

int64_t oracle_chunk_bytes(int64_t nbytes, int n_chunk, const int64_t *max_bytes,
                           const int64_t *chunk_bytes);

/* prm = {alpha_ns, bw_intra, lat_intra, bw_inter, lat_inter, delta} */
double oracle_cc_ns(int cc_type, int cc_algo, int64_t nbytes, int N, int M, int K, double lg,
                    const double *prm, int n_chunk, const int64_t *max_bytes,
                    const int64_t *chunk_bytes);

/* prm as above; message size over bandwidth plus latency on the bottleneck link */
double oracle_cc_ns_alpha_beta(int64_t nbytes, int N, int M, const double *prm);

/* Composes scenarios [s0, s1).  Outputs are [n_ops][n_scen] (only the columns in
 * range are written); any output pointer may be NULL. */
int oracle_compose(const oracle_graph *g, const oracle_scen *sc, int32_t s0, int32_t s1,
                   int32_t refine_passes, uint64_t tie_seed, int64_t *start, int64_t *finish,
                   int64_t *makespan, double *cc_ns, uint8_t *overlapped);

#ifdef __cplusplus
}
#endif
#endif
