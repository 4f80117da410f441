/*
 * echo_oracle.c -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, single-threaded CPU restatement of what the Echo simulator
 * (arXiv 2412.12487) computes on its hot path.  It exists to check the CUDA path
 * and is never part of it: only the tests, the smoke check and the benchmark's
 * CPU-baseline leg load it.  It shares no code, header, table or helper with the
 * product library.
 *
 * What it follows:
 *   - Sec. 4.2 (Timeline Composing): an event-driven simulator walks the per-rank
 *     execution graphs and puts every op on its rank's compute, communication or
 *     memcpy timeline.  Each (rank, stream) timeline runs its ops one after the
 *     other in issue order.
 *   - Sec. 5.2 (synchronization): a collective starts when the last member
 *     communicator has launched; a send/recv waits for its peer.  Both are a join
 *     over the members' launch conditions.
 *   - Sec. 5.3, Eqs. 2-5 (execution time): ring all-gather, ring reduce-scatter,
 *     ring all-reduce and tree all-reduce closed forms, with eta = number of
 *     chunks and the chunk size of Table 6.
 *   - Sec. 2.3 (slowdown factor = time with overlapping comm / time without) and
 *     Sec. 3 (the validator adjusts overlapped ops after composing): a compute op
 *     whose first-pass interval overlaps a communication op on the same rank is
 *     stretched by its factor and the timeline is composed again.
 *
 * Readings where the paper is silent or garbled:
 *   time is int64 ns, sources start at 0; a rank has any number of serial streams
 *   (its compute timeline plus comm/memcpy timelines); overlap means
 *   a positive-length intersection of [start, finish) intervals and slows the
 *   whole kernel (variants: only the overlapped length is slowed; a comm op's
 *   interval on rank r opens when r has launched it, the latest finish among its
 *   launch conditions on r, rather than when the last member has); the bare "(N-1)" inside Eqs. 3-4 is read as a per-step latency,
 *   so every ring step costs L + p/B; send/recv costs eta chunk transfers over the
 *   intra- or inter-node link; AUTO all-reduce takes the faster of ring and tree
 *   (ties to ring); an all-reduce policy (ring, tree or auto for every all-reduce)
 *   may replace the per-op algorithm; N = 1 or 0 bytes costs 0; slowed duration =
 *   rint(d * factor).
 *
 * Parity pins: see tests/test_oracle_pins.py.  Every function here is pinned
 * (closed forms, Table 6, brute force, invariants); none is "parity unpinned".
 */
#include "echo_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

enum { K_COMPUTE = 0, K_MEMCPY = 1, K_COLL = 2, K_P2P = 3 };
enum { T_AR = 0, T_AG = 1, T_RS = 2, T_SR = 3 };
enum { A_RING = 0, A_TREE = 1, A_AUTO = 2 };

/* Table 6 (H800, 32 GPUs): chunk size per tensor size.  MB read as 2^20 bytes,
 * chunk sizes are 10^3 bytes.  Between the printed sizes the next printed size's
 * chunk applies; below 4 MB and above 256 MB the end values are kept. */
static const int64_t kTableMaxBytes[5] = {4LL << 20, 8LL << 20, 64LL << 20, 128LL << 20, INT64_MAX};
static const int64_t kTableChunk[5] = {18000, 36000, 72000, 144000, 288000};

int64_t oracle_chunk_bytes(int64_t nbytes, int n_chunk, const int64_t *max_bytes,
                           const int64_t *chunk_bytes) {
  if (n_chunk <= 0 || !max_bytes || !chunk_bytes) {
    n_chunk = 5;
    max_bytes = kTableMaxBytes;
    chunk_bytes = kTableChunk;
  }
  for (int i = 0; i < n_chunk; ++i)
    if (nbytes <= max_bytes[i]) return chunk_bytes[i];
  return chunk_bytes[n_chunk - 1];
}

static int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }

/* Eqs. 2-4: ring collectives.  eta rounds of chunks; each of the eta*(N-1) steps
 * (2*eta*(N-1) for all-reduce) moves p = S/(N*eta) bytes over the ring's slowest
 * link (inter-node when the group spans nodes). */
static double ring_time(int type, int64_t S, int N, int M, const double *prm, int64_t C) {
  double alpha = prm[0], Ba = prm[1], La = prm[2], Be = prm[3], Le = prm[4], delta = prm[5];
  int64_t eta = ceil_div(S, (int64_t)N * C);
  if (eta < 1) eta = 1;
  double p = (double)S / ((double)N * (double)eta);
  double L = (M > 1) ? Le : La;
  double B = (M > 1) ? Be : Ba;
  double t = L + p / B;
  if (type == T_AG) return alpha + (double)(eta * (N - 1)) * t;
  if (type == T_RS) return alpha + (double)(eta * (N - 1)) * t + delta * (double)S;
  return alpha + (double)(2 * eta * (N - 1)) * t + delta * (double)S; /* all-reduce */
}

/* Eq. 5: tree all-reduce.  eta chunks pipelined through K-1 intra-node hops up
 * and down (beta each) and log2(M) inter-node levels up and down (gamma each). */
static double tree_time(int64_t S, int M, int K, double lg, const double *prm, int64_t C) {
  double alpha = prm[0], Ba = prm[1], La = prm[2], Be = prm[3], Le = prm[4], delta = prm[5];
  int64_t eta = ceil_div(S, C);
  if (eta < 1) eta = 1;
  double pt = (double)S / (double)eta;
  double beta = La + pt / Ba;
  double gamma = (M > 1) ? Le + pt / Be : beta;
  return alpha + gamma * (double)(eta - 1) + 2.0 * beta * (double)(K - 1) + 2.0 * gamma * lg +
         delta * (double)S;
}

double oracle_cc_ns(int cc_type, int cc_algo, int64_t nbytes, int N, int M, int K, double lg,
                    const double *prm, int n_chunk, const int64_t *max_bytes,
                    const int64_t *chunk_bytes) {
  if (N <= 1 || nbytes <= 0) return 0.0;
  int64_t C = oracle_chunk_bytes(nbytes, n_chunk, max_bytes, chunk_bytes);
  if (cc_type == T_SR) {
    /* send/recv: eta chunk transfers over the link joining the two ranks */
    double alpha = prm[0];
    double L = (M > 1) ? prm[4] : prm[2];
    double B = (M > 1) ? prm[3] : prm[1];
    int64_t eta = ceil_div(nbytes, C);
    if (eta < 1) eta = 1;
    return alpha + (double)eta * (L + ((double)nbytes / (double)eta) / B);
  }
  if (cc_type != T_AR) return ring_time(cc_type, nbytes, N, M, prm, C);
  if (cc_algo == A_RING) return ring_time(T_AR, nbytes, N, M, prm, C);
  if (cc_algo == A_TREE) return tree_time(nbytes, M, K, lg, prm, C);
  double r = ring_time(T_AR, nbytes, N, M, prm, C);
  double t = tree_time(nbytes, M, K, lg, prm, C);
  return (t < r) ? t : r;
}

/* Total length covered by the intervals [lo[i], hi[i]) (their union): sort by
 * start, then sweep, counting each stretch once. */
static void sort_intervals(int64_t *lo, int64_t *hi, int64_t m) {
  for (int64_t i = 1; i < m; ++i) { /* insertion sort: the lists are short */
    int64_t a = lo[i], b = hi[i], j = i - 1;
    while (j >= 0 && lo[j] > a) {
      lo[j + 1] = lo[j];
      hi[j + 1] = hi[j];
      --j;
    }
    lo[j + 1] = a;
    hi[j + 1] = b;
  }
}
static int64_t union_length(int64_t *lo, int64_t *hi, int64_t m) {
  sort_intervals(lo, hi, m);
  int64_t total = 0, covered = INT64_MIN;
  for (int64_t i = 0; i < m; ++i) {
    int64_t a = lo[i] > covered ? lo[i] : covered;
    if (hi[i] > a) {
      total += hi[i] - a;
      covered = hi[i];
    }
  }
  return total;
}

/* The alpha-beta model that Sec. 2.3 describes for the simulators Echo compares
 * against (NCCL-Predictor, Sec. 8.3): a collective takes its message size over the
 * bandwidth plus the latency.  Read here on the group's bottleneck link, the
 * inter-node one when the group spans nodes; N = 1 or 0 bytes costs 0. */
double oracle_cc_ns_alpha_beta(int64_t nbytes, int N, int M, const double *prm) {
  if (N <= 1 || nbytes <= 0) return 0.0;
  double L = (M > 1) ? prm[4] : prm[2];
  double B = (M > 1) ? prm[3] : prm[1];
  return L + (double)nbytes / B;
}

/* ------------------------------------------------------------------------------ */
/* event-driven timeline composer (Sec. 4.2)                                      */
/* ------------------------------------------------------------------------------ */

typedef struct {
  int64_t t;
  uint64_t key;
  int32_t op;
} event_t;

static int ev_less(const event_t *a, const event_t *b) {
  if (a->t != b->t) return a->t < b->t;
  return a->key < b->key;
}

static void heap_push(event_t *h, int64_t *n, event_t e) {
  int64_t i = (*n)++;
  h[i] = e;
  while (i > 0) {
    int64_t p = (i - 1) / 2;
    if (!ev_less(&h[i], &h[p])) break;
    event_t tmp = h[i];
    h[i] = h[p];
    h[p] = tmp;
    i = p;
  }
}

static event_t heap_pop(event_t *h, int64_t *n) {
  event_t top = h[0];
  h[0] = h[--(*n)];
  int64_t i = 0;
  for (;;) {
    int64_t l = 2 * i + 1, r = l + 1, m = i;
    if (l < *n && ev_less(&h[l], &h[m])) m = l;
    if (r < *n && ev_less(&h[r], &h[m])) m = r;
    if (m == i) break;
    event_t tmp = h[i];
    h[i] = h[m];
    h[m] = tmp;
    i = m;
  }
  return top;
}

static uint64_t mix64(uint64_t x) {
  x += 0x9e3779b97f4a7c15ULL;
  x = (x ^ (x >> 30)) * 0xbf58476d1ce4e5b9ULL;
  x = (x ^ (x >> 27)) * 0x94d049bb133111ebULL;
  return x ^ (x >> 31);
}

typedef struct {
  int64_t V;
  const int64_t *pred_off;
  const int32_t *pred_idx;
  int64_t *succ_off; /* data successors */
  int32_t *succ_idx;
  int64_t *opq_off;  /* (queue, position) pairs of every op */
  int32_t *opq_q;
  int64_t *opq_pos;
  const int64_t *q_off;
  const int32_t *q_ops;
  int32_t *cnt;
  event_t *heap;
  uint64_t tie_seed;
} sim_t;

/* One composition: every op starts when all of its launch conditions hold (it
 * heads each of its timelines and its data producers have finished); time only
 * moves forward by popping the earliest finish event. */
static int simulate(sim_t *S, const int64_t *d, int64_t *st, int64_t *fin) {
  int64_t V = S->V, nh = 0, done = 0;
  for (int64_t v = 0; v < V; ++v)
    S->cnt[v] = (int32_t)((S->pred_off[v + 1] - S->pred_off[v]) + (S->opq_off[v + 1] - S->opq_off[v]));
  for (int64_t v = 0; v < V; ++v)
    for (int64_t k = S->opq_off[v]; k < S->opq_off[v + 1]; ++k)
      if (S->opq_pos[k] == 0) S->cnt[v]--; /* first in its timeline: nothing ahead */
  for (int64_t v = 0; v < V; ++v) {
    if (S->cnt[v] == 0) {
      st[v] = 0;
      event_t e = {d[v], S->tie_seed ? mix64((uint64_t)v ^ S->tie_seed) : (uint64_t)v, (int32_t)v};
      heap_push(S->heap, &nh, e);
    }
  }
  while (nh > 0) {
    event_t e = heap_pop(S->heap, &nh);
    int64_t now = e.t;
    int32_t u = e.op;
    fin[u] = now;
    done++;
    /* wake data consumers */
    for (int64_t k = S->succ_off[u]; k < S->succ_off[u + 1]; ++k) {
      int32_t w = S->succ_idx[k];
      if (--S->cnt[w] == 0) {
        st[w] = now;
        event_t x = {now + d[w], S->tie_seed ? mix64((uint64_t)w ^ S->tie_seed) : (uint64_t)w, w};
        heap_push(S->heap, &nh, x);
      }
    }
    /* the next op on each of u's timelines may now launch */
    for (int64_t k = S->opq_off[u]; k < S->opq_off[u + 1]; ++k) {
      int32_t q = S->opq_q[k];
      int64_t nxt = S->q_off[q] + S->opq_pos[k] + 1;
      if (nxt < S->q_off[q + 1]) {
        int32_t w = S->q_ops[nxt];
        if (--S->cnt[w] == 0) {
          st[w] = now;
          event_t x = {now + d[w], S->tie_seed ? mix64((uint64_t)w ^ S->tie_seed) : (uint64_t)w, w};
          heap_push(S->heap, &nh, x);
        }
      }
    }
  }
  return done == V ? 0 : ORACLE_E_DEADLOCK;
}

int oracle_compose(const oracle_graph *g, const oracle_scen *sc, int32_t s0, int32_t s1,
                   int32_t refine_passes, uint64_t tie_seed, int64_t *start, int64_t *finish,
                   int64_t *makespan, double *cc_ns, uint8_t *overlapped) {
  int64_t V = g->n_ops;
  int32_t S = sc->n_scen;
  if (V < 0 || S < 0 || s0 < 0 || s1 > S || s0 > s1 || refine_passes < 0) return ORACLE_E_INVALID;
  if (sc->ar_algo_policy < 0 || sc->ar_algo_policy > 3) return ORACLE_E_INVALID;
  int64_t nq = (int64_t)g->n_streams * g->n_ranks;
  int rc = 0;

  /* per-op timeline memberships, data successors, group shape (N, M, K, log2 M) */
  sim_t sim;
  memset(&sim, 0, sizeof sim);
  sim.V = V;
  sim.pred_off = g->pred_off;
  sim.pred_idx = g->pred_idx;
  sim.q_off = g->q_off;
  sim.q_ops = g->q_ops;
  sim.tie_seed = tie_seed;
  int64_t E = g->pred_off[V];
  int64_t QE = g->q_off[nq];
  sim.succ_off = calloc((size_t)V + 1, sizeof(int64_t));
  sim.succ_idx = malloc((size_t)(E > 0 ? E : 1) * sizeof(int32_t));
  sim.opq_off = calloc((size_t)V + 1, sizeof(int64_t));
  sim.opq_q = malloc((size_t)(QE > 0 ? QE : 1) * sizeof(int32_t));
  sim.opq_pos = malloc((size_t)(QE > 0 ? QE : 1) * sizeof(int64_t));
  sim.cnt = malloc((size_t)(V > 0 ? V : 1) * sizeof(int32_t));
  sim.heap = malloc((size_t)(V > 0 ? V : 1) * sizeof(event_t));
  int64_t *fill = calloc((size_t)V + 1, sizeof(int64_t));
  int64_t *d0 = malloc((size_t)(V > 0 ? V : 1) * sizeof(int64_t));
  int64_t *d = malloc((size_t)(V > 0 ? V : 1) * sizeof(int64_t));
  int64_t *st = malloc((size_t)(V > 0 ? V : 1) * sizeof(int64_t));
  int64_t *fn = malloc((size_t)(V > 0 ? V : 1) * sizeof(int64_t));
  uint8_t *ov = calloc((size_t)(V > 0 ? V : 1), 1);
  int64_t *cst = malloc((size_t)(QE > 0 ? QE : 1) * sizeof(int64_t)); /* one rank's comm intervals */
  int64_t *cfn = malloc((size_t)(QE > 0 ? QE : 1) * sizeof(int64_t));
  int64_t *clo = malloc((size_t)(QE > 0 ? QE : 1) * sizeof(int64_t)); /* clipped to one kernel */
  int64_t *chi = malloc((size_t)(QE > 0 ? QE : 1) * sizeof(int64_t));
  int64_t *olen = calloc((size_t)(V > 0 ? V : 1), sizeof(int64_t)); /* overlapped length */
  uint8_t *onr = calloc((size_t)(V > 0 ? V : 1), 1); /* op runs on the rank at hand */
  int32_t G = g->n_groups;
  int32_t *gN = calloc((size_t)(G > 0 ? G : 1), sizeof(int32_t));
  int32_t *gM = calloc((size_t)(G > 0 ? G : 1), sizeof(int32_t));
  int32_t *gK = calloc((size_t)(G > 0 ? G : 1), sizeof(int32_t));
  double *glg = calloc((size_t)(G > 0 ? G : 1), sizeof(double));
  if (!sim.succ_off || !sim.succ_idx || !sim.opq_off || !sim.opq_q || !sim.opq_pos || !sim.cnt ||
      !sim.heap || !fill || !d0 || !d || !st || !fn || !ov || !cst || !cfn || !clo || !chi || !olen || !onr || !gN || !gM ||
      !gK || !glg) {
    rc = ORACLE_E_NOMEM;
    goto out;
  }
  for (int64_t e = 0; e < E; ++e) sim.succ_off[g->pred_idx[e] + 1]++;
  for (int64_t v = 0; v < V; ++v) sim.succ_off[v + 1] += sim.succ_off[v];
  for (int64_t v = 0; v < V; ++v)
    for (int64_t e = g->pred_off[v]; e < g->pred_off[v + 1]; ++e) {
      int32_t u = g->pred_idx[e];
      sim.succ_idx[sim.succ_off[u] + fill[u]++] = (int32_t)v;
    }
  for (int64_t k = 0; k < QE; ++k) sim.opq_off[g->q_ops[k] + 1]++;
  for (int64_t v = 0; v < V; ++v) sim.opq_off[v + 1] += sim.opq_off[v];
  memset(fill, 0, (size_t)(V + 1) * sizeof(int64_t));
  for (int64_t q = 0; q < nq; ++q)
    for (int64_t k = g->q_off[q]; k < g->q_off[q + 1]; ++k) {
      int32_t v = g->q_ops[k];
      int64_t slot = sim.opq_off[v] + fill[v]++;
      sim.opq_q[slot] = (int32_t)q;
      sim.opq_pos[slot] = k - g->q_off[q];
    }
  for (int32_t gi = 0; gi < G; ++gi) {
    int64_t a = g->grp_off[gi], b = g->grp_off[gi + 1];
    int32_t N = (int32_t)(b - a), M = 0, K = 0;
    /* distinct nodes and the largest per-node member count, by direct counting */
    for (int64_t i = a; i < b; ++i) {
      int32_t node = g->grp_rank[i] / g->gpus_per_node;
      int seen = 0, here = 0;
      for (int64_t j = a; j < i; ++j)
        if (g->grp_rank[j] / g->gpus_per_node == node) seen = 1;
      for (int64_t j = a; j < b; ++j)
        if (g->grp_rank[j] / g->gpus_per_node == node) here++;
      if (!seen) M++;
      if (here > K) K = here;
    }
    gN[gi] = N;
    gM[gi] = M;
    gK[gi] = K;
    glg[gi] = log2((double)M);
  }

  for (int32_t s = s0; s < s1; ++s) {
    double prm[6] = {sc->alpha_ns[s], sc->bw_intra[s], sc->lat_intra[s],
                     sc->bw_inter[s], sc->lat_inter[s], sc->delta[s]};
    for (int64_t v = 0; v < V; ++v) {
      uint8_t k = g->kind[v];
      if (k == K_COLL || k == K_P2P) {
        int32_t gi = g->group[v];
        /* an all-reduce policy replaces every all-reduce's own algorithm */
        const int algo = g->cc_type[v] == T_AR && sc->ar_algo_policy > 0 ? sc->ar_algo_policy - 1 : g->cc_algo[v];
        double T = sc->cc_model == 1
                       ? oracle_cc_ns_alpha_beta(g->cc_bytes[v], gN[gi], gM[gi], prm)
                       : oracle_cc_ns(g->cc_type[v], algo, g->cc_bytes[v], gN[gi], gM[gi], gK[gi],
                                      glg[gi], prm, sc->n_chunk, sc->chunk_max_bytes, sc->chunk_bytes);
        if (cc_ns) cc_ns[v * S + s] = T;
        d0[v] = llrint(T);
      } else {
        d0[v] = sc->dur[v * S + s];
      }
      d[v] = d0[v];
    }
    rc = simulate(&sim, d, st, fn);
    if (rc) goto out;
    memset(ov, 0, (size_t)(V > 0 ? V : 1));
    for (int32_t pass = 0; pass < refine_passes; ++pass) {
      /* validator: a compute op of rank r is slowed when its interval overlaps,
       * with positive length, the interval of any comm op that rank r takes part in */
      for (int32_t r = 0; r < g->n_ranks; ++r) {
        int64_t qa = (int64_t)g->n_streams * r, qb = qa + g->n_streams, nc = 0;
        for (int64_t j = g->q_off[qa]; j < g->q_off[qb]; ++j) onr[g->q_ops[j]] = 1;
        for (int64_t q = qa; q < qb; ++q)
          for (int64_t j = g->q_off[q]; j < g->q_off[q + 1]; ++j) {
            int32_t w = g->q_ops[j];
            if (g->kind[w] != K_COLL && g->kind[w] != K_P2P) continue;
            if (sc->comm_interval == 1) {
              /* rank r has launched w once the op before it on this timeline and
               * its data producers that run on r have finished */
              int64_t t = 0;
              if (j > g->q_off[q] && fn[g->q_ops[j - 1]] > t) t = fn[g->q_ops[j - 1]];
              for (int64_t e = g->pred_off[w]; e < g->pred_off[w + 1]; ++e) {
                int32_t u = g->pred_idx[e];
                if (onr[u] && fn[u] > t) t = fn[u];
              }
              cst[nc] = t;
            } else {
              cst[nc] = st[w];
            }
            cfn[nc] = fn[w];
            nc++;
          }
        for (int64_t j = g->q_off[qa]; j < g->q_off[qb]; ++j) onr[g->q_ops[j]] = 0;
        for (int64_t i = g->q_off[qa]; i < g->q_off[qb]; ++i) {
          int32_t v = g->q_ops[i];
          if (g->kind[v] != K_COMPUTE) continue;
          /* the parts of the rank's comm intervals inside the kernel's interval; the
           * kernel is overlapped when they cover a positive length */
          int64_t m = 0;
          for (int64_t j = 0; j < nc; ++j) {
            int64_t lo = st[v] > cst[j] ? st[v] : cst[j];
            int64_t hi = fn[v] < cfn[j] ? fn[v] : cfn[j];
            if (lo < hi) {
              clo[m] = lo;
              chi[m] = hi;
              m++;
            }
          }
          ov[v] = m > 0;
          olen[v] = union_length(clo, chi, m);
        }
      }
      for (int64_t v = 0; v < V; ++v) {
        if (g->kind[v] == K_COMPUTE && ov[v]) {
          double f = sc->slowdown[(int64_t)g->kclass[v] * S + s];
          if (sc->overlap_model == 1) /* the overlapped part of the kernel runs f times longer */
            d[v] = llrint((double)d0[v] + (f - 1.0) * (double)olen[v]);
          else /* the whole kernel does (Sec. 2.3) */
            d[v] = llrint((double)d0[v] * f);
        } else {
          d[v] = d0[v];
        }
      }
      rc = simulate(&sim, d, st, fn);
      if (rc) goto out;
    }
    int64_t mk = 0;
    for (int64_t v = 0; v < V; ++v) {
      if (start) start[v * S + s] = st[v];
      if (finish) finish[v * S + s] = fn[v];
      if (overlapped) overlapped[v * S + s] = ov[v];
      if (fn[v] > mk) mk = fn[v];
    }
    if (makespan) makespan[s] = mk;
  }

out:
  free(sim.succ_off);
  free(sim.succ_idx);
  free(sim.opq_off);
  free(sim.opq_q);
  free(sim.opq_pos);
  free(sim.cnt);
  free(sim.heap);
  free(fill);
  free(d0);
  free(d);
  free(st);
  free(fn);
  free(ov);
  free(cst);
  free(cfn);
  free(clo);
  free(chi);
  free(olen);
  free(onr);
  free(gN);
  free(gM);
  free(gK);
  free(glg);
  return rc;
}
