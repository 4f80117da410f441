// echo_host.cpp -- host side of the C ABI declared in include/echo.h: input
// validation, topological levelling and renumbering, collective-signature dedup,
// device memory, kernel launches and readback.
#include <cuda_runtime.h>

#include <algorithm>
#include <array>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <map>
#include <new>
#include <string>
#include <tuple>
#include <vector>

#include "echo.h"
#include "echo_internal.h"

using echo::CcSig;
using echo::ChunkTable;

namespace {

// Table 6 of the paper (Sec. 8.3): chunk size per tensor size, MB read as MiB.
const int64_t kDefaultMax[5] = {4LL << 20, 8LL << 20, 64LL << 20, 128LL << 20, INT64_MAX};
const int64_t kDefaultChunk[5] = {18000, 36000, 72000, 144000, 288000};

struct Err {
  int code = ECHO_OK;
  std::string msg;
};

int fail(Err &e, int code, const char *fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  e.code = code;
  e.msg = buf;
  return code;
}

// Everything derived from a graph on the host.
struct GraphBuild {
  int64_t V = 0, E = 0, QE = 0, L = 0, max_width = 0;
  int64_t V_ext = 0;  // the caller's ops (more than V when replicas are folded)
  int32_t R = 0, NS = 0, gpn = 1;
  std::vector<int32_t> int2ext, ext2int;
  int64_t Ls = 0, n_seg = 0;           // segment levels, segments
  std::vector<int64_t> seg_lvl_off;    // [Ls+1] segments of each segment level
  std::vector<int64_t> seg_node_off;   // [n_seg+1] nodes of each segment (internal ids)
  std::vector<int32_t> seg_int;        // [V] segment of each internal node
  std::vector<int64_t> nq_off;
  std::vector<int32_t> nq;
  std::vector<int64_t> dp_off;
  std::vector<int32_t> dp;
  std::vector<uint8_t> kcl, is_comm, local;
  std::vector<int64_t> q_off;
  std::vector<int32_t> q_ops_int;
  std::vector<CcSig> sigs;
  std::vector<int32_t> sig_count, comm_node, comm_sig, node_sig;
  std::vector<int64_t> cand_off;      // [R+1] overlap candidates of each rank (compute ops, issue order)
  std::vector<int32_t> cand_ops;      // (internal ids)
  std::vector<uint8_t> cand_flag;     // [V] 1 for an overlap candidate
  int64_t n_cand = 0;                 // overlap candidates
  std::vector<int32_t> cidx;          // [V] level-order index of a candidate (by internal id), -1 otherwise
  std::vector<int32_t> cand_cidx;     // level-order index of each entry of cand_ops
  std::vector<int32_t> cand_node;     // internal id of each candidate, in level order
  std::vector<uint8_t> cand_kcl;      // kernel class of each entry of cand_ops
  std::vector<uint8_t> q_rel;         // [queue entries] 1 for a comm op that can overlap a compute op
                                      // of the entry's rank in some scenario (see overlap_candidates)
  int32_t n_cq = 0;                   // comm timelines per rank in cq_off (max over ranks)
  std::vector<int64_t> cq_off;        // [R*n_cq+1] comm ops of each (rank, comm timeline)
  std::vector<int32_t> cq_ops;        // internal ids, in issue order
  std::vector<int32_t> lq_off;        // [cq_ops+1] launch conditions of each cq_ops entry on its rank
  std::vector<int32_t> lq_ops;        // (internal ids; the latest one on each of the rank's timelines)
  std::vector<int64_t> seg_words;     // [n_seg] record words of each segment
  // [V] 1 for an op whose finish a later step reads besides the next op of its
  // chain: an overlap candidate, a comm op the validator's cursors visit, or one
  // of their launch conditions (a segment's tail is always kept: later heads read it)
  std::vector<uint8_t> keep;
  std::vector<int64_t> hin_off;       // [n_seg+1] inputs of each segment's head
  std::vector<int32_t> hin;           // (internal ids, each the tail of an earlier segment)
  int32_t max_kclass = -1;
  // programs of the dataflow composer (one per rank; see echo_internal.h)
  bool df_ok = false;
  std::vector<int64_t> df_off;
  std::vector<uint32_t> df_rec, df_opnd;
  int64_t df_slots = 0, df_exports = 0;
  int32_t df_wpb = 1;  // warps per block: a block holds df_wpb consecutive ranks (for block joins)
  bool stageable = true;              // every head has < 2^16 inputs
};

bool finite_nonneg(double x) { return std::isfinite(x) && x >= 0.0; }

constexpr int64_t kStepNodes = 2048;     // nodes of one composition step (a level or a part of one)
constexpr int64_t kStepSegments = 1024;  // segments of one composition step

// Compute ops that can overlap a comm op of their rank in some scenario: the only
// ones the validator pass (Sec. 3, 6) tests.  This pruning is a static analysis of
// this library, not a step of the paper; it never changes a result.  A rank's
// compute timeline is a serial chain, so for a comm op w on rank r the compute ops
// of r up to the latest one that reaches w finish before w starts, and those from
// the earliest one that w reaches on start after w ends: only positions in
// between, (anc(w), desc(w)), can intersect w's interval, whatever the durations.
// anc and desc follow the edges among rank r's own ops (data edges and the order
// of r's timelines); paths through other ranks are ignored, which only widens the
// ranges.  Needs the internal numbering (a topological order), q_off/q_ops_int
// and dp.
void overlap_candidates(GraphBuild &b) {
  const int64_t V = b.V;
  const int32_t R = b.R, NS = b.NS;
  std::vector<int64_t> su_off(V + 1, 0);  // data successors
  for (int64_t q = 0; q < b.dp_off[V]; ++q) su_off[b.dp[q] + 1]++;
  for (int64_t v = 0; v < V; ++v) su_off[v + 1] += su_off[v];
  std::vector<int32_t> su(std::max<int64_t>(su_off[V], 1));
  {
    std::vector<int64_t> fill(su_off.begin(), su_off.end() - 1);
    for (int64_t v = 0; v < V; ++v)
      for (int64_t q = b.dp_off[v]; q < b.dp_off[v + 1]; ++q) su[fill[b.dp[q]]++] = (int32_t)v;
  }
  std::vector<int32_t> loc(V, -1);
  b.cand_off.assign(R + 1, 0);
  b.cand_ops.clear();
  b.cand_flag.assign(V, 0);
  b.cand_kcl.clear();
  b.q_rel.assign(std::max<int64_t>(b.q_off[(int64_t)R * NS], 1), 0);
  std::vector<int32_t> nodes, cpos, prv, nxt, anc, desc;
  std::vector<int64_t> cover;
  for (int32_t r = 0; r < R; ++r) {
    nodes.clear();
    for (int32_t k = 0; k < NS; ++k)
      for (int64_t i = b.q_off[(int64_t)r * NS + k]; i < b.q_off[(int64_t)r * NS + k + 1]; ++i)
        nodes.push_back(b.q_ops_int[i]);
    std::sort(nodes.begin(), nodes.end());  // a topological order
    const int64_t m = (int64_t)nodes.size();
    for (int64_t j = 0; j < m; ++j) loc[nodes[j]] = (int32_t)j;
    const int64_t c0 = b.q_off[(int64_t)r * NS], n = b.q_off[(int64_t)r * NS + 1] - c0;
    cpos.assign(m, -1);
    prv.assign(m, -1);
    nxt.assign(m, -1);
    for (int64_t i = c0; i < c0 + n; ++i) cpos[loc[b.q_ops_int[i]]] = (int32_t)(i - c0);
    for (int32_t k = 0; k < NS; ++k)
      for (int64_t i = b.q_off[(int64_t)r * NS + k] + 1; i < b.q_off[(int64_t)r * NS + k + 1]; ++i) {
        prv[loc[b.q_ops_int[i]]] = loc[b.q_ops_int[i - 1]];
        nxt[loc[b.q_ops_int[i - 1]]] = loc[b.q_ops_int[i]];
      }
    anc.assign(m, -1);
    for (int64_t j = 0; j < m; ++j) {  // latest compute position of r reaching the op
      int32_t x = cpos[j];
      if (prv[j] >= 0) x = std::max(x, anc[prv[j]]);
      for (int64_t q = b.dp_off[nodes[j]]; q < b.dp_off[nodes[j] + 1]; ++q)
        if (loc[b.dp[q]] >= 0) x = std::max(x, anc[loc[b.dp[q]]]);
      anc[j] = x;
    }
    desc.assign(m, (int32_t)n);
    for (int64_t j = m - 1; j >= 0; --j) {  // earliest compute position of r the op reaches
      int32_t x = cpos[j] >= 0 ? cpos[j] : (int32_t)n;
      if (nxt[j] >= 0) x = std::min(x, desc[nxt[j]]);
      for (int64_t q = su_off[nodes[j]]; q < su_off[nodes[j] + 1]; ++q)
        if (loc[su[q]] >= 0) x = std::min(x, desc[loc[su[q]]]);
      desc[j] = x;
    }
    cover.assign(n + 1, 0);
    for (int64_t j = 0; j < m; ++j)
      if (b.is_comm[nodes[j]] && anc[j] + 1 < desc[j]) {
        cover[anc[j] + 1]++;
        cover[desc[j]]--;
      }
    // the comm ops the validator's cursors visit on this rank: only those whose
    // range holds a compute position (a tensor-parallel all-reduce between its
    // producer and its consumer never overlaps a compute op of the rank, so its
    // interval can be skipped without changing any decision or covered length)
    for (int32_t k = 1; k < NS; ++k)
      for (int64_t i = b.q_off[(int64_t)r * NS + k]; i < b.q_off[(int64_t)r * NS + k + 1]; ++i) {
        const int32_t w = b.q_ops_int[i];
        b.q_rel[i] = b.is_comm[w] && anc[loc[w]] + 1 < desc[loc[w]];
      }
    int64_t run = 0;
    for (int64_t p = 0; p < n; ++p) {
      run += cover[p];
      if (run > 0) {
        const int32_t v = b.q_ops_int[c0 + p];
        b.cand_ops.push_back(v);
        b.cand_kcl.push_back(b.kcl[v]);
        b.cand_flag[v] = 1;
      }
    }
    b.cand_off[r + 1] = (int64_t)b.cand_ops.size();
    for (int64_t j = 0; j < m; ++j) loc[nodes[j]] = -1;
  }
  // level order of the candidates (by internal id): each segment level's candidates
  // are then one contiguous range, and so are each segment's
  b.n_cand = b.cand_off[R];
  b.cidx.assign(V, -1);
  b.cand_node.clear();
  for (int64_t v = 0; v < V; ++v)
    if (b.cand_flag[v]) {
      b.cidx[v] = (int32_t)b.cand_node.size();
      b.cand_node.push_back((int32_t)v);
    }
  if (b.cand_node.empty()) b.cand_node.push_back(0);
  b.cand_cidx.resize(b.cand_ops.size());
  for (size_t k = 0; k < b.cand_ops.size(); ++k) b.cand_cidx[k] = b.n_cand ? b.cidx[b.cand_ops[k]] : 0;
  if (b.cand_ops.empty()) b.cand_ops.push_back(0);
  if (b.cand_kcl.empty()) b.cand_kcl.push_back(0);
  if (b.cand_cidx.empty()) b.cand_cidx.push_back(0);
}


// The dataflow composer's programs: every rank's ops in internal order with their
// inputs on the rank (the latest op of one of its timelines: shared memory; an
// earlier op of the rank: its stored finish), the inputs produced by other warps
// (export flags) and, for comm ops, the partial slots of their members.  A comm
// op's data producers run on its members, each member taking its own; one that
// runs on no member is taken by the first member.
void build_dataflow(GraphBuild &b) {
  const int64_t V = b.V;
  const int32_t R = b.R, NS = b.NS;
  b.df_ok = false;
  b.df_off.assign(R + 1, 0);
  b.df_rec.clear();
  b.df_opnd.clear();
  if (V >= (int64_t)(echo::kDfPayload + 1u)) return;
  // ranks of each op, ascending, with the op's timeline on each
  std::vector<int64_t> ro_off(V + 1, 0);
  for (int64_t q = 0; q < (int64_t)R * NS; ++q)
    for (int64_t i = b.q_off[q]; i < b.q_off[q + 1]; ++i) ro_off[b.q_ops_int[i] + 1]++;
  for (int64_t v = 0; v < V; ++v) ro_off[v + 1] += ro_off[v];
  std::vector<int32_t> ro(std::max<int64_t>(ro_off[V], 1));
  std::vector<int8_t> rt(ro.size());
  {
    std::vector<int64_t> fill(ro_off.begin(), ro_off.end() - 1);
    for (int64_t q = 0; q < (int64_t)R * NS; ++q)
      for (int64_t i = b.q_off[q]; i < b.q_off[q + 1]; ++i) {
        const int64_t at = fill[b.q_ops_int[i]]++;
        ro[at] = (int32_t)(q / NS);
        rt[at] = (int8_t)(q % NS);
      }
  }
  auto runs_on = [&](int32_t u, int32_t r) {
    return std::binary_search(ro.data() + ro_off[u], ro.data() + ro_off[u + 1], r);
  };
  auto members = [&](int32_t v) { return ro_off[v + 1] - ro_off[v]; };
  // Block joins: a comm op whose members are exactly the ranks of one block of
  // df_wpb consecutive ranks (aligned) joins through shared memory.  The width is the
  // one (dividing R, at most 8) whose blocks hold the most comm ops.
  auto aligned_group = [&](int64_t v, int32_t w) {
    if (members((int32_t)v) != w) return false;
    const int32_t r0 = ro[ro_off[v]];
    return r0 % w == 0 && ro[ro_off[v] + w - 1] == r0 + w - 1;
  };
  b.df_wpb = 1;
  {
    int64_t best = 0;
    for (int32_t w = 2; w <= 8; w *= 2) {
      if (R % w) continue;
      int64_t n = 0;
      for (int64_t v = 0; v < V; ++v) n += b.is_comm[v] && aligned_group(v, w);
      if (n > best) {
        best = n;
        b.df_wpb = w;
      }
    }
  }
  // partial slots (block joins take a per-block sequence number instead), and the
  // producers of each comm op that run on none of its members
  std::vector<int64_t> slot(V, 0);
  std::vector<uint8_t> uncovered(std::max<int64_t>(b.dp_off[V], 1), 0);
  std::vector<uint32_t> bseq(R / b.df_wpb, 0);
  b.df_slots = 0;
  for (int64_t v = 0; v < V; ++v) {
    if (!b.is_comm[v]) continue;
    if (b.df_wpb > 1 && aligned_group(v, b.df_wpb)) {
      slot[v] = echo::kDfBlockJoin | bseq[ro[ro_off[v]] / b.df_wpb]++;
    } else if (members((int32_t)v) > 1) {
      slot[v] = b.df_slots;
      b.df_slots += members((int32_t)v);
    }
    for (int64_t e = b.dp_off[v]; e < b.dp_off[v + 1]; ++e) {
      const int32_t u = b.dp[e];
      bool cov = false;
      for (int64_t k = ro_off[u]; k < ro_off[u + 1] && !cov; ++k) cov = runs_on((int32_t)v, ro[k]);
      uncovered[e] = !cov;
    }
  }
  // exports: ops another warp waits for
  std::vector<int64_t> exp_id(V, -1);
  b.df_exports = 0;
  auto export_op = [&](int32_t u) {
    if (exp_id[u] < 0) exp_id[u] = b.df_exports++;
  };
  for (int64_t v = 0; v < V; ++v) {
    if (b.is_comm[v] && members((int32_t)v) > (int64_t)echo::kDfDirectMembers) export_op((int32_t)v);
    for (int64_t e = b.dp_off[v]; e < b.dp_off[v + 1]; ++e) {
      const int32_t u = b.dp[e];
      if (b.is_comm[v] ? uncovered[e] != 0 : !runs_on(u, ro[ro_off[v]])) export_op(u);
    }
  }
  if (b.df_exports >= (int64_t)(echo::kDfPayload + 1u)) return;
  // the programs, written in one pass over the ops in internal order (each rank's
  // entries land in its own range, in that order); per rank only the latest op of
  // each timeline and the previous op are kept
  for (int32_t r = 0; r < R; ++r) b.df_off[r + 1] = b.df_off[r] + (b.q_off[(int64_t)(r + 1) * NS] - b.q_off[(int64_t)r * NS]);
  b.df_rec.assign((size_t)b.df_off[R] * 8, 0u);
  std::vector<int64_t> cnt(R, 0);
  std::vector<int32_t> last((size_t)R * NS, -1), prev(R, -1);
  std::vector<int8_t> prev_tl(R, 0);
  std::vector<uint32_t> extra;
  auto timeline_on = [&](int32_t u, int32_t r) -> int {  // u's timeline on rank r, -1 if none
    const int32_t *lo = ro.data() + ro_off[u], *hi = ro.data() + ro_off[u + 1];
    const int32_t *p = std::lower_bound(lo, hi, r);
    return p != hi && *p == r ? rt[p - ro.data()] : -1;
  };
  for (int64_t v = 0; v < V; ++v) {
    const bool comm = b.is_comm[v];
    const int64_t nm = members((int32_t)v);
    for (int64_t j = ro_off[v]; j < ro_off[v + 1]; ++j) {
      const int32_t r = ro[j], k = rt[j];
      const int64_t me = j - ro_off[v];
      int32_t *lr = last.data() + (size_t)r * NS;
      extra.clear();
      uint32_t regs = lr[k] >= 0 ? 1u << k : 0u;  // the op before it on its timeline
      for (int64_t e = b.dp_off[v]; e < b.dp_off[v + 1]; ++e) {
        const int32_t u = b.dp[e];
        const int ku = timeline_on(u, r);
        if (ku >= 0) {  // runs on this rank
          if (lr[ku] == u)
            regs |= 1u << ku;
          else
            extra.push_back((echo::kDfInLocal << 30) | (uint32_t)u);
        } else if (comm ? (uncovered[e] && me == 0) : true) {
          extra.push_back((echo::kDfInRemote << 30) | (uint32_t)exp_id[u]);
        }
      }
      // the previous op of the program, when an input, comes from a register
      bool use_prev = false;
      if (prev[r] >= 0 && ((regs >> prev_tl[r]) & 1) && lr[prev_tl[r]] == prev[r]) {
        use_prev = true;
        regs &= ~(1u << prev_tl[r]);
      }
      const bool two_hop = comm && nm > (int64_t)echo::kDfDirectMembers;
      const bool publish = exp_id[v] >= 0 && (!comm || me == 0);
      if (extra.size() > 0xFF || nm > 0xFFFF || b.df_opnd.size() + extra.size() >= (size_t)UINT32_MAX) return;
      const uint32_t hdr = (uint32_t)k | (comm ? echo::kDfComm : 0u) | (publish ? echo::kDfExport : 0u) |
                           (two_hop ? echo::kDfTwoHop : 0u) | (use_prev ? echo::kDfPrev : 0u) |
                           ((uint32_t)extra.size() << 8) | (regs << 16);
      uint32_t *w = b.df_rec.data() + (size_t)(b.df_off[r] + cnt[r]++) * 8;
      w[0] = (uint32_t)v;
      w[1] = b.cidx[v] >= 0 ? (uint32_t)b.cidx[v] : ~0u;
      w[2] = hdr;
      w[3] = (uint32_t)b.df_opnd.size();
      w[4] = comm ? (uint32_t)slot[v] : 0u;  // (kDfBlockJoin | sequence number for a block join)
      w[5] = comm ? (uint32_t)nm | ((uint32_t)me << 16) : 0u;
      w[6] = publish || two_hop ? (uint32_t)exp_id[v] : 0u;
      w[7] = 0u;
      b.df_opnd.insert(b.df_opnd.end(), extra.begin(), extra.end());
      lr[k] = (int32_t)v;
      prev[r] = (int32_t)v;
      prev_tl[r] = (int8_t)k;
    }
  }
  if (b.df_slots >= (int64_t)echo::kDfBlockJoin) return;
  for (uint32_t n : bseq)
    if (n >= echo::kDfBlockJoin) return;
  if (b.df_rec.empty()) b.df_rec.assign(8, 0);
  if (b.df_opnd.empty()) b.df_opnd.push_back(0);
  b.df_ok = true;
}

// `shape`, when given, replaces the (N, M, K) of every group computed from its
// members (a folded graph keeps the shapes of the caller's groups).  `programs`:
// also build the dataflow composer's programs (not needed to validate a graph).
using Shape = std::array<int32_t, 3>;
int build_graph(const echo_graph_desc *g, GraphBuild &b, Err &e, const std::vector<Shape> *shape = nullptr,
                bool programs = true) {
  if (!g) return fail(e, ECHO_E_INVALID_ARG, "graph descriptor is NULL");
  const int64_t V = g->n_ops;
  if (V < 0 || V >= INT32_MAX) return fail(e, ECHO_E_INVALID_ARG, "n_ops %lld out of range", (long long)V);
  if (g->n_ranks < 1 || g->n_ranks > 65535)
    return fail(e, ECHO_E_UNSUPPORTED, "n_ranks %d outside [1, 65535]", g->n_ranks);
  if (g->n_streams < 1 || g->n_streams > echo::kMaxStreams)
    return fail(e, ECHO_E_UNSUPPORTED, "n_streams %d outside [1, %d]", g->n_streams, echo::kMaxStreams);
  if (g->gpus_per_node < 1) return fail(e, ECHO_E_INVALID_ARG, "gpus_per_node must be >= 1");
  if (g->n_groups < 0) return fail(e, ECHO_E_INVALID_ARG, "n_groups must be >= 0");
  const int32_t R = g->n_ranks, NS = g->n_streams;
  const int64_t NQ = (int64_t)R * NS;
  if (!g->pred_off || !g->q_off) return fail(e, ECHO_E_INVALID_ARG, "pred_off and q_off are required");
  if (V > 0 && (!g->kind || !g->kclass || !g->group || !g->cc_type || !g->cc_algo || !g->cc_bytes))
    return fail(e, ECHO_E_INVALID_ARG, "per-op arrays are required when n_ops > 0");
  if (g->n_groups > 0 && (!g->grp_off || !g->grp_rank))
    return fail(e, ECHO_E_INVALID_ARG, "grp_off/grp_rank are required when n_groups > 0");

  // data dependencies
  if (g->pred_off[0] != 0) return fail(e, ECHO_E_BAD_GRAPH, "pred_off[0] must be 0");
  for (int64_t v = 0; v < V; ++v)
    if (g->pred_off[v + 1] < g->pred_off[v]) return fail(e, ECHO_E_BAD_GRAPH, "pred_off decreases at op %lld", (long long)v);
  const int64_t E = g->pred_off[V];
  if (E > 0 && !g->pred_idx) return fail(e, ECHO_E_INVALID_ARG, "pred_idx is NULL");
  if (E >= INT32_MAX) return fail(e, ECHO_E_UNSUPPORTED, "too many edges");
  for (int64_t v = 0; v < V; ++v)
    for (int64_t k = g->pred_off[v]; k < g->pred_off[v + 1]; ++k) {
      int32_t u = g->pred_idx[k];
      if (u < 0 || u >= V) return fail(e, ECHO_E_BAD_GRAPH, "op %lld: predecessor %d out of range", (long long)v, u);
      if (u == v) return fail(e, ECHO_E_CYCLE, "op %lld depends on itself", (long long)v);
    }
  // groups
  std::vector<std::vector<int32_t>> members(g->n_groups);
  if (g->n_groups > 0) {
    if (g->grp_off[0] != 0) return fail(e, ECHO_E_BAD_GRAPH, "grp_off[0] must be 0");
    for (int32_t gi = 0; gi < g->n_groups; ++gi) {
      if (g->grp_off[gi + 1] < g->grp_off[gi]) return fail(e, ECHO_E_BAD_GRAPH, "grp_off decreases at group %d", gi);
      for (int64_t k = g->grp_off[gi]; k < g->grp_off[gi + 1]; ++k) {
        int32_t r = g->grp_rank[k];
        if (r < 0 || r >= R) return fail(e, ECHO_E_BAD_GRAPH, "group %d: rank %d out of range", gi, r);
        members[gi].push_back(r);
      }
      std::sort(members[gi].begin(), members[gi].end());
      if (std::adjacent_find(members[gi].begin(), members[gi].end()) != members[gi].end())
        return fail(e, ECHO_E_BAD_GRAPH, "group %d repeats a rank", gi);
      if (members[gi].empty()) return fail(e, ECHO_E_BAD_GRAPH, "group %d is empty", gi);
    }
  }
  // ops
  int32_t max_kc = -1;
  for (int64_t v = 0; v < V; ++v) {
    uint8_t k = g->kind[v];
    if (k > ECHO_OP_P2P) return fail(e, ECHO_E_BAD_GRAPH, "op %lld: kind %d", (long long)v, k);
    if (k == ECHO_OP_COMPUTE) {
      if (g->kclass[v] == echo::kNotSlowable) return fail(e, ECHO_E_BAD_GRAPH, "op %lld: kclass 255 is reserved", (long long)v);
      max_kc = std::max<int32_t>(max_kc, g->kclass[v]);
    }
    if (k == ECHO_OP_COLL || k == ECHO_OP_P2P) {
      int32_t gi = g->group[v];
      if (gi < 0 || gi >= g->n_groups) return fail(e, ECHO_E_BAD_GRAPH, "op %lld: group %d out of range", (long long)v, gi);
      if (g->cc_bytes[v] < 0) return fail(e, ECHO_E_INVALID_ARG, "op %lld: negative message size", (long long)v);
      uint8_t t = g->cc_type[v];
      if (k == ECHO_OP_P2P) {
        if (t != ECHO_CC_SENDRECV) return fail(e, ECHO_E_BAD_GRAPH, "op %lld: P2P op needs cc_type SENDRECV", (long long)v);
        if (members[gi].size() > 2) return fail(e, ECHO_E_BAD_GRAPH, "op %lld: P2P group has more than 2 ranks", (long long)v);
      } else {
        if (t > ECHO_CC_REDUCESCATTER) return fail(e, ECHO_E_BAD_GRAPH, "op %lld: collective cc_type %d", (long long)v, t);
        if (t == ECHO_CC_ALLREDUCE && g->cc_algo[v] > ECHO_ALGO_AUTO)
          return fail(e, ECHO_E_BAD_GRAPH, "op %lld: cc_algo %d", (long long)v, g->cc_algo[v]);
      }
    }
  }
  // timelines
  if (g->q_off[0] != 0) return fail(e, ECHO_E_BAD_GRAPH, "q_off[0] must be 0");
  for (int64_t q = 0; q < NQ; ++q)
    if (g->q_off[q + 1] < g->q_off[q]) return fail(e, ECHO_E_BAD_GRAPH, "q_off decreases at timeline %lld", (long long)q);
  const int64_t QE = g->q_off[NQ];
  if (QE > 0 && !g->q_ops) return fail(e, ECHO_E_INVALID_ARG, "q_ops is NULL");
  if (QE >= INT32_MAX) return fail(e, ECHO_E_UNSUPPORTED, "too many timeline entries");
  std::vector<int32_t> cnt(V, 0);
  std::vector<int64_t> comm_keys;
  for (int64_t q = 0; q < NQ; ++q) {
    int32_t r = (int32_t)(q / NS), k = (int32_t)(q % NS);
    for (int64_t i = g->q_off[q]; i < g->q_off[q + 1]; ++i) {
      int32_t v = g->q_ops[i];
      if (v < 0 || v >= V) return fail(e, ECHO_E_BAD_GRAPH, "timeline (%d,%d): op %d out of range", r, k, v);
      uint8_t kd = g->kind[v];
      if ((k == 0) != (kd == ECHO_OP_COMPUTE))
        return fail(e, ECHO_E_BAD_GRAPH, "op %d of kind %d on stream %d of rank %d (stream 0 holds exactly the compute ops)", v, kd, k, r);
      cnt[v]++;
      if (kd == ECHO_OP_COLL || kd == ECHO_OP_P2P) {
        const auto &m = members[g->group[v]];
        if (!std::binary_search(m.begin(), m.end(), r))
          return fail(e, ECHO_E_BAD_GRAPH, "comm op %d on rank %d, which is not in its group", v, r);
        comm_keys.push_back((int64_t)v * R + r);
      }
    }
  }
  std::sort(comm_keys.begin(), comm_keys.end());
  if (std::adjacent_find(comm_keys.begin(), comm_keys.end()) != comm_keys.end())
    return fail(e, ECHO_E_BAD_GRAPH, "a comm op is issued twice on one rank");
  for (int64_t v = 0; v < V; ++v) {
    uint8_t kd = g->kind[v];
    int64_t want = (kd == ECHO_OP_COLL || kd == ECHO_OP_P2P) ? (int64_t)members[g->group[v]].size() : 1;
    if (cnt[v] != want)
      return fail(e, ECHO_E_BAD_GRAPH, "op %lld appears on %d timelines, expected %lld", (long long)v, cnt[v], (long long)want);
  }

  // Kahn levelling over data + issue-order dependencies; level = ASAP depth
  std::vector<int64_t> succ_off(V + 1, 0);
  for (int64_t k = 0; k < E; ++k) succ_off[g->pred_idx[k] + 1]++;
  for (int64_t v = 0; v < V; ++v) succ_off[v + 1] += succ_off[v];
  std::vector<int32_t> succ(E > 0 ? E : 1);
  {
    std::vector<int64_t> fill(succ_off.begin(), succ_off.end() - 1);
    for (int64_t v = 0; v < V; ++v)
      for (int64_t k = g->pred_off[v]; k < g->pred_off[v + 1]; ++k) succ[fill[g->pred_idx[k]]++] = (int32_t)v;
  }
  // next op on each timeline of an op: (op, next) pairs
  std::vector<int64_t> nx_off(V + 1, 0);
  std::vector<int32_t> indeg(V, 0);
  for (int64_t v = 0; v < V; ++v) indeg[v] = (int32_t)(g->pred_off[v + 1] - g->pred_off[v]);
  for (int64_t q = 0; q < NQ; ++q)
    for (int64_t i = g->q_off[q]; i + 1 < g->q_off[q + 1]; ++i) {
      nx_off[g->q_ops[i] + 1]++;
      indeg[g->q_ops[i + 1]]++;
    }
  for (int64_t v = 0; v < V; ++v) nx_off[v + 1] += nx_off[v];
  std::vector<int32_t> nx(nx_off[V] > 0 ? nx_off[V] : 1);
  {
    std::vector<int64_t> fill(nx_off.begin(), nx_off.end() - 1);
    for (int64_t q = 0; q < NQ; ++q)
      for (int64_t i = g->q_off[q]; i + 1 < g->q_off[q + 1]; ++i) nx[fill[g->q_ops[i]]++] = g->q_ops[i + 1];
  }
  std::vector<int32_t> level(V, 0), order;
  order.reserve(V);
  for (int64_t v = 0; v < V; ++v)
    if (indeg[v] == 0) order.push_back((int32_t)v);
  for (size_t h = 0; h < order.size(); ++h) {
    int32_t u = order[h];
    auto relax = [&](int32_t w) {
      level[w] = std::max(level[w], level[u] + 1);
      if (--indeg[w] == 0) order.push_back(w);
    };
    for (int64_t k = succ_off[u]; k < succ_off[u + 1]; ++k) relax(succ[k]);
    for (int64_t k = nx_off[u]; k < nx_off[u + 1]; ++k) relax(nx[k]);
  }
  if ((int64_t)order.size() != V)
    return fail(e, ECHO_E_CYCLE, "the dependencies form a cycle (%lld of %lld ops orderable)", (long long)order.size(), (long long)V);

  int64_t L = 0;
  for (int64_t v = 0; v < V; ++v) L = std::max<int64_t>(L, level[v] + 1);
  b.V = V;
  b.V_ext = V;
  b.E = E;
  b.QE = QE;
  b.L = L;
  b.R = R;
  b.NS = NS;
  b.gpn = g->gpus_per_node;
  b.max_kclass = max_kc;
  b.max_width = 0;
  {
    std::vector<int64_t> w(L, 0);
    for (int64_t v = 0; v < V; ++v) w[level[v]]++;
    for (int64_t l = 0; l < L; ++l) b.max_width = std::max(b.max_width, w[l]);
  }
  // Chain contraction.  v continues the segment of its predecessor u when u is v's
  // only distinct input and v is u's only distinct consumer.  Along a segment the
  // finish times are running sums of the durations, so only a segment's head reads
  // other ops (timeline frontiers, data predecessors) and only its tail is read by
  // other ops or advances a timeline.
  std::vector<int64_t> mp_off(V + 1, 0);
  std::vector<int32_t> mp;  // distinct predecessors over data and issue-order edges
  {
    std::vector<int64_t> cnt(V + 1, 0);
    for (int64_t v = 0; v < V; ++v) cnt[v + 1] = g->pred_off[v + 1] - g->pred_off[v];
    for (int64_t q = 0; q < NQ; ++q)
      for (int64_t i = g->q_off[q] + 1; i < g->q_off[q + 1]; ++i) cnt[g->q_ops[i] + 1]++;
    for (int64_t v = 0; v < V; ++v) cnt[v + 1] += cnt[v];
    std::vector<int32_t> tmp(cnt[V] > 0 ? cnt[V] : 1);
    std::vector<int64_t> fill(cnt.begin(), cnt.end() - 1);
    for (int64_t v = 0; v < V; ++v)
      for (int64_t k = g->pred_off[v]; k < g->pred_off[v + 1]; ++k) tmp[fill[v]++] = g->pred_idx[k];
    for (int64_t q = 0; q < NQ; ++q)
      for (int64_t i = g->q_off[q] + 1; i < g->q_off[q + 1]; ++i) tmp[fill[g->q_ops[i]]++] = g->q_ops[i - 1];
    mp.reserve(cnt[V]);
    for (int64_t v = 0; v < V; ++v) {
      std::sort(tmp.begin() + cnt[v], tmp.begin() + cnt[v + 1]);
      int32_t prev = -1;
      for (int64_t k = cnt[v]; k < cnt[v + 1]; ++k)
        if (tmp[k] != prev) {
          mp.push_back(tmp[k]);
          prev = tmp[k];
        }
      mp_off[v + 1] = (int64_t)mp.size();
    }
  }
  std::vector<int32_t> out_cnt(V, 0);
  for (int32_t u : mp) out_cnt[u]++;
  std::vector<int32_t> seg_of(V, -1), nxt(V, -1);
  std::vector<int32_t> seg_len, seg_head, seg_tail;  // by creation order
  for (int32_t v : order) {  // topological order
    if (mp_off[v + 1] - mp_off[v] == 1) {
      const int32_t u = mp[mp_off[v]];
      const int32_t su = seg_of[u];
      if (out_cnt[u] == 1 && seg_tail[su] == u && seg_len[su] < echo::kMaxSegment) {
        seg_of[v] = su;
        seg_len[su]++;
        seg_tail[su] = v;
        nxt[u] = v;
        continue;
      }
    }
    seg_of[v] = (int32_t)seg_len.size();
    seg_len.push_back(1);
    seg_head.push_back(v);
    seg_tail.push_back(v);
  }
  const int64_t NSg = (int64_t)seg_len.size();
  // segment levels: ASAP depth of the contracted graph (only heads have inputs)
  std::vector<int32_t> seg_lvl(NSg, 0);
  for (int32_t v : order) {
    const int32_t sv = seg_of[v];
    if (seg_head[sv] != v) continue;
    int32_t lv = 0;
    for (int64_t k = mp_off[v]; k < mp_off[v + 1]; ++k) lv = std::max(lv, seg_lvl[seg_of[mp[k]]] + 1);
    seg_lvl[sv] = lv;
  }
  int64_t Ls = 0;
  for (int64_t t = 0; t < NSg; ++t) Ls = std::max<int64_t>(Ls, seg_lvl[t] + 1);
  b.Ls = Ls;
  b.n_seg = NSg;
  b.seg_lvl_off.assign(Ls + 1, 0);
  for (int64_t t = 0; t < NSg; ++t) b.seg_lvl_off[seg_lvl[t] + 1]++;
  for (int64_t l = 0; l < Ls; ++l) b.seg_lvl_off[l + 1] += b.seg_lvl_off[l];
  std::vector<int32_t> seg_order(NSg);  // internal segment id -> creation id
  {
    std::vector<int64_t> cur(b.seg_lvl_off.begin(), b.seg_lvl_off.end() - 1);
    for (int64_t t = 0; t < NSg; ++t) seg_order[cur[seg_lvl[t]]++] = (int32_t)t;
    // within a level the heaviest segments first (inputs and tail timelines weigh
    // twice a chain step), so that a warp's lanes hold segments of similar weight
    std::vector<int32_t> ntl(V, 0);
    for (int64_t i = 0; i < QE; ++i) ntl[g->q_ops[i]]++;
    std::vector<int64_t> cost(NSg);
    for (int64_t t = 0; t < NSg; ++t) {
      const int32_t h = seg_head[t], z = seg_tail[t];
      cost[t] = 2 * (ntl[h] + (g->pred_off[h + 1] - g->pred_off[h]) + ntl[z]) + seg_len[t];
    }
    for (int64_t l = 0; l < Ls; ++l)
      std::stable_sort(seg_order.begin() + b.seg_lvl_off[l], seg_order.begin() + b.seg_lvl_off[l + 1],
                       [&](int32_t x, int32_t y) { return cost[x] > cost[y]; });
  }
  // internal numbering: segment levels in order, each segment's chain contiguous
  b.seg_node_off.assign(NSg + 1, 0);
  b.seg_int.assign(V, 0);
  b.int2ext.assign(V, 0);
  b.ext2int.assign(V, 0);
  {
    int64_t i = 0;
    for (int64_t t = 0; t < NSg; ++t) {
      b.seg_node_off[t] = i;
      for (int32_t v = seg_head[seg_order[t]]; v >= 0; v = nxt[v]) {
        b.int2ext[i] = v;
        b.ext2int[v] = (int32_t)i;
        b.seg_int[i] = (int32_t)t;
        ++i;
      }
    }
    b.seg_node_off[NSg] = i;
  }
  // Inputs of every segment head: its distinct predecessors over data and issue
  // order (each the tail of an earlier segment, as a chain only continues through
  // an op's single consumer), less any that is itself a direct predecessor of
  // another input: that one finishes no earlier, so the maximum is unchanged.
  b.hin_off.assign(NSg + 1, 0);
  b.hin.clear();
  for (int64_t t = 0; t < NSg; ++t) {
    const int32_t v = b.int2ext[b.seg_node_off[t]];
    const int32_t *p0 = mp.data() + mp_off[v], *p1 = mp.data() + mp_off[v + 1];
    for (const int32_t *pu = p0; pu < p1; ++pu) {
      bool dominated = false;
      for (const int32_t *pw = p0; pw < p1 && !dominated; ++pw)
        if (pw != pu) dominated = std::binary_search(mp.data() + mp_off[*pw], mp.data() + mp_off[*pw + 1], *pu);
      if (!dominated) b.hin.push_back(b.ext2int[*pu]);
    }
    b.hin_off[t + 1] = (int64_t)b.hin.size();
  }
  // timelines of every internal node
  b.nq_off.assign(V + 1, 0);
  for (int64_t i = 0; i < QE; ++i) b.nq_off[b.ext2int[g->q_ops[i]] + 1]++;
  for (int64_t v = 0; v < V; ++v) b.nq_off[v + 1] += b.nq_off[v];
  b.nq.assign(QE > 0 ? QE : 1, 0);
  b.q_off.assign(g->q_off, g->q_off + NQ + 1);
  b.q_ops_int.assign(QE > 0 ? QE : 1, 0);
  {
    std::vector<int64_t> fill(b.nq_off.begin(), b.nq_off.end() - 1);
    for (int64_t q = 0; q < NQ; ++q)
      for (int64_t i = g->q_off[q]; i < g->q_off[q + 1]; ++i) {
        int32_t in = b.ext2int[g->q_ops[i]];
        b.nq[fill[in]++] = (int32_t)q;
        b.q_ops_int[i] = in;
      }
  }
  // data predecessors in internal ids
  b.dp_off.assign(V + 1, 0);
  b.dp.assign(E > 0 ? E : 1, 0);
  for (int64_t i = 0; i < V; ++i) {
    int32_t v = b.int2ext[i];
    int64_t n = g->pred_off[v + 1] - g->pred_off[v];
    b.dp_off[i + 1] = b.dp_off[i] + n;
    for (int64_t k = 0; k < n; ++k) b.dp[b.dp_off[i] + k] = b.ext2int[g->pred_idx[g->pred_off[v] + k]];
  }
  b.kcl.assign(V, echo::kNotSlowable);
  b.is_comm.assign(V, 0);
  b.local.assign(V, 0);
  b.node_sig.assign(V, -1);
  // group shape: N members, M distinct nodes, K largest per-node count, log2(M)
  std::vector<int32_t> gN(g->n_groups), gM(g->n_groups), gK(g->n_groups);
  for (int32_t gi = 0; gi < g->n_groups; ++gi) {
    std::map<int32_t, int32_t> per_node;
    for (int32_t r : members[gi]) per_node[r / g->gpus_per_node]++;
    int32_t K = 0;
    for (auto &kv : per_node) K = std::max(K, kv.second);
    gN[gi] = (int32_t)members[gi].size();
    gM[gi] = (int32_t)per_node.size();
    gK[gi] = K;
    if (shape) {
      gN[gi] = (*shape)[gi][0];
      gM[gi] = (*shape)[gi][1];
      gK[gi] = (*shape)[gi][2];
    }
  }
  std::map<std::tuple<int32_t, int32_t, int64_t, int32_t, int32_t, int32_t>, int32_t> sig_of;
  for (int64_t i = 0; i < V; ++i) {
    int32_t v = b.int2ext[i];
    uint8_t kd = g->kind[v];
    if (kd == ECHO_OP_COMPUTE) b.kcl[i] = g->kclass[v];
    if (kd == ECHO_OP_COMPUTE || kd == ECHO_OP_MEMCPY) b.local[i] = 1;
    if (kd == ECHO_OP_COLL || kd == ECHO_OP_P2P) {
      b.is_comm[i] = 1;
      int32_t gi = g->group[v];
      int32_t t = g->cc_type[v];
      int32_t a = (t == ECHO_CC_ALLREDUCE) ? g->cc_algo[v] : ECHO_ALGO_RING;
      auto key = std::make_tuple(t, a, g->cc_bytes[v], gN[gi], gM[gi], gK[gi]);
      auto it = sig_of.find(key);
      int32_t s;
      if (it == sig_of.end()) {
        s = (int32_t)b.sigs.size();
        sig_of.emplace(key, s);
        CcSig cs;
        cs.nbytes = g->cc_bytes[v];
        cs.type = t;
        cs.algo = a;
        cs.N = gN[gi];
        cs.M = gM[gi];
        cs.K = gK[gi];
        cs.pad = 0;
        cs.lg = std::log2((double)gM[gi]);
        b.sigs.push_back(cs);
        b.sig_count.push_back(0);
      } else {
        s = it->second;
      }
      b.sig_count[s]++;
      b.comm_node.push_back((int32_t)i);
      b.comm_sig.push_back(s);
      b.node_sig[i] = s;
    }
  }
  overlap_candidates(b);
  // the comm ops that can overlap a compute op of their rank, on each of the
  // rank's timelines that hold any, in issue order
  for (int32_t r = 0; r < R; ++r) {
    int32_t n = 0;
    for (int32_t k = 1; k < NS; ++k) {
      const int64_t q = (int64_t)r * NS + k;
      for (int64_t i = g->q_off[q]; i < g->q_off[q + 1]; ++i)
        if (b.q_rel[i]) {
          ++n;
          break;
        }
    }
    b.n_cq = std::max(b.n_cq, n);
  }
  // With each entry, the ops whose finish its rank waits for before it launches
  // the comm op (for the validator variant that counts a comm op's interval on a
  // rank from that rank's launch): the op before it on its timeline and its data
  // producers that run on the rank.  A timeline is serial, so only the latest of
  // them on each of the rank's timelines is kept.
  b.cq_off.assign((size_t)R * b.n_cq + 1, 0);
  b.lq_off.assign(1, 0);
  b.lq_ops.clear();
  {
    std::vector<int32_t> tl(V, -1);  // timeline of an op of the rank at hand
    std::vector<int64_t> tpos(V, 0), best(NS);
    for (int32_t r = 0; r < R; ++r) {
      for (int32_t k = 0; k < NS; ++k)
        for (int64_t i = g->q_off[(int64_t)r * NS + k]; i < g->q_off[(int64_t)r * NS + k + 1]; ++i) {
          tl[b.q_ops_int[i]] = k;
          tpos[b.q_ops_int[i]] = i;
        }
      int32_t j = 0;
      for (int32_t k = 1; k < NS; ++k) {
        const int64_t q = (int64_t)r * NS + k;
        const size_t before = b.cq_ops.size();
        for (int64_t i = g->q_off[q]; i < g->q_off[q + 1]; ++i) {
          const int32_t w = b.q_ops_int[i];
          if (!b.q_rel[i]) continue;
          b.cq_ops.push_back(w);
          std::fill(best.begin(), best.end(), -1);
          if (i > g->q_off[q]) best[k] = i - 1;
          for (int64_t e = b.dp_off[w]; e < b.dp_off[w + 1]; ++e) {
            const int32_t u = b.dp[e];
            if (tl[u] >= 0) best[tl[u]] = std::max(best[tl[u]], tpos[u]);
          }
          for (int32_t kk = 0; kk < NS; ++kk)
            if (best[kk] >= 0) b.lq_ops.push_back(b.q_ops_int[best[kk]]);
          b.lq_off.push_back((int32_t)b.lq_ops.size());
        }
        if (b.cq_ops.size() > before) b.cq_off[(size_t)r * b.n_cq + ++j] = (int64_t)b.cq_ops.size();
      }
      for (; j < b.n_cq; ++j) b.cq_off[(size_t)r * b.n_cq + j + 1] = (int64_t)b.cq_ops.size();
      for (int32_t k = 0; k < NS; ++k)
        for (int64_t i = g->q_off[(int64_t)r * NS + k]; i < g->q_off[(int64_t)r * NS + k + 1]; ++i)
          tl[b.q_ops_int[i]] = -1;
    }
  }
  if (b.cq_ops.empty()) {
    b.cq_ops.push_back(0);
    b.lq_off.push_back(0);
  }
  if (b.lq_ops.empty()) b.lq_ops.push_back(0);
  b.keep.assign(V, 0);
  for (int64_t v = 0; v < V; ++v) b.keep[v] = b.cand_flag[v];
  const int64_t n_cqe = b.cq_off.back();  // (cq_ops and lq_off hold a placeholder when empty)
  for (int64_t e = 0; e < n_cqe; ++e) {
    b.keep[b.cq_ops[e]] = 1;
    for (int32_t q = b.lq_off[e]; q < b.lq_off[e + 1]; ++q) b.keep[b.lq_ops[q]] = 1;
  }
  b.seg_words.assign(NSg, 0);
  for (int64_t t = 0; t < NSg; ++t) {
    const int64_t nin = b.hin_off[t + 1] - b.hin_off[t];
    if (nin > 0xFFFF) b.stageable = false;
    bool cand = false, kept = false;
    for (int64_t v = b.seg_node_off[t]; v < b.seg_node_off[t + 1]; ++v) {
      cand = cand || b.cand_flag[v];
      kept = kept || (b.keep[v] && v + 1 < b.seg_node_off[t + 1]);
    }
    b.seg_words[t] = 4 + nin + (cand ? 3 : 0) + (kept ? 2 : 0);
  }
  // every input of a segment comes from an earlier level (the kernels' contract)
  {
    std::vector<int32_t> lvl(NSg, 0);
    for (int64_t l = 0; l < Ls; ++l)
      for (int64_t t = b.seg_lvl_off[l]; t < b.seg_lvl_off[l + 1]; ++t) lvl[t] = (int32_t)l;
    for (int64_t t = 0; t < NSg; ++t)
      for (int64_t q = b.hin_off[t]; q < b.hin_off[t + 1]; ++q)
        if (lvl[b.seg_int[b.hin[q]]] >= lvl[t])
          return fail(e, ECHO_E_BAD_GRAPH, "internal: segment %lld reads level %d from level %d", (long long)t,
                      lvl[b.seg_int[b.hin[q]]], lvl[t]);
  }
  if (programs) build_dataflow(b);
  return ECHO_OK;
}

// Ring sizes of the staged compose kernels for scenario blocks of `sigma`.  The
// duration and record rings must hold two consecutive segment levels (the one
// being composed and the one before it, which slower threads may still read);
// whatever more they hold is prefetch look-ahead.  Preference: a larger duration
// ring, then a larger value ring (more predecessors served from shared memory).
// Replica folding.  In DDP mode Echo composes a single copy of the workload of
// each DP group (Sec. 8.5).  Generalised here: the caller marks rank b as a
// replica of a representative rank a (replica_of[b] = a), meaning that b runs the
// same ops as a, timeline by timeline and position by position.  rho maps every
// op to its representative: an op that runs on some representative rank is its
// own (a DP all-reduce shared by the replicas, say); an op that runs only on
// replica ranks maps to the op at the same place on the representatives.  When
//   (i)   d(x) = d(rho x) for every op (checked per scenario batch, on the device),
//   (ii)  rho(preds(x)) = rho(preds(rho x)) as sets, and
//   (iii) the folded graph -- the representatives, with predecessors rho(preds) --
//         is acyclic,
// the folded longest-path times t satisfy the full graph's recurrence through
// f(x) = t(rho x), and as that recurrence has one solution, f(x) = t(rho x)
// exactly.  (ii) holds for issue order by the positional mapping and is checked
// here for data dependencies; the validator additionally needs a replica rank's
// launch conditions to mirror those of its representative, also checked.
struct Fold {
  std::vector<int32_t> rho;     // [V] representative of each op (caller ids)
  std::vector<int32_t> keep;    // folded id -> caller id
  std::vector<int32_t> red;     // [V] caller id -> folded id of its representative
  std::vector<int32_t> pairs;   // (replica op, representative) of every local replica-only op
  std::vector<uint8_t> kind, kclass, cc_type, cc_algo;
  std::vector<int32_t> group, pred_idx, q_ops, grp_rank;
  std::vector<int64_t> cc_bytes, pred_off, q_off, grp_off;
  std::vector<Shape> shape;     // [folded groups] (N, M, K) of the caller's group
  echo_graph_desc desc{};
};

// Checks `replica_of` against the graph `g` (already validated) and builds the
// folded graph in F.  F.keep stays empty when no rank is marked as a replica.
int build_fold(const echo_graph_desc *g, const int32_t *replica_of, Fold &F, Err &e) {
  const int64_t V = g->n_ops;
  const int32_t R = g->n_ranks, NS = g->n_streams;
  const int64_t NQ = (int64_t)R * NS, QE = g->q_off[NQ];
  bool any = false;
  for (int32_t r = 0; r < R; ++r) {
    const int32_t a = replica_of[r];
    if (a < 0 || a >= R) return fail(e, ECHO_E_INVALID_ARG, "replica_of[%d] = %d out of range", r, a);
    if (replica_of[a] != a)
      return fail(e, ECHO_E_BAD_GRAPH, "replica_of: rank %d mirrors rank %d, which is itself a replica", r, a);
    any = any || a != r;
  }
  if (!any) return ECHO_OK;
  auto is_rep = [&](int32_t r) { return replica_of[r] == r; };
  // ranks of each op, ascending (CSR), and whether it runs on a representative
  std::vector<int64_t> ro_off(V + 1, 0);
  for (int64_t i = 0; i < QE; ++i) ro_off[g->q_ops[i] + 1]++;
  for (int64_t v = 0; v < V; ++v) ro_off[v + 1] += ro_off[v];
  std::vector<int32_t> ro(std::max<int64_t>(QE, 1));
  std::vector<uint8_t> on_rep(V, 0);
  {
    std::vector<int64_t> fill(ro_off.begin(), ro_off.end() - 1);
    for (int64_t q = 0; q < NQ; ++q)
      for (int64_t i = g->q_off[q]; i < g->q_off[q + 1]; ++i) {
        const int32_t v = g->q_ops[i], r = (int32_t)(q / NS);
        ro[fill[v]++] = r;
        if (is_rep(r)) on_rep[v] = 1;
      }
  }
  auto runs_on = [&](int32_t u, int32_t r) {
    return std::binary_search(ro.data() + ro_off[u], ro.data() + ro_off[u + 1], r);
  };
  // the positional mapping
  F.rho.assign(V, -1);
  for (int32_t b = 0; b < R; ++b) {
    const int32_t a = replica_of[b];
    if (a == b) continue;
    for (int32_t k = 0; k < NS; ++k) {
      const int64_t qa = (int64_t)a * NS + k, qb = (int64_t)b * NS + k;
      const int64_t n = g->q_off[qb + 1] - g->q_off[qb];
      if (n != g->q_off[qa + 1] - g->q_off[qa])
        return fail(e, ECHO_E_BAD_GRAPH, "replica_of: timeline %d of rank %d holds %lld ops, of rank %d %lld", k, b,
                    (long long)n, a, (long long)(g->q_off[qa + 1] - g->q_off[qa]));
      for (int64_t i = 0; i < n; ++i) {
        const int32_t x = g->q_ops[g->q_off[qb] + i], y = g->q_ops[g->q_off[qa] + i];
        if (on_rep[x] ? x != y : (F.rho[x] >= 0 && F.rho[x] != y))
          return fail(e, ECHO_E_BAD_GRAPH, "replica_of: op %d (rank %d, timeline %d, position %lld) does not mirror op %d of rank %d",
                      x, b, k, (long long)i, y, a);
        if (!on_rep[x]) F.rho[x] = y;
      }
    }
  }
  for (int64_t v = 0; v < V; ++v)
    if (on_rep[v]) F.rho[v] = (int32_t)v;
  // group shapes of the caller's groups
  std::vector<Shape> gshape(g->n_groups);
  for (int32_t gi = 0; gi < g->n_groups; ++gi) {
    std::map<int32_t, int32_t> per_node;
    for (int64_t k = g->grp_off[gi]; k < g->grp_off[gi + 1]; ++k) per_node[g->grp_rank[k] / g->gpus_per_node]++;
    int32_t K = 0;
    for (auto &kv : per_node) K = std::max(K, kv.second);
    gshape[gi] = {(int32_t)(g->grp_off[gi + 1] - g->grp_off[gi]), (int32_t)per_node.size(), K};
  }
  auto is_comm = [&](int64_t v) { return g->kind[v] == ECHO_OP_COLL || g->kind[v] == ECHO_OP_P2P; };
  std::vector<int32_t> s1, s2;
  auto rho_set = [&](int32_t v, std::vector<int32_t> &out, int32_t on_rank) {
    out.clear();
    for (int64_t k = g->pred_off[v]; k < g->pred_off[v + 1]; ++k) {
      const int32_t u = g->pred_idx[k];
      if (on_rank < 0 || runs_on(u, on_rank)) out.push_back(F.rho[u]);
    }
    std::sort(out.begin(), out.end());
    out.erase(std::unique(out.begin(), out.end()), out.end());
  };
  for (int64_t x = 0; x < V; ++x) {
    if (on_rep[x]) continue;
    const int32_t y = F.rho[x];
    // same op
    bool same = g->kind[x] == g->kind[y] && (g->kind[x] != ECHO_OP_COMPUTE || g->kclass[x] == g->kclass[y]);
    if (same && is_comm(x))
      same = g->cc_type[x] == g->cc_type[y] && g->cc_bytes[x] == g->cc_bytes[y] &&
             (g->cc_type[x] != ECHO_CC_ALLREDUCE || g->cc_algo[x] == g->cc_algo[y]) &&
             gshape[g->group[x]] == gshape[g->group[y]];
    if (!same) return fail(e, ECHO_E_BAD_GRAPH, "replica_of: op %lld differs from its representative %d", (long long)x, y);
    // it runs on the replicas of exactly the representative ranks that run y
    s1.clear();
    for (int64_t k = ro_off[x]; k < ro_off[x + 1]; ++k) s1.push_back(replica_of[ro[k]]);
    std::sort(s1.begin(), s1.end());
    s2.clear();
    for (int64_t k = ro_off[y]; k < ro_off[y + 1]; ++k)
      if (is_rep(ro[k])) s2.push_back(ro[k]);
    if (std::adjacent_find(s1.begin(), s1.end()) != s1.end() || s1 != s2)
      return fail(e, ECHO_E_BAD_GRAPH, "replica_of: op %lld and its representative %d run on different ranks", (long long)x, y);
    // (ii) for data dependencies
    rho_set((int32_t)x, s1, -1);
    rho_set(y, s2, -1);
    if (s1 != s2)
      return fail(e, ECHO_E_BAD_GRAPH, "replica_of: the producers of op %lld do not mirror those of op %d", (long long)x, y);
  }
  // launch conditions on each replica rank mirror those on its representative
  for (int32_t b = 0; b < R; ++b) {
    const int32_t a = replica_of[b];
    if (a == b) continue;
    for (int32_t k = 1; k < NS; ++k) {
      const int64_t qa = (int64_t)a * NS + k, qb = (int64_t)b * NS + k;
      for (int64_t i = 0; i < g->q_off[qb + 1] - g->q_off[qb]; ++i) {
        const int32_t x = g->q_ops[g->q_off[qb] + i], y = g->q_ops[g->q_off[qa] + i];
        if (!is_comm(x)) continue;
        rho_set(x, s1, b);
        rho_set(y, s2, a);
        if (s1 != s2)
          return fail(e, ECHO_E_BAD_GRAPH, "replica_of: the producers of op %d on rank %d do not mirror those on rank %d", x, b, a);
      }
    }
  }
  // the folded graph
  F.red.assign(V, -1);
  F.keep.clear();
  for (int64_t v = 0; v < V; ++v)
    if (F.rho[v] == v) {
      F.red[v] = (int32_t)F.keep.size();
      F.keep.push_back((int32_t)v);
    }
  for (int64_t v = 0; v < V; ++v) F.red[v] = F.red[F.rho[v]];
  const int64_t Vf = (int64_t)F.keep.size();
  std::vector<int32_t> gmap(g->n_groups, -1);
  F.grp_off.assign(1, 0);
  F.grp_rank.clear();
  F.shape.clear();
  F.kind.resize(Vf);
  F.kclass.resize(Vf);
  F.cc_type.resize(Vf);
  F.cc_algo.resize(Vf);
  F.group.resize(Vf);
  F.cc_bytes.resize(Vf);
  F.pred_off.assign(Vf + 1, 0);
  F.pred_idx.clear();
  for (int64_t j = 0; j < Vf; ++j) {
    const int32_t v = F.keep[j];
    F.kind[j] = g->kind[v];
    F.kclass[j] = g->kclass[v];
    F.cc_type[j] = g->cc_type[v];
    F.cc_algo[j] = g->cc_algo[v];
    F.cc_bytes[j] = g->cc_bytes[v];
    F.group[j] = 0;
    if (is_comm(v)) {
      const int32_t gi = g->group[v];
      if (gmap[gi] < 0) {  // the group's representative members
        gmap[gi] = (int32_t)F.shape.size();
        for (int64_t k = g->grp_off[gi]; k < g->grp_off[gi + 1]; ++k)
          if (is_rep(g->grp_rank[k])) F.grp_rank.push_back(g->grp_rank[k]);
        F.grp_off.push_back((int64_t)F.grp_rank.size());
        F.shape.push_back(gshape[gi]);
      }
      F.group[j] = gmap[gi];
    }
    s1.clear();
    for (int64_t k = g->pred_off[v]; k < g->pred_off[v + 1]; ++k) s1.push_back(F.red[g->pred_idx[k]]);
    std::sort(s1.begin(), s1.end());
    s1.erase(std::unique(s1.begin(), s1.end()), s1.end());
    F.pred_idx.insert(F.pred_idx.end(), s1.begin(), s1.end());
    F.pred_off[j + 1] = (int64_t)F.pred_idx.size();
  }
  F.q_off.assign(NQ + 1, 0);
  F.q_ops.clear();
  for (int64_t q = 0; q < NQ; ++q) {
    if (is_rep((int32_t)(q / NS)))
      for (int64_t i = g->q_off[q]; i < g->q_off[q + 1]; ++i) F.q_ops.push_back(F.red[g->q_ops[i]]);
    F.q_off[q + 1] = (int64_t)F.q_ops.size();
  }
  F.pairs.clear();
  for (int64_t x = 0; x < V; ++x)
    if (F.rho[x] != x && !is_comm(x)) {
      F.pairs.push_back((int32_t)x);
      F.pairs.push_back(F.rho[x]);
    }
  echo_graph_desc &d = F.desc;
  d = echo_graph_desc{};
  d.n_ops = Vf;
  d.n_ranks = R;
  d.n_streams = NS;
  d.gpus_per_node = g->gpus_per_node;
  d.n_groups = (int32_t)F.shape.size();
  d.kind = F.kind.data();
  d.kclass = F.kclass.data();
  d.group = F.group.data();
  d.cc_type = F.cc_type.data();
  d.cc_algo = F.cc_algo.data();
  d.cc_bytes = F.cc_bytes.data();
  d.pred_off = F.pred_off.data();
  d.pred_idx = F.pred_idx.data();
  d.q_off = F.q_off.data();
  d.q_ops = F.q_ops.data();
  d.grp_off = F.grp_off.data();
  d.grp_rank = F.grp_rank.data();
  d.replica_of = nullptr;
  return ECHO_OK;
}

// The folded graph of `g` when its replica_of marks replicas: `fb` composes it,
// with int2ext / ext2int / V_ext in the caller's ids.  Returns ECHO_OK with
// *folded = false when there is nothing to fold.
int build_folded(const echo_graph_desc *g, GraphBuild &fb, Fold &F, bool *folded, Err &e, bool programs = true) {
  *folded = false;
  if (!g->replica_of) return ECHO_OK;
  int rc = build_fold(g, g->replica_of, F, e);
  if (rc || F.keep.empty()) return rc;
  Err e2;
  rc = build_graph(&F.desc, fb, e2, &F.shape, programs);
  if (rc) return fail(e, ECHO_E_BAD_GRAPH, "replica_of: the folded graph is not valid (%s)", e2.msg.c_str());
  for (auto &x : fb.int2ext) x = F.keep[x];
  std::vector<int32_t> e2i(g->n_ops);
  for (int64_t v = 0; v < g->n_ops; ++v) e2i[v] = fb.ext2int[F.red[v]];
  fb.ext2int.swap(e2i);
  fb.V_ext = g->n_ops;
  *folded = true;
  return ECHO_OK;
}

// The steps of the staged kernels for scenario blocks of `sigma`.  The segments of
// one level are independent, so a wide level may run as several consecutive
// steps: each step holds at most `cap` nodes and kStepSegments segments, so that
// two consecutive steps fit the shared-memory rings (the numbering stays as it is).
struct Steps {
  int64_t L = 0;
  std::vector<int64_t> off;    // [L+1] segments of each step
  std::vector<int64_t> words;  // [L] record block words (padded to 4)
  std::vector<int64_t> cand;   // [L+1] first level-order candidate of each step
};

Steps make_steps(const GraphBuild &b, int64_t cap) {
  Steps st;
  st.off.assign(1, 0);
  for (int64_t l = 0; l < b.Ls; ++l) {
    int64_t t = b.seg_lvl_off[l];
    while (t < b.seg_lvl_off[l + 1]) {
      int64_t u = t + 1;  // one segment always fits (at most kMaxSegment nodes)
      while (u < b.seg_lvl_off[l + 1] && u - t < kStepSegments && b.seg_node_off[u + 1] - b.seg_node_off[t] <= cap)
        ++u;
      st.off.push_back(u);
      t = u;
    }
  }
  st.L = (int64_t)st.off.size() - 1;
  st.words.assign(st.L, 0);
  st.cand.assign(st.L + 1, b.n_cand);
  for (int64_t l = 0; l < st.L; ++l) {
    int64_t w = 0;
    for (int64_t t = st.off[l]; t < st.off[l + 1]; ++t) w += b.seg_words[t];
    st.words[l] = (w + 3) & ~(int64_t)3;
    const int32_t first = (int32_t)b.seg_node_off[st.off[l]];
    st.cand[l] = std::lower_bound(b.cand_node.begin(), b.cand_node.begin() + b.n_cand, first) - b.cand_node.begin();
  }
  return st;
}

echo::StagedPlan plan_staged(const GraphBuild &b, const Steps &st, int sigma, size_t smem_cap) {
  echo::StagedPlan best;
  if (!b.stageable || st.L == 0) return best;
  auto pow2 = [](int64_t x) {
    int k = 0;
    while (((int64_t)1 << k) < x) ++k;
    return k;
  };
  int64_t rows2 = 0, words2 = 0, segmax = 0, prow = 0, pword = 0, crows2 = 0, pcand = 0;
  for (int64_t l = 0; l < st.L; ++l) {
    const int64_t r = b.seg_node_off[st.off[l + 1]] - b.seg_node_off[st.off[l]];
    const int64_t nc = st.cand[l + 1] - st.cand[l];
    crows2 = std::max(crows2, nc + pcand);
    pcand = nc;
    rows2 = std::max(rows2, r + prow);
    words2 = std::max(words2, st.words[l] + pword);
    segmax = std::max(segmax, st.off[l + 1] - st.off[l]);
    prow = r;
    pword = st.words[l];
  }
  const int dmin = std::max(pow2(rows2), 4), rmin = std::max(pow2(words2), 4);
  const int cring = std::max(pow2(crows2), 4);  // candidate ring: two levels' candidates
  const int vwant = std::min(std::max(pow2(4 * segmax), 6), 12);
  for (int d = dmin + 2; d >= dmin; --d)
    for (int v = vwant; v >= 6; --v)
      for (int r = rmin + 1; r >= rmin; --r) {
        const size_t need = echo::staged_layout(sigma, v, (size_t)1 << d, r, (size_t)1 << cring).total;
        if (need <= smem_cap && d < 31 && r < 31 && cring < 31) {
          best.ok = true;
          best.dring_log2 = d;
          best.vring_log2 = v;
          best.rring_log2 = r;
          best.cring_log2 = cring;
          best.smem = need;
          // the pipelined kernel's duration ring takes every row the rest leaves:
          // more levels in flight hide more of each level's copy latency
          const int64_t row = (int64_t)sigma * 8, fixed = (int64_t)echo::staged_layout(sigma, v, 0, r, 0).total;
          const int64_t crows = std::max<int64_t>(crows2, 2), room = (int64_t)smem_cap - fixed;
          best.pipe_crows = (uint32_t)crows;
          best.pipe_drows = (uint32_t)std::max<int64_t>(room / row, (int64_t)1 << d);
          best.pipe_drows_c = (uint32_t)std::max<int64_t>((room - crows * row) / row, (int64_t)1 << d);
          return best;
        }
      }
  return best;
}

// Record blocks of every segment level for scenario blocks of `sigma` and a value
// ring of 2^vlog2 segments, and the per-level metadata (word offset of the block,
// first node, first segment).  A head's inputs recent enough to be in the value
// ring become byte offsets of their slots, the others node ids.
void build_records(const GraphBuild &b, const Steps &stp, int sigma, int vlog2, std::vector<uint32_t> &recs,
                   std::vector<uint32_t> &meta) {
  const int64_t R = (int64_t)1 << vlog2;
  const uint32_t row = (uint32_t)sigma * 8;
  recs.clear();
  meta.assign(4 * (stp.L + 1), 0);
  std::vector<uint32_t> far;
  for (int64_t l = 0; l < stp.L; ++l) {
    const int64_t s0 = stp.off[l], s1 = stp.off[l + 1];
    const int64_t i0 = b.seg_node_off[s0];
    const size_t base = recs.size();
    meta[4 * l] = (uint32_t)base;
    meta[4 * l + 1] = (uint32_t)i0;
    meta[4 * l + 2] = (uint32_t)s0;
    meta[4 * l + 3] = (uint32_t)stp.cand[l];
    recs.resize(base + 4 * (s1 - s0), 0);
    for (int64_t t = s0; t < s1; ++t) {
      const int64_t h = b.seg_node_off[t], z = b.seg_node_off[t + 1] - 1;
      const size_t hd = base + 4 * (t - s0);
      recs[hd] = (uint32_t)(recs.size() - base);
      recs[hd + 2] = (uint32_t)(h - i0);
      recs[hd + 3] = (uint32_t)(z - h + 1);
      far.clear();
      uint32_t nin = 0;
      for (int64_t q = b.hin_off[t]; q < b.hin_off[t + 1]; ++q) {
        // an input's value-ring slot is rewritten by segment seg+R, which must not
        // be in segment levels <= l
        const int64_t u = b.hin[q], su = b.seg_int[u];
        if (su + R >= s1) {
          recs.push_back((uint32_t)(su & (R - 1)) * row);
          ++nin;
        } else {
          far.push_back((uint32_t)u);
        }
      }
      recs.insert(recs.end(), far.begin(), far.end());
      recs[hd + 1] = nin | ((uint32_t)far.size() << 16);
      // chain nodes that are overlap candidates: a 64-bit mask over the chain and the
      // level-order index of the first of them
      uint64_t mask = 0;
      int64_t c_first = -1;
      for (int64_t v = h; v <= z; ++v)
        if (b.cand_flag[v]) {
          mask |= 1ull << (v - h);
          if (c_first < 0) c_first = b.cidx[v];
        }
      if (mask) {
        recs[hd + 3] |= 1u << 16;
        recs.push_back((uint32_t)mask);
        recs.push_back((uint32_t)(mask >> 32));
        recs.push_back((uint32_t)c_first);
      }
      // chain positions before the tail whose finish a later step reads
      uint64_t kmask = 0;
      for (int64_t v = h; v < z; ++v)
        if (b.keep[v]) kmask |= 1ull << (v - h);
      if (kmask) {
        recs[hd + 3] |= 1u << 17;
        recs.push_back((uint32_t)kmask);
        recs.push_back((uint32_t)(kmask >> 32));
      }
    }
    while (recs.size() % 4) recs.push_back(0);
  }
  meta[4 * stp.L] = (uint32_t)recs.size();
  meta[4 * stp.L + 1] = (uint32_t)b.V;
  meta[4 * stp.L + 2] = (uint32_t)b.n_seg;
  meta[4 * stp.L + 3] = (uint32_t)stp.cand[stp.L];
  if (recs.empty()) recs.assign(4, 0);
}

// ------------------------------------------------------------------------------------
template <typename T>
struct DevArr {
  T *p = nullptr;
  size_t n = 0;
};

}  // namespace

struct echo_ctx {
  int device = 0;
  int sms = 0;
  cudaStream_t stream = nullptr;
  bool own_stream = false;
  std::string err;
  int state = 0;  // 0 empty, 1 graph, 2 scenarios, 3 estimated, 4 composed
  GraphBuild gb;
  std::vector<void *> graph_allocs, scen_allocs;
  // replica folding: the other build of the graph (the full one while the folded
  // one is active, and the reverse), pairs of rows whose durations must match
  bool fold_ok = false, fold_active = false;
  GraphBuild gb_alt;
  std::vector<void *> fold_allocs;
  int32_t *fold_pairs = nullptr, *fold_flag = nullptr;
  int64_t n_fold_pairs = 0;
  std::vector<void *> raw_allocs;  // the caller's durations as uploaded
  size_t raw_cap = 0;
  // device graph
  int64_t *seg_lvl_off = nullptr, *seg_node_off = nullptr, *nq_off = nullptr, *dp_off = nullptr, *q_off = nullptr;
  int64_t *cq_off = nullptr;
  uint8_t *cand_kcl = nullptr;
  int32_t *cq_ops = nullptr, *lq_off = nullptr, *lq_ops = nullptr;
  int64_t *cand_off = nullptr;
  int32_t *cand_ops = nullptr;
  uint8_t *cand_flag = nullptr;
  int32_t *nq = nullptr, *dp = nullptr, *q_ops = nullptr, *int2ext = nullptr, *ext2int = nullptr;
  int32_t *node_sig = nullptr, *comm_node = nullptr, *comm_sig = nullptr, *sig_count = nullptr;
  uint8_t *kcl = nullptr, *local = nullptr;
  CcSig *sigs = nullptr;
  int32_t *status = nullptr;
  // scenarios
  int32_t S = 0, C = 0, sigma = 1;
  size_t scen_vs = 0;  // elements of each [op][scenario] matrix (blocked layout, padded)
  echo::MatLayout lay{0, 0};
  ChunkTable tbl{};
  double *prm = nullptr, *sums = nullptr, *comm_sum = nullptr, *cc_ns = nullptr;
  double *sf = nullptr;     // slowdown factors [C][S]
  void *raw = nullptr;
  int64_t *dur = nullptr, *f[2] = {nullptr, nullptr}, *mk = nullptr, *cc_dur = nullptr;
  int64_t *gfrontier = nullptr;
  int64_t *deff = nullptr;                // full validator durations, for kernels without a candidate ring
  int64_t *cd[2] = {nullptr, nullptr};    // candidates' durations of the validator's passes (compact)
  echo::MatLayout lay_c{0, 0};            // [n_cand][S] compact layout
  size_t cd_elems = 0;                    // elements of each compact matrix
  int32_t *cand_cidx = nullptr, *cidx = nullptr, *cand_node = nullptr;
  uint8_t *ov = nullptr;
  uint32_t *d_recs = nullptr, *d_meta = nullptr;
  echo::StagedPlan plan;
  Steps steps;  // composition steps of the staged kernels
  uint32_t rec_words = 0;
  std::vector<double> h_sums, h_maxsf;
  int final_f = 0;
  const int64_t *final_cd = nullptr;  // candidates' durations of the last composition (null: the original)
  bool have_ov = false;
  echo::OverlapArgs last_ov{};  // inputs of the last validator pass (to recompute its decisions)
  int kernel_choice = 0;            // 0 automatic, 1 direct, 2 staged, 3 pipelined, 4 dataflow (tuning and tests)
  // dataflow composer
  bool use_df = false;
  int64_t *df_off = nullptr;
  uint32_t *df_rec = nullptr, *df_opnd = nullptr;
  uint64_t *df_part = nullptr, *df_xval = nullptr;
  size_t df_part_elems = 0, df_xval_elems = 0;
  uint32_t df_epoch = 0;
  int32_t *df_abort = nullptr;
  int cc_model = ECHO_CC_MODEL_WHITEBOX;
  int est_policy = ECHO_AR_PER_OP;  // all-reduce policy of the current estimates
  long long wait_limit_cycles = 0;  // bound of every device-side wait
  int32_t skip_level = -1;          // failure injection for tests
  // scratch for readback / queries
  void *stage = nullptr;
  size_t stage_bytes = 0;
  // profiling
  bool prof = false;
  std::vector<std::pair<std::string, std::pair<cudaEvent_t, cudaEvent_t>>> recs;
  std::vector<cudaEvent_t> ev_pool;
};

namespace {

int set_err(echo_ctx *c, int code, const std::string &msg) {
  if (c) c->err = msg;
  return code;
}

int cuda_fail(echo_ctx *c, cudaError_t e, const char *what) {
  std::string m = std::string(what) + ": " + cudaGetErrorString(e);
  if (e == cudaErrorMemoryAllocation) return set_err(c, ECHO_E_OOM, m);
  return set_err(c, ECHO_E_CUDA, m);
}

#define CK(call, what)                           \
  do {                                           \
    cudaError_t _e = (call);                     \
    if (_e != cudaSuccess) return cuda_fail(c, _e, what); \
  } while (0)

template <typename T>
int dalloc(echo_ctx *c, std::vector<void *> &owner, T **p, size_t n) {
  size_t bytes = std::max<size_t>(n, 1) * sizeof(T);
  void *q = nullptr;
  cudaError_t e = cudaMalloc(&q, bytes);
  if (e != cudaSuccess) {
    (void)cudaGetLastError();
    return set_err(c, ECHO_E_OOM, "cudaMalloc of " + std::to_string(bytes) + " bytes failed");
  }
  owner.push_back(q);
  *p = static_cast<T *>(q);
  return ECHO_OK;
}

template <typename T>
int upload(echo_ctx *c, std::vector<void *> &owner, T **p, const std::vector<T> &h) {
  int rc = dalloc(c, owner, p, h.size());
  if (rc) return rc;
  if (!h.empty()) CK(cudaMemcpyAsync(*p, h.data(), h.size() * sizeof(T), cudaMemcpyHostToDevice, c->stream), "upload");
  return ECHO_OK;
}

void free_all(std::vector<void *> &v) {
  for (void *p : v) cudaFree(p);
  v.clear();
}

int stage_reserve(echo_ctx *c, size_t bytes) {
  if (c->stage_bytes >= bytes) return ECHO_OK;
  if (c->stage) cudaFree(c->stage);
  c->stage = nullptr;
  c->stage_bytes = 0;
  cudaError_t e = cudaMalloc(&c->stage, bytes);
  if (e != cudaSuccess) {
    (void)cudaGetLastError();
    return set_err(c, ECHO_E_OOM, "cudaMalloc of the readback buffer failed");
  }
  c->stage_bytes = bytes;
  return ECHO_OK;
}

template <typename F>
cudaError_t timed(echo_ctx *c, const char *name, F &&launch) {
  if (!c->prof) return launch();
  auto get = [&]() {
    cudaEvent_t ev;
    if (!c->ev_pool.empty()) {
      ev = c->ev_pool.back();
      c->ev_pool.pop_back();
    } else {
      cudaEventCreate(&ev);
    }
    return ev;
  };
  cudaEvent_t a = get(), b = get();
  cudaEventRecord(a, c->stream);
  cudaError_t e = launch();
  cudaEventRecord(b, c->stream);
  c->recs.push_back({name, {a, b}});
  return e;
}

int check_ctx(echo_ctx *c) {
  if (!c) return ECHO_E_INVALID_ARG;
  cudaError_t e = cudaSetDevice(c->device);
  if (e != cudaSuccess) return cuda_fail(c, e, "cudaSetDevice");
  return ECHO_OK;
}

int pick_sigma(int32_t S, int sms) {
  if (const char *e = std::getenv("ECHO_SIGMA")) {  // tuning override: 1, 2, 4, 8 or 16
    int v = std::atoi(e);
    if (v == 1 || v == 2 || v == 4 || v == 8 || v == 16) return v;
  }
  int want = (S + sms - 1) / std::max(sms, 1);
  int s = 1;
  while (s < want && s < 16) s <<= 1;
  return s;
}

int sync_status(echo_ctx *c, int32_t *host_status) {
  CK(cudaMemcpyAsync(host_status, c->status, sizeof(int32_t), cudaMemcpyDeviceToHost, c->stream), "status readback");
  CK(cudaStreamSynchronize(c->stream), "cudaStreamSynchronize");
  return ECHO_OK;
}

int check_params(echo_ctx *c, int64_t n, const double *alpha, const double *bwa, const double *lata,
                 const double *bwe, const double *late, const double *delta) {
  if (n > 0 && (!alpha || !bwa || !lata || !bwe || !late || !delta))
    return set_err(c, ECHO_E_INVALID_ARG, "link parameter arrays are required");
  for (int64_t s = 0; s < n; ++s) {
    if (!finite_nonneg(alpha[s]) || !finite_nonneg(lata[s]) || !finite_nonneg(late[s]) || !finite_nonneg(delta[s]))
      return set_err(c, ECHO_E_INVALID_ARG, "alpha, latencies and delta must be finite and >= 0 (entry " + std::to_string(s) + ")");
    if (!(std::isfinite(bwa[s]) && bwa[s] > 0.0) || !(std::isfinite(bwe[s]) && bwe[s] > 0.0))
      return set_err(c, ECHO_E_INVALID_ARG, "bandwidths must be finite and > 0 (entry " + std::to_string(s) + ")");
  }
  return ECHO_OK;
}

int make_table(echo_ctx *c, int32_t n, const int64_t *mx, const int64_t *cb, ChunkTable *t) {
  std::memset(t, 0, sizeof *t);
  if (n == 0) {
    t->n = 5;
    for (int i = 0; i < 5; ++i) {
      t->max_bytes[i] = kDefaultMax[i];
      t->chunk[i] = kDefaultChunk[i];
    }
    return ECHO_OK;
  }
  if (n < 0 || n > echo::kMaxChunk) return set_err(c, ECHO_E_UNSUPPORTED, "chunk table size outside [0, 16]");
  if (!mx || !cb) return set_err(c, ECHO_E_INVALID_ARG, "chunk table arrays are NULL");
  t->n = n;
  for (int i = 0; i < n; ++i) {
    if (cb[i] <= 0) return set_err(c, ECHO_E_INVALID_ARG, "chunk sizes must be > 0");
    if (i > 0 && mx[i] < mx[i - 1]) return set_err(c, ECHO_E_INVALID_ARG, "chunk_max_bytes must be ascending");
    t->max_bytes[i] = mx[i];
    t->chunk[i] = cb[i];
  }
  return ECHO_OK;
}

// Device copies of the active graph build c->gb.
int upload_graph(echo_ctx *c) {
  free_all(c->graph_allocs);
  const GraphBuild &B = c->gb;
  auto &o = c->graph_allocs;
  int rc;
  if ((rc = upload(c, o, &c->seg_lvl_off, B.seg_lvl_off)) || (rc = upload(c, o, &c->seg_node_off, B.seg_node_off)) ||
      (rc = upload(c, o, &c->cand_kcl, B.cand_kcl)) ||
      (rc = upload(c, o, &c->cq_off, B.cq_off)) || (rc = upload(c, o, &c->cq_ops, B.cq_ops)) ||
      (rc = upload(c, o, &c->lq_off, B.lq_off)) || (rc = upload(c, o, &c->lq_ops, B.lq_ops)) ||
      (rc = upload(c, o, &c->cand_off, B.cand_off)) || (rc = upload(c, o, &c->cand_ops, B.cand_ops)) ||
      (rc = upload(c, o, &c->cand_flag, B.cand_flag)) || (rc = upload(c, o, &c->cand_cidx, B.cand_cidx)) ||
      (rc = upload(c, o, &c->cidx, B.cidx)) || (rc = upload(c, o, &c->cand_node, B.cand_node)) ||
      (rc = upload(c, o, &c->nq_off, B.nq_off)) ||
      (rc = upload(c, o, &c->nq, B.nq)) || (rc = upload(c, o, &c->dp_off, B.dp_off)) ||
      (rc = upload(c, o, &c->dp, B.dp)) || (rc = upload(c, o, &c->q_off, B.q_off)) ||
      (rc = upload(c, o, &c->q_ops, B.q_ops_int)) || (rc = upload(c, o, &c->int2ext, B.int2ext)) ||
      (rc = upload(c, o, &c->ext2int, B.ext2int)) || (rc = upload(c, o, &c->node_sig, B.node_sig)) ||
      (rc = upload(c, o, &c->comm_node, B.comm_node)) || (rc = upload(c, o, &c->comm_sig, B.comm_sig)) ||
      (rc = upload(c, o, &c->sig_count, B.sig_count)) || (rc = upload(c, o, &c->kcl, B.kcl)) ||
      (rc = upload(c, o, &c->local, B.local)) ||
      (rc = upload(c, o, &c->sigs, B.sigs)) ||
      (B.df_ok && ((rc = upload(c, o, &c->df_off, B.df_off)) || (rc = upload(c, o, &c->df_rec, B.df_rec)) ||
                   (rc = upload(c, o, &c->df_opnd, B.df_opnd))))) {
    free_all(c->graph_allocs);
    return rc;
  }
  CK(cudaStreamSynchronize(c->stream), "graph upload");
  return ECHO_OK;
}

// Makes the folded (want = true) or the full build of the graph the active one.
int activate_fold(echo_ctx *c, bool want) {
  if (!c->fold_ok || want == c->fold_active) return ECHO_OK;
  std::swap(c->gb, c->gb_alt);
  c->fold_active = want;
  free_all(c->scen_allocs);
  c->scen_vs = 0;
  const int rc = upload_graph(c);
  if (rc) {  // no device graph any more: the graph must be loaded again
    c->state = 0;
    c->fold_ok = false;
  }
  return rc;
}

}  // namespace

extern "C" {

const char *echo_strerror(int s) {
  switch (s) {
    case ECHO_OK: return "ok";
    case ECHO_E_INVALID_ARG: return "invalid argument";
    case ECHO_E_BAD_GRAPH: return "malformed graph";
    case ECHO_E_CYCLE: return "dependency cycle";
    case ECHO_E_STATE: return "call out of order";
    case ECHO_E_OOM: return "out of memory";
    case ECHO_E_CUDA: return "CUDA error";
    case ECHO_E_TIMEOUT: return "device wait timed out";
    case ECHO_E_OVERFLOW: return "time overflow";
    case ECHO_E_BOUNDS: return "a device-side index check failed";
    case ECHO_E_UNSUPPORTED: return "unsupported size";
    default: return "unknown status";
  }
}

int echo_last_error(echo_ctx *c, char *buf, size_t n) {
  if (!c || !buf || n == 0) return ECHO_E_INVALID_ARG;
  std::snprintf(buf, n, "%s", c->err.c_str());
  return ECHO_OK;
}

int echo_create(echo_ctx **out, int device, void *cuda_stream) {
  if (!out) return ECHO_E_INVALID_ARG;
  *out = nullptr;
  int n = 0;
  if (cudaGetDeviceCount(&n) != cudaSuccess || device < 0 || device >= n) {
    (void)cudaGetLastError();
    return ECHO_E_INVALID_ARG;
  }
  echo_ctx *c = new (std::nothrow) echo_ctx();
  if (!c) return ECHO_E_OOM;
  c->device = device;
  if (cudaSetDevice(device) != cudaSuccess ||
      cudaDeviceGetAttribute(&c->sms, cudaDevAttrMultiProcessorCount, device) != cudaSuccess) {
    delete c;
    return ECHO_E_CUDA;
  }
  if (cuda_stream) {
    c->stream = static_cast<cudaStream_t>(cuda_stream);
  } else {
    if (cudaStreamCreateWithFlags(&c->stream, cudaStreamNonBlocking) != cudaSuccess) {
      delete c;
      return ECHO_E_CUDA;
    }
    c->own_stream = true;
  }
  void *st = nullptr;
  if (cudaMalloc(&st, sizeof(int32_t)) != cudaSuccess) {
    if (c->own_stream) cudaStreamDestroy(c->stream);
    delete c;
    return ECHO_E_OOM;
  }
  c->status = static_cast<int32_t *>(st);
  if (const char *e = std::getenv("ECHO_COMPOSE_KERNEL")) {  // tuning and tests: force a compose kernel
    const std::string k(e);
    c->kernel_choice = k == "direct" ? 1 : k == "staged" ? 2 : k == "pipelined" ? 3 : k == "dataflow" ? 4 : 0;
  }
  // device waits give up after 2 s (tests shorten this and inject a level that never arrives)
  int clock_khz = 0;
  cudaDeviceGetAttribute(&clock_khz, cudaDevAttrClockRate, device);
  double limit_ms = 2000.0;
  if (const char *e = std::getenv("ECHO_TEST_WAIT_LIMIT_MS")) limit_ms = std::atof(e);
  c->wait_limit_cycles = (long long)(std::max(clock_khz, 1000) * limit_ms);
  if (const char *e = std::getenv("ECHO_TEST_SKIP_LEVEL")) c->skip_level = std::atoi(e);
  *out = c;
  return ECHO_OK;
}

int echo_destroy(echo_ctx *c) {
  if (!c) return ECHO_OK;
  cudaSetDevice(c->device);
  cudaStreamSynchronize(c->stream);
  free_all(c->graph_allocs);
  free_all(c->scen_allocs);
  free_all(c->fold_allocs);
  free_all(c->raw_allocs);
  if (c->stage) cudaFree(c->stage);
  if (c->status) cudaFree(c->status);
  for (auto &r : c->recs) {
    cudaEventDestroy(r.second.first);
    cudaEventDestroy(r.second.second);
  }
  for (auto ev : c->ev_pool) cudaEventDestroy(ev);
  if (c->own_stream) cudaStreamDestroy(c->stream);
  delete c;
  return ECHO_OK;
}

int echo_check_graph(const echo_graph_desc *g, int64_t *n_levels, int64_t *max_width) {
  GraphBuild b;
  Err e;
  int rc = build_graph(g, b, e, nullptr, false);
  if (rc) return rc;
  if (n_levels) *n_levels = b.L;
  if (max_width) *max_width = b.max_width;
  return ECHO_OK;
}

int echo_check_replicas(const echo_graph_desc *g, int64_t *n_ops_folded) {
  GraphBuild b, fb;
  Fold F;
  Err e;
  bool folded = false;
  int rc = build_graph(g, b, e, nullptr, false);
  if (!rc) rc = build_folded(g, fb, F, &folded, e, false);
  if (rc) return rc;
  if (n_ops_folded) *n_ops_folded = folded ? fb.V : b.V;
  return ECHO_OK;
}

int echo_overlap_candidates(const echo_graph_desc *g, uint8_t *flags, int64_t *n_candidates) {
  GraphBuild b;
  Err e;
  const int rc = build_graph(g, b, e, nullptr, false);
  if (rc) return rc;
  if (flags)
    for (int64_t v = 0; v < b.V; ++v) flags[v] = b.cand_flag[b.ext2int[v]];
  if (n_candidates) *n_candidates = b.n_cand;
  return ECHO_OK;
}

int echo_load_graph(echo_ctx *c, const echo_graph_desc *g) {
  int rc = check_ctx(c);
  if (rc) return rc;
  GraphBuild b, fb;
  Fold F;
  Err e;
  bool folded = false;
  if ((rc = build_graph(g, b, e)) || (rc = build_folded(g, fb, F, &folded, e))) return set_err(c, rc, e.msg);
  CK(cudaStreamSynchronize(c->stream), "cudaStreamSynchronize");
  free_all(c->graph_allocs);
  free_all(c->scen_allocs);
  free_all(c->fold_allocs);
  c->scen_vs = 0;
  c->state = 0;
  c->fold_ok = c->fold_active = folded;
  c->n_fold_pairs = 0;
  if (folded) {  // compose the folded graph until a scenario batch breaks the symmetry
    c->gb = std::move(fb);
    c->gb_alt = std::move(b);
    c->n_fold_pairs = (int64_t)F.pairs.size() / 2;
    if (F.pairs.empty()) F.pairs.assign(2, 0);
    if ((rc = upload(c, c->fold_allocs, &c->fold_pairs, F.pairs)) ||
        (rc = dalloc(c, c->fold_allocs, &c->fold_flag, 1)))
      return rc;
  } else {
    c->gb = std::move(b);
    c->gb_alt = GraphBuild{};
  }
  if ((rc = upload_graph(c))) return rc;
  c->state = 1;
  return ECHO_OK;
}

int echo_load_scenarios(echo_ctx *c, const echo_scen_desc *sc) {
  int rc = check_ctx(c);
  if (rc) return rc;
  if (c->state < 1) return set_err(c, ECHO_E_STATE, "load a graph first");
  if (!sc) return set_err(c, ECHO_E_INVALID_ARG, "scenario descriptor is NULL");
  const GraphBuild &B = c->gb;  // (the active build: folded or full)
  const int64_t Vx = B.V_ext;
  const int32_t S = sc->n_scen;
  if (S < 1) return set_err(c, ECHO_E_INVALID_ARG, "n_scen must be >= 1");
  if (sc->n_kclass < 1 || sc->n_kclass <= B.max_kclass)
    return set_err(c, ECHO_E_INVALID_ARG, "n_kclass must exceed every compute op's kclass");
  if (Vx > 0 && !sc->dur) return set_err(c, ECHO_E_INVALID_ARG, "dur is NULL");
  if (sc->dur_bits != 0 && sc->dur_bits != 32 && sc->dur_bits != 64)
    return set_err(c, ECHO_E_INVALID_ARG, "dur_bits must be 32 or 64");
  if (!sc->slowdown) return set_err(c, ECHO_E_INVALID_ARG, "slowdown is NULL");
  if ((rc = check_params(c, S, sc->alpha_ns, sc->bw_intra, sc->lat_intra, sc->bw_inter, sc->lat_inter, sc->delta)))
    return rc;
  const int32_t C = sc->n_kclass;
  std::vector<double> maxsf(S, 1.0);
  for (int64_t k = 0; k < (int64_t)C * S; ++k) {
    double x = sc->slowdown[k];
    if (!(std::isfinite(x) && x > 0.0 && x <= 1e6))
      return set_err(c, ECHO_E_INVALID_ARG, "slowdown factors must be in (0, 1e6]");
    maxsf[k % S] = std::max(maxsf[k % S], x);
  }
  ChunkTable tbl;
  if ((rc = make_table(c, sc->n_chunk, sc->chunk_max_bytes, sc->chunk_bytes, &tbl))) return rc;

  CK(cudaStreamSynchronize(c->stream), "cudaStreamSynchronize");
  c->state = 1;
  // the caller's durations, as given, on the device
  const int bits = sc->dur_bits == 32 ? 32 : 64;
  const size_t raw_bytes = (size_t)Vx * S * (bits / 8);
  if (raw_bytes > c->raw_cap) {
    free_all(c->raw_allocs);
    c->raw = nullptr;
    c->raw_cap = 0;
    uint8_t *p = nullptr;
    if ((rc = dalloc(c, c->raw_allocs, &p, raw_bytes))) return rc;
    c->raw = p;
    c->raw_cap = raw_bytes;
  }
  if (Vx > 0)
    CK(cudaMemcpyAsync(c->raw, sc->dur, raw_bytes, cudaMemcpyHostToDevice, c->stream), "duration upload");
  if (c->fold_ok) {
    // the folded graph gives the full graph's times when every replica op's
    // durations equal its representative's in every scenario
    int32_t h_flag = 0;
    CK(cudaMemsetAsync(c->fold_flag, 0, sizeof(int32_t), c->stream), "memset");
    CK(timed(c, "replica_check", [&] {
         return echo::launch_replica_check(c->raw, bits, c->fold_pairs, c->n_fold_pairs, S, c->fold_flag, c->stream);
       }), "replica check launch");
    CK(cudaMemcpyAsync(&h_flag, c->fold_flag, sizeof h_flag, cudaMemcpyDeviceToHost, c->stream), "flag readback");
    CK(cudaStreamSynchronize(c->stream), "cudaStreamSynchronize");
    if ((rc = activate_fold(c, h_flag == 0))) return rc;
  }
  const int64_t V = B.V;
  // The dataflow composer (rows of 32 scenarios, a warp per rank) is serial in
  // the length of the longest rank program, the levelled ones in their number of
  // steps.  Measured on GB300: a program entry costs about 0.22 us while at most
  // 8 warps share an SM, and proportionally more beyond (0.24 us on GPT-1.3B x 256,
  // 0.37 us at 13.5 warps per SM on the 1024-rank workload, 0.52 us at 20 on
  // GPT-175B x 1024); a levelled step costs about 1.1 us.  The cheaper estimate
  // wins (when every warp can be resident).
  const int32_t n_groups = (S + 31) / 32;
  bool use_df = false;
  if (B.df_ok && (c->kernel_choice == 0 || c->kernel_choice == 4) &&
      echo::dataflow_fits((int64_t)B.R * n_groups, B.NS, B.df_wpb, c->device)) {
    int64_t longest = 0;
    for (int32_t r = 0; r < B.R; ++r) longest = std::max(longest, B.df_off[r + 1] - B.df_off[r]);
    const double warps_per_sm = (double)B.R * n_groups / std::max(c->sms, 1);
    const double df_us = (double)longest * 0.22 * std::max(1.0, warps_per_sm / 8.0);
    const double lev_us = (double)make_steps(B, kStepNodes).L * 1.1;
    use_df = c->kernel_choice == 4 || df_us < lev_us;
  }
  const int sigma = use_df ? 32 : pick_sigma(S, c->sms);
  int slog2 = 0;
  while ((1 << slog2) < sigma) ++slog2;
  // [op][scenario] matrices are stored in scenario blocks of sigma (the last padded)
  const size_t VS = (size_t)V * (size_t)((S + sigma - 1) / sigma) * sigma;
  const int32_t G = (int32_t)B.sigs.size();
  if (c->scen_vs != VS || c->S != S || c->C != C || c->sigma != sigma || c->use_df != use_df) {
    free_all(c->scen_allocs);
    c->scen_vs = 0;
    auto &o = c->scen_allocs;
    bool in_smem = true;
    echo::compose_smem_bytes(B.R * B.NS, sigma, &in_smem);
    int64_t nblk = (S + sigma - 1) / sigma;
    const size_t CS = (size_t)std::max<int64_t>(B.n_cand, 1) * (size_t)nblk * sigma;  // compact matrices
    if ((rc = dalloc(c, o, &c->prm, (size_t)6 * S)) || (rc = dalloc(c, o, &c->sf, (size_t)C * S)) ||
        (rc = dalloc(c, o, &c->sums, (size_t)S)) || (rc = dalloc(c, o, &c->comm_sum, (size_t)S)) ||
        (rc = dalloc(c, o, &c->dur, VS)) ||
        (rc = dalloc(c, o, &c->f[0], VS)) || (rc = dalloc(c, o, &c->f[1], VS)) ||
        (rc = dalloc(c, o, &c->cd[0], CS)) || (rc = dalloc(c, o, &c->ov, VS)) ||
        (rc = dalloc(c, o, &c->mk, (size_t)S)) || (rc = dalloc(c, o, &c->cc_ns, (size_t)G * S)) ||
        (rc = dalloc(c, o, &c->cc_dur, (size_t)G * S)) ||
        (!in_smem && (rc = dalloc(c, o, &c->gfrontier, (size_t)nblk * B.R * B.NS * sigma)))) {
      free_all(c->scen_allocs);
      return rc;
    }
    if (in_smem) c->gfrontier = nullptr;
    c->use_df = use_df;
    if (use_df) {
      c->df_part_elems = (size_t)std::max<int64_t>(B.df_slots, 1) * n_groups * 32;
      c->df_xval_elems = (size_t)std::max<int64_t>(B.df_exports, 1) * n_groups * 32;
      if ((rc = dalloc(c, o, &c->df_part, c->df_part_elems)) || (rc = dalloc(c, o, &c->df_xval, c->df_xval_elems)) ||
          (rc = dalloc(c, o, &c->df_abort, 1))) {
        free_all(c->scen_allocs);
        return rc;
      }
      // zeroed words carry tag 0, which no launch uses
      CK(cudaMemsetAsync(c->df_part, 0, c->df_part_elems * sizeof(uint64_t), c->stream), "memset");
      CK(cudaMemsetAsync(c->df_xval, 0, c->df_xval_elems * sizeof(uint64_t), c->stream), "memset");
    }
    // padding lanes of the duration matrices stay zero
    CK(cudaMemsetAsync(c->dur, 0, VS * sizeof(int64_t), c->stream), "memset");
    CK(cudaMemsetAsync(c->cd[0], 0, CS * sizeof(int64_t), c->stream), "memset");
    c->cd[1] = nullptr;   // second compact buffer: allocated when refine_passes > 1
    c->deff = nullptr;    // allocated when a kernel without a candidate ring composes a second pass
    // launch shape of the staged kernels (threads and blocks per SM may be overridden
    // for tuning: ECHO_STAGED_THREADS, ECHO_BLOCKS_PER_SM)
    int optin = 0, per_sm = 0;
    cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, c->device);
    cudaDeviceGetAttribute(&per_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, c->device);
    int threads = sigma == 16 ? 1024 : sigma == 8 ? 512 : sigma == 4 ? 256 : 512;
    int bps = 1;
    if (const char *e = std::getenv("ECHO_STAGED_THREADS")) threads = std::atoi(e);
    if (const char *e = std::getenv("ECHO_BLOCKS_PER_SM")) bps = std::max(1, std::atoi(e));
    const size_t cap = std::min((size_t)std::max(optin - 1024, 0), (size_t)(per_sm / bps) - 1024);
    // the widest steps whose rings fit
    for (int64_t step_cap = kStepNodes; !use_df; step_cap /= 2) {
      c->steps = make_steps(B, step_cap);
      c->plan = plan_staged(B, c->steps, sigma, cap);
      if (c->plan.ok || step_cap <= 2 * echo::kMaxSegment) break;
    }
    if (use_df) c->plan = echo::StagedPlan{};
    const Steps &st = c->steps;
    c->plan.threads = threads;
    if (c->plan.ok) {
      // the pipelined kernel moves whole rows of even width and arms each step's
      // byte count on one mbarrier (transaction counts stay below 2^20)
      int64_t max_bytes = 0;
      for (int64_t l = 0; l < st.L; ++l) {
        const int64_t rows = B.seg_node_off[st.off[l + 1]] - B.seg_node_off[st.off[l]];
        max_bytes = std::max(max_bytes, rows * sigma * 8 + st.words[l] * 4 + 32 + (st.cand[l + 1] - st.cand[l]) * sigma * 8);
      }
      c->plan.pipelined = sigma % 2 == 0 && max_bytes < (1 << 20);
      std::vector<uint32_t> recs, meta;
      build_records(B, st, sigma, c->plan.vring_log2, recs, meta);
      c->rec_words = meta[4 * st.L];
      if ((rc = upload(c, o, &c->d_recs, recs)) || (rc = upload(c, o, &c->d_meta, meta))) {
        free_all(c->scen_allocs);
        return rc;
      }
    }
    c->scen_vs = VS;
    c->S = S;
    c->C = C;
    c->sigma = sigma;
    c->lay = echo::MatLayout{V, slog2};
    c->lay_c = echo::MatLayout{B.n_cand, slog2};
    c->cd_elems = CS;
  }
  c->tbl = tbl;
  c->h_maxsf = maxsf;
  // parameters
  const double *src[6] = {sc->alpha_ns, sc->bw_intra, sc->lat_intra, sc->bw_inter, sc->lat_inter, sc->delta};
  for (int k = 0; k < 6; ++k)
    CK(cudaMemcpyAsync(c->prm + (size_t)k * S, src[k], S * sizeof(double), cudaMemcpyHostToDevice, c->stream), "parameter upload");
  CK(cudaMemcpyAsync(c->sf, sc->slowdown, (size_t)C * S * sizeof(double), cudaMemcpyHostToDevice, c->stream),
     "slowdown upload");
  CK(cudaMemsetAsync(c->sums, 0, S * sizeof(double), c->stream), "memset");
  CK(cudaMemsetAsync(c->status, 0, sizeof(int32_t), c->stream), "memset");
  if (V > 0) {
    CK(timed(c, "permute_rows", [&] {
         return echo::launch_permute_rows(c->raw, bits, c->int2ext, c->local, V, S, c->lay, c->dur, c->sums,
                                          c->status, c->stream);
       }), "permute_rows launch");
  }
  c->h_sums.assign(S, 0.0);
  CK(cudaMemcpyAsync(c->h_sums.data(), c->sums, S * sizeof(double), cudaMemcpyDeviceToHost, c->stream), "sum readback");
  int32_t st = 0;
  if ((rc = sync_status(c, &st))) return rc;
  if (st == echo::kDevNegativeDuration) return set_err(c, ECHO_E_INVALID_ARG, "negative duration in dur");
  c->state = 2;
  return ECHO_OK;
}

// CC estimates of every signature and scenario under all-reduce policy `policy`,
// scattered into the duration rows of the comm ops, with the overflow check.
static int run_estimate(echo_ctx *c, int policy) {
  const GraphBuild &B = c->gb;
  const int32_t S = c->S, G = (int32_t)B.sigs.size();
  c->state = 2;
  echo::ScenParams p{c->prm, c->prm + S, c->prm + 2 * (size_t)S, c->prm + 3 * (size_t)S,
                     c->prm + 4 * (size_t)S, c->prm + 5 * (size_t)S};
  CK(cudaMemsetAsync(c->status, 0, sizeof(int32_t), c->stream), "memset");
  CK(cudaMemsetAsync(c->comm_sum, 0, S * sizeof(double), c->stream), "memset");
  CK(timed(c, "cc_estimate", [&] {
       return echo::launch_cc_estimate(c->sigs, G, p, S, c->tbl, c->sig_count, c->cc_ns, c->cc_dur,
                                       c->comm_sum, c->status, c->cc_model, policy, c->stream);
     }), "cc_estimate launch");
  CK(timed(c, "cc_scatter", [&] {
       return echo::launch_cc_scatter(c->comm_node, c->comm_sig, (int64_t)B.comm_node.size(), c->cc_dur, S,
                                      c->lay, c->dur, c->stream);
     }), "cc_scatter launch");
  std::vector<double> comm(S, 0.0);
  CK(cudaMemcpyAsync(comm.data(), c->comm_sum, S * sizeof(double), cudaMemcpyDeviceToHost, c->stream), "readback");
  int32_t st = 0;
  int rc;
  if ((rc = sync_status(c, &st))) return rc;
  if (st == echo::kDevCcOverflow) return set_err(c, ECHO_E_OVERFLOW, "a collective's estimated time is not below 2^61 ns");
  // every finish time is at most the sum of all (slowed) durations of its scenario
  for (int32_t s = 0; s < S; ++s) {
    double bound = c->h_sums[s] * c->h_maxsf[s] + comm[s] + (double)B.V + 1.0;
    if (!(bound < 2305843009213693952.0))
      return set_err(c, ECHO_E_OVERFLOW, "scenario " + std::to_string(s) + ": total duration could overflow int64");
  }
  c->est_policy = policy;
  c->state = 3;
  return ECHO_OK;
}

int echo_estimate_collectives(echo_ctx *c) {
  int rc = check_ctx(c);
  if (rc) return rc;
  if (c->state < 2) return set_err(c, ECHO_E_STATE, "load scenarios first");
  return run_estimate(c, ECHO_AR_PER_OP);
}

int echo_compose(echo_ctx *c, const echo_compose_opts *opts) {
  int rc = check_ctx(c);
  if (rc) return rc;
  if (c->state < 3) return set_err(c, ECHO_E_STATE, "estimate the collectives first");
  int32_t refine = opts ? opts->refine_passes : 1;
  if (refine < 0 || refine > 8) return set_err(c, ECHO_E_INVALID_ARG, "refine_passes outside [0, 8]");
  const int32_t model = opts ? opts->overlap_model : ECHO_OVERLAP_WHOLE;
  if (model != ECHO_OVERLAP_WHOLE && model != ECHO_OVERLAP_PROPORTIONAL)
    return set_err(c, ECHO_E_INVALID_ARG, "unknown overlap model");
  const int32_t civ = opts ? opts->comm_interval : ECHO_COMM_EXECUTION;
  if (civ != ECHO_COMM_EXECUTION && civ != ECHO_COMM_LAUNCH)
    return set_err(c, ECHO_E_INVALID_ARG, "unknown comm interval");
  const int32_t policy = opts ? opts->ar_algo_policy : ECHO_AR_PER_OP;
  if (policy < ECHO_AR_PER_OP || policy > ECHO_AR_AUTO)
    return set_err(c, ECHO_E_INVALID_ARG, "unknown all-reduce policy");
  if (policy != c->est_policy && (rc = run_estimate(c, policy))) return rc;
  const char *dbg_env = std::getenv("ECHO_DEBUG_BOUNDS");
  const int32_t dbg = (opts && opts->debug_bounds) || (dbg_env && std::atoi(dbg_env) != 0) ? 1 : 0;
  const GraphBuild &B = c->gb;
  // the pipelined and dataflow kernels read the validator's durations of the
  // candidates (compact rows); the others compose from a full matrix built for them
  const bool ring = c->use_df || (c->plan.ok && c->plan.pipelined && (c->kernel_choice == 0 || c->kernel_choice == 3));
  if (refine > 1 && !c->cd[1]) {
    if ((rc = dalloc(c, c->scen_allocs, &c->cd[1], c->cd_elems))) return rc;
    CK(cudaMemsetAsync(c->cd[1], 0, c->cd_elems * sizeof(int64_t), c->stream), "memset");
  }
  if (refine > 0 && !ring && !c->deff) {
    if ((rc = dalloc(c, c->scen_allocs, &c->deff, c->scen_vs))) return rc;
  }
  c->state = 3;
  // the inputs of a validator pass, kept to recompute its decisions on demand
  // (echo_read_overlap runs the overlap test on them again)
  auto overlap_args = [&](const int64_t *f_prev, const int64_t *cd_used, int64_t *cd_next) {
    echo::OverlapArgs o{};
    o.lay = c->lay;
    o.lay_c = c->lay_c;
    o.S = c->S;
    o.n_streams = B.NS;
    o.n_ranks = B.R;
    {  // pieces of each rank's list: enough warps for about sixteen waves (16 warps
       // per SM; shorter pieces even out the last wave: 9.27 -> 8.79 ms on the
       // 1024-rank workload, 1.24 -> 1.09 ms on GPT-175B against four waves), each
       // piece at least 64 candidates long
      const int64_t base = (int64_t)B.R * ((c->S + 31) / 32), want = 16 * 16 * (int64_t)c->sms;
      const int64_t per_rank = B.n_cand / std::max<int32_t>(B.R, 1);
      o.parts = (int32_t)std::max<int64_t>(1, std::min((want + base - 1) / base, per_rank / 64));
    }
    o.cand_kcl = c->cand_kcl;
    o.cand_off = c->cand_off;
    o.cand_ops = c->cand_ops;
    o.cand_cidx = c->cand_cidx;
    o.n_cq = B.n_cq;
    o.cq_off = c->cq_off;
    o.cq_ops = c->cq_ops;
    o.lq_off = civ == ECHO_COMM_LAUNCH ? c->lq_off : nullptr;
    o.lq_ops = c->lq_ops;
    o.kcl = c->kcl;
    o.f = f_prev;
    o.dur = c->dur;
    o.cd_used = cd_used;
    o.sf = c->sf;
    o.model = model;
    o.cd_next = cd_next;
    o.ov = nullptr;  // the decisions are recomputed on demand by echo_read_overlap
    o.n_kclass = c->C;
    o.dbg = dbg;
    o.status = c->status;
    return o;
  };
  // one composition with durations `d` (and, for the pipelined and dataflow
  // kernels, the candidates' durations `cdur`) into `f`
  // (final_pass: the readback reads every finish of this composition)
  auto compose_pass = [&](const int64_t *d, const int64_t *cdur, int64_t *f, bool adjusted,
                          bool final_pass) -> cudaError_t {
    const char *name = adjusted ? "compose_adjusted" : "compose";
    if (c->use_df) {
      echo::DataflowArgs a{};
      a.S = c->S;
      a.G = (c->S + 31) / 32;
      a.R = B.R;
      a.n_streams = B.NS;
      a.V = B.V;
      a.n_cand = B.n_cand;
      a.n_slots = std::max<int64_t>(B.df_slots, 1);
      a.n_exports = std::max<int64_t>(B.df_exports, 1);
      a.off = c->df_off;
      a.rec = c->df_rec;
      a.opnd = c->df_opnd;
      a.dur = d;
      a.cdur = cdur;
      a.f = f;
      a.part = c->df_part;
      a.xval = c->df_xval;
      // tags run 1..7; before they start over, every word is zeroed so that none
      // written (or left unwritten by an aborted launch) carries a current tag
      cudaError_t err;
      if (++c->df_epoch > 7) {
        c->df_epoch = 1;
        if ((err = cudaMemsetAsync(c->df_part, 0, c->df_part_elems * sizeof(uint64_t), c->stream)) != cudaSuccess ||
            (err = cudaMemsetAsync(c->df_xval, 0, c->df_xval_elems * sizeof(uint64_t), c->stream)) != cudaSuccess)
          return err;
      }
      a.epoch = c->df_epoch;
      a.abort_flag = c->df_abort;
      a.makespan = c->mk;
      a.status = c->status;
      a.wait_limit_cycles = c->wait_limit_cycles;
      a.skip_slot = c->skip_level;
      a.n_opnd = (int64_t)B.df_opnd.size();
      a.wpb = B.df_wpb;
      a.dbg = dbg;
      if ((err = cudaMemsetAsync(c->mk, 0, (size_t)c->S * sizeof(int64_t), c->stream)) != cudaSuccess ||
          (err = cudaMemsetAsync(c->df_abort, 0, sizeof(int32_t), c->stream)) != cudaSuccess)
        return err;
      return timed(c, name, [&] { return echo::launch_compose_dataflow(a, c->stream); });
    }
    if (c->plan.ok && c->kernel_choice != 1) {
      echo::StagedArgs a{};
      a.S = c->S;
      a.L = (int32_t)c->steps.L;
      a.n_rows = (uint32_t)B.V;
      a.n_words = c->rec_words;
      a.vlog2 = c->plan.vring_log2;
      a.dlog2 = c->plan.dring_log2;
      a.rlog2 = c->plan.rring_log2;
      a.clog2 = c->plan.cring_log2;
      a.d_rows = (uint32_t)1 << c->plan.dring_log2;
      a.c_rows = (uint32_t)1 << c->plan.cring_log2;
      a.meta = c->d_meta;
      a.recs = c->d_recs;
      a.dur = d;
      a.cdur = cdur;
      a.n_cand = (uint32_t)B.n_cand;
      a.f = f;
      a.makespan = c->mk;
      a.status = c->status;
      a.wait_limit_cycles = c->wait_limit_cycles;
      a.skip_level = c->skip_level;
      a.store_all = final_pass;
      a.dbg = dbg;
      const bool pipe = c->plan.pipelined && (c->kernel_choice == 0 || c->kernel_choice == 3);
      if (pipe) {
        a.d_rows = cdur ? c->plan.pipe_drows_c : c->plan.pipe_drows;
        a.c_rows = cdur ? c->plan.pipe_crows : 0;
      }
      if (pipe)
        return timed(c, name, [&] { return echo::launch_compose_pipelined(a, c->sigma, c->plan, c->stream); });
      return timed(c, name, [&] { return echo::launch_compose_staged(a, c->sigma, c->plan, c->stream); });
    }
    echo::ComposeArgs a{};
    a.V = B.V;
    a.lay = c->lay;
    a.S = c->S;
    a.L = (int32_t)B.Ls;
    a.n_queues = B.R * B.NS;
    a.seg_lvl_off = c->seg_lvl_off;
    a.seg_node_off = c->seg_node_off;
    a.nq_off = c->nq_off;
    a.nq = c->nq;
    a.dp_off = c->dp_off;
    a.dp = c->dp;
    a.dur = d;
    a.f = f;
    a.makespan = c->mk;
    a.gfrontier = c->gfrontier;
    a.dbg = dbg;
    a.status = c->status;
    return timed(c, "compose_direct", [&] { return echo::launch_compose(a, c->sigma, c->stream); });
  };
  CK(cudaMemsetAsync(c->status, 0, sizeof(int32_t), c->stream), "memset");
  CK(compose_pass(c->dur, nullptr, c->f[0], false, refine == 0), "compose launch");
  const int64_t *cd_used = nullptr;
  for (int32_t p = 1; p <= refine; ++p) {
    echo::OverlapArgs o = overlap_args(c->f[(p - 1) % 2], cd_used, c->cd[(p - 1) % 2]);
    CK(timed(c, "overlap", [&] { return echo::launch_overlap(o, c->stream); }), "overlap launch");
    if (ring) {
      CK(compose_pass(c->dur, o.cd_next, c->f[p % 2], true, p == refine), "compose launch");
    } else {
      CK(cudaMemcpyAsync(c->deff, c->dur, c->scen_vs * sizeof(int64_t), cudaMemcpyDeviceToDevice, c->stream),
         "duration copy");
      CK(timed(c, "scatter_candidates", [&] {
           return echo::launch_scatter_candidates(c->cand_node, B.n_cand, c->S, c->lay, c->lay_c, o.cd_next, c->deff,
                                                  c->stream);
         }), "scatter launch");
      CK(compose_pass(c->deff, nullptr, c->f[p % 2], true, p == refine), "compose launch");
    }
    cd_used = o.cd_next;
    c->last_ov = o;
  }
  c->final_f = refine % 2;
  c->final_cd = cd_used;
  c->have_ov = refine > 0;
  c->state = 4;
  return ECHO_OK;
}

// Device-side failures of the last composition (a bounded wait that gave up).
static int composition_status(echo_ctx *c) {
  int32_t st = 0;
  int rc = sync_status(c, &st);
  if (rc) return rc;
  if (st == echo::kDevTimeout) {
    if (c->use_df) {  // words a warp never wrote must not carry a later launch's tag
      cudaError_t e = cudaMemsetAsync(c->df_part, 0, c->df_part_elems * sizeof(uint64_t), c->stream);
      if (e == cudaSuccess) e = cudaMemsetAsync(c->df_xval, 0, c->df_xval_elems * sizeof(uint64_t), c->stream);
      if (e == cudaSuccess) e = cudaStreamSynchronize(c->stream);
      if (e != cudaSuccess) {
        // the words may still hold stale tags: drop the scenario buffers, so that
        // the next echo_load_scenarios allocates and zeroes fresh ones
        (void)cudaGetLastError();
        free_all(c->scen_allocs);
        c->scen_vs = 0;
        c->state = 1;
        return cuda_fail(c, e, "clearing the dataflow words after a timeout");
      }
    }
    return set_err(c, ECHO_E_TIMEOUT, "a device-side wait of the composer gave up");
  }
  if (st == echo::kDevBounds) return set_err(c, ECHO_E_BOUNDS, "a debug-bounds index check failed on the device");
  return ECHO_OK;
}

static int read_range_check(echo_ctx *c, int64_t op0, int64_t op1, int need_state) {
  if (c->state < need_state) return set_err(c, ECHO_E_STATE, "nothing to read yet");
  if (op0 < 0 || op1 < op0 || op1 > c->gb.V_ext) return set_err(c, ECHO_E_INVALID_ARG, "op range out of bounds");
  return ECHO_OK;
}

int echo_read_times(echo_ctx *c, int64_t op0, int64_t op1, int32_t s0, int32_t s1, int64_t *start,
                    int64_t *finish) {
  int rc = check_ctx(c);
  if (rc) return rc;
  if ((rc = read_range_check(c, op0, op1, 4))) return rc;
  if (s0 < 0 || s1 > c->S || s1 < s0 || (s1 == s0 && op1 > op0))
    return set_err(c, ECHO_E_INVALID_ARG, "scenario range out of bounds");
  if ((rc = composition_status(c))) return rc;
  const int32_t Sr = s1 - s0;
  if (Sr == 0) return ECHO_OK;
  const int64_t rows_per = std::max<int64_t>(1, (int64_t)(64 << 20) / Sr);
  if ((rc = stage_reserve(c, (size_t)std::min<int64_t>(rows_per, std::max<int64_t>(op1 - op0, 1)) * Sr * 16)))
    return rc;
  for (int64_t a = op0; a < op1; a += rows_per) {
    int64_t b = std::min(op1, a + rows_per);
    int64_t n = (b - a) * Sr;
    int64_t *ds = static_cast<int64_t *>(c->stage);
    int64_t *df = ds + n;
    CK(timed(c, "readback", [&] {
         return echo::launch_readback(c->ext2int, a, b, s0, s1, c->lay, c->f[c->final_f], c->dur, c->cidx, c->lay_c,
                                      c->final_cd, start ? ds : nullptr, finish ? df : nullptr, c->stream);
       }), "readback launch");
    if (start)
      CK(cudaMemcpyAsync(start + (a - op0) * Sr, ds, n * sizeof(int64_t), cudaMemcpyDefault, c->stream), "copy out");
    if (finish)
      CK(cudaMemcpyAsync(finish + (a - op0) * Sr, df, n * sizeof(int64_t), cudaMemcpyDefault, c->stream), "copy out");
    CK(cudaStreamSynchronize(c->stream), "readback");
  }
  return ECHO_OK;
}

int echo_read_makespan(echo_ctx *c, int64_t *out) {
  int rc = check_ctx(c);
  if (rc) return rc;
  if (!out) return set_err(c, ECHO_E_INVALID_ARG, "output is NULL");
  if (c->state < 4) return set_err(c, ECHO_E_STATE, "compose first");
  if ((rc = composition_status(c))) return rc;
  CK(cudaMemcpyAsync(out, c->mk, c->S * sizeof(int64_t), cudaMemcpyDeviceToHost, c->stream), "D2H");
  CK(cudaStreamSynchronize(c->stream), "makespan readback");
  return ECHO_OK;
}

int echo_read_cc(echo_ctx *c, int64_t op0, int64_t op1, double *out) {
  int rc = check_ctx(c);
  if (rc) return rc;
  if (!out) return set_err(c, ECHO_E_INVALID_ARG, "output is NULL");
  if ((rc = read_range_check(c, op0, op1, 3))) return rc;
  const int32_t S = c->S;
  const int64_t rows_per = std::max<int64_t>(1, (int64_t)(64 << 20) / S);
  if ((rc = stage_reserve(c, (size_t)std::min<int64_t>(rows_per, std::max<int64_t>(op1 - op0, 1)) * S * 16)))
    return rc;
  for (int64_t a = op0; a < op1; a += rows_per) {
    int64_t b = std::min(op1, a + rows_per);
    int64_t n = (b - a) * S;
    double *d = static_cast<double *>(c->stage);
    CK(timed(c, "read_cc", [&] {
         return echo::launch_read_cc(c->ext2int, a, b, S, c->node_sig, c->cc_ns, d, c->stream);
       }), "read_cc launch");
    CK(cudaMemcpyAsync(out + (a - op0) * S, d, n * sizeof(double), cudaMemcpyDeviceToHost, c->stream), "D2H");
    CK(cudaStreamSynchronize(c->stream), "read_cc");
  }
  return ECHO_OK;
}

int echo_read_overlap(echo_ctx *c, int64_t op0, int64_t op1, uint8_t *out) {
  int rc = check_ctx(c);
  if (rc) return rc;
  if (!out) return set_err(c, ECHO_E_INVALID_ARG, "output is NULL");
  if ((rc = read_range_check(c, op0, op1, 4))) return rc;
  const int32_t S = c->S;
  const int64_t rows_per = std::max<int64_t>(1, (int64_t)(64 << 20) / S);
  if ((rc = stage_reserve(c, (size_t)std::min<int64_t>(rows_per, std::max<int64_t>(op1 - op0, 1)) * S * 16)))
    return rc;
  if ((rc = composition_status(c))) return rc;
  const uint8_t *ov = nullptr;
  if (c->have_ov) {
    // the last pass's inputs (its finish times and durations) are still intact:
    // run its overlap test again, keeping only the decisions
    echo::OverlapArgs o = c->last_ov;
    o.cd_next = nullptr;
    o.ov = c->ov;
    CK(timed(c, "overlap", [&] { return echo::launch_overlap(o, c->stream); }), "overlap launch");
    ov = c->ov;
  }
  for (int64_t a = op0; a < op1; a += rows_per) {
    int64_t b = std::min(op1, a + rows_per);
    int64_t n = (b - a) * S;
    uint8_t *d = static_cast<uint8_t *>(c->stage);
    CK(timed(c, "read_overlap", [&] {
         return echo::launch_read_ov(c->ext2int, a, b, S, c->lay, ov, c->cand_flag, d, c->stream);
       }), "read_overlap launch");
    CK(cudaMemcpyAsync(out + (a - op0) * S, d, n, cudaMemcpyDeviceToHost, c->stream), "D2H");
    CK(cudaStreamSynchronize(c->stream), "read_overlap");
  }
  return ECHO_OK;
}

int echo_cc_query(echo_ctx *c, const echo_cc_query_desc *q, double *out_ns) {
  int rc = check_ctx(c);
  if (rc) return rc;
  if (!q || (q->n > 0 && !out_ns)) return set_err(c, ECHO_E_INVALID_ARG, "query descriptor or output is NULL");
  const int64_t n = q->n;
  if (n < 0) return set_err(c, ECHO_E_INVALID_ARG, "negative query count");
  if (n == 0) return ECHO_OK;
  if (!q->cc_type || !q->cc_algo || !q->nbytes || !q->n_ranks || !q->n_nodes)
    return set_err(c, ECHO_E_INVALID_ARG, "query arrays are required");
  if ((rc = check_params(c, n, q->alpha_ns, q->bw_intra, q->lat_intra, q->bw_inter, q->lat_inter, q->delta))) return rc;
  ChunkTable tbl;
  if ((rc = make_table(c, q->n_chunk, q->chunk_max_bytes, q->chunk_bytes, &tbl))) return rc;
  std::vector<double> lg(n);
  std::vector<double> lg_cache(4097, -1.0);
  for (int64_t i = 0; i < n; ++i) {
    if (q->cc_type[i] > ECHO_CC_SENDRECV || (q->cc_type[i] == ECHO_CC_ALLREDUCE && q->cc_algo[i] > ECHO_ALGO_AUTO))
      return set_err(c, ECHO_E_INVALID_ARG, "query " + std::to_string(i) + ": bad type or algorithm");
    if (q->nbytes[i] < 0 || q->n_ranks[i] < 1 || q->n_nodes[i] < 1 || q->n_nodes[i] > q->n_ranks[i])
      return set_err(c, ECHO_E_INVALID_ARG, "query " + std::to_string(i) + ": need bytes >= 0 and 1 <= M <= N");
    int32_t m = q->n_nodes[i];
    if (m <= 4096) {
      if (lg_cache[m] < 0) lg_cache[m] = std::log2((double)m);
      lg[i] = lg_cache[m];
    } else {
      lg[i] = std::log2((double)m);
    }
  }
  // one staging allocation holds every query array: 6 param doubles, lg, bytes, N, M, type, algo, out
  const size_t per = 6 * 8 + 8 + 8 + 4 + 4 + 1 + 1 + 8;
  if ((rc = stage_reserve(c, per * (size_t)n + 256))) return rc;
  char *base = static_cast<char *>(c->stage);
  double *dprm = reinterpret_cast<double *>(base);
  double *dlg = dprm + 6 * n;
  int64_t *dbytes = reinterpret_cast<int64_t *>(dlg + n);
  double *dout = reinterpret_cast<double *>(dbytes + n);
  int32_t *dN = reinterpret_cast<int32_t *>(dout + n);
  int32_t *dM = dN + n;
  uint8_t *dtype = reinterpret_cast<uint8_t *>(dM + n);
  uint8_t *dalgo = dtype + n;
  const double *src[6] = {q->alpha_ns, q->bw_intra, q->lat_intra, q->bw_inter, q->lat_inter, q->delta};
  for (int k = 0; k < 6; ++k)
    CK(cudaMemcpyAsync(dprm + (size_t)k * n, src[k], n * sizeof(double), cudaMemcpyHostToDevice, c->stream), "H2D");
  CK(cudaMemcpyAsync(dlg, lg.data(), n * sizeof(double), cudaMemcpyHostToDevice, c->stream), "H2D");
  CK(cudaMemcpyAsync(dbytes, q->nbytes, n * sizeof(int64_t), cudaMemcpyHostToDevice, c->stream), "H2D");
  CK(cudaMemcpyAsync(dN, q->n_ranks, n * sizeof(int32_t), cudaMemcpyHostToDevice, c->stream), "H2D");
  CK(cudaMemcpyAsync(dM, q->n_nodes, n * sizeof(int32_t), cudaMemcpyHostToDevice, c->stream), "H2D");
  CK(cudaMemcpyAsync(dtype, q->cc_type, n, cudaMemcpyHostToDevice, c->stream), "H2D");
  CK(cudaMemcpyAsync(dalgo, q->cc_algo, n, cudaMemcpyHostToDevice, c->stream), "H2D");
  echo::ScenParams p{dprm, dprm + n, dprm + 2 * n, dprm + 3 * n, dprm + 4 * n, dprm + 5 * n};
  CK(timed(c, "cc_query", [&] {
       return echo::launch_cc_query(n, dtype, dalgo, dbytes, dN, dM, dlg, p, tbl, dout, c->stream);
     }), "cc_query launch");
  CK(cudaMemcpyAsync(out_ns, dout, n * sizeof(double), cudaMemcpyDeviceToHost, c->stream), "D2H");
  CK(cudaStreamSynchronize(c->stream), "cc_query");
  return ECHO_OK;
}

int echo_graph_info_get(echo_ctx *c, echo_graph_info *info) {
  if (!c || !info) return ECHO_E_INVALID_ARG;
  if (c->state < 1) return set_err(c, ECHO_E_STATE, "load a graph first");
  const GraphBuild &B = c->gb;
  info->n_ops = B.V_ext;
  info->n_ops_composed = B.V;
  info->replicas_folded = c->fold_active ? 1 : 0;
  info->n_edges = B.E;
  info->n_levels = B.L;
  info->max_width = B.max_width;
  info->n_queue_entries = B.QE;
  info->n_comm_ops = (int64_t)B.comm_node.size();
  info->n_signatures = (int64_t)B.sigs.size();
  info->n_segments = B.n_seg;
  info->n_segment_levels = B.Ls;
  info->n_overlap_candidates = B.cand_off.empty() ? 0 : B.cand_off.back();
  info->n_validator_comm_entries = B.cq_off.empty() ? 0 : B.cq_off.back();
  info->n_kept_finishes = B.V;
  if (!c->use_df) {  // segment tails and the ops whose finish the validator reads
    int64_t n = 0;
    for (int64_t t = 0; t < B.n_seg; ++t)
      for (int64_t v = B.seg_node_off[t]; v < B.seg_node_off[t + 1]; ++v)
        n += (v + 1 == B.seg_node_off[t + 1]) || B.keep[v];
    info->n_kept_finishes = n;
  }
  info->n_ranks = B.R;
  info->n_streams = B.NS;
  info->sigma = c->sigma;
  return ECHO_OK;
}

int echo_set_cc_model(echo_ctx *c, int model) {
  int rc = check_ctx(c);
  if (rc) return rc;
  if (model != ECHO_CC_MODEL_WHITEBOX && model != ECHO_CC_MODEL_ALPHA_BETA)
    return set_err(c, ECHO_E_INVALID_ARG, "unknown collective cost model");
  c->cc_model = model;
  if (c->state > 2) c->state = 2;  // the estimates must be made again
  return ECHO_OK;
}

int echo_set_profiling(echo_ctx *c, int enable) {
  if (!c) return ECHO_E_INVALID_ARG;
  c->prof = enable != 0;
  return ECHO_OK;
}

int echo_read_profile(echo_ctx *c, echo_kernel_stat *out, int cap, int *n) {
  int rc = check_ctx(c);
  if (rc) return rc;
  if (!n || (cap > 0 && !out)) return set_err(c, ECHO_E_INVALID_ARG, "output is NULL");
  CK(cudaStreamSynchronize(c->stream), "profile sync");
  std::vector<std::string> names;
  std::vector<std::pair<int64_t, double>> acc;
  for (auto &r : c->recs) {
    float ms = 0.f;
    cudaEventElapsedTime(&ms, r.second.first, r.second.second);
    size_t k = std::find(names.begin(), names.end(), r.first) - names.begin();
    if (k == names.size()) {
      names.push_back(r.first);
      acc.push_back({0, 0.0});
    }
    acc[k].first++;
    acc[k].second += ms;
    c->ev_pool.push_back(r.second.first);
    c->ev_pool.push_back(r.second.second);
  }
  c->recs.clear();
  int m = 0;
  for (size_t k = 0; k < names.size() && m < cap; ++k, ++m) {
    std::snprintf(out[m].name, sizeof out[m].name, "%s", names[k].c_str());
    out[m].launches = acc[k].first;
    out[m].total_ms = acc[k].second;
  }
  *n = m;
  return ECHO_OK;
}

}  // extern "C"
