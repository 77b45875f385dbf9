// LLM-free Monte Carlo tree search over an op's schedule space.
//
// Sec. 3.2 of the paper: nodes are programs and edges transformations;
// selection descends by UCT(P_i) = Q(P_i)/N(P_i) + c sqrt(ln N(parent)/N(P_i));
// expansion applies proposed transformations to the selected leaf and does
// not add a program already in the tree; a rollout applies q random legal
// transformations to obtain P_sim whose objective is the new node's reward;
// backpropagation adds the reward to Q and 1 to N of every ancestor. The
// proposal engine is the paper's non-LLM policy (App. G): a transformation
// drawn uniformly from the valid set. B = 2 and c = sqrt(2) (Sec. 4.1). The
// objective is measured on the device (speedup t(P0)/t(P)), not predicted.
//
// Readings where the paper is silent:
//  * UCT with N = 0 is undefined: unvisited children are taken first, in
//    child order; UCT ties go to the lower child index.
//  * Horizon T (Eq. 1) defaults to 8 and rollout length q to 2.
//  * Each new child and its rollout program are measured (a "sample" is a
//    distinct measured program); measurements are cached by schedule.
//  * Random draws come from a counter-based splitmix64 stream:
//    draw(n) = mix(key + (n + 1) * 0x9E3779B97F4A7C15), key = mix(seed), and
//    an index in [0, m) is ((draw >> 11) * m) >> 53.
#include <cmath>
#include <cstring>
#include <memory>
#include <new>
#include <unordered_map>
#include <vector>

#include "rc_internal.h"

namespace {

uint64_t mix64(uint64_t z) {
  z ^= z >> 30;
  z *= 0xBF58476D1CE4E5B9ull;
  z ^= z >> 27;
  z *= 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

struct Node {
  std::unique_ptr<rc_schedule_s> sched;
  uint64_t hash;
  int64_t parent;
  int depth;
  std::vector<int64_t> children;
  bool expanded = false;  // expansion was attempted
  bool open = true;       // this node or a descendant can still be expanded
  double Q = 0.0;
  int64_t N = 0;
  uint64_t sim_hash = 0;  // program whose measurement is this node's reward
};

struct Pending {
  const rc_schedule_s* sched;
  uint64_t hash;
};

}  // namespace

struct rc_search_s {
  const rc_op_s* op;
  rc_search_opts o;
  uint64_t key;
  uint64_t ctr = 0;
  std::vector<rc_transform> space;
  std::vector<Node> nodes;
  std::unordered_map<uint64_t, int64_t> in_tree;         // schedule hash -> node
  std::unordered_map<uint64_t, double> reward;           // measured programs
  std::unordered_map<uint64_t, rc_measurement> meas;     // their measurements
  std::vector<std::unique_ptr<rc_schedule_s>> owned;     // schedules handed out
  std::vector<Pending> pending;                          // last batch, in order
  std::vector<int64_t> awaiting;                         // nodes waiting for their reward
  double t0_ms = 0.0;                                    // P0 median time
  bool root_measured = false;
  int64_t iterations = 0;
  uint64_t best_hash = 0;
  double best_reward = -1.0;
  const rc_schedule_s* best_sched = nullptr;

  uint64_t draw() { return mix64(key + (++ctr) * 0x9E3779B97F4A7C15ull); }
  size_t index(size_t m) { return (size_t)(((draw() >> 11) * (unsigned __int128)m) >> 53); }

  // Apply one transformation; nullptr if illegal.
  std::unique_ptr<rc_schedule_s> apply(const rc_schedule_s* s, const rc_transform& t) {
    rc_schedule* out = nullptr;
    if (rc_schedule_apply(op, s, &t, 1, &out) != RC_OK) return nullptr;
    return std::unique_ptr<rc_schedule_s>(out);
  }

  void backprop(int64_t n, double r) {
    for (int64_t a = n; a >= 0; a = nodes[a].parent) {
      nodes[a].Q += r;
      nodes[a].N += 1;
    }
  }

  bool expandable(const Node& nd) const { return !nd.expanded && nd.depth < o.horizon; }

  void refresh_open(int64_t n) {
    for (int64_t a = n; a >= 0; a = nodes[a].parent) {
      Node& nd = nodes[a];
      bool op_ = expandable(nd);
      for (int64_t c : nd.children) op_ = op_ || nodes[c].open;
      if (op_ == nd.open && a != n) break;
      nd.open = op_;
    }
  }

  // UCT descent over open children (Sec. 3.2).
  int64_t select() {
    if (!nodes[0].open) return -1;
    int64_t cur = 0;
    while (!expandable(nodes[cur])) {
      const Node& nd = nodes[cur];
      int64_t best = -1;
      double best_v = -INFINITY;
      for (int64_t c : nd.children) {
        const Node& ch = nodes[c];
        if (!ch.open) continue;
        if (ch.N == 0) {
          best = c;
          break;
        }
        const double v = ch.Q / ch.N + o.c * std::sqrt(std::log((double)nd.N) / ch.N);
        if (v > best_v) {
          best_v = v;
          best = c;
        }
      }
      if (best < 0) return -1;
      cur = best;
    }
    return cur;
  }

  const rc_schedule_s* own(std::unique_ptr<rc_schedule_s> s) {
    owned.push_back(std::move(s));
    return owned.back().get();
  }
};

extern "C" rc_status rc_search_create(const rc_op* op, const rc_search_opts* opts, rc_search** out) {
  if (!op || !out) return rc_fail(RC_ERR_INVALID_ARG, "rc_search_create: NULL argument");
  *out = nullptr;
  rc_search_opts o;
  o.seed = 0;
  o.c = std::sqrt(2.0);
  o.branching = 2;
  o.horizon = 8;
  o.rollout = 2;
  o.max_tries = 64;
  if (opts) {
    o.seed = opts->seed;
    if (opts->c > 0) o.c = opts->c;
    if (opts->branching > 0) o.branching = opts->branching;
    if (opts->horizon > 0) o.horizon = opts->horizon;
    if (opts->rollout >= 0) o.rollout = opts->rollout;
    if (opts->max_tries > 0) o.max_tries = opts->max_tries;
  }
  auto* s = new (std::nothrow) rc_search_s;
  if (!s) return rc_fail(RC_ERR_OOM, "rc_search_create: out of host memory");
  s->op = op;
  s->o = o;
  s->key = mix64(o.seed);
  size_t n = 0;
  rc_transform_space(op, nullptr, 0, &n);
  s->space.resize(n);
  if (n) rc_transform_space(op, s->space.data(), n, &n);
  rc_schedule* root = nullptr;
  rc_status st = rc_schedule_apply(op, nullptr, nullptr, 0, &root);
  if (st != RC_OK) {
    delete s;
    return st;
  }
  Node r;
  r.sched.reset(root);
  r.hash = rc_schedule_hash(root);
  r.parent = -1;
  r.depth = 0;
  r.sim_hash = r.hash;
  s->in_tree[r.hash] = 0;
  s->nodes.push_back(std::move(r));
  *out = s;
  return RC_OK;
}

extern "C" rc_status rc_search_step(rc_search* s, const rc_measurement* results, size_t n_results,
                                    const rc_schedule** next, size_t cap, size_t* n_next) {
  if (!s || !n_next || (n_results && !results) || (cap && !next))
    return rc_fail(RC_ERR_INVALID_ARG, "rc_search_step: NULL argument");
  *n_next = 0;
  if (n_results != s->pending.size())
    return rc_fail(RC_ERR_INVALID_ARG, "rc_search_step: expected %zu results, got %zu",
                   s->pending.size(), n_results);
  // 1) record the measurements of the previous batch
  for (size_t i = 0; i < n_results; ++i) {
    const Pending& p = s->pending[i];
    const rc_measurement& m = results[i];
    if (!s->root_measured) {
      if (m.status != RC_OK || !(m.ms_median > 0))
        return rc_fail(RC_ERR_INVALID_ARG, "rc_search_step: the root program P0 must measure successfully");
      s->t0_ms = m.ms_median;
      s->root_measured = true;
    }
    const double r = (m.status == RC_OK && m.ms_median > 0) ? s->t0_ms / m.ms_median : 0.0;
    s->reward[p.hash] = r;
    s->meas[p.hash] = m;
    s->meas[p.hash].sched_hash = p.hash;
    if (r > s->best_reward) {
      s->best_reward = r;
      s->best_hash = p.hash;
      s->best_sched = p.sched;
    }
  }
  s->pending.clear();
  // 2) backpropagate the rewards of nodes whose rollout program is now measured
  for (int64_t n : s->awaiting) s->backprop(n, s->reward[s->nodes[n].sim_hash]);
  s->awaiting.clear();

  auto request = [&](const rc_schedule_s* sc, uint64_t h) {
    if (s->reward.count(h)) return;
    for (const Pending& p : s->pending)
      if (p.hash == h) return;
    s->pending.push_back({sc, h});
  };

  if (!s->root_measured) {
    const Node& r = s->nodes[0];
    s->pending.push_back({r.sched.get(), r.hash});
    s->awaiting.push_back(0);
  } else {
    // 3) select / expand / rollout until at least one program needs measuring
    for (int guard = 0; guard < 4096 && s->pending.empty(); ++guard) {
      const int64_t leaf = s->select();
      if (leaf < 0) break;
      s->nodes[leaf].expanded = true;
      std::vector<int64_t> kids;
      for (int tries = 0; (int)kids.size() < s->o.branching && tries < s->o.max_tries && !s->space.empty();
           ++tries) {
        const rc_transform& t = s->space[s->index(s->space.size())];
        auto c = s->apply(s->nodes[leaf].sched.get(), t);
        if (!c) continue;
        const uint64_t h = rc_schedule_hash(c.get());
        if (s->in_tree.count(h)) continue;  // keep the tree acyclic (Sec. 3.2)
        Node nd;
        nd.sched = std::move(c);
        nd.hash = h;
        nd.parent = leaf;
        nd.depth = s->nodes[leaf].depth + 1;
        const int64_t id = (int64_t)s->nodes.size();
        s->in_tree[h] = id;
        s->nodes.push_back(std::move(nd));
        s->nodes[leaf].children.push_back(id);
        kids.push_back(id);
      }
      for (int64_t id : kids) {
        // rollout: q random legal transformations from the new node
        std::unique_ptr<rc_schedule_s> cur(new rc_schedule_s(*s->nodes[id].sched));
        for (int q = 0; q < s->o.rollout; ++q) {
          for (int tries = 0; tries < s->o.max_tries && !s->space.empty(); ++tries) {
            auto nx = s->apply(cur.get(), s->space[s->index(s->space.size())]);
            if (nx) {
              cur = std::move(nx);
              break;
            }
          }
        }
        const uint64_t sh = rc_schedule_hash(cur.get());
        s->nodes[id].sim_hash = sh;
        request(s->nodes[id].sched.get(), s->nodes[id].hash);
        if (sh != s->nodes[id].hash) {
          auto it = s->in_tree.find(sh);
          request(it != s->in_tree.end() ? s->nodes[it->second].sched.get() : s->own(std::move(cur)), sh);
        }
        s->awaiting.push_back(id);
      }
      for (int64_t id : kids) s->refresh_open(id);
      s->refresh_open(leaf);
      ++s->iterations;
      if (s->pending.empty()) {
        // every program of this expansion was measured before: back up now
        for (int64_t n : s->awaiting) s->backprop(n, s->reward[s->nodes[n].sim_hash]);
        s->awaiting.clear();
      }
    }
  }
  if (s->pending.empty()) return rc_fail(RC_ERR_EXHAUSTED, "rc_search_step: search space exhausted");
  if (cap < s->pending.size())
    return rc_fail(RC_ERR_INVALID_ARG, "rc_search_step: next[] needs %zu entries", s->pending.size());
  for (size_t i = 0; i < s->pending.size(); ++i) next[i] = s->pending[i].sched;
  *n_next = s->pending.size();
  return RC_OK;
}

extern "C" rc_status rc_search_best(const rc_search* s, const rc_schedule** best, rc_measurement* m) {
  if (!s || !best) return rc_fail(RC_ERR_INVALID_ARG, "rc_search_best: NULL argument");
  if (!s->best_sched) return rc_fail(RC_ERR_INVALID_ARG, "rc_search_best: nothing measured yet");
  *best = s->best_sched;
  if (m) *m = s->meas.at(s->best_hash);
  return RC_OK;
}

extern "C" rc_status rc_search_get_stats(const rc_search* s, rc_search_stats* st) {
  if (!s || !st) return rc_fail(RC_ERR_INVALID_ARG, "rc_search_get_stats: NULL argument");
  st->nodes = (int64_t)s->nodes.size();
  st->samples = (int64_t)s->reward.size();
  st->iterations = s->iterations;
  st->best_reward = s->best_reward;
  return RC_OK;
}

extern "C" rc_status rc_search_node(const rc_search* s, int64_t i, int64_t* parent, double* q, int64_t* n,
                                    uint64_t* sched_hash) {
  if (!s) return rc_fail(RC_ERR_INVALID_ARG, "rc_search_node: NULL search");
  if (i < 0 || i >= (int64_t)s->nodes.size()) return rc_fail(RC_ERR_INVALID_ARG, "rc_search_node: index");
  const Node& nd = s->nodes[i];
  if (parent) *parent = nd.parent;
  if (q) *q = nd.Q;
  if (n) *n = nd.N;
  if (sched_hash) *sched_hash = nd.hash;
  return RC_OK;
}

extern "C" void rc_search_destroy(rc_search* s) { delete s; }
