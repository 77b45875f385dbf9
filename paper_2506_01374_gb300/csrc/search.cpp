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
//
// Optional learned surrogate (opts.surrogate = 1). Sec. 3.2 scores rollouts
// with a learned, hardware-informed surrogate f-hat instead of running them,
// and the cost model screens proposed transformations before they join the
// tree, pruning low-value ones (App. "LLM proposal validity"). Here f-hat is
// learned online from the measurements the search consumes: a ridge
// regression of log device time on one-hot features of the knob values
// (each knob's value, and the value pairs of knob pairs that interact in
// the kernels), one model per op stage when the measurements carry per-stage
// times (the op time is then the sum of the stage predictions), else one
// model of the op time. Once fitted (>= kMinFit samples), a rollout program
// that was not measured is scored as reward = t(P0) / f-hat(P_sim) and only
// expanded nodes are measured; with opts.screen = k > 1, an expansion draws
// up to k * B distinct legal proposals and keeps the B with the lowest
// predicted time (ties in draw order).
#include <algorithm>
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
  uint64_t sim_hash = 0;  // program whose measurement (or prediction) is this node's reward
  const rc_schedule_s* sim_sched = nullptr;
};

struct Pending {
  const rc_schedule_s* sched;
  uint64_t hash;
};

// Knob fields of rc_knobs in declaration order, and the pairs whose joint
// value gets its own feature.
enum { F_TM, F_TN, F_TK, F_UN, F_ST, F_SK, F_RA, F_GR, F_PE, F_FU, F_LA, F_VE, F_LO, F_COUNT };
int32_t knob_field(const rc_knobs& k, int f) {
  const int32_t v[F_COUNT] = {k.tile_m, k.tile_n, k.tile_k,     k.unroll, k.stages, k.split_k, k.raster,
                              k.group,  k.persistent, k.fuse, k.layout, k.vec,    k.location};
  return v[f];
}
constexpr int kPairs[][2] = {{F_TM, F_TN}, {F_TN, F_TK}, {F_TN, F_ST}, {F_TK, F_ST}, {F_TM, F_ST},
                             {F_TM, F_PE}, {F_TN, F_PE}, {F_TN, F_SK}, {F_PE, F_UN}, {F_TM, F_UN},
                             {F_TN, F_UN}, {F_PE, F_LO}, {F_TM, F_FU}, {F_RA, F_GR}};
constexpr int kNumPairs = sizeof(kPairs) / sizeof(kPairs[0]);
constexpr double kRidge = 1.0;        // penalty of every feature weight
constexpr double kRidgeBias = 1e-6;   // (almost) free intercept
constexpr int kMinFit = 24;           // samples before the surrogate is used

// Ridge regression y ~ w . x over sparse 0/1 features (feature 0 = intercept).
struct Ridge {
  std::unordered_map<uint64_t, int> index;  // feature key -> column
  std::vector<std::vector<int>> rows;       // training rows (active columns)
  std::vector<double> ys;
  std::vector<double> w;                    // fitted weights (size = columns at fit time)

  static uint64_t key(int model, int kind, int32_t a, int32_t b) {
    return mix64(((uint64_t)(uint32_t)model << 48) ^ ((uint64_t)(uint32_t)kind << 40) ^
                 ((uint64_t)(uint32_t)a << 20) ^ (uint64_t)(uint32_t)b ^ 0x5DEECE66Dull);
  }
  // Active columns of a knob vector (stage g's features; the intercept,
  // column 0, is not included); unseen features get a column when add =
  // true, else are skipped.
  void features(int g, const rc_knobs& k, bool add, std::vector<int>& f) {
    auto col = [&](uint64_t kk) {
      auto it = index.find(kk);
      if (it != index.end()) {
        f.push_back(it->second);
      } else if (add) {
        const int c = (int)index.size() + 1;
        index.emplace(kk, c);
        f.push_back(c);
      }
    };
    for (int i = 0; i < F_COUNT; ++i) col(key(g, i, knob_field(k, i), 0));
    for (int p = 0; p < kNumPairs; ++p)
      col(key(g, 100 + p, knob_field(k, kPairs[p][0]), knob_field(k, kPairs[p][1])));
  }
  // Row of the knob vectors ks[0..n) (stage g0 + i for ks[i]): intercept + their features.
  std::vector<int> row(const rc_knobs* ks, int n, int g0, bool add) {
    std::vector<int> f{0};
    for (int i = 0; i < n; ++i) features(g0 + i, ks[i], add, f);
    return f;
  }
  void add(const rc_knobs* ks, int n, int g0, double y) {
    rows.push_back(row(ks, n, g0, true));
    ys.push_back(y);
  }
  // Solve (X^T X + diag(lambda)) w = X^T y by Cholesky.
  void fit() {
    const size_t F = index.size() + 1;
    std::vector<double> A(F * F, 0.0), b(F, 0.0);
    for (size_t r = 0; r < rows.size(); ++r) {
      for (int i : rows[r]) {
        b[i] += ys[r];
        for (int j : rows[r]) A[(size_t)i * F + j] += 1.0;
      }
    }
    A[0] += kRidgeBias;
    for (size_t i = 1; i < F; ++i) A[i * F + i] += kRidge;
    for (size_t j = 0; j < F; ++j) {  // A = L L^T, L in the lower triangle
      double d = A[j * F + j];
      for (size_t k = 0; k < j; ++k) d -= A[j * F + k] * A[j * F + k];
      const double ljj = std::sqrt(d);
      A[j * F + j] = ljj;
      for (size_t i = j + 1; i < F; ++i) {
        double v = A[i * F + j];
        for (size_t k = 0; k < j; ++k) v -= A[i * F + k] * A[j * F + k];
        A[i * F + j] = v / ljj;
      }
    }
    std::vector<double> z(F);
    for (size_t i = 0; i < F; ++i) {  // L z = b
      double v = b[i];
      for (size_t k = 0; k < i; ++k) v -= A[i * F + k] * z[k];
      z[i] = v / A[i * F + i];
    }
    w.assign(F, 0.0);
    for (size_t i = F; i-- > 0;) {  // L^T w = z
      double v = z[i];
      for (size_t k = i + 1; k < F; ++k) v -= A[k * F + i] * w[k];
      w[i] = v / A[i * F + i];
    }
  }
  double predict(const rc_knobs* ks, int n, int g0) {
    double y = 0.0;
    for (int c : row(ks, n, g0, false))
      if ((size_t)c < w.size()) y += w[c];
    return y;
  }
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
  double t0_ms = 0.0;                                    // objective of the root program
  bool root_measured = false;
  int64_t iterations = 0;
  uint64_t best_hash = 0;
  double best_reward = -1.0;
  const rc_schedule_s* best_sched = nullptr;
  // learned surrogate: one ridge model per stage (per-stage times) or one for the op
  std::vector<Ridge> models;
  int per_stage = -1;  // -1 undecided, 1 per-stage models, 0 one op model
  size_t n_train = 0;     // measurements in the training set
  size_t n_fit = 0;       // measurements of the current fit
  int64_t predicted = 0;  // rollout rewards taken from the surrogate

  void train(const rc_schedule_s* sc, const rc_measurement& m) {
    if (!o.surrogate || m.status != RC_OK || !(m.ms_median > 0)) return;
    const int S = sc->n_stages;
    bool stages_ok = S > 1 && m.n_stages == S;
    for (int g = 0; stages_ok && g < S; ++g) stages_ok = m.stage_ms[g] > 0;
    if (per_stage < 0) {
      per_stage = stages_ok ? 1 : 0;
      models.resize(per_stage ? S : 1);
    }
    if (per_stage == 1 && !stages_ok) return;  // keep the training set homogeneous
    if (per_stage == 1) {
      for (int g = 0; g < S; ++g) models[g].add(&sc->k[g], 1, g, std::log(m.stage_ms[g]));
    } else {
      models[0].add(sc->k, S, 0, std::log(m.ms_median));  // features of stage g keyed by g
    }
    ++n_train;
  }
  bool surrogate_ready() const { return o.surrogate && n_fit >= (size_t)kMinFit; }
  void maybe_refit() {
    if (!o.surrogate || n_train < (size_t)kMinFit) return;
    if (n_fit == 0 || n_train - n_fit >= std::max<size_t>(4, n_fit / 8)) {
      for (Ridge& r : models) r.fit();
      n_fit = n_train;
    }
  }
  bool in_task(int g) const { return o.stage_mask == 0 || (g < 32 && ((o.stage_mask >> g) & 1u)); }
  // The objective of a measurement: the op's median time, or with a stage
  // mask the sum of the selected stages' medians.
  double objective(const rc_measurement& m) const {
    if (!o.stage_mask || m.n_stages != nodes[0].sched->n_stages) return m.ms_median;
    double t = 0.0;
    for (int g = 0; g < m.n_stages; ++g) {
      if (!in_task(g)) continue;
      if (!(m.stage_ms[g] > 0)) return m.ms_median;
      t += m.stage_ms[g];
    }
    return t;
  }
  // Predicted objective (ms) of a schedule.
  double predict_ms(const rc_schedule_s* sc) {
    const int S = sc->n_stages;
    if (per_stage == 1) {
      double t = 0.0;
      for (int g = 0; g < S; ++g)
        if (in_task(g)) t += std::exp(models[g].predict(&sc->k[g], 1, g));
      return t;
    }
    return std::exp(models[0].predict(sc->k, S, 0));
  }

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

  // Rollout reward of node n: the measured speedup of its rollout program,
  // else (surrogate mode) t(P0) / f-hat(P_sim).
  double node_reward(int64_t n) {
    const Node& nd = nodes[n];
    auto it = reward.find(nd.sim_hash);
    if (it != reward.end()) return it->second;
    ++predicted;
    const double t = predict_ms(nd.sim_sched);
    return t > 0 ? t0_ms / t : 0.0;
  }

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
  o.surrogate = 0;
  o.screen = 1;
  o.stage_mask = 0;
  o.root = nullptr;
  if (opts) {
    o.seed = opts->seed;
    if (opts->c > 0) o.c = opts->c;
    if (opts->branching > 0) o.branching = opts->branching;
    if (opts->horizon > 0) o.horizon = opts->horizon;
    if (opts->rollout >= 0) o.rollout = opts->rollout;
    if (opts->max_tries > 0) o.max_tries = opts->max_tries;
    if (opts->surrogate < 0 || opts->surrogate > 1)
      return rc_fail(RC_ERR_INVALID_ARG, "rc_search_create: surrogate must be 0 or 1");
    o.surrogate = opts->surrogate;
    if (opts->screen > 1) o.screen = opts->screen;
    const int S = op->n_stages;
    if (S < 32 && (opts->stage_mask >> S) != 0)
      return rc_fail(RC_ERR_INVALID_ARG, "rc_search_create: stage_mask names a stage the op does not have");
    o.stage_mask = opts->stage_mask;
    if (opts->root && (opts->root->op_kind != op->d.kind || opts->root->n_stages != S))
      return rc_fail(RC_ERR_INVALID_ARG, "rc_search_create: root is a schedule of another op");
    o.root = opts->root;
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
  if (o.stage_mask) {  // one task: only the selected stages' transformations
    std::vector<rc_transform> keep;
    for (const rc_transform& t : s->space)
      if (t.stage < 32 && ((o.stage_mask >> t.stage) & 1u)) keep.push_back(t);
    s->space.swap(keep);
  }
  rc_schedule* root = nullptr;
  rc_status st = rc_schedule_apply(op, o.root, nullptr, 0, &root);
  if (st != RC_OK) {
    delete s;
    return st;
  }
  s->o.root = nullptr;  // copied above; the caller's schedule is not referenced afterwards
  Node r;
  r.sched.reset(root);
  r.hash = rc_schedule_hash(root);
  r.parent = -1;
  r.depth = 0;
  r.sim_hash = r.hash;
  r.sim_sched = r.sched.get();
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
      if (m.status != RC_OK || !(m.ms_median > 0) || !(s->objective(m) > 0))
        return rc_fail(RC_ERR_INVALID_ARG, "rc_search_step: the root program must measure successfully");
      s->t0_ms = s->objective(m);
      s->root_measured = true;
    }
    const double r = (m.status == RC_OK && m.ms_median > 0) ? s->t0_ms / s->objective(m) : 0.0;
    s->reward[p.hash] = r;
    s->meas[p.hash] = m;
    s->meas[p.hash].sched_hash = p.hash;
    s->train(p.sched, m);
    if (r > s->best_reward) {
      s->best_reward = r;
      s->best_hash = p.hash;
      s->best_sched = p.sched;
    }
  }
  s->pending.clear();
  s->maybe_refit();
  // 2) backpropagate the rewards of nodes whose rollout program is now measured (or predicted)
  for (int64_t n : s->awaiting) s->backprop(n, s->node_reward(n));
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
      // proposals: B distinct legal new programs, or with screening up to
      // screen * B of them of which the B with the lowest predicted time stay
      const bool screen = s->surrogate_ready() && s->o.screen > 1;
      const int want = screen ? s->o.branching * s->o.screen : s->o.branching;
      std::vector<std::unique_ptr<rc_schedule_s>> props;
      std::vector<uint64_t> prop_hash;
      for (int tries = 0; (int)props.size() < want && tries < s->o.max_tries * (screen ? s->o.screen : 1) &&
                          !s->space.empty();
           ++tries) {
        const rc_transform& t = s->space[s->index(s->space.size())];
        auto c = s->apply(s->nodes[leaf].sched.get(), t);
        if (!c) continue;
        const uint64_t h = rc_schedule_hash(c.get());
        if (s->in_tree.count(h)) continue;  // keep the tree acyclic (Sec. 3.2)
        bool dup = false;
        for (uint64_t ph : prop_hash) dup = dup || ph == h;
        if (dup) continue;
        props.push_back(std::move(c));
        prop_hash.push_back(h);
      }
      std::vector<size_t> keep(props.size());
      for (size_t i = 0; i < keep.size(); ++i) keep[i] = i;
      if (screen && (int)props.size() > s->o.branching) {
        std::vector<double> pred(props.size());
        for (size_t i = 0; i < props.size(); ++i) pred[i] = s->predict_ms(props[i].get());
        std::stable_sort(keep.begin(), keep.end(), [&](size_t a, size_t b) { return pred[a] < pred[b]; });
        keep.resize(s->o.branching);
        std::sort(keep.begin(), keep.end());  // children in draw order
      }
      for (size_t i : keep) {
        std::unique_ptr<rc_schedule_s> c = std::move(props[i]);
        const uint64_t h = prop_hash[i];
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
        if (sh == s->nodes[id].hash) {
          s->nodes[id].sim_sched = s->nodes[id].sched.get();
        } else {
          auto it = s->in_tree.find(sh);
          const rc_schedule_s* sim =
              it != s->in_tree.end() ? s->nodes[it->second].sched.get() : s->own(std::move(cur));
          s->nodes[id].sim_sched = sim;
          // with a fitted surrogate the rollout program is predicted, not measured
          if (!s->surrogate_ready()) request(sim, sh);
        }
        s->awaiting.push_back(id);
      }
      for (int64_t id : kids) s->refresh_open(id);
      s->refresh_open(leaf);
      ++s->iterations;
      if (s->pending.empty()) {
        // every program of this expansion was measured before (or is predicted): back up now
        for (int64_t n : s->awaiting) s->backprop(n, s->node_reward(n));
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
  st->model_samples = (int64_t)s->n_fit;
  int64_t cols = 0;
  for (const Ridge& r : s->models) cols += (int64_t)r.w.size();
  st->model_features = cols;
  st->predicted = s->predicted;
  return RC_OK;
}

extern "C" rc_status rc_search_predict(rc_search* s, const rc_schedule* sched, double* ms) {
  if (!s || !sched || !ms) return rc_fail(RC_ERR_INVALID_ARG, "rc_search_predict: NULL argument");
  if (sched->op_kind != s->op->d.kind || sched->n_stages != s->nodes[0].sched->n_stages)
    return rc_fail(RC_ERR_INVALID_ARG, "rc_search_predict: schedule of another op");
  if (!s->o.surrogate || s->n_fit == 0)
    return rc_fail(RC_ERR_INVALID_ARG, "rc_search_predict: no fitted surrogate (surrogate off or too few samples)");
  *ms = s->predict_ms(sched);
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
