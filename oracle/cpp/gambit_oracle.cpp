// CPU oracle for the beam-decode hot path of thought-level beam search, in plain C++17.
//
// This is test infrastructure, not the product: only the tests, the smoke check and the
// CPU-baseline legs of the benchmark load it.  It shares no code with the CUDA library.
// Every routine is the plain definition of what the GPU path computes, written for a
// reader to check against the paper, not for speed:
//
//  * decode attention (Section 3.1; Algorithm 1, "Generate"): for each query head h,
//    s_t = scale * q_h . K_t over the beam's whole materialised context, two-pass
//    softmax (max, then sum of exp), o_h = sum_t p_t V_t, all in fp64; query head h
//    reads KV head h / (Hq / Hkv);
//  * the probe sigma(w . h + b) in fp64 and the running mean of Algorithm 1,
//    s_bar <- s_bar + (x - s_bar) / n, in fp32 with the subtraction, division and
//    addition each rounded on its own (this file is compiled with -ffp-contract=off);
//  * the Tournament of Algorithm 1 (Eq. 2: Case 1 under capacity; Eq. 3: Case 2 at
//    capacity, zero-sum) with a stable ranking;
//  * the paged pool: per-slot block tables, page reference counts, lowest-free-page
//    allocation, copy-on-write of a shared partial tail page, and fork without copying
//    (Section 3.1, the paragraph after Eq. 3: a branched child inherits its parent's KV,
//    pruning frees only the blocks nobody else holds);
//  * beam KV materialised by copying: every slot keeps its full K and V arrays and a
//    branched child gets a copy of its parent's arrays.
//
// Readings where the paper is silent, the same as the GPU path's: ties in the ranking keep
// the lower slot first, +0 and -0 tie, a NaN mean ranks after every number; with fan-out f
// each parent gets f - 1 children (the last one the remainder) and the parents are the
// first ceil(K / (f - 1)) eligible survivors in rank order; when the eligible survivors
// cannot supply K children only K_eff = min(K, (f - 1) |B|) traces are pruned; child k
// (children in parent-rank order) takes the k-th smallest freed slot (pruned slots in
// Case 2, vacant slots in Case 1) and inherits the parent's length, running mean and step
// count, with gen = 0 and a fresh lineage id; a step that cannot get all its pages changes
// nothing and reports out of memory; holders of a shared partial tail page decide in slot
// order against the current reference count, so every holder but the last copies.
#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <functional>
#include <map>
#include <queue>
#include <string>
#include <vector>

namespace {

constexpr int kOk = 0, kErrInvalid = 1, kErrOom = 2, kErrState = 4;
constexpr uint32_t kPromptWriter = 0xFFFFFFFFu;

// ---- attention ---------------------------------------------------------------------------

// Softmax weights over L keys for one query: p_t = exp(s_t - max s) / sum_u exp(s_u - max s).
void softmax_weights(const double* q, const double* K, int L, int D, int stride, double scale,
                     std::vector<double>& p) {
  p.resize(L);
  double m = -INFINITY;
  for (int t = 0; t < L; ++t) {
    double s = 0.0;
    for (int d = 0; d < D; ++d) s += q[d] * K[(size_t)t * stride + d];
    p[t] = scale * s;
    m = std::max(m, p[t]);
  }
  double sum = 0.0;
  for (int t = 0; t < L; ++t) {
    p[t] = std::exp(p[t] - m);
    sum += p[t];
  }
  for (int t = 0; t < L; ++t) p[t] /= sum;
}

// ---- tournament --------------------------------------------------------------------------

struct Plan {
  int kase = 0;                            // 0: nothing to do, 1: under capacity, 2: at capacity
  std::vector<int> order;                  // active slots, best first
  std::vector<int> pruned;                 // ascending
  std::vector<std::pair<int, int>> children;  // (child slot, parent slot)
};

// Active slots best first: higher mean first, ties by slot (stable), NaN after every number.
std::vector<int> rank_order(const float* mean, const uint8_t* active, int n) {
  std::vector<int> order;
  for (int s = 0; s < n; ++s)
    if (active[s]) order.push_back(s);
  std::stable_sort(order.begin(), order.end(), [&](int a, int b) {
    const double ma = mean[a], mb = mean[b];
    const bool na = std::isnan(ma), nb = std::isnan(mb);
    if (na || nb) return !na && nb;      // a number before a NaN; two NaNs keep slot order
    return ma > mb;                      // +0 and -0 compare equal and keep slot order
  });
  return order;
}

Plan tournament(const float* mean, const uint8_t* active, const uint8_t* eligible, int n, int capacity, int K,
                int fanout) {
  Plan plan;
  plan.order = rank_order(mean, active, n);
  const int N = (int)plan.order.size();
  if (N == 0) return plan;
  if (N < capacity) {
    // Case 1 (Eq. 2): the top min(C - N, |B|) eligible traces get one child each, in vacant slots.
    plan.kase = 1;
    std::vector<int> B, vacant;
    for (int s : plan.order)
      if (eligible[s]) B.push_back(s);
    for (int s = 0; s < capacity; ++s)
      if (!active[s]) vacant.push_back(s);
    const int m = std::min(capacity - N, (int)B.size());
    for (int k = 0; k < m; ++k) plan.children.push_back({vacant[k], B[k]});
    return plan;
  }
  // Case 2 (Eq. 3), fan-out f: prune the bottom K_eff, the top eligible survivors branch.
  plan.kase = 2;
  K = std::max(0, std::min(K, N));
  std::vector<int> B;
  for (int r = 0; r < N - K; ++r)
    if (eligible[plan.order[r]]) B.push_back(plan.order[r]);
  const long long cap_children = (long long)(fanout - 1) * (long long)B.size();
  const int k_eff = (int)std::min<long long>(K, cap_children);
  if (k_eff == 0) return plan;
  plan.pruned.assign(plan.order.end() - k_eff, plan.order.end());
  std::sort(plan.pruned.begin(), plan.pruned.end());
  for (int k = 0; k < k_eff; ++k) plan.children.push_back({plan.pruned[k], B[k / (fanout - 1)]});
  return plan;
}

// ---- the paged pool --------------------------------------------------------------------------

struct Run {
  uint32_t writer;
  int64_t start, end;
};

struct Pool {
  int64_t num_pages;
  int max_beams, max_pages, P;
  int capacity;
  int status = kOk;
  uint32_t next_lineage = 1;
  std::vector<int64_t> refcnt;
  std::priority_queue<int64_t, std::vector<int64_t>, std::greater<int64_t>> free_pages;  // lowest id first
  std::vector<std::vector<int64_t>> tables;
  // Per-slot state in the dtypes the Python wrapper views directly.
  std::vector<int64_t> seq_len, gen, nsteps;
  std::vector<uint8_t> active;
  std::vector<float> mean;
  std::vector<uint32_t> lineage;
  std::vector<std::vector<Run>> history;     // which writer wrote which positions of each context
  std::vector<int64_t> cow;                  // (slot, old page, new page, rows) per copy-on-write
  // The last tournament's plan, for the caller to read.
  Plan last;

  Pool(int64_t np, int mb, int mp, int ps)
      : num_pages(np), max_beams(mb), max_pages(mp), P(ps), capacity(mb), refcnt(np, 0), tables(mb),
        seq_len(mb, 0), gen(mb, 0), nsteps(mb, 0), active(mb, 0), mean(mb, 0.f), lineage(mb, 0), history(mb) {
    for (int64_t p = 0; p < np; ++p) free_pages.push(p);
  }

  void set_error(int code) {
    if (status == kOk) status = code;
  }
  int64_t alloc() {
    const int64_t p = free_pages.top();
    free_pages.pop();
    refcnt[p] = 1;
    return p;
  }
  void unref(int64_t p) {
    if (--refcnt[p] == 0) free_pages.push(p);
  }
  int64_t pages_of(int64_t L) const { return (L + P - 1) / P; }

  bool seed(int n_beams, int64_t prompt_len) {
    const int64_t npg = pages_of(prompt_len);
    if (npg > max_pages || npg > (int64_t)free_pages.size()) return false;
    std::vector<int64_t> pages;
    for (int64_t i = 0; i < npg; ++i) pages.push_back(alloc());
    for (int64_t p : pages) refcnt[p] = n_beams;
    for (int b = 0; b < n_beams; ++b) {
      tables[b] = pages;
      seq_len[b] = prompt_len;
      active[b] = 1;
      gen[b] = 0;
      mean[b] = 0.f;
      nsteps[b] = 0;
      lineage[b] = next_lineage + (uint32_t)b;
      history[b] = {{kPromptWriter, 0, prompt_len}};
    }
    next_lineage += (uint32_t)n_beams;
    return true;
  }

  // Pages one decode step needs: a fresh page at each page boundary, and one copy per holder
  // of a shared partial tail page but the last.
  int64_t step_needs() const {
    int64_t need = 0;
    std::map<int64_t, int64_t> tail_holders;
    for (int b = 0; b < max_beams; ++b) {
      if (!active[b]) continue;
      if (seq_len[b] % P == 0)
        ++need;
      else
        ++tail_holders[tables[b][seq_len[b] / P]];
    }
    for (const auto& th : tail_holders) need += std::min(th.second, refcnt[th.first] - 1);
    return need;
  }

  // Reserve position seq_len[b] of every active beam, slots ascending.
  bool begin_step() {
    for (int b = 0; b < max_beams; ++b)
      if (active[b] && seq_len[b] % P == 0 && seq_len[b] / P >= max_pages) {
        set_error(kErrOom);
        return false;
      }
    if (step_needs() > (int64_t)free_pages.size()) {
      set_error(kErrOom);
      return false;
    }
    for (int b = 0; b < max_beams; ++b) {
      if (!active[b]) continue;
      const int64_t L = seq_len[b];
      if (L % P == 0) {
        tables[b].push_back(alloc());
      } else {
        const int64_t old = tables[b][L / P];
        if (refcnt[old] > 1) {
          const int64_t fresh = alloc();
          --refcnt[old];
          tables[b][L / P] = fresh;
          cow.insert(cow.end(), {b, old, fresh, L % P});
        }
      }
      seq_len[b] = L + 1;
      gen[b] += 1;
      std::vector<Run>& h = history[b];
      if (!h.empty() && h.back().writer == (uint32_t)b && h.back().end == L)
        h.back().end = L + 1;
      else
        h.push_back({(uint32_t)b, L, L + 1});
    }
    return true;
  }

  // Each (slot, parent): the slot's old references go first, then it takes the parent's table
  // (a reference on every page, nothing copied), length, mean and step count, gen 0 and a
  // fresh lineage id.
  void make_children(const std::vector<std::pair<int, int>>& children) {
    for (const auto& c : children)
      if (active[c.first])
        for (int64_t p : tables[c.first]) unref(p);
    for (size_t k = 0; k < children.size(); ++k) {
      const int s = children[k].first, par = children[k].second;
      tables[s] = tables[par];
      for (int64_t p : tables[s]) ++refcnt[p];
      seq_len[s] = seq_len[par];
      mean[s] = mean[par];
      nsteps[s] = nsteps[par];
      gen[s] = 0;
      lineage[s] = next_lineage + (uint32_t)k;
      active[s] = 1;
      history[s] = history[par];
    }
    next_lineage += (uint32_t)children.size();
  }

  void prune_branch(int K, int fanout, int64_t warmup, const uint8_t* mask, int32_t* parent_of, uint8_t* pruned) {
    std::vector<uint8_t> elig(max_beams);
    for (int s = 0; s < max_beams; ++s) elig[s] = active[s] && gen[s] >= warmup && (!mask || mask[s]);
    std::vector<uint8_t> was_active = active;
    last = tournament(mean.data(), active.data(), elig.data(), max_beams, capacity, K, fanout);
    make_children(last.children);
    for (int s = 0; s < max_beams; ++s) {
      parent_of[s] = was_active[s] ? s : -1;
      pruned[s] = 0;
    }
    for (const auto& c : last.children) parent_of[c.first] = c.second;
    for (int s : last.pruned) pruned[s] = 1;
  }

  void fork_slots(const int32_t* parent_of) {
    std::vector<std::pair<int, int>> children;
    for (int s = 0; s < max_beams; ++s) {
      const int p = parent_of[s];
      if (p < 0 || p == s) continue;
      if (p >= max_beams)
        set_error(kErrInvalid);
      else
        children.push_back({s, p});
    }
    make_children(children);
  }

  void release(const int32_t* slots, int n) {
    for (int i = 0; i < n; ++i) {
      const int s = slots[i];
      if (s < 0 || s >= max_beams) {
        set_error(kErrInvalid);
        continue;
      }
      if (!active[s]) {
        set_error(kErrState);
        continue;
      }
      for (int64_t p : tables[s]) unref(p);
      tables[s].clear();
      active[s] = 0;
      seq_len[s] = 0;
      gen[s] = 0;
      history[s].clear();
    }
  }

  // Reference-count conservation and the free-page identity; "" when they hold.
  std::string check() const {
    std::vector<int64_t> counted(num_pages, 0);
    int64_t held = 0;
    for (int b = 0; b < max_beams; ++b) {
      if (!active[b]) continue;
      if ((int64_t)tables[b].size() != pages_of(seq_len[b])) return "table length of slot " + std::to_string(b);
      for (int64_t p : tables[b]) ++counted[p];
      held += (int64_t)tables[b].size();
    }
    int64_t sum = 0, in_use = 0;
    for (int64_t p = 0; p < num_pages; ++p) {
      if (counted[p] != refcnt[p]) return "refcount of page " + std::to_string(p);
      sum += refcnt[p];
      in_use += refcnt[p] > 0;
    }
    if (sum != held) return "sum of refcounts";
    if ((int64_t)free_pages.size() != num_pages - in_use) return "free-page count";
    auto q = free_pages;
    int64_t prev = -1;
    while (!q.empty()) {
      const int64_t p = q.top();
      q.pop();
      if (p == prev || refcnt[p] != 0) return "free set holds page " + std::to_string(p);
      prev = p;
    }
    return "";
  }
};

// ---- beam KV materialised by copying -----------------------------------------------------------

struct BeamKV {
  int layers, Hkv, D;
  std::vector<std::vector<std::vector<float>>> K, V;  // [slot][layer] -> [L][Hkv][D]
  BeamKV(int nl, int mb, int hkv, int d)
      : layers(nl), Hkv(hkv), D(d), K(mb, std::vector<std::vector<float>>(nl)), V(mb, std::vector<std::vector<float>>(nl)) {}
  size_t row() const { return (size_t)Hkv * D; }
};

thread_local std::string g_msg;

}  // namespace

extern "C" {

// o[h] = sum_t softmax_t(scale * q[h] . K[t][h/G]) V[t][h/G]; q [Hq][D], K, V [L][Hkv][D], all fp64.
void gbo_decode_attention(const double* q, int Hq, int D, const double* K, const double* V, int L, int Hkv,
                          double scale, double* out) {
  const int G = Hq / Hkv;
  std::vector<double> p;
  for (int h = 0; h < Hq; ++h) {
    const int kh = h / G;
    softmax_weights(q + (size_t)h * D, K + (size_t)kh * D, L, D, Hkv * D, scale, p);
    for (int d = 0; d < D; ++d) {
      double o = 0.0;
      for (int t = 0; t < L; ++t) o += p[t] * V[((size_t)t * Hkv + kh) * D + d];
      out[(size_t)h * D + d] = o;
    }
  }
}

// The softmax weights of one query over L keys (K [L][D]), fp64.
void gbo_softmax_weights(const double* q, const double* K, int L, int D, double scale, double* p_out) {
  std::vector<double> p;
  softmax_weights(q, K, L, D, D, scale, p);
  std::copy(p.begin(), p.end(), p_out);
}

// sigma(w . h_i + b) for n rows h [n][H], fp64.
void gbo_probe_score(const double* h, int n, int H, const double* w, double bias, double* out) {
  for (int i = 0; i < n; ++i) {
    double z = 0.0;
    for (int d = 0; d < H; ++d) z += h[(size_t)i * H + d] * w[d];
    z += bias;
    out[i] = 1.0 / (1.0 + std::exp(-z));
  }
}

// One running-mean step in fp32: n counts the scores seen before x; returns the new mean.
float gbo_running_mean_update(float mean, int n, float x) {
  volatile float d = x - mean;             // each operation rounded to fp32 on its own
  volatile float q = d / (float)(n + 1);
  volatile float m = mean + q;
  return m;
}

// The Tournament over n slots: writes the case, the rank order (n_order entries), the pruned
// slots ascending and the (child, parent) pairs; returns the number of children.
int gbo_tournament(const float* mean, const uint8_t* active, const uint8_t* eligible, int n, int capacity, int K,
                   int fanout, int* kase, int* order, int* n_order, int* pruned, int* n_pruned, int* children) {
  const Plan p = tournament(mean, active, eligible, n, capacity, K, fanout);
  *kase = p.kase;
  *n_order = (int)p.order.size();
  std::copy(p.order.begin(), p.order.end(), order);
  *n_pruned = (int)p.pruned.size();
  std::copy(p.pruned.begin(), p.pruned.end(), pruned);
  for (size_t k = 0; k < p.children.size(); ++k) {
    children[2 * k] = p.children[k].first;
    children[2 * k + 1] = p.children[k].second;
  }
  return (int)p.children.size();
}

void* gbo_pool_new(int64_t num_pages, int max_beams, int max_pages, int page_size) {
  return new Pool(num_pages, max_beams, max_pages, page_size);
}
void gbo_pool_free(void* pool) { delete static_cast<Pool*>(pool); }
void* gbo_pool_clone(void* pool) { return new Pool(*static_cast<Pool*>(pool)); }

// Direct views of the per-slot state and the reference counts (the wrapper reads and writes them).
void* gbo_pool_array(void* pool, int which) {
  Pool* p = static_cast<Pool*>(pool);
  switch (which) {
    case 0: return p->seq_len.data();
    case 1: return p->active.data();
    case 2: return p->gen.data();
    case 3: return p->mean.data();
    case 4: return p->nsteps.data();
    case 5: return p->lineage.data();
    case 6: return p->refcnt.data();
  }
  return nullptr;
}

int gbo_pool_seed(void* pool, int n_beams, int64_t prompt_len) { return static_cast<Pool*>(pool)->seed(n_beams, prompt_len); }
int gbo_pool_begin_step(void* pool) { return static_cast<Pool*>(pool)->begin_step(); }
int gbo_pool_status(void* pool) { return static_cast<Pool*>(pool)->status; }
void gbo_pool_set_status(void* pool, int status) { static_cast<Pool*>(pool)->status = status; }
void gbo_pool_set_capacity(void* pool, int c) { static_cast<Pool*>(pool)->capacity = c; }
int gbo_pool_capacity(void* pool) { return static_cast<Pool*>(pool)->capacity; }
int64_t gbo_pool_num_free(void* pool) { return (int64_t) static_cast<Pool*>(pool)->free_pages.size(); }
uint32_t gbo_pool_next_lineage(void* pool) { return static_cast<Pool*>(pool)->next_lineage; }

void gbo_pool_prune_branch(void* pool, int K, int fanout, int64_t warmup, const uint8_t* mask, int32_t* parent_of,
                           uint8_t* pruned) {
  static_cast<Pool*>(pool)->prune_branch(K, fanout, warmup, mask, parent_of, pruned);
}
// The last tournament's plan: the case, then the sizes of its lists.
int gbo_pool_last_plan(void* pool, int* order, int* n_order, int* pruned, int* n_pruned, int* children,
                       int* n_children) {
  const Plan& p = static_cast<Pool*>(pool)->last;
  *n_order = (int)p.order.size();
  *n_pruned = (int)p.pruned.size();
  *n_children = (int)p.children.size();
  if (order) std::copy(p.order.begin(), p.order.end(), order);
  if (pruned) std::copy(p.pruned.begin(), p.pruned.end(), pruned);
  if (children)
    for (size_t k = 0; k < p.children.size(); ++k) {
      children[2 * k] = p.children[k].first;
      children[2 * k + 1] = p.children[k].second;
    }
  return p.kase;
}
void gbo_pool_fork_slots(void* pool, const int32_t* parent_of) { static_cast<Pool*>(pool)->fork_slots(parent_of); }
void gbo_pool_release(void* pool, const int32_t* slots, int n) { static_cast<Pool*>(pool)->release(slots, n); }

// Table of a slot: returns its length and copies up to cap entries.
int gbo_pool_table(void* pool, int slot, int64_t* out, int cap) {
  const std::vector<int64_t>& t = static_cast<Pool*>(pool)->tables[slot];
  std::copy(t.begin(), t.begin() + std::min<size_t>(t.size(), (size_t)cap), out);
  return (int)t.size();
}
// Writer history of a slot as (writer, start, end) triples: returns the run count.
int gbo_pool_history(void* pool, int slot, int64_t* out, int cap) {
  const std::vector<Run>& h = static_cast<Pool*>(pool)->history[slot];
  for (size_t i = 0; i < h.size() && (int)i < cap; ++i) {
    out[3 * i] = h[i].writer;
    out[3 * i + 1] = h[i].start;
    out[3 * i + 2] = h[i].end;
  }
  return (int)h.size();
}
// Copy-on-write events so far as (slot, old page, new page, rows) quadruples: returns the count.
int gbo_pool_cow_events(void* pool, int64_t* out, int cap) {
  const std::vector<int64_t>& c = static_cast<Pool*>(pool)->cow;
  const int n = (int)(c.size() / 4);
  std::copy(c.begin(), c.begin() + 4 * std::min(n, cap), out);
  return n;
}
// Invariant check: returns "" when they hold, else what failed.
const char* gbo_pool_check(void* pool) {
  g_msg = static_cast<Pool*>(pool)->check();
  return g_msg.c_str();
}

void* gbo_kv_new(int layers, int max_beams, int Hkv, int D) { return new BeamKV(layers, max_beams, Hkv, D); }
void gbo_kv_free(void* kv) { delete static_cast<BeamKV*>(kv); }
// Append n rows [n][Hkv][D] to a slot's layer.
void gbo_kv_append(void* kv, int slot, int layer, const float* k, const float* v, int n) {
  BeamKV* s = static_cast<BeamKV*>(kv);
  const size_t m = (size_t)n * s->row();
  s->K[slot][layer].insert(s->K[slot][layer].end(), k, k + m);
  s->V[slot][layer].insert(s->V[slot][layer].end(), v, v + m);
}
// A branched child gets a copy of its parent's arrays (every layer).
void gbo_kv_branch(void* kv, int child, int parent) {
  BeamKV* s = static_cast<BeamKV*>(kv);
  s->K[child] = s->K[parent];
  s->V[child] = s->V[parent];
}
void gbo_kv_release(void* kv, int slot) {
  BeamKV* s = static_cast<BeamKV*>(kv);
  for (int l = 0; l < s->layers; ++l) {
    s->K[slot][l].clear();
    s->V[slot][l].clear();
  }
}
// Rows held for (slot, layer); copies them (widened to fp64) when k_out / v_out are given.
int gbo_kv_get(void* kv, int slot, int layer, double* k_out, double* v_out) {
  const BeamKV* s = static_cast<BeamKV*>(kv);
  const std::vector<float>& K = s->K[slot][layer];
  const std::vector<float>& V = s->V[slot][layer];
  if (k_out) std::copy(K.begin(), K.end(), k_out);
  if (v_out) std::copy(V.begin(), V.end(), v_out);
  return (int)(K.size() / s->row());
}

}  // extern "C"
