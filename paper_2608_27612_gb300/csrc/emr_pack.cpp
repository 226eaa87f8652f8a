// Host side of libemr: grid descriptor (Eq. 1), genome packer, status strings.
#include <pthread.h>

#include <algorithm>
#include <atomic>
#include <chrono>
#include <cmath>
#include <condition_variable>
#include <functional>
#include <memory>
#include <mutex>
#include <cstring>
#include <thread>
#include <utility>
#include <vector>

#include "emr_internal.h"

using namespace emr;

namespace {

inline size_t align16(size_t x) { return (x + 15) & ~size_t(15); }

// Host worker threads kept across calls (starting threads costs as much as
// packing a few dozen genomes). run() executes fn(0 .. n-1) on the workers and
// the caller and returns when all are done; one job at a time (a caller that
// finds the pool busy runs its job alone). A worker that finishes a job watches
// for the next one for kSpinMicros before it sleeps, so that calls in quick
// succession (a packing pipeline) hand out their tasks without waking threads.
// shutdown() (emr_pack_release, and the library's unload) stops and joins the
// workers; the next run() starts a fresh pool. A process forked from this one
// starts a fresh pool too.
class WorkerPool {
 public:
  static constexpr int kSpinMicros = 400;

  static WorkerPool& get() {
    static std::once_flag once;
    std::call_once(once, [] { pthread_atfork(nullptr, nullptr, [] { instance() = nullptr; }); });
    std::lock_guard<std::mutex> lk(create_mu());
    if (!instance()) instance() = new WorkerPool();
    return *instance();
  }

  // Stop and join the workers and free the pool (never while a job runs on it).
  static void shutdown() {
    WorkerPool* p;
    {
      std::lock_guard<std::mutex> lk(create_mu());
      p = instance();
      instance() = nullptr;
    }
    if (!p) return;
    {
      std::lock_guard<std::mutex> job(p->job_mu_);  // a job in progress finishes first
      std::lock_guard<std::mutex> lk(p->mu_);
      p->stop_.store(true);
    }
    p->cv_.notify_all();
    for (std::thread& t : p->threads_)
      if (t.joinable()) t.join();
    delete p;
  }

  void run(int n, const std::function<void(int)>& fn) {
    std::unique_lock<std::mutex> job_lock(job_mu_, std::try_to_lock);
    if (!job_lock.owns_lock() || n <= 1) {
      for (int t = 0; t < n; t++) fn(t);
      return;
    }
    ensure(n - 1);
    uint64_t g;
    {
      std::lock_guard<std::mutex> lk(mu_);
      job_ = &fn;
      n_ = n;
      left_.store(n - 1);
      g = gen_.load() + 1;
      claim_.store((g << 32) | 1u, std::memory_order_release);  // task 0 is the caller's
      gen_.store(g, std::memory_order_release);
    }
    cv_.notify_all();  // the workers asleep; the spinning ones have seen gen_
    fn(0);
    for (int t; (t = claim(g, n)) >= 0;) {  // help with the tasks not yet taken
      fn(t);
      left_.fetch_sub(1, std::memory_order_acq_rel);
    }
    // the workers' last tasks: short, so wait by spinning, then on the condition variable
    for (int k = 0; left_.load(std::memory_order_acquire) != 0 && k < 4096; k++) {
    }
    if (left_.load(std::memory_order_acquire) != 0) {
      std::unique_lock<std::mutex> lk(mu_);
      done_cv_.wait(lk, [&] { return left_.load(std::memory_order_acquire) == 0; });
    }
    std::lock_guard<std::mutex> lk(mu_);
    job_ = nullptr;
  }

 private:
  static WorkerPool*& instance() {
    static WorkerPool* p = nullptr;
    return p;
  }
  static std::mutex& create_mu() {
    static std::mutex m;
    return m;
  }

  void ensure(int workers) {
    while (int(threads_.size()) < workers) threads_.emplace_back([this] { loop(); });
  }

  // The next task of job generation g (of n tasks), or -1 when it has none left or a newer
  // job was posted: a task is claimed together with its job's generation, so a thread late
  // to a finished job never runs the next job's tasks with the old function.
  int claim(uint64_t g, int n) {
    uint64_t c = claim_.load(std::memory_order_acquire);
    for (;;) {
      if ((c >> 32) != (g & 0xffffffffu) || int(c & 0xffffffffu) >= n) return -1;
      if (claim_.compare_exchange_weak(c, c + 1, std::memory_order_acq_rel)) return int(c & 0xffffffffu);
    }
  }

  void loop() {
    uint64_t seen = gen_.load(std::memory_order_acquire);
    for (;;) {
      // watch for a new job for a while, then sleep until one is posted
      const auto t0 = std::chrono::steady_clock::now();
      for (int k = 1; gen_.load(std::memory_order_acquire) == seen && !stop_.load(); k++) {
        if ((k & 255) == 0 && std::chrono::steady_clock::now() - t0 > std::chrono::microseconds(kSpinMicros)) {
          std::unique_lock<std::mutex> lk(mu_);
          cv_.wait(lk, [&] { return stop_.load() || gen_.load(std::memory_order_acquire) != seen; });
          break;
        }
      }
      if (stop_.load()) return;
      const std::function<void(int)>* fn;
      int n;
      {
        std::lock_guard<std::mutex> lk(mu_);
        seen = gen_.load(std::memory_order_acquire);
        fn = job_;
        n = n_;
      }
      if (!fn) continue;
      for (int t; (t = claim(seen, n)) >= 0;) {
        (*fn)(t);
        if (left_.fetch_sub(1, std::memory_order_acq_rel) == 1) {
          std::lock_guard<std::mutex> lk(mu_);
          done_cv_.notify_all();
        }
      }
    }
  }

  std::mutex job_mu_, mu_;
  std::condition_variable cv_, done_cv_;
  const std::function<void(int)>* job_ = nullptr;
  int n_ = 0;
  std::atomic<int> left_{0};
  std::atomic<uint64_t> gen_{0}, claim_{0};  // claim_: generation (high 32 bits) and next task
  std::atomic<bool> stop_{false};
  std::vector<std::thread> threads_;
};

uint32_t compact_bits(uint64_t m) {  // even bits of m, packed
  m &= 0x5555555555555555ull;
  m = (m | (m >> 1)) & 0x3333333333333333ull;
  m = (m | (m >> 2)) & 0x0f0f0f0f0f0f0f0full;
  m = (m | (m >> 4)) & 0x00ff00ff00ff00ffull;
  m = (m | (m >> 8)) & 0x0000ffff0000ffffull;
  m = (m | (m >> 16)) & 0x00000000ffffffffull;
  return uint32_t(m);
}

// Relative per-query work of one activation, for scheduling only.
int act_cost(int a) {
  static const int c[6] = {0, 5, 6, 3, 7, 1};
  return (a >= 0 && a < 6) ? c[a] : 8;
}

struct Edge {
  int s, d;
  float w;
  int ord;  // position among the genome's enabled connections (the large-genome merge restores it)
};

// Buffers reused across genomes (capacity kept; no allocation per genome once warm).
struct Scratch {
  std::vector<std::pair<int32_t, int>> ids;  // (id, local index), sorted by id
  std::vector<Edge> es;
  std::vector<int> indeg, order, ready, stack, slot, kept;
  std::vector<int> succ_beg, succ, pred_beg, pred, fill;
  std::vector<char> reach;
  std::vector<unsigned> has_in;
  std::vector<uint64_t> seen;  // per destination: the sources seen (genomes up to 64 nodes)
  std::vector<int> in_cnt, in_beg;
  std::vector<PackEdge> in_edges;
  std::vector<int> table;  // id - id_min -> local index (-1: none), when the ids span a small range
  int64_t id_min = 0;
};

// Scratch of the packing tasks of one call, kept across calls so that a warm
// packer allocates nothing. One caller at a time uses the shared set (a caller
// that finds it in use packs with its own); release() (from emr_pack_release)
// frees the memory, and the next call grows it again.
struct PackBuffers {
  static constexpr int kTasks = 16;
  std::mutex mu;
  Scratch scratch[kTasks];
  static PackBuffers& get() {
    static PackBuffers* b = new PackBuffers();
    return *b;
  }
  void release() {
    std::lock_guard<std::mutex> lk(mu);
    for (int t = 0; t < kTasks; t++) scratch[t] = Scratch();
  }
};

int local_of(const Scratch& S, int32_t id) {
  if (!S.table.empty()) {  // ids span a small range: direct lookup
    const int64_t k = int64_t(id) - S.id_min;
    return (k >= 0 && k < int64_t(S.table.size())) ? S.table[size_t(k)] : -1;
  }
  auto it = std::lower_bound(S.ids.begin(), S.ids.end(), std::make_pair(id, -1));
  return (it != S.ids.end() && it->first == id) ? it->second : -1;
}

// CSR adjacency (by source for succ, by destination for pred) over the enabled edges.
void build_csr(int n, const std::vector<Edge>& es, bool by_src, std::vector<int>& beg, std::vector<int>& adj,
               std::vector<int>& fill) {
  beg.assign(n + 1, 0);
  for (auto& e : es) beg[(by_src ? e.s : e.d) + 1]++;
  for (int v = 0; v < n; v++) beg[v + 1] += beg[v];
  adj.resize(es.size());
  fill.assign(n, 0);
  for (auto& e : es) {
    const int k = by_src ? e.s : e.d;
    adj[beg[k] + fill[k]++] = by_src ? e.d : e.s;
  }
}

// Topological order (Kahn, ties by id), dead-node removal, input folding and
// per-side variation flags for one genome. Its records go to on[] (room for
// n1 - n0 nodes) and oe[] (room for c1 - c0 edges), the unused rest zeroed;
// *out is its genome record, node_beg and edge_beg left to the caller.
emr_status pack_one(int64_t n0, int64_t n1, int64_t c0, int64_t c1, const int32_t* node_id,
                    const int32_t* node_kind, const int32_t* node_act, const float* node_bias,
                    const int32_t* conn_src, const int32_t* conn_dst, const float* conn_w,
                    const uint8_t* conn_en, Scratch& S, PackNode* on, PackEdge* oe, PackGenome* out) {
  const int n = int(n1 - n0);
  if (n <= 0 || n > 1 << 20) return EMR_ERR_ARG;
  S.ids.clear();
  int out_node = -1;
  for (int k = 0; k < n; k++) {
    const int kind = node_kind[n0 + k];
    if (kind < 0 || kind > EMR_KIND_OUTPUT) return EMR_ERR_ARG;
    if (kind >= EMR_KIND_HIDDEN && (node_act[n0 + k] < 0 || node_act[n0 + k] > EMR_ACT_ABS)) return EMR_ERR_ARG;
    if (kind == EMR_KIND_OUTPUT) {
      if (out_node >= 0) return EMR_ERR_ARG;
      out_node = k;
    }
    S.ids.push_back({node_id[n0 + k], k});
  }
  if (out_node < 0) return EMR_ERR_ARG;
  if (!std::is_sorted(S.ids.begin(), S.ids.end())) std::sort(S.ids.begin(), S.ids.end());
  for (size_t k = 1; k < S.ids.size(); k++)
    if (S.ids[k].first == S.ids[k - 1].first) return EMR_ERR_ARG;  // duplicate id
  S.table.clear();
  const int64_t span = int64_t(S.ids.back().first) - S.ids.front().first + 1;
  if (span <= 4 * int64_t(n) + 64) {
    S.id_min = S.ids.front().first;
    S.table.assign(size_t(span), -1);
    for (auto& pr : S.ids) S.table[size_t(int64_t(pr.first) - S.id_min)] = pr.second;
  }
  S.es.clear();
  for (int64_t c = c0; c < c1; c++) {
    if (!conn_en[c]) continue;
    const int ls = local_of(S, conn_src[c]), ld = local_of(S, conn_dst[c]);
    if (ls < 0 || ld < 0) return EMR_ERR_ARG;
    if (node_kind[n0 + ld] < EMR_KIND_HIDDEN) return EMR_ERR_ARG;
    S.es.push_back({ls, ld, conn_w[c]});
  }
  // Parallel connections (same source and destination) become one edge whose
  // weight is their sum in connection order; an edge of weight 0 contributes
  // nothing and is dropped. Every evaluator then sees at most one edge per
  // (source, destination), each of nonzero weight.
  if (n <= 64) {  // a source mask per destination finds repeats without sorting
    S.seen.assign(size_t(n), 0ull);
    bool repeat = false;
    for (auto& e : S.es) {
      const uint64_t bit = 1ull << e.s;
      repeat = repeat || (S.seen[e.d] & bit);
      S.seen[e.d] |= bit;
    }
    size_t m = 0;
    for (size_t k = 0; k < S.es.size(); k++) {
      Edge e = S.es[k];
      if (repeat) {  // fold later repeats into the first occurrence, in connection order
        size_t f = 0;
        while (f < m && !(S.es[f].s == e.s && S.es[f].d == e.d)) f++;
        if (f < m) {
          S.es[f].w += e.w;
          continue;
        }
      }
      S.es[m++] = e;
    }
    S.es.resize(m);
  } else {
    for (size_t k = 0; k < S.es.size(); k++) S.es[k].ord = int(k);
    std::stable_sort(S.es.begin(), S.es.end(),
                     [](const Edge& a, const Edge& b) { return a.d != b.d ? a.d < b.d : a.s < b.s; });
    size_t m = 0;
    for (size_t k = 0; k < S.es.size();) {
      Edge e = S.es[k++];  // the first occurrence: the sort is stable
      while (k < S.es.size() && S.es[k].s == e.s && S.es[k].d == e.d) e.w += S.es[k++].w;
      S.es[m++] = e;
    }
    S.es.resize(m);
    // back to the order of first occurrence, the order the path above keeps
    std::sort(S.es.begin(), S.es.end(), [](const Edge& a, const Edge& b) { return a.ord < b.ord; });
  }
  S.es.erase(std::remove_if(S.es.begin(), S.es.end(), [](const Edge& e) { return e.w == 0.f; }), S.es.end());
  S.reach.assign(n, 0);
  if (n <= 64) {
    // Kahn's algorithm and the reachability on bit masks: bit k of succ[v] / pred[v] is local
    // node k; the ready set holds nodes by rank in id order, so its lowest bit is the ready
    // node of smallest id.
    uint64_t succ[64], pred[64];
    int indeg[64];
    uint8_t rank_of[64], node_at[64];
    for (int k = 0; k < n; k++) {
      succ[k] = pred[k] = 0;
      indeg[k] = 0;
    }
    for (auto& e : S.es) {  // parallel edges are merged: one per source
      succ[e.s] |= 1ull << e.d;
      pred[e.d] |= 1ull << e.s;
      indeg[e.d]++;
    }
    for (int r = 0; r < n; r++) {
      node_at[r] = uint8_t(S.ids[size_t(r)].second);
      rank_of[S.ids[size_t(r)].second] = uint8_t(r);
    }
    uint64_t ready = 0;
    for (int k = 0; k < n; k++)
      if (indeg[k] == 0) ready |= 1ull << rank_of[k];
    S.order.clear();
    while (ready) {
      const int v = node_at[__builtin_ctzll(ready)];
      ready &= ready - 1;
      S.order.push_back(v);
      for (uint64_t m = succ[v]; m; m &= m - 1) {
        const int u = __builtin_ctzll(m);
        if (--indeg[u] == 0) ready |= 1ull << rank_of[u];
      }
    }
    if (int(S.order.size()) != n) return EMR_ERR_CYCLE;
    // the nodes from which the output is reachable
    uint64_t reach = 1ull << out_node, todo = reach;
    while (todo) {
      const int v = __builtin_ctzll(todo);
      todo &= todo - 1;
      const uint64_t fresh = pred[v] & ~reach;
      reach |= fresh;
      todo |= fresh;
    }
    for (int k = 0; k < n; k++) S.reach[size_t(k)] = char((reach >> k) & 1u);
  } else {
    build_csr(n, S.es, true, S.succ_beg, S.succ, S.fill);
    build_csr(n, S.es, false, S.pred_beg, S.pred, S.fill);
    // Kahn's algorithm over every node; ready nodes leave in ascending id order.
    S.indeg.assign(n, 0);
    for (auto& e : S.es) S.indeg[e.d]++;
    S.order.clear();
    S.ready.clear();
    auto by_id = [&](int a, int b) { return node_id[n0 + a] > node_id[n0 + b]; };  // min-heap on id
    for (int v = 0; v < n; v++)
      if (S.indeg[v] == 0) S.ready.push_back(v);
    std::make_heap(S.ready.begin(), S.ready.end(), by_id);
    while (!S.ready.empty()) {
      std::pop_heap(S.ready.begin(), S.ready.end(), by_id);
      const int v = S.ready.back();
      S.ready.pop_back();
      S.order.push_back(v);
      for (int k = S.succ_beg[v]; k < S.succ_beg[v + 1]; k++)
        if (--S.indeg[S.succ[k]] == 0) {
          S.ready.push_back(S.succ[k]);
          std::push_heap(S.ready.begin(), S.ready.end(), by_id);
        }
    }
    if (int(S.order.size()) != n) return EMR_ERR_CYCLE;
    // Keep the non-input nodes from which the output is reachable.
    S.stack.assign(1, out_node);
    S.reach[out_node] = 1;
    while (!S.stack.empty()) {
      const int v = S.stack.back();
      S.stack.pop_back();
      for (int k = S.pred_beg[v]; k < S.pred_beg[v + 1]; k++)
        if (!S.reach[S.pred[k]]) { S.reach[S.pred[k]] = 1; S.stack.push_back(S.pred[k]); }
    }
  }
  S.slot.assign(n, -1);
  S.kept.clear();
  for (int v : S.order)
    if (S.reach[v] && node_kind[n0 + v] >= EMR_KIND_HIDDEN) { S.slot[v] = int(S.kept.size()); S.kept.push_back(v); }
  if (S.kept.empty() || S.kept.back() != out_node) return EMR_ERR_ARG;  // output must be last
  if (S.kept.size() > 65535) return EMR_ERR_RANGE;
  const int nk = int(S.kept.size());
  std::memset(on, 0, sizeof(PackNode) * size_t(n));  // the kept nodes' records, then zeros
  S.has_in.assign(nk, 0);  // bit k: has an enabled in-connection from input kind k
  S.in_cnt.assign(nk, 0);
  for (int t = 0; t < nk; t++) {
    const int v = S.kept[t];
    on[t].act = uint8_t(node_act[n0 + v]);
    on[t].bias = node_bias[n0 + v];
  }
  for (auto& e : S.es) {
    const int t = S.slot[e.d];
    if (t < 0) continue;
    const int sk = node_kind[n0 + e.s];
    if (sk < EMR_KIND_HIDDEN) {
      on[t].w_in[sk] += e.w;
      S.has_in[t] |= 1u << sk;
    } else {
      if (S.slot[e.s] < 0) return EMR_ERR_ARG;  // cannot happen: a source of a kept node is kept
      S.in_cnt[t]++;
    }
  }
  // in-edges from kept non-input nodes, grouped by destination (each group in the order of
  // the edges' first connections)
  S.in_beg.assign(nk + 1, 0);
  for (int t = 0; t < nk; t++) S.in_beg[t + 1] = S.in_beg[t] + S.in_cnt[t];
  if (S.in_beg[nk] > 65535) return EMR_ERR_RANGE;
  if (S.in_beg[nk] > c1 - c0) return EMR_ERR_ARG;  // cannot happen: an edge per kept connection at most
  std::memset(oe, 0, sizeof(PackEdge) * size_t(c1 - c0));
  S.fill.assign(nk, 0);
  for (auto& e : S.es) {
    const int t = S.slot[e.d];
    if (t < 0 || node_kind[n0 + e.s] < EMR_KIND_HIDDEN) continue;
    oe[S.in_beg[t] + S.fill[t]++] = PackEdge{uint16_t(S.slot[e.s]), 0, e.w};
  }
  PackGenome& g = *out;
  g = PackGenome{};
  g.n_nodes = uint16_t(nk);
  for (int t = 0; t < nk; t++) {
    on[t].edge_beg = uint16_t(S.in_beg[t]);
    on[t].edge_cnt = uint16_t(S.in_cnt[t]);
  }
  g.n_edges = uint16_t(S.in_beg[nk]);
  for (int side = 0; side < 2; side++) {
    const int gx = side == EMR_SIDE_OUT ? EMR_KIND_X2 : EMR_KIND_X1;
    const int gy = side == EMR_SIDE_OUT ? EMR_KIND_Y2 : EMR_KIND_Y1;
    int nv = 0, nve = 0, nj = 0;
    uint32_t cost = 0;
    for (int t = 0; t < nk; t++) {
      // the grid coordinates the node depends on: its own grid inputs and those of its sources
      uint32_t ax = ((S.has_in[t] >> gx) & 1u) * kAxisX | ((S.has_in[t] >> gy) & 1u) * kAxisY;
      int vin = 0;
      for (int k = S.in_beg[t]; k < S.in_beg[t + 1]; k++) {
        const uint32_t sa = (on[oe[k].src].axes >> (2 * side)) & 3u;
        if (sa) { ax |= sa; vin++; }
      }
      if (ax) {
        on[t].vary |= uint8_t(1u << side);
        on[t].axes |= uint8_t(ax << (2 * side));
        nv++;
        nve += vin;
        // per-query work: a node of one coordinate is evaluated once per tile row or column
        if (ax == kAxisXY) { nj++; cost += 2 + vin + act_cost(on[t].act); }
      }
    }
    if (nv > EMR_MAX_VARYING || nve > EMR_MAX_VEDGES) return EMR_ERR_RANGE;
    g.n_varying[side] = uint16_t(nv);
    g.n_vedges[side] = uint16_t(nve);
    g.n_joint[side] = uint16_t(nj);
    g.cost[side] = cost + (nv > nj ? 1u : 0u);
  }
  return EMR_OK;
}

}  // namespace

void emr::host_parallel(int n, const std::function<void(int)>& fn) { WorkerPool::get().run(n, fn); }

extern "C" {

emr_status emr_grid_build(int32_t D, int64_t chunk, emr_grid* grid) {
  if (!grid) return EMR_ERR_ARG;
  if (D < 0 || D > EMR_MAX_DEPTH) return EMR_ERR_RANGE;
  if (chunk < 0 || (chunk > 0 && (chunk < 4096 || (chunk & (chunk - 1)) != 0))) return EMR_ERR_ARG;
  std::memset(grid, 0, sizeof *grid);
  grid->D = D;
  grid->chunk = chunk;
  int64_t words = 0;
  for (int d = 0; d < EMR_MAX_DEPTH + 2; d++) {  // entries past D + 1 repeat the totals
    const int e = d <= D + 1 ? d : D + 1;
    grid->level_off[d] = level_offset(e);
    grid->halo_off[d] = halo_offset(e);
    grid->word_off[d] = words;
    if (d <= D) words += ((int64_t(1) << (2 * (d + 1))) + 31) / 32;
  }
  grid->n_total = grid->level_off[D + 1];
  grid->n_halo = grid->halo_off[D + 1];
  grid->n_words = words;
  return EMR_OK;
}

emr_status emr_index_to_ij(int64_t gidx, int32_t* d, int32_t* i, int32_t* j) {
  if (gidx < 0 || gidx >= level_offset(EMR_MAX_DEPTH + 1)) return EMR_ERR_RANGE;
  int lv = 0;
  while (level_offset(lv + 1) <= gidx) lv++;
  uint64_t m = uint64_t(gidx - level_offset(lv));
  if (d) *d = lv;
  if (i) *i = int32_t(compact_bits(m));
  if (j) *j = int32_t(compact_bits(m >> 1));
  return EMR_OK;
}

emr_status emr_pack_size(int32_t P, const int64_t* node_ptr, const int64_t* conn_ptr, size_t* bytes) {
  if (P < 0 || !bytes || (P > 0 && (!node_ptr || !conn_ptr))) return EMR_ERR_ARG;
  int64_t nn = P ? node_ptr[P] - node_ptr[0] : 0, nc = P ? conn_ptr[P] - conn_ptr[0] : 0;
  if (nn < 0 || nc < 0) return EMR_ERR_ARG;
  *bytes = align16(sizeof(PackHeader)) + align16(sizeof(PackGenome) * size_t(P)) +
           align16(sizeof(PackNode) * size_t(nn)) + align16(sizeof(PackEdge) * size_t(nc)) + 16;
  return EMR_OK;
}

emr_status emr_pack_population(int32_t P, const int64_t* node_ptr, const int32_t* node_id,
                               const int32_t* node_kind, const int32_t* node_act, const float* node_bias,
                               const int64_t* conn_ptr, const int32_t* conn_src, const int32_t* conn_dst,
                               const float* conn_w, const uint8_t* conn_enabled, void* buf, size_t cap,
                               size_t* used, int32_t* bad_genome) {
  if (bad_genome) *bad_genome = -1;
  if (P <= 0 || !node_ptr || !node_id || !node_kind || !node_act || !node_bias || !conn_ptr ||
      (!buf && cap > 0) || !used)
    return EMR_ERR_ARG;
  const bool has_conns = conn_ptr[P] > conn_ptr[0];
  if (has_conns && (!conn_src || !conn_dst || !conn_w || !conn_enabled)) return EMR_ERR_ARG;
  // Layout: genome g's node records start at node index node_ptr[g] - node_ptr[0] and its edge
  // records at conn_ptr[g] - conn_ptr[0] (room for all its input nodes and connections; the
  // unused rest is zeroed), so every genome packs straight into the blob, independently.
  const int64_t nn = node_ptr[P] - node_ptr[0], nc = conn_ptr[P] - conn_ptr[0];
  if (nn < 0 || nc < 0) return EMR_ERR_ARG;
  if (nn > int64_t(UINT32_MAX) || nc > int64_t(UINT32_MAX)) return EMR_ERR_RANGE;
  PackHeader h{};
  h.magic = kPackMagic;
  h.version = kPackVersion;
  h.P = P;
  h.off_genomes = align16(sizeof(PackHeader));
  h.off_nodes = h.off_genomes + align16(sizeof(PackGenome) * size_t(P));
  h.off_edges = h.off_nodes + align16(sizeof(PackNode) * size_t(nn));
  h.total_bytes = h.off_edges + align16(sizeof(PackEdge) * size_t(nc));
  *used = size_t(h.total_bytes);
  if (cap < h.total_bytes) return EMR_ERR_CAPACITY;
  auto* base = static_cast<uint8_t*>(buf);
  // the genome records, nodes and edges are written below; clear the alignment gaps between sections
  auto clear = [&](uint64_t from, uint64_t to) {
    if (to > from) std::memset(base + from, 0, size_t(to - from));
  };
  clear(sizeof(PackHeader), h.off_genomes);
  clear(h.off_genomes + sizeof(PackGenome) * uint64_t(P), h.off_nodes);
  clear(h.off_nodes + sizeof(PackNode) * uint64_t(nn), h.off_edges);
  clear(h.off_edges + sizeof(PackEdge) * uint64_t(nc), h.total_bytes);
  auto* gt = reinterpret_cast<PackGenome*>(base + h.off_genomes);
  auto* nt = reinterpret_cast<PackNode*>(base + h.off_nodes);
  auto* et = reinterpret_cast<PackEdge*>(base + h.off_edges);
  // per-task scratch kept across calls; a caller that finds it in use packs with its own
  PackBuffers& shared = PackBuffers::get();
  std::unique_lock<std::mutex> buf_lock(shared.mu, std::try_to_lock);
  std::unique_ptr<PackBuffers> own;
  if (!buf_lock.owns_lock()) own.reset(new PackBuffers());
  PackBuffers& B = own ? *own : shared;
  // Genomes are independent: host tasks take chunks of kChunk genomes from a shared counter,
  // each with its own scratch; the lowest failing genome index is reported.
  constexpr int kChunk = 8;
  const int n_chunks = (P + kChunk - 1) / kChunk;
  const int hw = int(std::max(1u, std::thread::hardware_concurrency()));
  // a task's share costs about as much to hand out as packing a few genomes
  const int n_tasks = std::max(1, std::min({hw, PackBuffers::kTasks, P / 32}));
  struct TaskOut {
    int32_t bad = -1;
    emr_status rc = EMR_OK;
    int32_t max_nodes = 0, max_edges = 0, max_varying[2] = {0, 0}, max_vedges[2] = {0, 0};
  };
  TaskOut outs[PackBuffers::kTasks];
  std::atomic<int> next_chunk{0};
  auto work = [&](int t) {
    Scratch& scratch = B.scratch[t];
    TaskOut& o = outs[t];
    o = TaskOut();
    for (int c; (c = next_chunk.fetch_add(1, std::memory_order_relaxed)) < n_chunks;) {
      const int g_end = std::min(P, (c + 1) * kChunk);
      for (int g = c * kChunk; g < g_end; g++) {
        emr_status rc = EMR_OK;
        if (node_ptr[g + 1] < node_ptr[g] || conn_ptr[g + 1] < conn_ptr[g]) rc = EMR_ERR_ARG;
        const int64_t nb = node_ptr[g] - node_ptr[0], eb = conn_ptr[g] - conn_ptr[0];
        PackGenome& pg = gt[g];
        if (rc == EMR_OK)
          rc = pack_one(node_ptr[g], node_ptr[g + 1], conn_ptr[g], conn_ptr[g + 1], node_id, node_kind, node_act,
                        node_bias, conn_src, conn_dst, conn_w, conn_enabled, scratch, nt + nb, et + eb, &pg);
        if (rc != EMR_OK) {
          if (o.bad < 0 || g < o.bad) {
            o.bad = g;
            o.rc = rc;
          }
          continue;
        }
        pg.node_beg = uint32_t(nb);
        pg.edge_beg = uint32_t(eb);
        o.max_nodes = std::max<int32_t>(o.max_nodes, pg.n_nodes);
        o.max_edges = std::max<int32_t>(o.max_edges, pg.n_edges);
        for (int sd = 0; sd < 2; sd++) {
          o.max_varying[sd] = std::max<int32_t>(o.max_varying[sd], pg.n_varying[sd]);
          o.max_vedges[sd] = std::max<int32_t>(o.max_vedges[sd], pg.n_vedges[sd]);
        }
      }
    }
  };
  if (n_tasks == 1) {
    work(0);
  } else {
    WorkerPool::get().run(n_tasks, work);
  }
  int32_t bad = -1;
  emr_status bad_rc = EMR_OK;
  for (int t = 0; t < n_tasks; t++) {
    const TaskOut& o = outs[t];
    if (o.bad >= 0 && (bad < 0 || o.bad < bad)) {
      bad = o.bad;
      bad_rc = o.rc;
    }
    h.max_nodes = std::max(h.max_nodes, o.max_nodes);
    h.max_edges = std::max(h.max_edges, o.max_edges);
    for (int sd = 0; sd < 2; sd++) {
      h.max_varying[sd] = std::max(h.max_varying[sd], o.max_varying[sd]);
      h.max_vedges[sd] = std::max(h.max_vedges[sd], o.max_vedges[sd]);
    }
  }
  if (bad >= 0) {
    if (bad_genome) *bad_genome = bad;
    return bad_rc;
  }
  std::memcpy(base, &h, sizeof h);
  return EMR_OK;
}

emr_status emr_pack_info(const void* pack_host, int32_t* P, int32_t* max_varying_out, int32_t* max_varying_in) {
  if (!pack_host) return EMR_ERR_ARG;
  const PackHeader* h = pack_header(pack_host);
  if (h->magic != kPackMagic || h->version != kPackVersion) return EMR_ERR_ARG;
  if (P) *P = h->P;
  if (max_varying_out) *max_varying_out = h->max_varying[EMR_SIDE_OUT];
  if (max_varying_in) *max_varying_in = h->max_varying[EMR_SIDE_IN];
  return EMR_OK;
}

void emr_pack_release(void) {
  WorkerPool::shutdown();
  PackBuffers::get().release();
}

// The worker threads are joined when libemr is unloaded (or the process exits),
// so no thread outlives the library's code.
__attribute__((destructor)) static void emr_pack_unload() { WorkerPool::shutdown(); }

// Contiguous genome ranges of balanced cost for population-parallel work
// (Table 1: the CPPN query, variance and mask stages split over the
// population). A pair's weight is its packed per-query work estimate plus the
// filter's per-query work; a pair whose output is constant over the grid, or an
// unused per-genome slot, weighs 1 (its tiles are only cleared).
emr_status emr_partition_genomes(const void* pack_host, const emr_query* q, int32_t n_parts, int32_t* g_begin) {
  if (!pack_host || !q || q->S <= 0 || !q->side_host || n_parts <= 0 || !g_begin) return EMR_ERR_ARG;
  const PackHeader* h = pack_header(pack_host);
  if (h->magic != kPackMagic || h->version != kPackVersion || h->P <= 0) return EMR_ERR_ARG;
  const PackGenome* gt =
      reinterpret_cast<const PackGenome*>(static_cast<const uint8_t*>(pack_host) + h->off_genomes);
  constexpr uint64_t kFilterWork = 6;  // variance and band screen per query, in the cost estimate's units
  const int32_t P = h->P, S = q->S;
  std::vector<uint64_t> prefix(size_t(P) + 1, 0);
  for (int32_t g = 0; g < P; g++) {
    uint64_t w = 0;
    for (int32_t s = 0; s < S; s++) {
      const int64_t si = q->per_genome ? int64_t(g) * S + s : s;
      const int32_t side = q->side_host[si];
      if (side != EMR_SIDE_OUT && side != EMR_SIDE_IN) return EMR_ERR_ARG;
      const bool unused = q->per_genome && q->count_host && s >= q->count_host[g];
      w += (unused || gt[g].n_varying[side] == 0) ? 1 : uint64_t(gt[g].cost[side]) + kFilterWork;
    }
    prefix[size_t(g) + 1] = prefix[size_t(g)] + w;
  }
  const uint64_t total = prefix[size_t(P)];
  g_begin[0] = 0;
  for (int32_t k = 1; k < n_parts; k++) {
    // the boundary nearest to k / n_parts of the total, never before the previous one
    const uint64_t target = total / uint64_t(n_parts) * uint64_t(k) + total % uint64_t(n_parts) * uint64_t(k) / uint64_t(n_parts);
    int32_t g = int32_t(std::lower_bound(prefix.begin(), prefix.end(), target) - prefix.begin());
    if (g > 0 && target - prefix[size_t(g) - 1] < prefix[size_t(g)] - target) g--;
    g_begin[k] = std::max(std::min(g, P), g_begin[k - 1]);
  }
  g_begin[n_parts] = P;
  return EMR_OK;
}

const char* emr_strerror(emr_status s) {
  switch (s) {
    case EMR_OK: return "ok";
    case EMR_ERR_ARG: return "invalid argument";
    case EMR_ERR_CYCLE: return "genome has a cycle among its enabled connections";
    case EMR_ERR_RANGE: return "size beyond a documented limit";
    case EMR_ERR_CAPACITY: return "output buffer or workspace too small";
    case EMR_ERR_CUDA: return "CUDA error";
    case EMR_ERR_TIMEOUT: return "host-side wait timed out";
    case EMR_ERR_ALLOC: return "host allocation failed";
    default: return "unknown status";
  }
}

int32_t emr_version(void) { return 100; }

}  // extern "C"
