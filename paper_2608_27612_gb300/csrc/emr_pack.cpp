// Host side of libemr: grid descriptor (Eq. 1), genome packer, status strings.
#include <pthread.h>

#include <algorithm>
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
// finds the pool busy runs its job alone). shutdown() (emr_pack_release, and
// the library's unload) stops and joins the workers; the next run() starts a
// fresh pool. A process forked from this one starts a fresh pool too.
class WorkerPool {
 public:
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
      p->stop_ = true;
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
    {
      std::lock_guard<std::mutex> lk(mu_);
      job_ = &fn;
      n_ = n;
      next_ = 1;  // task 0 is the caller's
      left_ = n - 1;
      gen_++;
    }
    cv_.notify_all();
    fn(0);
    for (;;) {  // help with the remaining tasks, then wait for the workers' last ones
      int t;
      {
        std::lock_guard<std::mutex> lk(mu_);
        if (next_ >= n_) break;
        t = next_++;
      }
      fn(t);
      std::lock_guard<std::mutex> lk(mu_);
      if (--left_ == 0) break;
    }
    std::unique_lock<std::mutex> lk(mu_);
    done_cv_.wait(lk, [&] { return left_ == 0 || (next_ >= n_ && left_ == 0); });
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

  void loop() {
    uint64_t seen = 0;
    for (;;) {
      std::unique_lock<std::mutex> lk(mu_);
      cv_.wait(lk, [&] { return stop_ || (gen_ != seen && job_ && next_ < n_); });
      if (stop_) return;
      seen = gen_;
      while (job_ && next_ < n_) {
        const int t = next_++;
        const std::function<void(int)>* fn = job_;
        lk.unlock();
        (*fn)(t);
        lk.lock();
        if (--left_ == 0) done_cv_.notify_all();
      }
    }
  }

  std::mutex job_mu_, mu_;
  std::condition_variable cv_, done_cv_;
  const std::function<void(int)>* job_ = nullptr;
  int n_ = 0, next_ = 0, left_ = 0;
  uint64_t gen_ = 0;
  bool stop_ = false;
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

// A genome's packed record; its nodes and edges are appended to its thread's
// arrays (node_beg / edge_beg are positions there until the blob is assembled).
struct GenomeOut {
  PackGenome g{};
};

struct Edge {
  int s, d;
  float w;
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

// Packing buffers of the tasks of one call, kept across calls so that a warm
// packer allocates nothing: scratch, the tasks' node and edge records, the
// genome table. One caller at a time uses the shared set; release() (from
// emr_pack_release) frees their memory, and the next call grows them again.
struct PackBuffers {
  static constexpr int kTasks = 16;
  std::mutex mu;
  Scratch scratch[kTasks];
  std::vector<PackNode> nodes[kTasks];
  std::vector<PackEdge> edges[kTasks];
  std::vector<GenomeOut> gs;
  static PackBuffers& get() {
    static PackBuffers* b = new PackBuffers();
    return *b;
  }
  void release() {
    std::lock_guard<std::mutex> lk(mu);
    for (int t = 0; t < kTasks; t++) {
      scratch[t] = Scratch();
      std::vector<PackNode>().swap(nodes[t]);
      std::vector<PackEdge>().swap(edges[t]);
    }
    std::vector<GenomeOut>().swap(gs);
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
// per-side variation flags for one genome.
emr_status pack_one(int64_t n0, int64_t n1, int64_t c0, int64_t c1, const int32_t* node_id,
                    const int32_t* node_kind, const int32_t* node_act, const float* node_bias,
                    const int32_t* conn_src, const int32_t* conn_dst, const float* conn_w,
                    const uint8_t* conn_en, Scratch& S, std::vector<PackNode>& nodes,
                    std::vector<PackEdge>& edges, GenomeOut* out) {
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
    std::stable_sort(S.es.begin(), S.es.end(),
                     [](const Edge& a, const Edge& b) { return a.d != b.d ? a.d < b.d : a.s < b.s; });
    size_t m = 0;
    for (size_t k = 0; k < S.es.size();) {
      Edge e = S.es[k++];
      while (k < S.es.size() && S.es[k].s == e.s && S.es[k].d == e.d) e.w += S.es[k++].w;
      S.es[m++] = e;
    }
    S.es.resize(m);
  }
  S.es.erase(std::remove_if(S.es.begin(), S.es.end(), [](const Edge& e) { return e.w == 0.f; }), S.es.end());
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
  S.reach.assign(n, 0);
  S.stack.assign(1, out_node);
  S.reach[out_node] = 1;
  while (!S.stack.empty()) {
    const int v = S.stack.back();
    S.stack.pop_back();
    for (int k = S.pred_beg[v]; k < S.pred_beg[v + 1]; k++)
      if (!S.reach[S.pred[k]]) { S.reach[S.pred[k]] = 1; S.stack.push_back(S.pred[k]); }
  }
  S.slot.assign(n, -1);
  S.kept.clear();
  for (int v : S.order)
    if (S.reach[v] && node_kind[n0 + v] >= EMR_KIND_HIDDEN) { S.slot[v] = int(S.kept.size()); S.kept.push_back(v); }
  if (S.kept.empty() || S.kept.back() != out_node) return EMR_ERR_ARG;  // output must be last
  if (S.kept.size() > 65535) return EMR_ERR_RANGE;
  const int nk = int(S.kept.size());
  const size_t nb = nodes.size();
  nodes.resize(nb + size_t(nk));  // value-initialised records
  PackNode* on = nodes.data() + nb;
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
  // in-edges from kept non-input nodes, grouped by destination (ascending source)
  S.in_beg.assign(nk + 1, 0);
  for (int t = 0; t < nk; t++) S.in_beg[t + 1] = S.in_beg[t] + S.in_cnt[t];
  if (S.in_beg[nk] > 65535) return EMR_ERR_RANGE;
  const size_t eb = edges.size();
  edges.resize(eb + size_t(S.in_beg[nk]));
  PackEdge* oe = edges.data() + eb;
  S.fill.assign(nk, 0);
  for (auto& e : S.es) {
    const int t = S.slot[e.d];
    if (t < 0 || node_kind[n0 + e.s] < EMR_KIND_HIDDEN) continue;
    oe[S.in_beg[t] + S.fill[t]++] = PackEdge{uint16_t(S.slot[e.s]), 0, e.w};
  }
  PackGenome& g = out->g;
  g = PackGenome{};
  g.node_beg = uint32_t(nb);
  g.edge_beg = uint32_t(eb);
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
  // per-task buffers kept across calls; a caller that finds them in use packs with its own
  PackBuffers& shared = PackBuffers::get();
  std::unique_lock<std::mutex> buf_lock(shared.mu, std::try_to_lock);
  std::unique_ptr<PackBuffers> own;
  if (!buf_lock.owns_lock()) own.reset(new PackBuffers());
  PackBuffers& B = own ? *own : shared;
  std::vector<GenomeOut>& gs = B.gs;
  gs.resize(size_t(P));
  // Genomes are independent: pack them on several host threads, each with its
  // own scratch; the lowest failing genome index is reported.
  const int hw = int(std::max(1u, std::thread::hardware_concurrency()));
  // a thread's share costs about as much to hand out as packing a few genomes
  const int n_threads = std::max(1, std::min({hw, PackBuffers::kTasks, P / 32}));
  emr_status t_rc[PackBuffers::kTasks];
  int32_t t_bad[PackBuffers::kTasks];
  std::vector<PackNode>* t_nodes = B.nodes;
  std::vector<PackEdge>* t_edges = B.edges;
  auto g_lo = [&](int t) { return int(int64_t(P) * t / n_threads); };
  auto work = [&](int t) {
    Scratch& scratch = B.scratch[t];
    t_rc[t] = EMR_OK;
    t_bad[t] = -1;
    t_nodes[t].clear();
    t_edges[t].clear();
    const int64_t n_lo = node_ptr[g_lo(t)], n_hi = node_ptr[g_lo(t + 1)];
    t_nodes[t].reserve(size_t(std::max<int64_t>(0, n_hi - n_lo)));
    for (int g = g_lo(t); g < g_lo(t + 1); g++) {
      emr_status rc = EMR_OK;
      if (node_ptr[g + 1] < node_ptr[g] || conn_ptr[g + 1] < conn_ptr[g]) rc = EMR_ERR_ARG;
      if (rc == EMR_OK)
        rc = pack_one(node_ptr[g], node_ptr[g + 1], conn_ptr[g], conn_ptr[g + 1], node_id, node_kind, node_act,
                      node_bias, conn_src, conn_dst, conn_w, conn_enabled, scratch, t_nodes[t], t_edges[t], &gs[g]);
      if (rc != EMR_OK) {
        t_rc[t] = rc;
        t_bad[t] = g;
        return;
      }
    }
  };
  if (n_threads == 1) {
    work(0);
  } else {
    WorkerPool::get().run(n_threads, work);
  }
  for (int t = 0; t < n_threads; t++)
    if (t_rc[t] != EMR_OK) {
      if (bad_genome) *bad_genome = t_bad[t];
      return t_rc[t];
    }
  size_t nn = 0, ne = 0;
  std::vector<size_t> t_nb(n_threads), t_eb(n_threads);  // each thread's first node / edge in the blob
  for (int t = 0; t < n_threads; t++) {
    t_nb[t] = nn;
    t_eb[t] = ne;
    nn += t_nodes[t].size();
    ne += t_edges[t].size();
  }
  PackHeader h{};
  h.magic = kPackMagic;
  h.version = kPackVersion;
  h.P = P;
  h.off_genomes = align16(sizeof(PackHeader));
  h.off_nodes = h.off_genomes + align16(sizeof(PackGenome) * size_t(P));
  h.off_edges = h.off_nodes + align16(sizeof(PackNode) * nn);
  h.total_bytes = h.off_edges + align16(sizeof(PackEdge) * ne);
  *used = size_t(h.total_bytes);
  if (cap < h.total_bytes) return EMR_ERR_CAPACITY;
  auto* base = static_cast<uint8_t*>(buf);
  // every record is written in full below; only the alignment gaps between sections are cleared
  auto clear = [&](uint64_t from, uint64_t to) {
    if (to > from) std::memset(base + from, 0, size_t(to - from));
  };
  clear(sizeof(PackHeader), h.off_genomes);
  clear(h.off_genomes + sizeof(PackGenome) * uint64_t(P), h.off_nodes);
  clear(h.off_nodes + sizeof(PackNode) * uint64_t(nn), h.off_edges);
  clear(h.off_edges + sizeof(PackEdge) * uint64_t(ne), h.total_bytes);
  auto* gt = reinterpret_cast<PackGenome*>(base + h.off_genomes);
  auto* nt = reinterpret_cast<PackNode*>(base + h.off_nodes);
  auto* et = reinterpret_cast<PackEdge*>(base + h.off_edges);
  for (int t = 0; t < n_threads; t++) {
    if (!t_nodes[t].empty()) std::memcpy(nt + t_nb[t], t_nodes[t].data(), t_nodes[t].size() * sizeof(PackNode));
    if (!t_edges[t].empty()) std::memcpy(et + t_eb[t], t_edges[t].data(), t_edges[t].size() * sizeof(PackEdge));
  }
  for (int t = 0; t < n_threads; t++)
    for (int g = g_lo(t); g < g_lo(t + 1); g++) {
      gs[g].g.node_beg += uint32_t(t_nb[t]);
      gs[g].g.edge_beg += uint32_t(t_eb[t]);
    }
  for (int g = 0; g < P; g++) {
    const PackGenome pg = gs[g].g;
    gt[g] = pg;
    h.max_nodes = std::max<int32_t>(h.max_nodes, pg.n_nodes);
    h.max_edges = std::max<int32_t>(h.max_edges, pg.n_edges);
    for (int s = 0; s < 2; s++) {
      h.max_varying[s] = std::max<int32_t>(h.max_varying[s], pg.n_varying[s]);
      h.max_vedges[s] = std::max<int32_t>(h.max_vedges[s], pg.n_vedges[s]);
    }
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
