// Substrate network assembly (host C++). ES-HyperNEAT's construction, which
// the paper's Section 2 summarises and Section 6 configures: Phase 1 connects
// each substrate input to the positions its outgoing query keeps (the hidden
// nodes), Phase 2 repeats that from every newly discovered hidden node for a
// fixed number of rounds, Phase 3 connects the hidden nodes that the incoming
// query of each substrate output keeps, and nodes that lie on no path from an
// input to an output are pruned. Every query round runs on the device path
// (emr_eval_prepare, emr_eval_filter, emr_mask_combine_types,
// emr_compact_records); the host keeps the graph.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstring>
#include <list>
#include <string>
#include <thread>
#include <unordered_map>
#include <vector>

#include "../../include/emr.h"
#include "emr_internal.h"

namespace {

inline size_t up256(size_t x) { return (x + 255) & ~size_t(255); }

// fn(g) for g in [0, n) on the library's host worker threads (genomes are independent).
template <class F>
void parallel_for(int32_t n, F fn) {
  const int hw = int(std::max(1u, std::thread::hardware_concurrency()));
  const int nt = std::max(1, std::min({hw, 16, n / 16}));
  if (nt == 1) {
    for (int32_t g = 0; g < n; g++) fn(g);
    return;
  }
  emr::host_parallel(nt, [&](int t) {
    for (int32_t g = int32_t(int64_t(n) * t / nt); g < int32_t(int64_t(n) * (t + 1) / nt); g++) fn(g);
  });
}

// Device workspace carve-up for one query batch of up to n_pairs pairs.
struct AsmLayout {
  size_t eval_bytes, cws_bytes;
  size_t off_a, off_b, off_side, off_count, off_eval, off_split, off_band, off_mask, off_cws, off_idx, off_w,
      off_cnt, off_off, total;
};

emr_status asm_layout(const void* pack_host, int32_t P, int32_t S, const emr_grid* g, int64_t list_cap,
                      AsmLayout* L) {
  // the record workspace depends on the pack and the number of pairs only: size it with a
  // per-genome query of S slots
  std::vector<float> a(size_t(P) * S, 0.f), b(size_t(P) * S, 0.f);
  std::vector<int32_t> side(size_t(P) * S, EMR_SIDE_OUT), count(size_t(P), S);
  emr_query q{};
  q.S = S;
  q.per_genome = 1;
  q.a_host = a.data();
  q.b_host = b.data();
  q.side_host = side.data();
  q.count_host = count.data();
  emr_status rc = emr_eval_workspace_size(pack_host, &q, &L->eval_bytes);
  if (rc != EMR_OK) return rc;
  const int64_t n_pairs = int64_t(P) * S;
  if (n_pairs > 0x7fffffffLL) return EMR_ERR_RANGE;
  rc = emr_compact_workspace_size(g, int32_t(n_pairs), &L->cws_bytes);
  if (rc != EMR_OK) return rc;
  size_t o = 0;
  L->off_a = o; o += up256(size_t(n_pairs) * 4);
  L->off_b = o; o += up256(size_t(n_pairs) * 4);
  L->off_side = o; o += up256(size_t(n_pairs) * 4);
  L->off_count = o; o += up256(size_t(P) * 4);
  L->off_eval = o; o += up256(L->eval_bytes);
  const size_t plane = size_t(n_pairs) * size_t(g->n_words) * 4;
  L->off_split = o; o += up256(plane);
  L->off_band = o; o += up256(plane);
  L->off_mask = o; o += up256(plane);
  L->off_cws = o; o += up256(L->cws_bytes);
  L->off_idx = o; o += up256(size_t(list_cap) * 4);
  L->off_w = o; o += up256(size_t(list_cap) * 4);
  L->off_cnt = o; o += up256(size_t(n_pairs) * 8);
  L->off_off = o; o += up256(size_t(n_pairs + 1) * 8);
  L->total = o;
  return EMR_OK;
}

struct Conn {
  int64_t src, dst;  // global index of a hidden position, or -1 - k for substrate node k
  float w;
  uint8_t type;
};

struct GenomeGraph {
  std::vector<int64_t> hidden;                 // discovered positions, discovery order
  std::unordered_map<int64_t, int32_t> seen;   // position -> index in hidden
  std::vector<Conn> conns, to_outputs;         // phase 1-2 connections; phase 3 candidates
  size_t frontier_beg = 0, frontier_end = 0;   // hidden[frontier_beg, frontier_end): next round's sources
};

// Grid coordinates (Eq. 1) of global index p, exact in fp32.
void coords(int64_t p, float* x, float* y) {
  int32_t d, i, j;
  emr_index_to_ij(p, &d, &i, &j);
  const double s = std::ldexp(1.0, -(d + 1));
  *x = float((2.0 * i + 1.0) * s - 1.0);
  *y = float((2.0 * j + 1.0) * s - 1.0);
}

// Connection type of a connection from src to dst (Section 6), both as points.
uint8_t conn_type(float xs, float ys, float xt, float yt) {
  if (xs == xt && ys == yt) return 3;
  return ys < yt ? 0 : ys > yt ? 1 : 2;
}

// One query batch on the device: slots (host arrays) -> lists on the host.
struct Runner {
  const void* pack_host;
  const void* pack_dev;
  const emr_grid* g;
  float theta, band, w_min;
  int32_t mode, types, P;
  uint8_t* ws;
  AsmLayout L;
  int64_t list_cap;
  cudaStream_t st;
  std::vector<int64_t> offsets;
  std::vector<int32_t> idx;
  std::vector<float> w;

  emr_status run(int32_t S, int32_t per_genome, const std::vector<float>& a, const std::vector<float>& b,
                 const std::vector<int32_t>& side, const std::vector<int32_t>& count) {
    const size_t ns = a.size();
    float* a_dev = reinterpret_cast<float*>(ws + L.off_a);
    float* b_dev = reinterpret_cast<float*>(ws + L.off_b);
    int32_t* side_dev = reinterpret_cast<int32_t*>(ws + L.off_side);
    int32_t* count_dev = reinterpret_cast<int32_t*>(ws + L.off_count);
    if (cudaMemcpyAsync(a_dev, a.data(), ns * 4, cudaMemcpyHostToDevice, st) != cudaSuccess ||
        cudaMemcpyAsync(b_dev, b.data(), ns * 4, cudaMemcpyHostToDevice, st) != cudaSuccess ||
        cudaMemcpyAsync(side_dev, side.data(), ns * 4, cudaMemcpyHostToDevice, st) != cudaSuccess ||
        (per_genome && cudaMemcpyAsync(count_dev, count.data(), size_t(P) * 4, cudaMemcpyHostToDevice, st) !=
                           cudaSuccess))
      return EMR_ERR_CUDA;
    emr_query q{};
    q.S = S;
    q.per_genome = per_genome;
    q.a_host = a.data();
    q.b_host = b.data();
    q.side_host = side.data();
    q.count_host = per_genome ? count.data() : nullptr;
    q.a_dev = a_dev;
    q.b_dev = b_dev;
    q.side_dev = side_dev;
    q.count_dev = per_genome ? count_dev : nullptr;
    const int64_t n_pairs = int64_t(P) * S;
    uint32_t* split = reinterpret_cast<uint32_t*>(ws + L.off_split);
    uint32_t* bandb = reinterpret_cast<uint32_t*>(ws + L.off_band);
    uint32_t* mask = reinterpret_cast<uint32_t*>(ws + L.off_mask);
    int64_t* off_dev = reinterpret_cast<int64_t*>(ws + L.off_off);
    emr_status rc;
    if ((rc = emr_eval_prepare(pack_host, pack_dev, &q, ws + L.off_eval, L.eval_bytes, st)) != EMR_OK) return rc;
    if ((rc = emr_eval_filter(pack_host, &q, g, theta, band, w_min, split, bandb, nullptr, ws + L.off_eval,
                              L.eval_bytes, st)) != EMR_OK)
      return rc;
    if ((rc = emr_mask_combine_types(split, bandb, &q, g, int32_t(n_pairs), mode, types, mask, st)) != EMR_OK)
      return rc;
    if ((rc = emr_compact_records(mask, pack_host, &q, ws + L.off_eval, L.eval_bytes, g,
                                  reinterpret_cast<int32_t*>(ws + L.off_idx), reinterpret_cast<float*>(ws + L.off_w),
                                  list_cap, reinterpret_cast<int64_t*>(ws + L.off_cnt), off_dev, ws + L.off_cws,
                                  L.cws_bytes, st)) != EMR_OK)
      return rc;
    offsets.resize(size_t(n_pairs + 1));
    if (cudaMemcpyAsync(offsets.data(), off_dev, size_t(n_pairs + 1) * 8, cudaMemcpyDeviceToHost, st) != cudaSuccess ||
        cudaStreamSynchronize(st) != cudaSuccess)
      return EMR_ERR_CUDA;
    const int64_t total = offsets[size_t(n_pairs)];
    if (total > list_cap) return EMR_ERR_CAPACITY;
    idx.resize(size_t(total));
    w.resize(size_t(total));
    if (total > 0 &&
        (cudaMemcpyAsync(idx.data(), ws + L.off_idx, size_t(total) * 4, cudaMemcpyDeviceToHost, st) != cudaSuccess ||
         cudaMemcpyAsync(w.data(), ws + L.off_w, size_t(total) * 4, cudaMemcpyDeviceToHost, st) != cudaSuccess ||
         cudaStreamSynchronize(st) != cudaSuccess))
      return EMR_ERR_CUDA;
    return EMR_OK;
  }
};

// ---- connection cache --------------------------------------------------------------
//
// Discovered lists keyed by (genome content, query slot, query parameters). A
// genome is identified by the bytes of its packed records, so an identical
// genome in a later population (an elite, or a clone) hits; entries are evicted
// least recently used beyond the byte budget.

struct SlotKey {
  int64_t genome;  // id in the cache's genome table
  uint32_t a, b;   // slot coordinates (fp32 bits)
  int32_t side, D, mode, types;
  uint32_t theta, band, w_min;
  bool operator==(const SlotKey& o) const { return std::memcmp(this, &o, sizeof(SlotKey)) == 0; }
};
struct SlotKeyHash {
  size_t operator()(const SlotKey& k) const {
    const auto* p = reinterpret_cast<const uint8_t*>(&k);
    uint64_t h = 1469598103934665603ull;  // FNV-1a
    for (size_t i = 0; i < sizeof(SlotKey); i++) h = (h ^ p[i]) * 1099511628211ull;
    return size_t(h);
  }
};

struct List {
  std::vector<int32_t> idx;
  std::vector<float> w;
};

struct Slot {
  float a, b;
  int32_t side;
};

}  // namespace

struct emr_cache {
  size_t max_bytes = 0, bytes = 0;
  int64_t hits = 0, misses = 0;
  std::unordered_map<std::string, int64_t> genomes;
  std::list<SlotKey> lru;  // most recent first
  struct Entry {
    std::list<SlotKey>::iterator at;
    List list;
  };
  std::unordered_map<SlotKey, Entry, SlotKeyHash> map;

  static size_t cost(const List& l) { return l.idx.size() * 8 + sizeof(Entry) + sizeof(SlotKey) + 64; }
  bool get(const SlotKey& k, List* out) {
    auto it = map.find(k);
    if (it == map.end()) { misses++; return false; }
    hits++;
    lru.splice(lru.begin(), lru, it->second.at);
    *out = it->second.list;
    return true;
  }
  void put(const SlotKey& k, const List& l) {
    if (map.count(k)) return;
    const size_t c = cost(l);
    if (c > max_bytes) return;
    while (bytes + c > max_bytes && !lru.empty()) {
      auto it = map.find(lru.back());
      bytes -= cost(it->second.list);
      map.erase(it);
      lru.pop_back();
    }
    lru.push_front(k);
    map.emplace(k, Entry{lru.begin(), l});
    bytes += c;
  }
};

namespace {

// Content identity of genome g of a packed blob: its kept node and edge records.
std::string genome_bytes(const void* pack_host, int32_t g) {
  const auto* base = static_cast<const uint8_t*>(pack_host);
  const auto* h = emr::pack_header(pack_host);
  const auto* gt = reinterpret_cast<const emr::PackGenome*>(base + h->off_genomes) + g;
  std::string s;
  s.append(reinterpret_cast<const char*>(&gt->n_nodes), 4);
  s.append(reinterpret_cast<const char*>(base + h->off_nodes) + size_t(gt->node_beg) * sizeof(emr::PackNode),
           size_t(gt->n_nodes) * sizeof(emr::PackNode));
  s.append(reinterpret_cast<const char*>(base + h->off_edges) + size_t(gt->edge_beg) * sizeof(emr::PackEdge),
           size_t(gt->n_edges) * sizeof(emr::PackEdge));
  return s;
}

uint32_t bits(float f) {
  uint32_t u;
  std::memcpy(&u, &f, 4);
  return u;
}

// Lists of every genome's slots (slots[g]): from the cache where present, the
// rest from the device in batches of at most slots_max slots per genome, then
// added to the cache.
emr_status query_slots(Runner& R, emr_cache* cache, const std::vector<int64_t>& gid, int32_t D,
                       const std::vector<std::vector<Slot>>& slots, int32_t slots_max,
                       std::vector<std::vector<List>>& out) {
  const int32_t P = R.P;
  auto key = [&](int32_t g, const Slot& sl) {
    SlotKey k;
    std::memset(&k, 0, sizeof(k));
    k.genome = gid[size_t(g)];
    k.a = bits(sl.a);
    k.b = bits(sl.b);
    k.side = sl.side;
    k.D = D;
    k.mode = R.mode;
    k.types = R.types;
    k.theta = bits(R.theta);
    k.band = bits(R.band);
    k.w_min = bits(R.w_min);
    return k;
  };
  out.assign(size_t(P), {});
  std::vector<std::vector<int32_t>> miss(static_cast<size_t>(P));
  for (int32_t g = 0; g < P; g++) {
    out[size_t(g)].resize(slots[size_t(g)].size());
    for (size_t k = 0; k < slots[size_t(g)].size(); k++)
      if (!cache || !cache->get(key(g, slots[size_t(g)][k]), &out[size_t(g)][k]))
        miss[size_t(g)].push_back(int32_t(k));
  }
  std::vector<size_t> cursor(static_cast<size_t>(P), 0);
  for (;;) {
    int32_t S = 0;
    for (int32_t g = 0; g < P; g++)
      S = std::max<int32_t>(S, int32_t(std::min<size_t>(size_t(slots_max), miss[size_t(g)].size() - cursor[size_t(g)])));
    if (S == 0) return EMR_OK;
    std::vector<float> a(size_t(P) * S, 0.f), b(size_t(P) * S, 0.f);
    std::vector<int32_t> side(size_t(P) * S, EMR_SIDE_OUT), count(static_cast<size_t>(P), 0);
    for (int32_t g = 0; g < P; g++) {
      const int32_t n = int32_t(std::min<size_t>(size_t(S), miss[size_t(g)].size() - cursor[size_t(g)]));
      count[size_t(g)] = n;
      for (int32_t s = 0; s < n; s++) {
        const Slot& sl = slots[size_t(g)][size_t(miss[size_t(g)][cursor[size_t(g)] + size_t(s)])];
        a[size_t(g) * S + s] = sl.a;
        b[size_t(g) * S + s] = sl.b;
        side[size_t(g) * S + s] = sl.side;
      }
    }
    emr_status rc = R.run(S, 1, a, b, side, count);
    if (rc != EMR_OK) return rc;
    for (int32_t g = 0; g < P; g++) {
      for (int32_t s = 0; s < count[size_t(g)]; s++) {
        const int32_t k = miss[size_t(g)][cursor[size_t(g)] + size_t(s)];
        const int64_t r = int64_t(g) * S + s;
        List& l = out[size_t(g)][size_t(k)];
        l.idx.assign(R.idx.begin() + R.offsets[size_t(r)], R.idx.begin() + R.offsets[size_t(r) + 1]);
        l.w.assign(R.w.begin() + R.offsets[size_t(r)], R.w.begin() + R.offsets[size_t(r) + 1]);
        if (cache) cache->put(key(g, slots[size_t(g)][size_t(k)]), l);
      }
      cursor[size_t(g)] += size_t(count[size_t(g)]);
    }
  }
}

}  // namespace

extern "C" {

emr_status emr_assemble_workspace_size(const void* pack_host, int32_t n_in, int32_t n_out, int32_t slots_max,
                                       const emr_grid* grid, int64_t list_cap, size_t* bytes) {
  int32_t P = 0;
  if (!bytes || !grid || n_in <= 0 || n_out <= 0 || slots_max <= 0 || list_cap <= 0) return EMR_ERR_ARG;
  emr_status rc = emr_pack_info(pack_host, &P, nullptr, nullptr);
  if (rc != EMR_OK) return rc;
  AsmLayout L;
  if ((rc = asm_layout(pack_host, P, std::max(slots_max, n_in + n_out), grid, list_cap, &L)) != EMR_OK) return rc;
  *bytes = L.total;
  return EMR_OK;
}

emr_status emr_assemble(const void* pack_host, const void* pack_dev, int32_t n_in, const float* in_x,
                        const float* in_y, int32_t n_out, const float* out_x, const float* out_y,
                        const emr_grid* grid, float theta, float band, float w_min, int32_t mode, int32_t types,
                        int32_t rounds, int32_t slots_max, void* ws, size_t ws_bytes, int64_t list_cap,
                        int64_t* node_off, int32_t* hidden, int64_t hidden_cap, int64_t* conn_off, int32_t* conn_src,
                        int32_t* conn_dst, float* conn_w, uint8_t* conn_type_out, int64_t conn_cap, emr_cache* cache,
                        void* stream) {
  if (!pack_dev || !ws || n_in <= 0 || n_out <= 0 || !in_x || !in_y || !out_x || !out_y || rounds < 0 ||
      slots_max <= 0 || list_cap <= 0 || !node_off || !conn_off || hidden_cap < 0 || conn_cap < 0 ||
      (hidden_cap > 0 && !hidden) || (conn_cap > 0 && (!conn_src || !conn_dst || !conn_w || !conn_type_out)))
    return EMR_ERR_ARG;
  if ((mode != EMR_EAGER && mode != EMR_GATED) || types < 0 || types > EMR_CONN_ALL) return EMR_ERR_ARG;
  int32_t P = 0;
  emr_status rc = emr_pack_info(pack_host, &P, nullptr, nullptr);
  if (rc != EMR_OK) return rc;
  Runner R{pack_host, pack_dev, grid, theta, band, w_min, mode, types, P, static_cast<uint8_t*>(ws), {}, list_cap,
           static_cast<cudaStream_t>(stream), {}, {}, {}};
  const int32_t S_max = std::max(slots_max, n_in + n_out);
  if ((rc = asm_layout(pack_host, P, S_max, grid, list_cap, &R.L)) != EMR_OK) return rc;
  if (ws_bytes < R.L.total) return EMR_ERR_CAPACITY;
  std::vector<GenomeGraph> G(static_cast<size_t>(P));

  std::vector<int64_t> gid(static_cast<size_t>(P), 0);
  if (cache)
    for (int32_t g = 0; g < P; g++)
      gid[size_t(g)] = cache->genomes.emplace(genome_bytes(pack_host, g), int64_t(cache->genomes.size())).first->second;

  // Phase 1 and the queries of Phase 3: outgoing from each input, incoming to each output
  {
    std::vector<Slot> io;
    for (int32_t k = 0; k < n_in; k++) io.push_back({in_x[k], in_y[k], EMR_SIDE_OUT});
    for (int32_t k = 0; k < n_out; k++) io.push_back({out_x[k], out_y[k], EMR_SIDE_IN});
    std::vector<std::vector<Slot>> slots(static_cast<size_t>(P), io);
    std::vector<std::vector<List>> lists;
    if ((rc = query_slots(R, cache, gid, grid->D, slots, n_in + n_out, lists)) != EMR_OK) return rc;
    parallel_for(P, [&](int32_t g) {
      GenomeGraph& gg = G[size_t(g)];
      for (int32_t s = 0; s < n_in + n_out; s++) {
        const List& l = lists[size_t(g)][size_t(s)];
        for (size_t e = 0; e < l.idx.size(); e++) {
          const int64_t p = l.idx[e];
          float x, y;
          coords(p, &x, &y);
          if (s < n_in) {
            gg.conns.push_back({-1 - s, p, l.w[e], conn_type(in_x[s], in_y[s], x, y)});
            if (gg.seen.emplace(p, int32_t(gg.hidden.size())).second) gg.hidden.push_back(p);
          } else {
            const int32_t o = s - n_in;
            gg.to_outputs.push_back({p, -1 - (n_in + o), l.w[e], conn_type(x, y, out_x[o], out_y[o])});
          }
        }
      }
      gg.frontier_beg = 0;
      gg.frontier_end = gg.hidden.size();
    });
  }

  // Phase 2: outgoing queries from each newly discovered hidden node, `rounds` times
  for (int32_t round = 0; round < rounds; round++) {
    std::vector<std::vector<Slot>> slots(static_cast<size_t>(P));
    parallel_for(P, [&](int32_t g) {
      const GenomeGraph& gg = G[size_t(g)];
      for (size_t h = gg.frontier_beg; h < gg.frontier_end; h++) {
        Slot sl{0.f, 0.f, EMR_SIDE_OUT};
        coords(gg.hidden[h], &sl.a, &sl.b);
        slots[size_t(g)].push_back(sl);
      }
    });
    std::vector<std::vector<List>> lists;
    if ((rc = query_slots(R, cache, gid, grid->D, slots, slots_max, lists)) != EMR_OK) return rc;
    parallel_for(P, [&](int32_t g) {
      GenomeGraph& gg = G[size_t(g)];
      for (size_t k = 0; k < slots[size_t(g)].size(); k++) {
        const int64_t src = gg.hidden[gg.frontier_beg + k];
        const Slot& sl = slots[size_t(g)][k];
        const List& l = lists[size_t(g)][k];
        for (size_t e = 0; e < l.idx.size(); e++) {
          const int64_t p = l.idx[e];
          float x, y;
          coords(p, &x, &y);
          gg.conns.push_back({src, p, l.w[e], conn_type(sl.a, sl.b, x, y)});
          if (gg.seen.emplace(p, int32_t(gg.hidden.size())).second) gg.hidden.push_back(p);
        }
      }
      gg.frontier_beg = gg.frontier_end;
      gg.frontier_end = gg.hidden.size();
    });
  }

  // Phase 3 and pruning; nodes are numbered inputs, outputs, then kept hidden
  // positions in ascending global index; connections sorted by (dst, src)
  struct Out { int32_t src, dst; float w; uint8_t t; };
  std::vector<std::vector<int64_t>> kept_of(static_cast<size_t>(P));
  std::vector<std::vector<Out>> out_of(static_cast<size_t>(P));
  parallel_for(P, [&](int32_t g) {
    GenomeGraph& gg = G[size_t(g)];
    for (const Conn& c : gg.to_outputs)
      if (gg.seen.count(c.src)) gg.conns.push_back(c);
    const int32_t H = int32_t(gg.hidden.size()), NS = n_in + n_out, N = NS + H;
    auto node = [&](int64_t v) -> int32_t { return v < 0 ? int32_t(-1 - v) : NS + gg.seen.at(v); };
    std::vector<std::vector<int32_t>> fwd(static_cast<size_t>(N)), bwd(static_cast<size_t>(N));
    for (const Conn& c : gg.conns) {
      fwd[size_t(node(c.src))].push_back(node(c.dst));
      bwd[size_t(node(c.dst))].push_back(node(c.src));
    }
    auto reach = [&](const std::vector<std::vector<int32_t>>& adj, int32_t beg, int32_t end) {
      std::vector<uint8_t> vis(static_cast<size_t>(N), 0);
      std::vector<int32_t> stack;
      for (int32_t v = beg; v < end; v++) { vis[size_t(v)] = 1; stack.push_back(v); }
      while (!stack.empty()) {
        const int32_t v = stack.back();
        stack.pop_back();
        for (int32_t u : adj[size_t(v)])
          if (!vis[size_t(u)]) { vis[size_t(u)] = 1; stack.push_back(u); }
      }
      return vis;
    };
    const std::vector<uint8_t> from_in = reach(fwd, 0, n_in), to_out = reach(bwd, n_in, NS);
    std::vector<int64_t> kept;
    for (int32_t h = 0; h < H; h++)
      if (from_in[size_t(NS + h)] && to_out[size_t(NS + h)]) kept.push_back(gg.hidden[size_t(h)]);
    std::sort(kept.begin(), kept.end());
    std::unordered_map<int64_t, int32_t> id;
    for (size_t k = 0; k < kept.size(); k++) id[kept[k]] = NS + int32_t(k);
    auto new_id = [&](int64_t v) -> int32_t {
      if (v < 0) return int32_t(-1 - v);
      auto it = id.find(v);
      return it == id.end() ? -1 : it->second;
    };
    std::vector<Out>& outc = out_of[size_t(g)];
    for (const Conn& c : gg.conns) {
      const int32_t s = new_id(c.src), d = new_id(c.dst);
      if (s >= 0 && d >= 0) outc.push_back({s, d, c.w, c.type});
    }
    std::sort(outc.begin(), outc.end(), [](const Out& x, const Out& y) {
      return x.dst != y.dst ? x.dst < y.dst : x.src < y.src;
    });
    kept_of[size_t(g)] = std::move(kept);
    gg = GenomeGraph();  // release the graph early
  });
  int64_t n_hidden_total = 0, n_conn_total = 0;
  node_off[0] = 0;
  conn_off[0] = 0;
  for (int32_t g = 0; g < P; g++) {
    const std::vector<int64_t>& kept = kept_of[size_t(g)];
    const std::vector<Out>& outc = out_of[size_t(g)];
    for (size_t k = 0; k < kept.size(); k++, n_hidden_total++)
      if (n_hidden_total < hidden_cap) hidden[n_hidden_total] = int32_t(kept[k]);
    for (size_t k = 0; k < outc.size(); k++, n_conn_total++)
      if (n_conn_total < conn_cap) {
        conn_src[n_conn_total] = outc[k].src;
        conn_dst[n_conn_total] = outc[k].dst;
        conn_w[n_conn_total] = outc[k].w;
        conn_type_out[n_conn_total] = outc[k].t;
      }
    node_off[g + 1] = n_hidden_total;
    conn_off[g + 1] = n_conn_total;
  }
  return (n_hidden_total > hidden_cap || n_conn_total > conn_cap) ? EMR_ERR_CAPACITY : EMR_OK;
}

emr_status emr_cache_create(size_t max_bytes, emr_cache** cache) {
  if (!cache) return EMR_ERR_ARG;
  *cache = nullptr;
  try {
    *cache = new emr_cache();
  } catch (...) {
    return EMR_ERR_ALLOC;
  }
  (*cache)->max_bytes = max_bytes;
  return EMR_OK;
}

emr_status emr_cache_destroy(emr_cache* cache) {
  delete cache;
  return EMR_OK;
}

emr_status emr_cache_clear(emr_cache* cache) {
  if (!cache) return EMR_ERR_ARG;
  const size_t mb = cache->max_bytes;
  *cache = emr_cache();
  cache->max_bytes = mb;
  return EMR_OK;
}

emr_status emr_cache_stats(const emr_cache* cache, int64_t* hits, int64_t* misses, int64_t* entries,
                           int64_t* bytes) {
  if (!cache) return EMR_ERR_ARG;
  if (hits) *hits = cache->hits;
  if (misses) *misses = cache->misses;
  if (entries) *entries = int64_t(cache->map.size());
  if (bytes) *bytes = int64_t(cache->bytes);
  return EMR_OK;
}

}  // extern "C"
