// Internal layouts shared by libemr's host code and kernels (not part of the ABI).
#pragma once

#include <stdint.h>

#include <functional>

#include "../../include/emr.h"

namespace emr {

constexpr uint32_t kPackMagic = 0x504d5245u;  // "EMRP"
constexpr uint32_t kPackVersion = 2;

// Packed population blob: header, genome table, node records, edge records.
// Every section starts on a 16-byte boundary; offsets are bytes from the blob start.
struct PackHeader {
  uint32_t magic, version;
  int32_t P;
  int32_t max_nodes;       // kept non-input nodes of the largest genome
  int32_t max_varying[2];  // per query side (EMR_SIDE_OUT, EMR_SIDE_IN)
  int32_t max_vedges[2];   // edges between varying nodes, per side
  int32_t max_edges;       // edges between kept non-input nodes
  int32_t reserved;
  uint64_t off_genomes, off_nodes, off_edges, total_bytes;
};
static_assert(sizeof(PackHeader) == 72, "pack header layout");

struct PackGenome {
  uint32_t node_beg;       // first node record
  uint32_t edge_beg;       // first edge record
  uint16_t n_nodes;        // kept non-input nodes, topological order (output last)
  uint16_t n_edges;        // edges between them
  uint16_t n_varying[2];   // nodes whose value varies over the grid, per side
  uint16_t n_vedges[2];    // edges whose source and destination both vary, per side
  uint32_t cost[2];        // per-query work estimate, per side (scheduling only)
  uint16_t n_joint[2];     // varying nodes that depend on both grid coordinates, per side
};
static_assert(sizeof(PackGenome) == 32, "pack genome layout");

struct PackNode {
  uint8_t act;             // EMR_ACT_*
  uint8_t vary;            // bit s: varies over the grid under query side s
  uint8_t axes;            // bits 2 s, 2 s + 1: depends on the grid x, y coordinate under query side s
  uint8_t reserved;
  uint16_t edge_beg;       // first in-edge, relative to the genome's edge_beg
  uint16_t edge_cnt;       // in-edges from kept non-input nodes
  float bias;
  float w_in[5];           // summed weights of in-connections from x1, y1, x2, y2, bias
};
static_assert(sizeof(PackNode) == 32, "pack node layout");

// Grid coordinates a varying node depends on (PackNode::axes per side; the
// records' node and edge fields): x only, y only, or both ("joint").
constexpr uint32_t kAxisX = 1, kAxisY = 2, kAxisXY = 3;

struct PackEdge {
  uint16_t src;            // source: index among the genome's kept non-input nodes
  uint16_t reserved;
  float w;
};
static_assert(sizeof(PackEdge) == 8, "pack edge layout");

inline const PackHeader* pack_header(const void* blob) { return static_cast<const PackHeader*>(blob); }

// fn(0 .. n-1) on the library's persistent host worker threads and the caller;
// returns when every call has returned (emr_pack.cpp).
void host_parallel(int n, const std::function<void(int)>& fn);

// Grid helpers (Eq. 1 numbering, depth-major Morton).
inline int64_t level_offset(int d) { return ((int64_t(1) << (2 * (d + 1))) - 4) / 3; }
inline int64_t halo_offset(int d) { return 8 * ((int64_t(1) << d) - 1); }

// Evaluation tiles: depth d is covered by square Morton blocks of side
// min(2^{d+1}, kTileSide); tiles are numbered depth by depth.
constexpr int kTileLog = 6;
constexpr int kTileSide = 1 << kTileLog;
inline int tile_side(int d) { return (d + 1) < kTileLog ? (1 << (d + 1)) : kTileSide; }
inline int64_t tiles_in_level(int d) { return (d + 1) <= kTileLog ? 1 : (int64_t(1) << (2 * (d + 1 - kTileLog))); }

}  // namespace emr
