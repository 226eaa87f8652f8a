// libemr device code for sm_103a: per-pair CPPN specialisation, tiled CPPN
// evaluation with the fused variance/band epilogue, filter planes, mask
// combination and ordered compaction.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstring>
#include <utility>
#include <vector>

#include "emr_internal.h"

using namespace emr;

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kBlock = 128;  // threads per evaluation tile CTA

// Programmatic dependent launch: a kernel launched to overlap its predecessor
// (launch_overlapped) runs pdl_wait() before it reads the predecessor's results,
// which returns once the predecessor has completed and its writes are visible
// (at once for a kernel launched the ordinary way); pdl_trigger() lets the next
// such launch begin.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
// A launch that overlaps its predecessor without reading its results still has to
// complete after it (later kernels in the stream read every launch's output): its
// last CTA waits for the predecessor as it exits, after its own work, so that a
// chain of such launches adds no CTA lifetime per launch to the stream's timeline.
struct PdlWaitAtExit {
  bool on;
  __device__ __forceinline__ ~PdlWaitAtExit() {
    if (on) pdl_wait();
  }
};
__device__ __forceinline__ bool last_cta() {
  return blockIdx.x == gridDim.x - 1 && blockIdx.y == gridDim.y - 1 && blockIdx.z == gridDim.z - 1;
}

// ---- grid arithmetic ---------------------------------------------------------

__host__ __device__ __forceinline__ uint32_t compact1by1(uint32_t x) {
  x &= 0x55555555u;
  x = (x | (x >> 1)) & 0x33333333u;
  x = (x | (x >> 2)) & 0x0f0f0f0fu;
  x = (x | (x >> 4)) & 0x00ff00ffu;
  x = (x | (x >> 8)) & 0x0000ffffu;
  return x;
}
__host__ __device__ __forceinline__ uint32_t spread1by1(uint32_t x) {
  x &= 0x0000ffffu;
  x = (x | (x << 8)) & 0x00ff00ffu;
  x = (x | (x << 4)) & 0x0f0f0f0fu;
  x = (x | (x << 2)) & 0x33333333u;
  x = (x | (x << 1)) & 0x55555555u;
  return x;
}
__device__ __forceinline__ uint32_t morton2(uint32_t i, uint32_t j) { return spread1by1(i) | (spread1by1(j) << 1); }

// Eq. 1 coordinate of grid index i at depth d: (2i+1) 2^-(d+1) - 1, exact in fp32 for d <= 22.
__device__ __forceinline__ float grid_coord(int i, float scale) { return fmaf(float(2 * i + 1), scale, -1.0f); }

// ---- activations (fp32) --------------------------------------------------------
// All transcendental parts run on the MUFU (special function unit) through its
// approximate instructions with denormal flushing (values below 2^-126 only
// move by less than 2^-126): sigmoid(z) = 1 / (1 + 2^(-z log2 e)),
// tanh(z) = 1 - 2 / (1 + 2^(2 z log2 e)), gauss(z) = 2^(-z^2 log2 e), and sin
// after a two-constant Cody-Waite reduction by 2 pi (constants: 2 pi rounded
// to fp32 and the fp32 rounding of the remainder; the multiple k is rounded to
// nearest with the 1.5 * 2^23 shift, valid for |z| < 2^24).
constexpr float kTwoPiHi = 0x1.921fb6p+2f;
constexpr float kTwoPiLo = -0x1.777a5cp-23f;
constexpr float kInvTwoPi = 0x1.45f306p-3f;
constexpr float kLog2e = 0x1.715476p+0f;
constexpr float kRoundShift = 0x1.8p+23f;

__device__ __forceinline__ float mufu_ex2(float x) {
  float r;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}
__device__ __forceinline__ float mufu_rcp(float x) {
  float r;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}
__device__ __forceinline__ float mufu_sin(float x) {
  float r;
  asm("sin.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}

__device__ __forceinline__ float act_sigmoid(float z) { return mufu_rcp(1.0f + mufu_ex2(z * -kLog2e)); }
__device__ __forceinline__ float act_tanh(float z) {
  return fmaf(-2.0f, mufu_rcp(1.0f + mufu_ex2(z * (2.0f * kLog2e))), 1.0f);
}
__device__ __forceinline__ float act_gauss(float z) { return mufu_ex2(z * (z * -kLog2e)); }
__device__ __forceinline__ float act_sin(float z) {
  const float k = fmaf(z, kInvTwoPi, kRoundShift) - kRoundShift;
  float r = fmaf(-k, kTwoPiHi, z);
  r = fmaf(-k, kTwoPiLo, r);
  return mufu_sin(r);
}

__device__ __forceinline__ float act_apply(int a, float z) {
  switch (a) {
    case EMR_ACT_SIGMOID: return act_sigmoid(z);
    case EMR_ACT_TANH: return act_tanh(z);
    case EMR_ACT_GAUSS: return act_gauss(z);
    case EMR_ACT_SIN: return act_sin(z);
    case EMR_ACT_ABS: return fabsf(z);
    default: return z;
  }
}

__device__ __forceinline__ void act_apply4(int a, float& z0, float& z1, float& z2, float& z3) {
  switch (a) {
    case EMR_ACT_SIGMOID: z0 = act_sigmoid(z0); z1 = act_sigmoid(z1); z2 = act_sigmoid(z2); z3 = act_sigmoid(z3); break;
    case EMR_ACT_TANH: z0 = act_tanh(z0); z1 = act_tanh(z1); z2 = act_tanh(z2); z3 = act_tanh(z3); break;
    case EMR_ACT_GAUSS: z0 = act_gauss(z0); z1 = act_gauss(z1); z2 = act_gauss(z2); z3 = act_gauss(z3); break;
    case EMR_ACT_SIN: z0 = act_sin(z0); z1 = act_sin(z1); z2 = act_sin(z2); z3 = act_sin(z3); break;
    case EMR_ACT_ABS: z0 = fabsf(z0); z1 = fabsf(z1); z2 = fabsf(z2); z3 = fabsf(z3); break;
    default: break;
  }
}

// ---- packed pairs of fp32 -----------------------------------------------------------
// Two fp32 values in one 64-bit register pair, for the f32x2 add / mul / fma
// instructions: one issue slot for two lanes' worth of arithmetic, each half
// rounded exactly as the scalar instruction rounds it (so a packed evaluation
// gives the scalar one's bits). MUFU operations stay scalar, on the halves.
typedef unsigned long long f2;
__device__ __forceinline__ f2 f2_pack(float lo, float hi) {
  f2 r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void f2_unpack(f2 v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ float f2_lo(f2 v) {
  float lo, hi;
  f2_unpack(v, lo, hi);
  return lo;
}
__device__ __forceinline__ f2 f2_add(f2 a, f2 b) {
  f2 r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ f2 f2_mul(f2 a, f2 b) {
  f2 r;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ f2 f2_fma(f2 a, f2 b, f2 c) {
  f2 r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
  return r;
}
__device__ __forceinline__ f2 f2_splat(float c) { return f2_pack(c, c); }
__device__ __forceinline__ f2 f2_ex2(f2 v) {
  float a, b;
  f2_unpack(v, a, b);
  return f2_pack(mufu_ex2(a), mufu_ex2(b));
}
__device__ __forceinline__ f2 f2_rcp(f2 v) {
  float a, b;
  f2_unpack(v, a, b);
  return f2_pack(mufu_rcp(a), mufu_rcp(b));
}
// The activations above, on pairs, operation for operation: sigmoid and tanh
// add 1 to the power of two, sin's reduction computes fma(k, -c, r) for
// fma(-k, c, r) (the same exact product) and adds -shift for "- shift".
template <int NPP>
__device__ __forceinline__ void act_apply_pairs(int a, f2 (&z)[NPP]) {
  switch (a) {
    case EMR_ACT_SIGMOID: {
      const f2 c = f2_splat(-kLog2e), one = f2_splat(1.0f);
#pragma unroll
      for (int p = 0; p < NPP; p++) z[p] = f2_rcp(f2_add(one, f2_ex2(f2_mul(z[p], c))));
      break;
    }
    case EMR_ACT_TANH: {
      const f2 c = f2_splat(2.0f * kLog2e), one = f2_splat(1.0f), m2 = f2_splat(-2.0f);
#pragma unroll
      for (int p = 0; p < NPP; p++) z[p] = f2_fma(m2, f2_rcp(f2_add(one, f2_ex2(f2_mul(z[p], c)))), one);
      break;
    }
    case EMR_ACT_GAUSS: {
      const f2 c = f2_splat(-kLog2e);
#pragma unroll
      for (int p = 0; p < NPP; p++) z[p] = f2_ex2(f2_mul(z[p], f2_mul(z[p], c)));
      break;
    }
    case EMR_ACT_SIN: {
      const f2 inv = f2_splat(kInvTwoPi), sh = f2_splat(kRoundShift), nsh = f2_splat(-kRoundShift);
      const f2 nhi = f2_splat(-kTwoPiHi), nlo = f2_splat(-kTwoPiLo);
#pragma unroll
      for (int p = 0; p < NPP; p++) {
        const f2 k = f2_add(f2_fma(z[p], inv, sh), nsh);
        const f2 r = f2_fma(k, nlo, f2_fma(k, nhi, z[p]));
        float a0, a1;
        f2_unpack(r, a0, a1);
        z[p] = f2_pack(mufu_sin(a0), mufu_sin(a1));
      }
      break;
    }
    case EMR_ACT_ABS:
#pragma unroll
      for (int p = 0; p < NPP; p++) {
        float a0, a1;
        f2_unpack(z[p], a0, a1);
        z[p] = f2_pack(fabsf(a0), fabsf(a1));
      }
      break;
    default:
      break;
  }
}

// ---- filter arithmetic shared by every kernel ------------------------------------
// All kernels take the same fp32 decisions, operation for operation:
//   variance: S = sum_c (w_c - m)^2 with m = (w0 + w1 + w2 + w3) / 4; V = S / 4 and
//     V > theta is tested as S > 4 theta (scaling by 4 is exact);
//   band: with squared differences to the four neighbours, B > band is tested as
//     max(min(dt^2, db^2), min(dl^2, dr^2)) > band^2 (squaring is monotone on
//     |d|; it changes the fp32 decision only within one rounding of the band).
__device__ __forceinline__ float sqdiff(float a, float b) {
  const float t = a - b;
  return t * t;
}
// Sixteen times the population variance of four values, as the sum of their six
// squared pairwise differences (sum over i < j of (w_i - w_j)^2 equals four times
// the sum of squared deviations from the mean). The four sibling differences
// (w0 w1, w2 w3 along x; w0 w2, w1 w3 along y) are the band test's as well.
__device__ __forceinline__ float var16(float w0, float w1, float w2, float w3) {
  return ((sqdiff(w0, w1) + sqdiff(w2, w3)) + (sqdiff(w0, w2) + sqdiff(w1, w3))) +
         (sqdiff(w0, w3) + sqdiff(w1, w2));
}
__device__ __forceinline__ bool band_pass_sq(float dl2, float dr2, float db2, float dt2, float band2) {
  return fmaxf(fminf(dt2, db2), fminf(dl2, dr2)) > band2;
}

// Band-bit planes are quad-major from depth 3 on: in each block of 128
// positions (32 sibling quads), word c holds child c of the 32 quads (bit =
// quad). Depths 0..2 use the position-major layout of the other planes.
constexpr int kQuadMajorFrom = 3;

// Bits b (8 of them) spread to positions 0, 4, ..., 28.
__device__ __forceinline__ uint32_t spread_nibbles(uint32_t b) {
  b &= 0xffu;
  b = (b | (b << 12)) & 0x000f000fu;
  b = (b | (b << 6)) & 0x03030303u;
  b = (b | (b << 3)) & 0x11111111u;
  return b;
}

// Band-bit word of the 8 quads (32 positions) of lane group g from the four
// per-child ballots: bit 4 i + c of the word is child c of quad 8 g + i.
__device__ __forceinline__ uint32_t band_word(uint32_t b0, uint32_t b1, uint32_t b2, uint32_t b3, int g) {
  const int sh = 8 * g;
  return spread_nibbles(b0 >> sh) | (spread_nibbles(b1 >> sh) << 1) | (spread_nibbles(b2 >> sh) << 2) |
         (spread_nibbles(b3 >> sh) << 3);
}

// ---- per-pair specialisation ---------------------------------------------------
// A pair's record: header {nv, nve, out_const, flags}, then nv_cap float4
// {c0, wx, wy, info} with info = act | axes << 4 | edge_beg << 8 | edge_cnt << 20
// (axes: the grid coordinates the node depends on, kAxisX / kAxisY / kAxisXY),
// then nve_cap uint2 {source slot | source axes << 16, weight bits}, each
// node's edges ascending in (source axes, source slot). Varying slots follow
// the genome's topological order; the output is the last slot. nv = 0: the
// output is the same at every position (out_const); unused per-genome slots are
// recorded as constant 0 (no variance, no band value, nothing kept).
//
// Every evaluator computes a node's input in one order, so that all of them
// give the same fp32 value at a position:
//   x only:  a = fma(wx, x, c0), then its edges (all from x-only sources);
//   y only:  a = fma(wy, y, c0), then its edges (all from y-only sources);
//   joint:   sx = fma(wx, x, c0) and the edges from x-only sources,
//            sy = wy * y and the edges from y-only sources,
//            a = sx + sy, then the edges from joint sources;
// each edge adds fma(w, v_source, a); the node's value is act(a).
// Pairs with at most kDenseMax varying nodes also get, for the tile kernels'
// node tables, a table program per grid axis, the joint-node block and the
// joint nodes' activations (the dense block, at dense_off()):
//   program of axis a: kDenseMax float4 entries {c0, c, info, 0}, in slot order,
//     one per node with a row on that axis (info: row | kEntMul | kEntJoint |
//     act << 7 | first source << 10 | source count << 18), and kEntSrcCap
//     float2 sources {row of the source (int bits), weight}, in slot order;
//     rows of axis a: the joint nodes first (row m: the axis-a part of joint node
//     m's input), then the nodes of coordinate a alone (their values);
//   joint block: kDenseMax x kDenseMax floats, row-major, entry (m, m2) the
//     weight of the edge from joint node m2 to joint node m (m2 < m), else 0;
//   joint activations: kDenseMax int32.
constexpr int kDenseMax = 12;
constexpr uint32_t kEntMul = 1u << 5, kEntJoint = 1u << 6;
constexpr int kEntSrcCap = kDenseMax * (kDenseMax - 1) / 2;
struct SpecLayout {
  int64_t stride;
  int32_t nv_cap, nve_cap;
  __host__ __device__ int64_t coef_off() const { return 16; }
  __host__ __device__ int64_t edge_off() const { return 16 + 16 * int64_t(nv_cap); }
  __host__ __device__ int64_t dense_off() const { return (edge_off() + 8 * int64_t(nve_cap) + 15) & ~int64_t(15); }
  __host__ __device__ int64_t ent_off() const { return dense_off(); }
  __host__ __device__ int64_t esrc_off() const { return ent_off() + 2 * 16 * kDenseMax; }
  __host__ __device__ int64_t wj_off() const { return esrc_off() + 2 * 8 * kEntSrcCap; }
  __host__ __device__ int64_t jact_off() const { return wj_off() + 4 * kDenseMax * kDenseMax; }
  __host__ __device__ int64_t end_off() const { return jact_off() + 4 * kDenseMax; }
};

inline SpecLayout spec_layout(int nv_cap, int nve_cap) {
  SpecLayout L;
  L.nv_cap = std::max(nv_cap, 1);
  L.nve_cap = std::max(nve_cap, 1);
  L.stride = (L.end_off() + 15) & ~int64_t(15);
  return L;
}

// Kernel class of a pair by its varying-node count nv and its joint-node count
// nj: 0 = interpreter (nv above kDenseMax); otherwise by the joint nodes, the
// only ones evaluated per position: 1 = up to 12, 2 = up to 8, 3 = up to 6,
// 4 = up to 4, 5 = up to 2, 6 = none (the output depends on one coordinate, or
// on none: constant outputs are the last pairs of class 6). Classes run in this
// order, heaviest first.
constexpr int kClasses = 7;
constexpr int kClassNone = kClasses - 1;
__host__ __device__ __forceinline__ int pair_class(int nv, int nj) {
  return nv > kDenseMax ? 0 : nj > 8 ? 1 : nj > 6 ? 2 : nj > 4 ? 3 : nj > 2 ? 4 : nj > 0 ? 5 : kClassNone;
}

// Header word 3 of a record: its kernel class (bits 0..3) and, when nv <=
// kDenseMax, the joint-node count (bits 4..7) and the slot masks of the x-only
// (bits 8..19) and y-only (bits 20..31) nodes.
constexpr int kHdrJointShift = 4, kHdrXShift = 8, kHdrYShift = 20;

struct QueryDev {
  const float *a, *b;
  const int32_t *side, *count;
  int32_t S, per_genome;
};

// Pair schedule: by kernel class (heaviest class first), then by estimated
// cost, heaviest first: order[rank] = pair, by a counting sort over kCostBins
// bins of the pairs' bins (bins[r]), run by one CTA of nthreads threads (a
// multiple of 32, at most 1024; each thread scans kCostBins / nthreads bins).
// Up to nthreads * kSchedRegBins pairs, each thread reads its pairs' bins once,
// all at a time, and keeps them in registers for both passes.
constexpr int kClassBins = 256;
constexpr int kCostBins = kClasses * kClassBins;
constexpr int kSchedRegBins = 32;
__device__ void schedule_block(const int32_t* __restrict__ bins, int64_t n_pairs, int32_t* __restrict__ order,
                               int32_t* hist, int32_t* wsum) {
  const int nthreads = blockDim.x, tid = threadIdx.x;
  for (int k = tid; k < kCostBins; k += nthreads) hist[k] = 0;
  __syncthreads();
  const bool in_regs = n_pairs <= int64_t(nthreads) * kSchedRegBins;
  int rb[kSchedRegBins];  // bin of pair tid + i * nthreads (-1: none)
  if (in_regs) {
#pragma unroll
    for (int i = 0; i < kSchedRegBins; i++) {
      const int64_t r = tid + int64_t(i) * nthreads;
      rb[i] = r < n_pairs ? __ldcg(bins + r) : -1;
    }
#pragma unroll
    for (int i = 0; i < kSchedRegBins; i++)
      if (rb[i] >= 0) atomicAdd(&hist[rb[i]], 1);
  } else {
#pragma unroll 4
    for (int64_t r = tid; r < n_pairs; r += nthreads) atomicAdd(&hist[__ldcg(bins + r)], 1);
  }
  __syncthreads();
  // exclusive scan: thread tid owns bins [tid * per, (tid + 1) * per)
  const int per = kCostBins / nthreads, lane = tid & 31, warp = tid >> 5;
  int local = 0;
  for (int k = 0; k < per; k++) local += hist[tid * per + k];
  int x = local;
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) wsum[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int t = lane < nthreads / 32 ? wsum[lane] : 0;
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, t, o);
      if (lane >= o) t += y;
    }
    wsum[lane] = t;
  }
  __syncthreads();
  int run = (warp ? wsum[warp - 1] : 0) + x - local;
  for (int k = 0; k < per; k++) {
    const int v = hist[tid * per + k];
    hist[tid * per + k] = run;
    run += v;
  }
  __syncthreads();
  if (in_regs) {
#pragma unroll
    for (int i = 0; i < kSchedRegBins; i++)
      if (rb[i] >= 0) order[atomicAdd(&hist[rb[i]], 1)] = int32_t(tid + i * nthreads);
    return;
  }
#pragma unroll 4
  for (int64_t r = tid; r < n_pairs; r += nthreads) order[atomicAdd(&hist[__ldcg(bins + r)], 1)] = int32_t(r);
}

// One thread per pair: fold the constant inputs (the slot's node coordinates
// and the bias) and every node that does not vary over the grid into per-node
// constants; list the edges between varying nodes.
constexpr int kSpecWarps = 4;   // pairs per CTA: a warp per pair
constexpr int kSpecSmemNodes = 128;  // genomes up to this many kept nodes keep their values in shared memory
// genomes up to this many kept nodes and edges are staged in shared memory, and
// their records built there before one coalesced copy out
constexpr int kSpecStageNodes = 48, kSpecStageEdges = 96;

__global__ void __launch_bounds__(32 * kSpecWarps) spec_kernel(const uint8_t* __restrict__ pack, QueryDev q,
                                                               int64_t n_pairs, SpecLayout L,
                                                               uint8_t* __restrict__ spec,
                                                               float* __restrict__ scratch, int32_t scratch_stride,
                                                               int32_t* __restrict__ order, int32_t* __restrict__ bins,
                                                               unsigned int* __restrict__ done) {
  pdl_trigger();  // a tile launch set to overlap this kernel waits for its completion in every CTA
  __shared__ float s_cval[kSpecWarps][kSpecSmemNodes];
  __shared__ int32_t s_hist[kCostBins];
  __shared__ int32_t s_wsum[32];
  __shared__ __align__(16) PackNode s_nd[kSpecWarps][kSpecStageNodes];
  __shared__ __align__(16) PackEdge s_ed[kSpecWarps][kSpecStageEdges];
  __shared__ float4 s_cf[kSpecWarps][kSpecStageNodes];
  __shared__ uint2 s_ve[kSpecWarps][kSpecStageEdges];
  __shared__ __align__(16) float s_W[kSpecWarps][kDenseMax * kDenseMax];
  __shared__ int s_last;
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int64_t r = int64_t(blockIdx.x) * kSpecWarps + wid;
  auto pair_record = [&]() {
  const PackHeader* h = reinterpret_cast<const PackHeader*>(pack);
  const PackGenome* gt = reinterpret_cast<const PackGenome*>(pack + h->off_genomes);
  const PackNode* nt = reinterpret_cast<const PackNode*>(pack + h->off_nodes);
  const PackEdge* et = reinterpret_cast<const PackEdge*>(pack + h->off_edges);
  int g = int(r / q.S), s = int(r % q.S);
  uint8_t* rec = spec + r * L.stride;
  int32_t* hdr = reinterpret_cast<int32_t*>(rec);
  if (q.per_genome && q.count && s >= q.count[g]) {  // unused slot: constant 0, nothing kept
    if (lane == 0) {
      hdr[0] = 0; hdr[1] = 0; hdr[2] = 0; hdr[3] = pair_class(0, 0);
      bins[r] = kCostBins - 1;
    }
    return;
  }
  const PackGenome G = gt[g];
  if (lane == 0) {  // the pair's schedule bin: its class, then its cost, heaviest first
    const int64_t si = q.per_genome ? int64_t(g) * q.S + s : s;
    const int side = q.side[si] ? 1 : 0;
    const int c = int(min(G.cost[side], uint32_t(kClassBins - 1)));
    bins[r] = pair_class(G.n_varying[side], G.n_joint[side]) * kClassBins + (kClassBins - 1 - c);
  }
  // stage a small genome's node and edge records (coalesced, by the warp)
  const bool staged = G.n_nodes <= kSpecStageNodes && G.n_edges <= kSpecStageEdges;
  if (staged) {
    const int4* ns = reinterpret_cast<const int4*>(nt + G.node_beg);
    int4* nd_s = reinterpret_cast<int4*>(s_nd[wid]);
    for (int k = lane; k < 2 * int(G.n_nodes); k += 32) nd_s[k] = ns[k];
    const uint2* es = reinterpret_cast<const uint2*>(et + G.edge_beg);
    uint2* ed_s = reinterpret_cast<uint2*>(s_ed[wid]);
    for (int k = lane; k < int(G.n_edges); k += 32) ed_s[k] = es[k];
    __syncwarp();
  }
  const PackNode* NS = staged ? s_nd[wid] : nt + G.node_beg;
  const PackEdge* ES = staged ? s_ed[wid] : et + G.edge_beg;
  float4* coef_g = reinterpret_cast<float4*>(rec + L.coef_off());
  uint2* ve_g = reinterpret_cast<uint2*>(rec + L.edge_off());
  float4* coef = staged ? s_cf[wid] : coef_g;  // records are built here (staged: copied out below)
  uint2* ve = staged ? s_ve[wid] : ve_g;
  int nv = 0, nve = 0;
  int32_t hdr3 = 0;
  {
    const int64_t si = q.per_genome ? int64_t(g) * q.S + s : s;
    const int side = q.side[si] ? 1 : 0;
    const float a = q.a[si], b = q.b[si];
    float in[5] = {0.f, 0.f, 0.f, 0.f, 1.f};
    int gx, gy;
    if (side == EMR_SIDE_OUT) { in[EMR_KIND_X1] = a; in[EMR_KIND_Y1] = b; gx = EMR_KIND_X2; gy = EMR_KIND_Y2; }
    else { in[EMR_KIND_X2] = a; in[EMR_KIND_Y2] = b; gx = EMR_KIND_X1; gy = EMR_KIND_Y1; }
    float* cval = G.n_nodes <= kSpecSmemNodes ? s_cval[wid] : scratch + r * scratch_stride;
    const int n = G.n_nodes;
    const uint32_t vbit = 1u << side;
    // The constants: the nodes that do not vary, in topological order (each folds its sources'
    // values), by lane 0. A node that does not vary has no varying source.
    float out_const = 0.f;
    if (lane == 0) {
      for (int t = 0; t < n; t++) {
        const PackNode nd = NS[t];
        if (nd.vary & vbit) continue;
        const PackEdge* ed = ES + nd.edge_beg;
        float z = nd.bias;
        for (int k = 0; k < 5; k++) z = fmaf(nd.w_in[k], in[k], z);
        for (int e = 0; e < nd.edge_cnt; e++) z = fmaf(ed[e].w, cval[ed[e].src], z);
        cval[t] = act_apply(nd.act, z);
        out_const = cval[t];
      }
    }
    // the varying nodes' record indices (their order among the varying nodes), in their value
    // slots, by the warp
    for (int t0 = 0; t0 < n; t0 += 32) {
      const int t = t0 + lane;
      const bool v = t < n && (NS[t].vary & vbit);
      const uint32_t bal = __ballot_sync(kFull, v);
      if (v) cval[t] = __uint_as_float(uint32_t(nv + __popc(bal & ((1u << lane) - 1u))));
      nv += __popc(bal);
    }
    __syncwarp();  // lane 0's constants and every record index are visible to the warp
    // Each varying node's record, by its lane: the constant part of its input (the inputs of
    // fixed value, then its sources that do not vary, in edge order) and its edges from varying
    // sources, ascending (source axes, source index); edge offsets by a warp scan.
    uint32_t xm = 0, ym = 0;
    int nj = 0, k0 = 0;
    for (int t0 = 0; t0 < n; t0 += 32) {
      const int t = t0 + lane;
      const bool v = t < n && (NS[t].vary & vbit);
      PackNode nd{};
      int cnt = 0;
      if (v) {
        nd = NS[t];
        const PackEdge* ed = ES + nd.edge_beg;
        for (int e = 0; e < nd.edge_cnt; e++) cnt += (NS[ed[e].src].vary & vbit) ? 1 : 0;
      }
      int incl = cnt;  // inclusive warp scan of the edge counts
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int u = __shfl_up_sync(kFull, incl, o);
        if (lane >= o) incl += u;
      }
      const int total = __shfl_sync(kFull, incl, 31);
      const int eb = nve + incl - cnt;
      const uint32_t bal = __ballot_sync(kFull, v);
      const int slot = k0 + __popc(bal & ((1u << lane) - 1u));
      const uint32_t ax = v ? (uint32_t(nd.axes) >> (2 * side)) & 3u : 0u;
      if (v) {
        float c0 = nd.bias;
        for (int k = 0; k < 5; k++)
          if (k != gx && k != gy) c0 = fmaf(nd.w_in[k], in[k], c0);
        const PackEdge* ed = ES + nd.edge_beg;
        int ne = eb;
        for (int e = 0; e < nd.edge_cnt; e++) {
          const PackNode& src = NS[ed[e].src];
          if (src.vary & vbit) {
            const uint32_t sa = (uint32_t(src.axes) >> (2 * side)) & 3u;
            ve[ne++] = make_uint2(__float_as_uint(cval[ed[e].src]) | (sa << 16), __float_as_uint(ed[e].w));
          } else {
            c0 = fmaf(ed[e].w, cval[ed[e].src], c0);
          }
        }
        for (int e = eb + 1; e < ne; e++) {  // (insertion sort, a few edges)
          const uint2 key = ve[e];
          int f = e - 1;
          while (f >= eb && ve[f].x > key.x) { ve[f + 1] = ve[f]; f--; }
          ve[f + 1] = key;
        }
        const uint32_t info = uint32_t(nd.act) | (ax << 4) | (uint32_t(eb) << 8) | (uint32_t(cnt) << 20);
        coef[slot] = make_float4(c0, nd.w_in[gx], nd.w_in[gy], __uint_as_float(info));
      }
      nj += __popc(__ballot_sync(kFull, ax == kAxisXY));
      const bool dense_slot = slot < kDenseMax;
      xm |= __reduce_or_sync(kFull, ax == kAxisX && dense_slot ? 1u << slot : 0u);
      ym |= __reduce_or_sync(kFull, ax == kAxisY && dense_slot ? 1u << slot : 0u);
      nve += total;
      k0 += __popc(bal);
    }
    out_const = __shfl_sync(kFull, out_const, 0);
    hdr3 = int32_t(pair_class(nv, nj) |
                   (nv <= kDenseMax ? uint32_t(nj) << kHdrJointShift | xm << kHdrXShift | ym << kHdrYShift : 0u));
    if (lane == 0) {
      hdr[0] = nv;
      hdr[1] = nve;
      reinterpret_cast<float*>(hdr)[2] = out_const;
      hdr[3] = hdr3;
    }
  }
  const uint32_t h3 = uint32_t(hdr3);
  __syncwarp();  // the lanes' coefficient and edge records are visible to the warp
  if (staged) {
    for (int k = lane; k < nv; k += 32) coef_g[k] = coef[k];
    for (int k = lane; k < nve; k += 32) ve_g[k] = ve[k];
  }
  if (nv <= kDenseMax) {  // the dense block: built in shared memory by the warp's lanes, then copied out
    float* Ws = s_W[wid];
    for (int k = lane; k < kDenseMax * kDenseMax; k += 32) Ws[k] = 0.f;
    __syncwarp();
    if (lane < nv) {  // lane k fills row k (at most one edge per source: parallel connections are merged)
      const uint32_t info = __float_as_uint(coef[lane].w);
      const int eb = int((info >> 8) & 0xfffu), ec = int(info >> 20);
      for (int e = eb; e < eb + ec; e++) Ws[lane * kDenseMax + int(ve[e].x & 0xffffu)] += __uint_as_float(ve[e].y);
    }
    __syncwarp();
    // the tile kernels' table programs (lane k: slot k), joint block and joint activations
    const int nj = int((h3 >> kHdrJointShift) & 0xfu);
    const uint32_t xm = (h3 >> kHdrXShift) & 0xfffu, ym = (h3 >> kHdrYShift) & 0xfffu;
    const uint32_t jm = ((1u << nv) - 1u) & ~(xm | ym);
    float4* ent_g = reinterpret_cast<float4*>(rec + L.ent_off());
    float2* esrc_g = reinterpret_cast<float2*>(rec + L.esrc_off());
    for (int a = 0; a < 2; a++) {
      const int k = lane;
      const uint32_t om = a ? ym : xm, bit = 1u << k, below = bit - 1u;
      const bool on = k < nv && ((om | jm) & bit) != 0u;
      const bool joint = (jm & bit) != 0u;
      uint32_t sm = 0;  // sources: earlier nodes of this coordinate alone with an edge into k
      if (on)
        for (uint32_t b = om & below; b; b &= b - 1u)
          if (Ws[k * kDenseMax + __ffs(b) - 1] != 0.f) sm |= b & (0u - b);
      const int cnt = __popc(sm);
      int beg = cnt;  // exclusive prefix over the lanes
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(kFull, beg, o);
        if (lane >= o) beg += y;
      }
      beg -= cnt;
      if (on) {
        const float4 cf = coef[k];
        const int row = joint ? __popc(jm & below) : nj + __popc(om & below);
        const uint32_t info = uint32_t(row) | (joint && a ? kEntMul : 0u) | (joint ? kEntJoint : 0u) |
                              ((__float_as_uint(cf.w) & 7u) << 7) | (uint32_t(beg) << 10) | (uint32_t(cnt) << 18);
        ent_g[a * kDenseMax + __popc((om | jm) & below)] = make_float4(cf.x, a ? cf.z : cf.y, __uint_as_float(info), 0.f);
        int q = beg;
        for (uint32_t b = sm; b; b &= b - 1u) {
          const int j = __ffs(b) - 1;
          esrc_g[a * kEntSrcCap + q++] =
              make_float2(__int_as_float(nj + __popc(om & ((1u << j) - 1u))), Ws[k * kDenseMax + j]);
        }
      }
    }
    auto slot_of = [&](int m) {  // joint node m is the m-th set bit of jm
      uint32_t b = jm;
      for (int q = 0; q < m; q++) b &= b - 1u;
      return b ? __ffs(b) - 1 : 0;
    };
    float* wj_g = reinterpret_cast<float*>(rec + L.wj_off());
    for (int t = lane; t < kDenseMax * kDenseMax; t += 32) {
      const int m = t / kDenseMax, m2 = t % kDenseMax;
      wj_g[t] = m < nj && m2 < m ? Ws[slot_of(m) * kDenseMax + slot_of(m2)] : 0.f;
    }
    if (lane < kDenseMax)
      reinterpret_cast<int32_t*>(rec + L.jact_off())[lane] =
          lane < nj ? int32_t(__float_as_uint(coef[slot_of(lane)].w) & 0xfu) : 0;
  }
  };
  if (r < n_pairs) pair_record();  // whole warps
  // the last CTA to finish orders the pairs by their bins (no waiting: the others have
  // published their bins before counting themselves done)
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) s_last = atomicAdd(done, 1u) == gridDim.x - 1;
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  schedule_block(bins, n_pairs, order, s_hist, s_wsum);
  if (threadIdx.x == 0) *done = 0u;  // ready for the next call
}

// ---- evaluation tiles ------------------------------------------------------------

enum { kModeMaterialise = 0, kModeFused = 1 };

// Output views: band_bits and out may be chunk-local buffers. Band word w of
// pair r is bandb[r * band_stride + w - band_shift]; output at global index p of
// pair r is out[r * out_stride + p - out_shift]. Whole-grid calls use strides
// n_words / n_total and shifts 0. The split plane is always whole-grid.
constexpr int kPyramidTop = 4;  // depths 0..4 (side <= 32) share one CTA

struct TileArgs {
  const uint8_t* spec;
  SpecLayout L;
  const int32_t* order;
  int64_t rank_beg;
  int32_t n_tiles, tile_beg;
  int64_t band_stride, band_shift, out_stride, out_shift;
  int32_t D, mode;
  float theta, band, w_min;
  int32_t lvl_tile_beg[EMR_MAX_DEPTH + 2];
  int64_t n_total, n_halo, n_words;
  int64_t level_off[EMR_MAX_DEPTH + 2], halo_off[EMR_MAX_DEPTH + 2], word_off[EMR_MAX_DEPTH + 2];
  float* out;
  float* out_halo;
  uint32_t* split;
  uint32_t* bandb;
  uint8_t* tile_flags;  // fused, optional: [pair][dense tile] set to 1 where a band bit is set
  int64_t n_dense;
};

// Input of one node (its value before the activation) at NP points, from the
// record's edge list in the evaluators' common order (see the record layout):
// coefficients c, edges [eb, ee), source values val(slot, p).
template <int NP, class Val>
__device__ __forceinline__ void node_input_sparse(const float4 c, const uint2* __restrict__ ve, int eb, int ee,
                                                  const float (&x)[NP], const float (&y)[NP], Val val,
                                                  float (&z)[NP]) {
  const uint32_t ax = (__float_as_uint(c.w) >> 4) & 3u;
  float sy[NP];
#pragma unroll
  for (int p = 0; p < NP; p++) {
    z[p] = ax == kAxisY ? fmaf(c.z, y[p], c.x) : fmaf(c.y, x[p], c.x);
    sy[p] = __fmul_rn(c.z, y[p]);
  }
  bool merged = ax != kAxisXY;  // joint: x part in z, y part in sy until the first joint source
  for (int e = eb; e < ee; e++) {
    const uint2 E = ve[e];
    const uint32_t sa = E.x >> 16;
    const int src = int(E.x & 0xffffu);
    const float we = __uint_as_float(E.y);
    if (!merged && sa == kAxisY) {
#pragma unroll
      for (int p = 0; p < NP; p++) sy[p] = fmaf(we, val(src, p), sy[p]);
      continue;
    }
    if (!merged && sa == kAxisXY) {
#pragma unroll
      for (int p = 0; p < NP; p++) z[p] = __fadd_rn(z[p], sy[p]);
      merged = true;
    }
#pragma unroll
    for (int p = 0; p < NP; p++) z[p] = fmaf(we, val(src, p), z[p]);
  }
  if (!merged) {
#pragma unroll
    for (int p = 0; p < NP; p++) z[p] = __fadd_rn(z[p], sy[p]);
  }
}

// CPPN at four points by interpreting the pair's record: node values live in
// shared memory, one float4 (four points) per thread and varying node.
__device__ __forceinline__ void eval4_interp(const float4* __restrict__ coef, const uint2* __restrict__ ve,
                                             float4* __restrict__ vals, int nv, float out_const, int tid,
                                             const float (&x)[4], const float (&y)[4], float (&w)[4]) {
  if (nv == 0) {
    w[0] = w[1] = w[2] = w[3] = out_const;
    return;
  }
  float z[4];
  auto val = [&](int src, int p) {
    const float4& v = vals[src * kBlock + tid];
    return p == 0 ? v.x : p == 1 ? v.y : p == 2 ? v.z : v.w;
  };
  for (int k = 0; k < nv; k++) {
    const float4 c = coef[k];
    const uint32_t info = __float_as_uint(c.w);
    const int eb = int((info >> 8) & 0xfffu), ee = eb + int(info >> 20);
    node_input_sparse<4>(c, ve, eb, ee, x, y, val, z);
    act_apply4(int(info & 0xfu), z[0], z[1], z[2], z[3]);
    if (k + 1 < nv) vals[k * kBlock + tid] = make_float4(z[0], z[1], z[2], z[3]);
  }
  w[0] = z[0]; w[1] = z[1]; w[2] = z[2]; w[3] = z[3];
}

__global__ void __launch_bounds__(kBlock) tile_kernel(const TileArgs A) {
  extern __shared__ float4 smem4[];
  pdl_trigger();  // the dense classes may follow as SMs free up
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t rank = A.rank_beg + blockIdx.x / A.n_tiles;
  const int tile = A.tile_beg + int(blockIdx.x % A.n_tiles);
  const int r = A.order[rank];
  const uint8_t* rec = A.spec + int64_t(r) * A.L.stride;
  const int nv = reinterpret_cast<const int32_t*>(rec)[0];
  const int nve = reinterpret_cast<const int32_t*>(rec)[1];
  const float out_const = reinterpret_cast<const float*>(rec)[2];
  int d = 0;
  while (A.lvl_tile_beg[d + 1] <= tile) d++;
  const int T = d + 1 < kTileLog ? (1 << (d + 1)) : kTileSide;
  const uint32_t mb = uint32_t(tile - A.lvl_tile_beg[d]) * uint32_t(T * T);  // first Morton index of the tile
  const int i0 = int(compact1by1(mb)), j0 = int(compact1by1(mb >> 1));
  const int n = 1 << (d + 1);
  const float scale = __int_as_float((127 - (d + 1)) << 23);  // 2^-(d+1)

  // shared memory: record (coefficients, edges) | node values | output tile with its ring
  float4* coef = smem4;
  uint2* ve = reinterpret_cast<uint2*>(smem4 + A.L.nv_cap);
  float4* vals = smem4 + A.L.nv_cap + (A.L.nve_cap + 1) / 2;
  float* wt = reinterpret_cast<float*>(vals + A.L.nv_cap * kBlock);
  const int pitch = T + 2;
  {
    const float4* gc = reinterpret_cast<const float4*>(rec + A.L.coef_off());
    for (int k = tid; k < nv; k += kBlock) coef[k] = gc[k];
    const uint2* ge = reinterpret_cast<const uint2*>(rec + A.L.edge_off());
    for (int k = tid; k < nve; k += kBlock) ve[k] = ge[k];
  }
  __syncthreads();

  const bool fused = A.mode == kModeFused;
  const int nq = T * T / 4;
  const bool ring = fused || A.out_halo != nullptr;
  const int items = nq + (ring ? T : 0);
  const int64_t pair_pos = int64_t(r) * A.out_stride - A.out_shift + A.level_off[d];
  const int64_t band_base = int64_t(r) * A.band_stride - A.band_shift;
  for (int base = 0; base < items; base += kBlock) {
    const int q = base + tid;
    const bool valid = q < items;
    const bool is_main = q < nq;
    int li[4], lj[4];
    bool use = valid;
    if (is_main) {
      const int pi = int(compact1by1(uint32_t(q))), pj = int(compact1by1(uint32_t(q) >> 1));
#pragma unroll
      for (int c = 0; c < 4; c++) { li[c] = 2 * pi + (c & 1); lj[c] = 2 * pj + (c >> 1); }
    } else {
      const int hq = valid ? q - nq : 0;
#pragma unroll
      for (int c = 0; c < 4; c++) {
        const int k = 4 * hq + c, sd = k / T, u = k - sd * T;
        li[c] = sd == 0 ? -1 : sd == 1 ? T : u;
        lj[c] = sd == 2 ? -1 : sd == 3 ? T : u;
      }
      if (!fused) {  // materialised: only ring points outside the domain are evaluated
        const int sd = (4 * hq) / T;
        const bool outside = (sd == 0 && i0 == 0) || (sd == 1 && i0 + T == n) || (sd == 2 && j0 == 0) ||
                             (sd == 3 && j0 + T == n);
        use = valid && outside;
      }
    }
    float w[4] = {0.f, 0.f, 0.f, 0.f};
    if (__any_sync(kFull, use)) {
      float x[4], y[4];
#pragma unroll
      for (int c = 0; c < 4; c++) { x[c] = grid_coord(i0 + li[c], scale); y[c] = grid_coord(j0 + lj[c], scale); }
      eval4_interp(coef, ve, vals, nv, out_const, tid, x, y, w);
    }
    if (!fused) {
      if (is_main) {
        *reinterpret_cast<float4*>(A.out + pair_pos + mb + 4 * q) = make_float4(w[0], w[1], w[2], w[3]);
      } else if (use) {
#pragma unroll
        for (int c = 0; c < 4; c++) {
          const int gi = i0 + li[c], gj = j0 + lj[c];
          const int sd = gi < 0 ? 0 : gi >= n ? 1 : gj < 0 ? 2 : 3;
          const int t = sd < 2 ? gj : gi;
          A.out_halo[int64_t(r) * A.n_halo + A.halo_off[d] + sd * n + t] = w[c];
        }
      }
      continue;
    }
    // fused: the four children of parent q give its variance (Section 3.2)
    if (d >= 1) {
      const unsigned bal = __ballot_sync(kFull, is_main && var16(w[0], w[1], w[2], w[3]) > 16.f * A.theta);
      const int q0 = base + warp * 32;
      if (lane == 0 && q0 < nq)
        A.split[int64_t(r) * A.n_words + A.word_off[d - 1] + (mb / 4 + uint32_t(q0)) / 32] = bal;
    }
    if (valid) {
#pragma unroll
      for (int c = 0; c < 4; c++) wt[(lj[c] + 1) * pitch + (li[c] + 1)] = w[c];
    }
  }
  if (!fused) return;
  __syncthreads();
  bool any_pass = false;
  // band value of each position from its four neighbours at distance 2^-d
  for (int base = 0; base < nq; base += kBlock) {
    const int q = base + tid;
    const bool valid = q < nq;
    const int pi = int(compact1by1(uint32_t(q))), pj = int(compact1by1(uint32_t(q) >> 1));
    const float band2 = A.band * A.band;
    bool pass[4] = {false, false, false, false};
    float w[4];
#pragma unroll
    for (int c = 0; c < 4; c++) {
      const int li = 2 * pi + (c & 1) + 1, lj = 2 * pj + (c >> 1) + 1;
      w[c] = valid ? wt[lj * pitch + li] : 0.f;
      if (valid) {
        pass[c] = band_pass_sq(sqdiff(w[c], wt[lj * pitch + li - 1]), sqdiff(w[c], wt[lj * pitch + li + 1]),
                               sqdiff(w[c], wt[(lj - 1) * pitch + li]), sqdiff(w[c], wt[(lj + 1) * pitch + li]), band2);
        if (A.w_min > 0.f) pass[c] = pass[c] && fabsf(w[c]) > A.w_min;
      }
    }
    const uint32_t b0 = __ballot_sync(kFull, pass[0]), b1 = __ballot_sync(kFull, pass[1]);
    const uint32_t b2 = __ballot_sync(kFull, pass[2]), b3 = __ballot_sync(kFull, pass[3]);
    any_pass = any_pass || (b0 | b1 | b2 | b3) != 0u;
    const int q0 = base + warp * 32;
    if (d >= kQuadMajorFrom) {
      if (lane < 4 && q0 < nq)
        A.bandb[band_base + A.word_off[d] + 4 * ((mb + 4u * uint32_t(q0)) >> 7) + lane] =
            lane == 0 ? b0 : lane == 1 ? b1 : lane == 2 ? b2 : b3;
    } else if (q0 == 0 && lane * 32 < 4 * nq) {
      A.bandb[band_base + A.word_off[d] + lane] = band_word(b0, b1, b2, b3, lane);
    }
    if (A.out && (pass[0] | pass[1] | pass[2] | pass[3])) {
#pragma unroll
      for (int c = 0; c < 4; c++)
        if (pass[c]) A.out[pair_pos + mb + 4 * q + c] = w[c];
    }
  }
  // dense tile numbering: depths 0..4 share tile 0, interpreter tile t >= 5 is dense tile t - 4
  if (A.tile_flags && __syncthreads_or(any_pass) && tid == 0)
    A.tile_flags[int64_t(r) * A.n_dense + (tile <= kPyramidTop ? 0 : tile - kPyramidTop)] = 1;
}

// ---- register-resident tiles (pairs with at most kDenseMax varying nodes) ---------
//
// A CTA of 128 threads owns one tile: either a 64 x 64 Morton block of one
// depth >= 5, or (tile 0 of a pair) the whole of depths 0..4. A node that
// depends on one grid coordinate has one value per tile column (x) or row (y):
// the CTA first evaluates those nodes at the tile's distinct coordinates into
// shared-memory tables, together with the x part and the y part of every joint
// node's input (both coordinates). Then each thread evaluates sibling quads
// (the four children of one parent cell): a joint node's input is its x part
// plus its y part from the tables, plus its edges from joint sources, with the
// joint nodes' values in registers (loop unrolled to NJMAX with a uniform early
// exit, so every register index is static). An output of one coordinate is
// read from its table. The quad's variance comes straight from its four
// results; the band value needs the neighbours, taken from the tile in shared
// memory after a barrier (the ring of out-of-tile neighbours is evaluated by the
// tile too).

struct DTileArgs {
  const uint8_t* spec;
  SpecLayout L;
  const int32_t* order;
  int64_t rank_beg;
  int32_t n_tiles, tile_beg;
  int32_t tiles_per_cta;  // consecutive tiles of one pair per CTA (blockIdx.x: tile group)
  int64_t band_stride, band_shift, out_stride, out_shift;
  int32_t D, mode;
  float theta, band, w_min;
  int64_t n_total, n_halo, n_words;
  int64_t level_off[EMR_MAX_DEPTH + 2], halo_off[EMR_MAX_DEPTH + 2], word_off[EMR_MAX_DEPTH + 2];
  float* out;
  float* out_halo;
  uint32_t* split;
  uint32_t* bandb;
  uint8_t* tile_flags;  // fused, optional: [pair][dense tile] set to 1 where a band bit is set
  int64_t n_dense;
  int32_t wait_at_start;  // pyramid kernel: the launch overlaps the record kernel, whose records it reads
};

template <int NP>
__device__ __forceinline__ void act_applyN(int a, float (&z)[NP]) {
  switch (a) {
    case EMR_ACT_SIGMOID:
#pragma unroll
      for (int p = 0; p < NP; p++) z[p] = act_sigmoid(z[p]);
      break;
    case EMR_ACT_TANH:
#pragma unroll
      for (int p = 0; p < NP; p++) z[p] = act_tanh(z[p]);
      break;
    case EMR_ACT_GAUSS:
#pragma unroll
      for (int p = 0; p < NP; p++) z[p] = act_gauss(z[p]);
      break;
    case EMR_ACT_SIN:
#pragma unroll
      for (int p = 0; p < NP; p++) z[p] = act_sin(z[p]);
      break;
    case EMR_ACT_ABS:
#pragma unroll
      for (int p = 0; p < NP; p++) z[p] = fabsf(z[p]);
      break;
    default:
      break;
  }
}

// Node tables of a dense tile CTA, [axis][row][column]. Rows of axis a: first
// the joint nodes (row m: the axis-a part of joint node m's input), then the
// nodes of coordinate a alone (their values), in slot order. Tile-local
// coordinate index i sits at column i + 2, so the columns of sibling positions
// (2 c, 2 c + 1) are 8-byte aligned. A 64 x 64 tile uses i = -1 .. 64 (ring
// included); the pyramid tile keeps depth d at columns seg(d) + i + 2,
// i = -1 .. 2^(d+1).
constexpr int kTabFull = kTileSide + 4;
__host__ __device__ constexpr int tab_seg(int d) { return (2 << d) - 2 + 4 * d; }
constexpr int kTabPyr = tab_seg(kPyramidTop + 1);

// Table program of one axis (built per pair by spec_kernel, see the record
// layout): kEntMul: the input starts as c * coordinate (the y part of a joint
// node); kEntJoint: the row holds the input, no activation.

// Table columns: every entry of the axis at the NC coordinate values cv,
// columns pos (the common order of the record layout; a node of one coordinate
// has sources of that coordinate only).
template <int NC>
__device__ __forceinline__ void table_columns(const float (&cv)[NC], const int (&pos)[NC], int n_ent,
                                              const float4* __restrict__ ent, const float2* __restrict__ src,
                                              float* __restrict__ tab, int tw) {
  for (int e = 0; e < n_ent; e++) {
    const float4 E = ent[e];
    const uint32_t info = __float_as_uint(E.z);
    float z[NC];
#pragma unroll
    for (int c = 0; c < NC; c++) z[c] = (info & kEntMul) ? __fmul_rn(E.y, cv[c]) : fmaf(E.y, cv[c], E.x);
    const int sb = int((info >> 10) & 0xffu), se = sb + int(info >> 18);
    for (int k = sb; k < se; k++) {
      const float2 S = src[k];
      const float* col = tab + __float_as_int(S.x) * tw;
#pragma unroll
      for (int c = 0; c < NC; c++) z[c] = fmaf(S.y, col[pos[c]], z[c]);
    }
    if (!(info & kEntJoint)) act_applyN<NC>(int((info >> 7) & 7u), z);
    float* out = tab + int(info & 31u) * tw;
#pragma unroll
    for (int c = 0; c < NC; c++) out[pos[c]] = z[c];
  }
}
// (NC = 1: one column.)
__device__ __forceinline__ void table_column(float cv, int pos, int n_ent, const float4* __restrict__ ent,
                                             const float2* __restrict__ src, float* __restrict__ tab, int tw) {
  const float c1[1] = {cv};
  const int p1[1] = {pos};
  table_columns<1>(c1, p1, n_ent, ent, src, tab, tw);
}

// The joint nodes of a pair at NP points: init(m, z) gives joint node m's x
// part plus y part; its edges from earlier joint nodes (WJ, row-major NJMAX x
// NJMAX, 0 where there is no edge) follow in slot order. w: the last joint
// node's value, the output.
template <int NJMAX, int NP, class Init>
__device__ __forceinline__ void eval_joint(int nj, const float* __restrict__ WJ, const int* __restrict__ jact,
                                           Init init, float (&w)[NP]) {
  // node m is computed in w; entering node m + 1 keeps it as v[m] for the later nodes
  float v[NJMAX > 1 ? NJMAX - 1 : 1][NP];
#pragma unroll
  for (int m = 0; m < NJMAX; m++) {
    if (m >= nj) break;
    if (m > 0) {
#pragma unroll
      for (int p = 0; p < NP; p++) v[m - 1][p] = w[p];
    }
    init(m, w);
#pragma unroll
    for (int m2 = 0; m2 < m; m2++) {
      const float wk = WJ[m * NJMAX + m2];
      if (wk != 0.f) {
#pragma unroll
        for (int p = 0; p < NP; p++) w[p] = fmaf(wk, v[m2][p], w[p]);
      }
    }
    act_applyN<NP>(jact[m], w);
  }
}

// Per-CTA view of a pair for the table evaluators.
struct PairTabs {
  const float* tx;  // axis-0 table
  const float* ty;  // axis-1 table
  int tw;           // table row length
  int nv, nj;
  bool out_x;       // output of one coordinate: x (else y)
  int orow;         // its row
  float out_const;
};

// Output at NP points given by their table columns (xp, yp).
template <int NJMAX, int NP>
__device__ __forceinline__ void eval_points(const PairTabs& T, const float* __restrict__ WJ,
                                            const int* __restrict__ jact, const int (&xp)[NP], const int (&yp)[NP],
                                            float (&w)[NP]) {
  if constexpr (NJMAX > 0) {
    if (T.nj > 0) {
      auto init = [&](int m, float (&z)[NP]) {
        const float* sx = T.tx + m * T.tw;
        const float* sy = T.ty + m * T.tw;
#pragma unroll
        for (int p = 0; p < NP; p++) z[p] = __fadd_rn(sx[xp[p]], sy[yp[p]]);
      };
      eval_joint<NJMAX, NP>(T.nj, WJ, jact, init, w);
      return;
    }
  }
  if (T.nv == 0) {
#pragma unroll
    for (int p = 0; p < NP; p++) w[p] = T.out_const;
    return;
  }
  const float* t = (T.out_x ? T.tx : T.ty) + T.orow * T.tw;
#pragma unroll
  for (int p = 0; p < NP; p++) w[p] = t[T.out_x ? xp[p] : yp[p]];
}

// The joint nodes of a pair at 2 NPP points held as NPP packed pairs (eval_joint
// on pairs): WJ2 holds each joint weight twice (both halves of a pair).
template <int NJMAX, int NPP, class Init>
__device__ __forceinline__ void eval_joint_pairs(int nj, const f2* __restrict__ WJ2, const int* __restrict__ jact,
                                                 Init init, f2 (&w)[NPP]) {
  f2 v[NJMAX > 1 ? NJMAX - 1 : 1][NPP];
#pragma unroll
  for (int m = 0; m < NJMAX; m++) {
    if (m >= nj) break;
    if (m > 0) {
#pragma unroll
      for (int p = 0; p < NPP; p++) v[m - 1][p] = w[p];
    }
    init(m, w);
#pragma unroll
    for (int m2 = 0; m2 < m; m2++) {
      const f2 wk = WJ2[m * NJMAX + m2];
      if (f2_lo(wk) != 0.f) {
#pragma unroll
        for (int p = 0; p < NPP; p++) w[p] = f2_fma(wk, v[m2][p], w[p]);
      }
    }
    act_apply_pairs<NPP>(jact[m], w);
  }
}

// Output at QPE sibling quads of a 64 x 64 tile: quad h has its children at
// table columns xq[h], xq[h] + 1 and rows yq[h], yq[h] + 1 (both even), read as
// pairs; w[4 h + c] is child c (x fastest). Joint node m's parts are row m.
template <int NJMAX, int QPE>
__device__ __forceinline__ void eval_quads(const PairTabs& T, const float* __restrict__ WJ,
                                           const int* __restrict__ jact, const int (&xq)[QPE], const int (&yq)[QPE],
                                           float (&w)[4 * QPE]) {
  if constexpr (NJMAX > 0) {
    if (T.nj > 0) {
      auto init = [&](int m, float (&z)[4 * QPE]) {
        const float* sx = T.tx + m * kTabFull;
        const float* sy = T.ty + m * kTabFull;
#pragma unroll
        for (int h = 0; h < QPE; h++) {
          const float2 a = *reinterpret_cast<const float2*>(sx + xq[h]);
          const float2 b = *reinterpret_cast<const float2*>(sy + yq[h]);
          z[4 * h + 0] = __fadd_rn(a.x, b.x);
          z[4 * h + 1] = __fadd_rn(a.y, b.x);
          z[4 * h + 2] = __fadd_rn(a.x, b.y);
          z[4 * h + 3] = __fadd_rn(a.y, b.y);
        }
      };
      eval_joint<NJMAX, 4 * QPE>(T.nj, WJ, jact, init, w);
      return;
    }
  }
  if (T.nv == 0) {
#pragma unroll
    for (int p = 0; p < 4 * QPE; p++) w[p] = T.out_const;
    return;
  }
  const float* t = (T.out_x ? T.tx : T.ty) + T.orow * kTabFull;
#pragma unroll
  for (int h = 0; h < QPE; h++) {
    const float2 a = *reinterpret_cast<const float2*>(t + (T.out_x ? xq[h] : yq[h]));
    w[4 * h + 0] = a.x;
    w[4 * h + 1] = T.out_x ? a.y : a.x;
    w[4 * h + 2] = T.out_x ? a.x : a.y;
    w[4 * h + 3] = a.y;
  }
}

// eval_quads with the joint nodes on packed pairs (children 0, 1 and 2, 3 of
// each quad), the joint weights twice each in WJ2: the same bits in about half
// the issue slots of the fp32 work, for kernels whose registers hold the pairs.
template <int NJMAX, int QPE>
__device__ __forceinline__ void eval_quads_packed(const PairTabs& T, const f2* __restrict__ WJ2,
                                                  const int* __restrict__ jact, const int (&xq)[QPE],
                                                  const int (&yq)[QPE], float (&w)[4 * QPE]) {
  if constexpr (NJMAX > 0) {
    if (T.nj > 0) {
      auto init = [&](int m, f2 (&z)[2 * QPE]) {
        const float* sx = T.tx + m * kTabFull;
        const float* sy = T.ty + m * kTabFull;
#pragma unroll
        for (int h = 0; h < QPE; h++) {
          const f2 a = *reinterpret_cast<const f2*>(sx + xq[h]);  // the x parts of columns xq, xq + 1
          const float2 b = *reinterpret_cast<const float2*>(sy + yq[h]);
          z[2 * h + 0] = f2_add(a, f2_splat(b.x));
          z[2 * h + 1] = f2_add(a, f2_splat(b.y));
        }
      };
      f2 z[2 * QPE];
      eval_joint_pairs<NJMAX, 2 * QPE>(T.nj, WJ2, jact, init, z);
#pragma unroll
      for (int h = 0; h < QPE; h++) {
        f2_unpack(z[2 * h + 0], w[4 * h + 0], w[4 * h + 1]);
        f2_unpack(z[2 * h + 1], w[4 * h + 2], w[4 * h + 3]);
      }
      return;
    }
  }
  if (T.nv == 0) {
#pragma unroll
    for (int p = 0; p < 4 * QPE; p++) w[p] = T.out_const;
    return;
  }
  const float* t = (T.out_x ? T.tx : T.ty) + T.orow * kTabFull;
#pragma unroll
  for (int h = 0; h < QPE; h++) {
    const float2 a = *reinterpret_cast<const float2*>(t + (T.out_x ? xq[h] : yq[h]));
    w[4 * h + 0] = a.x;
    w[4 * h + 1] = T.out_x ? a.y : a.x;
    w[4 * h + 2] = T.out_x ? a.x : a.y;
    w[4 * h + 3] = a.y;
  }
}

// Split and band words that dense tile `tile` of pair r covers, set to 0: the
// planes of a pair whose output is constant over the grid (every variance and
// band value is exactly 0). Words as the tile kernels write them: tile 0 the
// parents of depths 1..4 and the band words of depths 0..4, tile t >= 1 the 32
// parent words and 128 band words of its 64 x 64 block.
__device__ __forceinline__ void zero_tile(const DTileArgs& A, int r, int tile, int tid, int nthreads) {
  uint32_t* split_row = A.split + int64_t(r) * A.n_words;
  const int64_t band_base = int64_t(r) * A.band_stride - A.band_shift;
  if (tile > 0) {
    int u = tile - 1, d = kPyramidTop + 1;
    while (u >= (1 << (2 * (d - kPyramidTop - 1)))) { u -= 1 << (2 * (d - kPyramidTop - 1)); d++; }
    const uint32_t mb = uint32_t(u) * uint32_t(kTileSide * kTileSide);
    for (int k = tid; k < 32; k += nthreads) split_row[A.word_off[d - 1] + mb / 128 + k] = 0u;
    for (int k = tid; k < 128; k += nthreads) A.bandb[band_base + A.word_off[d] + mb / 32 + k] = 0u;
    return;
  }
  const int d_hi = min(A.D, kPyramidTop);
  for (int d = 0; d <= d_hi; d++) {
    const int nq = 1 << (2 * d);
    if (d >= 1)
      for (int k = tid; k < (nq + 31) / 32; k += nthreads) split_row[A.word_off[d - 1] + k] = 0u;
    for (int k = tid; k < (4 * nq + 31) / 32; k += nthreads) A.bandb[band_base + A.word_off[d] + k] = 0u;
  }
}

// Fused mode: the planes of constant-output pairs (ranks rank_beg + blockIdx.y);
// the CTAs of a pair take its tiles in turn.
__global__ void __launch_bounds__(128) zero_tiles_kernel(const DTileArgs A) {
  const int r = A.order[A.rank_beg + blockIdx.y];
  for (int t = A.tile_beg + int(blockIdx.x); t < A.tile_beg + A.n_tiles; t += int(gridDim.x))
    zero_tile(A, r, t, threadIdx.x, blockDim.x);
}

// The shared tile stores position (i, j) of a T x T tile at row j + 2, column
// i + 2 (pitch T + 4): two-column padding keeps sibling pairs 8-byte aligned;
// the ring of out-of-tile neighbours sits in columns / rows 1 and T + 2.
constexpr int kPad = 2;
constexpr int kWtFull = (kTileSide + 2 * kPad) * (kTileSide + 2 * kPad);
// The pyramid tile's padded grids of depths 0..4, one after the other; its node
// tables follow them in the same buffer.
// sum over e < d of (2^(e+1) + 4)^2 = (4^(d+1) - 4) / 3 + 16 (2^d - 1) + 16 d (kPad = 2)
static_assert(kPad == 2, "wt_seg's closed form");
__host__ __device__ constexpr int wt_seg(int d) { return ((4 << (2 * d)) - 4) / 3 + 16 * ((1 << d) - 1) + 16 * d; }
constexpr int kWtPyr = wt_seg(kPyramidTop + 1);
constexpr int kTileBuf = kWtFull + 2 * kDenseMax * kTabFull;
static_assert(kWtPyr % 4 == 0 && kWtPyr + 2 * kDenseMax * kTabPyr <= kTileBuf, "pyramid tables fit the tile buffer");

// Plane words of a 64 x 64 tile whose output depends on one coordinate. In a
// word of 32 sibling quads (Morton order), quad bit b has x = 8 xhi + (b0 b2 b4)
// and y = 4 yhi + (b1 b3), with xhi = word bits (1, 3) and yhi = word bits
// (0, 2, 4). Given a bit per column pair (x) or row pair (y), the word places
// it at every quad of that column (row).
__device__ __forceinline__ uint32_t word_of_columns(uint32_t bits32, uint32_t w) {
  const uint32_t xhi = ((w >> 1) & 1u) | ((w >> 2) & 2u);
  const uint32_t b = (bits32 >> (8 * xhi)) & 0xffu;
  // column bit k to Morton position spread(k) (y = 0), then the four rows (offsets 0, 2, 8, 10)
  const uint32_t m = (b & 3u) | ((b & 0xcu) << 2) | ((b & 0x30u) << 12) | ((b & 0xc0u) << 14);
  return m * 0x505u;
}
__device__ __forceinline__ uint32_t word_of_rows(uint32_t bits32, uint32_t w) {
  const uint32_t yhi = (w & 1u) | ((w >> 1) & 2u) | ((w >> 2) & 4u);
  const uint32_t n = (bits32 >> (4 * yhi)) & 0xfu;
  // row bit k to Morton position 2 spread(k) (x = 0), then the eight columns
  const uint32_t m = (n & 1u) | ((n & 2u) << 1) | ((n & 4u) << 6) | ((n & 8u) << 7);
  return m * 0x00330033u;
}

// CTAs resident per SM that each class is compiled for (bounds its registers).
constexpr int dense_min_blocks(int njmax, int tpb) { return (njmax <= 4 ? 2048 : njmax <= 8 ? 1536 : 1024) / tpb / 2; }

// The tile of depths 0..min(D, 4) of pair r (dense tile 0), by all TPB threads of the CTA:
// in fused mode its split and band words and its tile flag, in materialise mode its outputs
// and halo points. The pair's table programs, joint block and joint activations are in
// shared memory (s_ent, s_esrc, s_WJ, s_jact); s_buf holds kWtPyr floats of padded
// per-depth outputs, then the two axes' node tables (2 kDenseMax rows of kTabPyr).
template <int NJMAX, int TPB>
__device__ __forceinline__ void pyramid_tile(const DTileArgs& A, const int r, const int nv, const int nj,
                                             const uint32_t xm, const uint32_t ym, const float out_const,
                                             const float4 (*s_ent)[kDenseMax], const float2 (*s_esrc)[kEntSrcCap],
                                             const float* s_WJ, const int* s_jact, float* s_buf) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const uint32_t jm = ((1u << nv) - 1u) & ~(xm | ym);
  const bool ax_x = (xm | jm) != 0u, ax_y = (ym | jm) != 0u;
  const int n_ent_x = __popc((xm | jm) & ((1u << nv) - 1u)), n_ent_y = __popc((ym | jm) & ((1u << nv) - 1u));
  const bool fused = A.mode == kModeFused;
  const bool wfilter = A.w_min > 0.f;
  const float theta16 = 16.f * A.theta, band2 = A.band * A.band;
  uint32_t* split_row = A.split + int64_t(r) * A.n_words;
  const int64_t band_base = int64_t(r) * A.band_stride - A.band_shift;
  const int64_t prow = int64_t(r) * A.out_stride - A.out_shift;
  const int d_hi = min(A.D, kPyramidTop);
  float* s_wt = s_buf;
  float* tab = s_buf + kWtPyr;
  // node tables: depth e's coordinates -1 .. 2^(e+1) at columns tab_seg(e) + 1 ..
  {
    const int P = (4 << d_hi) - 2 + 2 * (d_hi + 1);  // sum over depths of 2^(d+1) + 2
    const int n_items = (ax_x ? P : 0) + (ax_y ? P : 0);
    for (int u = tid; u < n_items; u += TPB) {
      const int a = ax_x && u < P ? 0 : 1;
      int e = 0, v = a == 1 && ax_x ? u - P : u;
      while (v >= (2 << e) + 2) { v -= (2 << e) + 2; e++; }
      table_column(grid_coord(v - 1, __int_as_float((127 - (e + 1)) << 23)), tab_seg(e) + v + 1,
                   a ? n_ent_y : n_ent_x, s_ent[a], s_esrc[a], tab + a * kDenseMax * kTabPyr, kTabPyr);
    }
  }
  __syncthreads();
  PairTabs T;
  T.tx = tab;
  T.ty = tab + kDenseMax * kTabPyr;
  T.tw = kTabPyr;
  T.nv = nv;
  T.nj = nj;
  T.out_x = nv > 0 && ((xm >> (nv - 1)) & 1u) != 0u;
  T.orow = __popc(T.out_x ? xm : ym) - 1;  // an output of one coordinate (no joint node): its axis' last row
  T.out_const = out_const;

  // ---- tile 0: depths 0..min(D, 4). One pass evaluates the quads and ring points
  // of every depth (work items: the quads of depth 0, 1, ..., then four ring
  // points at a time), one barrier, then each depth is filtered from shared memory.
  const bool ring = fused || A.out_halo != nullptr;
  const int n_quads = ((4 << (2 * d_hi)) - 1) / 3;       // quads of depths 0..d_hi
  const int n_items = n_quads + (ring ? (4 << d_hi) - 2 : 0);  // + ring groups (side / 4 ... of each depth)
  // work item u's depth, its four points (li, lj) in that depth's grid (ring points
  // outside [0, 2^(e+1))), and whether it is a quad
  auto item_points = [&](int u, int& e, int (&li)[4], int (&lj)[4]) {
    e = 0;
    const bool quad = u < n_quads;
    if (quad) {
      while (((4 << (2 * e)) - 1) / 3 <= u) e++;
      const uint32_t q = uint32_t(u - ((1 << (2 * e)) - 1) / 3);
      const int pi = int(compact1by1(q)), pj = int(compact1by1(q >> 1));
#pragma unroll
      for (int c = 0; c < 4; c++) { li[c] = 2 * pi + (c & 1); lj[c] = 2 * pj + (c >> 1); }
    } else {
      const int g = u - n_quads;
      while ((2 << (e + 1)) - 2 <= g) e++;
      const int Te = 1 << (e + 1);
#pragma unroll
      for (int c = 0; c < 4; c++) {  // ring point t lies on side t / Te
        const int t = 4 * (g - ((2 << e) - 2)) + c, sd = t >> (e + 1), uu = t & (Te - 1);
        li[c] = sd == 0 ? -1 : sd == 1 ? Te : uu;
        lj[c] = sd == 2 ? -1 : sd == 3 ? Te : uu;
      }
    }
    return quad;
  };
  auto store_item = [&](int u, bool quad, int e, const int (&li)[4], const int (&lj)[4], const float* w) {
    const int Te = 1 << (e + 1), pitch = Te + 2 * kPad;
    if (fused) {
      const int sb = wt_seg(e);  // this depth's padded grid in shared memory
#pragma unroll
      for (int c = 0; c < 4; c++) s_wt[sb + (lj[c] + kPad) * pitch + li[c] + kPad] = w[c];
    } else if (quad) {
      const uint32_t q = uint32_t(u - ((1 << (2 * e)) - 1) / 3);
      *reinterpret_cast<float4*>(A.out + prow + A.level_off[e] + 4 * q) = make_float4(w[0], w[1], w[2], w[3]);
    } else {
#pragma unroll
      for (int c = 0; c < 4; c++) {
        const int hs = li[c] < 0 ? 0 : li[c] >= Te ? 1 : lj[c] < 0 ? 2 : 3;
        A.out_halo[int64_t(r) * A.n_halo + A.halo_off[e] + hs * Te + (hs < 2 ? lj[c] : li[c])] = w[c];
      }
    }
  };
  // IPT items a pass (their points evaluated together). Two measured slower than one (more
  // registers and spills in the block kernel than the extra work in flight gains).
  constexpr int IPT = 1;
  for (int u0 = tid; u0 < n_items; u0 += IPT * TPB) {
    int e[IPT], li[IPT][4], lj[IPT][4], xp[4 * IPT], yp[4 * IPT];
    bool quad[IPT], valid[IPT];
#pragma unroll
    for (int k = 0; k < IPT; k++) {
      const int u = u0 + k * TPB;
      valid[k] = u < n_items;
      quad[k] = item_points(valid[k] ? u : u0, e[k], li[k], lj[k]);  // past the end: item u0 again
#pragma unroll
      for (int c = 0; c < 4; c++) {
        xp[4 * k + c] = tab_seg(e[k]) + li[k][c] + 2;
        yp[4 * k + c] = tab_seg(e[k]) + lj[k][c] + 2;
      }
    }
    float w[4 * IPT];
    eval_points<NJMAX, 4 * IPT>(T, s_WJ, s_jact, xp, yp, w);
#pragma unroll
    for (int k = 0; k < IPT; k++)
      if (valid[k]) store_item(u0 + k * TPB, quad[k], e[k], li[k], lj[k], w + 4 * k);
  }
  if (!fused) return;
  __syncthreads();
  // Variance and band test of depths 0..d_hi, one item per quad: depths d_hi .. 3 in whole
  // warps of 32 quads (their band words are quad-major), then depths 2, 1 and 0 packed into one
  // warp (lanes 0-15, 16-19 and 20). The band screen of the 64 x 64 tiles applies: a quad with
  // 16 V <= band^2 has no passing position, and the full test runs only in warps where some
  // quad fails the screen.
  int n_big = 0;
  for (int e = kQuadMajorFrom; e <= d_hi; e++) n_big += 1 << (2 * e);
  const int n_band_items = n_big + 32;
  auto depth_of = [&](int u, int* q) {  // an item of the whole-warp depths
    int e = d_hi;
    while (u >= (1 << (2 * e))) { u -= 1 << (2 * e); e--; }
    *q = u;
    return e;
  };
  bool any_pass = false;
  for (int base = 0; base < n_band_items; base += TPB) {
    const int u = base + tid;
    int e = -1, q = 0;
    if (u < n_big) {
      e = depth_of(u, &q);
    } else if (u < n_band_items) {
      const int v = u - n_big;
      e = v < 16 ? 2 : v < 20 ? 1 : v == 20 ? 0 : -1;
      q = v < 16 ? v : v < 20 ? v - 16 : 0;
      if (e > d_hi) e = -1;
    }
    bool pass[4] = {false, false, false, false}, split = false, screened_out = true;
    float w[4] = {0.f, 0.f, 0.f, 0.f};
    const float* t = s_wt;
    int pitch = 0;
    if (e >= 0) {
      const int Te = 1 << (e + 1);
      const int sb = wt_seg(e);
      pitch = Te + 2 * kPad;
      const int pi = int(compact1by1(uint32_t(q))), pj = int(compact1by1(uint32_t(q) >> 1));
      t = s_wt + sb + (2 * pj + kPad) * pitch + 2 * pi + kPad;
      w[0] = t[0]; w[1] = t[1]; w[2] = t[pitch]; w[3] = t[pitch + 1];
      // the four children give the parent's variance (Section 3.2)
      const float v16 = var16(w[0], w[1], w[2], w[3]);
      split = v16 > theta16;
      screened_out = v16 <= band2;
    }
    if (__any_sync(kFull, !screened_out) && !screened_out) {
      const float L[4] = {t[-1], w[0], t[pitch - 1], w[2]}, R[4] = {w[1], t[2], w[3], t[pitch + 2]};
      const float Bo[4] = {t[-pitch], t[-pitch + 1], w[0], w[1]};
      const float U[4] = {w[2], w[3], t[2 * pitch], t[2 * pitch + 1]};
#pragma unroll
      for (int c = 0; c < 4; c++) {
        pass[c] = band_pass_sq(sqdiff(w[c], L[c]), sqdiff(w[c], R[c]), sqdiff(w[c], Bo[c]), sqdiff(w[c], U[c]),
                               band2);
        if (wfilter) pass[c] = pass[c] && fabsf(w[c]) > A.w_min;
      }
    }
    const uint32_t bs = __ballot_sync(kFull, split);
    const uint32_t b0 = __ballot_sync(kFull, pass[0]), b1 = __ballot_sync(kFull, pass[1]);
    const uint32_t b2 = __ballot_sync(kFull, pass[2]), b3 = __ballot_sync(kFull, pass[3]);
    any_pass = any_pass || (b0 | b1 | b2 | b3) != 0u;
    const int wbase = base + warp * 32;  // this warp's first item
    if (wbase < n_big) {
      int q0;
      const int ew = depth_of(wbase, &q0);
      if (lane == 0) split_row[A.word_off[ew - 1] + q0 / 32] = bs;
      if (lane < 4)
        A.bandb[band_base + A.word_off[ew] + 4 * (q0 / 32) + lane] = lane == 0 ? b0 : lane == 1 ? b1 : lane == 2 ? b2 : b3;
    } else if (wbase == n_big) {  // depths 2, 1, 0: position-major words
      if (d_hi >= 2) {
        if (lane == 0) split_row[A.word_off[1]] = bs & 0xffffu;
        if (lane < 2) A.bandb[band_base + A.word_off[2] + lane] = band_word(b0, b1, b2, b3, lane);
      }
      if (d_hi >= 1) {
        if (lane == 2) split_row[A.word_off[0]] = (bs >> 16) & 0xfu;
        if (lane == 3)
          A.bandb[band_base + A.word_off[1]] = band_word((b0 >> 16) & 0xfu, (b1 >> 16) & 0xfu, (b2 >> 16) & 0xfu,
                                                         (b3 >> 16) & 0xfu, 0);
      }
      if (lane == 4)
        A.bandb[band_base + A.word_off[0]] = band_word((b0 >> 20) & 1u, (b1 >> 20) & 1u, (b2 >> 20) & 1u,
                                                       (b3 >> 20) & 1u, 0);
    }
    if (A.out && e >= 0 && (pass[0] | pass[1] | pass[2] | pass[3])) {
      const int64_t lrow = prow + A.level_off[e];
#pragma unroll
      for (int c = 0; c < 4; c++)
        if (pass[c]) A.out[lrow + 4 * q + c] = w[c];
    }
  }
  if (A.tile_flags && __syncthreads_or(any_pass) && tid == 0) A.tile_flags[int64_t(r) * A.n_dense] = 1;
}

template <int NJMAX, int TPB>
__global__ void __launch_bounds__(TPB, dense_min_blocks(NJMAX, TPB)) tile_kernel_dense(const DTileArgs A) {
  static_assert(NJMAX <= kDenseMax, "joint block holds at most kDenseMax rows");
  static_assert(TPB >= 64 && TPB <= 256 && (TPB & (TPB - 1)) == 0, "tile work divides evenly");
  constexpr int QPT = kTileSide * kTileSide / 4 / TPB;  // quads per thread in a 64 x 64 tile
  constexpr int P64 = kTileSide + 2 * kPad;
  constexpr int NJ1 = NJMAX > 0 ? NJMAX : 1;
  __shared__ __align__(16) float s_WJ[NJ1 * NJ1];
  __shared__ int s_jact[NJ1];
  __shared__ float4 s_ent[2][kDenseMax];  // table programs of the two axes
  __shared__ float2 s_esrc[2][kEntSrcCap];
  __shared__ __align__(16) float s_buf[kTileBuf];  // output tile with its ring, then the node tables
  // quad TPB k of a tile: its column and row offsets (in positions) and its shared-tile offset
  __shared__ int4 s_kq[QPT];
  // The next class's launch (other pairs, other outputs) may start filling the SMs
  // this one frees. When this launch overlaps its predecessor, its last CTA waits,
  // as it exits, for the predecessor to complete, so that this launch completes only
  // after it (later kernels in the stream read every launch's planes).
  pdl_trigger();
  const PdlWaitAtExit pdl_exit{last_cta()};
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (tid < QPT) {
    const int dx = int(compact1by1(uint32_t(TPB * tid))), dy = int(compact1by1(uint32_t(TPB * tid) >> 1));
    s_kq[tid] = make_int4(2 * dx, 2 * dy, 2 * dx + 2 * dy * P64, 0);
  }
  // ---- the pair: one record for the CTA's tiles
  const int64_t rank = A.rank_beg + blockIdx.y;
  const int r = A.order[rank];
  const uint8_t* rec = A.spec + int64_t(r) * A.L.stride;
  const int nv = reinterpret_cast<const int32_t*>(rec)[0];
  const float out_const = reinterpret_cast<const float*>(rec)[2];
  const uint32_t h3 = reinterpret_cast<const uint32_t*>(rec)[3];
  const int nj = int((h3 >> kHdrJointShift) & 0xfu);
  const uint32_t xm = (h3 >> kHdrXShift) & 0xfffu, ym = (h3 >> kHdrYShift) & 0xfffu;
  const uint32_t jm = ((1u << nv) - 1u) & ~(xm | ym);
  const bool fused = A.mode == kModeFused;
  const bool wfilter = A.w_min > 0.f;
  const float theta16 = 16.f * A.theta, band2 = A.band * A.band;
  const int t_beg = A.tile_beg + int(blockIdx.x) * A.tiles_per_cta;
  const int t_end = min(t_beg + A.tiles_per_cta, A.tile_beg + A.n_tiles);
  if (fused && nv == 0) {  // constant output: every variance and band value is exactly 0
    for (int t = t_beg; t < t_end; t++) zero_tile(A, r, t, tid, TPB);
    return;
  }
  {  // the pair's table programs, joint block and joint activations (built by spec_kernel)
    const float4* gent = reinterpret_cast<const float4*>(rec + A.L.ent_off());
    const float2* gsrc = reinterpret_cast<const float2*>(rec + A.L.esrc_off());
    for (int k = tid; k < 2 * kDenseMax; k += TPB) s_ent[k / kDenseMax][k % kDenseMax] = gent[k];
    for (int k = tid; k < 2 * kEntSrcCap; k += TPB) s_esrc[k / kEntSrcCap][k % kEntSrcCap] = gsrc[k];
    if constexpr (NJMAX > 0) {
      const float* gwj = reinterpret_cast<const float*>(rec + A.L.wj_off());
      for (int t = tid; t < NJMAX * NJMAX; t += TPB) s_WJ[t] = gwj[(t / NJMAX) * kDenseMax + t % NJMAX];
      if (tid < NJMAX) s_jact[tid] = reinterpret_cast<const int32_t*>(rec + A.L.jact_off())[tid];
    }
  }
  const bool ax_x = (xm | jm) != 0u, ax_y = (ym | jm) != 0u;
  const int n_ent_x = __popc((xm | jm) & ((1u << nv) - 1u)), n_ent_y = __popc((ym | jm) & ((1u << nv) - 1u));
  __syncthreads();
  uint32_t* split_row = A.split + int64_t(r) * A.n_words;
  const int64_t band_base = int64_t(r) * A.band_stride - A.band_shift;
  const int64_t prow = int64_t(r) * A.out_stride - A.out_shift;
  const int d_hi = min(A.D, kPyramidTop);
  float* s_wt = s_buf;

  // ---- one tile of the pair
  auto run_tile = [&](const int tile) {
    if (tile > 0) {  // a 64 x 64 tile; tile 0 (depths 0..4) below
      // geometry: a 64 x 64 tile of depth d >= 5 at Morton block mb
      int d = 0, i0 = 0, j0 = 0;
      uint32_t mb = 0;
      {
        int u = tile - 1;
        d = kPyramidTop + 1;
        while (u >= (1 << (2 * (d - kPyramidTop - 1)))) { u -= 1 << (2 * (d - kPyramidTop - 1)); d++; }
        mb = uint32_t(u) * uint32_t(kTileSide * kTileSide);
        i0 = int(compact1by1(mb));
        j0 = int(compact1by1(mb >> 1));
      }
      const int tw = kTabFull;
      float* tab = s_buf + kWtFull;
      // node tables, one coordinate per thread. A 64 x 64 tile with nodes on one axis
      // takes its 66 coordinates (ring included); with both, the 64 + 64 inside the
      // tile, and the four ring coordinates only where a ring is evaluated.
      auto column = [&](int a, float cv, int pos) {
        table_column(cv, pos, a ? n_ent_y : n_ent_x, s_ent[a], s_esrc[a], tab + a * kDenseMax * tw, tw);
      };
      {
        const float scale = __int_as_float((127 - (d + 1)) << 23);
        const int n_items = ax_x && ax_y ? 2 * kTileSide : (ax_x || ax_y) ? kTileSide + 2 : 0;
        for (int u = tid; u < n_items; u += TPB) {
          const int a = ax_x && ax_y ? u / kTileSide : ax_x ? 0 : 1;
          const int i = ax_x && ax_y ? u % kTileSide : u - 1;
          column(a, grid_coord((a ? j0 : i0) + i, scale), i + 2);
        }
      }
      __syncthreads();
      // the ring coordinates of a 64 x 64 tile with nodes on both axes (CTA-uniform call)
      auto ring_columns = [&]() {
        if (ax_x && ax_y) {
          if (tid < 4) {
            const int a = tid >> 1, i = tid & 1 ? kTileSide : -1;
            column(a, grid_coord((a ? j0 : i0) + i, __int_as_float((127 - (d + 1)) << 23)), i + 2);
          }
          __syncthreads();
        }
      };
      PairTabs T;
      T.tx = tab;
      T.ty = tab + kDenseMax * tw;
      T.tw = tw;
      T.nv = nv;
      T.nj = nj;
      T.out_x = nv > 0 && ((xm >> (nv - 1)) & 1u) != 0u;
      T.orow = __popc(T.out_x ? xm : ym) - 1;  // an output of one coordinate (no joint node): its axis' last row
      T.out_const = out_const;

      if constexpr (NJMAX == 0) {
        if (tile > 0 && fused && !A.out && nv > 0) {
          // ---- a 64 x 64 tile whose output f depends on one coordinate: every quad of a
          // column pair (x) or row pair (y) has the children f0, f1 (twice), so its
          // variance is 16 V = 4 (f0 - f1)^2 (the six-difference sum, exactly), and a
          // position's band value is the smaller squared difference to its two
          // neighbours along that coordinate (the other axis gives 0). Each warp takes
          // the 32 pairs (one per lane) and writes a quarter of the tile's words.
          const float* f = (T.out_x ? T.tx : T.ty) + T.orow * kTabFull;  // coordinate i at i + 2
          const float fl = f[2 * lane + 1], f0 = f[2 * lane + 2], f1 = f[2 * lane + 3], fr = f[2 * lane + 4];
          const float s01 = sqdiff(f0, f1);
          bool g0 = fminf(sqdiff(f0, fl), s01) > band2, g1 = fminf(s01, sqdiff(f1, fr)) > band2;
          if (wfilter) {
            g0 = g0 && fabsf(f0) > A.w_min;
            g1 = g1 && fabsf(f1) > A.w_min;
          }
          const uint32_t S = __ballot_sync(kFull, 4.f * s01 > theta16);
          const uint32_t G0 = __ballot_sync(kFull, g0), G1 = __ballot_sync(kFull, g1);
          // band word 4 j + c holds child c of the quads of split word j: child c lies in the
          // pair's first or second column (c & 1) or row (c >> 1)
          const uint32_t j = uint32_t(tid) >> 2, c = uint32_t(tid) & 3u;
          const uint32_t gsel = (T.out_x ? (c & 1u) : (c >> 1)) ? G1 : G0;
          A.bandb[band_base + A.word_off[d] + mb / 32 + tid] = T.out_x ? word_of_columns(gsel, j) : word_of_rows(gsel, j);
          if (tid < 32)
            split_row[A.word_off[d - 1] + mb / 128 + tid] =
                T.out_x ? word_of_columns(S, uint32_t(tid)) : word_of_rows(S, uint32_t(tid));
          if (A.tile_flags && tid == 0 && (G0 | G1) != 0u) A.tile_flags[int64_t(r) * A.n_dense + tile] = 1;
          return;
        }
      }
      {
        // ---- a full 64 x 64 tile of one depth >= 5: 4 quads and 1 ring point per thread
        const int n = 1 << (d + 1);
        const int64_t lrow = prow + A.level_off[d];
        // quad q = tid + TPB k of the tile has parent (pl + dx(k), ql + dy(k)), where
        // (dx, dy) are the Morton coordinates of TPB k (its bits lie above tid's)
        const int pl = int(compact1by1(uint32_t(tid))), ql = int(compact1by1(uint32_t(tid) >> 1));
        const int xb = 2 * pl + 2, yb = 2 * ql + 2;  // table columns of this thread's quad k = 0
        const int sbase = (2 * ql + kPad) * P64 + 2 * pl + kPad;
        uint32_t* split_k = split_row + A.word_off[d - 1] + mb / 128 + warp;  // this warp's parents, k = 0
        uint32_t* band_k = A.bandb + (band_base + A.word_off[d] + 4 * (mb / 128 + warp));
        // QPE quads per evaluation: quads k .. k + QPE - 1 share one pass over the joint nodes
        constexpr int QPE = NJMAX <= 6 ? 2 : 1;
        // A position passes the band test only if both differences along one axis
        // exceed the band, and one of them is to its sibling in the quad. The sum of the
        // six squared sibling differences (16 V, rounded upward monotonically) bounds
        // each of them, so a quad with 16 V within band^2 has no passing position,
        // whatever its neighbours; need: some quad of this thread may have one.
        bool need = false;
  #pragma unroll 1
        for (int k0 = 0; k0 < QPT; k0 += QPE) {
          float w[4 * QPE];
          int4 kq[QPE];
          int xq[QPE], yq[QPE];
  #pragma unroll
          for (int h = 0; h < QPE; h++) {
            kq[h] = s_kq[k0 + h];
            xq[h] = xb + kq[h].x;
            yq[h] = yb + kq[h].y;
          }
          eval_quads<NJMAX, QPE>(T, s_WJ, s_jact, xq, yq, w);
  #pragma unroll
          for (int h = 0; h < QPE; h++) {
            const int k = k0 + h;
            const float* wq = w + 4 * h;
            if (fused) {
              // the four children give the parent's variance (Section 3.2)
              const float v16 = var16(wq[0], wq[1], wq[2], wq[3]);
              const unsigned bal = __ballot_sync(kFull, v16 > theta16);
              if (lane == 0) split_k[(TPB / 32) * k] = bal;
              need = need || !(v16 <= band2);
            } else {
              *reinterpret_cast<float4*>(A.out + lrow + mb + 4 * (tid + TPB * k)) =
                  make_float4(wq[0], wq[1], wq[2], wq[3]);
            }
          }
        }
        if (fused && !__syncthreads_or(need)) {  // no position of the tile can pass
          if (lane == 0)
            for (int k = 0; k < QPT; k++) *reinterpret_cast<uint4*>(band_k + 4 * (TPB / 32) * k) = make_uint4(0, 0, 0, 0);
          return;
        }
        if (fused || A.out_halo) ring_columns();
        if (fused) {  // a tile the band screen lets through (rare): its outputs again, into the shared tile
  #pragma unroll 1
          for (int k0 = 0; k0 < QPT; k0 += QPE) {
            float w[4 * QPE];
            int4 kq[QPE];
            int xq[QPE], yq[QPE];
  #pragma unroll
            for (int h = 0; h < QPE; h++) {
              kq[h] = s_kq[k0 + h];
              xq[h] = xb + kq[h].x;
              yq[h] = yb + kq[h].y;
            }
            eval_quads<NJMAX, QPE>(T, s_WJ, s_jact, xq, yq, w);
  #pragma unroll
            for (int h = 0; h < QPE; h++) {
              float* t = s_wt + sbase + kq[h].z;
              *reinterpret_cast<float2*>(t) = make_float2(w[4 * h + 0], w[4 * h + 1]);
              *reinterpret_cast<float2*>(t + P64) = make_float2(w[4 * h + 2], w[4 * h + 3]);
            }
          }
        }
        // ring: 4 sides x 64 points, evaluated four at a time by threads 0..63
        // (point t = 4 tid + c lies on side t / 64, the same for all four)
        if (tid < kTileSide && (fused || A.out_halo)) {
          const int sd = tid >> 4, u0 = 4 * (tid & 15);
          int li[4], lj[4], xp[4], yp[4];
          float w[4];
  #pragma unroll
          for (int c = 0; c < 4; c++) {
            li[c] = sd == 0 ? -1 : sd == 1 ? kTileSide : u0 + c;
            lj[c] = sd == 2 ? -1 : sd == 3 ? kTileSide : u0 + c;
            xp[c] = li[c] + 2;
            yp[c] = lj[c] + 2;
          }
          const int gi = i0 + li[0], gj = j0 + lj[0];  // a side lies wholly inside or outside the domain
          const bool outside = gi < 0 || gi >= n || gj < 0 || gj >= n;
          if (fused || outside) {  // materialised: only points outside the domain are written
            eval_points<NJMAX, 4>(T, s_WJ, s_jact, xp, yp, w);
  #pragma unroll
            for (int c = 0; c < 4; c++) {
              if (fused) {
                s_wt[(lj[c] + kPad) * P64 + li[c] + kPad] = w[c];
              } else {
                const int pi_ = i0 + li[c], pj_ = j0 + lj[c];
                const int hs = pi_ < 0 ? 0 : pi_ >= n ? 1 : pj_ < 0 ? 2 : 3;
                A.out_halo[int64_t(r) * A.n_halo + A.halo_off[d] + hs * n + (hs < 2 ? pj_ : pi_)] = w[c];
              }
            }
          }
        }
        if (!fused) return;
        __syncthreads();
        // band value of each position from its four neighbours at distance 2^-d
        bool any_pass = false;
  #pragma unroll 2
        for (int k = 0; k < QPT; k++) {
          const float* t = s_wt + sbase + s_kq[k].z;  // (2pi, 2pj)
          const float2 w01 = *reinterpret_cast<const float2*>(t), w23 = *reinterpret_cast<const float2*>(t + P64);
          const float2 bel = *reinterpret_cast<const float2*>(t - P64), abv = *reinterpret_cast<const float2*>(t + 2 * P64);
          const float l0 = t[-1], l2 = t[P64 - 1], r1 = t[2], r3 = t[P64 + 2];
          const float w[4] = {w01.x, w01.y, w23.x, w23.y};
          const float L[4] = {l0, w[0], l2, w[2]}, R[4] = {w[1], r1, w[3], r3};
          const float Bo[4] = {bel.x, bel.y, w[0], w[1]}, U[4] = {w[2], w[3], abv.x, abv.y};
          bool pass[4];
          // squared differences between siblings are shared by both
          const float h01 = sqdiff(w[0], w[1]), h23 = sqdiff(w[2], w[3]);
          const float v02 = sqdiff(w[0], w[2]), v13 = sqdiff(w[1], w[3]);
          const float DL[4] = {sqdiff(w[0], L[0]), h01, sqdiff(w[2], L[2]), h23};
          const float DR[4] = {h01, sqdiff(w[1], R[1]), h23, sqdiff(w[3], R[3])};
          const float DB[4] = {sqdiff(w[0], Bo[0]), sqdiff(w[1], Bo[1]), v02, v13};
          const float DT[4] = {v02, v13, sqdiff(w[2], U[2]), sqdiff(w[3], U[3])};
  #pragma unroll
          for (int c = 0; c < 4; c++) pass[c] = band_pass_sq(DL[c], DR[c], DB[c], DT[c], band2);
          if (wfilter) {
  #pragma unroll
            for (int c = 0; c < 4; c++) pass[c] = pass[c] && fabsf(w[c]) > A.w_min;
          }
          const uint32_t b0 = __ballot_sync(kFull, pass[0]), b1 = __ballot_sync(kFull, pass[1]);
          const uint32_t b2 = __ballot_sync(kFull, pass[2]), b3 = __ballot_sync(kFull, pass[3]);
          any_pass = any_pass || (b0 | b1 | b2 | b3) != 0u;
          if (lane == 0)  // the four quad-major words of this warp's 32 quads
            *reinterpret_cast<uint4*>(band_k + 4 * (TPB / 32) * k) = make_uint4(b0, b1, b2, b3);
          if (A.out && (pass[0] | pass[1] | pass[2] | pass[3])) {
            float* o = A.out + lrow + mb + 4 * (tid + TPB * k);
  #pragma unroll
            for (int c = 0; c < 4; c++)
              if (pass[c]) o[c] = w[c];
          }
        }
        if (A.tile_flags && __syncthreads_or(any_pass) && tid == 0) A.tile_flags[int64_t(r) * A.n_dense + tile] = 1;
        return;
      }
    }
    pyramid_tile<NJMAX, TPB>(A, r, nv, nj, xm, ym, out_const, s_ent, s_esrc, s_WJ, s_jact, s_buf);
  };

  for (int t = t_beg; t < t_end; t++) {
    if (t > t_beg) __syncthreads();  // the previous tile's reads of the shared buffer are done
    run_tile(t);
  }
}

// The depths 0..4 tile (dense tile 0) of the pairs in one launch, fused mode: a CTA
// per pair, the record's table programs, joint block and activations staged in
// shared memory, then pyramid_tile. The block kernel does the same among its other
// paths; this kernel holds only this one, so its CTAs fetch less code.
constexpr int kPyrTPB = 128;  // threads per pyramid CTA
template <int NJMAX>
__global__ void __launch_bounds__(kPyrTPB, dense_min_blocks(NJMAX, kPyrTPB)) tile_kernel_pyramid(const DTileArgs A) {
  constexpr int NJ1 = NJMAX > 0 ? NJMAX : 1;
  __shared__ __align__(16) float s_WJ[NJ1 * NJ1];
  __shared__ int s_jact[NJ1];
  __shared__ float4 s_ent[2][kDenseMax];
  __shared__ float2 s_esrc[2][kEntSrcCap];
  __shared__ __align__(16) float s_buf[kWtPyr + 2 * kDenseMax * kTabPyr];
  // Launched to overlap the record kernel, every CTA waits for its records first; the
  // launches after this one may start only then (they read the records unwaited).
  if (A.wait_at_start) pdl_wait();
  pdl_trigger();
  const PdlWaitAtExit pdl_exit{last_cta()};
  const int tid = threadIdx.x;
  const int r = A.order[A.rank_beg + blockIdx.y];
  const uint8_t* rec = A.spec + int64_t(r) * A.L.stride;
  const int nv = reinterpret_cast<const int32_t*>(rec)[0];
  const float out_const = reinterpret_cast<const float*>(rec)[2];
  const uint32_t h3 = reinterpret_cast<const uint32_t*>(rec)[3];
  const int nj = int((h3 >> kHdrJointShift) & 0xfu);
  const uint32_t xm = (h3 >> kHdrXShift) & 0xfffu, ym = (h3 >> kHdrYShift) & 0xfffu;
  if (nv == 0) {  // constant output: every variance and band value is exactly 0
    zero_tile(A, r, 0, tid, kPyrTPB);
    return;
  }
  {
    const float4* gent = reinterpret_cast<const float4*>(rec + A.L.ent_off());
    const float2* gsrc = reinterpret_cast<const float2*>(rec + A.L.esrc_off());
    for (int k = tid; k < 2 * kDenseMax; k += kPyrTPB) s_ent[k / kDenseMax][k % kDenseMax] = gent[k];
    for (int k = tid; k < 2 * kEntSrcCap; k += kPyrTPB) s_esrc[k / kEntSrcCap][k % kEntSrcCap] = gsrc[k];
    if constexpr (NJMAX > 0) {
      const float* gwj = reinterpret_cast<const float*>(rec + A.L.wj_off());
      for (int t = tid; t < NJMAX * NJMAX; t += kPyrTPB) s_WJ[t] = gwj[(t / NJMAX) * kDenseMax + t % NJMAX];
      if (tid < NJMAX) s_jact[tid] = reinterpret_cast<const int32_t*>(rec + A.L.jact_off())[tid];
    }
  }
  __syncthreads();
  pyramid_tile<NJMAX, kPyrTPB>(A, r, nv, nj, xm, ym, out_const, s_ent, s_esrc, s_WJ, s_jact, s_buf);
}

// The 64 x 64 tiles of pairs whose output depends on one coordinate (no joint
// node; fused mode, no output buffer): a warp per tile, four tiles at a time per
// CTA, no block barrier. The warp evaluates the output's axis table at the
// tile's 64 coordinates (two per lane), then filters per column (row) pair as
// in tile_kernel_dense; the two ring coordinates are evaluated only where an
// edge column's band test can pass (its pair's squared difference exceeds
// band^2: otherwise the smaller difference cannot).
constexpr int kOneAxisWarps = 4;
constexpr int kOneAxisBlocks = 12;  // CTAs per SM the kernel is compiled for
__global__ void __launch_bounds__(32 * kOneAxisWarps, kOneAxisBlocks) tile_kernel_one_axis(const DTileArgs A) {
  __shared__ float4 s_ent[kDenseMax];
  __shared__ float2 s_esrc[kEntSrcCap];
  __shared__ __align__(16) float s_tab[kOneAxisWarps][kDenseMax * kTabFull];
  pdl_trigger();
  const PdlWaitAtExit pdl_exit{last_cta()};
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int r = A.order[A.rank_beg + blockIdx.y];
  const uint8_t* rec = A.spec + int64_t(r) * A.L.stride;
  const int nv = reinterpret_cast<const int32_t*>(rec)[0];
  const uint32_t h3 = reinterpret_cast<const uint32_t*>(rec)[3];
  const uint32_t xm = (h3 >> kHdrXShift) & 0xfffu, ym = (h3 >> kHdrYShift) & 0xfffu;
  const bool out_x = nv > 0 && ((xm >> (nv - 1)) & 1u) != 0u;
  const int a = out_x ? 0 : 1;
  const uint32_t om = out_x ? xm : ym;
  const int n_ent = __popc(om & ((1u << nv) - 1u)), orow = __popc(om) - 1;
  {
    const float4* gent = reinterpret_cast<const float4*>(rec + A.L.ent_off()) + a * kDenseMax;
    const float2* gsrc = reinterpret_cast<const float2*>(rec + A.L.esrc_off()) + a * kEntSrcCap;
    if (tid < kDenseMax) s_ent[tid] = gent[tid];
    for (int k = tid; k < kEntSrcCap; k += 32 * kOneAxisWarps) s_esrc[k] = gsrc[k];
  }
  __syncthreads();
  if (nv == 0) return;  // (constant pairs are not launched here)
  uint32_t* split_row = A.split + int64_t(r) * A.n_words;
  const int64_t band_base = int64_t(r) * A.band_stride - A.band_shift;
  const bool wfilter = A.w_min > 0.f;
  const float theta16 = 16.f * A.theta, band2 = A.band * A.band;
  float* tab = s_tab[warp];
  const float* f = tab + orow * kTabFull;  // coordinate i at i + 2
  const int t_beg = A.tile_beg + int(blockIdx.x) * A.tiles_per_cta;
  const int t_end = min(t_beg + A.tiles_per_cta, A.tile_beg + A.n_tiles);
  for (int tile = t_beg + warp; tile < t_end; tile += kOneAxisWarps) {
    int u = tile - 1, d = kPyramidTop + 1;
    while (u >= (1 << (2 * (d - kPyramidTop - 1)))) { u -= 1 << (2 * (d - kPyramidTop - 1)); d++; }
    const uint32_t mb = uint32_t(u) * uint32_t(kTileSide * kTileSide);
    const int c0 = int(compact1by1(out_x ? mb : mb >> 1));  // first column (row) of the tile
    const float scale = __int_as_float((127 - (d + 1)) << 23);
    __syncwarp();  // the previous tile's reads of this warp's table are done
    table_column(grid_coord(c0 + lane, scale), lane + 2, n_ent, s_ent, s_esrc, tab, kTabFull);
    table_column(grid_coord(c0 + lane + 32, scale), lane + 34, n_ent, s_ent, s_esrc, tab, kTabFull);
    __syncwarp();
    const float f0 = f[2 * lane + 2], f1 = f[2 * lane + 3];
    const float s01 = sqdiff(f0, f1);
    const bool ring_l = __shfl_sync(kFull, s01 > band2, 0), ring_r = __shfl_sync(kFull, s01 > band2, 31);
    if (ring_l || ring_r) {
      if (lane == 0 && ring_l) table_column(grid_coord(c0 - 1, scale), 1, n_ent, s_ent, s_esrc, tab, kTabFull);
      if (lane == 1 && ring_r) table_column(grid_coord(c0 + 64, scale), 66, n_ent, s_ent, s_esrc, tab, kTabFull);
      __syncwarp();
    }
    // (an edge neighbour not evaluated is only read where the pair's own difference decides)
    const float fl = f[2 * lane + 1], fr = f[2 * lane + 4];
    bool g0 = fminf(sqdiff(f0, fl), s01) > band2, g1 = fminf(s01, sqdiff(f1, fr)) > band2;
    if (wfilter) {
      g0 = g0 && fabsf(f0) > A.w_min;
      g1 = g1 && fabsf(f1) > A.w_min;
    }
    const uint32_t S = __ballot_sync(kFull, 4.f * s01 > theta16);
    const uint32_t G0 = __ballot_sync(kFull, g0), G1 = __ballot_sync(kFull, g1);
    uint32_t* band_t = A.bandb + (band_base + A.word_off[d] + mb / 32);
#pragma unroll
    for (int k = 0; k < 4; k++) {  // band word 4 j + c: child c of the quads of split word j
      const uint32_t wi = uint32_t(4 * lane + k), j = wi >> 2, c = wi & 3u;
      const uint32_t gsel = (out_x ? (c & 1u) : (c >> 1)) ? G1 : G0;
      band_t[wi] = out_x ? word_of_columns(gsel, j) : word_of_rows(gsel, j);
    }
    split_row[A.word_off[d - 1] + mb / 128 + lane] =
        out_x ? word_of_columns(S, uint32_t(lane)) : word_of_rows(S, uint32_t(lane));
    if (A.tile_flags && lane == 0 && (G0 | G1) != 0u) A.tile_flags[int64_t(r) * A.n_dense + tile] = 1;
  }
}

// The 64 x 64 tiles of pairs with joint nodes (fused mode, no output buffer): a
// warp per tile, kWarpTiles tiles of one pair at a time per CTA. The warp fills
// its own node tables (the tile's 64 + 64 coordinates, two per lane and axis),
// then each lane evaluates 32 sibling quads (quad l + 32 k: the lanes' ballot
// for k is split word k of the tile) two per pass (one above 6 joint nodes). A
// tile whose band screen fires (rare) is left to the whole CTA after the warps'
// tiles: its tables and ring again, its outputs into a shared tile (which takes
// the place of the other warps' tables), and the band test from shared memory,
// 128 threads at a time; every other tile stores zero band words.
constexpr int kWarpTiles = 4;
constexpr int warp_min_blocks(int njmax) { return njmax <= 2 ? 7 : njmax <= 8 ? 6 : 4; }

// Column (row) offset of quad 32 k of a 64 x 64 tile, in positions: Morton bits
// 6, 8 of the quad index are x bits 3, 4 (bits 5, 7, 9: y bits 2, 3, 4).
__device__ __forceinline__ int warp_quad_dx(int k) { return 2 * (8 * ((k >> 1) & 1) + 16 * ((k >> 3) & 1)); }
__device__ __forceinline__ int warp_quad_dy(int k) { return 2 * (4 * (k & 1) + 8 * ((k >> 2) & 1) + 16 * ((k >> 4) & 1)); }

// The warp kernel's quads on packed pairs up to 8 joint nodes (measured). The 3..4-joint class
// needs its six-CTA budget for them: under seven CTAs' registers the moves that form the pairs
// took as many issue slots as the packed arithmetic saved. The 9..12-joint class (128 registers
// at four CTAs per SM) stays scalar.
__host__ __device__ constexpr bool warp_packed(int njmax) { return njmax <= 8; }
template <int NJMAX, int QPE>
__device__ __forceinline__ void warp_quads(const PairTabs& T, const float* __restrict__ WJ, const f2* __restrict__ WJ2,
                                           const int* __restrict__ jact, const int (&xq)[QPE], const int (&yq)[QPE],
                                           float (&w)[4 * QPE]) {
  if constexpr (warp_packed(NJMAX))
    eval_quads_packed<NJMAX, QPE>(T, WJ2, jact, xq, yq, w);
  else
    eval_quads<NJMAX, QPE>(T, WJ, jact, xq, yq, w);
}

template <int NJMAX>
__global__ void __launch_bounds__(32 * kWarpTiles, warp_min_blocks(NJMAX)) tile_kernel_warp(const DTileArgs A) {
  static_assert(NJMAX >= 1 && NJMAX <= kDenseMax, "pairs with joint nodes");
  // quads per pass (measured): four up to 4 joint nodes, two above
  constexpr int QPE = NJMAX <= 4 ? 4 : 2;
  __shared__ __align__(16) float s_WJ[NJMAX * NJMAX];
  __shared__ f2 s_WJ2[NJMAX * NJMAX];  // the same weights twice each, for the packed quads
  __shared__ int s_jact[NJMAX];
  __shared__ float4 s_ent[2][kDenseMax];
  __shared__ float2 s_esrc[2][kEntSrcCap];
  __shared__ __align__(16) float s_tab[kWarpTiles][2 * kDenseMax * kTabFull];
  __shared__ int s_defer[kWarpTiles];  // the CTA's tiles whose band screen fired
  __shared__ int s_ndefer;
  static_assert(kWarpTiles >= 4 && (kWarpTiles - 1) * 2 * kDenseMax * kTabFull >= kWtFull,
                "the shared output tile fits in the tables of warps 1..kWarpTiles-1");
  pdl_trigger();
  const PdlWaitAtExit pdl_exit{last_cta()};
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (tid == 0) s_ndefer = 0;
  const int r = A.order[A.rank_beg + blockIdx.y];
  const uint8_t* rec = A.spec + int64_t(r) * A.L.stride;
  const int nv = reinterpret_cast<const int32_t*>(rec)[0];
  const uint32_t h3 = reinterpret_cast<const uint32_t*>(rec)[3];
  const int nj = int((h3 >> kHdrJointShift) & 0xfu);
  const uint32_t xm = (h3 >> kHdrXShift) & 0xfffu, ym = (h3 >> kHdrYShift) & 0xfffu;
  const uint32_t jm = ((1u << nv) - 1u) & ~(xm | ym);
  {
    const float4* gent = reinterpret_cast<const float4*>(rec + A.L.ent_off());
    const float2* gsrc = reinterpret_cast<const float2*>(rec + A.L.esrc_off());
    const float* gwj = reinterpret_cast<const float*>(rec + A.L.wj_off());
    for (int k = tid; k < 2 * kDenseMax; k += 32 * kWarpTiles) s_ent[k / kDenseMax][k % kDenseMax] = gent[k];
    for (int k = tid; k < 2 * kEntSrcCap; k += 32 * kWarpTiles) s_esrc[k / kEntSrcCap][k % kEntSrcCap] = gsrc[k];
    for (int t = tid; t < NJMAX * NJMAX; t += 32 * kWarpTiles) {
      const float wk = gwj[(t / NJMAX) * kDenseMax + t % NJMAX];
      s_WJ[t] = wk;
      s_WJ2[t] = f2_splat(wk);
    }
    if (tid < NJMAX) s_jact[tid] = reinterpret_cast<const int32_t*>(rec + A.L.jact_off())[tid];
  }
  __syncthreads();
  const int n_ent_x = __popc((xm | jm) & ((1u << nv) - 1u)), n_ent_y = __popc((ym | jm) & ((1u << nv) - 1u));
  uint32_t* split_row = A.split + int64_t(r) * A.n_words;
  const int64_t band_base = int64_t(r) * A.band_stride - A.band_shift;
  const bool wfilter = A.w_min > 0.f;
  const float theta16 = 16.f * A.theta, band2 = A.band * A.band;
  float* tx = s_tab[warp];
  float* ty = tx + kDenseMax * kTabFull;
  PairTabs T;
  T.tx = tx;
  T.ty = ty;
  T.tw = kTabFull;
  T.nv = nv;
  T.nj = nj;
  T.out_x = false;
  T.orow = 0;
  T.out_const = 0.f;
  // this lane's quads: parent (pl, ql) + (dx(k), dy(k)) / 2 of quad lane + 32 k
  const int pl = int(compact1by1(uint32_t(lane))), ql = int(compact1by1(uint32_t(lane) >> 1));
  const int xb = 2 * pl + 2, yb = 2 * ql + 2;  // table columns of its quad k = 0
  const int t_beg = A.tile_beg + int(blockIdx.x) * A.tiles_per_cta;
  const int t_end = min(t_beg + A.tiles_per_cta, A.tile_beg + A.n_tiles);
  for (int tile = t_beg + warp; tile < t_end; tile += kWarpTiles) {
    int u = tile - 1, d = kPyramidTop + 1;
    while (u >= (1 << (2 * (d - kPyramidTop - 1)))) { u -= 1 << (2 * (d - kPyramidTop - 1)); d++; }
    const uint32_t mb = uint32_t(u) * uint32_t(kTileSide * kTileSide);
    const int i0 = int(compact1by1(mb)), j0 = int(compact1by1(mb >> 1));
    const float scale = __int_as_float((127 - (d + 1)) << 23);
    __syncwarp();  // the previous tile's reads of this warp's tables are done
    {
      const int pos[2] = {lane + 2, lane + 34};
      const float cx[2] = {grid_coord(i0 + lane, scale), grid_coord(i0 + lane + 32, scale)};
      table_columns<2>(cx, pos, n_ent_x, s_ent[0], s_esrc[0], tx, kTabFull);
      const float cy[2] = {grid_coord(j0 + lane, scale), grid_coord(j0 + lane + 32, scale)};
      table_columns<2>(cy, pos, n_ent_y, s_ent[1], s_esrc[1], ty, kTabFull);
    }
    __syncwarp();
    uint32_t* split_k = split_row + A.word_off[d - 1] + mb / 128;  // split word k of the tile
    // A position passes the band test only if both differences along one axis
    // exceed the band, and one of them is to its sibling in the quad; 16 V bounds
    // each sibling difference, so a quad with 16 V within band^2 has none.
    bool need = false;
#pragma unroll 1
    for (int k0 = 0; k0 < 32; k0 += QPE) {
      float w[4 * QPE];
      int xq[QPE], yq[QPE];
#pragma unroll
      for (int h = 0; h < QPE; h++) {
        xq[h] = xb + warp_quad_dx(k0 + h);
        yq[h] = yb + warp_quad_dy(k0 + h);
      }
      warp_quads<NJMAX, QPE>(T, s_WJ, s_WJ2, s_jact, xq, yq, w);
#pragma unroll
      for (int h = 0; h < QPE; h++) {
        // the four children give the parent's variance (Section 3.2)
        const float v16 = var16(w[4 * h + 0], w[4 * h + 1], w[4 * h + 2], w[4 * h + 3]);
        const unsigned bal = __ballot_sync(kFull, v16 > theta16);
        if (lane == 0) split_k[k0 + h] = bal;
        need = need || !(v16 <= band2);
      }
    }
    uint32_t* band_t = A.bandb + (band_base + A.word_off[d] + mb / 32);  // 128 quad-major words
    if (!__any_sync(kFull, need)) {  // no position of the tile can pass
      reinterpret_cast<uint4*>(band_t)[lane] = make_uint4(0u, 0u, 0u, 0u);
      continue;
    }
    if (lane == 0) s_defer[atomicAdd(&s_ndefer, 1)] = tile;  // the CTA's band test, below
  }
  __syncthreads();  // every warp's tiles are done: the tables are free
  const int n_defer = s_ndefer;
  // A tile whose band screen fired: its band test by the whole CTA. Its tables (ring
  // coordinates included) go to warp 0's slot, its outputs and ring into a shared tile
  // over the other slots (position (i, j) at row j + kPad, column i + kPad), then each
  // thread tests quads tid + 128 k from shared memory.
  constexpr int P64 = kTileSide + 2 * kPad;
  constexpr int NT = 32 * kWarpTiles;
  float* s_wt = s_tab[1];
  T.tx = s_tab[0];
  T.ty = s_tab[0] + kDenseMax * kTabFull;
  for (int q = 0; q < n_defer; q++) {
    const int tile = s_defer[q];
    int u = tile - 1, d = kPyramidTop + 1;
    while (u >= (1 << (2 * (d - kPyramidTop - 1)))) { u -= 1 << (2 * (d - kPyramidTop - 1)); d++; }
    const uint32_t mb = uint32_t(u) * uint32_t(kTileSide * kTileSide);
    const int i0 = int(compact1by1(mb)), j0 = int(compact1by1(mb >> 1));
    const float scale = __int_as_float((127 - (d + 1)) << 23);
    if (q > 0) __syncthreads();  // the previous tile's reads of the tables and the shared tile are done
    for (int v = tid; v < 2 * (kTileSide + 2); v += NT) {  // coordinates -1 .. 64 of each axis
      const int ax = v / (kTileSide + 2), i = v % (kTileSide + 2) - 1;
      table_column(grid_coord((ax ? j0 : i0) + i, scale), i + 2, ax ? n_ent_y : n_ent_x, s_ent[ax], s_esrc[ax],
                   ax ? const_cast<float*>(T.ty) : const_cast<float*>(T.tx), kTabFull);
    }
    __syncthreads();
#pragma unroll 1
    for (int k0 = 0; k0 < kTileSide * kTileSide / 4 / NT; k0 += QPE) {  // the tile's quads into the shared tile
      float w[4 * QPE];
      int xq[QPE], yq[QPE], so[QPE];
#pragma unroll
      for (int h = 0; h < QPE; h++) {
        const uint32_t qi = uint32_t(tid + NT * (k0 + h));
        const int px = int(compact1by1(qi)), py = int(compact1by1(qi >> 1));
        xq[h] = 2 * px + 2;
        yq[h] = 2 * py + 2;
        so[h] = (2 * py + kPad) * P64 + 2 * px + kPad;
      }
      warp_quads<NJMAX, QPE>(T, s_WJ, s_WJ2, s_jact, xq, yq, w);
#pragma unroll
      for (int h = 0; h < QPE; h++) {
        *reinterpret_cast<float2*>(s_wt + so[h]) = make_float2(w[4 * h + 0], w[4 * h + 1]);
        *reinterpret_cast<float2*>(s_wt + so[h] + P64) = make_float2(w[4 * h + 2], w[4 * h + 3]);
      }
    }
    if (tid < kTileSide) {  // the ring: 4 sides x 64 points, four at a time
      const int sd = tid >> 4, u0 = 4 * (tid & 15);
      int li[4], lj[4], xp[4], yp[4];
      float w[4];
#pragma unroll
      for (int c = 0; c < 4; c++) {
        li[c] = sd == 0 ? -1 : sd == 1 ? kTileSide : u0 + c;
        lj[c] = sd == 2 ? -1 : sd == 3 ? kTileSide : u0 + c;
        xp[c] = li[c] + 2;
        yp[c] = lj[c] + 2;
      }
      eval_points<NJMAX, 4>(T, s_WJ, s_jact, xp, yp, w);
#pragma unroll
      for (int c = 0; c < 4; c++) s_wt[(lj[c] + kPad) * P64 + li[c] + kPad] = w[c];
    }
    __syncthreads();
    uint32_t* band_t = A.bandb + (band_base + A.word_off[d] + mb / 32);
    bool any_pass = false;
#pragma unroll 1
    for (int k = 0; k < kTileSide * kTileSide / 4 / NT; k++) {
      const uint32_t qi = uint32_t(tid + NT * k);  // quad lane + 32 (warp + kWarpTiles k)
      const int px = int(compact1by1(qi)), py = int(compact1by1(qi >> 1));
      const float* t = s_wt + (2 * py + kPad) * P64 + 2 * px + kPad;  // child 0
      const float2 w01 = *reinterpret_cast<const float2*>(t), w23 = *reinterpret_cast<const float2*>(t + P64);
      const float2 bel = *reinterpret_cast<const float2*>(t - P64), abv = *reinterpret_cast<const float2*>(t + 2 * P64);
      const float w[4] = {w01.x, w01.y, w23.x, w23.y};
      const float L[4] = {t[-1], w[0], t[P64 - 1], w[2]}, R[4] = {w[1], t[2], w[3], t[P64 + 2]};
      const float Bo[4] = {bel.x, bel.y, w[0], w[1]}, U[4] = {w[2], w[3], abv.x, abv.y};
      bool pass[4];
#pragma unroll
      for (int c = 0; c < 4; c++) {
        pass[c] = band_pass_sq(sqdiff(w[c], L[c]), sqdiff(w[c], R[c]), sqdiff(w[c], Bo[c]), sqdiff(w[c], U[c]), band2);
        if (wfilter) pass[c] = pass[c] && fabsf(w[c]) > A.w_min;
      }
      const uint32_t b0 = __ballot_sync(kFull, pass[0]), b1 = __ballot_sync(kFull, pass[1]);
      const uint32_t b2 = __ballot_sync(kFull, pass[2]), b3 = __ballot_sync(kFull, pass[3]);
      any_pass = any_pass || (b0 | b1 | b2 | b3) != 0u;
      if (lane < 4)  // quad-major words of quads 32 kk .. 32 kk + 31, kk = warp + kWarpTiles k
        band_t[4 * (warp + kWarpTiles * k) + lane] = lane == 0 ? b0 : lane == 1 ? b1 : lane == 2 ? b2 : b3;
    }
    if (__syncthreads_or(any_pass) && A.tile_flags && tid == 0) A.tile_flags[int64_t(r) * A.n_dense + tile] = 1;
  }
}

// ---- filter planes from a materialised evaluation ---------------------------------

struct GridDev {
  int32_t D;
  int64_t n_total, n_halo, n_words, n_qblocks;
  int64_t level_off[EMR_MAX_DEPTH + 2], halo_off[EMR_MAX_DEPTH + 2], word_off[EMR_MAX_DEPTH + 2];
  int64_t qblk_off[EMR_MAX_DEPTH + 2];  // first block of 32 sibling quads of each depth
};

__device__ __forceinline__ int level_of_word(const GridDev& G, int64_t wi) {
  int d = 0;
  while (G.word_off[d + 1] <= wi) d++;
  return d;
}

// Bits of word wi (depth d) that correspond to grid positions (depths 0 and 1 fill part of a word).
__device__ __forceinline__ uint32_t valid_bits(const GridDev& G, int d, int64_t wi) {
  const uint32_t m0 = uint32_t(wi - G.word_off[d]) * 32u;
  const uint32_t cnt = 1u << (2 * (d + 1));
  return cnt - m0 >= 32 ? kFull : ((1u << (cnt - m0)) - 1u);
}

// One warp per block of 32 sibling quads (128 positions) of one depth; lane =
// quad. Each lane reads its four outputs, their children (variance) and their
// neighbours (band) from the materialised outputs.
__global__ void planes_kernel(const float* __restrict__ out, const float* __restrict__ out_halo, GridDev G,
                              int64_t n_pairs, float theta, float band, float w_min, uint32_t* __restrict__ split,
                              uint32_t* __restrict__ bandb, float* __restrict__ var_dbg) {
  const int lane = threadIdx.x & 31;
  const int64_t wg = (int64_t(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  if (wg >= n_pairs * G.n_qblocks) return;
  const int64_t r = wg / G.n_qblocks, qb = wg % G.n_qblocks;
  int d = 0;
  while (G.qblk_off[d + 1] <= qb) d++;
  const uint32_t b = uint32_t(qb - G.qblk_off[d]);
  const uint32_t q = 32u * b + uint32_t(lane);  // quad (parent) index at depth d
  const uint32_t nq = 1u << (2 * d);
  const bool valid = q < nq;
  const int n = 1 << (d + 1);
  const float theta16 = 16.f * theta, band2 = band * band;
  const float* o = out + r * G.n_total;
  bool sp[4] = {false, false, false, false}, bp[4] = {false, false, false, false};
  if (valid) {
    const int pi = int(compact1by1(q)), pj = int(compact1by1(q >> 1));
    const float4 w4 = *reinterpret_cast<const float4*>(o + G.level_off[d] + 4 * int64_t(q));
    const float w[4] = {w4.x, w4.y, w4.z, w4.w};
#pragma unroll
    for (int c = 0; c < 4; c++) {
      const int i = 2 * pi + (c & 1), j = 2 * pj + (c >> 1);
      const uint32_t m = 4 * q + uint32_t(c);
      float S = 0.f;
      if (d < G.D) {
        const float4 ch = *reinterpret_cast<const float4*>(o + G.level_off[d + 1] + 4 * int64_t(m));
        S = var16(ch.x, ch.y, ch.z, ch.w);
        sp[c] = S > theta16;
      }
      if (var_dbg) var_dbg[r * G.n_total + G.level_off[d] + m] = 0.0625f * S;
      float nbv[4];
      const int ni[4] = {i - 1, i + 1, i, i}, nj[4] = {j, j, j - 1, j + 1};
#pragma unroll
      for (int k = 0; k < 4; k++) {
        if (ni[k] >= 0 && ni[k] < n && nj[k] >= 0 && nj[k] < n) {
          nbv[k] = o[G.level_off[d] + morton2(uint32_t(ni[k]), uint32_t(nj[k]))];
        } else {
          const int sd = ni[k] < 0 ? 0 : ni[k] >= n ? 1 : nj[k] < 0 ? 2 : 3;
          const int t = sd < 2 ? nj[k] : ni[k];
          nbv[k] = out_halo[r * G.n_halo + G.halo_off[d] + sd * n + t];
        }
      }
      bp[c] = band_pass_sq(sqdiff(w[c], nbv[0]), sqdiff(w[c], nbv[1]), sqdiff(w[c], nbv[2]), sqdiff(w[c], nbv[3]),
                           band2);
      if (w_min > 0.f) bp[c] = bp[c] && fabsf(w[c]) > w_min;
    }
  }
  const uint32_t s0 = __ballot_sync(kFull, sp[0]), s1 = __ballot_sync(kFull, sp[1]);
  const uint32_t s2 = __ballot_sync(kFull, sp[2]), s3 = __ballot_sync(kFull, sp[3]);
  const uint32_t b0 = __ballot_sync(kFull, bp[0]), b1 = __ballot_sync(kFull, bp[1]);
  const uint32_t b2 = __ballot_sync(kFull, bp[2]), b3 = __ballot_sync(kFull, bp[3]);
  // position-major words of this block: 4 (fewer at depths 0..2)
  const int nw = int(min(4u, (4u * nq - 128u * b + 31u) / 32u));
  const int64_t w0 = r * G.n_words + G.word_off[d] + 4 * int64_t(b);
  if (lane < nw) split[w0 + lane] = band_word(s0, s1, s2, s3, lane);
  if (d >= kQuadMajorFrom) {
    if (lane < 4) bandb[w0 + lane] = lane == 0 ? b0 : lane == 1 ? b1 : lane == 2 ? b2 : b3;
  } else if (lane < nw) {
    bandb[w0 + lane] = band_word(b0, b1, b2, b3, lane);
  }
}

// A (possibly chunk-local) bit plane: word w of pair r is p[r * stride + w - shift].
struct PlaneView {
  uint32_t* p;
  int64_t stride, shift;
  __device__ __forceinline__ uint32_t& at(int64_t r, int64_t w) const { return p[r * stride + w - shift]; }
};

// Active bits (Eq. 2: every ancestor split) of the 32 positions of word wi at
// depth d; the ancestors at each shallower depth lie in a single word.
__device__ __forceinline__ uint32_t active_bits(const uint32_t* sp, const GridDev& G, int d, int64_t wi) {
  const uint32_t m0 = uint32_t(wi - G.word_off[d]) * 32u;
  uint32_t act = kFull;
  for (int k = 1; k <= d && act; k++) {
    const uint32_t a0 = m0 >> (2 * k);
    const uint32_t aw = sp[G.word_off[d - k] + (a0 >> 5)];
    uint32_t bits = 0;
    for (int bb = 0; bb < 32; bb++) {
      const uint32_t anc = (m0 + uint32_t(bb)) >> (2 * k);
      bits |= ((aw >> (anc & 31u)) & 1u) << bb;
    }
    act &= bits;
  }
  return act;
}

// Connection-type filter (Section 6 taxonomy): a connection between a pair's
// query slot (a, b) and a grid position is a self-loop when both are the same
// point, else forward / backward / lateral as the source's y is below / above /
// equal to the target's (outgoing side: the slot is the source; incoming: the
// position is). types: EMR_CONN_* bits to keep; EMR_CONN_ALL disables it.
struct TypeFilter {
  int32_t types;
  QueryDev q;
};

// Row r (y offset) and column c (x offset) of the 32 Morton positions of a word:
// bits 1 and 3 of the position in the word carry y, bits 0, 2 and 4 carry x.
__device__ __forceinline__ uint32_t word_row_bits(int r) { return 0x00330033u << (((r & 1) << 1) | ((r & 2) << 2)); }
__device__ __forceinline__ uint32_t word_col_bits(int c) {
  return 0x0505u << ((c & 1) | ((c & 2) << 1) | ((c & 4) << 2));
}

// Kept-type bits of the 32 positions of position-major word wi (depth d) for pair r.
__device__ __noinline__ uint32_t type_bits(const TypeFilter& tf, int64_t r, const GridDev& G, int d, int64_t wi) {
  const int64_t si = tf.q.per_genome ? r : r % tf.q.S;
  const float a = tf.q.a[si], b = tf.q.b[si];
  const bool out_side = tf.q.side[si] == EMR_SIDE_OUT;
  const uint32_t m0 = uint32_t(wi - G.word_off[d]) * 32u;
  const int i0 = int(compact1by1(m0)), j0 = int(compact1by1(m0 >> 1));
  const float scale = __int_as_float((127 - (d + 1)) << 23);
  uint32_t fw = 0u, bw = 0u, lw = 0u, sw = 0u;
  for (int rr = 0; rr < 4; rr++) {
    const float y = grid_coord(j0 + rr, scale);
    const float ys = out_side ? b : y, yt = out_side ? y : b;
    const uint32_t row = word_row_bits(rr);
    if (ys < yt) {
      fw |= row;
    } else if (ys > yt) {
      bw |= row;
    } else {
      lw |= row;
      for (int c = 0; c < 8; c++)  // the slot itself, if it is a position of this row
        if (grid_coord(i0 + c, scale) == a) sw |= row & word_col_bits(c);
    }
  }
  lw &= ~sw;
  return ((tf.types & EMR_CONN_F) ? fw : 0u) | ((tf.types & EMR_CONN_B) ? bw : 0u) |
         ((tf.types & EMR_CONN_L) ? lw : 0u) | ((tf.types & EMR_CONN_S) ? sw : 0u);
}

// mask = band AND NOT split (no split at depth D); gated: AND Eq. 2's active bit.
// One thread per group of 4 words (one 128-position block from depth 3 on; the
// 4 words of depths 0..2 form group 0), pair = blockIdx.y; groups cover words
// [w0, w0 + nw) (w0 and nw multiples of 4, or nw reaching n_words). split is a
// whole-grid plane. Planes start at pair r0 (the type filter's slots are absolute).
// Mask words wi .. wi + nwk - 1 (a group of 4 words: one 128-position block from
// depth 3 on, or the 4 words of depths 0..2) of pair r: band (re-interleaved to
// position-major) AND NOT split, gated AND active, AND kept connection types.
// sp: the pair's split row; bw: its band words (indexed by global word); ra: the
// pair's absolute number for the type filter.
__device__ __forceinline__ void combine_group(const uint32_t* __restrict__ sp, const uint32_t* bw, const GridDev& G,
                                              int64_t wi, int nwk, int gated, const TypeFilter& tf, int64_t ra,
                                              uint32_t (&m)[4]) {
  if (wi >= G.word_off[kQuadMajorFrom]) {
    int d = kQuadMajorFrom;
    while (G.word_off[d + 1] <= wi) d++;
    const uint4 bq = *reinterpret_cast<const uint4*>(bw + wi);
    const uint4 sq = d < G.D ? *reinterpret_cast<const uint4*>(sp + wi) : make_uint4(0, 0, 0, 0);
    const uint32_t s4[4] = {sq.x, sq.y, sq.z, sq.w};
#pragma unroll
    for (int c = 0; c < 4; c++) {  // re-interleave the block's four child words
      m[c] = band_word(bq.x, bq.y, bq.z, bq.w, c) & ~s4[c];
      if (gated && m[c]) m[c] &= active_bits(sp, G, d, wi + c);
      if (tf.types != EMR_CONN_ALL && m[c]) m[c] &= type_bits(tf, ra, G, d, wi + c);
    }
  } else {
    for (int c = 0; c < 4; c++) {
      m[c] = 0u;
      if (c >= nwk) continue;
      const int64_t wc = wi + c;
      int d = 0;
      while (G.word_off[d + 1] <= wc) d++;
      uint32_t keep = bw[wc] & valid_bits(G, d, wc);
      if (d < G.D) keep &= ~sp[wc];
      if (gated && keep) keep &= active_bits(sp, G, d, wc);
      if (tf.types != EMR_CONN_ALL && keep) keep &= type_bits(tf, ra, G, d, wc);
      m[c] = keep;
    }
  }
}

__global__ void combine_kernel(const uint32_t* __restrict__ split, PlaneView band, PlaneView mask, GridDev G,
                               int64_t w0, int64_t nw, int gated, TypeFilter tf, int64_t r0) {
  const int64_t k = (int64_t(blockIdx.x) * blockDim.x + threadIdx.x) * 4;
  if (k >= nw) return;
  const int64_t r = blockIdx.y;
  const int64_t wi = w0 + k;
  const uint32_t* sp = split + r * G.n_words;
  const int nwk = nw - k < 4 ? int(nw - k) : 4;
  uint32_t m[4];
  combine_group(sp, &band.at(r, 0), G, wi, nwk, gated, tf, r0 + r, m);
  if (wi >= G.word_off[kQuadMajorFrom]) {
    *reinterpret_cast<uint4*>(&mask.at(r, wi)) = make_uint4(m[0], m[1], m[2], m[3]);
  } else {
    for (int c = 0; c < nwk; c++) mask.at(r, wi + c) = m[c];
  }
}

// ---- ordered compaction -----------------------------------------------------------

constexpr int kCompactBlock = 256;  // words per compaction block (8192 positions)

__device__ __forceinline__ int block_exclusive_scan(int v, int* sh, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(kFull, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) sh[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int t = lane < nw ? sh[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(kFull, t, o);
      if (lane >= o) t += y;
    }
    if (lane < nw) sh[lane] = t;
  }
  __syncthreads();
  const int before = warp ? sh[warp - 1] : 0;
  if (total) *total = sh[nw - 1];
  __syncthreads();
  return before + x - v;
}

// Four words of pair r starting at word wi (a multiple of 4) with the bits that
// are not grid positions cleared; words past w_end read as 0.
__device__ __forceinline__ void load_mask4(const PlaneView& mask, const GridDev& G, int64_t r, int64_t wi,
                                           int64_t w_end, uint32_t (&m)[4]) {
  if (wi + 4 <= w_end && wi >= G.word_off[kQuadMajorFrom]) {
    const uint4 v = *reinterpret_cast<const uint4*>(&mask.at(r, wi));
    m[0] = v.x; m[1] = v.y; m[2] = v.z; m[3] = v.w;
    return;
  }
#pragma unroll
  for (int c = 0; c < 4; c++) {
    const int64_t wc = wi + c;
    m[c] = wc < w_end ? mask.at(r, wc) & valid_bits(G, level_of_word(G, wc), wc) : 0u;
  }
}

// grid (blocks of kCompactBlock * 4 words, pairs): set bits per block.
__global__ void compact_count_kernel(PlaneView mask, GridDev G, int64_t w0, int64_t nw, int nb, int64_t r0,
                                     int32_t* __restrict__ bcount) {
  __shared__ int sh[32];
  const int64_t r = r0 + blockIdx.y;
  const int64_t k = (int64_t(blockIdx.x) * kCompactBlock + threadIdx.x) * 4;
  uint32_t m[4] = {0u, 0u, 0u, 0u};
  if (k < nw) load_mask4(mask, G, r, w0 + k, w0 + nw, m);
  const int c = __popc(m[0]) + __popc(m[1]) + __popc(m[2]) + __popc(m[3]);
  int total;
  block_exclusive_scan(c, sh, &total);
  if (threadIdx.x == 0) bcount[r * nb + blockIdx.x] = total;
}

// One CTA per pair: exclusive scan of its block counts.
__global__ void compact_scan_pair_kernel(const int32_t* __restrict__ bcount, int nb, int32_t* __restrict__ boff,
                                         int64_t* __restrict__ counts) {
  __shared__ int sh[32];
  const int64_t r = blockIdx.x;
  int carry = 0;
  for (int k0 = 0; k0 < nb; k0 += blockDim.x) {
    const int k = k0 + threadIdx.x;
    const int v = k < nb ? bcount[r * nb + k] : 0;
    int total;
    const int ex = block_exclusive_scan(v, sh, &total);
    if (k < nb) boff[r * nb + k] = carry + ex;
    carry += total;
  }
  if (threadIdx.x == 0) counts[r] = carry;
}

// One CTA: exclusive scan of the pair counts (int64).
__global__ void compact_scan_pairs_kernel(const int64_t* __restrict__ counts, int64_t n_pairs,
                                          int64_t* __restrict__ offsets) {
  __shared__ long long sh[32];
  pdl_wait();  // the counts
  pdl_trigger();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  long long carry = 0;
  for (int64_t k0 = 0; k0 < n_pairs; k0 += blockDim.x) {
    const int64_t k = k0 + threadIdx.x;
    const long long v = k < n_pairs ? counts[k] : 0;
    long long x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const long long y = __shfl_up_sync(kFull, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) sh[warp] = x;
    __syncthreads();
    if (warp == 0) {
      long long t = lane < nw ? sh[lane] : 0;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const long long y = __shfl_up_sync(kFull, t, o);
        if (lane >= o) t += y;
      }
      if (lane < nw) sh[lane] = t;
    }
    __syncthreads();
    const long long before = warp ? sh[warp - 1] : 0;
    if (k < n_pairs) offsets[k] = carry + before + x - v;
    carry += sh[nw - 1];
    __syncthreads();
  }
  if (threadIdx.x == 0) offsets[n_pairs] = carry;
}

// CPPN output of one grid point from a pair's record, in the evaluators'
// common order (see the record layout), so the value equals the one the tile
// kernels computed at that position. Node values go to a local array.
__device__ float eval_record_point(const uint8_t* rec, const SpecLayout& L, float x, float y) {
  const int nv = reinterpret_cast<const int32_t*>(rec)[0];
  const float out_const = reinterpret_cast<const float*>(rec)[2];
  const float4* coef = reinterpret_cast<const float4*>(rec + L.coef_off());
  const uint2* ve = reinterpret_cast<const uint2*>(rec + L.edge_off());
  float v[EMR_MAX_VARYING];
  const float xs[1] = {x}, ys[1] = {y};
  float z[1] = {out_const};
  for (int k = 0; k < nv; k++) {
    const float4 c = coef[k];
    const uint32_t info = __float_as_uint(c.w);
    const int eb = int((info >> 8) & 0xfffu), ee = eb + int(info >> 20);
    node_input_sparse<1>(c, ve, eb, ee, xs, ys, [&](int src, int) { return v[src]; }, z);
    z[0] = act_apply(int(info & 0xfu), z[0]);
    v[k] = z[0];
  }
  return z[0];
}

// Per-pair records (pair r at spec + r * L.stride) from which the kept weights
// are recomputed instead of read from materialised outputs.
struct RecordSource {
  const uint8_t* spec;
  SpecLayout L;
};

// when out is NULL and rs.spec is set, the weights are recomputed from the records.
__global__ void compact_write_kernel(PlaneView mask, const float* __restrict__ out, int64_t out_stride,
                                     int64_t out_shift, GridDev G, int64_t w0, int64_t nw, int nb,
                                     int64_t r0, const int32_t* __restrict__ boff,
                                     const int64_t* __restrict__ offsets, int64_t cap, int32_t* __restrict__ idx,
                                     float* __restrict__ wv) {
  __shared__ int sh[32];
  const int64_t r = r0 + blockIdx.y;
  const int64_t k = (int64_t(blockIdx.x) * kCompactBlock + threadIdx.x) * 4;
  uint32_t m[4] = {0u, 0u, 0u, 0u};
  if (k < nw) load_mask4(mask, G, r, w0 + k, w0 + nw, m);
  const int ex = block_exclusive_scan(__popc(m[0]) + __popc(m[1]) + __popc(m[2]) + __popc(m[3]), sh, nullptr);
  if (!(m[0] | m[1] | m[2] | m[3])) return;
  int64_t dst = offsets[r] + boff[r * nb + blockIdx.x] + ex;
  for (int c = 0; c < 4; c++) {
    if (!m[c]) continue;
    const int64_t wi = w0 + k + c;
    const int d = level_of_word(G, wi);
    const int64_t gbase = G.level_off[d] + (wi - G.word_off[d]) * 32;
    for (uint32_t v = m[c]; v; v &= v - 1, dst++) {
      const int64_t gidx = gbase + __ffs(v) - 1;
      if (dst < cap) {
        idx[dst] = int32_t(gidx);
        if (out && wv) wv[dst] = out[r * out_stride + gidx - out_shift];
      }
    }
  }
}

// The pair whose list holds entry t: the last r with offsets[r] <= t.
__device__ __forceinline__ int64_t pair_of_entry(const int64_t* __restrict__ offsets, int64_t n_pairs, int64_t t) {
  int64_t lo = 0, hi = n_pairs;  // offsets[lo] <= t < offsets[hi]
  while (hi - lo > 1) {
    const int64_t mid = (lo + hi) >> 1;
    if (offsets[mid] <= t) lo = mid; else hi = mid;
  }
  return lo;
}

// Weights of the listed kept positions, recomputed from the records: one entry
// per thread (kept positions cluster, so a thread per mask word would evaluate
// long runs serially). The entry's pair is the last r with offsets[r] <= t.
__global__ void __launch_bounds__(kCompactBlock) kept_weights_kernel(RecordSource rs, GridDev G,
                                                                     const int64_t* __restrict__ offsets,
                                                                     int64_t n_pairs, int64_t cap,
                                                                     const int32_t* __restrict__ idx,
                                                                     float* __restrict__ wv) {
  const int64_t total = offsets[n_pairs] < cap ? offsets[n_pairs] : cap;
  for (int64_t t = int64_t(blockIdx.x) * kCompactBlock + threadIdx.x; t < total;
       t += int64_t(gridDim.x) * kCompactBlock) {
    const int64_t lo = pair_of_entry(offsets, n_pairs, t);
    const int64_t gidx = idx[t];
    int d = 0;
    while (G.level_off[d + 1] <= gidx) d++;
    const uint32_t m = uint32_t(gidx - G.level_off[d]);
    const float scale = __int_as_float((127 - (d + 1)) << 23);  // 2^-(d+1)
    const float x = grid_coord(int(compact1by1(m)), scale), y = grid_coord(int(compact1by1(m >> 1)), scale);
    wv[t] = eval_record_point(rs.spec + lo * rs.L.stride, rs.L, x, y);
  }
}

// Connection type code of each list entry (0 forward, 1 backward, 2 lateral,
// 3 self; Section 6 taxonomy), from the pair's query slot and the position.
__global__ void __launch_bounds__(kCompactBlock) conn_types_kernel(QueryDev q, GridDev G,
                                                                   const int64_t* __restrict__ offsets,
                                                                   int64_t n_pairs, int64_t cap,
                                                                   const int32_t* __restrict__ idx,
                                                                   uint8_t* __restrict__ type) {
  const int64_t total = offsets[n_pairs] < cap ? offsets[n_pairs] : cap;
  for (int64_t t = int64_t(blockIdx.x) * kCompactBlock + threadIdx.x; t < total;
       t += int64_t(gridDim.x) * kCompactBlock) {
    const int64_t r = pair_of_entry(offsets, n_pairs, t);
    const int64_t si = q.per_genome ? r : r % q.S;
    const float a = q.a[si], b = q.b[si];
    const bool out_side = q.side[si] == EMR_SIDE_OUT;
    const int64_t gidx = idx[t];
    int d = 0;
    while (G.level_off[d + 1] <= gidx) d++;
    const uint32_t m = uint32_t(gidx - G.level_off[d]);
    const float scale = __int_as_float((127 - (d + 1)) << 23);
    const float x = grid_coord(int(compact1by1(m)), scale), y = grid_coord(int(compact1by1(m >> 1)), scale);
    const float xs = out_side ? a : x, ys = out_side ? b : y, xt = out_side ? x : a, yt = out_side ? y : b;
    type[t] = (xs == xt && ys == yt) ? 3 : ys < yt ? 0 : ys > yt ? 1 : 2;
  }
}

// Eq. 2 gate of n listed entries (global entry numbers e0 .. e0 + n - 1 of
// lists with the given offsets): keep[t] = 1 when every ancestor of the entry's
// position split, read from the complete split plane.
__global__ void __launch_bounds__(kCompactBlock) gate_kernel(const uint32_t* __restrict__ split, GridDev G,
                                                             const int64_t* __restrict__ offsets, int64_t n_pairs,
                                                             int64_t e0, int64_t n, const int32_t* __restrict__ idx,
                                                             uint8_t* __restrict__ keep) {
  for (int64_t t = int64_t(blockIdx.x) * kCompactBlock + threadIdx.x; t < n; t += int64_t(gridDim.x) * kCompactBlock) {
    const int64_t r = pair_of_entry(offsets, n_pairs, e0 + t);
    const int64_t gidx = idx[t];
    int d = 0;
    while (G.level_off[d + 1] <= gidx) d++;
    const uint32_t m = uint32_t(gidx - G.level_off[d]);
    const uint32_t* sp = split + r * G.n_words;
    bool act = true;
    for (int k = 1; k <= d && act; k++) {
      const uint32_t am = m >> (2 * k);  // ancestor at depth d - k
      act = (sp[G.word_off[d - k] + (am >> 5)] >> (am & 31u)) & 1u;
    }
    keep[t] = act ? 1 : 0;
  }
}

// ---- selection over flagged tiles ---------------------------------------------------
//
// Mask combine, ordered compaction and kept weights in two passes (count, write)
// that visit only the tiles whose flag says some band bit is set: every other
// tile's mask is 0 whatever its split bits. One CTA per pair.

constexpr int kSelectThreads = 128;

// Words [*wb, *we) of dense tile t: tile 0 holds depths 0..min(D, 4), tile t >= 1 the
// 128 words of one 64 x 64 block of a depth >= 5.
__device__ __forceinline__ void tile_words(const GridDev& G, int32_t t, int64_t* wb, int64_t* we) {
  if (t == 0) {
    *wb = 0;
    *we = G.word_off[(G.D < kPyramidTop ? G.D : kPyramidTop) + 1];
  } else {
    *wb = G.word_off[kPyramidTop + 1] + int64_t(t - 1) * (kTileSide * kTileSide / 32);
    *we = *wb + kTileSide * kTileSide / 32;
  }
}

// One warp per pair (kSelectThreads / 32 pairs a CTA): the flags are read 32 at a
// time and the flagged tiles taken in ascending order from the ballot; scans are
// warp shuffles, so no CTA barrier is needed. Every loop is warp-uniform.

__device__ __forceinline__ int warp_exclusive_scan(int v, int* total) {
  const int lane = threadIdx.x & 31;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(kFull, x, o);
    if (lane >= o) x += y;
  }
  *total = __shfl_sync(kFull, x, 31);
  return x - v;
}

__global__ void __launch_bounds__(kSelectThreads) select_count_kernel(const uint32_t* __restrict__ split,
                                                                      const uint32_t* __restrict__ bandb,
                                                                      const uint8_t* __restrict__ flags,
                                                                      int64_t n_dense, GridDev G_arg, int gated,
                                                                      TypeFilter tf, int64_t n_pairs,
                                                                      int64_t* __restrict__ counts,
                                                                      int32_t* __restrict__ tile_base,
                                                                      int64_t* __restrict__ items,
                                                                      unsigned long long* __restrict__ n_items) {
  __shared__ GridDev G;  // dynamically indexed below: a shared copy instead of a local one
  for (int k = threadIdx.x; k < int(sizeof(GridDev) / 4); k += blockDim.x)
    reinterpret_cast<int*>(&G)[k] = reinterpret_cast<const int*>(&G_arg)[k];
  __syncthreads();
  pdl_wait();  // the tile launches' planes and flags
  pdl_trigger();
  const int lane = threadIdx.x & 31;
  const int64_t r = (int64_t(blockIdx.x) * kSelectThreads + threadIdx.x) >> 5;
  if (r >= n_pairs) return;  // whole warps
  const uint32_t* sp = split + r * G.n_words;
  const uint32_t* bw = bandb + r * G.n_words;
  int run = 0;  // entries of the pair's earlier flagged tiles
  for (int64_t t0 = 0; t0 < n_dense; t0 += 32) {
    const int64_t t = t0 + lane;
    uint32_t bal = __ballot_sync(kFull, t < n_dense && flags[r * n_dense + t]);
    for (; bal; bal &= bal - 1) {
      const int64_t tt = t0 + __ffs(bal) - 1;
      int64_t wb, we;
      tile_words(G, int32_t(tt), &wb, &we);
      int sum = 0;
      for (int64_t wi = wb + 4 * lane; wi < we; wi += 128) {
        uint32_t m[4];
        combine_group(sp, bw, G, wi, we - wi < 4 ? int(we - wi) : 4, gated, tf, r, m);
        sum += __popc(m[0]) + __popc(m[1]) + __popc(m[2]) + __popc(m[3]);
      }
#pragma unroll
      for (int o = 16; o; o >>= 1) sum += __shfl_xor_sync(kFull, sum, o);
      if (lane == 0 && sum > 0) {  // a work item for the write kernel
        tile_base[r * n_dense + tt] = run;
        items[atomicAdd(n_items, 1ull)] = r * n_dense + tt;
      }
      run += sum;
    }
  }
  if (lane == 0) counts[r] = run;
}

// One warp per work item (pair, tile with kept positions): the tile's list
// entries go to offsets[pair] + tile_base, in ascending global index.
__global__ void __launch_bounds__(kSelectThreads) select_write_kernel(const uint32_t* __restrict__ split,
                                                                      const uint32_t* __restrict__ bandb,
                                                                      int64_t n_dense, GridDev G_arg, int gated,
                                                                      TypeFilter tf,
                                                                      const int32_t* __restrict__ tile_base,
                                                                      const int64_t* __restrict__ items,
                                                                      const unsigned long long* __restrict__ n_items,
                                                                      const int64_t* __restrict__ offsets,
                                                                      int64_t cap, int32_t* __restrict__ idx,
                                                                      float* __restrict__ wv) {
  __shared__ GridDev G;  // dynamically indexed below: a shared copy instead of a local one
  for (int k = threadIdx.x; k < int(sizeof(GridDev) / 4); k += blockDim.x)
    reinterpret_cast<int*>(&G)[k] = reinterpret_cast<const int*>(&G_arg)[k];
  __syncthreads();
  pdl_wait();  // the offsets (and, before them, the work items)
  pdl_trigger();
  const int lane = threadIdx.x & 31;
  const int64_t n = int64_t(*n_items);
  const int64_t warps = int64_t(gridDim.x) * (kSelectThreads / 32);
  for (int64_t it = (int64_t(blockIdx.x) * kSelectThreads + threadIdx.x) >> 5; it < n; it += warps) {
    const int64_t item = items[it], r = item / n_dense, t = item - r * n_dense;
    const uint32_t* sp = split + r * G.n_words;
    const uint32_t* bw = bandb + r * G.n_words;
    int64_t base = offsets[r] + tile_base[item];
    int64_t wb, we;
    tile_words(G, int32_t(t), &wb, &we);
    for (int64_t w0 = wb; w0 < we; w0 += 128) {
      const int64_t wi = w0 + 4 * lane;
      uint32_t m[4] = {0u, 0u, 0u, 0u};
      if (wi < we) combine_group(sp, bw, G, wi, we - wi < 4 ? int(we - wi) : 4, gated, tf, r, m);
      int total;
      const int ex = warp_exclusive_scan(__popc(m[0]) + __popc(m[1]) + __popc(m[2]) + __popc(m[3]), &total);
      int64_t dst = base + ex;
      // one non-empty word at a time across the warp, lane l its bit l: consecutive set
      // bits go to consecutive entries, so the stores coalesce
#pragma unroll
      for (int c = 0; c < 4; c++) {
        int64_t gb = 0;
        if (m[c]) {
          int d = 0;
          while (G.word_off[d + 1] <= wi + c) d++;
          gb = G.level_off[d] + (wi + c - G.word_off[d]) * 32;
        }
        for (uint32_t nz = __ballot_sync(kFull, m[c] != 0u); nz; nz &= nz - 1) {
          const int src = __ffs(nz) - 1;
          const uint32_t word = __shfl_sync(kFull, m[c], src);
          const int64_t wd = __shfl_sync(kFull, dst, src);
          const int64_t wg = __shfl_sync(kFull, gb, src);
          if ((word >> lane) & 1u) {
            const int64_t e = wd + __popc(word & ((1u << lane) - 1u));
            if (e < cap) {
              idx[e] = int32_t(wg + lane);
              if (wv) wv[e] = __int_as_float(int32_t(r));  // the pair, for select_weights_kernel
            }
          }
        }
        dst += __popc(m[c]);
      }
      base += total;
    }
  }
}

// Kept weights of the selected entries, one entry per thread: the write kernel
// left each entry's pair number in its weight slot (pairs have very unequal
// list lengths, so a warp per pair would leave a few long lists on the tail).
__global__ void __launch_bounds__(kCompactBlock) select_weights_kernel(RecordSource rs, GridDev G,
                                                                       const int64_t* __restrict__ offsets,
                                                                       int64_t n_pairs, int64_t cap,
                                                                       const int32_t* __restrict__ idx,
                                                                       float* __restrict__ wv) {
  pdl_wait();  // the entries and their pairs
  const int64_t total = offsets[n_pairs] < cap ? offsets[n_pairs] : cap;
  for (int64_t e = int64_t(blockIdx.x) * kCompactBlock + threadIdx.x; e < total;
       e += int64_t(gridDim.x) * kCompactBlock) {
    const int64_t r = __float_as_int(wv[e]);
    const int64_t gidx = idx[e];
    int d = 0;
    while (G.level_off[d + 1] <= gidx) d++;
    const uint32_t m = uint32_t(gidx - G.level_off[d]);
    const float scale = __int_as_float((127 - (d + 1)) << 23);  // 2^-(d+1)
    const float x = grid_coord(int(compact1by1(m)), scale), y = grid_coord(int(compact1by1(m >> 1)), scale);
    wv[e] = eval_record_point(rs.spec + r * rs.L.stride, rs.L, x, y);
  }
}

constexpr int kSubtreeMaxDepth = 11;  // aggregates of 4^D cells per pair must stay addressable and modest

// ---- subtree-leaf variance (the ES-HyperNEAT reading of a cell's variance) ----
//
// A depth-e cell's depth-D descendants are a contiguous Morton range of 4^(D-e)
// leaves, so aggregates (mean, M2 = sum of squared deviations) merge level by
// level: four children of n leaves each give mean = average of their means and
// M2 = the sum of their M2 plus n times the squared deviations of their means.
// One launch per level; cell idx of the launch is pair idx >> 2(e+1), Morton
// index idx & (4^(e+1) - 1). The loop over cells is warp-uniform (the split
// words come from ballots).
__global__ void __launch_bounds__(256) subtree_level_kernel(const float* __restrict__ out,
                                                            const float2* __restrict__ child,
                                                            float2* __restrict__ agg, int e, GridDev G,
                                                            int64_t n_pairs, float theta,
                                                            uint32_t* __restrict__ split, float* __restrict__ var_out) {
  const int lane = threadIdx.x & 31;
  const int lg = 2 * (e + 1);                      // log2 of the cells of level e
  const int64_t cells = int64_t(1) << lg, total = n_pairs * cells;
  const float n_child = float(int64_t(1) << (2 * (G.D - e - 1)));  // leaves under each child
  const float n_cell = 4.f * n_child;
  const int64_t stride = int64_t(gridDim.x) * blockDim.x;
  for (int64_t base = int64_t(blockIdx.x) * blockDim.x + (threadIdx.x & ~31); base < total; base += stride) {
    const int64_t idx = base + lane;
    const bool valid = idx < total;
    bool bit = false;
    if (valid) {
      const int64_t r = idx >> lg, m = idx & (cells - 1);
      float c[4], M[4] = {0.f, 0.f, 0.f, 0.f};
      if (e == G.D - 1) {
        const float4 x = *reinterpret_cast<const float4*>(out + r * G.n_total + G.level_off[G.D] + 4 * m);
        c[0] = x.x; c[1] = x.y; c[2] = x.z; c[3] = x.w;
      } else {
#pragma unroll
        for (int k = 0; k < 4; k++) {
          const float2 a = child[4 * idx + k];
          c[k] = a.x;
          M[k] = a.y;
        }
      }
      const float mean = ((c[0] + c[1]) + (c[2] + c[3])) * 0.25f;
      const float d0 = c[0] - mean, d1 = c[1] - mean, d2 = c[2] - mean, d3 = c[3] - mean;
      const float m2 = ((M[0] + M[1]) + (M[2] + M[3])) + n_child * ((d0 * d0 + d1 * d1) + (d2 * d2 + d3 * d3));
      agg[idx] = make_float2(mean, m2);
      bit = m2 > theta * n_cell;
      if (var_out) var_out[r * G.n_total + G.level_off[e] + m] = m2 / n_cell;
    }
    const uint32_t bal = __ballot_sync(0xffffffffu, bit);
    if (valid) {
      const int64_t r = idx >> lg, m = idx & (cells - 1);
      if (cells >= 32) {
        if (lane == 0) split[r * G.n_words + G.word_off[e] + (m >> 5)] = bal;
      } else if (m == 0) {  // 4 or 16 cells: the pair's word holds lanes lane .. lane + cells - 1
        split[r * G.n_words + G.word_off[e]] = (bal >> lane) & uint32_t((int64_t(1) << cells) - 1);
      }
    }
  }
}

// HyperNEAT's weight scaling of list entries: a connection whose output
// magnitude exceeds the threshold is expressed, its magnitude mapped linearly
// from (thr, 1] onto (0, w_max] (magnitudes above 1 clamp to 1); others become 0.
__global__ void __launch_bounds__(kCompactBlock) scale_weights_kernel(float* __restrict__ w,
                                                                      const int64_t* __restrict__ offsets,
                                                                      int64_t n_pairs, int64_t cap, float thr,
                                                                      float w_max) {
  const int64_t total = offsets[n_pairs] < cap ? offsets[n_pairs] : cap;
  for (int64_t e = int64_t(blockIdx.x) * kCompactBlock + threadIdx.x; e < total;
       e += int64_t(gridDim.x) * kCompactBlock) {
    const float v = w[e], a = fabsf(v);
    w[e] = a > thr ? copysignf((fminf(a, 1.0f) - thr) / (1.0f - thr) * w_max, v) : 0.0f;
  }
}

// ---- host helpers ---------------------------------------------------------------

inline emr_status cuda_status(cudaError_t e) { return e == cudaSuccess ? EMR_OK : EMR_ERR_CUDA; }

inline bool grid_ok(const emr_grid* g) { return g && g->D >= 0 && g->D <= EMR_MAX_DEPTH && g->n_total > 0; }

GridDev grid_dev(const emr_grid* g) {
  GridDev G{};
  G.D = g->D;
  G.n_total = g->n_total;
  G.n_halo = g->n_halo;
  G.n_words = g->n_words;
  int64_t qb = 0;
  for (int d = 0; d < EMR_MAX_DEPTH + 2; d++) {  // entries past D + 1 repeat the totals
    const int e = d <= g->D + 1 ? d : g->D + 1;
    G.level_off[d] = g->level_off[e];
    G.halo_off[d] = g->halo_off[e];
    G.word_off[d] = g->word_off[e];
    G.qblk_off[d] = qb;
    if (d <= g->D) qb += ((int64_t(1) << (2 * d)) + 31) / 32;
  }
  G.n_qblocks = G.qblk_off[g->D + 1];
  return G;
}

struct EvalPlan {
  int64_t n_pairs;
  int64_t n_class[kClasses];  // pairs per kernel class (schedule order)
  int64_t n_const;            // pairs whose output is constant over the grid: the last ranks of kClassNone
  SpecLayout L;
  int32_t scratch_stride;
  size_t spec_bytes, scratch_bytes, order_bytes, sched_bytes, total;
};

emr_status eval_plan(const void* pack_host, const emr_query* q, EvalPlan* p) {
  if (!pack_host || !q || q->S <= 0 || !q->a_host || !q->b_host || !q->side_host) return EMR_ERR_ARG;
  const PackHeader* h = pack_header(pack_host);
  if (h->magic != kPackMagic || h->version != kPackVersion || h->P <= 0) return EMR_ERR_ARG;
  const PackGenome* gt =
      reinterpret_cast<const PackGenome*>(static_cast<const uint8_t*>(pack_host) + h->off_genomes);
  bool sides[2] = {false, false};
  const int64_t ns = q->per_genome ? int64_t(h->P) * q->S : q->S;
  for (int64_t k = 0; k < ns; k++) {
    if (q->side_host[k] != EMR_SIDE_OUT && q->side_host[k] != EMR_SIDE_IN) return EMR_ERR_ARG;
    sides[q->side_host[k]] = true;
  }
  int nv = 0, nve = 0;
  for (int s = 0; s < 2; s++)
    if (sides[s]) { nv = std::max(nv, h->max_varying[s]); nve = std::max(nve, h->max_vedges[s]); }
  p->n_pairs = int64_t(h->P) * q->S;
  for (int c = 0; c < kClasses; c++) p->n_class[c] = 0;
  p->n_const = 0;
  for (int g = 0; g < h->P; g++)
    for (int s = 0; s < q->S; s++) {
      int nvar = 0, nj = 0;  // unused slots evaluate to a constant
      if (!(q->per_genome && q->count_host && s >= q->count_host[g])) {
        const int64_t si = q->per_genome ? int64_t(g) * q->S + s : s;
        nvar = gt[g].n_varying[q->side_host[si]];
        nj = gt[g].n_joint[q->side_host[si]];
      }
      p->n_class[pair_class(nvar, nj)]++;
      if (nvar == 0) p->n_const++;
    }
  p->L = spec_layout(nv, nve);
  p->scratch_stride = std::max(h->max_nodes, 1);
  p->spec_bytes = size_t(p->n_pairs) * size_t(p->L.stride);
  p->scratch_bytes = (size_t(p->n_pairs) * size_t(p->scratch_stride) * 4 + 255) & ~size_t(255);
  p->order_bytes = (size_t(p->n_pairs) * 4 + 255) & ~size_t(255);
  p->sched_bytes = (size_t(p->n_pairs) * 4 + 16 + 255) & ~size_t(255);  // pair bins, then the done counter
  p->total = ((p->spec_bytes + 255) & ~size_t(255)) + p->scratch_bytes + p->order_bytes + p->sched_bytes;
  return EMR_OK;
}

QueryDev query_dev(const emr_query* q) {
  QueryDev d;
  d.a = q->a_dev;
  d.b = q->b_dev;
  d.side = q->side_dev;
  d.count = q->count_dev;
  d.S = q->S;
  d.per_genome = q->per_genome;
  return d;
}

void ws_layout(const EvalPlan& p, void* ws, uint8_t** spec, int32_t** order, float** scratch = nullptr) {
  uint8_t* base = static_cast<uint8_t*>(ws);
  *spec = base;
  float* sc = reinterpret_cast<float*>(base + ((p.spec_bytes + 255) & ~size_t(255)));
  *order = reinterpret_cast<int32_t*>(reinterpret_cast<uint8_t*>(sc) + p.scratch_bytes);
  if (scratch) *scratch = sc;
}

// Specialise every pair and order the pairs by cost, into the workspace.
emr_status prepare(const void* pack_dev, const emr_query* q, const EvalPlan& p, void* ws, cudaStream_t st,
                   uint8_t** spec, int32_t** order) {
  float* scratch;
  ws_layout(p, ws, spec, order, &scratch);
  int32_t* bins = reinterpret_cast<int32_t*>(reinterpret_cast<uint8_t*>(*order) + p.order_bytes);
  auto* done = reinterpret_cast<unsigned int*>(bins + p.n_pairs);
  if (cudaMemsetAsync(done, 0, sizeof(unsigned int), st) != cudaSuccess) return EMR_ERR_CUDA;
  const QueryDev qd = query_dev(q);
  const uint8_t* pk = static_cast<const uint8_t*>(pack_dev);
  spec_kernel<<<unsigned((p.n_pairs + kSpecWarps - 1) / kSpecWarps), 32 * kSpecWarps, 0, st>>>(
      pk, qd, p.n_pairs, p.L, *spec, scratch, p.scratch_stride, *order, bins, done);
  return cuda_status(cudaGetLastError());
}

size_t tile_smem_bytes(const SpecLayout& L) {
  return 16 * size_t(L.nv_cap) + 16 * size_t((L.nve_cap + 1) / 2) + 16 * size_t(L.nv_cap) * kBlock +
         4 * size_t(kTileSide + 2) * size_t(kTileSide + 2);
}

int64_t dense_tiles(int D) {
  int64_t t = 1;
  for (int d = kPyramidTop + 1; d <= D; d++) t += tiles_in_level(d);
  return t;
}

constexpr int kDenseTPB = 128;  // threads per dense tile CTA

// Streaming multiprocessors of the current device (queried once per device).
int sm_count() {
  static int cached[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 1;
  if (dev < 64 && cached[dev] > 0) return cached[dev];
  int n = 1;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1) n = 1;
  if (dev < 64) cached[dev] = n;
  return n;
}

// Waves of resident CTAs a dense launch keeps at least, when it groups tiles.
constexpr int kDenseMinWaves = 2;

// A launch that may begin while the previous kernel in the stream drains
// (programmatic dependent launch): for tile launches of other pairs, which
// touch none of the previous launch's outputs. *overlap: whether this launch
// may overlap its predecessor; set for the next one.
template <class... KArgs, class... Args>
cudaError_t launch_overlapped(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                              bool* overlap, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = *overlap ? 1 : 0;
  *overlap = true;
  return cudaLaunchKernelEx(&cfg, kern, args...);
}

// Dense tiles a CTA-wide launch takes in fused mode (tile_kernel_pyramid, or the block kernel
// tile_kernel_dense; the rest run a warp per tile): the depths 0..4 tile, and at depth 5 also
// the grid's one 64 x 64 tile, on the block kernel (a warp launch of one tile per pair would
// leave three of a CTA's four warps idle).
inline int32_t block_tiles(int64_t n_dense) { return n_dense == 2 ? 2 : 1; }

template <int NJMAX>
emr_status launch_dense(const DTileArgs& A0, int64_t rank_beg, int64_t n_ranks, cudaStream_t st, bool* overlap) {
  if (n_ranks <= 0) return EMR_OK;
  DTileArgs A = A0;
  // consecutive tiles of a pair share a CTA (one record load and one prologue for
  // all of them) while the launch still fills every SM kDenseMinWaves times
  const int64_t slots = int64_t(sm_count()) * dense_min_blocks(NJMAX, kDenseTPB);
  int g = 8;
  while (g > 1 && n_ranks * ((A.n_tiles + g - 1) / g) < kDenseMinWaves * slots) g >>= 1;
  A.tiles_per_cta = g;
  const unsigned gx = unsigned((A.n_tiles + g - 1) / g);
  for (int64_t r0 = 0; r0 < n_ranks; r0 += 65535) {  // grid y: ranks, at most 65535 a launch
    A.rank_beg = rank_beg + r0;
    const dim3 grid(gx, unsigned(std::min<int64_t>(65535, n_ranks - r0)));
    const cudaError_t e = launch_overlapped(tile_kernel_dense<NJMAX, kDenseTPB>, grid, dim3(kDenseTPB), 0, st,
                                            overlap, A);
    if (e != cudaSuccess) return cuda_status(e);
  }
  return cuda_status(cudaGetLastError());
}

// Dense tile 0 of n_ranks pairs through tile_kernel_pyramid (fused mode, no output buffer).
template <int NJMAX>
emr_status launch_pyramid(const DTileArgs& A0, int64_t rank_beg, int64_t n_ranks, cudaStream_t st, bool* overlap) {
  if (n_ranks <= 0) return EMR_OK;
  DTileArgs A = A0;
  for (int64_t r0 = 0; r0 < n_ranks; r0 += 65535) {  // grid y: ranks, at most 65535 a launch
    A.rank_beg = rank_beg + r0;
    const dim3 grid(1, unsigned(std::min<int64_t>(65535, n_ranks - r0)));
    const cudaError_t e = launch_overlapped(tile_kernel_pyramid<NJMAX>, grid, dim3(kPyrTPB), 0, st, overlap, A);
    if (e != cudaSuccess) return cuda_status(e);
  }
  return cuda_status(cudaGetLastError());
}

template <int NJMAX>
emr_status launch_warp(const DTileArgs& A0, int64_t rank_beg, int64_t n_ranks, cudaStream_t st, bool* overlap) {
  if (n_ranks <= 0 || A0.n_tiles <= 0) return EMR_OK;
  DTileArgs A = A0;
  // a tile per warp: short CTAs balance best (measured against longer groups); the kernel
  // keeps at most one deferred band test per warp
  const int g = kWarpTiles;
  A.tiles_per_cta = g;
  const unsigned gx = unsigned((A.n_tiles + g - 1) / g);
  for (int64_t r0 = 0; r0 < n_ranks; r0 += 65535) {
    A.rank_beg = rank_beg + r0;
    const dim3 grid(gx, unsigned(std::min<int64_t>(65535, n_ranks - r0)));
    const cudaError_t e =
        launch_overlapped(tile_kernel_warp<NJMAX>, grid, dim3(32 * kWarpTiles), 0, st, overlap, A);
    if (e != cudaSuccess) return cuda_status(e);
  }
  return cuda_status(cudaGetLastError());
}

// A class of pairs with joint nodes, tiles [D.tile_beg, D.tile_beg + D.n_tiles): in fused
// mode without an output buffer the depths 0..4 tile through tile_kernel_dense and the
// 64 x 64 tiles a warp each (launch_tiles itself gives a full range's depths 0..4 tiles to
// one tile_kernel_pyramid launch); otherwise all through tile_kernel_dense.
template <int NJMAX>
emr_status launch_joint_class(const DTileArgs& D, int64_t rank_beg, int64_t n_ranks, cudaStream_t st,
                              bool* overlap, bool warp_tiles) {
  if (n_ranks <= 0) return EMR_OK;
  if (!warp_tiles) return launch_dense<NJMAX>(D, rank_beg, n_ranks, st, overlap);
  emr_status rc;
  const int32_t end = D.tile_beg + D.n_tiles;
  // the block kernel takes the depths 0..4 tile, the warp kernel the 64 x 64 tiles (with a
  // single 64 x 64 tile, D = 5, the block kernel takes it too)
  const int32_t split_at = std::min<int32_t>(end, block_tiles(D.n_dense));
  if (D.tile_beg < split_at) {
    DTileArgs D0 = D;
    D0.n_tiles = split_at - D.tile_beg;
    if ((rc = launch_dense<NJMAX>(D0, rank_beg, n_ranks, st, overlap)) != EMR_OK) return rc;
  }
  if (end <= split_at) return EMR_OK;
  DTileArgs D1 = D;
  D1.tile_beg = std::max<int32_t>(D.tile_beg, split_at);
  D1.n_tiles = end - D1.tile_beg;
  return launch_warp<NJMAX>(D1, rank_beg, n_ranks, st, overlap);
}

emr_status launch_one_axis(const DTileArgs& A0, int64_t rank_beg, int64_t n_ranks, cudaStream_t st, bool* overlap) {
  if (n_ranks <= 0 || A0.n_tiles <= 0) return EMR_OK;
  DTileArgs A = A0;
  const int64_t slots = int64_t(sm_count()) * kOneAxisBlocks;
  int g = 32;  // tiles per CTA, a warp taking every kOneAxisWarps-th
  while (g > kOneAxisWarps && n_ranks * ((A.n_tiles + g - 1) / g) < kDenseMinWaves * slots) g >>= 1;
  A.tiles_per_cta = g;
  const unsigned gx = unsigned((A.n_tiles + g - 1) / g);
  for (int64_t r0 = 0; r0 < n_ranks; r0 += 65535) {
    A.rank_beg = rank_beg + r0;
    const dim3 grid(gx, unsigned(std::min<int64_t>(65535, n_ranks - r0)));
    const cudaError_t e = launch_overlapped(tile_kernel_one_axis, grid, dim3(32 * kOneAxisWarps), 0, st, overlap, A);
    if (e != cudaSuccess) return cuda_status(e);
  }
  return cuda_status(cudaGetLastError());
}

// Tile range (dense numbering: tile 0 = depths 0..4, then the 64 x 64 tiles of
// depths 5..D in global-index order) and output views of one launch set.
struct TileRange {
  int32_t beg = 0, end = -1;  // end < 0: all tiles
  int64_t band_stride = -1, band_shift = 0, out_stride = -1, out_shift = 0;
};

emr_status launch_tiles(const EvalPlan& p, const emr_grid* g, const uint8_t* spec, const int32_t* order, int mode,
                        float theta, float band, float w_min, float* out, float* out_halo, uint32_t* split,
                        uint32_t* bandb, cudaStream_t st, TileRange tr = TileRange(),
                        uint8_t* tile_flags = nullptr, bool after_records = false) {
  // after_records: the record kernel is this stream's last launch and the tile flags are
  // already zeroed, so the first tile launch may overlap it (when that launch waits for it)
  emr_status rc = EMR_OK;
  const int32_t n_dense = int32_t(dense_tiles(g->D));
  if (tile_flags && !after_records &&
      cudaMemsetAsync(tile_flags, 0, size_t(p.n_pairs) * size_t(n_dense), st) != cudaSuccess)
    return EMR_ERR_CUDA;
  if (tr.end < 0) tr.end = n_dense;
  if (tr.band_stride < 0) tr.band_stride = g->n_words;
  if (tr.out_stride < 0) tr.out_stride = g->n_total;
  if (tr.beg < 0 || tr.end > n_dense || tr.beg >= tr.end) return tr.beg == tr.end ? EMR_OK : EMR_ERR_ARG;
  // class 0: interpreter (more than kDenseMax varying nodes); its tiles are one
  // per depth for depths 0..5, then the same 64 x 64 tiles (dense tile t >= 1 is
  // interpreter tile t + 4).
  if (p.n_class[0] > 0) {
    TileArgs A{};
    A.spec = spec;
    A.L = p.L;
    A.order = order;
    A.rank_beg = 0;
    A.D = g->D;
    A.mode = mode;
    A.theta = theta;
    A.band = band;
    A.w_min = w_min;
    int32_t t = 0;
    for (int d = 0; d <= g->D; d++) {
      A.lvl_tile_beg[d] = t;
      t += int32_t(tiles_in_level(d));
    }
    for (int d = g->D + 1; d < EMR_MAX_DEPTH + 2; d++) A.lvl_tile_beg[d] = t;
    const int32_t ib = tr.beg == 0 ? 0 : tr.beg + 4;
    const int32_t ie = tr.end >= n_dense ? t : tr.end + 4;
    A.tile_beg = ib;
    A.n_tiles = ie - ib;
    A.band_stride = tr.band_stride;
    A.band_shift = tr.band_shift;
    A.out_stride = tr.out_stride;
    A.out_shift = tr.out_shift;
    A.n_total = g->n_total;
    A.n_halo = g->n_halo;
    A.n_words = g->n_words;
    for (int d = 0; d < EMR_MAX_DEPTH + 2; d++) {
      A.level_off[d] = g->level_off[d];
      A.halo_off[d] = g->halo_off[d];
      A.word_off[d] = g->word_off[d];
    }
    A.out = out;
    A.out_halo = out_halo;
    A.split = split;
    A.bandb = bandb;
    A.tile_flags = tile_flags;
    A.n_dense = n_dense;
    const int64_t blocks = p.n_class[0] * int64_t(A.n_tiles);
    if (blocks > 0x7fffffffLL) return EMR_ERR_RANGE;
    const size_t smem = tile_smem_bytes(p.L);
    if (smem > 227 * 1024) return EMR_ERR_RANGE;
    cudaError_t e = cudaFuncSetAttribute(tile_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
    if (e != cudaSuccess) return EMR_ERR_CUDA;
    if (blocks > 0) tile_kernel<<<unsigned(blocks), kBlock, smem, st>>>(A);
    if ((rc = cuda_status(cudaGetLastError())) != EMR_OK) return rc;
  }
  DTileArgs D{};
  D.spec = spec;
  D.L = p.L;
  D.order = order;
  D.tile_beg = tr.beg;
  D.n_tiles = tr.end - tr.beg;
  D.band_stride = tr.band_stride;
  D.band_shift = tr.band_shift;
  D.out_stride = tr.out_stride;
  D.out_shift = tr.out_shift;
  D.D = g->D;
  D.mode = mode;
  D.theta = theta;
  D.band = band;
  D.w_min = w_min;
  D.n_total = g->n_total;
  D.n_halo = g->n_halo;
  D.n_words = g->n_words;
  for (int d = 0; d < EMR_MAX_DEPTH + 2; d++) {
    D.level_off[d] = g->level_off[d];
    D.halo_off[d] = g->halo_off[d];
    D.word_off[d] = g->word_off[d];
  }
  D.out = out;
  D.out_halo = out_halo;
  D.split = split;
  D.bandb = bandb;
  D.tile_flags = tile_flags;
  D.n_dense = n_dense;
  // the class launches after the first overlap their predecessor's last wave
  bool overlap = p.n_class[0] > 0;
  const bool warp_tiles = mode == kModeFused && !out;
  // first rank of each joint class (12, 8, 6, 4 joint nodes at most)
  const int64_t b1 = p.n_class[0], b2 = b1 + p.n_class[1], b3 = b2 + p.n_class[2], b4 = b3 + p.n_class[3];
  const int64_t b5 = b4 + p.n_class[4];
  int64_t beg = b5 + p.n_class[5];
  const int32_t bt = block_tiles(n_dense);
  // non-constant one-coordinate pairs: ranks beg .. beg + n_one - 1 (the constant ones follow)
  const int64_t n_one = p.n_class[kClassNone] - p.n_const;
  const bool one_fused = mode == kModeFused && !out && n_one > 0;
  bool one_tile0_done = false;
  if (warp_tiles && D.tile_beg < bt && D.tile_beg + D.n_tiles > bt) {
    // the depths 0..4 tile of every pair in one tile_kernel_pyramid launch (the 12-joint
    // class in one of its own), then every class's warp launch (depths 5..D): the pyramid
    // kernel's latency-bound CTAs share the SMs with the warp launches that follow. The
    // pairs of up to 8 joint nodes and the one-coordinate pairs are consecutive ranks; one
    // launch of the 8-joint kernel for all of them measured faster than a launch per class.
    DTileArgs D0 = D, D1 = D;
    D0.n_tiles = bt - D.tile_beg;
    D1.tile_beg = bt;
    D1.n_tiles = D.tile_beg + D.n_tiles - bt;
    if (after_records && !overlap) {  // the depths 0..4 launches overlap the record kernel
      overlap = true;
      D0.wait_at_start = 1;
    }
    if ((rc = launch_pyramid<12>(D0, b1, p.n_class[1], st, &overlap)) != EMR_OK) return rc;
    if ((rc = launch_pyramid<8>(D0, b2, beg + (one_fused ? n_one : 0) - b2, st, &overlap)) != EMR_OK) return rc;
    one_tile0_done = one_fused;
    if ((rc = launch_warp<12>(D1, b1, p.n_class[1], st, &overlap)) != EMR_OK) return rc;
    if ((rc = launch_warp<8>(D1, b2, p.n_class[2], st, &overlap)) != EMR_OK) return rc;
    if ((rc = launch_warp<6>(D1, b3, p.n_class[3], st, &overlap)) != EMR_OK) return rc;
    if ((rc = launch_warp<4>(D1, b4, p.n_class[4], st, &overlap)) != EMR_OK) return rc;
    if ((rc = launch_warp<2>(D1, b5, p.n_class[5], st, &overlap)) != EMR_OK) return rc;
  } else {
    if ((rc = launch_joint_class<12>(D, b1, p.n_class[1], st, &overlap, warp_tiles)) != EMR_OK) return rc;
    if ((rc = launch_joint_class<8>(D, b2, p.n_class[2], st, &overlap, warp_tiles)) != EMR_OK) return rc;
    if ((rc = launch_joint_class<6>(D, b3, p.n_class[3], st, &overlap, warp_tiles)) != EMR_OK) return rc;
    if (warp_tiles && D.tile_beg + D.n_tiles > bt) {
      if ((rc = launch_joint_class<4>(D, b4, p.n_class[4], st, &overlap, warp_tiles)) != EMR_OK) return rc;
      if ((rc = launch_joint_class<2>(D, b5, p.n_class[5], st, &overlap, warp_tiles)) != EMR_OK) return rc;
    } else {
      // block tiles only: the 1..2-joint pairs (the ranks after the 3..4-joint ones) with them in one
      // launch (a launch of its own pays more than the smaller kernel saves)
      if ((rc = launch_joint_class<4>(D, b4, p.n_class[4] + p.n_class[5], st, &overlap, warp_tiles)) != EMR_OK)
        return rc;
    }
  }
  if (one_fused) {
    // one-coordinate outputs: the depths 0..4 tile through the block kernel (unless the
    // pyramid launch took it), the 64 x 64 tiles (depths 5..D) a warp each
    const int64_t n5 = n_one;
    const int32_t split_at = std::min<int32_t>(tr.end, block_tiles(n_dense));
    if (tr.beg < split_at && !one_tile0_done) {
      DTileArgs D0 = D;
      D0.n_tiles = split_at - tr.beg;
      if ((rc = launch_dense<0>(D0, beg, n5, st, &overlap)) != EMR_OK) return rc;
    }
    const int32_t t1 = std::max<int32_t>(tr.beg, split_at);
    if (t1 < tr.end) {
      DTileArgs D1 = D;
      D1.tile_beg = t1;
      D1.n_tiles = tr.end - t1;
      if ((rc = launch_one_axis(D1, beg, n5, st, &overlap)) != EMR_OK) return rc;
    }
  } else if (mode != kModeFused || p.n_const == 0) {
    return launch_dense<0>(D, beg, p.n_class[kClassNone], st, &overlap);
  } else if ((rc = launch_dense<0>(D, beg, p.n_class[kClassNone] - p.n_const, st, &overlap)) != EMR_OK) {
    return rc;
  }
  if (mode != kModeFused) return EMR_OK;
  // with tile flags, a constant-output pair has none set and its planes are never read: leave them
  if (tile_flags) return EMR_OK;
  const int64_t c0 = beg + p.n_class[kClassNone] - p.n_const;
  for (int64_t r0 = 0; r0 < p.n_const; r0 += 65535) {  // grid y: pairs, at most 65535 a launch
    D.rank_beg = c0 + r0;
    const int64_t nc = std::min<int64_t>(65535, p.n_const - r0);
    const int64_t gx = std::max<int64_t>(1, std::min<int64_t>(D.n_tiles, 64));
    const dim3 grid(static_cast<unsigned>(gx), static_cast<unsigned>(nc));
    zero_tiles_kernel<<<grid, 128, 0, st>>>(D);
  }
  return cuda_status(cudaGetLastError());
}

emr_status launch_combine(const uint32_t* split, PlaneView band, PlaneView mask, const emr_grid* g, int64_t n_pairs,
                          int64_t w0, int64_t nw, int gated, cudaStream_t st, TypeFilter tf, int64_t r0 = 0) {
  if (n_pairs <= 0 || nw <= 0) return EMR_OK;
  if (n_pairs > 65535) {  // grid y limit: split the pairs
    for (int64_t q0 = 0; q0 < n_pairs; q0 += 65535) {
      const int64_t nr = std::min<int64_t>(65535, n_pairs - q0);
      PlaneView b2 = band, m2 = mask;
      b2.p += q0 * band.stride;
      m2.p += q0 * mask.stride;
      emr_status rc = launch_combine(split + q0 * g->n_words, b2, m2, g, nr, w0, nw, gated, st, tf, r0 + q0);
      if (rc != EMR_OK) return rc;
    }
    return EMR_OK;
  }
  const int64_t groups = (nw + 3) / 4;
  dim3 grid(unsigned((groups + 255) / 256), unsigned(n_pairs));
  combine_kernel<<<grid, 256, 0, st>>>(split, band, mask, grid_dev(g), w0, nw, gated, tf, r0);
  return cuda_status(cudaGetLastError());
}

TypeFilter no_type_filter() {
  TypeFilter tf{};
  tf.types = EMR_CONN_ALL;
  return tf;
}

emr_status launch_combine(const uint32_t* split, const uint32_t* bandb, const emr_grid* g, int64_t n_pairs, int gated,
                          uint32_t* mask, cudaStream_t st, TypeFilter tf = no_type_filter()) {
  return launch_combine(split, PlaneView{const_cast<uint32_t*>(bandb), g->n_words, 0},
                        PlaneView{mask, g->n_words, 0}, g, n_pairs, 0, g->n_words, gated, st, tf);
}

constexpr int64_t kCompactWords = 4 * kCompactBlock;  // words per compaction block

size_t compact_ws_bytes(int64_t nw, int64_t n_pairs) {
  const int64_t nb = (nw + kCompactWords - 1) / kCompactWords;
  return size_t(2 * 4 * nb * n_pairs + 256);
}

// Ordered compaction of words [w0, w0 + nw) of every pair.
emr_status launch_compact(PlaneView mask, const float* out, int64_t out_stride, int64_t out_shift, const emr_grid* g,
                          int64_t n_pairs, int64_t w0, int64_t nw, int32_t* idx, float* w, int64_t cap, int64_t* counts,
                          int64_t* offsets, void* ws, cudaStream_t st, RecordSource rs = RecordSource{nullptr, {}}) {
  const int nb = int((nw + kCompactWords - 1) / kCompactWords);
  const int64_t nblk = int64_t(nb) * n_pairs;
  if (n_pairs <= 0 || n_pairs > 0x7fffffffLL) return EMR_ERR_RANGE;
  int32_t* bcount = static_cast<int32_t*>(ws);
  int32_t* boff = bcount + nblk;
  const GridDev G = grid_dev(g);
  for (int64_t r0 = 0; r0 < n_pairs; r0 += 65535) {  // grid y holds at most 65535 pairs
    const dim3 grid(unsigned(nb), unsigned(std::min<int64_t>(65535, n_pairs - r0)));
    compact_count_kernel<<<grid, kCompactBlock, 0, st>>>(mask, G, w0, nw, nb, r0, bcount);
  }
  compact_scan_pair_kernel<<<unsigned(n_pairs), 256, 0, st>>>(bcount, nb, boff, counts);
  compact_scan_pairs_kernel<<<1, 1024, 0, st>>>(counts, n_pairs, offsets);
  for (int64_t r0 = 0; r0 < n_pairs; r0 += 65535) {
    const dim3 grid(unsigned(nb), unsigned(std::min<int64_t>(65535, n_pairs - r0)));
    compact_write_kernel<<<grid, kCompactBlock, 0, st>>>(mask, out, out_stride, out_shift, G, w0, nw, nb, r0, boff,
                                                         offsets, cap, idx, w);
  }
  if (w && !out && rs.spec && cap > 0) {
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) !=
        cudaSuccess)
      return EMR_ERR_CUDA;
    kept_weights_kernel<<<unsigned(8 * sms), kCompactBlock, 0, st>>>(rs, G, offsets, n_pairs, cap, idx, w);
  }
  return cuda_status(cudaGetLastError());
}

}  // namespace

extern "C" {

emr_status emr_eval_workspace_size(const void* pack_host, const emr_query* q, size_t* bytes) {
  if (!bytes) return EMR_ERR_ARG;
  EvalPlan p;
  emr_status rc = eval_plan(pack_host, q, &p);
  if (rc != EMR_OK) return rc;
  *bytes = p.total;
  return EMR_OK;
}

emr_status emr_eval_prepare(const void* pack_host, const void* pack_dev, const emr_query* q, void* ws,
                            size_t ws_bytes, void* stream) {
  if (!pack_dev || !ws || !q || !q->a_dev || !q->b_dev || !q->side_dev) return EMR_ERR_ARG;
  EvalPlan p;
  emr_status rc = eval_plan(pack_host, q, &p);
  if (rc != EMR_OK) return rc;
  if (ws_bytes < p.total) return EMR_ERR_CAPACITY;
  uint8_t* spec;
  int32_t* order;
  return prepare(pack_dev, q, p, ws, static_cast<cudaStream_t>(stream), &spec, &order);
}

emr_status emr_eval(const void* pack_host, const emr_query* q, const emr_grid* grid, float* out, float* out_halo,
                    void* ws, size_t ws_bytes, void* stream) {
  if (!grid_ok(grid) || !out || !ws) return EMR_ERR_ARG;
  EvalPlan p;
  emr_status rc = eval_plan(pack_host, q, &p);
  if (rc != EMR_OK) return rc;
  if (ws_bytes < p.total) return EMR_ERR_CAPACITY;
  uint8_t* spec;
  int32_t* order;
  ws_layout(p, ws, &spec, &order);
  return launch_tiles(p, grid, spec, order, kModeMaterialise, 0.f, 0.f, 0.f, out, out_halo, nullptr, nullptr,
                      static_cast<cudaStream_t>(stream));
}

emr_status emr_mask_combine(const uint32_t* split, const uint32_t* band_bits, const emr_grid* grid, int32_t n_pairs,
                            int32_t mode, uint32_t* mask, void* stream) {
  if (!split || !band_bits || !mask || !grid_ok(grid) || n_pairs <= 0 || (mode != EMR_EAGER && mode != EMR_GATED))
    return EMR_ERR_ARG;
  return launch_combine(split, band_bits, grid, n_pairs, mode == EMR_GATED, mask, static_cast<cudaStream_t>(stream));
}

emr_status emr_mask_combine_types(const uint32_t* split, const uint32_t* band_bits, const emr_query* q,
                                  const emr_grid* grid, int32_t n_pairs, int32_t mode, int32_t types, uint32_t* mask,
                                  void* stream) {
  if (!split || !band_bits || !mask || !grid_ok(grid) || n_pairs <= 0 || (mode != EMR_EAGER && mode != EMR_GATED))
    return EMR_ERR_ARG;
  if (!q || q->S <= 0 || !q->a_dev || !q->b_dev || !q->side_dev || n_pairs % q->S != 0 || types < 0 ||
      types > EMR_CONN_ALL)
    return EMR_ERR_ARG;
  TypeFilter tf;
  tf.types = types;
  tf.q = query_dev(q);
  return launch_combine(split, band_bits, grid, n_pairs, mode == EMR_GATED, mask, static_cast<cudaStream_t>(stream),
                        tf);
}

emr_status emr_subtree_workspace_size(const emr_grid* grid, int32_t n_pairs, size_t* bytes) {
  if (!grid_ok(grid) || n_pairs <= 0 || !bytes) return EMR_ERR_ARG;
  if (grid->D > kSubtreeMaxDepth) return EMR_ERR_RANGE;
  const size_t a = size_t(1) << (2 * grid->D), b = grid->D >= 1 ? a / 4 : 1;
  *bytes = size_t(n_pairs) * (a + b) * 8 + 512;
  return EMR_OK;
}

emr_status emr_subtree_split(const float* out, const emr_grid* grid, int32_t n_pairs, float theta, uint32_t* split,
                             float* var_out, void* ws, size_t ws_bytes, void* stream) {
  size_t need = 0;
  emr_status rc = emr_subtree_workspace_size(grid, n_pairs, &need);
  if (rc != EMR_OK) return rc;
  if (!out || !split || !ws || !(theta >= 0.f)) return EMR_ERR_ARG;
  if (ws_bytes < need) return EMR_ERR_CAPACITY;
  if (grid->D == 0) return EMR_OK;  // a single level: every position is a leaf
  const size_t a = size_t(1) << (2 * grid->D);
  float2* buf[2] = {static_cast<float2*>(ws),
                    reinterpret_cast<float2*>(static_cast<uint8_t*>(ws) + ((size_t(n_pairs) * a * 8 + 255) & ~size_t(255)))};
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return EMR_ERR_CUDA;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const GridDev G = grid_dev(grid);
  for (int e = grid->D - 1, k = 0; e >= 0; e--, k ^= 1) {
    const int64_t total = int64_t(n_pairs) << (2 * (e + 1));
    const int64_t blocks = std::min<int64_t>((total + 255) / 256, int64_t(16) * sms);
    subtree_level_kernel<<<unsigned(blocks), 256, 0, st>>>(out, buf[k ^ 1], buf[k], e, G, n_pairs, theta, split,
                                                           var_out);
  }
  return cuda_status(cudaGetLastError());
}

emr_status emr_scale_weights(float* w, const int64_t* offsets, int32_t n_pairs, int64_t cap, float w_thr,
                             float w_max, void* stream) {
  if (!offsets || n_pairs <= 0 || cap < 0 || (cap > 0 && !w) || !(w_thr >= 0.f && w_thr < 1.f) || !(w_max > 0.f))
    return EMR_ERR_ARG;
  if (cap == 0) return EMR_OK;
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return EMR_ERR_CUDA;
  scale_weights_kernel<<<unsigned(8 * sms), kCompactBlock, 0, static_cast<cudaStream_t>(stream)>>>(
      w, offsets, n_pairs, cap, w_thr, w_max);
  return cuda_status(cudaGetLastError());
}

emr_status emr_conn_types(const int32_t* idx, const int64_t* offsets, const emr_query* q, const emr_grid* grid,
                          int32_t n_pairs, int64_t cap, uint8_t* type, void* stream) {
  if (!offsets || !grid_ok(grid) || n_pairs <= 0 || cap < 0 || (cap > 0 && (!idx || !type))) return EMR_ERR_ARG;
  if (!q || q->S <= 0 || !q->a_dev || !q->b_dev || !q->side_dev || n_pairs % q->S != 0) return EMR_ERR_ARG;
  if (cap == 0) return EMR_OK;
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return EMR_ERR_CUDA;
  conn_types_kernel<<<unsigned(8 * sms), kCompactBlock, 0, static_cast<cudaStream_t>(stream)>>>(
      query_dev(q), grid_dev(grid), offsets, n_pairs, cap, idx, type);
  return cuda_status(cudaGetLastError());
}

emr_status emr_substrate_config(int32_t config, int32_t* types, int32_t* hidden_rounds) {
  static const int32_t kTypes[6] = {EMR_CONN_F, EMR_CONN_F, EMR_CONN_F | EMR_CONN_B, EMR_CONN_F | EMR_CONN_L,
                                    EMR_CONN_F | EMR_CONN_S, EMR_CONN_ALL};
  if (config < EMR_SUBSTRATE_FEEDFORWARD || config > EMR_SUBSTRATE_FULL) return EMR_ERR_ARG;
  if (types) *types = kTypes[config];
  if (hidden_rounds) *hidden_rounds = config == EMR_SUBSTRATE_FEEDFORWARD ? 0 : 1;
  return EMR_OK;
}

emr_status emr_variance_filter(const float* out, const float* out_halo, const emr_grid* grid, int32_t P, int32_t S,
                               float theta, float band, float w_min, int32_t mode, uint32_t* mask, uint32_t* split,
                               uint32_t* band_bits, float* var_dbg, void* stream) {
  if (!out || !out_halo || !grid_ok(grid) || P <= 0 || S <= 0 || !mask || !split || !band_bits) return EMR_ERR_ARG;
  if (!(theta >= 0.f) || !(band >= 0.f) || !(w_min >= 0.f) || (mode != EMR_EAGER && mode != EMR_GATED))
    return EMR_ERR_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int64_t n_pairs = int64_t(P) * S;
  const GridDev G = grid_dev(grid);
  const int64_t threads = n_pairs * G.n_qblocks * 32;
  if ((threads + 255) / 256 > 0x7fffffffLL) return EMR_ERR_RANGE;
  planes_kernel<<<unsigned((threads + 255) / 256), 256, 0, st>>>(out, out_halo, G, n_pairs, theta, band, w_min, split,
                                                                 band_bits, var_dbg);
  emr_status rc = cuda_status(cudaGetLastError());
  if (rc != EMR_OK) return rc;
  return launch_combine(split, band_bits, grid, n_pairs, mode == EMR_GATED, mask, st);
}

emr_status emr_eval_filter(const void* pack_host, const emr_query* q, const emr_grid* grid, float theta, float band,
                           float w_min, uint32_t* split, uint32_t* band_bits, float* out, void* ws, size_t ws_bytes,
                           void* stream) {
  if (!grid_ok(grid) || !split || !band_bits || !ws) return EMR_ERR_ARG;
  if (!(theta >= 0.f) || !(band >= 0.f) || !(w_min >= 0.f)) return EMR_ERR_ARG;
  EvalPlan p;
  emr_status rc = eval_plan(pack_host, q, &p);
  if (rc != EMR_OK) return rc;
  if (ws_bytes < p.total) return EMR_ERR_CAPACITY;
  uint8_t* spec;
  int32_t* order;
  ws_layout(p, ws, &spec, &order);
  return launch_tiles(p, grid, spec, order, kModeFused, theta, band, w_min, out, nullptr, split, band_bits,
                      static_cast<cudaStream_t>(stream));
}

emr_status emr_compact_workspace_size(const emr_grid* grid, int32_t n_pairs, size_t* bytes) {
  if (!grid_ok(grid) || n_pairs <= 0 || !bytes) return EMR_ERR_ARG;
  *bytes = compact_ws_bytes(grid->n_words, n_pairs);
  return EMR_OK;
}

emr_status emr_compact_records(const uint32_t* mask, const void* pack_host, const emr_query* q, const void* eval_ws,
                               size_t eval_ws_bytes, const emr_grid* grid, int32_t* idx, float* w, int64_t cap,
                               int64_t* counts, int64_t* offsets, void* ws, size_t ws_bytes, void* stream) {
  if (!mask || !grid_ok(grid) || (!idx && cap > 0) || cap < 0 || !counts || !offsets || !ws || !eval_ws)
    return EMR_ERR_ARG;
  EvalPlan p;
  emr_status rc = eval_plan(pack_host, q, &p);
  if (rc != EMR_OK) return rc;
  if (eval_ws_bytes < p.total || ws_bytes < compact_ws_bytes(grid->n_words, p.n_pairs)) return EMR_ERR_CAPACITY;
  return launch_compact(PlaneView{const_cast<uint32_t*>(mask), grid->n_words, 0}, nullptr, 0, 0, grid, p.n_pairs, 0,
                        grid->n_words, idx, w, cap, counts, offsets, ws, static_cast<cudaStream_t>(stream),
                        RecordSource{static_cast<const uint8_t*>(eval_ws), p.L});
}

emr_status emr_eval_filter_tiles(const void* pack_host, const emr_query* q, const emr_grid* grid, float theta,
                                 float band, float w_min, uint32_t* split, uint32_t* band_bits, uint8_t* tile_flags,
                                 void* ws, size_t ws_bytes, void* stream) {
  if (!grid_ok(grid) || !split || !band_bits || !tile_flags || !ws) return EMR_ERR_ARG;
  if (!(theta >= 0.f) || !(band >= 0.f) || !(w_min >= 0.f)) return EMR_ERR_ARG;
  EvalPlan p;
  emr_status rc = eval_plan(pack_host, q, &p);
  if (rc != EMR_OK) return rc;
  if (ws_bytes < p.total) return EMR_ERR_CAPACITY;
  uint8_t* spec;
  int32_t* order;
  ws_layout(p, ws, &spec, &order);
  return launch_tiles(p, grid, spec, order, kModeFused, theta, band, w_min, nullptr, nullptr, split, band_bits,
                      static_cast<cudaStream_t>(stream), TileRange(), tile_flags);
}

static size_t select_ws_bytes(int64_t n_pairs, int64_t n_dense) {
  return 256 + ((size_t(n_pairs) * size_t(n_dense) * 4 + 255) & ~size_t(255)) + size_t(n_pairs) * size_t(n_dense) * 8;
}

emr_status emr_select_workspace_size(const emr_grid* grid, int32_t n_pairs, size_t* bytes) {
  if (!grid_ok(grid) || n_pairs <= 0 || !bytes) return EMR_ERR_ARG;
  *bytes = select_ws_bytes(n_pairs, dense_tiles(grid->D));
  return EMR_OK;
}

static emr_status select_launch(const EvalPlan& p, const uint32_t* split, const uint32_t* band_bits,
                                const uint8_t* tile_flags, const emr_query* q, const void* eval_ws,
                                const emr_grid* grid, int32_t mode, int32_t types, int32_t* idx, float* w, int64_t cap,
                                int64_t* counts, int64_t* offsets, void* ws, cudaStream_t st,
                                bool items_zeroed = false);

emr_status emr_select(const uint32_t* split, const uint32_t* band_bits, const uint8_t* tile_flags,
                      const void* pack_host, const emr_query* q, const void* eval_ws, size_t eval_ws_bytes,
                      const emr_grid* grid, int32_t mode, int32_t types, int32_t* idx, float* w, int64_t cap,
                      int64_t* counts, int64_t* offsets, void* ws, size_t ws_bytes, void* stream) {
  if (!split || !band_bits || !tile_flags || !eval_ws || !grid_ok(grid) || (!idx && cap > 0) || cap < 0 ||
      !counts || !offsets || !ws || (mode != EMR_EAGER && mode != EMR_GATED) || types < 0 || types > EMR_CONN_ALL)
    return EMR_ERR_ARG;
  EvalPlan p;
  emr_status rc = eval_plan(pack_host, q, &p);
  if (rc != EMR_OK) return rc;
  if (eval_ws_bytes < p.total) return EMR_ERR_CAPACITY;
  if (p.n_pairs <= 0 || p.n_pairs > 0x7fffffffLL) return EMR_ERR_RANGE;
  if (ws_bytes < select_ws_bytes(p.n_pairs, dense_tiles(grid->D))) return EMR_ERR_CAPACITY;
  return select_launch(p, split, band_bits, tile_flags, q, eval_ws, grid, mode, types, idx, w, cap, counts, offsets,
                       ws, static_cast<cudaStream_t>(stream));
}

// Planes, tile flags and selection workspace of emr_discover after the records.
struct DiscoverLayout {
  size_t split, band, flags, sel, total;
};

static DiscoverLayout discover_layout(const EvalPlan& p, const emr_grid* g) {
  auto up = [](size_t x) { return (x + 255) & ~size_t(255); };
  DiscoverLayout L;
  const size_t plane = size_t(p.n_pairs) * size_t(g->n_words) * 4;
  const int64_t n_dense = dense_tiles(g->D);
  L.split = up(p.total);
  L.band = L.split + up(plane);
  L.flags = L.band + up(plane);
  L.sel = L.flags + up(size_t(p.n_pairs) * size_t(n_dense));
  L.total = L.sel + up(select_ws_bytes(p.n_pairs, n_dense));
  return L;
}

emr_status emr_discover_workspace_size(const void* pack_host, const emr_query* q, const emr_grid* grid,
                                       size_t* bytes) {
  if (!bytes || !grid_ok(grid)) return EMR_ERR_ARG;
  EvalPlan p;
  emr_status rc = eval_plan(pack_host, q, &p);
  if (rc != EMR_OK) return rc;
  *bytes = discover_layout(p, grid).total;
  return EMR_OK;
}

emr_status emr_copy_async(void* dst, const void* src, size_t bytes, void* stream) {
  if (bytes == 0) return EMR_OK;
  if (!dst || !src) return EMR_ERR_ARG;
  return cuda_status(cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDefault, static_cast<cudaStream_t>(stream)));
}

emr_status emr_discover(const void* pack_host, const void* pack_dev, const emr_query* q, const emr_grid* grid,
                        float theta, float band, float w_min, int32_t mode, int32_t types, void* ws, size_t ws_bytes,
                        int32_t* idx, float* w, int64_t cap, int64_t* counts, int64_t* offsets, void* stream) {
  if (!pack_dev || !ws || !grid_ok(grid) || (!idx && cap > 0) || cap < 0 || !counts || !offsets ||
      (mode != EMR_EAGER && mode != EMR_GATED) || types < 0 || types > EMR_CONN_ALL)
    return EMR_ERR_ARG;
  if (!(theta >= 0.f) || !(band >= 0.f) || !(w_min >= 0.f)) return EMR_ERR_ARG;
  EvalPlan p;
  emr_status rc = eval_plan(pack_host, q, &p);
  if (rc != EMR_OK) return rc;
  if (p.n_pairs <= 0 || p.n_pairs > 0x7fffffffLL) return EMR_ERR_RANGE;
  const DiscoverLayout L = discover_layout(p, grid);
  if (ws_bytes < L.total) return EMR_ERR_CAPACITY;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  uint8_t* base = static_cast<uint8_t*>(ws);
  uint8_t* spec;
  int32_t* order;
  uint8_t* flags = base + L.flags;
  // the selection's work-item counter and the tile flags, zeroed ahead: the first tile launch
  // may then overlap the record kernel and the selection's first kernel the tile launches
  // (adjacent in the workspace: one memset)
  if (cudaMemsetAsync(flags, 0, L.sel - L.flags + sizeof(unsigned long long), st) != cudaSuccess)
    return EMR_ERR_CUDA;
  if ((rc = prepare(pack_dev, q, p, ws, st, &spec, &order)) != EMR_OK) return rc;
  auto* split = reinterpret_cast<uint32_t*>(base + L.split);
  auto* bandb = reinterpret_cast<uint32_t*>(base + L.band);
  if ((rc = launch_tiles(p, grid, spec, order, kModeFused, theta, band, w_min, nullptr, nullptr, split, bandb, st,
                         TileRange(), flags, true)) != EMR_OK)
    return rc;
  return select_launch(p, split, bandb, flags, q, ws, grid, mode, types, idx, w, cap, counts, offsets,
                       base + L.sel, st, true);
}

// Selection over the flagged tiles: count, scan, write, kept weights. Each kernel
// overlaps its predecessor's end and waits for its results before reading them.
// items_zeroed: the work-item counter was zeroed earlier in the stream (then the
// count kernel may overlap the tile launches too).
static emr_status select_launch(const EvalPlan& p, const uint32_t* split, const uint32_t* band_bits,
                                const uint8_t* tile_flags, const emr_query* q, const void* eval_ws,
                                const emr_grid* grid, int32_t mode, int32_t types, int32_t* idx, float* w, int64_t cap,
                                int64_t* counts, int64_t* offsets, void* ws, cudaStream_t st,
                                bool items_zeroed) {
  const int64_t n_dense = dense_tiles(grid->D);
  TypeFilter tf = no_type_filter();
  if (types != EMR_CONN_ALL) {
    tf.types = types;
    tf.q = query_dev(q);
  }
  const GridDev G = grid_dev(grid);
  auto* n_items = static_cast<unsigned long long*>(ws);
  auto* tile_base = reinterpret_cast<int32_t*>(static_cast<uint8_t*>(ws) + 256);
  auto* items = reinterpret_cast<int64_t*>(static_cast<uint8_t*>(ws) + 256 +
                                           ((size_t(p.n_pairs) * size_t(n_dense) * 4 + 255) & ~size_t(255)));
  const int sms = sm_count();
  if (!items_zeroed && cudaMemsetAsync(n_items, 0, sizeof(unsigned long long), st) != cudaSuccess)
    return EMR_ERR_CUDA;
  bool overlap = items_zeroed;
  const unsigned blocks = unsigned((p.n_pairs + kSelectThreads / 32 - 1) / (kSelectThreads / 32));
  cudaError_t e = launch_overlapped(select_count_kernel, dim3(blocks), dim3(kSelectThreads), 0, st, &overlap, split,
                                    band_bits, tile_flags, n_dense, G, int(mode == EMR_GATED), tf, p.n_pairs, counts,
                                    tile_base, items, n_items);
  if (e == cudaSuccess)
    e = launch_overlapped(compact_scan_pairs_kernel, dim3(1), dim3(1024), 0, st, &overlap,
                          static_cast<const int64_t*>(counts), p.n_pairs, offsets);
  if (e == cudaSuccess)
    e = launch_overlapped(select_write_kernel, dim3(unsigned(16 * sms)), dim3(kSelectThreads), 0, st, &overlap, split,
                          band_bits, n_dense, G, int(mode == EMR_GATED), tf, static_cast<const int32_t*>(tile_base),
                          static_cast<const int64_t*>(items), static_cast<const unsigned long long*>(n_items),
                          static_cast<const int64_t*>(offsets), cap, idx, w);
  if (e == cudaSuccess && w && cap > 0)
    e = launch_overlapped(select_weights_kernel, dim3(unsigned(8 * sms)), dim3(kCompactBlock), 0, st, &overlap,
                          RecordSource{static_cast<const uint8_t*>(eval_ws), p.L}, G,
                          static_cast<const int64_t*>(offsets), p.n_pairs, cap, static_cast<const int32_t*>(idx), w);
  return cuda_status(e != cudaSuccess ? e : cudaGetLastError());
}

emr_status emr_compact(const uint32_t* mask, const float* out, const emr_grid* grid, int32_t n_pairs, int32_t* idx,
                       float* w, int64_t cap, int64_t* counts, int64_t* offsets, void* ws, size_t ws_bytes,
                       void* stream) {
  if (!mask || !grid_ok(grid) || n_pairs <= 0 || (!idx && cap > 0) || cap < 0 || !counts || !offsets || !ws ||
      (w && !out))
    return EMR_ERR_ARG;
  if (ws_bytes < compact_ws_bytes(grid->n_words, n_pairs)) return EMR_ERR_CAPACITY;
  return launch_compact(PlaneView{const_cast<uint32_t*>(mask), grid->n_words, 0}, out, grid->n_total, 0, grid,
                        n_pairs, 0, grid->n_words, idx, w, cap, counts, offsets, ws, static_cast<cudaStream_t>(stream));
}

}  // extern "C"

// ---- fused evaluation without caller-provided workspace ----------------------------
//
// Some callers cannot call cudaMalloc: a plugin inside a host application that
// owns every byte of device memory, or a latency-critical loop that must not
// take the implicit device synchronisation an allocation brings. For them,
// emr_eval_filter_noalloc keeps its scratch (the per-pair CPPN records, their
// scratch and the pair schedule) in the library's own static device array
// below. Each GPU that loads libemr holds this array until the process exits.

#include <mutex>

namespace {

constexpr size_t kStaticScratchBytes = size_t(16) << 20;  // 16 MiB per device
constexpr int kMaxDevices = 64;

static __device__ __align__(256) uint8_t g_static_scratch[kStaticScratchBytes];

std::mutex g_static_scratch_mu;
void* g_static_scratch_dev[kMaxDevices] = {};

// Device address of g_static_scratch on the current device. The first call on
// a device looks it up (cudaGetSymbolAddress, with that device current); later
// calls reuse the cached address. In host code the symbol itself is only a
// host-side stand-in and must never be handed to a kernel.
emr_status static_scratch_address(void** ptr) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return EMR_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return EMR_ERR_RANGE;
  std::lock_guard<std::mutex> lock(g_static_scratch_mu);
  if (!g_static_scratch_dev[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_static_scratch) != cudaSuccess || !p) return EMR_ERR_CUDA;
    g_static_scratch_dev[dev] = p;
  }
  *ptr = g_static_scratch_dev[dev];
  return EMR_OK;
}

}  // namespace

extern "C" emr_status emr_eval_filter_noalloc(const void* pack_host, const void* pack_dev, const emr_query* q,
                                              const emr_grid* grid, float theta, float band, float w_min,
                                              uint32_t* split, uint32_t* band_bits, float* out, void* stream) {
  if (!pack_dev || !grid_ok(grid) || !split || !band_bits || !q || !q->a_dev || !q->b_dev || !q->side_dev)
    return EMR_ERR_ARG;
  if (!(theta >= 0.f) || !(band >= 0.f) || !(w_min >= 0.f)) return EMR_ERR_ARG;
  EvalPlan p;
  emr_status rc = eval_plan(pack_host, q, &p);
  if (rc != EMR_OK) return rc;
  if (p.total > kStaticScratchBytes) return EMR_ERR_RANGE;  // population x slots too large for the static area
  void* ws = nullptr;
  if ((rc = static_scratch_address(&ws)) != EMR_OK) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  uint8_t* spec;
  int32_t* order;
  if ((rc = prepare(pack_dev, q, p, ws, st, &spec, &order)) != EMR_OK) return rc;
  return launch_tiles(p, grid, spec, order, kModeFused, theta, band, w_min, out, nullptr, split, band_bits, st);
}

// ---- a7: chunked streaming ------------------------------------------------------------
//
// The grid is cut into chunks of whole tiles (dense numbering) and processed
// from the highest global index down. A chunk's positions at depth d have
// their children at depth d + 1 in the same or an earlier chunk, so when a
// chunk has been evaluated its own split bits are final and its keep mask and
// compacted lists can be produced at once. Only the split plane is resident;
// band bits, masks and lists are per chunk, double-buffered (kept weights are
// recomputed from the per-pair records), and the lists are copied to the
// caller's host arrays on a second stream while the next chunk computes.

#include <chrono>
#include <thread>

namespace {

struct StreamPlan {
  EvalPlan ev;
  std::vector<std::pair<int32_t, int32_t>> chunks;  // tile ranges, processing order
  int64_t wpc, ppc;                                 // words / positions per chunk buffer row
  int64_t n_pairs, chunk_cap;
  size_t off_split, off_band[2], off_mask[2], off_cws[2], off_idx[2], off_w[2], off_cnt[2], off_off[2];
  size_t cws_bytes, total;
};

inline int64_t tile_pos(const emr_grid* g, int32_t t, int32_t n_dense) {
  if (t >= n_dense) return g->n_total;
  return t == 0 ? 0 : g->level_off[kPyramidTop + 1] + int64_t(t - 1) * kTileSide * kTileSide;
}
inline int64_t tile_word(const emr_grid* g, int32_t t, int32_t n_dense) {
  if (t >= n_dense) return g->n_words;
  return t == 0 ? 0 : g->word_off[kPyramidTop + 1] + int64_t(t - 1) * (kTileSide * kTileSide / 32);
}

// The grid's chunks as dense tile ranges, from the highest global index down:
// grid->chunk positions each (whole 64 x 64 tiles; 0 = one chunk), the tile of
// depths 0..4 joining the lowest chunk.
std::vector<std::pair<int32_t, int32_t>> grid_chunks(const emr_grid* g) {
  const int32_t n_dense = int32_t(dense_tiles(g->D));
  const int64_t tile_positions = int64_t(kTileSide) * kTileSide;
  const int32_t tpc = g->chunk > 0 ? int32_t(std::max<int64_t>(1, g->chunk / tile_positions)) : n_dense;
  std::vector<std::pair<int32_t, int32_t>> chunks;
  for (int32_t hi = n_dense; hi > 0;) {
    int32_t lo = std::max(hi - tpc, 1);
    if (lo == 1) lo = 0;  // the tile of depths 0..4 joins the last chunk
    chunks.push_back({lo, hi});
    hi = lo;
  }
  return chunks;
}

emr_status stream_plan(const void* pack_host, const emr_query* q, const emr_grid* g, int64_t chunk_cap,
                       StreamPlan* sp) {
  if (!grid_ok(g) || chunk_cap <= 0) return EMR_ERR_ARG;
  emr_status rc = eval_plan(pack_host, q, &sp->ev);
  if (rc != EMR_OK) return rc;
  const int32_t n_dense = int32_t(dense_tiles(g->D));
  sp->chunks = grid_chunks(g);
  sp->wpc = sp->ppc = 0;
  for (auto& c : sp->chunks) {
    sp->wpc = std::max(sp->wpc, tile_word(g, c.second, n_dense) - tile_word(g, c.first, n_dense));
    sp->ppc = std::max(sp->ppc, tile_pos(g, c.second, n_dense) - tile_pos(g, c.first, n_dense));
  }
  sp->wpc = (sp->wpc + 3) & ~int64_t(3);
  sp->ppc = (sp->ppc + 3) & ~int64_t(3);
  sp->n_pairs = sp->ev.n_pairs;
  sp->chunk_cap = chunk_cap;
  auto up = [](size_t x) { return (x + 255) & ~size_t(255); };
  size_t o = up(sp->ev.total);
  sp->off_split = o;
  o += up(size_t(sp->n_pairs) * size_t(g->n_words) * 4);
  sp->cws_bytes = compact_ws_bytes(sp->wpc, sp->n_pairs);
  for (int b = 0; b < 2; b++) {
    sp->off_band[b] = o; o += up(size_t(sp->n_pairs) * size_t(sp->wpc) * 4);
    sp->off_mask[b] = o; o += up(size_t(sp->n_pairs) * size_t(sp->wpc) * 4);
    sp->off_cws[b] = o; o += up(sp->cws_bytes);
    sp->off_idx[b] = o; o += up(size_t(chunk_cap) * 4);
    sp->off_w[b] = o; o += up(size_t(chunk_cap) * 4);
    sp->off_cnt[b] = o; o += up(size_t(sp->n_pairs) * 8);
    sp->off_off[b] = o; o += up(size_t(sp->n_pairs + 1) * 8);
  }
  sp->total = o;
  return EMR_OK;
}

}  // namespace

extern "C" emr_status emr_grid_chunk(const emr_grid* grid, int64_t chunk_idx, int64_t* n_chunks, int64_t* pos_beg,
                                     int64_t* pos_end) {
  if (!grid_ok(grid)) return EMR_ERR_ARG;
  if (grid->chunk < 0 || (grid->chunk > 0 && grid->chunk % (int64_t(kTileSide) * kTileSide) != 0))
    return EMR_ERR_ARG;
  const auto chunks = grid_chunks(grid);
  const int64_t n = int64_t(chunks.size());
  if (n_chunks) *n_chunks = n;
  if (!pos_beg && !pos_end) return EMR_OK;
  if (chunk_idx < 0 || chunk_idx >= n) return EMR_ERR_RANGE;
  const auto& c = chunks[size_t(n - 1 - chunk_idx)];  // ascending global index
  const int32_t n_dense = int32_t(dense_tiles(grid->D));
  if (pos_beg) *pos_beg = tile_pos(grid, c.first, n_dense);
  if (pos_end) *pos_end = tile_pos(grid, c.second, n_dense);
  return EMR_OK;
}

extern "C" emr_status emr_eval_chunk(const void* pack_host, const emr_query* q, const emr_grid* grid,
                                     int64_t chunk_idx, float* out, float* out_halo, void* ws, size_t ws_bytes,
                                     void* stream) {
  if (!grid_ok(grid) || !out || !ws) return EMR_ERR_ARG;
  int64_t n_chunks = 0, p_lo = 0, p_hi = 0;
  emr_status rc = emr_grid_chunk(grid, chunk_idx, &n_chunks, &p_lo, &p_hi);
  if (rc != EMR_OK) return rc;
  EvalPlan p;
  if ((rc = eval_plan(pack_host, q, &p)) != EMR_OK) return rc;
  if (ws_bytes < p.total) return EMR_ERR_CAPACITY;
  uint8_t* spec;
  int32_t* order;
  ws_layout(p, ws, &spec, &order);
  const auto chunks = grid_chunks(grid);
  const auto& c = chunks[size_t(n_chunks - 1 - chunk_idx)];
  TileRange tr;
  tr.beg = c.first;
  tr.end = c.second;
  tr.out_stride = p_hi - p_lo;
  tr.out_shift = p_lo;
  return launch_tiles(p, grid, spec, order, kModeMaterialise, 0.f, 0.f, 0.f, out, out_halo, nullptr, nullptr,
                      static_cast<cudaStream_t>(stream), tr);
}

namespace {

// Wait for an event with a host-side deadline (timeout_ms <= 0: no limit).
emr_status wait_event(cudaEvent_t ev, std::chrono::steady_clock::time_point deadline, bool limited) {
  for (;;) {
    const cudaError_t e = cudaEventQuery(ev);
    if (e == cudaSuccess) return EMR_OK;
    if (e != cudaErrorNotReady) return EMR_ERR_CUDA;
    if (limited && std::chrono::steady_clock::now() > deadline) return EMR_ERR_TIMEOUT;
    std::this_thread::sleep_for(std::chrono::microseconds(20));
  }
}

}  // namespace

extern "C" emr_status emr_stream_workspace_size(const void* pack_host, const emr_query* q, const emr_grid* grid,
                                                int64_t chunk_cap, size_t* bytes) {
  if (!bytes) return EMR_ERR_ARG;
  StreamPlan sp;
  emr_status rc = stream_plan(pack_host, q, grid, chunk_cap, &sp);
  if (rc != EMR_OK) return rc;
  *bytes = sp.total;
  return EMR_OK;
}

extern "C" emr_status emr_stream_mode(const void* pack_host, const void* pack_dev, const emr_query* q,
                                      const emr_grid* grid, float theta, float band, float w_min, int32_t mode,
                                      int32_t types, void* ws, size_t ws_bytes, int64_t chunk_cap, int32_t* h_idx,
                                      float* h_w, int64_t cap, int64_t* counts, int64_t* offsets, int64_t timeout_ms,
                                      void* stream) {
  if (!pack_dev || !ws || !counts || !offsets || cap < 0 || (cap > 0 && (!h_idx || !h_w)) || timeout_ms < 0)
    return EMR_ERR_ARG;
  if (!(theta >= 0.f) || !(band >= 0.f) || !(w_min >= 0.f)) return EMR_ERR_ARG;
  if ((mode != EMR_EAGER && mode != EMR_GATED) || types < 0 || types > EMR_CONN_ALL || !q) return EMR_ERR_ARG;
  TypeFilter tf;
  tf.types = types;
  tf.q = query_dev(q);
  StreamPlan sp;
  emr_status rc = stream_plan(pack_host, q, grid, chunk_cap, &sp);
  if (rc != EMR_OK) return rc;
  if (ws_bytes < sp.total) return EMR_ERR_CAPACITY;
  const auto deadline = std::chrono::steady_clock::now() + std::chrono::milliseconds(timeout_ms);
  const bool limited = timeout_ms > 0;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  uint8_t* base = static_cast<uint8_t*>(ws);
  uint8_t* spec;
  int32_t* order;
  if ((rc = prepare(pack_dev, q, sp.ev, ws, st, &spec, &order)) != EMR_OK) return rc;
  uint32_t* split = reinterpret_cast<uint32_t*>(base + sp.off_split);
  const int32_t n_dense = int32_t(dense_tiles(grid->D));
  const int64_t NP = sp.n_pairs;

  cudaStream_t cp = nullptr;
  cudaEvent_t ev_done[2] = {nullptr, nullptr}, ev_copied[2] = {nullptr, nullptr};
  int64_t* staging = nullptr;  // pinned: 2 x (n_pairs + 1) chunk offsets
  bool ok = cudaStreamCreateWithFlags(&cp, cudaStreamNonBlocking) == cudaSuccess &&
            cudaHostAlloc(reinterpret_cast<void**>(&staging), size_t(2 * (NP + 1)) * 8, cudaHostAllocDefault) ==
                cudaSuccess;
  for (int b = 0; b < 2 && ok; b++)
    ok = cudaEventCreateWithFlags(&ev_done[b], cudaEventDisableTiming) == cudaSuccess &&
         cudaEventCreateWithFlags(&ev_copied[b], cudaEventDisableTiming) == cudaSuccess;
  struct ChunkOut { int64_t at; std::vector<int64_t> off; };  // host position of its lists, per-pair offsets
  std::vector<ChunkOut> outs(sp.chunks.size());
  for (int64_t r = 0; r < NP; r++) counts[r] = 0;
  int64_t cursor = 0;
  bool overflow = false;
  rc = ok ? EMR_OK : EMR_ERR_CUDA;

  // Collect chunk k's lists: wait for its offsets, then copy its entries to the host arrays.
  auto collect = [&](size_t k) -> emr_status {
    const int b = int(k & 1);
    emr_status e = wait_event(ev_done[b], deadline, limited);
    if (e != EMR_OK) return e;
    const int64_t* off = staging + b * (NP + 1);
    const int64_t total = off[NP];
    if (total > sp.chunk_cap) overflow = true;
    const int64_t n = std::min(total, sp.chunk_cap);
    ChunkOut& co = outs[k];
    co.at = cursor;
    co.off.assign(off, off + NP + 1);
    for (int64_t r = 0; r < NP; r++) counts[r] += off[r + 1] - off[r];
    const int64_t fit = std::max<int64_t>(0, std::min(n, cap - cursor));
    if (fit < n) overflow = true;
    if (fit > 0) {
      if (cudaMemcpyAsync(h_idx + cursor, base + sp.off_idx[b], size_t(fit) * 4, cudaMemcpyDeviceToHost, cp) !=
              cudaSuccess ||
          cudaMemcpyAsync(h_w + cursor, base + sp.off_w[b], size_t(fit) * 4, cudaMemcpyDeviceToHost, cp) !=
              cudaSuccess)
        return EMR_ERR_CUDA;
    }
    cursor += fit;
    return cudaEventRecord(ev_copied[b], cp) == cudaSuccess ? EMR_OK : EMR_ERR_CUDA;
  };

  for (size_t k = 0; k < sp.chunks.size() && rc == EMR_OK; k++) {
    const int b = int(k & 1);
    const int32_t t_lo = sp.chunks[k].first, t_hi = sp.chunks[k].second;
    const int64_t w_lo = tile_word(grid, t_lo, n_dense), w_hi = tile_word(grid, t_hi, n_dense);
    const int64_t p_lo = tile_pos(grid, t_lo, n_dense);
    if (k >= 2 && cudaStreamWaitEvent(st, ev_copied[b], 0) != cudaSuccess) { rc = EMR_ERR_CUDA; break; }
    uint32_t* bandc = reinterpret_cast<uint32_t*>(base + sp.off_band[b]);
    uint32_t* maskc = reinterpret_cast<uint32_t*>(base + sp.off_mask[b]);
    TileRange tr;
    tr.beg = t_lo;
    tr.end = t_hi;
    tr.band_stride = sp.wpc;
    tr.band_shift = w_lo;
    tr.out_stride = sp.ppc;
    tr.out_shift = p_lo;
    if ((rc = launch_tiles(sp.ev, grid, spec, order, kModeFused, theta, band, w_min, nullptr, nullptr, split, bandc,
                           st, tr)) != EMR_OK)
      break;
    if ((rc = launch_combine(split, PlaneView{bandc, sp.wpc, w_lo}, PlaneView{maskc, sp.wpc, w_lo}, grid, NP, w_lo,
                             w_hi - w_lo, 0, st, tf)) != EMR_OK)
      break;
    if ((rc = launch_compact(PlaneView{maskc, sp.wpc, w_lo}, nullptr, 0, 0, grid, NP, w_lo, w_hi - w_lo,
                             reinterpret_cast<int32_t*>(base + sp.off_idx[b]),
                             reinterpret_cast<float*>(base + sp.off_w[b]), sp.chunk_cap,
                             reinterpret_cast<int64_t*>(base + sp.off_cnt[b]),
                             reinterpret_cast<int64_t*>(base + sp.off_off[b]), base + sp.off_cws[b], st,
                             RecordSource{spec, sp.ev.L})) != EMR_OK)
      break;
    if (cudaMemcpyAsync(staging + b * (NP + 1), base + sp.off_off[b], size_t(NP + 1) * 8, cudaMemcpyDeviceToHost,
                        st) != cudaSuccess ||
        cudaEventRecord(ev_done[b], st) != cudaSuccess) {
      rc = EMR_ERR_CUDA;
      break;
    }
    if (k >= 1) rc = collect(k - 1);
  }
  if (rc == EMR_OK && !sp.chunks.empty()) rc = collect(sp.chunks.size() - 1);
  for (int b = 0; b < 2 && rc == EMR_OK; b++)
    if (ev_copied[b]) rc = wait_event(ev_copied[b], deadline, limited);
  if (rc == EMR_OK) {
    // per-pair lists in ascending global index: chunks in reverse processing order
    offsets[0] = 0;
    for (int64_t r = 0; r < NP; r++) offsets[r + 1] = offsets[r] + counts[r];
    if (!overflow && cursor > 0) {
      std::vector<int32_t> ti(h_idx, h_idx + cursor);
      std::vector<float> tw(h_w, h_w + cursor);
      int64_t dst = 0;
      for (int64_t r = 0; r < NP; r++)
        for (size_t k = sp.chunks.size(); k-- > 0;) {
          const ChunkOut& co = outs[k];
          const int64_t n = co.off[r + 1] - co.off[r];
          std::copy(ti.begin() + co.at + co.off[r], ti.begin() + co.at + co.off[r] + n, h_idx + dst);
          std::copy(tw.begin() + co.at + co.off[r], tw.begin() + co.at + co.off[r] + n, h_w + dst);
          dst += n;
        }
    }
    if (overflow) rc = EMR_ERR_CAPACITY;
  }
  if (rc == EMR_OK && mode == EMR_GATED && cursor > 0) {
    // Eq. 2 needs every ancestor's split bit, final only now: gate the eager lists
    // (a superset) against the resident split plane, a buffer of entries at a time.
    int64_t* off_dev = reinterpret_cast<int64_t*>(base + sp.off_off[0]);
    int32_t* idx_dev = reinterpret_cast<int32_t*>(base + sp.off_idx[0]);
    uint8_t* keep_dev = base + sp.off_w[0];
    std::vector<uint8_t> keep(static_cast<size_t>(cursor));
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        cudaMemcpyAsync(off_dev, offsets, size_t(NP + 1) * 8, cudaMemcpyHostToDevice, st) != cudaSuccess)
      rc = EMR_ERR_CUDA;
    for (int64_t e0 = 0; e0 < cursor && rc == EMR_OK; e0 += sp.chunk_cap) {
      const int64_t n = std::min(sp.chunk_cap, cursor - e0);
      if (cudaMemcpyAsync(idx_dev, h_idx + e0, size_t(n) * 4, cudaMemcpyHostToDevice, st) != cudaSuccess) {
        rc = EMR_ERR_CUDA;
        break;
      }
      gate_kernel<<<unsigned(8 * sms), kCompactBlock, 0, st>>>(split, grid_dev(grid), off_dev, NP, e0, n, idx_dev,
                                                              keep_dev);
      if (cudaGetLastError() != cudaSuccess ||
          cudaMemcpyAsync(keep.data() + e0, keep_dev, size_t(n), cudaMemcpyDeviceToHost, st) != cudaSuccess ||
          cudaEventRecord(ev_done[0], st) != cudaSuccess) {
        rc = EMR_ERR_CUDA;
        break;
      }
      rc = wait_event(ev_done[0], deadline, limited);
    }
    if (rc == EMR_OK) {  // drop the ungated entries in place, pair by pair
      int64_t dst = 0;
      for (int64_t r = 0; r < NP; r++) {
        const int64_t beg = offsets[r], end = offsets[r + 1];
        offsets[r] = dst;
        for (int64_t e = beg; e < end; e++)
          if (keep[size_t(e)]) {
            h_idx[dst] = h_idx[e];
            h_w[dst] = h_w[e];
            dst++;
          }
        counts[r] = dst - offsets[r];
      }
      offsets[NP] = dst;
    }
  }
  // a timed-out call leaves its queued work running; release what is safe to release
  if (rc != EMR_ERR_TIMEOUT && staging) cudaFreeHost(staging);
  for (int b = 0; b < 2; b++) {
    if (ev_done[b]) cudaEventDestroy(ev_done[b]);
    if (ev_copied[b]) cudaEventDestroy(ev_copied[b]);
  }
  if (cp) cudaStreamDestroy(cp);
  return rc;
}

extern "C" emr_status emr_stream(const void* pack_host, const void* pack_dev, const emr_query* q,
                                 const emr_grid* grid, float theta, float band, float w_min, void* ws, size_t ws_bytes,
                                 int64_t chunk_cap, int32_t* h_idx, float* h_w, int64_t cap, int64_t* counts,
                                 int64_t* offsets, int64_t timeout_ms, void* stream) {
  return emr_stream_mode(pack_host, pack_dev, q, grid, theta, band, w_min, EMR_EAGER, EMR_CONN_ALL, ws, ws_bytes,
                         chunk_cap, h_idx, h_w, cap, counts, offsets, timeout_ms, stream);
}
