// gemm_tc.cuh — persistent, warp-specialised tcgen05 GEMM with the three
// epilogues of the GRPO LM-head path.
//
//   D[M x N] = A[M x K] * B[N x K]^T      (bf16 in, fp32 accumulate in TMEM)
//
// Tile 128 x 256 per CTA (kPair = 1) or 256 x 256 per CTA pair (kPair = 2,
// tcgen05 cta_group::2: each CTA stages its own 128 rows of A and half of B's
// 256 columns, the even CTA issues the MMAs for both, and each CTA's TMEM
// holds its 128 accumulator rows).  Roles per CTA (64 + 32 EpiShape::kWarps threads):
//   warp 0      TMA producer: 64-wide k-blocks (128-byte swizzle) into a ring
//               of shared-memory stages.
//   warp 1      owns 512 TMEM columns (two 256-column accumulators, so the
//               epilogue of tile i overlaps the MMAs of tile i + 1); one lane
//               of the issuing CTA issues the 128x256x16 / 256x256x16 MMAs.
//   warps 2..   epilogue (EpiShape::kWarps of them): one thread per accumulator row
//               (TMEM lane), 32 columns per tcgen05.ld; with 8 warps two share a
//               lane quarter and split the columns, their per-row log-softmax /
//               sampling state written as separate split entries.
//
// Epilogues:
//   kEpiLse  forward of the log-softmax (pi_theta in Eq. 1): per row a running
//            max and sum of exp over the tiles of one vocabulary split, plus
//            the logit of the target token; the logits never leave the SM.
//   kEpiLseZ the same, and the fp32 logits themselves are stored (through the
//            output tensor map, like kEpiF32), so that the backward forms dZ
//            from them instead of recomputing the GEMM.
//   kEpiDz   backward: recomputes the logits of one vocabulary chunk and
//            writes dZ = g (onehot(y) - softmax) as bf16.
//   kEpiF32  fp32 tile written as is or added to the existing values:
//            dW = dZ^T H, and dH += dZ W over the compacted rows.
//   Both write through a tensor map: each epilogue warp stages its 32 rows x
//   32 columns in shared memory and one lane issues a TMA store (or an L2
//   reduce-add), so the output leaves the SM as whole 32-row boxes instead of
//   32 scattered row segments per store instruction.
//   kEpiSample  the rollout draw o_t ~ softmax(z_t / temperature): per row the
//            running log-sum-exp of z / temperature and the running argmax of
//            z / temperature + Gumbel noise (Philox4x32-10, counter = (v / 4, t,
//            offset), key = seed); the logits never leave the SM.
//   kEpiSampleZ the same, and the fp32 logits z themselves are stored (as
//            kEpiLseZ does), for the nucleus (top-p) selection that follows.
//   kEpiAdam dW = dZ^T H consumed in place by an AdamW step on the matching
//            LM-head rows (fp32 master, both moments, bf16 weights out), so
//            dW itself is never stored; the weights and moments move through
//            shared memory with TMA loads and stores, 32 x 32 blocks per warp.
//
// Operands may be K-major (rows of the matrix run along K) or MN-major (rows
// run along M or N); the MN-major forms let dH read W and dW read dZ in the
// layout they already have.  dW's other operand is a transposed copy of the
// gathered hidden states (K-major), which measured faster than reading them
// MN-major.
#pragma once

#include <climits>

#include <cuda.h>
#include <stdint.h>

#include "ptx.cuh"

namespace grpo {

constexpr int kBK = 64;            // bf16 elements per 128-byte swizzle row
constexpr int kTileN = 256;        // accumulator columns per TMEM buffer
constexpr int kRowsCta = 128;      // accumulator rows per CTA (TMEM lanes)
constexpr int kTmemCols = 512;
constexpr int kRowAlign = 256;     // row padding of every token-indexed buffer
constexpr int kMaxHeads = 4;       // LM heads one forward launch can sweep

template <int kPair>
struct TileCfg {
  static constexpr int kTileM = kRowsCta * kPair;       // rows of one tile
  static constexpr int kBRows = kTileN / kPair;         // B rows (N) staged per CTA
  static constexpr int kABytes = kRowsCta * kBK * 2;    // 16 KB
  static constexpr int kBBytes = kBRows * kBK * 2;      // 32 KB (single) / 16 KB (pair)
  static constexpr int kStageBytes = kABytes + kBBytes;
};

enum { kEpiLse = 0, kEpiDz = 1, kEpiF32 = 2, kEpiAdam = 3, kEpiSample = 4, kEpiLseZ = 5, kEpiSampleZ = 6 };

// Epilogue warps per CTA: 4 = one per TMEM lane quarter (each thread walks its
// row's 256 columns); 8 = two per quarter, each taking half the columns.  The
// sampling epilogue (Philox and two logarithms per element) uses 8: measured
// on the 8B batch, 17.6 -> 16.7 ms.  The others keep 4: with 8, the dW GEMM
// of the same batch went from 15.7 to 16.7 ms per step.
template <int kEpi>
struct EpiShape {
  static constexpr int kWarps = kEpi == kEpiSample || kEpi == kEpiSampleZ ? 8 : 4;
  static constexpr int kHalves = kWarps / 4;    // column halves of a tile, one per warp of a quarter
  static constexpr int kThreads = 64 + 32 * kWarps;
  static constexpr bool kTmaOut =
      kEpi == kEpiDz || kEpi == kEpiF32 || kEpi == kEpiAdam || kEpi == kEpiLseZ || kEpi == kEpiSampleZ;
  // element type of the output tensor map: fp32 (128-byte rows of 32, 128-byte
  // swizzle) or bf16 (kEpiDz: 64-byte rows, 64-byte swizzle)
  static constexpr bool kOutF32 = kEpi == kEpiF32 || kEpi == kEpiLseZ || kEpi == kEpiAdam || kEpi == kEpiSampleZ;
  // one warp's 32 x 32 block in shared memory: bf16 dZ / fp32 output or
  // logits, two per warp; kEpiAdam: fp32 weights, first and second moments (4 KB each) and the
  // bf16 weights (2 KB), one per warp (the dW K-loop is long enough to hide it)
  static constexpr int kBlockBytes =
      kEpi == kEpiDz                        ? 32 * 32 * 2
      : kEpi == kEpiF32 || kEpi == kEpiLseZ || kEpi == kEpiSampleZ ? 32 * 32 * 4
      : kEpi == kEpiAdam                    ? 3 * 4096 + 2048
                                            : 0;
  static constexpr int kBlocks = kEpi == kEpiAdam ? 1 : 2;
  static constexpr int kOutBytes = kBlocks * kBlockBytes * kWarps;
};

// Operand-ring depth: 6 stages of 32 KB (pair) / 4 of 48 KB (single), one
// fewer for kEpiAdam and kEpiSampleZ (5 / 3), whose staging blocks take the
// room (kEpiSampleZ: 8 warps x 2 blocks of 4 KB).
template <int kPair, int kEpi>
__host__ __device__ constexpr int ring_stages() {
  return kEpi == kEpiAdam || kEpi == kEpiSampleZ ? (kPair == 2 ? 5 : 3) : (kPair == 2 ? 6 : 4);
}

// Dynamic shared memory of one CTA: the operand ring, the output staging
// blocks (1024-byte aligned, as the output swizzle needs), the barriers.
template <int kPair, int kEpi>
__host__ __device__ constexpr int smem_bytes() {
  return ring_stages<kPair, kEpi>() * TileCfg<kPair>::kStageBytes + EpiShape<kEpi>::kOutBytes + 1024 /*align*/ +
         256 /*barriers*/;
}

struct GemmArgs {
  const int* n_valid;   // device: number of compacted rows
  int M, N, K;          // extents; M or K is replaced by *n_valid when m_dyn / k_dyn
  int m_dyn, k_dyn;
  int a_off_m, a_off_k; // coordinate offsets into A's tensor map
  int b_off_n, b_off_k; // coordinate offsets into B's tensor map
  int n_per_unit;       // consecutive N tiles one CTA (pair) walks as one work unit
  int n_heads;          // B matrices (LM heads) swept against the same A, 1..kMaxHeads
  int group_m;          // raster: at most this many M tiles per group sharing the same N sweep
  int group_n;          // raster along N instead (when > 0): at most this many N units per group,
                        // their B tiles shared while the group sweeps every M tile
  int a_hint, b_hint;   // L2 eviction policy of A / B loads (kHint*)
  unsigned* status;     // device status word
  unsigned long long wait_ns;  // bound of every pipeline wait (0: kWaitLimitNs)
  int drop_kblock1;     // fault-injection test hook: CTA 0 skips the copies of its
                        // k-block number drop_kblock1 - 1 (0: never), so a wait runs out
  int drop_adam1;       // the same for kEpiAdam: CTA 0's epilogue warp 0 skips the loads of
                        // its weight block number drop_adam1 - 1 (0: never)
  int* gate;            // [gridDim.x] tiles each CTA has begun, zeroed before the launch
                        // (nullptr: no gate); see gate_wait
  int gate_slack;       // tiles a CTA may run ahead of the slowest ones
  int gate_lag;         // CTAs allowed to lag further behind

  // kEpiLse
  const int* yc;        // [M] target of each compacted row (-1: none)
  float* part_m;        // [units_n x halves x ldp] running max (log2 units); halves = EpiShape::kHalves
  float* part_s;        // [units_n x halves x ldp] running sum of 2^(z log2e - max)
  float* zy;            // [n_heads x ldp] logit of the target
  long ldp;

  // kEpiDz (output: bf16 through the output tensor map)
  const float* lse;     // [M] natural log-sum-exp of each row
  const float* gcoef;   // [M] dloss/dlogp of each row

  // kEpiF32 (output: fp32 through the output tensor map)
  int accumulate;       // 1: out += acc (L2 reduce-add), 0: out = acc

  const int* row_map;   // kEpiSample: token position of each compacted row

  // kEpiAdam: the accumulator is a dW tile; an AdamW step is applied to the
  // matching weights instead of storing dW.  The fp32 weights, both moments
  // and the bf16 weights are reached through tensor maps (the output map and
  // B maps 1..3, which a one-head launch does not otherwise use).
  float adam_b1, adam_b2, adam_eps, adam_lr;
  float adam_decay;     // 1 - lr * weight_decay
  float adam_bc1;       // 1 / (1 - beta1^step)
  float adam_bc2;       // 1 / (1 - beta2^step)

  // kEpiSample (row_map gives the token position t of each compacted row)
  float inv_temp;       // 1 / temperature
  uint32_t seed_lo, seed_hi, off_lo, off_hi;
  float* best_s;        // [units_n x halves x ldp] best perturbed score of the split entry
  int* best_c;          // [units_n x halves x ldp] its vocabulary column
  float* best_z;        // [units_n x halves x ldp] its z / temperature
};

struct TileSched {
  int m_tiles, n_tiles, units_head, units_n, total, k_blocks, m_rows;
  int group;  // M tiles (or, with GemmArgs::group_n, N units) per raster group, balanced
};

__device__ __forceinline__ TileSched make_sched(const GemmArgs& a, int tile_m) {
  TileSched s;
  const int nv = *a.n_valid;
  s.m_rows = a.m_dyn ? nv : a.M;
  const int K = a.k_dyn ? nv : a.K;
  s.m_tiles = (s.m_rows + tile_m - 1) / tile_m;
  s.n_tiles = (a.N + kTileN - 1) / kTileN;  // per head
  s.units_head = (s.n_tiles + a.n_per_unit - 1) / a.n_per_unit;
  s.units_n = s.units_head * max(1, a.n_heads);
  s.total = s.m_tiles * s.units_n;
  s.k_blocks = (K + kBK - 1) / kBK;
  // as few groups as group_m (group_n) allows, of near-equal height: a last
  // group of a few M tiles would stream all of B again for a sliver of the work
  const int along = a.group_n > 0 ? s.units_n : s.m_tiles;
  const int gmax = max(1, a.group_n > 0 ? a.group_n : a.group_m);
  const int ngroups = max(1, (along + gmax - 1) / gmax);
  s.group = max(1, (along + ngroups - 1) / ngroups);
  return s;
}

// Work unit u -> (m tile, n unit).  Groups of s.group consecutive M tiles
// sweep the N units together, so the CTAs running at the same time share B
// tiles (and A tiles) in L2.
__device__ __forceinline__ void unit_coords(const GemmArgs& a, const TileSched& s, int u, int& mt, int& un) {
  if (a.group_n > 0) {  // groups of s.group N units sweep every M tile
    const int per_group = s.group * s.m_tiles;
    const int g = u / per_group;
    const int first = g * s.group;
    const int gn = min(s.group, s.units_n - first);
    const int w = u - g * per_group;
    un = first + w % gn;
    mt = w / gn;
    return;
  }
  const int per_group = s.group * s.units_n;
  const int g = u / per_group;
  const int first = g * s.group;
  const int gm = min(s.group, s.m_tiles - first);
  const int w = u - g * per_group;
  mt = first + w % gm;
  un = w / gm;
}

// The pace gate of the persistent grid.  The CTAs sweeping one raster group
// read each B tile at about the same time only while they stay in step; left
// alone they drift apart by up to a work unit (the CTAs of a column start
// their units in different rounds), the B tiles between a column's first and
// last reader outgrow L2, and B is read from DRAM several times (measured: a
// W tile's readers spread over a median 13 tiles and the forward reading
// 24 GB for 5 GB of raster groups at 19,572 rows).  Each CTA publishes the
// number of tiles it has begun; before its k-th tile the producer warp waits
// until all CTAs but `lag` had begun tile k - slack.  The counters it tests
// were loaded when the previous tile began (so their latency hides behind that
// tile's copies, and a CTA in step goes on at once); only when those stale
// values fall short does it poll afresh.  The wait is a pace hint, not a
// dependency: it gives up after kGateNs and the CTA goes on, so it can delay
// a CTA but never stop one (a CTA that has issued all its loads publishes
// INT_MAX).
// A CTA never waits longer than a couple of tiles' time (about 20 us each at
// the 8B shape): in step the waits are far shorter, and a CTA that cannot
// start (its SM held by other work) should not hold the grid back for long.
constexpr unsigned long long kGateNs = 50000ull;  // 50 us
constexpr int kGateMaxCtas = 160;                   // counters a lane prefetches: 5 x 32
static_assert(kGateMaxCtas % 32 == 0, "whole counters per lane");

struct GatePrefetch {
  int v[kGateMaxCtas / 32];  // counters i = lane + 32 j, as loaded when the previous tile began
};

__device__ __forceinline__ int gate_behind(const GatePrefetch& p, int need, int n, int lane) {
  int behind = 0;
#pragma unroll
  for (int j = 0; j < kGateMaxCtas / 32; ++j) behind += lane + 32 * j < n && p.v[j] < need;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) behind += __shfl_xor_sync(0xffffffffu, behind, o);
  return behind;
}

__device__ __forceinline__ void gate_load(GatePrefetch& p, const volatile int* g, int n, int lane) {
#pragma unroll
  for (int j = 0; j < kGateMaxCtas / 32; ++j) p.v[j] = lane + 32 * j < n ? g[lane + 32 * j] : INT_MAX;
}

__device__ __forceinline__ void gate_wait(int* gate, int slack, int lag, int k, int lane, GatePrefetch& pre) {
  volatile int* g = gate;
  const int n = static_cast<int>(gridDim.x);
  if (lane == 0) g[blockIdx.x] = k;
  if (k > slack) {
    const int need = k - slack;
    if (gate_behind(pre, need, n, lane) > lag) {  // the stale counters fall short: poll
      const unsigned long long t0 = global_timer_ns();
      for (;;) {
        gate_load(pre, g, n, lane);
        if (gate_behind(pre, need, n, lane) <= lag) break;
        if (global_timer_ns() - t0 > kGateNs) break;
        __nanosleep(64);
      }
    }
  }
  gate_load(pre, g, n, lane);  // for the next tile: consumed when it begins
}

// ---------------------------------------------------------------- epilogue

// Per-row state of the epilogue for one work unit.
struct EpiRow {
  int r;          // accumulator row (compacted token / vocabulary row)
  bool rv;        // row inside M
  float run_m, run_s, zy_val;  // kEpiLse
  bool found;
  int y;
  float lse2, gr;  // kEpiDz
  int orow;        // kEpiSample: token position t
  float best_s, best_z;  // kEpiSample
  int best_c;
};

template <int kEpi>
__device__ __forceinline__ void epi_begin(EpiRow& e, const GemmArgs& a, int r, int m_rows) {
  const float kLog2e = 1.4426950408889634f;
  e.r = r;
  e.rv = r < m_rows;
  e.run_m = -INFINITY;
  e.run_s = 0.f;
  e.zy_val = 0.f;
  e.found = false;
  e.y = -1;
  e.lse2 = 0.f;
  e.gr = 0.f;
  e.orow = -1;
  e.best_s = -INFINITY;
  e.best_z = -INFINITY;
  e.best_c = -1;
  if (kEpi == kEpiSample || kEpi == kEpiSampleZ) {
    if (e.rv) e.orow = a.row_map[r];
  } else if (kEpi == kEpiLse || kEpi == kEpiLseZ) {
    e.y = e.rv ? a.yc[r] : -1;
  } else if (kEpi == kEpiDz) {
    if (e.rv) {
      e.y = a.yc[r];
      e.lse2 = a.lse[r] * kLog2e;
      e.gr = a.gcoef[r];
    }
  }
}

// One AdamW step of one weight element from its gradient g (fp32).
__device__ __forceinline__ void adam_update(float g, float& theta, float& m, float& v, const GemmArgs& a) {
  m = a.adam_b1 * m + (1.f - a.adam_b1) * g;
  v = a.adam_b2 * v + (1.f - a.adam_b2) * g * g;
  theta = theta * a.adam_decay - a.adam_lr * (m * a.adam_bc1) / (sqrtf(v * a.adam_bc2) + a.adam_eps);
}

// Output staging of one epilogue warp: two 32 x 32 blocks in shared memory,
// used in turn, and the tensor map of the output.
struct OutStage {
  uint32_t smem;             // first block (shared address); the second follows it
  int count;                 // blocks written so far by this warp
  const CUtensorMap* map;
  int lane;
  // kEpiAdam: the moments' and bf16 weights' maps, the block's load barrier
  const CUtensorMap* m_map;
  const CUtensorMap* v_map;
  const CUtensorMap* w_map;
  uint32_t ld_bar;
  uint32_t ld_phase;
  volatile int* abort;
  unsigned long long wlim;
  int blocks_loaded;         // kEpiAdam blocks this warp has loaded (fault-injection hook)
  bool first_warp;           // epilogue warp 0 of CTA 0 (fault-injection hook)
};

// Writes this warp's 32 x 32 output block (lane = row, `words` = the row's 64
// bytes of bf16 pairs or 128 bytes of fp32) to global memory at (x, y): the
// rows go into a shared block in the swizzle the output map declares (64-byte
// rows in the 64-byte swizzle, 128-byte rows in the 128-byte one: the 16-byte
// chunk index is XORed with bits 7.. of the offset, which also puts the writes
// of any 8 consecutive lanes on distinct bank groups), then lane 0 issues a
// TMA store, or an element-wise add at L2 when `reduce`.  kEvictFirst: the
// stored lines are the first L2 evicts (an output that is not read again
// while it could still be in L2 should not push out the operand tiles).
template <int kWords, bool kEvictFirst = false>
__device__ __forceinline__ void out_block(OutStage& o, const uint32_t* words, int x, int y, bool reduce) {
  constexpr int kRowBytes = kWords * 4;
  const uint32_t buf = o.smem + static_cast<uint32_t>(o.count & 1) * (32 * kRowBytes);
  // the store issued from this block two blocks ago must have read it
  if (o.lane == 0) bulk_wait_read_1();
  __syncwarp();
  const uint32_t row = buf + static_cast<uint32_t>(o.lane * kRowBytes);
  const uint32_t sw = kRowBytes == 64 ? (o.lane >> 1) & 3 : o.lane & 7;
#pragma unroll
  for (int j = 0; j < kWords / 4; ++j)
    st_shared_v4(row + 16u * (static_cast<uint32_t>(j) ^ sw), words[4 * j], words[4 * j + 1], words[4 * j + 2],
                 words[4 * j + 3]);
  fence_proxy_async_smem();
  __syncwarp();
  if (o.lane == 0) {
    if (reduce) tma_reduce_add_2d(o.map, buf, x, y);
    else if (kEvictFirst) tma_store_2d_hint(o.map, buf, x, y, l2_policy(kHintEvictFirst));
    else tma_store_2d(o.map, buf, x, y);
    bulk_commit();
  }
  ++o.count;
}

// One AdamW step on this warp's 32 x 32 block of LM-head weights at (x, y),
// whose gradient rows are in `g` (lane = row): lane 0 loads the fp32 weights
// and both moments with TMA (128-byte swizzle, zero-filled past the matrix),
// every lane updates its row in shared memory, and lane 0 stores the three
// blocks and the bf16 weights back (clipped at the matrix).  False if the load
// wait gave up (abort or time limit).
__device__ __forceinline__ bool adam_block(OutStage& o, const float* g, int x, int y, const GemmArgs& a) {
  const uint32_t th = o.smem, mo = o.smem + 4096, ve = o.smem + 8192, wb = o.smem + 12288;
  if (o.lane == 0) {
    bulk_wait_read_0();  // the previous block's stores have read the buffer
    mbar_arrive_expect_tx(o.ld_bar, 3 * 4096);
    // the test hook: these bytes never arrive, so the wait below runs out
    const bool drop = o.first_warp && ++o.blocks_loaded == a.drop_adam1;
    if (!drop) {
      tma_load_2d(th, o.map, o.ld_bar, x, y);
      tma_load_2d(mo, o.m_map, o.ld_bar, x, y);
      tma_load_2d(ve, o.v_map, o.ld_bar, x, y);
    }
  }
  const bool got = mbar_wait(o.ld_bar, o.ld_phase, o.abort, o.wlim);
  if (!got && o.lane == 0) {
    // the wait gave up: let the block's loads land before the buffer can be
    // released (they complete on ld_bar unless they were never issued)
    volatile int never = 0;
    if (!mbar_wait(o.ld_bar, o.ld_phase, &never, kDrainNs)) __nanosleep(kDrainPauseNs);
  }
  o.ld_phase ^= 1u;
  if (!__all_sync(0xffffffffu, got)) return false;
  const uint32_t row = static_cast<uint32_t>(o.lane * 128);
  const uint32_t sw = o.lane & 7;
  uint32_t wpk[16];
#pragma unroll
  for (int q = 0; q < 8; ++q) {
    const uint32_t off = row + 16u * (static_cast<uint32_t>(q) ^ sw);
    float4 p, m, v;
    ld_shared_v4(th + off, p);
    ld_shared_v4(mo + off, m);
    ld_shared_v4(ve + off, v);
    adam_update(g[4 * q + 0], p.x, m.x, v.x, a);
    adam_update(g[4 * q + 1], p.y, m.y, v.y, a);
    adam_update(g[4 * q + 2], p.z, m.z, v.z, a);
    adam_update(g[4 * q + 3], p.w, m.w, v.w, a);
    st_shared_v4(th + off, __float_as_uint(p.x), __float_as_uint(p.y), __float_as_uint(p.z), __float_as_uint(p.w));
    st_shared_v4(mo + off, __float_as_uint(m.x), __float_as_uint(m.y), __float_as_uint(m.z), __float_as_uint(m.w));
    st_shared_v4(ve + off, __float_as_uint(v.x), __float_as_uint(v.y), __float_as_uint(v.z), __float_as_uint(v.w));
    wpk[2 * q] = pack_bf16x2(p.x, p.y);
    wpk[2 * q + 1] = pack_bf16x2(p.z, p.w);
  }
  const uint32_t wrow = wb + static_cast<uint32_t>(o.lane * 64);
  const uint32_t wsw = (o.lane >> 1) & 3;
#pragma unroll
  for (int j = 0; j < 4; ++j)
    st_shared_v4(wrow + 16u * (static_cast<uint32_t>(j) ^ wsw), wpk[4 * j], wpk[4 * j + 1], wpk[4 * j + 2],
                 wpk[4 * j + 3]);
  fence_proxy_async_smem();
  __syncwarp();
  if (o.lane == 0) {
    tma_store_2d(o.map, th, x, y);
    tma_store_2d(o.m_map, mo, x, y);
    tma_store_2d(o.v_map, ve, x, y);
    tma_store_2d(o.w_map, wb, x, y);
    bulk_commit();
  }
  return true;
}

// One 256-column accumulator tile of this thread's row; `tbase` is the TMEM
// address of column 0 of the tile in this warp's lane quarter; `row0` is the
// accumulator row of lane 0 (the TMA row coordinate of the warp's block) and
// m_rows the rows of the output (M).
template <int kEpi>
__device__ __forceinline__ bool epi_tile(EpiRow& e, const GemmArgs& a, uint32_t tbase, int col0,
                                         bool have_acc, int half, OutStage& os, int row0, int m_rows) {
  const float kLog2e = 1.4426950408889634f;
  constexpr int kChunks = kTileN / 32 / EpiShape<kEpi>::kHalves;
#pragma unroll 1
  for (int c = half * kChunks; c < (half + 1) * kChunks; ++c) {
    float v[32];
    if (have_acc) {
      tmem_ld32(tbase + c * 32, v);
    } else {
#pragma unroll
      for (int j = 0; j < 32; ++j) v[j] = 0.f;
    }
    const int cb = col0 + c * 32;
    if (kEpi == kEpiLse || kEpi == kEpiLseZ) {
      // kEpiLseZ: the raw logits first (blocks wholly past M or N skipped, the
      // tensor map clips the rest); they are read again only by the backward's
      // dZ pass, long after they have left L2
      if (kEpi == kEpiLseZ && row0 < m_rows && cb < a.N) {
        uint32_t bits[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) bits[j] = __float_as_uint(v[j]);
        out_block<32, true>(os, bits, cb, row0, false);
      }
      if (cb + 32 > a.N) {
#pragma unroll
        for (int j = 0; j < 32; ++j)
          if (cb + j >= a.N) v[j] = -INFINITY;
      }
      const unsigned off = static_cast<unsigned>(e.y - cb);
      if (off < 32u) {
        float t = v[0];
#pragma unroll
        for (int j = 1; j < 32; ++j) t = (off == static_cast<unsigned>(j)) ? v[j] : t;
        e.zy_val = t;
        e.found = true;
      }
      float cm = v[0];
#pragma unroll
      for (int j = 1; j < 32; ++j) cm = fmaxf(cm, v[j]);
      const float nm = fmaxf(e.run_m, cm * kLog2e);
      if (nm != -INFINITY) {  // a half-tile past V is all -inf: nothing to add
        float acc = 0.f;
#pragma unroll
        for (int j = 0; j < 32; ++j) acc += fast_exp2(fmaf(v[j], kLog2e, -nm));
        e.run_s = e.run_s * fast_exp2(e.run_m - nm) + acc;
        e.run_m = nm;
      }
    } else if (kEpi == kEpiSample || kEpi == kEpiSampleZ) {
      // kEpiSampleZ: the raw logits first (as kEpiLseZ, evict-first), read
      // again by the nucleus selection after this GEMM
      if (kEpi == kEpiSampleZ && row0 < m_rows && cb < a.N) {
        uint32_t bits[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) bits[j] = __float_as_uint(v[j]);
        out_block<32, true>(os, bits, cb, row0, false);
      }
      // scaled logits (cols >= N: -inf) -> running LSE and running argmax of z + noise
#pragma unroll
      for (int j = 0; j < 32; ++j) v[j] = (cb + j < a.N) ? v[j] * a.inv_temp : -INFINITY;
      if (e.rv) {
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          const uint4 w = philox4x32_10(
              make_uint4(static_cast<uint32_t>((cb >> 2) + q), static_cast<uint32_t>(e.orow), a.off_lo, a.off_hi),
              a.seed_lo, a.seed_hi);
          const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const int j = 4 * q + k;
            const float sc = v[j] + gumbel_of(ws[k]);
            if (sc > e.best_s) {  // strict: the lowest column wins a tie
              e.best_s = sc;
              e.best_c = cb + j;
              e.best_z = v[j];
            }
          }
        }
      }
      float cm = v[0];
#pragma unroll
      for (int j = 1; j < 32; ++j) cm = fmaxf(cm, v[j]);
      const float nm = fmaxf(e.run_m, cm * kLog2e);
      if (nm != -INFINITY) {  // a half-tile past V is all -inf: nothing to add
        float acc = 0.f;
#pragma unroll
        for (int j = 0; j < 32; ++j) acc += fast_exp2(fmaf(v[j], kLog2e, -nm));
        e.run_s = e.run_s * fast_exp2(e.run_m - nm) + acc;
        e.run_m = nm;
      }
    } else if (kEpi == kEpiDz) {
      const int gc = a.b_off_n + cb;  // vocabulary id of column 0 of this group
      uint32_t packed[16];
#pragma unroll
      for (int j = 0; j < 32; j += 2) {
        float d0 = dz_value(v[j], e.lse2, e.gr, gc + j == e.y);
        float d1 = dz_value(v[j + 1], e.lse2, e.gr, gc + j + 1 == e.y);
        if (cb + j >= a.N || !e.rv) d0 = 0.f;
        if (cb + j + 1 >= a.N || !e.rv) d1 = 0.f;
        packed[j / 2] = pack_bf16x2(d0, d1);
      }
      out_block<16>(os, packed, cb, row0, false);
    } else if (kEpi == kEpiAdam) {
      // a block wholly past M or N is skipped; the tensor maps clip the rest
      if (row0 < m_rows && cb < a.N && !adam_block(os, v, cb, row0, a)) return false;
    } else {
      // kEpiF32: a block wholly past M or N is skipped; the tensor map clips
      // the rest (its rows are the output's M, its columns N)
      if (row0 < m_rows && cb < a.N) {
        uint32_t bits[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) bits[j] = __float_as_uint(v[j]);
        out_block<32>(os, bits, cb, row0, a.accumulate != 0);
      }
    }
  }
  return true;
}

template <int kEpi>
__device__ __forceinline__ void epi_end(const EpiRow& e, const GemmArgs& a, int un, int head, int half) {
  const long entry = static_cast<long>(un) * EpiShape<kEpi>::kHalves + half;  // split entry of this column half
  if ((kEpi == kEpiSample || kEpi == kEpiSampleZ) && e.rv) {
    const long at = entry * a.ldp + e.r;
    a.part_m[at] = e.run_m;
    a.part_s[at] = e.run_s;
    a.best_s[at] = e.best_s;
    a.best_c[at] = e.best_c;
    a.best_z[at] = e.best_z;
  }
  if ((kEpi == kEpiLse || kEpi == kEpiLseZ) && e.rv) {
    a.part_m[entry * a.ldp + e.r] = e.run_m;
    a.part_s[entry * a.ldp + e.r] = e.run_s;
    if (e.found) a.zy[static_cast<long>(head) * a.ldp + e.r] = e.zy_val;
  }
}

// ---------------------------------------------------------------- kernel body

// kBblk: B is K-major and stored in k-blocks [K / 64][N][64] (a 3-D tensor
// map), so that one stage of B is a single contiguous run however long K is.
template <int kPair, int kEpi, bool kAmn, bool kBmn, bool kBblk>
__device__ __forceinline__ void gemm_body(const CUtensorMap* tmA, const CUtensorMap* const* tmBs,
                                          const CUtensorMap* tmD, const GemmArgs& args) {
  using C = TileCfg<kPair>;
  using ES = EpiShape<kEpi>;
  constexpr int kStages = ring_stages<kPair, kEpi>();
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* out_stage = smem + kStages * C::kStageBytes;  // [warps][blocks] output staging
  uint64_t* bars = reinterpret_cast<uint64_t*>(out_stage + ES::kOutBytes);
  uint64_t* full_bar = bars;                          // [kStages] TMA -> MMA (issuing CTA)
  uint64_t* empty_bar = bars + kStages;               // [kStages] MMA -> TMA (each CTA)
  uint64_t* tfull_bar = bars + 2 * kStages;           // [2] MMA -> epilogue (each CTA)
  uint64_t* tempty_bar = bars + 2 * kStages + 2;      // [2] epilogue -> MMA (issuing CTA)
  uint64_t* done_bar = bars + 2 * kStages + 4;        // [1] all MMAs retired (issuing CTA)
  uint64_t* ld_bar = bars + 2 * kStages + 5;          // [4] kEpiAdam block loads (one per epilogue warp)
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * kStages + 9);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = kPair == 2 ? cluster_ctarank() : 0u;
  const bool issuer = rank == 0;
  const int unit0 = blockIdx.x / kPair;
  const int unit_stride = gridDim.x / kPair;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(smem_addr(&full_bar[i]), 1);
      mbar_init(smem_addr(&empty_bar[i]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_addr(&tfull_bar[i]), 1);
      mbar_init(smem_addr(&tempty_bar[i]), EpiShape<kEpi>::kWarps * kPair);  // one arrival per epilogue warp
    }
    mbar_init(smem_addr(done_bar), 1);
    if (kEpi == kEpiAdam)
      for (int i = 0; i < ES::kWarps; ++i) mbar_init(smem_addr(&ld_bar[i]), 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(tmA);
    for (int h = 0; h < args.n_heads; ++h) tma_prefetch_desc(tmBs[h]);
    if (ES::kTmaOut) tma_prefetch_desc(tmD);
  }
  if (warp == 1) {
    if (kPair == 2) {
      tmem_alloc_pair(smem_addr(tmem_slot), kTmemCols);
      tmem_relinquish_pair();
    } else {
      tmem_alloc(smem_addr(tmem_slot), kTmemCols);
      tmem_relinquish();
    }
  }
  tc_fence_before();
  if (kPair == 2) cluster_sync(); else __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  const TileSched sch = make_sched(args, C::kTileM);
  const int KB = sch.k_blocks;
  const unsigned long long wlim = args.wait_ns ? args.wait_ns : kWaitLimitNs;

  // Raises the abort flag of this CTA and of its peer.
  auto raise_abort = [&]() {
    *abort_flag = 1;
    if (kPair == 2) st_shared_cluster(mapa_shared(smem_addr(const_cast<int*>(abort_flag)), rank ^ 1u), 1u);
    atomicOr(args.status, kDevTimeout);
  };

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    // Lane 0 issues the copies; the whole warp takes the pace gate between tiles.
    {
      const uint64_t pol_a = l2_policy(args.a_hint);
      const uint64_t pol_b = l2_policy(args.b_hint);
      int stage = 0;
      uint32_t phase = 0;
      int uses[kStages];
#pragma unroll
      for (int s = 0; s < kStages; ++s) uses[s] = 0;
      bool ok = true;
      int kblock_count = 0;  // k-blocks this CTA has staged (fault-injection hook)
      int tiles_begun = 0;
      GatePrefetch gate_pre;
#pragma unroll
      for (int j = 0; j < kGateMaxCtas / 32; ++j) gate_pre.v[j] = 0;
      for (int u = unit0; u < sch.total && ok; u += unit_stride) {
        int mt, un;
        unit_coords(args, sch, u, mt, un);
        const int head = un / sch.units_head;
        const int nt0 = (un - head * sch.units_head) * args.n_per_unit;
        const int nt1 = min(sch.n_tiles, nt0 + args.n_per_unit);
        for (int nt = nt0; nt < nt1 && ok; ++nt) {
          if (args.gate) gate_wait(args.gate, args.gate_slack, args.gate_lag, tiles_begun, lane, gate_pre);
          ++tiles_begun;
          for (int kb = 0; kb < KB && lane == 0; ++kb) {
            if (!mbar_wait(smem_addr(&empty_bar[stage]), phase ^ 1u, abort_flag, wlim)) {
              ok = false;
              break;
            }
            const uint32_t fb_local = smem_addr(&full_bar[stage]);
            const uint32_t fb = kPair == 2 ? mapa_shared(fb_local, 0) : fb_local;
            if (issuer) mbar_arrive_expect_tx(fb_local, kPair * C::kStageBytes);
            const uint32_t sa = smem_addr(smem + stage * C::kStageBytes);
            const uint32_t sb = sa + C::kABytes;
            const int k0 = kb * kBK;
            const int m0 = mt * C::kTileM + static_cast<int>(rank) * kRowsCta;
            const int n0 = nt * kTileN + static_cast<int>(rank) * C::kBRows;
            const bool drop = blockIdx.x == 0 && ++kblock_count == args.drop_kblock1;
            auto load = [&](uint32_t dst, const CUtensorMap* map, int c0, int c1, uint64_t pol) {
              if (drop) return;  // the test hook: these bytes never arrive
              if (kPair == 2) tma_load_2d_pair_hint(dst, map, fb, c0, c1, pol);
              else tma_load_2d_hint(dst, map, fb, c0, c1, pol);
            };
            auto load_blk = [&](uint32_t dst, const CUtensorMap* map, int row, int kblk, uint64_t pol) {
              if (drop) return;
              if (kPair == 2) tma_load_3d_pair_hint(dst, map, fb, 0, row, kblk, pol);
              else tma_load_3d_hint(dst, map, fb, 0, row, kblk, pol);
            };
            if (!kAmn) {
              load(sa, tmA, k0 + args.a_off_k, m0 + args.a_off_m, pol_a);
            } else {
#pragma unroll
              for (int j = 0; j < kRowsCta / 64; ++j)
                load(sa + j * 8192, tmA, m0 + args.a_off_m + 64 * j, k0 + args.a_off_k, pol_a);
            }
            if (!kBmn && kBblk) {
              load_blk(sb, tmBs[head], n0 + args.b_off_n, (k0 + args.b_off_k) >> 6, pol_b);
            } else if (!kBmn) {
              load(sb, tmBs[head], k0 + args.b_off_k, n0 + args.b_off_n, pol_b);
            } else {
#pragma unroll
              for (int j = 0; j < C::kBRows / 64; ++j)
                load(sb + j * 8192, tmBs[head], n0 + args.b_off_n + 64 * j, k0 + args.b_off_k, pol_b);
            }
            ++uses[stage];
            if (++stage == kStages) {
              stage = 0;
              phase ^= 1u;
            }
          }
          ok = __shfl_sync(0xffffffffu, ok, 0);
        }
      }
      if (args.gate && lane == 0) {  // every copy issued: nobody waits for this CTA any more
        volatile int* g = args.gate;
        g[blockIdx.x] = INT_MAX;
      }
      if (lane == 0 && !ok) raise_abort();
      // Every stage this CTA filled must have been consumed (so its copies
      // have landed) before the CTA can exit.
      for (int s = 0; s < kStages && lane == 0; ++s)
        if (uses[s] > 0)
          mbar_wait(smem_addr(&empty_bar[s]), static_cast<uint32_t>(uses[s] - 1) & 1u, abort_flag, wlim);
      // After an abort those waits give up at once, and a stage may still
      // have copies in flight.  The issuing CTA's full barrier of a stage
      // counts every byte both CTAs of the pair loaded into it, so a bounded
      // wait on the phase of each stage's last fill returns once they have
      // landed (the teardown's cluster barrier then holds the peer until this
      // drain ends).  Where that phase cannot complete (a copy that was never
      // issued), and on the peer, whose copies only the issuing CTA's
      // barriers count, a fixed pause stands in for the wait.
      if (lane == 0 && *abort_flag) {
        bool drained = issuer;
        if (issuer) {
          volatile int never = 0;
          for (int s = 0; s < kStages; ++s)
            if (uses[s] > 0 && !mbar_wait(smem_addr(&full_bar[s]), static_cast<uint32_t>(uses[s] - 1) & 1u, &never,
                                          kDrainNs))
              drained = false;
        }
        if (!drained) __nanosleep(kDrainPauseNs);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0 && issuer) {
      constexpr uint32_t idesc = idesc_bf16_f32(C::kTileM, kTileN, kAmn, kBmn);
      int stage = 0;
      uint32_t phase = 0;
      int tile = 0;
      bool ok = true;
      for (int u = unit0; u < sch.total && ok; u += unit_stride) {
        int mt, un;
        unit_coords(args, sch, u, mt, un);
        const int head = un / sch.units_head;
        const int nt0 = (un - head * sch.units_head) * args.n_per_unit;
        const int nt1 = min(sch.n_tiles, nt0 + args.n_per_unit);
        for (int nt = nt0; nt < nt1 && ok; ++nt) {
          if (KB == 0) continue;
          const int buf = tile & 1;
          const uint32_t use = static_cast<uint32_t>(tile >> 1);
          if (!mbar_wait(smem_addr(&tempty_bar[buf]), (use & 1u) ^ 1u, abort_flag, wlim)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(buf * kTileN);
          for (int kb = 0; kb < KB; ++kb) {
            if (!mbar_wait(smem_addr(&full_bar[stage]), phase, abort_flag, wlim)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t sa = smem_addr(smem + stage * C::kStageBytes);
            const uint32_t sb = sa + C::kABytes;
#pragma unroll
            for (int kk = 0; kk < kBK / 16; ++kk) {
              const uint64_t ad = kAmn ? sdesc_sw128(sa + kk * 2048, 8192, 1024)
                                       : sdesc_sw128(sa + kk * 32, 16, 1024);
              const uint64_t bd = kBmn ? sdesc_sw128(sb + kk * 2048, 8192, 1024)
                                       : sdesc_sw128(sb + kk * 32, 16, 1024);
              const uint32_t acc = (kb | kk) != 0 ? 1u : 0u;
              if (kPair == 2) tc_mma_bf16_pair(d_tmem, ad, bd, idesc, acc);
              else tc_mma_bf16(d_tmem, ad, bd, idesc, acc);
            }
            if (kPair == 2) tc_commit_pair_mc(smem_addr(&empty_bar[stage]), 0x3);
            else tc_commit(smem_addr(&empty_bar[stage]));
            if (++stage == kStages) {
              stage = 0;
              phase ^= 1u;
            }
          }
          if (!ok) break;
          if (kPair == 2) tc_commit_pair_mc(smem_addr(&tfull_bar[buf]), 0x3);
          else tc_commit(smem_addr(&tfull_bar[buf]));
          ++tile;
        }
      }
      if (!ok) raise_abort();
      // Retire every MMA before TMEM is released (not cut short by the abort flag:
      // issued MMAs always finish).
      if (kPair == 2) tc_commit_pair_mc(smem_addr(done_bar), 0x1);
      else tc_commit(smem_addr(done_bar));
      volatile int never = 0;
      mbar_wait(smem_addr(done_bar), 0, &never, wlim);
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int quad = warp & 3;              // TMEM lanes quad*32 .. quad*32+31
    const int half = (warp - 2) / 4;         // which 128 of the tile's 256 columns
    const int row = static_cast<int>(rank) * kRowsCta + quad * 32 + lane;  // row within the tile
    const uint32_t lane_addr = tmem_base + (static_cast<uint32_t>(quad * 32) << 16);
    const uint32_t tempty0 = smem_addr(&tempty_bar[0]);
    const uint32_t tempty1 = smem_addr(&tempty_bar[1]);
    const uint32_t tempty_c0 = kPair == 2 ? mapa_shared(tempty0, 0) : tempty0;
    const uint32_t tempty_c1 = kPair == 2 ? mapa_shared(tempty1, 0) : tempty1;
    OutStage os{smem_addr(out_stage) + static_cast<uint32_t>((warp - 2) * ES::kBlocks * ES::kBlockBytes),
                0,
                tmD,
                lane,
                tmBs[1],
                tmBs[2],
                tmBs[3],
                smem_addr(&ld_bar[kEpi == kEpiAdam ? warp - 2 : 0]),
                0u,
                abort_flag,
                wlim,
                0,
                blockIdx.x == 0 && warp == 2};
    int tile = 0;
    bool ok = true;
    for (int u = unit0; u < sch.total && ok; u += unit_stride) {
      int mt, un;
      unit_coords(args, sch, u, mt, un);
      const int head = un / sch.units_head;
      const int nt0 = (un - head * sch.units_head) * args.n_per_unit;
      const int nt1 = min(sch.n_tiles, nt0 + args.n_per_unit);
      EpiRow e;
      epi_begin<kEpi>(e, args, mt * C::kTileM + row, sch.m_rows);
      const int row0 = mt * C::kTileM + row - lane;  // accumulator row of lane 0
      for (int nt = nt0; nt < nt1; ++nt) {
        const int buf = tile & 1;
        const uint32_t use = static_cast<uint32_t>(tile >> 1);
        const bool have_acc = KB > 0;
        if (have_acc) {
          // all lanes must agree before the warp-wide tcgen05.ld: a lane that gave up
          // (abort) while another saw the phase complete makes the whole warp give up
          const bool got = mbar_wait(smem_addr(&tfull_bar[buf]), use & 1u, abort_flag, wlim);
          if (!__all_sync(0xffffffffu, got)) {
            ok = false;
            break;
          }
          tc_fence_after();
        }
        const bool done = epi_tile<kEpi>(e, args, lane_addr + static_cast<uint32_t>(buf * kTileN), nt * kTileN,
                                         have_acc, half, os, row0, sch.m_rows);
        if (have_acc) {
          tc_fence_before();
          __syncwarp();
          if (lane == 0) {
            const uint32_t tb = buf ? tempty_c1 : tempty_c0;
            if (kPair == 2) mbar_arrive_cluster(tb); else mbar_arrive(tb);
          }
          ++tile;
        }
        if (!done) {  // a kEpiAdam block load gave up
          ok = false;
          break;
        }
      }
      if (!ok) break;
      epi_end<kEpi>(e, args, un, head, half);
    }
    if (!ok) raise_abort();
    // the output boxes in flight read shared memory and must land before exit
    if (ES::kTmaOut && lane == 0) bulk_wait_all();
  }

  // (after a timeout the producer has drained the copies it issued: above)
  tc_fence_before();
  if (kPair == 2) cluster_sync(); else __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    if (kPair == 2) tmem_dealloc_pair(tmem_base, kTmemCols);
    else tmem_dealloc(tmem_base, kTmemCols);
  }
}

// One tensor map per B matrix; B1..B3 are read only when args.n_heads > 1.
template <int kEpi, bool kAmn, bool kBmn, bool kBblk = false>
__global__ void __launch_bounds__(EpiShape<kEpi>::kThreads, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB0,
                   const __grid_constant__ CUtensorMap tmB1, const __grid_constant__ CUtensorMap tmB2,
                   const __grid_constant__ CUtensorMap tmB3, const __grid_constant__ CUtensorMap tmD,
                   const GemmArgs args) {
  const CUtensorMap* tmBs[kMaxHeads] = {&tmB0, &tmB1, &tmB2, &tmB3};
  gemm_body<1, kEpi, kAmn, kBmn, kBblk>(&tmA, tmBs, &tmD, args);
}

template <int kEpi, bool kAmn, bool kBmn, bool kBblk = false>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(EpiShape<kEpi>::kThreads, 1)
    gemm_tc_pair_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB0,
                        const __grid_constant__ CUtensorMap tmB1, const __grid_constant__ CUtensorMap tmB2,
                        const __grid_constant__ CUtensorMap tmB3, const __grid_constant__ CUtensorMap tmD,
                        const GemmArgs args) {
  const CUtensorMap* tmBs[kMaxHeads] = {&tmB0, &tmB1, &tmB2, &tmB3};
  gemm_body<2, kEpi, kAmn, kBmn, kBblk>(&tmA, tmBs, &tmD, args);
}

}  // namespace grpo
