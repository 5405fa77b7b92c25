// gemm_launch.cuh — the launch parameters of the GEMM kernels: work-unit
// widths, raster group heights, L2 eviction hints, the backward's vocabulary
// chunk, the layout of the transposed hidden states and the tile shape.
// Together with gemm_tc.cuh and ptx.cuh these set the GEMMs' DRAM traffic
// (the DRAM figures recorded from ncu are keyed on the three files).  Each
// default is the measured best; the environment variables named below
// override them (read at each call).
#pragma once

#include <algorithm>
#include <cstdint>
#include <cstdio>
#include <cstdlib>
#include <cstring>

#include "ptx.cuh"

namespace grpo {
namespace launch {

constexpr int kLseTilesPerUnit = 16;  // vocabulary tiles (of 256) per forward work unit
// Forward work units are narrowed (16 -> 8 -> 4 vocabulary tiles) while a batch
// has too few 256-row tiles to give every CTA pair of a GB300 (76) a unit: a
// decode step of 256 rows would otherwise leave half the pairs idle (measured:
// 0.36 ms and 52% of HBM bandwidth for the 1.27 GB head with 16-tile units).
constexpr int kNominalPairs = 76;
// Longest row of the transposed hidden states kept as plain rows.  Past it a
// GEMM stage (128 rows of 128 bytes) would touch one 2 MB page per row; the
// k-block layout keeps a stage contiguous.  Measured on the dW GEMM: plain rows
// faster at 64 KB and 512 KB rows (14.6 vs 15.7 ms and 128.7 vs 140.6 ms per
// step), k-blocks faster at 2 MB rows (147.6 vs 190.4 ms).
constexpr int64_t kMaxTransposedRowBytes = int64_t(1) << 20;
constexpr int64_t kDefaultVocabChunk = 16384;

inline int64_t round_up(int64_t x, int64_t m) { return (x + m - 1) / m * m; }

// Vocabulary columns per backward chunk: the dZ chunk buffer holds
// T x chunk bf16 values.  Multiple of 256; GRPO_VOCAB_CHUNK overrides.
inline int64_t vocab_chunk(int64_t V) {
  int64_t c = kDefaultVocabChunk;
  if (const char* e = std::getenv("GRPO_VOCAB_CHUNK")) {
    const long long v = std::atoll(e);
    if (v >= 256) c = round_up(v, 256);
  }
  return std::min<int64_t>(c, round_up(V, 256));
}

// Vocabulary tiles per forward work unit before any narrowing for small
// batches: kLseTilesPerUnit, or GRPO_LSE_TILES (4, 8, 16 or 32; read where
// the layout is made, so a workspace is sized and used with the same value).
inline int lse_tiles_per_unit() {
  if (const char* e = std::getenv("GRPO_LSE_TILES")) {
    const int v = std::atoi(e);
    if (v == 4 || v == 8 || v == 16 || v == 32) return v;
  }
  return kLseTilesPerUnit;
}

// N tiles one CTA (pair) walks per work unit in the backward GEMMs (dZ, dH,
// dW): consecutive tiles of a unit share the A tile.  GRPO_UNIT_N="z,h,w".
inline int units_n(int which) {
  int u[3] = {1, 1, 1};
  if (const char* e = std::getenv("GRPO_UNIT_N")) {
    int v[3];
    if (std::sscanf(e, "%d,%d,%d", &v[0], &v[1], &v[2]) == 3)
      for (int i = 0; i < 3; ++i) u[i] = v[i] > 0 ? v[i] : u[i];
  }
  return u[which];
}

// L2 policy of the A and B loads of GEMM `which` (LSE, dZ, dH, dW) as
// kHint* values; GRPO_L2_HINTS="aL,bL,aZ,bZ,aH,bH,aW,bW" overrides them.
inline void l2_hints(int which, int* a_hint, int* b_hint) {
  // Forward: keep A, stream W.  The backward GEMMs measured best without hints.
  int h[8] = {kHintEvictLast, kHintEvictFirst, kHintNone, kHintNone,
              kHintNone, kHintNone, kHintNone, kHintNone};
  if (const char* e = std::getenv("GRPO_L2_HINTS")) {
    int v[8];
    if (std::sscanf(e, "%d,%d,%d,%d,%d,%d,%d,%d", &v[0], &v[1], &v[2], &v[3], &v[4], &v[5], &v[6], &v[7]) == 8)
      for (int i = 0; i < 8; ++i) h[i] = (v[i] >= 0 && v[i] <= 2) ? v[i] : h[i];
  }
  *a_hint = h[2 * which];
  *b_hint = h[2 * which + 1];
}

// Layout of the transposed hidden states for T_pad tokens: k-blocks when a
// plain row would be longer than kMaxTransposedRowBytes;
// GRPO_HCT_LAYOUT=rows|blocks forces one (the tests cover both on small sizes).
inline bool hct_blocks(int64_t T_pad) {
  if (const char* e = std::getenv("GRPO_HCT_LAYOUT")) {
    if (std::strcmp(e, "rows") == 0) return false;
    if (std::strcmp(e, "blocks") == 0) return true;
  }
  return T_pad * 2 > kMaxTransposedRowBytes;
}

// Pace gate of the forward and sampling GEMMs (GemmArgs::gate): how many
// vocabulary tiles a CTA may run ahead of the slowest CTAs of the grid, and
// how many CTAs (per 64) may lag further; GRPO_GATE="slack[,lag]" overrides
// them (slack 0: no gate).
constexpr int kGateSlack = 1;  // tested against counters a tile old: about 2 tiles of spread
constexpr int kGateLagPer64 = 0;
constexpr int kGateSlots = 1024;  // CTAs a workspace's gate array holds
// Batches of fewer rows take no gate: a decode step's forward reads W about
// once anyway and runs below the power cap, so pacing only costs waits
// (2048 rows: 1.571 against 1.539 ms per draw with and without it).
constexpr int64_t kGateMinRows = 4096;

// Whether GEMM `which` (LSE and sampling forwards, dZ, dH, dW) takes the pace
// gate; GRPO_GATE_GEMMS="l,z,h,w" (1 or 0 each) overrides the defaults.
inline bool gate_on(int which) {
  int g[4] = {1, 0, 0, 0};
  if (const char* e = std::getenv("GRPO_GATE_GEMMS")) {
    int v[4];
    if (std::sscanf(e, "%d,%d,%d,%d", &v[0], &v[1], &v[2], &v[3]) == 4)
      for (int i = 0; i < 4; ++i) g[i] = v[i] != 0;
  }
  return g[which] != 0;
}

inline void gate_params(int grid, int* slack, int* lag) {
  int s = kGateSlack, l = kGateLagPer64;
  if (const char* e = std::getenv("GRPO_GATE")) {
    int a = -1, b = -1;
    const int n = std::sscanf(e, "%d,%d", &a, &b);
    if (n >= 1 && a >= 0) s = a;
    if (n == 2 && b >= 0 && b <= 64) l = b;
  }
  *slack = s;
  *lag = grid * l / 64;
}

// 2-CTA (cta_group::2) tiles unless GRPO_CTA_PAIR=0.
inline bool use_pairs() {
  const char* e = std::getenv("GRPO_CTA_PAIR");
  return !(e && e[0] == '0');
}

// Largest raster group (M tiles per group) of each GEMM: LSE, dZ, dH, dW,
// and the forward that stores the logits (4).  The kernel splits the M tiles
// into as few groups of near-equal height as this allows.  The forward GEMM
// re-reads A (the gathered hidden states) for every one of its ~600
// vocabulary tiles, while the CTAs working on one group share each W tile
// in L2: up to 24 M tiles (48 MB of A) per group.  Measured on 5,390 rows x
// 155,136 (22 M tiles): 6.57 GB of DRAM reads per forward launch with groups
// of 19 + 3 tiles, 4.02 GB with all 22 in one group, 11.5 GB with two of 11;
// at 19,572 rows the step time moved by less than run-to-run noise (59.6-61
// ms) between groups of 16, 19, 20 and 26.  The backward GEMMs measured best
// at 8; so did the forward that also stores the logits (47.5 against 47.8 ms
// per step at 19,572 tokens, 123 against 133 ms for the forward of 160,089
// tokens, whose logits stream through L2 beside the operand tiles).
// GRPO_GROUP_M="a,b,c,d[,e]" overrides the defaults.
inline int group_m(int which) {
  int g[5] = {24, 8, 8, 8, 8};
  if (const char* e = std::getenv("GRPO_GROUP_M")) {
    int v[5];
    const int n = std::sscanf(e, "%d,%d,%d,%d,%d", &v[0], &v[1], &v[2], &v[3], &v[4]);
    if (n >= 4)
      for (int i = 0; i < n; ++i) g[i] = v[i] > 0 ? v[i] : g[i];
  }
  return g[which];
}

// Raster along N for GEMM `which` (LSE, dZ, dH, dW): when > 0, groups of at
// most this many N units keep their B tiles in L2 while the group sweeps
// every M tile (group_m is then unused).  The dZ GEMM's B is a W chunk (134 MB
// at 16,384 columns) and its A the gathered hidden states (160 MB at 19,572
// rows): grouped by 8 M tiles it reads the W chunk once per group (10 times
// per launch at 77 M tiles), grouped by 16 N tiles (32 MB of W) it reads W
// once and A once per group (4 times).  dH and dW would read their larger A
// (the dZ chunk) that many times instead, so they keep the M groups.
// GRPO_GROUP_N="a,b,c,d" overrides (0: group along M).
inline int group_n(int which) {
  int g[4] = {0, 16, 0, 0};
  if (const char* e = std::getenv("GRPO_GROUP_N")) {
    int v[4];
    if (std::sscanf(e, "%d,%d,%d,%d", &v[0], &v[1], &v[2], &v[3]) == 4)
      for (int i = 0; i < 4; ++i) g[i] = v[i] >= 0 ? v[i] : g[i];
  }
  return g[which];
}

}  // namespace launch
}  // namespace grpo
