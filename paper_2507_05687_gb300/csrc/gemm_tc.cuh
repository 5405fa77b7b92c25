// gemm_tc.cuh — persistent, warp-specialised tcgen05 GEMM with the three
// epilogues of the GRPO LM-head path.
//
//   D[M x N] = A[M x K] * B[N x K]^T      (bf16 in, fp32 accumulate in TMEM)
//
// Roles (192 threads, one CTA per SM):
//   warp 0      TMA producer: streams 128x64 A and 256x64 B k-blocks into a
//               4-stage shared-memory ring (128-byte swizzle).
//   warp 1      allocates 512 TMEM columns; one lane issues tcgen05.mma
//               (128x256x16 per instruction) into one of two 256-column
//               accumulators, so the epilogue of tile i overlaps the MMAs of
//               tile i + 1.
//   warps 2..5  epilogue: one thread per accumulator row (TMEM lane), reading
//               32 columns per tcgen05.ld.
//
// Epilogues:
//   kEpiLse  forward of the log-softmax (pi_theta in Eq. 1): per row a running
//            max and sum of exp over the tiles of one vocabulary split, plus
//            the logit of the target token; the logits never leave the SM.
//   kEpiDz   backward: recomputes the logits of one vocabulary chunk and
//            writes dZ = g (onehot(y) - softmax) as bf16.
//   kEpiF32  plain fp32 store (optionally added to the existing values) with
//            an optional row map: dH += dZ W and dW = dZ^T H.
//
// Operands may be K-major (rows of the matrix run along K) or MN-major (rows
// run along M or N); the MN-major forms let dH and dW read W, H and dZ in the
// layout they already have, with no transposed copies.
#pragma once

#include <cuda.h>
#include <stdint.h>

#include "ptx.cuh"

namespace grpo {

constexpr int kBM = 128;                 // accumulator rows (TMEM lanes)
constexpr int kBN = 256;                 // accumulator columns per buffer
constexpr int kBK = 64;                  // bf16 elements per 128-byte swizzle row
constexpr int kStages = 4;
constexpr int kABytes = kBM * kBK * 2;   // 16 KB
constexpr int kBBytes = kBN * kBK * 2;   // 32 KB
constexpr int kStageBytes = kABytes + kBBytes;
constexpr int kGemmThreads = 192;
constexpr int kTmemCols = 512;
constexpr int kGemmSmemBytes = kStages * kStageBytes + 1024 /*align*/ + 256 /*barriers*/;

enum { kEpiLse = 0, kEpiDz = 1, kEpiF32 = 2 };

struct GemmArgs {
  const int* n_valid;   // device: number of compacted rows
  int M, N, K;          // extents; M or K is replaced by *n_valid when m_dyn / k_dyn
  int m_dyn, k_dyn;
  int a_off_m, a_off_k; // coordinate offsets into A's tensor map
  int b_off_n, b_off_k; // coordinate offsets into B's tensor map
  int n_per_unit;       // consecutive N tiles one CTA walks as one work unit
  int group_m;          // raster: M tiles per group sharing the same N sweep
  unsigned* status;     // device status word

  // kEpiLse
  const int* yc;        // [M] target of each compacted row (-1: none)
  float* part_m;        // [units_n x ldp] running max (log2 units)
  float* part_s;        // [units_n x ldp] running sum of 2^(z log2e - max)
  float* zy;            // [M] logit of the target
  long ldp;

  // kEpiDz
  const float* lse;     // [M] natural log-sum-exp of each row
  const float* gcoef;   // [M] dloss/dlogp of each row
  uint16_t* dz;         // [rows x ldz] bf16 output
  long ldz;

  // kEpiF32
  float* out;           // fp32 output
  long ldo;
  int accumulate;       // 1: out += acc, 0: out = acc
  const int* row_map;   // optional: output row of accumulator row r
};

struct TileSched {
  int m_tiles, n_tiles, units_n, total, k_blocks;
};

__device__ __forceinline__ TileSched make_sched(const GemmArgs& a) {
  TileSched s;
  const int nv = *a.n_valid;
  const int M = a.m_dyn ? nv : a.M;
  const int K = a.k_dyn ? nv : a.K;
  s.m_tiles = (M + kBM - 1) / kBM;
  s.n_tiles = (a.N + kBN - 1) / kBN;
  s.units_n = (s.n_tiles + a.n_per_unit - 1) / a.n_per_unit;
  s.total = s.m_tiles * s.units_n;
  s.k_blocks = (K + kBK - 1) / kBK;
  return s;
}

// Work unit u -> (m tile, n unit).  Groups of group_m consecutive M tiles
// sweep the N units together, so the CTAs running at the same time share B
// tiles (and A tiles) in L2.
__device__ __forceinline__ void unit_coords(const GemmArgs& a, const TileSched& s, int u, int& mt,
                                            int& un) {
  const int per_group = a.group_m * s.units_n;
  const int g = u / per_group;
  const int first = g * a.group_m;
  const int gm = min(a.group_m, s.m_tiles - first);
  const int w = u - g * per_group;
  mt = first + w % gm;
  un = w / gm;
}

template <int kEpi, bool kAmn, bool kBmn>
__global__ void __launch_bounds__(kGemmThreads, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const GemmArgs args) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kStages * kStageBytes);
  uint64_t* full_bar = bars;                  // [kStages] TMA -> MMA
  uint64_t* empty_bar = bars + kStages;       // [kStages] MMA -> TMA
  uint64_t* tfull_bar = bars + 2 * kStages;   // [2] MMA -> epilogue
  uint64_t* tempty_bar = bars + 2 * kStages + 2;  // [2] epilogue -> MMA
  uint64_t* done_bar = bars + 2 * kStages + 4;    // [1] all MMAs retired
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * kStages + 5);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(smem_addr(&full_bar[i]), 1);
      mbar_init(smem_addr(&empty_bar[i]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_addr(&tfull_bar[i]), 1);
      mbar_init(smem_addr(&tempty_bar[i]), 4 * 32);
    }
    mbar_init(smem_addr(done_bar), 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
  }
  if (warp == 1) {
    tmem_alloc(smem_addr(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  const TileSched sch = make_sched(args);
  const int KB = sch.k_blocks;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int uses[kStages] = {0, 0, 0, 0};
      bool ok = true;
      for (int u = blockIdx.x; u < sch.total && ok; u += gridDim.x) {
        int mt, un;
        unit_coords(args, sch, u, mt, un);
        const int nt0 = un * args.n_per_unit;
        const int nt1 = min(sch.n_tiles, nt0 + args.n_per_unit);
        for (int nt = nt0; nt < nt1 && ok; ++nt) {
          for (int kb = 0; kb < KB; ++kb) {
            if (!mbar_wait(smem_addr(&empty_bar[stage]), phase ^ 1u, abort_flag)) {
              ok = false;
              break;
            }
            const uint32_t fb = smem_addr(&full_bar[stage]);
            mbar_arrive_expect_tx(fb, kStageBytes);
            const uint32_t sa = smem_addr(smem + stage * kStageBytes);
            const uint32_t sb = sa + kABytes;
            const int k0 = kb * kBK;
            const int m0 = mt * kBM;
            const int n0 = nt * kBN;
            if (!kAmn) {
              tma_load_2d(sa, &tmA, fb, k0 + args.a_off_k, m0 + args.a_off_m);
            } else {
#pragma unroll
              for (int j = 0; j < kBM / 64; ++j)
                tma_load_2d(sa + j * 8192, &tmA, fb, m0 + args.a_off_m + 64 * j, k0 + args.a_off_k);
            }
            if (!kBmn) {
              tma_load_2d(sb, &tmB, fb, k0 + args.b_off_k, n0 + args.b_off_n);
            } else {
#pragma unroll
              for (int j = 0; j < kBN / 64; ++j)
                tma_load_2d(sb + j * 8192, &tmB, fb, n0 + args.b_off_n + 64 * j, k0 + args.b_off_k);
            }
            ++uses[stage];
            if (++stage == kStages) {
              stage = 0;
              phase ^= 1u;
            }
          }
        }
      }
      if (!ok) {
        *abort_flag = 1;
        atomicOr(args.status, kDevTimeout);
      }
      // Let every copy this thread started land before the CTA can exit.
      for (int s = 0; s < kStages; ++s)
        if (uses[s] > 0)
          mbar_wait(smem_addr(&full_bar[s]), static_cast<uint32_t>(uses[s] - 1) & 1u, abort_flag);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(kBM, kBN, kAmn, kBmn);
      int stage = 0;
      uint32_t phase = 0;
      int tile = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < sch.total && ok; u += gridDim.x) {
        int mt, un;
        unit_coords(args, sch, u, mt, un);
        const int nt0 = un * args.n_per_unit;
        const int nt1 = min(sch.n_tiles, nt0 + args.n_per_unit);
        for (int nt = nt0; nt < nt1 && ok; ++nt) {
          if (KB == 0) continue;
          const int buf = tile & 1;
          const uint32_t use = static_cast<uint32_t>(tile >> 1);
          if (!mbar_wait(smem_addr(&tempty_bar[buf]), (use & 1u) ^ 1u, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(buf * kBN);
          for (int kb = 0; kb < KB; ++kb) {
            if (!mbar_wait(smem_addr(&full_bar[stage]), phase, abort_flag)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t sa = smem_addr(smem + stage * kStageBytes);
            const uint32_t sb = sa + kABytes;
#pragma unroll
            for (int kk = 0; kk < kBK / 16; ++kk) {
              const uint64_t ad = kAmn ? sdesc_sw128(sa + kk * 2048, 8192, 1024)
                                       : sdesc_sw128(sa + kk * 32, 16, 1024);
              const uint64_t bd = kBmn ? sdesc_sw128(sb + kk * 2048, 8192, 1024)
                                       : sdesc_sw128(sb + kk * 32, 16, 1024);
              tc_mma_bf16(d_tmem, ad, bd, idesc, (kb | kk) != 0 ? 1u : 0u);
            }
            tc_commit(smem_addr(&empty_bar[stage]));
            if (++stage == kStages) {
              stage = 0;
              phase ^= 1u;
            }
          }
          if (!ok) break;
          tc_commit(smem_addr(&tfull_bar[buf]));
          ++tile;
        }
      }
      if (!ok) {
        *abort_flag = 1;
        atomicOr(args.status, kDevTimeout);
      }
      // Retire every MMA before TMEM is released.
      tc_commit(smem_addr(done_bar));
      mbar_wait(smem_addr(done_bar), 0, abort_flag);
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int quad = warp & 3;             // TMEM lanes quad*32 .. quad*32+31
    const int row = quad * 32 + lane;      // accumulator row of this thread
    const uint32_t lane_addr = tmem_base + (static_cast<uint32_t>(quad * 32) << 16);
    const int nv = *args.n_valid;
    const int Mrows = args.m_dyn ? nv : args.M;
    const float kLog2e = 1.4426950408889634f;
    int tile = 0;
    bool ok = true;
    for (int u = blockIdx.x; u < sch.total && ok; u += gridDim.x) {
      int mt, un;
      unit_coords(args, sch, u, mt, un);
      const int nt0 = un * args.n_per_unit;
      const int nt1 = min(sch.n_tiles, nt0 + args.n_per_unit);
      const int r = mt * kBM + row;
      const bool rv = r < Mrows;

      // per-unit state of the log-softmax epilogue
      float run_m = -INFINITY, run_s = 0.f, zy_val = 0.f;
      bool found = false;
      int y = -1;
      float lse2 = 0.f, gr = 0.f;
      int orow = -1;
      if (kEpi == kEpiLse) {
        y = rv ? args.yc[r] : -1;
      } else if (kEpi == kEpiDz) {
        if (rv) {
          y = args.yc[r];
          lse2 = args.lse[r] * kLog2e;
          gr = args.gcoef[r];
        }
      } else {
        if (rv) orow = args.row_map ? args.row_map[r] : r;
      }

      for (int nt = nt0; nt < nt1; ++nt) {
        const int buf = tile & 1;
        const uint32_t use = static_cast<uint32_t>(tile >> 1);
        const bool have_acc = KB > 0;
        if (have_acc) {
          if (!mbar_wait(smem_addr(&tfull_bar[buf]), use & 1u, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
        }
        const uint32_t tbase = lane_addr + static_cast<uint32_t>(buf * kBN);
        const int col0 = nt * kBN;
#pragma unroll 1
        for (int c = 0; c < kBN / 32; ++c) {
          float v[32];
          if (have_acc) {
            tmem_ld32(tbase + c * 32, v);
          } else {
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] = 0.f;
          }
          const int cb = col0 + c * 32;
          if (kEpi == kEpiLse) {
            if (cb + 32 > args.N) {
#pragma unroll
              for (int j = 0; j < 32; ++j)
                if (cb + j >= args.N) v[j] = -INFINITY;
            }
            const unsigned off = static_cast<unsigned>(y - cb);
            if (off < 32u) {
              float t = v[0];
#pragma unroll
              for (int j = 1; j < 32; ++j) t = (off == static_cast<unsigned>(j)) ? v[j] : t;
              zy_val = t;
              found = true;
            }
            float cm = v[0];
#pragma unroll
            for (int j = 1; j < 32; ++j) cm = fmaxf(cm, v[j]);
            const float nm = fmaxf(run_m, cm * kLog2e);
            float acc = 0.f;
#pragma unroll
            for (int j = 0; j < 32; ++j) acc += fast_exp2(fmaf(v[j], kLog2e, -nm));
            run_s = run_s * fast_exp2(run_m - nm) + acc;
            run_m = nm;
          } else if (kEpi == kEpiDz) {
            const int gc = args.b_off_n + cb;  // vocabulary id of column 0 of this group
            uint32_t packed[16];
#pragma unroll
            for (int j = 0; j < 32; j += 2) {
              float d0 = -gr * fast_exp2(fmaf(v[j], kLog2e, -lse2));
              float d1 = -gr * fast_exp2(fmaf(v[j + 1], kLog2e, -lse2));
              if (gc + j == y) d0 += gr;
              if (gc + j + 1 == y) d1 += gr;
              if (cb + j >= args.N || !rv) d0 = 0.f;
              if (cb + j + 1 >= args.N || !rv) d1 = 0.f;
              packed[j / 2] = pack_bf16x2(d0, d1);
            }
            uint4* dst = reinterpret_cast<uint4*>(args.dz + static_cast<long>(r) * args.ldz + cb);
#pragma unroll
            for (int q = 0; q < 4; ++q)
              dst[q] = make_uint4(packed[4 * q], packed[4 * q + 1], packed[4 * q + 2], packed[4 * q + 3]);
          } else {
            if (rv) {
              float* dst = args.out + static_cast<long>(orow) * args.ldo + cb;
              if (cb + 32 <= args.N) {
                float4* d4 = reinterpret_cast<float4*>(dst);
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                  float4 o = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
                  if (args.accumulate) {
                    const float4 p = d4[q];
                    o.x += p.x; o.y += p.y; o.z += p.z; o.w += p.w;
                  }
                  d4[q] = o;
                }
              } else {
#pragma unroll
                for (int j = 0; j < 32; ++j)
                  if (cb + j < args.N) dst[j] = args.accumulate ? dst[j] + v[j] : v[j];
              }
            }
          }
        }
        if (have_acc) {
          tc_fence_before();
          mbar_arrive(smem_addr(&tempty_bar[buf]));
          ++tile;
        }
      }
      if (!ok) break;
      if (kEpi == kEpiLse && rv) {
        args.part_m[static_cast<long>(un) * args.ldp + r] = run_m;
        args.part_s[static_cast<long>(un) * args.ldp + r] = run_s;
        if (found) args.zy[r] = zy_val;
      }
    }
    if (!ok) {
      *abort_flag = 1;
      atomicOr(args.status, kDevTimeout);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

}  // namespace grpo
