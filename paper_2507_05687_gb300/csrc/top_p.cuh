// top_p.cuh — nucleus (top-p) truncation of the rollout draw.
//
// o_t ~ softmax(z_t / temperature) restricted to its nucleus (Holtzman et al.,
// 2020): the shortest set of the most probable tokens whose mass reaches
// top_p, with every token tied with its least probable member.  Gumbel-max
// over that set draws from the distribution renormalised on it.  The logits
// z_t are the fp32 rows the forward GEMM stored (kEpiLseZ); one CTA works on
// one row at a time and reads it a few times (the first read from HBM, the
// rest mostly from L2):
//   1. max and sum of 2^((y - max) log2 e) over y = z / temperature -> LSE;
//   2. a histogram of the probability mass, in 2^-40 fixed point (so the sums
//      do not depend on the order of the atomics), over 2048 buckets of
//      1/64 nat below the row's maximum; the bucket where the mass counted
//      from the top reaches top_p holds the threshold;
//   3. if that bucket holds more than kTopPCand logits, the same over 2048
//      finer buckets spanning the bucket's own range (repeated; a bucket
//      whose logits are all equal is taken whole: ties stay together);
//   4. the bucket's logits in shared memory: the threshold y* is the largest
//      candidate y with (mass above the bucket) + (candidate mass >= y)
//      >= target;
//   5. the argmax over y >= y* of y + G (Philox4x32-10 word v mod 4 of counter
//      (v div 4, t, offset), key seed; the same noise and the same fp32
//      operations as the sampling GEMM's epilogue, so top_p = 1 draws the
//      same tokens), the lowest v on ties.
// Every reduction has a fixed order, so a row's draw is deterministic.
#pragma once

#include <stdint.h>

#include "ptx.cuh"

namespace grpo {

constexpr int kTopPThreads = 512;
constexpr int kTopPBuckets = 2048;
constexpr int kTopPCand = 1024;    // candidates resolved exactly in shared memory
constexpr int kTopPLevels = 6;     // histogram levels before the candidates fit

struct TopPShared {
  unsigned long long hist[kTopPBuckets];
  unsigned cnt[kTopPBuckets];
  float cy[kTopPCand];
  unsigned long long cq[kTopPCand];
  float lvl_hi[kTopPLevels];
  float lvl_scale[kTopPLevels];
  int lvl_b[kTopPLevels];
  float rf[kTopPThreads / 32], rg[kTopPThreads / 32];
  int ri[kTopPThreads / 32];
  unsigned long long cum_before, target;
  unsigned ncand;
  int nlvl, mode;  // mode: 0 histogram again, 1 collect candidates, 2 threshold found
  float ystar;
};

// Probability of tempered logit y in 2^-40 units (truncated).
__device__ __forceinline__ unsigned long long top_p_mass(float y, float lse) {
  const float kLog2e = 1.4426950408889634f;
  return __float2ull_rz(fast_exp2((y - lse) * kLog2e) * 1099511627776.0f);
}

__device__ __forceinline__ int top_p_bucket(float y, float hi, float scale) {
  return static_cast<int>(fminf((hi - y) * scale, static_cast<float>(kTopPBuckets - 1)));
}

// True when y lies in the chosen bucket of every one of the first n levels.
__device__ __forceinline__ bool top_p_in(const TopPShared& sh, float y, int n) {
  for (int l = 0; l < n; ++l)
    if (top_p_bucket(y, sh.lvl_hi[l], sh.lvl_scale[l]) != sh.lvl_b[l]) return false;
  return true;
}

// Block-wide max of v (every thread gets it).
__device__ __forceinline__ float top_p_block_max(TopPShared& sh, float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  const int w = threadIdx.x >> 5;
  __syncthreads();
  if ((threadIdx.x & 31) == 0) sh.rf[w] = v;
  __syncthreads();
  float r = sh.rf[0];
  for (int i = 1; i < kTopPThreads / 32; ++i) r = fmaxf(r, sh.rf[i]);
  return r;
}

// Block-wide min of v (every thread gets it).
__device__ __forceinline__ float top_p_block_min(TopPShared& sh, float v) {
  return -top_p_block_max(sh, -v);
}

__global__ void __launch_bounds__(kTopPThreads)
    top_p_kernel(const float* __restrict__ z, int64_t ldz, int V, const int* __restrict__ n_valid,
                 const int* __restrict__ cidx, float inv_temp, float top_p, uint32_t seed_lo, uint32_t seed_hi,
                 uint32_t off_lo, uint32_t off_hi, int32_t* __restrict__ tokens, float* __restrict__ logp,
                 unsigned* status) {
  const float kLog2e = 1.4426950408889634f;
  const float kLn2 = 0.69314718055994531f;
  __shared__ TopPShared sh;
  const int tid = threadIdx.x;
  const int nv = *n_valid;
  for (int r = blockIdx.x; r < nv; r += gridDim.x) {
    const float* zr = z + static_cast<int64_t>(r) * ldz;
    // 1. row maximum and sum of exponentials (online), fixed-order merge
    float m = -INFINITY, s = 0.f;
    for (int v = tid; v < V; v += kTopPThreads) {
      const float y = zr[v] * inv_temp;
      if (y > m) {
        s = s * fast_exp2((m - y) * kLog2e) + 1.f;
        m = y;
      } else {
        s += fast_exp2((y - m) * kLog2e);
      }
    }
    const float ymax = top_p_block_max(sh, m);
    float sc = m == -INFINITY ? 0.f : s * fast_exp2((m - ymax) * kLog2e);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sc += __shfl_xor_sync(0xffffffffu, sc, o);
    __syncthreads();
    if ((tid & 31) == 0) sh.rg[tid >> 5] = sc;
    __syncthreads();
    float ssum = 0.f;
    for (int i = 0; i < kTopPThreads / 32; ++i) ssum += sh.rg[i];
    const float lse = ymax + __log2f(ssum) * kLn2;

    // 2-4. the threshold y*
    if (tid == 0) {
      sh.nlvl = 0;
      sh.cum_before = 0ull;
      sh.mode = top_p >= 1.f ? 2 : 0;
      sh.ystar = -INFINITY;
      sh.lvl_hi[0] = ymax;
      sh.lvl_scale[0] = 64.f;
    }
    __syncthreads();
    while (sh.mode == 0) {
      const int L = sh.nlvl;
      for (int b = tid; b < kTopPBuckets; b += kTopPThreads) {
        sh.hist[b] = 0ull;
        sh.cnt[b] = 0u;
      }
      __syncthreads();
      const float hi = sh.lvl_hi[L], scale = sh.lvl_scale[L];
      for (int v = tid; v < V; v += kTopPThreads) {
        const float y = zr[v] * inv_temp;
        if (top_p_in(sh, y, L)) {
          const int b = top_p_bucket(y, hi, scale);
          atomicAdd(&sh.hist[b], top_p_mass(y, lse));
          atomicAdd(&sh.cnt[b], 1u);
        }
      }
      __syncthreads();
      if (tid == 0) {
        if (L == 0) {
          unsigned long long tot = 0ull;
          for (int b = 0; b < kTopPBuckets; ++b) tot += sh.hist[b];
          const double want = ceil(static_cast<double>(top_p) * static_cast<double>(tot));
          unsigned long long t = static_cast<unsigned long long>(want);
          sh.target = t < 1ull ? 1ull : (t > tot ? tot : t);
        }
        unsigned long long acc = sh.cum_before;
        int b = 0;
        for (; b < kTopPBuckets - 1; ++b) {
          if (acc + sh.hist[b] >= sh.target) break;
          acc += sh.hist[b];
        }
        sh.cum_before = acc;
        sh.lvl_b[L] = b;
        sh.nlvl = L + 1;
        sh.mode = sh.cnt[b] <= static_cast<unsigned>(kTopPCand) ? 1 : 0;
      }
      __syncthreads();
      if (sh.mode == 0) {
        // too many logits in the bucket: refine over its own range, or take it whole if they are equal
        float lo = INFINITY, hi2 = -INFINITY;
        for (int v = tid; v < V; v += kTopPThreads) {
          const float y = zr[v] * inv_temp;
          if (top_p_in(sh, y, L + 1)) {
            lo = fminf(lo, y);
            hi2 = fmaxf(hi2, y);
          }
        }
        lo = top_p_block_min(sh, lo);
        hi2 = top_p_block_max(sh, hi2);
        __syncthreads();
        if (tid == 0) {
          if (!(hi2 > lo) || L + 1 >= kTopPLevels) {
            sh.ystar = lo;  // all equal (or out of levels: the whole bucket)
            sh.mode = 2;
            if (hi2 > lo) atomicOr(status, kDevNonFinite);
          } else {
            sh.lvl_hi[L + 1] = hi2;
            sh.lvl_scale[L + 1] = static_cast<float>(kTopPBuckets - 1) / (hi2 - lo);
          }
        }
        __syncthreads();
      }
    }
    if (sh.mode == 1) {
      if (tid == 0) sh.ncand = 0u;
      __syncthreads();
      const int n = sh.nlvl;
      for (int v = tid; v < V; v += kTopPThreads) {
        const float y = zr[v] * inv_temp;
        if (top_p_in(sh, y, n)) {
          const unsigned i = atomicAdd(&sh.ncand, 1u);
          if (i < static_cast<unsigned>(kTopPCand)) {
            sh.cy[i] = y;
            sh.cq[i] = top_p_mass(y, lse);
          }
        }
      }
      __syncthreads();
      const int nc = min(static_cast<int>(sh.ncand), kTopPCand);
      float best = -INFINITY;
      for (int i = tid; i < nc; i += kTopPThreads) {
        const float yi = sh.cy[i];
        unsigned long long above = 0ull;
        for (int j = 0; j < nc; ++j) above += sh.cy[j] >= yi ? sh.cq[j] : 0ull;
        if (sh.cum_before + above >= sh.target) best = fmaxf(best, yi);
      }
      best = top_p_block_max(sh, best);
      if (tid == 0) sh.ystar = best;
      __syncthreads();
    }
    const float ystar = sh.ystar;

    // 5. Gumbel-max over y >= y*, the lowest v on ties
    const int t = cidx[r];
    float bs = -INFINITY, by = 0.f;
    int bv = -1;
    for (int g = tid; 4 * g < V; g += kTopPThreads) {
      const uint4 w = philox4x32_10(make_uint4(static_cast<uint32_t>(g), static_cast<uint32_t>(t), off_lo, off_hi),
                                    seed_lo, seed_hi);
      const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int v = 4 * g + k;
        if (v < V) {
          const float y = zr[v] * inv_temp;
          if (y >= ystar) {
            const float sc2 = y + gumbel_of(ws[k]);
            if (sc2 > bs) {
              bs = sc2;
              bv = v;
              by = y;
            }
          }
        }
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float os = __shfl_xor_sync(0xffffffffu, bs, o);
      const int ov = __shfl_xor_sync(0xffffffffu, bv, o);
      const float oy = __shfl_xor_sync(0xffffffffu, by, o);
      if (os > bs || (os == bs && ov >= 0 && (bv < 0 || ov < bv))) {
        bs = os;
        bv = ov;
        by = oy;
      }
    }
    __syncthreads();
    if ((tid & 31) == 0) {
      sh.rf[tid >> 5] = bs;
      sh.ri[tid >> 5] = bv;
      sh.rg[tid >> 5] = by;
    }
    __syncthreads();
    if (tid == 0) {
      for (int i = 1; i < kTopPThreads / 32; ++i) {
        const float os = sh.rf[i];
        const int ov = sh.ri[i];
        if (os > bs || (os == bs && ov >= 0 && (bv < 0 || ov < bv))) {
          bs = os;
          bv = ov;
          by = sh.rg[i];
        }
      }
      if (!isfinite(lse) || bv < 0) atomicOr(status, kDevNonFinite);
      tokens[t] = bv;
      logp[t] = by - lse;
    }
    __syncthreads();
  }
}

// Masked rows (and rows past the workspace's row capacity) of a top-p draw: token -1, log-prob 0.
__global__ void top_p_fill_kernel(const uint8_t* __restrict__ mask, const int* __restrict__ rank_of, int64_t T,
                                  int32_t* __restrict__ tokens, float* __restrict__ logp) {
  for (int64_t t = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; t < T;
       t += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    if (!mask[t] || rank_of[t] < 0) {
      tokens[t] = -1;
      logp[t] = 0.f;
    }
  }
}

}  // namespace grpo
