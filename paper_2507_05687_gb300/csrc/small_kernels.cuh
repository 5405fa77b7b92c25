// small_kernels.cuh — the O(T) kernels around the LM-head GEMMs:
// group advantages (Eq. 2), compaction of unmasked rows, the merge of the
// per-split log-sum-exp partials, the per-token loss terms of Eq. 1 with
// their derivative in logp, and the deterministic loss reduction.
#pragma once

#include <stdint.h>

#include "dz_rows.cuh"
#include "ptx.cuh"

namespace grpo {

constexpr int kScanChunk = 4096;   // tokens per block in the compaction kernels
constexpr int kScanThreads = 256;  // 16 tokens per thread
static_assert(kScanChunk == kScanThreads * 16, "one chunk per block of the compaction kernels");

// ------------------------------------------------------------------ Eq. 2

// fp64 sum over the lanes of one aligned segment of `width` lanes (power of 2).
__device__ __forceinline__ double seg_sum(double x, int width) {
  for (int o = width >> 1; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
}

// G a power of two <= 32: each warp holds 32/G groups, one reward per lane,
// and reduces each group with shuffles inside its G-lane segment.
__global__ void adv_segmented_kernel(const float* __restrict__ r, int64_t n, int G, float eps,
                                     float* __restrict__ adv) {
  const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  const int64_t base = i - (threadIdx.x & 31);
  if (base >= n) return;  // whole warp out of range (n % G == 0, groups never straddle warps)
  const bool in = i < n;
  const double x = in ? static_cast<double>(r[i]) : 0.0;
  const double mean = seg_sum(x, G) / G;
  const double d = in ? x - mean : 0.0;
  const double var = seg_sum(d * d, G) / (G - 1);
  const double sd = sqrt(var);
  if (in) adv[i] = static_cast<float>(d / (sd + static_cast<double>(eps)));
}

// Any G: one warp per group, lanes stride over its members.
__global__ void adv_warp_kernel(const float* __restrict__ r, int64_t n_groups, int G, float eps,
                                float* __restrict__ adv) {
  const int64_t g = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (g >= n_groups) return;
  const float* rg = r + g * G;
  double s = 0.0;
  for (int j = lane; j < G; j += 32) s += static_cast<double>(rg[j]);
  const double mean = seg_sum(s, 32) / G;
  double q = 0.0;
  for (int j = lane; j < G; j += 32) {
    const double d = static_cast<double>(rg[j]) - mean;
    q += d * d;
  }
  const double sd = sqrt(seg_sum(q, 32) / (G - 1));
  for (int j = lane; j < G; j += 32)
    adv[g * G + j] = static_cast<float>((static_cast<double>(rg[j]) - mean) / (sd + static_cast<double>(eps)));
}

// ------------------------------------------------------------------ compaction

__device__ __forceinline__ int block_exclusive_scan(int v, int* sh /*[32]*/, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) sh[warp] = x;
  __syncthreads();
  if (warp == 0) {
    const int nw = blockDim.x >> 5;
    int w = lane < nw ? sh[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    if (lane < nw) sh[lane] = w;  // inclusive warp totals
  }
  __syncthreads();
  const int before = (warp > 0 ? sh[warp - 1] : 0) + x - v;
  *total = sh[(blockDim.x >> 5) - 1];
  __syncthreads();
  return before;
}

// counts[b] = number of unmasked rows in chunk b.
__global__ void mask_count_kernel(const uint8_t* __restrict__ mask, int64_t T, int* __restrict__ counts) {
  __shared__ int sh[32];
  const int64_t base = static_cast<int64_t>(blockIdx.x) * kScanChunk + threadIdx.x * 16;
  int c = 0;
#pragma unroll
  for (int j = 0; j < 16; ++j) c += (base + j < T && mask[base + j] != 0) ? 1 : 0;
  int total;
  block_exclusive_scan(c, sh, &total);
  if (threadIdx.x == 0) counts[blockIdx.x] = total;
}

// Single block: offsets[b] = sum of counts before b; *n_valid = grand total.
// n_valid = the number of unmasked rows, clamped to the workspace's row
// capacity `cap` (kDevCapacity is set when it had to be clamped).
__global__ void count_scan_kernel(const int* __restrict__ counts, int nb, int* __restrict__ offsets,
                                  int* __restrict__ n_valid, int cap, unsigned* status) {
  __shared__ int sh[32];
  int carry = 0;
  for (int b0 = 0; b0 < nb; b0 += blockDim.x) {
    const int b = b0 + threadIdx.x;
    const int v = b < nb ? counts[b] : 0;
    int total;
    const int ex = block_exclusive_scan(v, sh, &total);
    if (b < nb) offsets[b] = carry + ex;
    carry += total;
  }
  if (threadIdx.x == 0) {
    *n_valid = min(carry, cap);
    if (carry > cap) atomicOr(status, kDevCapacity);
  }
}

// cidx[rank] = t for unmasked rows; rank_of[t] = rank or -1.
__global__ void mask_scatter_kernel(const uint8_t* __restrict__ mask, int64_t T,
                                    const int* __restrict__ offsets, int cap, int* __restrict__ cidx,
                                    int* __restrict__ rank_of) {
  __shared__ int sh[32];
  const int64_t base = static_cast<int64_t>(blockIdx.x) * kScanChunk + threadIdx.x * 16;
  uint32_t bits = 0;
  int c = 0;
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    const bool m = base + j < T && mask[base + j] != 0;
    bits |= (m ? 1u : 0u) << j;
    c += m ? 1 : 0;
  }
  int total;
  int pos = offsets[blockIdx.x] + block_exclusive_scan(c, sh, &total);
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    const int64_t t = base + j;
    if (t < T) {
      if (bits & (1u << j)) {
        // rows past the capacity get no compacted row (their outputs are 0
        // and the status word carries kDevCapacity)
        if (pos < cap) cidx[pos] = static_cast<int>(t);
        rank_of[t] = pos < cap ? pos : -1;
        ++pos;
      } else {
        rank_of[t] = -1;
      }
    }
  }
}

// The three kernels above in one block, for batches of at most kScanChunk
// rows (a decode step): the same cidx, rank_of, n_valid and capacity status,
// with two launches fewer.
__global__ void mask_compact_small_kernel(const uint8_t* __restrict__ mask, int64_t T, int cap,
                                          int* __restrict__ n_valid, int* __restrict__ cidx,
                                          int* __restrict__ rank_of, unsigned* status) {
  __shared__ int sh[32];
  const int64_t base = static_cast<int64_t>(threadIdx.x) * 16;
  uint32_t bits = 0;
  int c = 0;
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    const bool m = base + j < T && mask[base + j] != 0;
    bits |= (m ? 1u : 0u) << j;
    c += m ? 1 : 0;
  }
  int total;
  int pos = block_exclusive_scan(c, sh, &total);
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    const int64_t t = base + j;
    if (t < T) {
      if (bits & (1u << j)) {
        if (pos < cap) cidx[pos] = static_cast<int>(t);
        rank_of[t] = pos < cap ? pos : -1;
        ++pos;
      } else {
        rank_of[t] = -1;
      }
    }
  }
  if (threadIdx.x == 0) {
    *n_valid = min(total, cap);
    if (total > cap) atomicOr(status, kDevCapacity);
  }
}

// Hc[r] = H[cidx[r]] and yc[r] = targets[cidx[r]] for r < n_valid; rows
// n_valid .. round_up(n_valid, 256) are zero-filled (they feed K-loops over
// tokens and the last row tile).  One warp per row, 16-byte vectors.
__global__ void gather_rows_kernel(const uint16_t* __restrict__ H, const int32_t* __restrict__ targets,
                                   const int* __restrict__ cidx, const int* __restrict__ n_valid_p,
                                   int Hd, int64_t V, uint16_t* __restrict__ Hc, int* __restrict__ yc,
                                   unsigned* status) {
  const int nv = *n_valid_p;
  const int rows = (nv + 255) / 256 * 256;
  const int lane = threadIdx.x & 31;
  const int vec = Hd / 8;  // uint4 per row
  for (int r = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; r < rows;
       r += (gridDim.x * blockDim.x) >> 5) {
    uint4* dst = reinterpret_cast<uint4*>(Hc + static_cast<int64_t>(r) * Hd);
    if (r < nv) {
      const int t = cidx[r];
      const uint4* src = reinterpret_cast<const uint4*>(H + static_cast<int64_t>(t) * Hd);
      for (int j = lane; j < vec; j += 32) dst[j] = __ldg(src + j);
      if (lane == 0) {
        if (targets) {
          const int y = targets[t];
          const bool ok = y >= 0 && static_cast<int64_t>(y) < V;
          yc[r] = ok ? y : -1;
          if (!ok) atomicOr(status, kDevBadTarget);
        } else {
          yc[r] = -1;  // no targets (sampling)
        }
      }
    } else {
      for (int j = lane; j < vec; j += 32) dst[j] = make_uint4(0, 0, 0, 0);
      if (lane == 0) yc[r] = -1;
    }
  }
}

// |o_i|: unmasked rows of each response (for the Eq. 1 per-response mean).
__global__ void resp_len_kernel(const uint8_t* __restrict__ mask, int64_t n_resp, int64_t L,
                                int* __restrict__ len) {
  const int64_t i = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (i >= n_resp) return;
  int c = 0;
  for (int64_t j = lane; j < L; j += 32) c += mask[i * L + j] != 0;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
  if (lane == 0) len[i] = c;
}

// ------------------------------------------------------------------ merge + loss

// log-sum-exp of row r from the per-split partials (log2 units inside).
// The log-sum-exp of a row from its splits' running (max, sum) pairs:
// m = the largest max, s = the sum over splits j of ps_j 2^(pm_j - m), in one
// fixed order that a thread and a warp reach alike: 32 partial sums (partial l
// over the splits j = l, l + 32, ... in increasing j), then a butterfly over
// the partials (l + l^16 for l < 16, then l + l^8 for l < 8, ...).  Every
// merge of the same splits (log-probs, loss, sampling, the nucleus draw) gets
// the same bits.
__device__ __forceinline__ float split_term(const float* __restrict__ pm, const float* __restrict__ ps, long at,
                                            float m) {
  return __fmul_rn(ps[at], fast_exp2(pm[at] - m));
}

__device__ __forceinline__ float merge_lse(const float* __restrict__ pm, const float* __restrict__ ps,
                                           int nsplit, long ldp, int r) {
  float m = -INFINITY;
  for (int j = 0; j < nsplit; ++j) m = fmaxf(m, pm[j * ldp + r]);
  float p[32];
#pragma unroll
  for (int l = 0; l < 32; ++l) p[l] = 0.f;
  for (int j0 = 0; j0 < nsplit; j0 += 32) {
#pragma unroll
    for (int l = 0; l < 32; ++l)
      if (j0 + l < nsplit) p[l] = __fadd_rn(p[l], split_term(pm, ps, (j0 + l) * ldp + r, m));
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
#pragma unroll
    for (int l = 0; l < o; ++l) p[l] = __fadd_rn(p[l], p[l + o]);
  }
  return (m + __log2f(p[0])) * 0.6931471805599453f;
}

// merge_lse by one warp, the same value in every lane, bit for bit (lane l
// holds partial l; the butterfly runs over shuffles), with a row's splits read
// at once instead of one after another (a decode step has few rows and up to
// ~300 splits each).  Also returns the row's max m.
__device__ __forceinline__ float merge_lse_warp(const float* __restrict__ pm, const float* __restrict__ ps,
                                                int nsplit, long ldp, int r, int lane, float* m_out = nullptr) {
  float m = -INFINITY;
  for (int j = lane; j < nsplit; j += 32) m = fmaxf(m, pm[j * ldp + r]);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
  float s = 0.f;
  for (int j = lane; j < nsplit; j += 32) s = __fadd_rn(s, split_term(pm, ps, j * ldp + r, m));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s = __fadd_rn(s, __shfl_xor_sync(0xffffffffu, s, o));
  if (m_out) *m_out = m;
  return (m + __log2f(s)) * 0.6931471805599453f;
}

// logp_out[t] for every row (0 on padding and on rows with a bad target); one
// warp per row.
__global__ void logp_merge_kernel(const uint8_t* __restrict__ mask, const int* __restrict__ rank_of,
                                  int64_t T, const float* __restrict__ pm, const float* __restrict__ ps,
                                  int nsplit, long ldp, const float* __restrict__ zy,
                                  const int* __restrict__ yc, float* __restrict__ logp_out,
                                  unsigned* status) {
  const int lane = threadIdx.x & 31;
  const int64_t warps = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
  for (int64_t t = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5; t < T; t += warps) {
    float out = 0.f;
    const int r = mask[t] ? rank_of[t] : -1;
    if (r >= 0) {
      const float lse = merge_lse_warp(pm, ps, nsplit, ldp, r, lane);
      if (lane == 0 && !isfinite(lse)) atomicOr(status, kDevNonFinite);
      out = yc[r] >= 0 ? zy[r] - lse : 0.f;
    }
    if (lane == 0) logp_out[t] = out;
  }
}

// The sampled token of every row: the split with the best perturbed score
// (the lowest split on a tie, i.e. the lowest column), and its log-prob under
// softmax(z / temperature).  Masked rows: token -1, log-prob 0.
// The sampler's noise G_{t,v} for a [rows x cols] block: one thread per group
// of 4 columns (one Philox call), grid-stride over the block.
__global__ void gumbel_noise_kernel(uint32_t seed_lo, uint32_t seed_hi, uint32_t off_lo, uint32_t off_hi,
                                    int64_t row0, int64_t rows, int64_t cols, float* __restrict__ out) {
  const int64_t groups = (cols + 3) / 4;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < rows * groups;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t t = i / groups;
    const int64_t g = i - t * groups;
    const uint4 w = philox4x32_10(
        make_uint4(static_cast<uint32_t>(g), static_cast<uint32_t>(row0 + t), off_lo, off_hi), seed_lo, seed_hi);
    const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int64_t v = 4 * g + k;
      if (v < cols) out[t * cols + v] = gumbel_of(ws[k]);
    }
  }
}

__global__ void sample_merge_kernel(const uint8_t* __restrict__ mask, const int* __restrict__ rank_of, int64_t T,
                                    const float* __restrict__ pm, const float* __restrict__ ps,
                                    const float* __restrict__ bs, const int* __restrict__ bc,
                                    const float* __restrict__ bz, int nsplit, long ldp,
                                    int32_t* __restrict__ tokens, float* __restrict__ logp, unsigned* status) {
  // one warp per row: the best score over the splits (the lowest split on a tie), then the LSE
  const int lane = threadIdx.x & 31;
  const int64_t warps = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
  for (int64_t t = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5; t < T; t += warps) {
    int tok = -1;
    float lp = 0.f;
    const int r = mask[t] ? rank_of[t] : -1;
    if (r >= 0) {
      float best = -INFINITY;
      int jb = nsplit;
      for (int j = lane; j < nsplit; j += 32) {
        const float sc = bs[j * ldp + r];
        if (sc > best) {  // a lane's splits in increasing order: its lowest on a tie
          best = sc;
          jb = j;
        }
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const float ob = __shfl_xor_sync(0xffffffffu, best, o);
        const int oj = __shfl_xor_sync(0xffffffffu, jb, o);
        if (ob > best || (ob == best && oj < jb)) {
          best = ob;
          jb = oj;
        }
      }
      const float z = jb < nsplit ? bz[jb * ldp + r] : 0.f;
      tok = jb < nsplit ? bc[jb * ldp + r] : -1;
      const float lse = merge_lse_warp(pm, ps, nsplit, ldp, r, lane);
      if (lane == 0 && (!isfinite(lse) || tok < 0)) atomicOr(status, kDevNonFinite);
      lp = z - lse;
    }
    if (lane == 0) {
      tokens[t] = tok;
      logp[t] = lp;
    }
  }
}

// Per-token terms of Eq. 1 over compacted rows: lse_c, g_c (dloss/dlogp) and
// one fp64 partial sum of w_t l_t per block (fixed order, no atomics).
__global__ void loss_terms_kernel(const int* __restrict__ cidx, const int* __restrict__ n_valid_p,
                                  const float* __restrict__ pm, const float* __restrict__ ps,
                                  int nsplit, long ldp, const float* __restrict__ zy,
                                  const int* __restrict__ yc, const float* __restrict__ old_logp,
                                  const float* __restrict__ ref_logp, const float* __restrict__ adv,
                                  int64_t L, const int* __restrict__ resp_len, int64_t n_resp,
                                  int agg_mode, float norm, float clip_eps, float beta, float kl_clamp,
                                  float* __restrict__ lse_c, float* __restrict__ g_c,
                                  double* __restrict__ block_loss, unsigned* status) {
  __shared__ double sh[32];
  const int nv = *n_valid_p;
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  double contrib = 0.0;
  if (r < nv) {
    const int t = cidx[r];
    const int64_t i = t / L;
    float lse = merge_lse(pm, ps, nsplit, ldp, r);
    if (!isfinite(lse)) atomicOr(status, kDevNonFinite);
    const bool yok = yc[r] >= 0;
    float g = 0.f;
    if (yok && isfinite(lse)) {
      const float logp = zy[r] - lse;
      const float A = adv[i];
      const float rho = __expf(logp - old_logp[t]);
      const float s1 = rho * A;
      const float s2 = fminf(fmaxf(rho, 1.f - clip_eps), 1.f + clip_eps) * A;
      const bool unclipped = s1 <= s2;
      const float s = unclipped ? s1 : s2;
      const float dref = ref_logp[t] - logp;
      const float e = __expf(dref);
      const float k3 = e - dref - 1.f;
      // capped KL: above the cap the value is the cap and the slope 0 (a tie is inside;
      // an infinite cap leaves every value, NaN included, as it is)
      const bool kl_in = !(k3 > kl_clamp);
      const float kl = kl_in ? k3 : kl_clamp;
      const float ell = -s + beta * kl;
      // norm > 0 replaces the local count (N_valid, or n_resp) by a global one
      const float w = agg_mode == 0
                          ? 1.f / (norm > 0.f ? norm : static_cast<float>(nv))
                          : 1.f / ((norm > 0.f ? norm : static_cast<float>(n_resp)) * static_cast<float>(resp_len[i]));
      g = w * ((unclipped ? -A * rho : 0.f) + (kl_in ? beta * (1.f - e) : 0.f));
      contrib = static_cast<double>(w) * static_cast<double>(ell);
    } else {
      lse = 0.f;
    }
    lse_c[r] = lse;
    g_c[r] = g;
  }
  // block reduction in a fixed order
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) contrib += __shfl_xor_sync(0xffffffffu, contrib, o);
  if ((threadIdx.x & 31) == 0) sh[threadIdx.x >> 5] = contrib;
  __syncthreads();
  if (threadIdx.x < 32) {
    double x = threadIdx.x < (blockDim.x >> 5) ? sh[threadIdx.x] : 0.0;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    if (threadIdx.x == 0) block_loss[blockIdx.x] = x;
  }
}

// Single block: loss = sum of the block partials, in block order.
__global__ void loss_final_kernel(const double* __restrict__ block_loss, const int* __restrict__ n_valid_p,
                                  int threads_per_block, float* __restrict__ loss_out) {
  __shared__ double sh[32];
  const int nb = (*n_valid_p + threads_per_block - 1) / threads_per_block;
  double x = 0.0;
  for (int b = threadIdx.x; b < nb; b += blockDim.x) x += block_loss[b];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  if ((threadIdx.x & 31) == 0) sh[threadIdx.x >> 5] = x;
  __syncthreads();
  if (threadIdx.x < 32) {
    double y = threadIdx.x < (blockDim.x >> 5) ? sh[threadIdx.x] : 0.0;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) y += __shfl_xor_sync(0xffffffffu, y, o);
    if (threadIdx.x == 0) *loss_out = static_cast<float>(y);
  }
}

// One AdamW step over n contiguous fp32 elements (n % 4 == 0), 16-byte vectors,
// grid-stride: theta, m, v updated in place from the gradient g, bf16 copy out.
__global__ void adamw_kernel(float* __restrict__ theta, float* __restrict__ m, float* __restrict__ v,
                             const float* __restrict__ g, uint16_t* __restrict__ w_out, int64_t n4, float b1,
                             float b2, float eps, float lr, float decay, float bc1, float bc2) {
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n4;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    float4 t = __ldcs(reinterpret_cast<float4*>(theta) + i);
    float4 mm = __ldcs(reinterpret_cast<float4*>(m) + i);
    float4 vv = __ldcs(reinterpret_cast<float4*>(v) + i);
    const float4 gg = __ldcs(reinterpret_cast<const float4*>(g) + i);
    float* tp = &t.x;
    float* mp = &mm.x;
    float* vp = &vv.x;
    const float* gp = &gg.x;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      mp[k] = b1 * mp[k] + (1.f - b1) * gp[k];
      vp[k] = b2 * vp[k] + (1.f - b2) * gp[k] * gp[k];
      tp[k] = tp[k] * decay - lr * (mp[k] * bc1) / (sqrtf(vp[k] * bc2) + eps);
    }
    __stcs(reinterpret_cast<float4*>(theta) + i, t);
    __stcs(reinterpret_cast<float4*>(m) + i, mm);
    __stcs(reinterpret_cast<float4*>(v) + i, vv);
    reinterpret_cast<uint2*>(w_out)[i] = make_uint2(pack_bf16x2(t.x, t.y), pack_bf16x2(t.z, t.w));
  }
}

// The K-major copy of the gathered hidden states for the dW GEMM, for the
// rows r < round_up(n_valid, 256) that the token K-loop can reach (zero past
// n_valid): with ld_t > 0 plain rows, HcT[k][r] = Hc[r][k] (row stride ld_t);
// with ld_t == 0 k-blocks of 64 tokens, HcT[r / 64][k][r % 64] = Hc[r][k], where
// a GEMM stage is one contiguous run however long the rows are.  64 x 64 tiles
// through shared memory, 32-bit words (two bf16) on both sides.
__global__ void transpose_rows_kernel(const uint16_t* __restrict__ Hc, const int* __restrict__ n_valid_p, int Hd,
                                      int64_t ld_t, uint16_t* __restrict__ HcT) {
  __shared__ uint16_t tile[64][66];
  const int nv = *n_valid_p;
  const int rows = (nv + 255) / 256 * 256;
  const int col_tiles = Hd / 64;
  const int64_t tiles = static_cast<int64_t>(rows / 64) * col_tiles;
  const int w = threadIdx.x & 31;
  const int q = threadIdx.x >> 5;  // 0..7
  for (int64_t i = blockIdx.x; i < tiles; i += gridDim.x) {
    const int r0 = static_cast<int>(i / col_tiles) * 64;
    const int c0 = static_cast<int>(i % col_tiles) * 64;
#pragma unroll
    for (int k = 0; k < 8; ++k) {  // rows r0 + q + 8k, columns c0 + 2w, 2w + 1
      const int r = q + 8 * k;
      const uint32_t v = *reinterpret_cast<const uint32_t*>(Hc + static_cast<int64_t>(r0 + r) * Hd + c0 + 2 * w);
      tile[r][2 * w] = static_cast<uint16_t>(v & 0xFFFFu);
      tile[r][2 * w + 1] = static_cast<uint16_t>(v >> 16);
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < 8; ++k) {  // rows c0 + q + 8k, tokens r0 + 2w, 2w + 1
      const int c = q + 8 * k;
      const uint32_t v = static_cast<uint32_t>(tile[2 * w][c]) | (static_cast<uint32_t>(tile[2 * w + 1][c]) << 16);
      const int64_t at = ld_t > 0 ? static_cast<int64_t>(c0 + c) * ld_t + r0 + 2 * w
                                  : static_cast<int64_t>(r0) * Hd + static_cast<int64_t>(c0 + c) * 64 + 2 * w;
      *reinterpret_cast<uint32_t*>(HcT + at) = v;
    }
    __syncthreads();
  }
}

// dH[t] = dHc[rank_of[t]] for unmasked rows, 0 for padding rows: one warp per
// row, 16-byte accesses (the compacted rows are read once).
__global__ void dh_rows_kernel(const int* __restrict__ rank_of, int64_t T, int Hd, const float* __restrict__ dHc,
                               float* __restrict__ dH) {
  const int lane = threadIdx.x & 31;
  const int vec = Hd / 4;
  for (int64_t t = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5; t < T;
       t += (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5) {
    const int r = rank_of[t];
    float4* row = reinterpret_cast<float4*>(dH + t * Hd);
    if (r < 0) {
      for (int j = lane; j < vec; j += 32) __stcs(row + j, make_float4(0.f, 0.f, 0.f, 0.f));
    } else {
      const float4* src = reinterpret_cast<const float4*>(dHc + static_cast<int64_t>(r) * Hd);
      int j = lane;
      for (; j + 96 < vec; j += 128) {  // four 16-byte loads in flight per lane
        const float4 a = __ldcs(src + j), b = __ldcs(src + j + 32), c = __ldcs(src + j + 64),
                     d = __ldcs(src + j + 96);
        __stcs(row + j, a);
        __stcs(row + j + 32, b);
        __stcs(row + j + 64, c);
        __stcs(row + j + 96, d);
      }
      for (; j < vec; j += 32) __stcs(row + j, __ldcs(src + j));
    }
  }
}

// dZ chunk from the logits the forward GEMM stored (kEpiLseZ): dz_rows with
// one block per row at a time.
__global__ void dz_from_logits_kernel(const float* __restrict__ z, int64_t ldz, const float* __restrict__ lse,
                                      const float* __restrict__ gcoef, const int* __restrict__ yc,
                                      const int* __restrict__ n_valid, int64_t rows_cap, int64_t c0, int width,
                                      int vc, uint16_t* __restrict__ dz) {
  dz_rows(z, ldz, lse, gcoef, yc, *n_valid, rows_cap, c0, width, vc, dz, blockIdx.x, gridDim.x, threadIdx.x,
          blockDim.x);
}

}  // namespace grpo
