// top_p.cuh — nucleus (top-p) truncation of the rollout draw.
//
// o_t ~ softmax(z_t / temperature) restricted to its nucleus (Holtzman et al.,
// 2020): the shortest set of the most probable tokens whose mass reaches
// top_p, with every token tied with its least probable member.  Gumbel-max
// over that set draws from the distribution renormalised on it.
//
// The sampling GEMM (kEpiSampleZ) has already produced, per row, the log-sum-
// exp of y = z / temperature, the row maximum and the plain Gumbel-max winner
// over the whole vocabulary, and stored the fp32 logits z.  For a row whose
// plain winner falls outside the nucleus (see below):
//   1. a histogram of the probability mass, in 2^-40 fixed point (so the sums
//      do not depend on the order of the atomics), over 2048 buckets of
//      1/64 nat below the row maximum; the bucket where the mass counted from
//      the top reaches top_p holds the threshold;
//   2. that bucket's logits gathered in shared memory and sorted: the threshold
//      y* is the first y (largest first) at which the mass above the bucket
//      plus the running mass reaches the target; a bucket with more than
//      kTopPCand logits is histogrammed
//      again over its own range first (one whose logits are all equal is taken
//      whole: ties stay together);
//   3. the argmax over y >= y* of y + G with the GEMM's noise (Philox4x32-10
//      word v mod 4 of counter (v div 4, t, offset), key seed) and fp32
//      operations, the lowest v on ties.
// Before any of that, a pass with one CTA per row (top_p_fast_kernel) decides
// whether the plain winner w0 (the GEMM's argmax over the whole vocabulary,
// already written to the outputs by top_p_prep_kernel) is in the nucleus: it
// is exactly when the mass of the logits strictly above y_w0 is below the
// target (then y_w0 >= y*; otherwise the tokens above it already reach the
// target and y* > y_w0).  A winner inside is the nucleus winner too, its
// perturbed score beating every token; that is the case for about a fraction
// top_p of the rows.  Only the others go through steps 1-3 (top_p_kernel), and
// top_p = 1 needs neither kernel.
//
// A row of the remaining list is shared by a cluster of kTopPCtas CTAs
// (distributed shared memory): each walks an interleaved eighth of the row, and
// CTA 0 of the cluster holds the merged histogram, candidates and decisions,
// which the others read back after a cluster barrier.
// Every reduction has a fixed order, so a row's draw is deterministic.
#pragma once

#include <stdint.h>

#include "ptx.cuh"
#include "small_kernels.cuh"

namespace grpo {

constexpr int kTopPThreads = 256;
constexpr int kTopPCtas = 8;       // CTAs of a cluster sharing one row
constexpr int kTopPBuckets = 2048;
constexpr int kTopPCand = 1024;    // candidates resolved exactly in shared memory
constexpr int kTopPLevels = 6;     // histogram levels before the candidates fit
constexpr int kTopPWarps = kTopPThreads / 32;
static_assert(kTopPBuckets == kTopPCtas * kTopPThreads, "one histogram bucket per thread of the cluster in the merge");

// Shared memory of one CTA.  The fields marked "host" are used in CTA 0 of
// the cluster only (the other CTAs write into and read from CTA 0's copy).
struct TopPShared {
  unsigned long long hist[kTopPBuckets];   // this CTA's histogram; host: then the merged one
  float cy[kTopPCand];                     // host: the gathered candidates
  unsigned long long cq[kTopPCand];
  float ly[kTopPCand];                     // this CTA's candidates before they go to the host
  unsigned long long lq[kTopPCand];
  unsigned long long scan[kTopPThreads];   // host: per-thread bucket-range sums of the scan
  uint32_t slot_f[kTopPCtas], slot_g[kTopPCtas], slot_i[kTopPCtas];  // host: one partial per CTA
  float lvl_hi[kTopPLevels];
  float lvl_scale[kTopPLevels];
  int lvl_b[kTopPLevels];
  unsigned long long ra[kTopPWarps];
  float rf[kTopPWarps], rg[kTopPWarps];
  int ri[kTopPWarps];
  unsigned long long cum_before, target;   // host, copied to every CTA
  unsigned ncand;                          // host
  unsigned lcand, lbase;                   // this CTA's candidate count and its offset at the host
  float lse, y0, ystar;
  int nlvl;
  int mode;  // 0 histogram, 1 resolve the gathered candidates, 2 threshold known
};

// Probability of tempered logit y in 2^-40 units, truncated toward zero: the
// float p * 2^40 (< 2^41) turned into an integer from its fields (significand
// shifted by the exponent), which is exact and cheaper than a 64-bit convert.
__device__ __forceinline__ unsigned long long top_p_mass(float y, float lse) {
  const float kLog2e = 1.4426950408889634f;
  const uint32_t b = __float_as_uint(fast_exp2((y - lse) * kLog2e) * 1099511627776.0f);
  const int e = static_cast<int>((b >> 23) & 0xFFu) - 150;  // value = significand * 2^e
  const unsigned long long m = static_cast<unsigned long long>((b & 0x7FFFFFu) | 0x800000u);
  if (e <= -24 || e > 40 || (b >> 31)) return 0ull;  // below 1, not finite, or negative
  return e >= 0 ? m << e : m >> (-e);
}

__device__ __forceinline__ int top_p_bucket(float y, float hi, float scale) {
  return static_cast<int>(fminf(fmaxf((hi - y) * scale, 0.f), static_cast<float>(kTopPBuckets - 1)));
}

// True when y lies in the chosen bucket of every one of the first n levels.
__device__ __forceinline__ bool top_p_in(const TopPShared& sh, float y, int n) {
  for (int l = 0; l < n; ++l)
    if (top_p_bucket(y, sh.lvl_hi[l], sh.lvl_scale[l]) != sh.lvl_b[l]) return false;
  return true;
}

// The mass the nucleus must reach, in the units of top_p_mass: top_p of the
// whole (1 = 2^40).  The fixed-point masses of a row sum to 2^40 up to their
// truncation and the fp32 LSE's rounding (a relative 1e-6 or so), which moves
// the boundary by that much mass; should they sum to less than the target,
// the nucleus is the whole vocabulary.
__device__ __forceinline__ unsigned long long top_p_target(float top_p) {
  const unsigned long long one = 1ull << 40;
  const unsigned long long t = static_cast<unsigned long long>(ceil(static_cast<double>(top_p) * 1099511627776.0));
  return t < 1ull ? 1ull : (t > one ? one : t);
}

// Block-wide max of v (every thread gets it).
__device__ __forceinline__ float top_p_block_max(TopPShared& sh, float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  __syncthreads();
  if ((threadIdx.x & 31) == 0) sh.rf[threadIdx.x >> 5] = v;
  __syncthreads();
  float r = sh.rf[0];
  for (int i = 1; i < kTopPWarps; ++i) r = fmaxf(r, sh.rf[i]);
  return r;
}

// Walks this CTA's share of the row (kShare CTAs share it; rank is this
// CTA's place among them): groups of four logits (16-byte loads; the row's
// leading dimension is a multiple of 64, so a group never leaves the row's
// storage) g = rank * kTopPThreads + tid + k * kShare * kTopPThreads, kUnroll
// groups per thread in flight; f(v, y) for every v < V.
template <int kUnroll, int kShare = kTopPCtas, typename F>
__device__ __forceinline__ void top_p_walk(const float* zr, int V, float inv_temp, int rank, F f) {
  constexpr int kStride = kShare * kTopPThreads;
  const int groups = (V + 3) / 4;
  const float4* zq = reinterpret_cast<const float4*>(zr);
  int g0 = rank * kTopPThreads + threadIdx.x;
  // whole rounds: kUnroll unconditional loads in flight, then their logits
  for (; g0 + (kUnroll - 1) * kStride < groups - 1; g0 += kUnroll * kStride) {
    float4 q[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) q[u] = __ldcg(zq + g0 + u * kStride);
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int v = 4 * (g0 + u * kStride);  // every group here lies below the last, so v + 3 < V
      f(v, q[u].x * inv_temp);
      f(v + 1, q[u].y * inv_temp);
      f(v + 2, q[u].z * inv_temp);
      f(v + 3, q[u].w * inv_temp);
    }
  }
  // the rest, one group at a time (the last group may be partial)
  for (; g0 < groups; g0 += kStride) {
    const float4 q = __ldcg(zq + g0);
    const int v = 4 * g0;
    const float zz[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
    for (int k = 0; k < 4; ++k)
      if (v + k < V) f(v + k, zz[k] * inv_temp);
  }
}

// The threshold among the nc gathered candidates (host CTA, every thread; the
// result in every thread): the candidates sorted by y, largest first (bitonic
// sort, padded to a power of two with -inf), their masses summed in that order
// (fixed-order block scan); y* is the y at the first position where the mass
// above the bucket plus the running sum reaches the target.  Equal logits sit
// next to each other, so y*'s whole tie group counts toward the target.
// -inf if no position does (the nucleus is then the whole vocabulary).
__device__ __forceinline__ float top_p_resolve(TopPShared& sh, int nc) {
  const int tid = threadIdx.x;
  int n = 1;
  while (n < nc) n <<= 1;  // <= kTopPCand
  for (int i = nc + tid; i < n; i += kTopPThreads) {
    sh.cy[i] = -INFINITY;
    sh.cq[i] = 0ull;
  }
  __syncthreads();
  for (int k = 2; k <= n; k <<= 1) {
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int i = tid; i < n; i += kTopPThreads) {
        const int l = i ^ j;
        if (l > i) {
          const float a = sh.cy[i], b = sh.cy[l];
          if ((i & k) == 0 ? a < b : a > b) {  // descending runs where bit k is clear
            sh.cy[i] = b;
            sh.cy[l] = a;
            const unsigned long long t = sh.cq[i];
            sh.cq[i] = sh.cq[l];
            sh.cq[l] = t;
          }
        }
      }
      __syncthreads();
    }
  }
  // running sums: thread tid owns positions [tid * per, (tid + 1) * per)
  const int per = (n + kTopPThreads - 1) / kTopPThreads;
  const int b0 = tid * per;
  unsigned long long own = 0ull;
  for (int i = b0; i < b0 + per && i < n; ++i) own += sh.cq[i];
  unsigned long long inc = own;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned long long v = __shfl_up_sync(0xffffffffu, inc, o);
    if ((tid & 31) >= o) inc += v;
  }
  if ((tid & 31) == 31) sh.ra[tid >> 5] = inc;
  __syncthreads();
  unsigned long long acc = inc - own;
  for (int w = 0; w < (tid >> 5); ++w) acc += sh.ra[w];
  const unsigned long long need = sh.target - sh.cum_before;
  int first = n;
  for (int i = b0; i < b0 + per && i < n; ++i) {
    acc += sh.cq[i];
    if (acc >= need) {
      first = i;
      break;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) first = min(first, __shfl_xor_sync(0xffffffffu, first, o));
  __syncthreads();
  if ((tid & 31) == 0) sh.ri[tid >> 5] = first;
  __syncthreads();
  for (int w = 0; w < kTopPWarps; ++w) first = min(first, sh.ri[w]);
  return first < n ? sh.cy[first] : -INFINITY;
}

// The better of two perturbed scores (the lower token on a tie; -1 loses).
__device__ __forceinline__ bool top_p_better(float s, int v, float s0, int v0) {
  return s > s0 || (s == s0 && v >= 0 && (v0 < 0 || v < v0));
}

__global__ void __cluster_dims__(kTopPCtas, 1, 1) __launch_bounds__(kTopPThreads, 4)
    top_p_kernel(const float* __restrict__ z, int64_t ldz, int V, const int* __restrict__ n_slow,
                 const int* __restrict__ slow_rows, const unsigned long long* __restrict__ slow_target,
                 const int* __restrict__ cidx, const float* __restrict__ lse_r, const float* __restrict__ y0_r,
                 const float* __restrict__ hi_r, float inv_temp, uint32_t seed_lo, uint32_t seed_hi,
                 uint32_t off_lo, uint32_t off_hi, int32_t* __restrict__ tokens, float* __restrict__ logp,
                 unsigned* status) {
  __shared__ TopPShared sh;
  const int tid = threadIdx.x;
  const int rank = static_cast<int>(cluster_ctarank());
  const bool host = rank == 0;
  const int ns = *n_slow;
  // CTA 0's copy of a field
  auto at0 = [&](const void* p) { return mapa_shared(smem_addr(p), 0); };
  for (int si = blockIdx.x / kTopPCtas; si < ns; si += gridDim.x / kTopPCtas) {
    const int r = slow_rows[si];
    const float* zr = z + static_cast<int64_t>(r) * ldz;
    const int t = cidx[r];
    if (tid == 0) {
      sh.lse = lse_r[r];
      sh.y0 = y0_r[r];
      sh.target = slow_target[si];
      sh.lvl_hi[0] = hi_r[r];  // the row maximum of y (to rounding): the top of the first level
    }
    if (tid == 0) {
      sh.nlvl = 0;
      sh.cum_before = 0ull;
      sh.ystar = -INFINITY;
      sh.mode = 0;
      sh.lvl_scale[0] = 64.f;
    }
    __syncthreads();
    const float lse = sh.lse;
    while (sh.mode == 0) {
      const int L = sh.nlvl;
      for (int b = tid; b < kTopPBuckets; b += kTopPThreads) sh.hist[b] = 0ull;
      __syncthreads();
      const float hi = sh.lvl_hi[L], scale = sh.lvl_scale[L];
      top_p_walk<4>(zr, V, inv_temp, rank, [&](int, float y) {
        if (top_p_in(sh, y, L)) {
          const unsigned long long q = top_p_mass(y, lse);
          if (q) atomicAdd(&sh.hist[top_p_bucket(y, hi, scale)], q);  // far-tail logits add nothing
        }
      });
      cluster_sync();
      {  // merge the histograms: CTA k sums buckets [k * kTopPThreads, (k + 1) * kTopPThreads) over
         // the cluster in rank order and leaves the sums in CTA 0's histogram (disjoint slices, so no
         // CTA reads a bucket another one writes)
        const int b = rank * kTopPThreads + tid;
        unsigned long long part[kTopPCtas];
#pragma unroll
        for (int k = 0; k < kTopPCtas; ++k) part[k] = ld_shared_cluster_u64(mapa_shared(smem_addr(&sh.hist[b]), k));
        unsigned long long m = 0ull;
#pragma unroll
        for (int k = 0; k < kTopPCtas; ++k) m += part[k];
        st_shared_cluster_u64(at0(&sh.hist[b]), m);
      }
      cluster_sync();
      if (host) {  // find the bucket that holds the threshold
        // the first bucket where the mass from the top reaches the target: each
        // thread sums a range of buckets, thread 0 walks the range sums and then
        // the buckets of the one range that crosses
        constexpr int kPer = kTopPBuckets / kTopPThreads;
        unsigned long long part = 0ull;
#pragma unroll
        for (int i = 0; i < kPer; ++i) part += sh.hist[tid * kPer + i];
        sh.scan[tid] = part;
        __syncthreads();
        if (tid < 32) {
          // warp 0: lane l owns segments [l * kSeg, (l + 1) * kSeg); an inclusive
          // scan of the lane sums finds the lane whose segments cross
          constexpr int kSeg = kTopPThreads / 32;
          unsigned long long own = 0ull;
#pragma unroll
          for (int i = 0; i < kSeg; ++i) own += sh.scan[tid * kSeg + i];
          unsigned long long inc = own;
#pragma unroll
          for (int o = 1; o < 32; o <<= 1) {
            const unsigned long long n = __shfl_up_sync(0xffffffffu, inc, o);
            if (tid >= o) inc += n;
          }
          const unsigned cross = __ballot_sync(0xffffffffu, sh.cum_before + inc >= sh.target);
          const int ln = cross ? __ffs(cross) - 1 : 31;
          const unsigned long long before = __shfl_sync(0xffffffffu, inc - own, ln);
          sh.ra[0] = before;
          sh.ri[0] = ln;
        }
        __syncthreads();
        if (tid == 0) {
          constexpr int kSeg = kTopPThreads / 32;
          unsigned long long acc = sh.cum_before + sh.ra[0];
          int seg = sh.ri[0] * kSeg;
          for (; seg < (sh.ri[0] + 1) * kSeg - 1; ++seg) {
            if (acc + sh.scan[seg] >= sh.target) break;
            acc += sh.scan[seg];
          }
          int b = seg * kPer;
          for (; b < (seg + 1) * kPer - 1; ++b) {
            if (acc + sh.hist[b] >= sh.target) break;
            acc += sh.hist[b];
          }
          sh.cum_before = acc;
          sh.lvl_b[L] = b;
          sh.ncand = 0u;
        }
      }
      cluster_sync();
      if (tid == 0) {
        sh.lvl_b[L] = static_cast<int>(ld_shared_cluster(at0(&sh.lvl_b[L])));
        sh.cum_before = ld_shared_cluster_u64(at0(&sh.cum_before));
        sh.nlvl = L + 1;
      }
      __syncthreads();
      // gather the bucket's logits (and their range, in case they do not fit):
      // into this CTA's buffer first, then one reservation at the host and a copy
      if (tid == 0) sh.lcand = 0u;
      __syncthreads();
      float lo = INFINITY, hi2 = -INFINITY;
      top_p_walk<4>(zr, V, inv_temp, rank, [&](int, float y) {
        if (top_p_in(sh, y, L + 1)) {
          lo = fminf(lo, y);
          hi2 = fmaxf(hi2, y);
          const unsigned i = atomicAdd(&sh.lcand, 1u);
          if (i < static_cast<unsigned>(kTopPCand)) {
            sh.ly[i] = y;
            sh.lq[i] = top_p_mass(y, lse);
          }
        }
      });
      lo = -top_p_block_max(sh, -lo);
      hi2 = top_p_block_max(sh, hi2);
      if (tid == 0) {
        st_shared_cluster(at0(&sh.slot_f[rank]), __float_as_uint(lo));
        st_shared_cluster(at0(&sh.slot_g[rank]), __float_as_uint(hi2));
        sh.lbase = atom_add_shared_cluster(at0(&sh.ncand), sh.lcand);
      }
      __syncthreads();
      {
        const unsigned n = min(sh.lcand, static_cast<unsigned>(kTopPCand));
        const unsigned base = sh.lbase;
        for (unsigned i = tid; i < n && base + i < static_cast<unsigned>(kTopPCand); i += kTopPThreads) {
          st_shared_cluster(at0(&sh.cy[base + i]), __float_as_uint(sh.ly[i]));
          st_shared_cluster_u64(at0(&sh.cq[base + i]), sh.lq[i]);
        }
      }
      cluster_sync();
      if (host) {
        const int nc = static_cast<int>(min(sh.ncand, static_cast<unsigned>(kTopPCand)));
        if (sh.ncand <= static_cast<unsigned>(kTopPCand)) {
          const float best = top_p_resolve(sh, nc);
          if (tid == 0) {
            sh.ystar = best;
            sh.mode = 2;
          }
        } else if (tid == 0) {
          float l = INFINITY, h = -INFINITY;
          for (int k = 0; k < kTopPCtas; ++k) {
            l = fminf(l, __uint_as_float(sh.slot_f[k]));
            h = fmaxf(h, __uint_as_float(sh.slot_g[k]));
          }
          if (!(h > l) || L + 1 >= kTopPLevels) {
            sh.ystar = l;  // all equal (or out of levels: the whole bucket)
            sh.mode = 2;
            if (h > l) atomicOr(status, kDevNonFinite);
          } else {
            sh.lvl_hi[L + 1] = h;
            sh.lvl_scale[L + 1] = static_cast<float>(kTopPBuckets - 1) / (h - l);
          }
        }
      }
      cluster_sync();
      if (tid == 0) {
        sh.mode = static_cast<int>(ld_shared_cluster(at0(&sh.mode)));
        sh.ystar = __uint_as_float(ld_shared_cluster(at0(&sh.ystar)));
        sh.lvl_hi[L + 1 < kTopPLevels ? L + 1 : L] =
            __uint_as_float(ld_shared_cluster(at0(&sh.lvl_hi[L + 1 < kTopPLevels ? L + 1 : L])));
        sh.lvl_scale[L + 1 < kTopPLevels ? L + 1 : L] =
            __uint_as_float(ld_shared_cluster(at0(&sh.lvl_scale[L + 1 < kTopPLevels ? L + 1 : L])));
      }
      __syncthreads();
    }
    const float ystar = sh.ystar;
    {  // the plain winner is outside the nucleus: the argmax over it
      // Gumbel-max over y >= y*, the lowest v on ties
      float bs = -INFINITY, by = 0.f;
      int bv = -1;
      const int groups = (V + 3) / 4;
      for (int g = rank * kTopPThreads + tid; g < groups; g += kTopPCtas * kTopPThreads) {
        const float4 q = __ldcg(reinterpret_cast<const float4*>(zr) + g);
        const float yy[4] = {q.x * inv_temp, q.y * inv_temp, q.z * inv_temp, q.w * inv_temp};
        if (!(yy[0] >= ystar || yy[1] >= ystar || yy[2] >= ystar || yy[3] >= ystar)) continue;
        const uint4 w = philox4x32_10(make_uint4(static_cast<uint32_t>(g), static_cast<uint32_t>(t), off_lo, off_hi),
                                      seed_lo, seed_hi);
        const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const int v = 4 * g + k;
          if (v < V && yy[k] >= ystar) {
            const float sc2 = yy[k] + gumbel_of(ws[k]);
            if (sc2 > bs) {
              bs = sc2;
              bv = v;
              by = yy[k];
            }
          }
        }
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const float os = __shfl_xor_sync(0xffffffffu, bs, o);
        const int ov = __shfl_xor_sync(0xffffffffu, bv, o);
        const float oy = __shfl_xor_sync(0xffffffffu, by, o);
        if (top_p_better(os, ov, bs, bv)) {
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
        for (int i = 1; i < kTopPWarps; ++i)
          if (top_p_better(sh.rf[i], sh.ri[i], bs, bv)) {
            bs = sh.rf[i];
            bv = sh.ri[i];
            by = sh.rg[i];
          }
        st_shared_cluster(at0(&sh.slot_f[rank]), __float_as_uint(bs));
        st_shared_cluster(at0(&sh.slot_g[rank]), __float_as_uint(by));
        st_shared_cluster(at0(&sh.slot_i[rank]), static_cast<uint32_t>(bv));
      }
      cluster_sync();
      if (host && tid == 0) {
        bs = -INFINITY;
        bv = -1;
        by = 0.f;
        for (int k = 0; k < kTopPCtas; ++k) {
          const float os = __uint_as_float(sh.slot_f[k]);
          const int ov = static_cast<int>(sh.slot_i[k]);
          if (top_p_better(os, ov, bs, bv)) {
            bs = os;
            bv = ov;
            by = __uint_as_float(sh.slot_g[k]);
          }
        }
        if (!isfinite(lse) || bv < 0) atomicOr(status, kDevNonFinite);
        tokens[t] = bv;
        logp[t] = by - lse;
      }
    }
    cluster_sync();  // the host's slots are free again before the next row
  }
}

// Per unmasked row, the plain draw from the sampling GEMM's splits: written
// to the outputs (the nucleus selection replaces it only where the winner
// falls outside the nucleus), and the row's LSE, winner's y and maximum y kept
// for the selection (whose per-row accumulators it clears).  One warp per row reads the splits in parallel; the LSE
// sum runs in split order with merge_lse's rounding, and the winner is the best
// score with the lowest split on a tie, as sample_merge_kernel takes them, so
// the draw is the plain sampler's bit for bit.
__global__ void top_p_prep_kernel(const int* __restrict__ n_valid, const int* __restrict__ cidx,
                                  const float* __restrict__ pm, const float* __restrict__ ps,
                                  const float* __restrict__ bs, const int* __restrict__ bc,
                                  const float* __restrict__ bz, int nsplit, long ldp, float* __restrict__ lse_r,
                                  float* __restrict__ y0_r, float* __restrict__ hi_r,
                                  unsigned long long* __restrict__ row_above, unsigned* __restrict__ row_done,
                                  int32_t* __restrict__ tokens, float* __restrict__ logp, unsigned* status) {
  const float kLn2 = 0.69314718055994531f;
  const int lane = threadIdx.x & 31;
  const int nv = *n_valid;
  const int warps = static_cast<int>((static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5);
  for (int r = static_cast<int>((static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5); r < nv;
       r += warps) {
    float m = -INFINITY, best = -INFINITY;
    int jb = nsplit;
    for (int j = lane; j < nsplit; j += 32) {
      m = fmaxf(m, pm[j * ldp + r]);
      const float sc = bs[j * ldp + r];
      if (sc > best) {
        best = sc;
        jb = j;
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
      const float ob = __shfl_xor_sync(0xffffffffu, best, o);
      const int oj = __shfl_xor_sync(0xffffffffu, jb, o);
      if (ob > best || (ob == best && oj < jb)) {
        best = ob;
        jb = oj;
      }
    }
    float s = 0.f;
    for (int j0 = 0; j0 < nsplit; j0 += 32) {
      const int j = j0 + lane;
      const float term = j < nsplit ? __fmul_rn(ps[j * ldp + r], fast_exp2(pm[j * ldp + r] - m)) : 0.f;
      const int n = min(32, nsplit - j0);
      for (int k = 0; k < n; ++k) s = __fadd_rn(s, __shfl_sync(0xffffffffu, term, k));
    }
    if (lane == 0) {
      const float lse = (m + __log2f(s)) * kLn2;
      const int tok = jb < nsplit ? bc[jb * ldp + r] : -1;
      const float y0 = jb < nsplit ? bz[jb * ldp + r] : 0.f;
      if (!isfinite(lse) || tok < 0) atomicOr(status, kDevNonFinite);
      lse_r[r] = lse;
      y0_r[r] = y0;
      hi_r[r] = m * kLn2;
      row_above[r] = 0ull;  // the fast pass's per-row accumulators
      row_done[r] = 0u;
      const int t = cidx[r];
      tokens[t] = tok;
      logp[t] = y0 - lse;
    }
  }
}

// Is each row's plain winner in its nucleus?  The mass strictly above the
// winner (2^-40 fixed point, exact integer sums), against the target
// top_p_target: the winner is in exactly when that mass is below the target;
// a row whose winner is outside goes to the list top_p_kernel works through,
// with its target.  A row is cut into `slices` interleaved slices, one CTA
// each (more than one for batches with too few rows to fill the GPU): each
// adds its slice's mass into the row's accumulator with a device-wide atomic,
// fences, and counts itself done; the CTA that completes the count makes the
// decision (nothing waits for anything).  row_above / row_done start at 0
// (top_p_prep_kernel clears them).
__global__ void __launch_bounds__(kTopPThreads)
    top_p_fast_kernel(const float* __restrict__ z, int64_t ldz, int V, const int* __restrict__ n_valid,
                      int slices, const float* __restrict__ lse_r, const float* __restrict__ y0_r, float inv_temp,
                      float top_p, unsigned long long* __restrict__ row_above, unsigned* __restrict__ row_done,
                      int* __restrict__ slow_rows, unsigned long long* __restrict__ slow_target,
                      unsigned* __restrict__ n_slow) {
  constexpr int kUnroll = 8;
  __shared__ unsigned long long ra[kTopPWarps];
  __shared__ float wbuf[kTopPWarps][32 * 4 * kUnroll];  // one warp's logits above the winner in a round
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  float* buf = wbuf[tid >> 5];
  const int nv = *n_valid;
  const int groups = (V + 3) / 4;
  const int stride = slices * kTopPThreads;
  const int64_t items = static_cast<int64_t>(nv) * slices;
  for (int64_t it = blockIdx.x; it < items; it += gridDim.x) {
    const int r = static_cast<int>(it / slices);
    const int sl = static_cast<int>(it - static_cast<int64_t>(r) * slices);
    const float4* zq = reinterpret_cast<const float4*>(z + static_cast<int64_t>(r) * ldz);
    const float lse = lse_r[r], y0 = y0_r[r];
    unsigned long long above = 0ull;
    // whole rounds: most logits lie below the winner, so each warp gathers the
    // ones above it (ballot + prefix count) and computes their masses with all
    // lanes busy instead of a few lanes at a time
    // (the test uses the warp's last lane, so that every lane of a warp runs the
    // same rounds: the ballots need the whole warp)
    int g0 = sl * kTopPThreads + tid;
    for (; g0 - lane + 31 + (kUnroll - 1) * stride < groups - 1; g0 += kUnroll * stride) {
      float4 q[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) q[u] = __ldcg(zq + g0 + u * stride);
      int cnt = 0;
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const float yy[4] = {q[u].x * inv_temp, q[u].y * inv_temp, q[u].z * inv_temp, q[u].w * inv_temp};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const bool a = yy[k] > y0;
          const unsigned bal = __ballot_sync(0xffffffffu, a);
          if (a) buf[cnt + __popc(bal & ((1u << lane) - 1u))] = yy[k];
          cnt += __popc(bal);
        }
      }
      __syncwarp();
      for (int i = lane; i < cnt; i += 32) above += top_p_mass(buf[i], lse);
      __syncwarp();
    }
    // the rest, one group at a time (the last group may be partial)
    for (; g0 < groups; g0 += stride) {
      const float4 q = __ldcg(zq + g0);
      const float zz[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const float y = zz[k] * inv_temp;
        if (4 * g0 + k < V && y > y0) above += top_p_mass(y, lse);
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) above += __shfl_xor_sync(0xffffffffu, above, o);
    if ((tid & 31) == 0) ra[tid >> 5] = above;
    __syncthreads();
    if (tid == 0) {
      above = 0ull;
      for (int w = 0; w < kTopPWarps; ++w) above += ra[w];
      bool decide = true;
      if (slices > 1) {
        atomicAdd(&row_above[r], above);
        __threadfence();
        decide = atomicAdd(&row_done[r], 1u) == static_cast<unsigned>(slices - 1);
        if (decide) {
          __threadfence();
          above = atomicAdd(&row_above[r], 0ull);  // every slice's mass (each fenced before counting itself)
        }
      }
      const unsigned long long target = top_p_target(top_p);
      if (decide && above >= target) {
        const unsigned k = atomicAdd(n_slow, 1u);
        slow_rows[k] = r;
        slow_target[k] = target;
      }
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
