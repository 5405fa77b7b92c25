// top_p.cuh — nucleus (top-p) truncation of the rollout draw.
//
// o_t ~ softmax(z_t / temperature) restricted to its nucleus (Holtzman et al.,
// 2020): the shortest set of the most probable tokens whose mass reaches
// top_p, with every token tied with its least probable member.  Gumbel-max
// over that set draws from the distribution renormalised on it.
//
// The sampling GEMM (kEpiSampleZ) has already produced, per row, the log-sum-
// exp of y = z / temperature, the row maximum and the plain Gumbel-max winner
// w0 over the whole vocabulary, and stored the fp32 logits z.
//
// w0 is in the nucleus exactly when the mass of the logits strictly above
// y_w0 is below the target (then y_w0 >= y*; otherwise the tokens above it
// already reach the target and y* > y_w0).  A winner inside is the nucleus
// winner too, its perturbed score beating every token; that is the case for
// about a fraction top_p of the rows, and top_p = 1 needs no selection at all.
// Masses are probabilities in 2^-40 fixed point, so no sum depends on the
// order of the atomics that form it.  A streaming pass over every row's
// logits (top_p_fast_kernel) lists the rows whose winner may lie outside,
// from fp32 sums within a proven margin of the exact mass.
//
// A cluster of 2, 4 or 8 CTAs takes one listed row at a time (distributed
// shared memory; each CTA walks an interleaved share of the row).  Only the
// logits above y_w0 matter; the first level's histogram of their exact masses
// confirms the row (a row whose total falls short keeps its plain draw), and
// then y* > y_w0:
//   1. a histogram of their mass over 2048 buckets spanning [y_w0, max y]
//      (at most 1/64 nat each); the bucket where the mass counted from the top
//      reaches the target holds y*;
//   2. a second walk gathers that bucket's logits as candidates (every CTA
//      receives all of them); a bucket with more than kTopPCand logits is
//      histogrammed again over its own range first (one whose logits are all
//      equal is taken whole: ties stay together);
//   3. y* is the largest candidate y whose mass together with that of the
//      candidates above it reaches what the target still needs (an exact rank
//      count, the candidates split over the cluster);
//   4. the draw is the best perturbed score y + G over y >= y* (G: the GEMM's
//      noise, Philox4x32-10 word v mod 4 of counter (v div 4, t, offset), key
//      seed, fp32 operations, the lowest v on ties).  The sampling GEMM kept
//      each split entry's best score over all its tokens; an entry whose
//      winner has y >= y* contributes it as it is, and only the other entries
//      (about 1 - top_p of them where the distribution is flat) are walked.
// Every reduction has a fixed order or is exact, so a row's draw is
// deterministic.
#pragma once

#include <stdint.h>

#include <cstdlib>

#include "gemm_tc.cuh"
#include "ptx.cuh"
#include "small_kernels.cuh"

namespace grpo {

constexpr int kTopPThreads = 256;
constexpr int kTopPCtas = 16;      // most CTAs of a cluster sharing one row (clusters of 2, 4, 8 or 16)
constexpr int kTopPBuckets = 2048;
constexpr int kTopPCand = 1024;    // candidates resolved exactly in shared memory
constexpr int kTopPLevels = 6;     // histogram levels before the candidates fit
constexpr int kTopPWarps = kTopPThreads / 32;
// column halves of a tile in the sampling GEMM's split entries (one per epilogue warp of a lane quarter)
constexpr int kSampleHalves = EpiShape<kEpiSample>::kHalves;
static_assert(kTopPBuckets % kTopPCtas == 0, "whole histogram slices per CTA in the merge");

// Shared memory of one CTA.  The fields marked "host" are used in CTA 0 of
// the cluster only (the other CTAs write into and read from CTA 0's copy).
struct TopPShared {
  union {
    unsigned long long hist[kTopPBuckets];  // histogram pass: this CTA's histogram; then its slice merged
    struct {                                // gather pass: this CTA's candidates before they are broadcast
      float y[kTopPCand];
    } loc;
    struct {                                // the draw: this CTA's entries whose winner lies outside the nucleus
      int e[kTopPThreads];
      unsigned n;
    } out;
  };
  float cy[kTopPCand];                      // the cluster's candidates: every CTA holds all of them
  unsigned long long cq[kTopPCand];
  unsigned long long tot[kTopPCtas];        // every CTA: the merged mass of each CTA's histogram slice
  // one value per CTA: host only, the range of its candidates and its best draw; every CTA, its
  // part of the threshold search
  uint32_t slot_lo[kTopPCtas], slot_hi[kTopPCtas], slot_r[kTopPCtas], slot_f[kTopPCtas], slot_g[kTopPCtas],
      slot_i[kTopPCtas];
  float lvl_hi[kTopPLevels];
  float lvl_scale[kTopPLevels];
  int lvl_b[kTopPLevels];
  unsigned long long ra[kTopPWarps];
  float rf[kTopPWarps], rg[kTopPWarps];
  int ri[kTopPWarps];
  unsigned long long cum_before;            // every CTA: the mass above the chosen buckets
  unsigned long long cum_next;              // every CTA: cum_before of the next level, from the CTA that found it
  unsigned ncand;                           // host: the reservation counter; every CTA: the cluster's count
  unsigned lcand, lbase;                    // this CTA's candidate count and its offset in the cluster's list
  float ystar;
  int full;                                 // the threshold is known but the candidates did not all fit
};

// Probability of tempered logit y in 2^-40 units, truncated toward zero: the
// float f = p * 2^40 converted exactly.  A value that is not finite or not
// below 2^41 gives 0.  The conversion is a 32-bit one: below 2^32 f truncates
// directly; from 2^32 on f is a multiple of its ulp (at least 2^9), so f 2^-9
// is an integer below 2^32 and converts exactly, then shifts back.  (A
// 64-bit conversion per logit measured a third of the histogram walk.)
__device__ __forceinline__ unsigned long long top_p_mass(float y, float lse) {
  const float kLog2e = 1.4426950408889634f;
  const float f = fast_exp2((y - lse) * kLog2e) * 1099511627776.0f;
  if (!(f < 2199023255552.0f)) return 0ull;
  const bool big = f >= 4294967296.0f;
  const unsigned v = __float2uint_rz(big ? f * 0.001953125f : f);
  return static_cast<unsigned long long>(v) << (big ? 9 : 0);
}

// Adds q to a 64-bit histogram bucket with 32-bit shared atomics: q's low word
// into the bucket's low word, then its high word plus the carry out of that
// add (the old low word plus q's low word wrapped) into the high word.  The
// bucket ends as the exact sum whatever the order of the adds.
__device__ __forceinline__ void top_p_hist_add(unsigned long long* h, unsigned long long q) {
  unsigned* w = reinterpret_cast<unsigned*>(h);  // little-endian: w[0] is the low word
  const unsigned lo = static_cast<unsigned>(q);
  const unsigned old = atomicAdd(w, lo);
  const unsigned hi = static_cast<unsigned>(q >> 32) + (old + lo < old ? 1u : 0u);
  if (hi) atomicAdd(w + 1, hi);
}

__device__ __forceinline__ int top_p_bucket(float y, float hi, float scale) {
  return static_cast<int>(fminf(fmaxf((hi - y) * scale, 0.f), static_cast<float>(kTopPBuckets - 1)));
}

// True when y lies in the chosen bucket of every one of the first n levels;
// the first level's range and bucket come in registers (hi0, scale0, b0), the
// walks' common case, the deeper ones from shared memory.
__device__ __forceinline__ bool top_p_in(const TopPShared& sh, float hi0, float scale0, int b0, float y, int n) {
  if (n == 0) return true;
  if (top_p_bucket(y, hi0, scale0) != b0) return false;
  for (int l = 1; l < n; ++l)
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

// Walks this CTA's share of the row in a cluster of kC CTAs: groups of four
// logits (16-byte loads; the row's leading dimension is a multiple of 64, so a
// group never leaves the row's storage) g = rank * kTopPThreads + tid + k * kC
// * kTopPThreads, up to kUnroll groups per thread loaded together (the last
// round predicated), then f(g, q) for each.  Lanes of a partial last group
// past V are the caller's to skip.
template <int kC, int kUnroll, typename F>
__device__ __forceinline__ void top_p_groups(const float* zr, int V, int rank, F f) {
  constexpr int kStride = kC * kTopPThreads;
  const int groups = (V + 3) / 4;
  const float4* zq = reinterpret_cast<const float4*>(zr);
  for (int g0 = rank * kTopPThreads + static_cast<int>(threadIdx.x); g0 < groups; g0 += kUnroll * kStride) {
    float4 q[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int g = g0 + u * kStride;
      q[u] = g < groups ? __ldcg(zq + g) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int g = g0 + u * kStride;
      if (g < groups) f(g, q[u]);
    }
  }
}

// The better of two perturbed scores (the lower token on a tie; -1 loses).
__device__ __forceinline__ bool top_p_better(float s, int v, float s0, int v0) {
  return s > s0 || (s == s0 && v >= 0 && (v0 < 0 || v < v0));
}

// This CTA's part of the threshold search over the nc gathered candidates:
// y* is the largest candidate y whose mass M(y) = sum of q_j over the
// candidates with y_j >= y reaches `need` (the first position, largest y
// first, where the running sum reaches need: the running sum at the end of
// y's group of equal logits is M(y), and it grows down the list).  The CTA
// takes the candidates [rank * per, (rank + 1) * per) of a cluster of kC,
// tpi threads each (a power of two, so a candidate's threads share a warp;
// one thread each, in rounds, when there are more candidates than threads);
// returns the largest qualifying y of its candidates in every thread, -inf if
// none.
template <int kC>
__device__ __forceinline__ float top_p_rank_slice(TopPShared& sh, int nc, int rank, unsigned long long need) {
  const int per = (nc + kC - 1) / kC;  // <= kTopPCand / kC
  int tpi = 32;
  while (tpi > 1 && per * tpi > kTopPThreads) tpi >>= 1;
  const int step = kTopPThreads / tpi;  // candidates per round
  float best = -INFINITY;
  for (int k0 = 0; k0 < per; k0 += step) {  // the same rounds in every thread
    const int k = k0 + static_cast<int>(threadIdx.x) / tpi;
    const int i = rank * per + k;
    const bool act = k < per && i < nc;
    const float yi = act ? sh.cy[i] : INFINITY;
    unsigned long long m = 0ull;
    if (act)
      for (int j = static_cast<int>(threadIdx.x) & (tpi - 1); j < nc; j += tpi)
        if (sh.cy[j] >= yi) m += sh.cq[j];
    for (int o = tpi >> 1; o > 0; o >>= 1) m += __shfl_xor_sync(0xffffffffu, m, o);
    if (act && m >= need) best = fmaxf(best, yi);
  }
  return top_p_block_max(sh, best);
}

// Launched in clusters of kC CTAs (the launch sets the cluster shape; 16 is a
// non-portable size the launch enables).
template <int kC>
__global__ void __launch_bounds__(kTopPThreads, 4)
    top_p_kernel(const float* __restrict__ z, int64_t ldz, int V, const int* __restrict__ n_slow,
                 const int* __restrict__ slow_rows, const unsigned long long* __restrict__ slow_target,
                 const int* __restrict__ cidx, const float* __restrict__ lse_r, const float* __restrict__ y0_r,
                 const float* __restrict__ hi_r, const float* __restrict__ best_s, const int* __restrict__ best_c,
                 const float* __restrict__ best_z, int nsplit, long ldp, int unit_tiles, float inv_temp,
                 uint32_t seed_lo, uint32_t seed_hi, uint32_t off_lo, uint32_t off_hi, int32_t* __restrict__ tokens,
                 float* __restrict__ logp, unsigned* status) {
  __shared__ TopPShared sh;
  const int tid = threadIdx.x;
  const int rank = static_cast<int>(cluster_ctarank());
  const bool host = rank == 0;
  const int ns = *n_slow;
  // CTA k's copy of a field
  auto atk = [&](const void* p, int k) { return mapa_shared(smem_addr(p), static_cast<uint32_t>(k)); };
  for (int si = blockIdx.x / kC; si < ns; si += gridDim.x / kC) {
    const int r = slow_rows[si];
    const float* zr = z + static_cast<int64_t>(r) * ldz;
    const int t = cidx[r];
    const float lse = lse_r[r], y0 = y0_r[r];
    const unsigned long long target = slow_target[si];
    if (tid == 0) {
      // the first level spans the logits above the plain winner (y* > y0: the
      // mass above y0 reaches the target), at most 1/64 nat a bucket
      const float hi = hi_r[r];  // the row maximum of y (to rounding)
      sh.lvl_hi[0] = hi;
      sh.lvl_scale[0] = hi > y0 ? fminf(fmaxf(64.f, static_cast<float>(kTopPBuckets - 1) / (hi - y0)), 1e30f) : 64.f;
      sh.cum_before = 0ull;
      sh.full = 0;
    }
    // Each level: histogram the mass of the logits above y0 that lie in the
    // chosen buckets of the levels before; pick the bucket where the mass from
    // the top reaches the target; gather that bucket's logits as candidates
    // and, on the way, draw over the logits above it (all in the nucleus).
    float bs, by;  // this thread's best perturbed score, its token and logit (the draw below)
    int bv;
    int L = 0;
    bool skip_row = false;  // the row keeps its plain draw
    for (;;) {
      __syncthreads();
      for (int b = tid; b < kTopPBuckets; b += kTopPThreads) sh.hist[b] = 0ull;
      __syncthreads();
      {
        const float hi = sh.lvl_hi[L], scale = sh.lvl_scale[L];
        const float hi0 = sh.lvl_hi[0], scale0 = sh.lvl_scale[0];
        const int b0 = L > 0 ? sh.lvl_b[0] : 0;
        top_p_groups<kC, 8>(zr, V, rank, [&](int g, float4 q) {
          const float yy[4] = {q.x * inv_temp, q.y * inv_temp, q.z * inv_temp, q.w * inv_temp};
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            if (4 * g + k < V && yy[k] > y0 && top_p_in(sh, hi0, scale0, b0, yy[k], L)) {
              const unsigned long long m = top_p_mass(yy[k], lse);
              if (m) top_p_hist_add(&sh.hist[top_p_bucket(yy[k], hi, scale)], m);  // far tail adds nothing
            }
          }
        });
      }
      cluster_sync();
      {  // merge the histograms: CTA k sums its slice of kSlice buckets over the cluster in rank
         // order into its own histogram (only CTA k reads the buckets of slice k, so no CTA reads
         // a bucket another one writes) and sends the slice's total to every CTA
        constexpr int kSlice = kTopPBuckets / kC;
        unsigned long long t = 0ull;
#pragma unroll
        for (int p = tid; p < kSlice; p += kTopPThreads) {
          const int b = rank * kSlice + p;
          unsigned long long part[kC];
#pragma unroll
          for (int k = 0; k < kC; ++k) part[k] = ld_shared_cluster_u64(atk(&sh.hist[b], k));
          unsigned long long m = 0ull;
#pragma unroll
          for (int k = 0; k < kC; ++k) m += part[k];
          sh.hist[b] = m;
          t += m;
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
        if ((tid & 31) == 0) sh.ra[tid >> 5] = t;
        __syncthreads();
        if (tid < kC) {
          unsigned long long sum = 0ull;
          for (int w = 0; w < kTopPWarps; ++w) sum += sh.ra[w];
          st_shared_cluster_u64(atk(&sh.tot[rank], tid), sum);
        }
        if (host && tid == 0) sh.ncand = 0u;  // nobody reserves candidates before the next barrier
      }
      cluster_sync();
      // The slice that holds the threshold: the first where the mass from the top
      // reaches the target.  Every CTA decides alike from the same totals.
      int cs = -1;
      unsigned long long before = sh.cum_before;
      for (int k = 0; k < kC; ++k) {
        if (before + sh.tot[k] >= target) {
          cs = k;
          break;
        }
        before += sh.tot[k];
      }
      // level 0 holds every logit above the winner: when even their exact mass
      // falls short of the target, the winner is in the nucleus (no CTA touches
      // another's shared memory after the barrier above in this row)
      if (L == 0 && cs < 0) {
        skip_row = true;
        break;
      }
      if (cs < 0) {  // (the masses fell short at a deeper level) the last bucket, as a scan would end
        cs = kC - 1;
        before -= sh.tot[kC - 1];
      }
      if (rank == cs) {  // the bucket within this slice: one block scan over per-thread runs of buckets
        constexpr int kSlice = kTopPBuckets / kC;
        constexpr int kPer = (kSlice + kTopPThreads - 1) / kTopPThreads;  // consecutive buckets a thread sums
        const int lane = tid & 31, warp = tid >> 5;
        const int p0 = tid * kPer;  // this thread's first position in the slice
        unsigned long long own = 0ull;
#pragma unroll
        for (int i = 0; i < kPer; ++i)
          if (p0 + i < kSlice) own += sh.hist[rank * kSlice + p0 + i];
        unsigned long long inc = own;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const unsigned long long n = __shfl_up_sync(0xffffffffu, inc, o);
          if (lane >= o) inc += n;
        }
        if (lane == 31) sh.ra[warp] = inc;
        __syncthreads();
        unsigned long long pre = 0ull, all = 0ull;
        for (int w = 0; w < kTopPWarps; ++w) {
          if (w < warp) pre += sh.ra[w];
          all += sh.ra[w];
        }
        inc += pre;
        // the first thread whose runs reach the target holds the crossing (its runs
        // are consecutive, so it walks them alone)
        const unsigned hit = __ballot_sync(0xffffffffu, before + inc >= target);
        if (lane == 0) sh.ri[warp] = hit ? __ffs(hit) - 1 : 32;
        __syncthreads();
        int first = kTopPThreads;
        for (int w = 0; w < kTopPWarps; ++w)
          if (sh.ri[w] < 32) {
            first = w * 32 + sh.ri[w];
            break;
          }
        if (tid == first) {
          unsigned long long a = before + inc - own;  // the mass above this thread's runs
          int b = rank * kSlice + p0;
          for (int i = 0; i < kPer - 1 && p0 + i < kSlice - 1; ++i, ++b) {
            if (a + sh.hist[b] >= target) break;
            a += sh.hist[b];
          }
          for (int k = 0; k < kC; ++k) {
            st_shared_cluster(atk(&sh.lvl_b[L], k), static_cast<uint32_t>(b));
            st_shared_cluster_u64(atk(&sh.cum_next, k), a);
          }
        } else if (first == kTopPThreads && tid == 0) {
          // no crossing in the last slice (only at a deeper level): its last bucket
          const int b = rank * kSlice + kSlice - 1;
          const unsigned long long a = before + all - sh.hist[b];
          for (int k = 0; k < kC; ++k) {
            st_shared_cluster(atk(&sh.lvl_b[L], k), static_cast<uint32_t>(b));
            st_shared_cluster_u64(atk(&sh.cum_next, k), a);
          }
        }
      }
      cluster_sync();
      if (tid == 0) {
        sh.cum_before = sh.cum_next;
        sh.lcand = 0u;
      }
      __syncthreads();
      // gather the bucket's logits (and their range, in case they do not fit)
      // into this CTA's list
      float lo = INFINITY, hi2 = -INFINITY;
      const float hi0 = sh.lvl_hi[0], scale0 = sh.lvl_scale[0];
      const int b0 = sh.lvl_b[0];
      top_p_groups<kC, 8>(zr, V, rank, [&](int g, float4 q) {
        const float yy[4] = {q.x * inv_temp, q.y * inv_temp, q.z * inv_temp, q.w * inv_temp};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          if (4 * g + k < V && yy[k] > y0 && top_p_in(sh, hi0, scale0, b0, yy[k], L + 1)) {
            lo = fminf(lo, yy[k]);
            hi2 = fmaxf(hi2, yy[k]);
            const unsigned i = atomicAdd(&sh.lcand, 1u);
            if (i < static_cast<unsigned>(kTopPCand)) sh.loc.y[i] = yy[k];
          }
        }
      });
      lo = -top_p_block_max(sh, -lo);
      hi2 = top_p_block_max(sh, hi2);
      if (tid == 0) {
        st_shared_cluster(atk(&sh.slot_lo[rank], 0), __float_as_uint(lo));
        st_shared_cluster(atk(&sh.slot_hi[rank], 0), __float_as_uint(hi2));
        sh.lbase = atom_add_shared_cluster(atk(&sh.ncand, 0), sh.lcand);
      }
      __syncthreads();
      {  // this CTA's candidates into every CTA's list, at the offset it reserved
        const unsigned n = min(sh.lcand, static_cast<unsigned>(kTopPCand));
        const unsigned base = sh.lbase;
        for (unsigned i = tid; i < n && base + i < static_cast<unsigned>(kTopPCand); i += kTopPThreads) {
          const float y = sh.loc.y[i];
          const unsigned long long m = top_p_mass(y, lse);
#pragma unroll
          for (int k = 0; k < kC; ++k) {
            st_shared_cluster(atk(&sh.cy[base + i], k), __float_as_uint(y));
            st_shared_cluster_u64(atk(&sh.cq[base + i], k), m);
          }
        }
      }
      cluster_sync();
      if (tid == 0) {
        if (!host) sh.ncand = ld_shared_cluster(atk(&sh.ncand, 0));
        if (sh.ncand > static_cast<unsigned>(kTopPCand)) {
          // too many to resolve here: every CTA reads the bucket's range and
          // decides alike whether to histogram it once more
          float l = INFINITY, h = -INFINITY;
          for (int k = 0; k < kC; ++k) {
            l = fminf(l, __uint_as_float(ld_shared_cluster(atk(&sh.slot_lo[k], 0))));
            h = fmaxf(h, __uint_as_float(ld_shared_cluster(atk(&sh.slot_hi[k], 0))));
          }
          if (!(h > l) || L + 1 >= kTopPLevels) {
            sh.ystar = l;  // all equal (or out of levels: the whole bucket)
            sh.full = 1;
            if (host && h > l) atomicOr(status, kDevNonFinite);
          } else {
            sh.lvl_hi[L + 1] = h;
            sh.lvl_scale[L + 1] = static_cast<float>(kTopPBuckets - 1) / (h - l);
          }
        }
      }
      __syncthreads();
      const int nc = static_cast<int>(sh.ncand);
      if (nc <= kTopPCand) {
        const float c = top_p_rank_slice<kC>(sh, nc, rank, target - sh.cum_before);
        if (tid < kC) st_shared_cluster(atk(&sh.slot_r[rank], tid), __float_as_uint(c));  // to every CTA
        cluster_sync();
        if (tid == 0) {
          float ys = -INFINITY;
          for (int k = 0; k < kC; ++k) ys = fmaxf(ys, __uint_as_float(sh.slot_r[k]));
          sh.ystar = ys;
          sh.full = ys == -INFINITY;  // no crossing (the masses fell short): the whole vocabulary
        }
        __syncthreads();
        break;
      }
      if (sh.full) break;
      ++L;
    }
    if (skip_row) continue;  // the plain draw (already written) stands
    // The draw: the best perturbed score over the logits y >= y*, the lowest
    // token on ties.  The sampling GEMM kept, for every split entry (a
    // vocabulary unit of unit_tiles tiles, one column half of each tile), its
    // best score over all of the entry's tokens.  Where that winner lies in
    // the nucleus it is the entry's best over its nucleus tokens too; only the
    // other entries are walked, with the GEMM's noise (Philox4x32-10 word v
    // mod 4 of counter (v div 4, t, offset), fp32 operations).
    const float ystar = sh.ystar;
    bs = -INFINITY;
    bv = -1;
    by = 0.f;
    // This CTA's entries are e = rank + kC j.  Each thread classifies
    // one of them (the loads of all entries in flight together); the entries
    // whose winner lies outside are then walked as one list of 4-token groups.
    constexpr int kGroupsPerTile = kTileN / kSampleHalves / 4;  // 4-token groups of one tile's column half
    const int per_entry = unit_tiles * kGroupsPerTile;
    const int nj = nsplit > rank ? (nsplit - rank + kC - 1) / kC : 0;
    for (int base = 0; base < nj; base += kTopPThreads) {
      __syncthreads();  // the previous batch's list has been walked
      if (tid == 0) sh.out.n = 0u;
      __syncthreads();
      if (base + tid < nj) {
        const int e = rank + kC * (base + tid);
        const long at = static_cast<long>(e) * ldp + r;
        const float bz = best_z[at];
        if (bz >= ystar) {
          const float s0 = best_s[at];
          const int c = best_c[at];
          if (top_p_better(s0, c, bs, bv)) {
            bs = s0;
            bv = c;
            by = bz;
          }
        } else {
          sh.out.e[atomicAdd(&sh.out.n, 1u)] = e;
        }
      }
      __syncthreads();
      const int total = static_cast<int>(sh.out.n) * per_entry;
      constexpr int kU = 4;  // groups per thread loaded together
      for (int g0 = tid; g0 < total; g0 += kU * kTopPThreads) {
        float4 q[kU];
        int v0[kU];
#pragma unroll
        for (int u = 0; u < kU; ++u) {
          const int gi = g0 + u * kTopPThreads;
          v0[u] = V;
          if (gi < total) {
            const int e = sh.out.e[gi / per_entry];
            const int gl = gi - (gi / per_entry) * per_entry;
            v0[u] = (e / kSampleHalves) * unit_tiles * kTileN + (e % kSampleHalves) * (kTileN / kSampleHalves) +
                    (gl / kGroupsPerTile) * kTileN + 4 * (gl % kGroupsPerTile);
          }
          q[u] = v0[u] < V ? __ldcg(reinterpret_cast<const float4*>(zr + v0[u])) : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int u = 0; u < kU; ++u) {
          if (v0[u] >= V) continue;
          const float yy[4] = {q[u].x * inv_temp, q[u].y * inv_temp, q[u].z * inv_temp, q[u].w * inv_temp};
          if (!(yy[0] >= ystar || yy[1] >= ystar || yy[2] >= ystar || yy[3] >= ystar)) continue;
          const uint4 w = philox4x32_10(
              make_uint4(static_cast<uint32_t>(v0[u] >> 2), static_cast<uint32_t>(t), off_lo, off_hi), seed_lo, seed_hi);
          const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const int v = v0[u] + k;
            if (v < V && yy[k] >= ystar) {
              const float sc = yy[k] + gumbel_of(ws[k]);
              if (top_p_better(sc, v, bs, bv)) {
                bs = sc;
                bv = v;
                by = yy[k];
              }
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
      st_shared_cluster(atk(&sh.slot_f[rank], 0), __float_as_uint(bs));
      st_shared_cluster(atk(&sh.slot_g[rank], 0), __float_as_uint(by));
      st_shared_cluster(atk(&sh.slot_i[rank], 0), static_cast<uint32_t>(bv));
    }
    cluster_sync();
    if (host && tid == 0) {
      bs = -INFINITY;
      bv = -1;
      by = 0.f;
      for (int k = 0; k < kC; ++k) {
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
    // No barrier before the next row: the host's slots are written again only
    // after the next row's third cluster barrier, which the host reaches after
    // reading them here; nothing else of another CTA is touched after the one
    // above.
  }
}

// Per unmasked row, the plain draw from the sampling GEMM's splits: written
// to the outputs (the nucleus selection replaces it only where the winner
// falls outside the nucleus), and the row's LSE, winner's y and maximum y kept
// for the selection (whose per-row accumulators it clears).  One warp per row reads the splits in parallel; the LSE
// is merge_lse's (merge_lse_warp), and the winner is the best
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
    float best = -INFINITY;
    int jb = nsplit;
    for (int j = lane; j < nsplit; j += 32) {
      const float sc = bs[j * ldp + r];
      if (sc > best) {
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
    float m;
    const float lse = merge_lse_warp(pm, ps, nsplit, ldp, r, lane, &m);
    if (lane == 0) {
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

// Which rows' plain winner may lie outside its nucleus?  The winner is in
// exactly when the mass strictly above it, in the 2^-40 fixed point of
// top_p_mass, is below top_p_target.  This pass only sorts the rows: it sums
// the same per-logit values p_v 2^40 in fp32 over each thread's 32 logits of a
// chunk and adds those sums, truncated, as integers.  Against the exact
// fixed-point mass E that approximation A is off by at most 31 u A' (the fp32
// sums of 32 positive terms, u = 2^-24, A' <= 2^41) plus one unit per logit
// and per sum, so |A - E| < 2^23 + 2 V = top_p_margin(V): a row with A plus
// that margin below the target certainly keeps its winner, and every other row goes to the list
// top_p_kernel works through, which confirms it with the exact mass first
// (the total of its level-0 histogram) and leaves a row whose exact mass
// falls short with its plain draw.
//
// The stored logits stream through shared memory.  Each row is cut into
// chunks of kFastChunk logits, the chunks of all rows are numbered row by
// row, and each CTA takes one contiguous range of them (so the grid stays
// busy whatever the number of rows).  One thread keeps kFastStages chunks in
// flight with bulk copies that complete on a per-stage mbarrier, while all
// threads work through the oldest (each thread 32 logits of a chunk, 16-byte
// shared loads).  When the CTA leaves a row it adds its sum for the row into
// the row's accumulator (integer device atomics, so the order does not
// matter), fences, and
// adds the number of chunks it covered to the row's count; the CTA that
// completes the count decides (nothing waits for anything).  row_above /
// row_done start at 0 (top_p_prep_kernel clears them).  Every wait is
// bounded: on expiry the CTA sets kDevTimeout, lets the copies it issued
// land (bounded again) and returns.
constexpr int kFastChunk = 8192;   // logits per stage (32 KB)
constexpr int kFastStages = 3;
constexpr int kFastSmem = kFastStages * kFastChunk * 4 + kFastStages * 8;
static_assert(kFastChunk % (kTopPWarps * 128) == 0, "whole float4 rounds per warp");

// The bound on |A - E| above for a vocabulary of V, in units of 2^-40.
inline unsigned long long top_p_margin(int64_t V) { return (1ull << 23) + 2ull * static_cast<unsigned long long>(V); }

// log2 of the cluster size of the selection (1 to 4: clusters of 2, 4, 8 or
// 16 CTAs) for a draw over up to `rows` rows.  About a fraction 1 - top_p of
// the rows are listed (the winner falls outside its nucleus that often).  A
// cluster takes one listed row at a time, so few listed rows want large
// clusters (each row done sooner, while about 74 clusters of 8 fit on a
// GB300) and many want small ones (fewer cluster barriers per logit).
// Measured draws over V = 155,136 (the listed-row estimate in brackets):
// 256 rows at top_p 0.9 [33] 0.37 / 0.39 / 0.43 ms with clusters of 8 / 4 /
// 2, at 0.5 [166] 0.43 / 0.42 / 0.46; 2048 rows at 0.9 [266] 1.96-2.06 /
// 1.96-2.10 / 2.03-2.11, at 0.5 [1331] 2.59 / 2.48 / 2.46; 19,572 of 32,768
// rows at 0.5 [21299] 24.7-24.9 / 24.3-24.7 / 23.4-24.1 ms.  GRPO_TOP_P_CLUSTER=2|4|8
// overrides the choice (16: one round of rows for a decode step's few
// listed rows, each walked by twice as many CTAs).
inline int top_p_cluster_log2(int64_t rows, float top_p) {
  if (const char* e = std::getenv("GRPO_TOP_P_CLUSTER")) {
    const int c = std::atoi(e);
    if (c == 2) return 1;
    if (c == 4) return 2;
    if (c == 8) return 3;
    if (c == 16) return 4;
  }
  const double listed = static_cast<double>(rows) * (1.0 - static_cast<double>(top_p)) * 1.3;
  return listed <= 36.0 ? 4 : listed <= 100.0 ? 3 : listed <= 400.0 ? 2 : 1;
}

__global__ void __launch_bounds__(kTopPThreads, 2)
    top_p_fast_kernel(const float* __restrict__ z, int64_t ldz, int V, const int* __restrict__ n_valid,
                      const float* __restrict__ lse_r, const float* __restrict__ y0_r, float inv_temp,
                      float top_p, unsigned long long* __restrict__ row_above, unsigned* __restrict__ row_done,
                      int* __restrict__ slow_rows, unsigned long long* __restrict__ slow_target,
                      unsigned* __restrict__ n_slow, unsigned long long margin, unsigned* status) {
  constexpr int kSeg = kFastChunk / kTopPWarps;  // logits of a chunk one warp reads
  constexpr int kPer = kSeg / 128;               // float4 per lane
  extern __shared__ __align__(128) unsigned char fast_smem[];
  float* ring = reinterpret_cast<float*>(fast_smem);
  uint64_t* full = reinterpret_cast<uint64_t*>(fast_smem + kFastStages * kFastChunk * 4);
  __shared__ unsigned long long ra[kTopPWarps];
  __shared__ int never;  // the waits here have no abort flag: never set
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const int warp = tid >> 5;
  const int nv = *n_valid;
  const int cpr = (V + kFastChunk - 1) / kFastChunk;  // chunks per row
  const int64_t items = static_cast<int64_t>(nv) * cpr;
  const int64_t per = (items + gridDim.x - 1) / gridDim.x;
  const int64_t i0 = static_cast<int64_t>(blockIdx.x) * per;
  const int64_t i1 = min(items, i0 + per);
  if (i0 >= i1) return;
  if (tid == 0) {
    for (int s = 0; s < kFastStages; ++s) mbar_init(smem_addr(&full[s]), 1);
    never = 0;
    fence_mbar_init();
  }
  __syncthreads();
  const unsigned long long target = top_p_target(top_p);
  // thread 0: the copy of chunk `it` into stage s (whole 16-byte groups: the
  // row's storage, ldz >= V rounded up to 64, covers the last partial group,
  // whose extra lanes are skipped below)
  auto issue = [&](int64_t it, int s) {
    const int64_t r = it / cpr;
    const int c0 = static_cast<int>(it - r * cpr) * kFastChunk;
    const uint32_t bytes = static_cast<uint32_t>((min(kFastChunk, V - c0) + 3) & ~3) * 4u;
    const uint32_t bar = smem_addr(&full[s]);
    mbar_arrive_expect_tx(bar, bytes);
    bulk_load_1d(smem_addr(ring + s * kFastChunk), z + r * ldz + c0, bytes, bar);
  };
  if (tid == 0)
    for (int s = 0; s < kFastStages && i0 + s < i1; ++s) issue(i0 + s, s);

  int64_t row = i0 / cpr;
  unsigned long long above = 0ull;
  unsigned covered = 0;
  // this CTA's mass of `row` and its chunk count into the row's accumulators
  auto flush = [&]() {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) above += __shfl_xor_sync(0xffffffffu, above, o);
    if (lane == 0) ra[warp] = above;
    __syncthreads();
    if (tid == 0) {
      unsigned long long m = 0ull;
      for (int w = 0; w < kTopPWarps; ++w) m += ra[w];
      atomicAdd(&row_above[row], m);
      __threadfence();
      if (atomicAdd(&row_done[row], covered) + covered == static_cast<unsigned>(cpr)) {
        __threadfence();
        const unsigned long long total = atomicAdd(&row_above[row], 0ull);  // every CTA's sum, each fenced first
        if (total + margin >= target) {
          const unsigned k = atomicAdd(n_slow, 1u);
          slow_rows[k] = static_cast<int>(row);
          slow_target[k] = target;
        }
      }
    }
    __syncthreads();
    above = 0ull;
    covered = 0;
  };

  int64_t it = i0;
  bool ok = true;
  for (; it < i1; ++it) {
    const int k = static_cast<int>(it - i0);
    const int s = k % kFastStages;
    const int64_t r = it / cpr;
    if (r != row) {  // uniform across the CTA
      flush();
      row = r;
    }
    const bool got = mbar_wait(smem_addr(&full[s]), static_cast<uint32_t>(k / kFastStages) & 1u, &never);
    if (!__syncthreads_and(got)) {
      ok = false;
      break;
    }
    const int c0 = static_cast<int>(it - r * cpr) * kFastChunk;
    const int n = min(kFastChunk, V - c0);  // logits of this chunk inside the row
    const float y0 = y0_r[r], lse = lse_r[r];
    const float* seg = ring + s * kFastChunk + warp * kSeg;
    float4 q[kPer];
#pragma unroll
    for (int j = 0; j < kPer; ++j) q[j] = reinterpret_cast<const float4*>(seg)[lane + 32 * j];
    // p_v 2^40 exactly as top_p_mass forms it, summed over the logits above the winner
    const float kLog2e = 1.4426950408889634f;
    float acc = 0.f;
    if (n == kFastChunk) {
#pragma unroll
      for (int j = 0; j < kPer; ++j) {
        const float zz[4] = {q[j].x, q[j].y, q[j].z, q[j].w};
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
          const float y = zz[kk] * inv_temp;
          const float f = fast_exp2((y - lse) * kLog2e) * 1099511627776.0f;
          acc += y > y0 ? f : 0.f;
        }
      }
    } else {  // the row's last, partial chunk
#pragma unroll
      for (int j = 0; j < kPer; ++j) {
        const float zz[4] = {q[j].x, q[j].y, q[j].z, q[j].w};
        const int e0 = warp * kSeg + 4 * (lane + 32 * j);
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
          const float y = zz[kk] * inv_temp;
          const float f = fast_exp2((y - lse) * kLog2e) * 1099511627776.0f;
          acc += e0 + kk < n && y > y0 ? f : 0.f;
        }
      }
    }
    above += __float2ull_rz(acc);
    ++covered;
    __syncthreads();  // every warp is done with stage s
    if (tid == 0 && it + kFastStages < i1) issue(it + kFastStages, s);
  }
  if (ok) {
    flush();
    return;
  }
  // a copy did not arrive in time: report it, let the copies issued for the
  // chunks not yet consumed land (bounded), and give up on the rest
  if (tid == 0) {
    atomicOr(status, kDevTimeout);
    bool drained = true;
    for (int64_t j = it; j < i1 && j < it + kFastStages; ++j) {
      const int kj = static_cast<int>(j - i0);
      if (!mbar_wait(smem_addr(&full[kj % kFastStages]), static_cast<uint32_t>(kj / kFastStages) & 1u, &never,
                     kDrainNs))
        drained = false;
    }
    if (!drained) __nanosleep(kDrainPauseNs);
  }
  __syncthreads();
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
