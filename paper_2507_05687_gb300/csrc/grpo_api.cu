// grpo_api.cu — the C ABI of include/grpo.h: argument checks, workspace
// layout, TMA tensor maps and the launch sequence of each call.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <cmath>
#include <cstdint>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <type_traits>
#include <vector>

#include "../../include/grpo.h"
#include "gemm_launch.cuh"
#include "gemm_tc.cuh"
#include "small_kernels.cuh"
#include "top_p.cuh"

using namespace grpo;
using namespace grpo::launch;

namespace {

constexpr int kLossThreads = 256;

// Workspace layout (byte offsets); every region is 256-byte aligned, the
// bf16 matrices 1024-byte aligned.  Regions indexed by token position hold
// T_pad rows; regions indexed by compacted (unmasked) row hold `rows`, the
// row capacity: T_pad for a full workspace, less for one sized by
// grpo_workspace_bytes_rows for batches with few unmasked rows.
struct Layout {
  int64_t T_pad, rows, nsplit, nblk_scan, nblk_loss, vchunk;
  int64_t ldz;    // leading dimension (fp32 elements) of the stored logits; 0: not stored
  int lse_tiles;  // vocabulary tiles (of 256) per forward work unit
  size_t status, n_valid, gate, counts, offsets, cidx, rank_of, yc, zy, part_m, part_s, lse_c, g_c,
      block_loss, resp_len, best_s, best_c, best_z, Hc, HcT, dz, dhc, z, slow_rows, slow_tgt, n_slow, row_above,
      row_done, total;
};

bool make_layout(int64_t T, int32_t Hd, int64_t V, int32_t which, Layout* L, int64_t rows_cap = -1) {
  if (T < 0 || T >= (int64_t(1) << 31) || Hd <= 0 || Hd % 64 != 0 || V <= 0 ||
      V >= (int64_t(1) << 31) ||
      (which != GRPO_WS_LOGPROBS && which != GRPO_WS_LOSS && which != GRPO_WS_LOGPROBS_HEADS &&
       which != GRPO_WS_SAMPLE && which != GRPO_WS_LOSS_LOGITS && which != GRPO_WS_SAMPLE_TOP_P))
    return false;
  const bool loss = which == GRPO_WS_LOSS || which == GRPO_WS_LOSS_LOGITS;
  const size_t heads = which == GRPO_WS_LOGPROBS_HEADS ? kMaxHeads : 1;
  L->T_pad = round_up(std::max<int64_t>(T, 1), kRowAlign);
  const int64_t vtiles = (V + kTileN - 1) / kTileN;
  // partial (max, sum) entries per row: one per vocabulary split and column half
  L->lse_tiles = lse_tiles_per_unit();
  const int64_t m_tiles = (std::max<int64_t>(T, 1) + 2 * kRowsCta - 1) / (2 * kRowsCta);
  while (L->lse_tiles > 4 && m_tiles * ((vtiles + L->lse_tiles - 1) / L->lse_tiles) < kNominalPairs)
    L->lse_tiles /= 2;
  L->nsplit = (vtiles + L->lse_tiles - 1) / L->lse_tiles *
              (which == GRPO_WS_SAMPLE || which == GRPO_WS_SAMPLE_TOP_P ? EpiShape<kEpiSample>::kHalves
                                                                         : EpiShape<kEpiLse>::kHalves);
  L->rows = rows_cap < 0 ? L->T_pad : std::min(L->T_pad, round_up(std::max<int64_t>(rows_cap, 1), kRowAlign));
  L->nblk_scan = (std::max<int64_t>(T, 1) + kScanChunk - 1) / kScanChunk;
  L->nblk_loss = (L->rows + kLossThreads - 1) / kLossThreads;
  L->vchunk = loss ? vocab_chunk(V) : 0;
  L->ldz = which == GRPO_WS_LOSS_LOGITS || which == GRPO_WS_SAMPLE_TOP_P ? round_up(V, 64) : 0;
  size_t off = 0;
  auto take = [&](size_t bytes, size_t align) {
    off = (off + align - 1) / align * align;
    const size_t at = off;
    off += bytes;
    return at;
  };
  const size_t tp = static_cast<size_t>(L->T_pad);  // token rows
  const size_t cr = static_cast<size_t>(L->rows);   // compacted rows
  L->status = take(4, 256);
  L->n_valid = take(4, 4);
  L->gate = take(4 * kGateSlots, 256);  // the forward GEMM's pace gate, one counter per CTA
  L->counts = take(4 * L->nblk_scan, 256);
  L->offsets = take(4 * L->nblk_scan, 256);
  L->cidx = take(4 * cr, 256);
  L->rank_of = take(4 * tp, 256);
  L->yc = take(4 * cr, 256);
  L->zy = take(4 * cr * heads, 256);
  L->part_m = take(4 * cr * L->nsplit * heads, 256);
  L->part_s = take(4 * cr * L->nsplit * heads, 256);
  L->lse_c = take(4 * cr, 256);
  L->g_c = take(4 * cr, 256);
  L->block_loss = take(8 * L->nblk_loss, 256);
  L->resp_len = take(4 * tp, 256);
  const size_t best = which == GRPO_WS_SAMPLE || which == GRPO_WS_SAMPLE_TOP_P ? 4 * cr * L->nsplit : 0;
  L->best_s = take(best, 256);
  L->best_c = take(best, 256);
  L->best_z = take(best, 256);
  L->Hc = take(2 * cr * static_cast<size_t>(Hd), 1024);
  // H_c transposed (rows [Hd x rows], or k-blocks [rows / 64][Hd][64] when a
  // row would exceed kMaxTransposedRowBytes): the K-major B operand of the dW GEMM
  L->HcT = loss ? take(2 * cr * static_cast<size_t>(Hd), 1024) : off;
  L->dz = loss ? take(2 * cr * static_cast<size_t>(L->vchunk), 1024) : off;
  // dH over the compacted rows, accumulated across vocabulary chunks
  L->dhc = loss ? take(4 * cr * static_cast<size_t>(Hd), 1024) : off;
  // the fp32 logits [rows x ldz] of the forward, kept for the backward (last,
  // so that every other region sits where the plain loss layout has it)
  L->z = take(4 * cr * static_cast<size_t>(L->ldz), 1024);
  // the nucleus draw: the rows whose plain winner falls outside, their targets, their count
  const bool top_p = which == GRPO_WS_SAMPLE_TOP_P;
  L->slow_rows = take(top_p ? 4 * cr : 0, 256);
  L->slow_tgt = take(top_p ? 8 * cr : 0, 256);
  L->n_slow = take(top_p ? 4 : 0, 256);
  L->row_above = take(top_p ? 8 * cr : 0, 256);
  L->row_done = take(top_p ? 4 * cr : 0, 256);
  L->total = (off + 1023) / 1024 * 1024;
  return true;
}

// The layout a call uses with a workspace of ws_bytes: the full one when it
// fits, else the largest row capacity (a multiple of 256) that fits.  False
// when the arguments are invalid or not even 256 rows fit.
bool fit_layout(int64_t T, int32_t Hd, int64_t V, int32_t which, size_t ws_bytes, Layout* L) {
  if (!make_layout(T, Hd, V, which, L)) return false;
  if (ws_bytes >= L->total) return true;
  int64_t lo = 0, hi = L->T_pad / kRowAlign;  // lo fits (0 = none found), hi does not
  Layout t;
  while (hi - lo > 1) {
    const int64_t mid = (lo + hi) / 2;
    make_layout(T, Hd, V, which, &t, mid * kRowAlign);
    if (t.total <= ws_bytes) lo = mid;
    else hi = mid;
  }
  if (lo == 0) {
    make_layout(T, Hd, V, which, &t, kRowAlign);
    if (t.total > ws_bytes) return false;
    lo = 1;
  }
  return make_layout(T, Hd, V, which, L, lo * kRowAlign);
}

// The layout of a loss call with a workspace of ws_bytes.  By default the
// backward recomputes each vocabulary chunk of the logits and nothing of
// [tokens x vocabulary] size is stored.  The logits are kept from the forward
// to the backward only when ws_bytes is exactly a kept-logits size
// (grpo_workspace_bytes(_rows) with GRPO_WS_LOSS_LOGITS) and not also exactly
// the plain layout's size: the caller asked for that layout by its size.  A
// larger workspace of any other size keeps the plain layout, however much
// room it has.
bool fit_loss_layout(int64_t T, int32_t Hd, int64_t V, size_t ws_bytes, Layout* L) {
  if (!fit_layout(T, Hd, V, GRPO_WS_LOSS, ws_bytes, L)) return false;
  Layout kept;
  if (fit_layout(T, Hd, V, GRPO_WS_LOSS_LOGITS, ws_bytes, &kept) && kept.total == ws_bytes &&
      L->total != ws_bytes)
    *L = kept;
  return true;
}

// ---------------------------------------------------------------- driver entry points

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;

bool get_encode() {
  std::call_once(g_encode_once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  });
  return g_encode != nullptr;
}

// A 2-D tensor map over a row-major matrix [rows x cols] (leading dimension
// ld elements) with boxes of box_cols (inner) x box_rows: bf16 operands in the
// 128-byte swizzle by default (box_cols 64 = 128 bytes); the output maps of
// the epilogues use fp32 / the 64-byte swizzle as their boxes need.
// Out-of-range elements of a box read as zero and are not written.
bool encode_2d(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint64_t ld_elems,
               uint32_t box_cols, uint32_t box_rows, bool f32 = false,
               CUtensorMapSwizzle swizzle = CU_TENSOR_MAP_SWIZZLE_128B) {
  const cuuint64_t dims[2] = {cols, rows};
  const cuuint64_t strides[1] = {ld_elems * (f32 ? 4 : 2)};
  const cuuint32_t box[2] = {box_cols, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  const CUresult r = g_encode(map, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                              const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                              swizzle, CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// A 3-D tensor map over a bf16 operand stored in k-blocks [K / 64][rows][64]
// (64 contiguous K elements per row of a block): the box is 64 x box_rows x 1
// in the 128-byte swizzle, the same shared-memory tile as the 2-D K-major box.
bool encode_blk(CUtensorMap* map, const void* base, uint64_t rows, uint64_t k, uint32_t box_rows) {
  const cuuint64_t dims[3] = {64, rows, k / 64};
  const cuuint64_t strides[2] = {64 * 2, rows * 64 * 2};
  const cuuint32_t box[3] = {64, box_rows, 1};
  const cuuint32_t estr[3] = {1, 1, 1};
  const CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box,
                              estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

struct DeviceInfo {
  int sms = 0;
  int pairs = 0;        // CTA pairs of the pair kernels that can be resident at once
  int top_p_clusters[4] = {0, 0, 0, 0};  // clusters of 2, 4, 8, 16 CTAs of the nucleus selection resident at once
  int fast_ctas = 0;       // CTAs of the nucleus fast pass resident at once (all SMs)
  bool ok = false;
};

// Every variant's dynamic shared memory fits the 227 KB a CTA may opt into.
static_assert(smem_bytes<2, kEpiSampleZ>() <= 232448 && smem_bytes<1, kEpiSampleZ>() <= 232448 &&
                  smem_bytes<2, kEpiAdam>() <= 232448 && smem_bytes<2, kEpiF32>() <= 232448 &&
                  smem_bytes<1, kEpiF32>() <= 232448,
              "shared memory budget");

template <int E, bool A, bool B, bool BLK = false>
bool prepare_kernels(int* pairs) {
  if (cudaFuncSetAttribute(gemm_tc_kernel<E, A, B, BLK>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           smem_bytes<1, E>()) != cudaSuccess ||
      cudaFuncSetAttribute(gemm_tc_pair_kernel<E, A, B, BLK>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           smem_bytes<2, E>()) != cudaSuccess)
    return false;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * 1024, 1, 1);
  cfg.blockDim = dim3(EpiShape<E>::kThreads, 1, 1);
  cfg.dynamicSmemBytes = smem_bytes<2, E>();
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, gemm_tc_pair_kernel<E, A, B, BLK>, &cfg) != cudaSuccess) {
    cudaGetLastError();  // clear: without the query the single-CTA tiles are used
    n = 0;
  }
  *pairs = *pairs < 0 ? n : std::min(*pairs, n);
  return true;
}

// Per-device facts and the one-time opt-in to large dynamic shared memory.
bool device_info(DeviceInfo* out) {
  static std::mutex mu;
  static DeviceInfo cache[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return false;
  std::lock_guard<std::mutex> lk(mu);
  if (!cache[dev].ok) {
    int major = 0, minor = 0, sms = 0, pairs = -1;
    if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return false;
    if (major != 10 || minor != 3) return false;
    if (!prepare_kernels<kEpiLse, false, false>(&pairs) || !prepare_kernels<kEpiLseZ, false, false>(&pairs) ||
        !prepare_kernels<kEpiDz, false, false>(&pairs) ||
        !prepare_kernels<kEpiF32, false, true>(&pairs) || !prepare_kernels<kEpiF32, true, false>(&pairs) ||
        !prepare_kernels<kEpiF32, true, false, true>(&pairs) || !prepare_kernels<kEpiAdam, true, false, true>(&pairs) ||
        !prepare_kernels<kEpiAdam, true, false>(&pairs) || !prepare_kernels<kEpiSample, false, false>(&pairs) ||
        !prepare_kernels<kEpiSampleZ, false, false>(&pairs))
      return false;
    // the nucleus selection walks its rows in a loop over a fixed set of
    // clusters: launch no more than can be resident together (a cluster must
    // fit in one GPC, so this is below SMs x CTAs per SM / cluster size)
    auto resident_clusters = [](auto kernel, int cluster) {
      if (cluster > 8 &&
          cudaFuncSetAttribute(kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess) {
        cudaGetLastError();
        return 0;
      }
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = cluster;
      attr[0].val.clusterDim.y = 1;
      attr[0].val.clusterDim.z = 1;
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3(cluster * 1024, 1, 1);
      cfg.blockDim = dim3(kTopPThreads, 1, 1);
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      int n = 0;
      if (cudaOccupancyMaxActiveClusters(&n, kernel, &cfg) != cudaSuccess) {
        cudaGetLastError();
        n = 0;
      }
      return n;
    };
    cache[dev].sms = sms;
    cache[dev].pairs = std::max(pairs, 0);
    cache[dev].top_p_clusters[0] = resident_clusters(top_p_kernel<2>, 2);
    cache[dev].top_p_clusters[1] = resident_clusters(top_p_kernel<4>, 4);
    cache[dev].top_p_clusters[2] = resident_clusters(top_p_kernel<8>, 8);
    cache[dev].top_p_clusters[3] = resident_clusters(top_p_kernel<16>, 16);  // 0: not available
    // the nucleus fast pass streams the stored logits through a shared-memory
    // ring (kFastSmem bytes); its grid is what can be resident at once
    int per_sm = 0;
    if (cudaFuncSetAttribute(top_p_fast_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kFastSmem) !=
            cudaSuccess ||
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, top_p_fast_kernel, kTopPThreads, kFastSmem) !=
            cudaSuccess)
      return false;
    cache[dev].fast_ctas = std::max(1, per_sm) * sms;
    cache[dev].ok = true;
  }
  *out = cache[dev];
  return true;
}

// ---------------------------------------------------------------- tracing

struct TraceRec {
  int32_t kind;
  int64_t cols;
  cudaEvent_t start, stop;
};

struct Tracer {
  std::mutex mu;
  bool on = false;
  std::vector<TraceRec> recs;   // recorded launches
  std::vector<cudaEvent_t> pool;  // created events, reused across records
  size_t used = 0;

  cudaEvent_t next_event() {
    if (used == pool.size()) {
      cudaEvent_t e = nullptr;
      if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
      pool.push_back(e);
    }
    return pool[used++];
  }
};

Tracer& tracer() {
  static Tracer* t = new Tracer();  // never destroyed: events may outlive static teardown
  return *t;
}

// Brackets the launches made in its lifetime with two events when tracing is on.
class TraceScope {
 public:
  TraceScope(int32_t kind, int64_t cols, cudaStream_t s) : s_(s) {
    Tracer& t = tracer();
    std::lock_guard<std::mutex> lk(t.mu);
    if (!t.on) return;
    rec_.kind = kind;
    rec_.cols = cols;
    rec_.start = t.next_event();
    rec_.stop = t.next_event();
    if (rec_.start && rec_.stop && cudaEventRecord(rec_.start, s) == cudaSuccess) active_ = true;
  }
  ~TraceScope() {
    if (!active_) return;
    Tracer& t = tracer();
    std::lock_guard<std::mutex> lk(t.mu);
    if (cudaEventRecord(rec_.stop, s_) == cudaSuccess) t.recs.push_back(rec_);
  }

 private:
  cudaStream_t s_;
  TraceRec rec_{};
  bool active_ = false;
};

// Copy-out stream of grpo_loss_fwd_bwd_to_host: one per device, created on
// first use (a driver object, not device memory) and shared by calls, which
// enqueue under `mu` so a ring event is never re-recorded before its wait.
struct CopyOut {
  std::mutex mu;
  cudaStream_t stream = nullptr;
  static constexpr int kRing = 4;
  cudaEvent_t ready[kRing] = {};
  cudaEvent_t done = nullptr;
  bool ok = false;
};

CopyOut* copy_out_for_device() {
  static std::mutex mu;
  static CopyOut* per_dev[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  std::lock_guard<std::mutex> lk(mu);
  if (!per_dev[dev]) {
    CopyOut* c = new CopyOut();
    bool ok = cudaStreamCreateWithFlags(&c->stream, cudaStreamNonBlocking) == cudaSuccess &&
              cudaEventCreateWithFlags(&c->done, cudaEventDisableTiming) == cudaSuccess;
    for (int i = 0; ok && i < CopyOut::kRing; ++i)
      ok = cudaEventCreateWithFlags(&c->ready[i], cudaEventDisableTiming) == cudaSuccess;
    c->ok = ok;
    per_dev[dev] = c;
  }
  return per_dev[dev]->ok ? per_dev[dev] : nullptr;
}

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// A bf16 row-major matrix [rows x cols] with leading dimension ld (elements),
// or, with blk, a K-major operand of `rows` rows and `cols` = K stored in
// k-blocks [cols / 64][rows][64] (ld unused; cols a multiple of 64).
struct Operand {
  const void* base;
  uint64_t rows, cols, ld;
  bool blk = false;
};

// The output of a kEpiDz (bf16) or kEpiF32 (fp32) GEMM: a row-major matrix
// [rows x cols], leading dimension ld elements; accumulator row r, column n
// lands at (r, n), and what lies outside rows x cols is not written.
struct OutMat {
  void* base;
  uint64_t rows, cols, ld;
};

// Builds the tensor maps of A, of each B (one per LM head; a.n_heads of them)
// and of the output D for the tile shape of kPair and launches the persistent
// GEMM with at most one CTA (pair) per work unit.
template <int kPair, int E, bool AMN, bool BMN>
cudaError_t launch_gemm_cfg(const Operand& A, const Operand* B, const GemmArgs& args, int64_t max_m_rows,
                            const DeviceInfo& di, cudaStream_t s, const OutMat* D) {
  using C = TileCfg<kPair>;
  GemmArgs a = args;
  a.n_heads = std::max(1, std::min(a.n_heads, kMaxHeads));
  // the k-block form of B exists only for the dW GEMMs (fp32 output or the AdamW step)
  constexpr bool kBlkOk = !BMN && (E == kEpiF32 || E == kEpiAdam);
  const bool blk = B[0].blk;
  if (blk && !kBlkOk) return cudaErrorInvalidValue;
  CUtensorMap ta, tb[kMaxHeads], td;
  if (!encode_2d(&ta, A.base, A.rows, A.cols, A.ld, kBK, AMN ? 64 : kRowsCta)) return cudaErrorInvalidValue;
  for (int h = 0; h < kMaxHeads; ++h) {
    if (h >= a.n_heads) {
      tb[h] = tb[0];
      continue;
    }
    const bool ok = B[h].blk ? !BMN && encode_blk(&tb[h], B[h].base, B[h].rows, B[h].cols, C::kBRows)
                             : encode_2d(&tb[h], B[h].base, B[h].rows, B[h].cols, B[h].ld, kBK, BMN ? 64 : C::kBRows);
    if (!ok) return cudaErrorInvalidValue;
  }
  // 32 x 32 boxes: 64-byte bf16 rows in the 64-byte swizzle, 128-byte fp32 rows in the 128-byte one
  auto out_map = [](CUtensorMap* m, const OutMat* o, bool f32) {
    return o && aligned(o->base, 16) &&
           encode_2d(m, o->base, o->rows, o->cols, o->ld, 32, 32, f32,
                     f32 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B);
  };
  if (E == kEpiAdam) {
    // D[0..3]: fp32 weights (the output map), first and second moments, bf16
    // weights; the moments and the bf16 weights ride in the unused B slots 1..3
    if (a.n_heads != 1 || !D || !out_map(&td, &D[0], true) || !out_map(&tb[1], &D[1], true) ||
        !out_map(&tb[2], &D[2], true) || !out_map(&tb[3], &D[3], false))
      return cudaErrorInvalidValue;
  } else if (EpiShape<E>::kTmaOut) {
    if (!out_map(&td, D, EpiShape<E>::kOutF32)) return cudaErrorInvalidValue;
  } else {
    td = ta;  // not read
  }
  const int64_t n_tiles = (a.N + kTileN - 1) / kTileN;
  const int64_t units = ((max_m_rows + C::kTileM - 1) / C::kTileM) *
                        ((n_tiles + a.n_per_unit - 1) / a.n_per_unit) * a.n_heads;
  const unsigned grid = static_cast<unsigned>(
      kPair == 2 ? 2 * std::max<int64_t>(1, std::min<int64_t>(di.pairs, units))
                 : std::max<int64_t>(1, std::min<int64_t>(di.sms, units)));
  GemmArgs ag = a;
  if (ag.gate) {
    gate_params(static_cast<int>(grid), &ag.gate_slack, &ag.gate_lag);
    if (ag.gate_slack <= 0 || grid > static_cast<unsigned>(kGateMaxCtas) || max_m_rows < kGateMinRows) {
      ag.gate = nullptr;
    } else {
      const cudaError_t e = cudaMemsetAsync(ag.gate, 0, grid * sizeof(int), s);
      if (e != cudaSuccess) return e;
    }
  }
  auto go = [&](auto blk_tag) {
    constexpr bool BLK = decltype(blk_tag)::value;
    if (kPair == 2)
      gemm_tc_pair_kernel<E, AMN, BMN, BLK><<<grid, EpiShape<E>::kThreads, smem_bytes<2, E>(), s>>>(
          ta, tb[0], tb[1], tb[2], tb[3], td, ag);
    else
      gemm_tc_kernel<E, AMN, BMN, BLK><<<grid, EpiShape<E>::kThreads, smem_bytes<1, E>(), s>>>(
          ta, tb[0], tb[1], tb[2], tb[3], td, ag);
  };
  if constexpr (kBlkOk) {
    if (blk) go(std::true_type{});
    else go(std::false_type{});
  } else {
    go(std::false_type{});
  }
  return cudaGetLastError();
}

template <int E, bool AMN, bool BMN>
cudaError_t launch_gemm(const Operand& A, const Operand* B, const GemmArgs& a, int64_t max_m_rows,
                        const DeviceInfo& di, cudaStream_t s, const OutMat* D = nullptr) {
  return use_pairs() && di.pairs > 0 ? launch_gemm_cfg<2, E, AMN, BMN>(A, B, a, max_m_rows, di, s, D)
                                     : launch_gemm_cfg<1, E, AMN, BMN>(A, B, a, max_m_rows, di, s, D);
}

template <int E, bool AMN, bool BMN>
cudaError_t launch_gemm(const Operand& A, const Operand& B, const GemmArgs& a, int64_t max_m_rows,
                        const DeviceInfo& di, cudaStream_t s, const OutMat* D = nullptr) {
  return launch_gemm<E, AMN, BMN>(A, &B, a, max_m_rows, di, s, D);
}

template <typename T>
T* at(void* ws, size_t off) {
  return reinterpret_cast<T*>(static_cast<char*>(ws) + off);
}


// The pointer the row gather reads H through: H itself for device (or
// managed) memory; for page-locked host memory registered with CUDA its
// device-side address, so the gather reads the unmasked rows over the host
// link and the masked ones never cross it; nullptr for memory the device
// cannot read (pageable host memory).
const uint16_t* hidden_view(const uint16_t* H) {
  cudaPointerAttributes pa{};
  if (cudaPointerGetAttributes(&pa, H) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  if (pa.type == cudaMemoryTypeHost) {
    if (!pa.devicePointer) return nullptr;
    // the device address of H itself, whether the attributes describe H or its allocation's start
    const ptrdiff_t off = pa.hostPointer ? reinterpret_cast<const char*>(H) - static_cast<const char*>(pa.hostPointer) : 0;
    return reinterpret_cast<const uint16_t*>(static_cast<const char*>(pa.devicePointer) + off);
  }
  if (pa.type == cudaMemoryTypeUnregistered) return nullptr;
  return H;
}

// Compaction of unmasked rows + gather of their hidden states and targets.
cudaError_t run_compaction(const uint16_t* H, const int32_t* targets, const uint8_t* mask, int64_t T,
                           int32_t Hd, int64_t V, void* ws, const Layout& Ly, int sms,
                           cudaStream_t s) {
  unsigned* status = at<unsigned>(ws, Ly.status);
  int* n_valid = at<int>(ws, Ly.n_valid);
  cudaError_t e = cudaMemsetAsync(status, 0, 8, s);  // status word and n_valid
  if (e != cudaSuccess) return e;
  TraceScope trace(GRPO_K_COMPACT, 0, s);
  if (T > 0 && T <= kScanChunk) {  // one block does all three steps
    mask_compact_small_kernel<<<1, kScanThreads, 0, s>>>(mask, T, static_cast<int>(Ly.rows), n_valid,
                                                         at<int>(ws, Ly.cidx), at<int>(ws, Ly.rank_of), status);
  } else if (T > 0) {
    const int nb = static_cast<int>(Ly.nblk_scan);
    mask_count_kernel<<<nb, kScanThreads, 0, s>>>(mask, T, at<int>(ws, Ly.counts));
    count_scan_kernel<<<1, 1024, 0, s>>>(at<int>(ws, Ly.counts), nb, at<int>(ws, Ly.offsets), n_valid,
                                         static_cast<int>(Ly.rows), status);
    mask_scatter_kernel<<<nb, kScanThreads, 0, s>>>(mask, T, at<int>(ws, Ly.offsets), static_cast<int>(Ly.rows),
                                                      at<int>(ws, Ly.cidx), at<int>(ws, Ly.rank_of));
  }
  const int64_t rows = Ly.rows;
  const int gblocks = static_cast<int>(std::max<int64_t>(1, std::min<int64_t>(rows / 8 + 1, sms * 8)));
  gather_rows_kernel<<<gblocks, 256, 0, s>>>(H, targets, at<int>(ws, Ly.cidx), n_valid, Hd, V,
                                             at<uint16_t>(ws, Ly.Hc), at<int>(ws, Ly.yc), status);
  return cudaGetLastError();
}

// Forward GEMM with the log-softmax epilogue over all V columns of each of
// the n_heads LM heads (one launch; the heads share the gathered hidden states).
// With a layout that keeps the logits (one head), they are stored as well.
cudaError_t run_lse(const uint16_t* const* W, int n_heads, int32_t Hd, int64_t V, void* ws, const Layout& Ly,
                    const DeviceInfo& di, cudaStream_t s) {
  GemmArgs a{};
  a.n_valid = at<int>(ws, Ly.n_valid);
  a.M = 0;
  a.m_dyn = 1;
  a.N = static_cast<int>(V);
  a.K = Hd;
  a.n_per_unit = Ly.lse_tiles;
  a.n_heads = n_heads;
  a.group_m = group_m(Ly.ldz > 0 ? 4 : 0);
  if (gate_on(0)) a.gate = at<int>(ws, Ly.gate);
  // Fault-injection test hook (failure-detection tests): GRPO_TEST_DROP_KBLOCK=k
  // makes CTA 0 skip the copies of its k-th k-block (1-based) so its pipeline
  // wait runs out after 0.2 s and the call reports GRPO_ERR_TIMEOUT.
  if (const char* d = std::getenv("GRPO_TEST_DROP_KBLOCK")) {
    a.drop_kblock1 = std::atoi(d);
    if (a.drop_kblock1 > 0) a.wait_ns = 200000000ull;
  }
  // gathered hidden states: re-read for every vocabulary tile (evict last);
  // W: streamed, shared by the CTAs of one round (evict first)
  l2_hints(0, &a.a_hint, &a.b_hint);
  a.status = at<unsigned>(ws, Ly.status);
  a.yc = at<int>(ws, Ly.yc);
  a.part_m = at<float>(ws, Ly.part_m);
  a.part_s = at<float>(ws, Ly.part_s);
  a.zy = at<float>(ws, Ly.zy);
  a.ldp = Ly.rows;
  const Operand A{at<uint16_t>(ws, Ly.Hc), static_cast<uint64_t>(Ly.rows), static_cast<uint64_t>(Hd),
                  static_cast<uint64_t>(Hd)};
  Operand B[kMaxHeads];
  for (int h = 0; h < n_heads; ++h)
    B[h] = Operand{W[h], static_cast<uint64_t>(V), static_cast<uint64_t>(Hd), static_cast<uint64_t>(Hd)};
  TraceScope trace(GRPO_K_LSE_GEMM, V * n_heads, s);
  if (Ly.ldz > 0) {
    if (n_heads != 1) return cudaErrorInvalidValue;
    const OutMat Z{at<float>(ws, Ly.z), static_cast<uint64_t>(Ly.rows), static_cast<uint64_t>(V),
                   static_cast<uint64_t>(Ly.ldz)};
    return launch_gemm<kEpiLseZ, false, false>(A, B, a, Ly.rows, di, s, &Z);
  }
  return launch_gemm<kEpiLse, false, false>(A, B, a, Ly.rows, di, s);
}

grpo_status from_cuda(cudaError_t e) { return e == cudaSuccess ? GRPO_OK : GRPO_ERR_CUDA; }

// AdamW step fused into the dW GEMM (grpo_loss_fwd_bwd_adamw).
struct AdamParams {
  float* master;
  float* exp_avg;
  float* exp_avg_sq;
  uint16_t* w_out;
  float b1, b2, eps, lr, decay, bc1, bc2;
};

grpo_status loss_impl(const uint16_t* H, const uint16_t* W, const int32_t* targets, const uint8_t* mask,
                      const float* old_logp, const float* ref_logp, const float* adv, int64_t n_resp,
                      int64_t L, int32_t Hd, int64_t V, float clip_eps, float beta, int32_t agg_mode,
                      float norm, float* loss_out, float* dH, float* dW, const AdamParams* adam, void* ws,
                      size_t ws_bytes, void* stream, float* dW_host = nullptr, float kl_clamp = INFINITY,
                      void* const* chunk_events = nullptr, int32_t n_events = 0);

}  // namespace

extern "C" {

const char* grpo_status_string(grpo_status st) {
  switch (st) {
    case GRPO_OK: return "GRPO_OK";
    case GRPO_ERR_INVALID_ARG: return "GRPO_ERR_INVALID_ARG";
    case GRPO_ERR_WORKSPACE: return "GRPO_ERR_WORKSPACE";
    case GRPO_ERR_CUDA: return "GRPO_ERR_CUDA";
    case GRPO_ERR_DEVICE_CHECK: return "GRPO_ERR_DEVICE_CHECK";
    case GRPO_ERR_TIMEOUT: return "GRPO_ERR_TIMEOUT";
    case GRPO_ERR_UNSUPPORTED: return "GRPO_ERR_UNSUPPORTED";
    case GRPO_ERR_CAPACITY: return "GRPO_ERR_CAPACITY";
  }
  return "GRPO_ERR_UNKNOWN";
}

size_t grpo_workspace_bytes_rows(int64_t T, int64_t max_valid, int32_t Hd, int64_t V, int32_t which) {
  Layout L;
  if (max_valid < 0) return 0;
  return make_layout(T, Hd, V, which, &L, max_valid) ? L.total : 0;
}

size_t grpo_workspace_bytes(int64_t T, int32_t Hd, int64_t V, int32_t which) {
  Layout L;
  return make_layout(T, Hd, V, which, &L) ? L.total : 0;
}

int32_t grpo_loss_plan(int64_t T, int32_t Hd, int64_t V, size_t ws_bytes, int64_t* rows) {
  Layout L;
  if (!fit_loss_layout(T, Hd, V, ws_bytes, &L)) return -1;
  if (rows) *rows = L.rows;
  return L.ldz > 0 ? 1 : 0;
}

grpo_status grpo_group_advantages(const float* rewards, int64_t n_resp, int32_t G, float eps,
                                  float* adv_out, void* stream) {
  if (G < 2 || n_resp < 0 || n_resp % G != 0) return GRPO_ERR_INVALID_ARG;
  if (n_resp == 0) return GRPO_OK;
  if (!rewards || !adv_out) return GRPO_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  TraceScope trace(GRPO_K_ADVANTAGES, 0, s);
  if (G <= 32 && (G & (G - 1)) == 0) {
    const int64_t blocks = (n_resp + 255) / 256;
    adv_segmented_kernel<<<static_cast<unsigned>(blocks), 256, 0, s>>>(rewards, n_resp, G, eps, adv_out);
  } else {
    const int64_t groups = n_resp / G;
    const int64_t blocks = (groups * 32 + 255) / 256;
    adv_warp_kernel<<<static_cast<unsigned>(blocks), 256, 0, s>>>(rewards, groups, G, eps, adv_out);
  }
  return from_cuda(cudaGetLastError());
}

grpo_status grpo_token_logprobs(const uint16_t* H, const uint16_t* W, const int32_t* targets,
                                const uint8_t* mask, int64_t T, int32_t Hd, int64_t V,
                                float* logp_out, void* ws, size_t ws_bytes, void* stream) {
  Layout Ly;
  if (!make_layout(T, Hd, V, GRPO_WS_LOGPROBS, &Ly)) return GRPO_ERR_INVALID_ARG;
  if (!W) return GRPO_ERR_INVALID_ARG;
  if (T > 0 && (!H || !targets || !mask || !logp_out)) return GRPO_ERR_INVALID_ARG;
  if (!aligned(W, 16) || (H && !aligned(H, 16))) return GRPO_ERR_INVALID_ARG;
  if (!ws || !aligned(ws, 256) || !fit_layout(T, Hd, V, GRPO_WS_LOGPROBS, ws_bytes, &Ly))
    return GRPO_ERR_WORKSPACE;
  if (T == 0) return GRPO_OK;
  DeviceInfo di;
  if (!device_info(&di)) return GRPO_ERR_UNSUPPORTED;
  if (!get_encode()) return GRPO_ERR_CUDA;
  if (!(H = hidden_view(H))) return GRPO_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e = run_compaction(H, targets, mask, T, Hd, V, ws, Ly, di.sms, s);
  if (e == cudaSuccess) e = run_lse(&W, 1, Hd, V, ws, Ly, di, s);
  if (e == cudaSuccess) {
    const int blocks = static_cast<int>(std::min<int64_t>((T + 7) / 8, di.sms * 16));  // a warp per row
    TraceScope trace(GRPO_K_LOGP_MERGE, 0, s);
    logp_merge_kernel<<<blocks, 256, 0, s>>>(mask, at<int>(ws, Ly.rank_of), T, at<float>(ws, Ly.part_m),
                                             at<float>(ws, Ly.part_s), static_cast<int>(Ly.nsplit),
                                             Ly.rows, at<float>(ws, Ly.zy), at<int>(ws, Ly.yc),
                                             logp_out, at<unsigned>(ws, Ly.status));
    e = cudaGetLastError();
  }
  return from_cuda(e);
}

grpo_status grpo_token_logprobs_heads(const uint16_t* H, const uint16_t* const* W_heads, int32_t n_heads,
                                      const int32_t* targets, const uint8_t* mask, int64_t T, int32_t Hd,
                                      int64_t V, float* logp_out, void* ws, size_t ws_bytes, void* stream) {
  Layout Ly;
  if (!make_layout(T, Hd, V, GRPO_WS_LOGPROBS_HEADS, &Ly)) return GRPO_ERR_INVALID_ARG;
  if (n_heads < 1 || n_heads > kMaxHeads || !W_heads) return GRPO_ERR_INVALID_ARG;
  for (int h = 0; h < n_heads; ++h)
    if (!W_heads[h] || !aligned(W_heads[h], 16)) return GRPO_ERR_INVALID_ARG;
  if (T > 0 && (!H || !targets || !mask || !logp_out)) return GRPO_ERR_INVALID_ARG;
  if (H && !aligned(H, 16)) return GRPO_ERR_INVALID_ARG;
  if (!ws || !aligned(ws, 256) || !fit_layout(T, Hd, V, GRPO_WS_LOGPROBS_HEADS, ws_bytes, &Ly))
    return GRPO_ERR_WORKSPACE;
  if (T == 0) return GRPO_OK;
  DeviceInfo di;
  if (!device_info(&di)) return GRPO_ERR_UNSUPPORTED;
  if (!get_encode()) return GRPO_ERR_CUDA;
  if (!(H = hidden_view(H))) return GRPO_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e = run_compaction(H, targets, mask, T, Hd, V, ws, Ly, di.sms, s);
  if (e == cudaSuccess) e = run_lse(W_heads, n_heads, Hd, V, ws, Ly, di, s);
  if (e == cudaSuccess) {
    const int blocks = static_cast<int>(std::min<int64_t>((T + 7) / 8, di.sms * 16));  // a warp per row
    TraceScope trace(GRPO_K_LOGP_MERGE, 0, s);
    for (int h = 0; h < n_heads && e == cudaSuccess; ++h) {
      const size_t head_parts = static_cast<size_t>(h) * Ly.nsplit * Ly.rows;
      logp_merge_kernel<<<blocks, 256, 0, s>>>(mask, at<int>(ws, Ly.rank_of), T, at<float>(ws, Ly.part_m) + head_parts,
                                               at<float>(ws, Ly.part_s) + head_parts, static_cast<int>(Ly.nsplit),
                                               Ly.rows, at<float>(ws, Ly.zy) + static_cast<size_t>(h) * Ly.rows,
                                               at<int>(ws, Ly.yc), logp_out + static_cast<size_t>(h) * T,
                                               at<unsigned>(ws, Ly.status));
      e = cudaGetLastError();
    }
  }
  return from_cuda(e);
}

grpo_status grpo_sample_tokens(const uint16_t* H, const uint16_t* W, const uint8_t* mask, int64_t T, int32_t Hd,
                               int64_t V, float temperature, uint64_t seed, uint64_t offset, int32_t* tokens_out,
                               float* logp_out, void* ws, size_t ws_bytes, void* stream) {
  Layout Ly;
  if (!make_layout(T, Hd, V, GRPO_WS_SAMPLE, &Ly)) return GRPO_ERR_INVALID_ARG;
  if (!W || !aligned(W, 16)) return GRPO_ERR_INVALID_ARG;
  if (T > 0 && (!H || !mask || !tokens_out || !logp_out)) return GRPO_ERR_INVALID_ARG;
  if (H && !aligned(H, 16)) return GRPO_ERR_INVALID_ARG;
  if (!(temperature > 0.f) || !(temperature < INFINITY)) return GRPO_ERR_INVALID_ARG;
  if (!ws || !aligned(ws, 256) || !fit_layout(T, Hd, V, GRPO_WS_SAMPLE, ws_bytes, &Ly))
    return GRPO_ERR_WORKSPACE;
  if (T == 0) return GRPO_OK;
  DeviceInfo di;
  if (!device_info(&di)) return GRPO_ERR_UNSUPPORTED;
  if (!get_encode()) return GRPO_ERR_CUDA;
  if (!(H = hidden_view(H))) return GRPO_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e = run_compaction(H, nullptr, mask, T, Hd, V, ws, Ly, di.sms, s);
  if (e == cudaSuccess) {
    GemmArgs a{};
    a.n_valid = at<int>(ws, Ly.n_valid);
    a.m_dyn = 1;
    a.N = static_cast<int>(V);
    a.K = Hd;
    a.n_per_unit = Ly.lse_tiles;
    a.n_heads = 1;
    a.group_m = group_m(0);
    if (gate_on(0)) a.gate = at<int>(ws, Ly.gate);
    l2_hints(0, &a.a_hint, &a.b_hint);
    a.status = at<unsigned>(ws, Ly.status);
    a.row_map = at<int>(ws, Ly.cidx);
    a.part_m = at<float>(ws, Ly.part_m);
    a.part_s = at<float>(ws, Ly.part_s);
    a.best_s = at<float>(ws, Ly.best_s);
    a.best_c = at<int>(ws, Ly.best_c);
    a.best_z = at<float>(ws, Ly.best_z);
    a.ldp = Ly.rows;
    a.inv_temp = 1.f / temperature;
    a.seed_lo = static_cast<uint32_t>(seed);
    a.seed_hi = static_cast<uint32_t>(seed >> 32);
    a.off_lo = static_cast<uint32_t>(offset);
    a.off_hi = static_cast<uint32_t>(offset >> 32);
    const Operand A{at<uint16_t>(ws, Ly.Hc), static_cast<uint64_t>(Ly.rows), static_cast<uint64_t>(Hd),
                    static_cast<uint64_t>(Hd)};
    const Operand B{W, static_cast<uint64_t>(V), static_cast<uint64_t>(Hd), static_cast<uint64_t>(Hd)};
    TraceScope trace(GRPO_K_SAMPLE_GEMM, V, s);
    e = launch_gemm<kEpiSample, false, false>(A, B, a, Ly.rows, di, s);
  }
  if (e == cudaSuccess) {
    const int blocks = static_cast<int>(std::min<int64_t>((T + 7) / 8, di.sms * 16));  // a warp per row
    TraceScope trace(GRPO_K_LOGP_MERGE, 0, s);
    sample_merge_kernel<<<blocks, 256, 0, s>>>(mask, at<int>(ws, Ly.rank_of), T, at<float>(ws, Ly.part_m),
                                               at<float>(ws, Ly.part_s), at<float>(ws, Ly.best_s),
                                               at<int>(ws, Ly.best_c), at<float>(ws, Ly.best_z),
                                               static_cast<int>(Ly.nsplit), Ly.rows, tokens_out, logp_out,
                                               at<unsigned>(ws, Ly.status));
    e = cudaGetLastError();
  }
  return from_cuda(e);
}

grpo_status grpo_sample_tokens_top_p(const uint16_t* H, const uint16_t* W, const uint8_t* mask, int64_t T,
                                     int32_t Hd, int64_t V, float temperature, float top_p, uint64_t seed,
                                     uint64_t offset, int32_t* tokens_out, float* logp_out, void* ws, size_t ws_bytes,
                                     void* stream) {
  Layout Ly;
  if (!make_layout(T, Hd, V, GRPO_WS_SAMPLE_TOP_P, &Ly)) return GRPO_ERR_INVALID_ARG;
  if (!W || !aligned(W, 16)) return GRPO_ERR_INVALID_ARG;
  if (T > 0 && (!H || !mask || !tokens_out || !logp_out)) return GRPO_ERR_INVALID_ARG;
  if (H && !aligned(H, 16)) return GRPO_ERR_INVALID_ARG;
  if (!(temperature > 0.f) || !(temperature < INFINITY) || !(top_p > 0.f) || !(top_p <= 1.f))
    return GRPO_ERR_INVALID_ARG;
  if (!ws || !aligned(ws, 256) || !fit_layout(T, Hd, V, GRPO_WS_SAMPLE_TOP_P, ws_bytes, &Ly))
    return GRPO_ERR_WORKSPACE;
  if (T == 0) return GRPO_OK;
  DeviceInfo di;
  if (!device_info(&di)) return GRPO_ERR_UNSUPPORTED;
  if (!get_encode()) return GRPO_ERR_CUDA;
  if (!(H = hidden_view(H))) return GRPO_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // the sampling GEMM (running LSE and the plain Gumbel-max winner per split),
  // storing the logits of every unmasked row for the nucleus selection
  cudaError_t e = run_compaction(H, nullptr, mask, T, Hd, V, ws, Ly, di.sms, s);
  if (e == cudaSuccess) {
    GemmArgs a{};
    a.n_valid = at<int>(ws, Ly.n_valid);
    a.m_dyn = 1;
    a.N = static_cast<int>(V);
    a.K = Hd;
    a.n_per_unit = Ly.lse_tiles;
    a.n_heads = 1;
    a.group_m = group_m(4);
    if (gate_on(0)) a.gate = at<int>(ws, Ly.gate);
    l2_hints(0, &a.a_hint, &a.b_hint);
    a.status = at<unsigned>(ws, Ly.status);
    a.row_map = at<int>(ws, Ly.cidx);
    a.part_m = at<float>(ws, Ly.part_m);
    a.part_s = at<float>(ws, Ly.part_s);
    a.best_s = at<float>(ws, Ly.best_s);
    a.best_c = at<int>(ws, Ly.best_c);
    a.best_z = at<float>(ws, Ly.best_z);
    a.ldp = Ly.rows;
    a.inv_temp = 1.f / temperature;
    a.seed_lo = static_cast<uint32_t>(seed);
    a.seed_hi = static_cast<uint32_t>(seed >> 32);
    a.off_lo = static_cast<uint32_t>(offset);
    a.off_hi = static_cast<uint32_t>(offset >> 32);
    const Operand A{at<uint16_t>(ws, Ly.Hc), static_cast<uint64_t>(Ly.rows), static_cast<uint64_t>(Hd),
                    static_cast<uint64_t>(Hd)};
    const Operand B{W, static_cast<uint64_t>(V), static_cast<uint64_t>(Hd), static_cast<uint64_t>(Hd)};
    const OutMat Z{at<float>(ws, Ly.z), static_cast<uint64_t>(Ly.rows), static_cast<uint64_t>(V),
                   static_cast<uint64_t>(Ly.ldz)};
    TraceScope trace(GRPO_K_SAMPLE_GEMM, V, s);
    e = launch_gemm<kEpiSampleZ, false, false>(A, B, a, Ly.rows, di, s, &Z);
  }
  if (e == cudaSuccess) {
    TraceScope trace(GRPO_K_TOP_P, V, s);
    const int fb = static_cast<int>(std::min<int64_t>((T + 255) / 256, int64_t(di.sms) * 16));
    top_p_fill_kernel<<<fb, 256, 0, s>>>(mask, at<int>(ws, Ly.rank_of), T, tokens_out, logp_out);
    // the plain draw of every unmasked row, and per row what the selection needs
    // (workspace arrays the sampling path leaves unused: LSE, the winner's y,
    // the row maximum)
    float* lse_r = at<float>(ws, Ly.lse_c);
    float* y0_r = at<float>(ws, Ly.g_c);
    float* hi_r = at<float>(ws, Ly.zy);
    const int pb = static_cast<int>(std::min<int64_t>((Ly.rows + 7) / 8, int64_t(di.sms) * 8));
    top_p_prep_kernel<<<pb, 256, 0, s>>>(at<int>(ws, Ly.n_valid), at<int>(ws, Ly.cidx), at<float>(ws, Ly.part_m),
                                         at<float>(ws, Ly.part_s), at<float>(ws, Ly.best_s),
                                         at<int>(ws, Ly.best_c), at<float>(ws, Ly.best_z),
                                         static_cast<int>(Ly.nsplit), Ly.rows, lse_r, y0_r, hi_r,
                                         at<unsigned long long>(ws, Ly.row_above), at<unsigned>(ws, Ly.row_done),
                                         tokens_out, logp_out, at<unsigned>(ws, Ly.status));
    e = cudaGetLastError();
    if (e == cudaSuccess && top_p < 1.f) {
      unsigned* n_slow = at<unsigned>(ws, Ly.n_slow);
      e = cudaMemsetAsync(n_slow, 0, 4, s);
      // is the winner in the nucleus?  every CTA that can be resident, each
      // over one contiguous range of the rows' logit chunks (the unmasked row
      // count is only known on the device; CTAs past the work return at once)
      // test hook: GRPO_TEST_TOP_P_LIST_ALL=1 lists every row (a margin above
      // any mass), so the selection's exact confirmation decides each one
      unsigned long long margin = top_p_margin(V);
      if (const char* h = std::getenv("GRPO_TEST_TOP_P_LIST_ALL"))
        if (h[0] == '1') margin = 1ull << 42;
      if (e == cudaSuccess)
        top_p_fast_kernel<<<di.fast_ctas, kTopPThreads, kFastSmem, s>>>(
            at<float>(ws, Ly.z), Ly.ldz, static_cast<int>(V), at<int>(ws, Ly.n_valid), lse_r, y0_r,
            1.f / temperature, top_p, at<unsigned long long>(ws, Ly.row_above), at<unsigned>(ws, Ly.row_done),
            at<int>(ws, Ly.slow_rows), at<unsigned long long>(ws, Ly.slow_tgt), n_slow, margin,
            at<unsigned>(ws, Ly.status));
      // the rows whose winner falls outside: clusters of 2, 4 or 8 CTAs, one
      // row per cluster at a time, as many clusters as can be resident together
      int lg = top_p_cluster_log2(Ly.rows, top_p);
      while (lg > 1 && di.top_p_clusters[lg - 1] <= 0) --lg;  // a size this device cannot place
      const int64_t clusters = std::max<int64_t>(1, std::min<int64_t>(Ly.rows, di.top_p_clusters[lg - 1]));
      const int rb = static_cast<int>(clusters << lg);
      auto select = [&](auto kernel) {
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = 1u << lg;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(static_cast<unsigned>(rb), 1, 1);
        cfg.blockDim = dim3(kTopPThreads, 1, 1);
        cfg.stream = s;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        return cudaLaunchKernelEx(
            &cfg, kernel, at<float>(ws, Ly.z), Ly.ldz, static_cast<int>(V), reinterpret_cast<const int*>(n_slow),
            static_cast<const int*>(at<int>(ws, Ly.slow_rows)),
            static_cast<const unsigned long long*>(at<unsigned long long>(ws, Ly.slow_tgt)),
            static_cast<const int*>(at<int>(ws, Ly.cidx)), static_cast<const float*>(lse_r),
            static_cast<const float*>(y0_r), static_cast<const float*>(hi_r),
            static_cast<const float*>(at<float>(ws, Ly.best_s)), static_cast<const int*>(at<int>(ws, Ly.best_c)),
            static_cast<const float*>(at<float>(ws, Ly.best_z)), static_cast<int>(Ly.nsplit),
            static_cast<long>(Ly.rows), Ly.lse_tiles, 1.f / temperature, static_cast<uint32_t>(seed),
            static_cast<uint32_t>(seed >> 32), static_cast<uint32_t>(offset), static_cast<uint32_t>(offset >> 32),
            tokens_out, logp_out, at<unsigned>(ws, Ly.status));
      };
      if (e == cudaSuccess) {
        if (lg == 1) e = select(top_p_kernel<2>);
        else if (lg == 2) e = select(top_p_kernel<4>);
        else if (lg == 3) e = select(top_p_kernel<8>);
        else e = select(top_p_kernel<16>);
      }
      if (e == cudaSuccess) e = cudaGetLastError();
    }
  }
  return from_cuda(e);
}

grpo_status grpo_gumbel_noise(uint64_t seed, uint64_t offset, int64_t row0, int64_t rows, int64_t cols,
                              float* out, void* stream) {
  if (row0 < 0 || rows < 0 || cols < 0 || row0 > (int64_t(1) << 32) - rows || cols >= (int64_t(1) << 31))
    return GRPO_ERR_INVALID_ARG;
  if (rows > 0 && cols > 0 && rows > (int64_t(1) << 40) / cols) return GRPO_ERR_INVALID_ARG;
  if (rows == 0 || cols == 0) return GRPO_OK;
  if (!out || !aligned(out, 4)) return GRPO_ERR_INVALID_ARG;
  DeviceInfo di;
  if (!device_info(&di)) return GRPO_ERR_UNSUPPORTED;
  const int64_t work = rows * ((cols + 3) / 4);
  const int blocks = static_cast<int>(std::min<int64_t>((work + 255) / 256, int64_t(di.sms) * 16));
  gumbel_noise_kernel<<<blocks, 256, 0, static_cast<cudaStream_t>(stream)>>>(
      static_cast<uint32_t>(seed), static_cast<uint32_t>(seed >> 32), static_cast<uint32_t>(offset),
      static_cast<uint32_t>(offset >> 32), row0, rows, cols, out);
  return from_cuda(cudaGetLastError());
}

grpo_status grpo_loss_fwd_bwd(const uint16_t* H, const uint16_t* W, const int32_t* targets,
                              const uint8_t* mask, const float* old_logp, const float* ref_logp,
                              const float* adv, int64_t n_resp, int64_t L, int32_t Hd, int64_t V,
                              float clip_eps, float beta, int32_t agg_mode, float* loss_out,
                              float* dH, float* dW, void* ws, size_t ws_bytes, void* stream) {
  return grpo_loss_fwd_bwd_norm(H, W, targets, mask, old_logp, ref_logp, adv, n_resp, L, Hd, V, clip_eps,
                                beta, agg_mode, 0.f, loss_out, dH, dW, ws, ws_bytes, stream);
}

grpo_status grpo_loss_fwd_bwd_norm(const uint16_t* H, const uint16_t* W, const int32_t* targets,
                                   const uint8_t* mask, const float* old_logp, const float* ref_logp,
                                   const float* adv, int64_t n_resp, int64_t L, int32_t Hd, int64_t V,
                                   float clip_eps, float beta, int32_t agg_mode, float norm,
                                   float* loss_out, float* dH, float* dW, void* ws, size_t ws_bytes,
                                   void* stream) {
  return loss_impl(H, W, targets, mask, old_logp, ref_logp, adv, n_resp, L, Hd, V, clip_eps, beta, agg_mode,
                   norm, loss_out, dH, dW, nullptr, ws, ws_bytes, stream);
}

grpo_status grpo_loss_fwd_bwd_kl_clamp(const uint16_t* H, const uint16_t* W, const int32_t* targets,
                                       const uint8_t* mask, const float* old_logp, const float* ref_logp,
                                       const float* adv, int64_t n_resp, int64_t L, int32_t Hd, int64_t V,
                                       float clip_eps, float beta, int32_t agg_mode, float norm, float kl_clamp,
                                       float* loss_out, float* dH, float* dW, void* ws, size_t ws_bytes,
                                       void* stream) {
  return loss_impl(H, W, targets, mask, old_logp, ref_logp, adv, n_resp, L, Hd, V, clip_eps, beta, agg_mode,
                   norm, loss_out, dH, dW, nullptr, ws, ws_bytes, stream, nullptr, kl_clamp);
}

int64_t grpo_vocab_chunk_cols(int64_t V) { return V > 0 ? vocab_chunk(V) : 0; }

grpo_status grpo_loss_fwd_bwd_events(const uint16_t* H, const uint16_t* W, const int32_t* targets,
                                     const uint8_t* mask, const float* old_logp, const float* ref_logp,
                                     const float* adv, int64_t n_resp, int64_t L, int32_t Hd, int64_t V,
                                     float clip_eps, float beta, int32_t agg_mode, float norm, float* loss_out,
                                     float* dH, float* dW, void* const* chunk_events, int32_t n_events, void* ws,
                                     size_t ws_bytes, void* stream) {
  if (!chunk_events) return GRPO_ERR_INVALID_ARG;
  return loss_impl(H, W, targets, mask, old_logp, ref_logp, adv, n_resp, L, Hd, V, clip_eps, beta, agg_mode,
                   norm, loss_out, dH, dW, nullptr, ws, ws_bytes, stream, nullptr, INFINITY, chunk_events,
                   n_events);
}

grpo_status grpo_loss_fwd_bwd_to_host(const uint16_t* H, const uint16_t* W, const int32_t* targets,
                                      const uint8_t* mask, const float* old_logp, const float* ref_logp,
                                      const float* adv, int64_t n_resp, int64_t L, int32_t Hd, int64_t V,
                                      float clip_eps, float beta, int32_t agg_mode, float norm, float* loss_out,
                                      float* dH, float* dW, float* dW_host, void* ws, size_t ws_bytes,
                                      void* stream) {
  if (!dW_host || !aligned(dW_host, 16)) return GRPO_ERR_INVALID_ARG;
  return loss_impl(H, W, targets, mask, old_logp, ref_logp, adv, n_resp, L, Hd, V, clip_eps, beta, agg_mode,
                   norm, loss_out, dH, dW, nullptr, ws, ws_bytes, stream, dW_host);
}

grpo_status grpo_loss_fwd_bwd_adamw(const uint16_t* H, const uint16_t* W, const int32_t* targets,
                                    const uint8_t* mask, const float* old_logp, const float* ref_logp,
                                    const float* adv, int64_t n_resp, int64_t L, int32_t Hd, int64_t V,
                                    float clip_eps, float beta, int32_t agg_mode, float norm, float lr,
                                    float beta1, float beta2, float eps, float weight_decay, int64_t step,
                                    float* W_master, float* exp_avg, float* exp_avg_sq, uint16_t* W_out,
                                    float* loss_out, float* dH, void* ws, size_t ws_bytes, void* stream) {
  if (!W_master || !exp_avg || !exp_avg_sq || !W_out || !aligned(W_master, 16) || !aligned(exp_avg, 16) ||
      !aligned(exp_avg_sq, 16) || !aligned(W_out, 16))
    return GRPO_ERR_INVALID_ARG;
  if (step < 1 || !(lr >= 0.f) || !(beta1 >= 0.f && beta1 < 1.f) || !(beta2 >= 0.f && beta2 < 1.f) ||
      !(eps > 0.f) || !(weight_decay >= 0.f))
    return GRPO_ERR_INVALID_ARG;
  AdamParams ap{};
  ap.master = W_master;
  ap.exp_avg = exp_avg;
  ap.exp_avg_sq = exp_avg_sq;
  ap.w_out = W_out;
  ap.b1 = beta1;
  ap.b2 = beta2;
  ap.eps = eps;
  ap.lr = lr;
  ap.decay = static_cast<float>(1.0 - static_cast<double>(lr) * weight_decay);
  ap.bc1 = static_cast<float>(1.0 / (1.0 - std::pow(static_cast<double>(beta1), static_cast<double>(step))));
  ap.bc2 = static_cast<float>(1.0 / (1.0 - std::pow(static_cast<double>(beta2), static_cast<double>(step))));
  // dW is not stored: pass the master weights as a placeholder output pointer
  return loss_impl(H, W, targets, mask, old_logp, ref_logp, adv, n_resp, L, Hd, V, clip_eps, beta, agg_mode,
                   norm, loss_out, dH, W_master, &ap, ws, ws_bytes, stream);
}

}  // extern "C"

namespace {

grpo_status loss_impl(const uint16_t* H, const uint16_t* W, const int32_t* targets, const uint8_t* mask,
                      const float* old_logp, const float* ref_logp, const float* adv, int64_t n_resp,
                      int64_t L, int32_t Hd, int64_t V, float clip_eps, float beta, int32_t agg_mode,
                      float norm, float* loss_out, float* dH, float* dW, const AdamParams* adam, void* ws,
                      size_t ws_bytes, void* stream, float* dW_host, float kl_clamp, void* const* chunk_events,
                      int32_t n_events) {
  if (n_resp < 1 || L < 1 || n_resp > (int64_t(1) << 31) / L) return GRPO_ERR_INVALID_ARG;
  if (!(norm >= 0.f) || norm == INFINITY) return GRPO_ERR_INVALID_ARG;
  if (!(kl_clamp >= 0.f)) return GRPO_ERR_INVALID_ARG;
  const int64_t T = n_resp * L;
  Layout Ly;
  if (!make_layout(T, Hd, V, GRPO_WS_LOSS, &Ly)) return GRPO_ERR_INVALID_ARG;
  if (!H || !W || !targets || !mask || !old_logp || !ref_logp || !adv || !loss_out || !dH || !dW)
    return GRPO_ERR_INVALID_ARG;
  if (!(clip_eps >= 0.f) || !(beta == beta) || (agg_mode != GRPO_AGG_TOKEN_MEAN && agg_mode != GRPO_AGG_SEQ_MEAN))
    return GRPO_ERR_INVALID_ARG;
  if (!aligned(W, 16) || !aligned(H, 16) || !aligned(dH, 16) || !aligned(dW, 16))
    return GRPO_ERR_INVALID_ARG;
  if (!ws || !aligned(ws, 256) || !fit_loss_layout(T, Hd, V, ws_bytes, &Ly))
    return GRPO_ERR_WORKSPACE;
  if (chunk_events) {
    const int64_t chunks = (V + Ly.vchunk - 1) / Ly.vchunk;
    if (n_events < chunks) return GRPO_ERR_INVALID_ARG;
    for (int64_t c = 0; c < chunks; ++c)
      if (!chunk_events[c]) return GRPO_ERR_INVALID_ARG;
  }
  DeviceInfo di;
  if (!device_info(&di)) return GRPO_ERR_UNSUPPORTED;
  if (!get_encode()) return GRPO_ERR_CUDA;
  if (!(H = hidden_view(H))) return GRPO_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int sms = di.sms;
  int* n_valid = at<int>(ws, Ly.n_valid);
  unsigned* status = at<unsigned>(ws, Ly.status);

  cudaError_t e = run_compaction(H, targets, mask, T, Hd, V, ws, Ly, sms, s);
  if (e == cudaSuccess && agg_mode == GRPO_AGG_SEQ_MEAN) {
    TraceScope trace(GRPO_K_COMPACT, 0, s);
    const int64_t blocks = (n_resp * 32 + 255) / 256;
    resp_len_kernel<<<static_cast<unsigned>(blocks), 256, 0, s>>>(mask, n_resp, L, at<int>(ws, Ly.resp_len));
    e = cudaGetLastError();
  }
  const bool hct_blk = hct_blocks(Ly.rows);
  if (e == cudaSuccess) {
    TraceScope trace(GRPO_K_TRANSPOSE, 0, s);
    const int tb = static_cast<int>(std::min<int64_t>(Ly.rows / 64 * (Hd / 64), int64_t(sms) * 8));
    transpose_rows_kernel<<<tb, 256, 0, s>>>(at<uint16_t>(ws, Ly.Hc), n_valid, Hd, hct_blk ? 0 : Ly.rows,
                                             at<uint16_t>(ws, Ly.HcT));
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) e = run_lse(&W, 1, Hd, V, ws, Ly, di, s);
  if (e == cudaSuccess) {
    TraceScope trace(GRPO_K_LOSS, 0, s);
    loss_terms_kernel<<<static_cast<unsigned>(Ly.nblk_loss), kLossThreads, 0, s>>>(
        at<int>(ws, Ly.cidx), n_valid, at<float>(ws, Ly.part_m), at<float>(ws, Ly.part_s),
        static_cast<int>(Ly.nsplit), Ly.rows, at<float>(ws, Ly.zy), at<int>(ws, Ly.yc), old_logp,
        ref_logp, adv, L, at<int>(ws, Ly.resp_len), n_resp, agg_mode, norm, clip_eps, beta, kl_clamp,
        at<float>(ws, Ly.lse_c), at<float>(ws, Ly.g_c), at<double>(ws, Ly.block_loss), status);
    loss_final_kernel<<<1, 1024, 0, s>>>(at<double>(ws, Ly.block_loss), n_valid, kLossThreads, loss_out);
    e = cudaGetLastError();
  }
  if (e != cudaSuccess) return from_cuda(e);

  // Backward, one vocabulary chunk at a time.  With dW_host, each finished dW
  // chunk is copied to the host on the copy-out stream while the next chunks
  // compute; `s` waits for the last copy at the end.
  CopyOut* co = nullptr;
  std::unique_lock<std::mutex> co_lock;
  if (dW_host && !adam) {
    co = copy_out_for_device();
    if (!co) return GRPO_ERR_CUDA;
    co_lock = std::unique_lock<std::mutex>(co->mu);
  }
  int chunk = 0;
  uint16_t* Hc = at<uint16_t>(ws, Ly.Hc);
  uint16_t* dz = at<uint16_t>(ws, Ly.dz);
  float* dHc = at<float>(ws, Ly.dhc);
  const int64_t vc = Ly.vchunk;
  const uint64_t tp = static_cast<uint64_t>(Ly.rows), hd = static_cast<uint64_t>(Hd);  // compacted rows
  const Operand opHc{Hc, tp, hd, hd};
  const Operand opHcT{at<uint16_t>(ws, Ly.HcT), hd, tp, tp, hct_blk};
  const Operand opW{W, static_cast<uint64_t>(V), hd, hd};
  const Operand opDz{dz, tp, static_cast<uint64_t>(vc), static_cast<uint64_t>(vc)};
  const OutMat outDz{dz, tp, static_cast<uint64_t>(vc), static_cast<uint64_t>(vc)};
  const OutMat outDh{dHc, tp, hd, hd};
  for (int64_t c0 = 0; c0 < V && e == cudaSuccess; c0 += vc) {
    const int64_t width = std::min<int64_t>(vc, V - c0);
    if (Ly.ldz > 0) {  // dZ chunk = g (onehot - softmax) from the logits the forward kept
      TraceScope trace(GRPO_K_DZ_LOGITS, width, s);
      const int blocks = static_cast<int>(std::min<int64_t>(Ly.rows, int64_t(sms) * 8));
      dz_from_logits_kernel<<<blocks, 256, 0, s>>>(at<float>(ws, Ly.z), Ly.ldz, at<float>(ws, Ly.lse_c),
                                                   at<float>(ws, Ly.g_c), at<int>(ws, Ly.yc), n_valid, Ly.rows,
                                                   c0, static_cast<int>(width), static_cast<int>(vc), dz);
      e = cudaGetLastError();
    } else {  // dZ chunk = g (onehot - softmax) from recomputed logits
      GemmArgs a{};
      a.n_valid = n_valid;
      a.m_dyn = 1;
      a.N = static_cast<int>(width);
      a.K = Hd;
      a.b_off_n = static_cast<int>(c0);
      a.n_per_unit = units_n(0);
      a.group_m = group_m(1);
      a.group_n = group_n(1);
      if (gate_on(1)) a.gate = at<int>(ws, Ly.gate);
      l2_hints(1, &a.a_hint, &a.b_hint);
      a.status = status;
      a.yc = at<int>(ws, Ly.yc);
      a.lse = at<float>(ws, Ly.lse_c);
      a.gcoef = at<float>(ws, Ly.g_c);
      TraceScope trace(GRPO_K_DZ_GEMM, width, s);
      e = launch_gemm<kEpiDz, false, false>(opHc, opW, a, Ly.rows, di, s, &outDz);
    }
    if (e != cudaSuccess) break;
    {  // dHc (+)= dZ_c W_c: stored by the first chunk, added at L2 by the others
      GemmArgs h{};
      h.n_valid = n_valid;
      h.m_dyn = 1;
      h.N = Hd;
      h.K = static_cast<int>(width);
      h.b_off_k = static_cast<int>(c0);
      h.n_per_unit = units_n(1);
      h.group_m = group_m(2);
      if (gate_on(2)) h.gate = at<int>(ws, Ly.gate);
      l2_hints(2, &h.a_hint, &h.b_hint);
      h.status = status;
      h.accumulate = c0 > 0;
      TraceScope trace(GRPO_K_DH_GEMM, width, s);
      e = launch_gemm<kEpiF32, false, true>(opDz, opW, h, Ly.rows, di, s, &outDh);
    }
    if (e != cudaSuccess) break;
    {  // dW_c = dZ_c^T Hc (stored, or consumed by the AdamW step)
      GemmArgs w{};
      w.n_valid = n_valid;
      w.M = static_cast<int>(width);
      w.N = Hd;
      w.k_dyn = 1;
      w.n_per_unit = units_n(2);
      w.group_m = group_m(3);
      if (gate_on(3)) w.gate = at<int>(ws, Ly.gate);
      l2_hints(3, &w.a_hint, &w.b_hint);
      w.status = status;
      w.accumulate = 0;
      const OutMat outDw{dW + c0 * Hd, static_cast<uint64_t>(width), hd, hd};
      TraceScope trace(GRPO_K_DW_GEMM, width, s);
      if (adam) {
        const int64_t off = c0 * Hd;
        const uint64_t wd = static_cast<uint64_t>(width);
        const OutMat adam_maps[4] = {{adam->master + off, wd, hd, hd},
                                     {adam->exp_avg + off, wd, hd, hd},
                                     {adam->exp_avg_sq + off, wd, hd, hd},
                                     {adam->w_out + off, wd, hd, hd}};
        // fault-injection test hook: GRPO_TEST_DROP_ADAM=n makes CTA 0 skip the
        // loads of its n-th weight block, so that wait runs out after 0.2 s and
        // the call reports GRPO_ERR_TIMEOUT
        if (const char* d = std::getenv("GRPO_TEST_DROP_ADAM")) {
          w.drop_adam1 = std::atoi(d);
          if (w.drop_adam1 > 0) w.wait_ns = 200000000ull;
        }
        w.adam_b1 = adam->b1;
        w.adam_b2 = adam->b2;
        w.adam_eps = adam->eps;
        w.adam_lr = adam->lr;
        w.adam_decay = adam->decay;
        w.adam_bc1 = adam->bc1;
        w.adam_bc2 = adam->bc2;
        e = launch_gemm<kEpiAdam, true, false>(opDz, opHcT, w, width, di, s, adam_maps);
      } else {
        e = launch_gemm<kEpiF32, true, false>(opDz, opHcT, w, width, di, s, &outDw);
      }
    }
    if (e == cudaSuccess && chunk_events) e = cudaEventRecord(static_cast<cudaEvent_t>(chunk_events[chunk]), s);
    if (e == cudaSuccess && co) {
      cudaEvent_t ready = co->ready[chunk % CopyOut::kRing];
      e = cudaEventRecord(ready, s);
      if (e == cudaSuccess) e = cudaStreamWaitEvent(co->stream, ready, 0);
      if (e == cudaSuccess)
        e = cudaMemcpyAsync(dW_host + c0 * Hd, dW + c0 * Hd, static_cast<size_t>(width) * Hd * sizeof(float),
                            cudaMemcpyDeviceToHost, co->stream);
    }
    ++chunk;
  }
  if (e == cudaSuccess) {  // dH rows to their padded positions, padding rows 0
    TraceScope trace(GRPO_K_DH_ROWS, 0, s);
    const int rb = static_cast<int>(std::min<int64_t>((T + 7) / 8, sms * 8));
    dh_rows_kernel<<<rb, 256, 0, s>>>(at<int>(ws, Ly.rank_of), T, Hd, dHc, dH);
    e = cudaGetLastError();
  }
  if (co && e == cudaSuccess) {
    e = cudaEventRecord(co->done, co->stream);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(s, co->done, 0);
  }
  return from_cuda(e);
}

}  // namespace

extern "C" {

grpo_status grpo_adamw_step(float* W_master, float* exp_avg, float* exp_avg_sq, const float* grad,
                            uint16_t* W_out, int64_t n, float lr, float beta1, float beta2, float eps,
                            float weight_decay, int64_t step, void* stream) {
  if (n < 0 || n % 4 != 0) return GRPO_ERR_INVALID_ARG;
  if (n == 0) return GRPO_OK;
  if (!W_master || !exp_avg || !exp_avg_sq || !grad || !W_out || !aligned(W_master, 16) ||
      !aligned(exp_avg, 16) || !aligned(exp_avg_sq, 16) || !aligned(grad, 16) || !aligned(W_out, 16))
    return GRPO_ERR_INVALID_ARG;
  if (step < 1 || !(lr >= 0.f) || !(beta1 >= 0.f && beta1 < 1.f) || !(beta2 >= 0.f && beta2 < 1.f) ||
      !(eps > 0.f) || !(weight_decay >= 0.f))
    return GRPO_ERR_INVALID_ARG;
  DeviceInfo di;
  if (!device_info(&di)) return GRPO_ERR_UNSUPPORTED;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const float decay = static_cast<float>(1.0 - static_cast<double>(lr) * weight_decay);
  const float bc1 = static_cast<float>(1.0 / (1.0 - std::pow(static_cast<double>(beta1), static_cast<double>(step))));
  const float bc2 = static_cast<float>(1.0 / (1.0 - std::pow(static_cast<double>(beta2), static_cast<double>(step))));
  const int64_t n4 = n / 4;
  const int blocks = static_cast<int>(std::min<int64_t>((n4 + 255) / 256, static_cast<int64_t>(di.sms) * 8));
  TraceScope trace(GRPO_K_ADAMW, 0, s);
  adamw_kernel<<<blocks, 256, 0, s>>>(W_master, exp_avg, exp_avg_sq, grad, W_out, n4, beta1, beta2, eps, lr,
                                      decay, bc1, bc2);
  return from_cuda(cudaGetLastError());
}

grpo_status grpo_trace_enable(int32_t enable) {
  Tracer& t = tracer();
  std::lock_guard<std::mutex> lk(t.mu);
  if (enable) {
    t.recs.clear();
    t.used = 0;
    // create events up front so the first traced launches do not pay for it
    while (t.pool.size() < 1024) {
      cudaEvent_t e = nullptr;
      if (cudaEventCreate(&e) != cudaSuccess) break;
      t.pool.push_back(e);
    }
  }
  t.on = enable != 0;
  return GRPO_OK;
}

int32_t grpo_trace_read(int32_t* kind, int64_t* cols, float* ms, int32_t max_records) {
  Tracer& t = tracer();
  std::lock_guard<std::mutex> lk(t.mu);
  const int32_t n = static_cast<int32_t>(t.recs.size());
  for (int32_t i = 0; i < n && i < max_records; ++i) {
    const TraceRec& r = t.recs[i];
    float dt = 0.f;
    if (cudaEventSynchronize(r.stop) != cudaSuccess ||
        cudaEventElapsedTime(&dt, r.start, r.stop) != cudaSuccess)
      return -1;
    if (kind) kind[i] = r.kind;
    if (cols) cols[i] = r.cols;
    if (ms) ms[i] = dt;
  }
  return n;
}

grpo_status grpo_check_device_status(void* ws, void* stream) {
  if (!ws) return GRPO_ERR_INVALID_ARG;
  unsigned word = 0;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaMemcpyAsync(&word, ws, sizeof(word), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return GRPO_ERR_CUDA;
  if (word & kDevTimeout) return GRPO_ERR_TIMEOUT;
  if (word & kDevCapacity) return GRPO_ERR_CAPACITY;
  if (word) return GRPO_ERR_DEVICE_CHECK;
  return GRPO_OK;
}

// ---------------------------------------------------------------- no-allocation variant
//
// grpo_token_logprobs_noalloc runs grpo_token_logprobs unchanged, with its
// scratch space taken from a fixed array in device memory that is part of this
// library instead of from a caller-provided workspace.

}  // extern "C"

namespace {

constexpr size_t kStaticScratchBytes = size_t(64) << 20;  // 64 MiB on every device that loads the library
static __device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

// Device address of g_static_scratch in the current device's context.  The
// host-side symbol is only a stand-in, never a device address.  Looked up on
// every call (a table lookup in the runtime once the module is loaded), so a
// context made after cudaDeviceReset gets its own address, never a stale one;
// the first call on a device loads the module and should come before any
// stream capture.
void* static_scratch() {
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_static_scratch) != cudaSuccess) return nullptr;
  return p;
}

}  // namespace

extern "C" grpo_status grpo_token_logprobs_noalloc(const uint16_t* H, const uint16_t* W,
                                                   const int32_t* targets, const uint8_t* mask,
                                                   int64_t T, int32_t Hd, int64_t V, float* logp_out,
                                                   void* stream) {
  const size_t need = grpo_workspace_bytes(T, Hd, V, GRPO_WS_LOGPROBS);
  if (need == 0) return GRPO_ERR_INVALID_ARG;
  if (need > kStaticScratchBytes) return GRPO_ERR_WORKSPACE;
  void* ws = static_scratch();
  if (!ws) return GRPO_ERR_CUDA;
  return grpo_token_logprobs(H, W, targets, mask, T, Hd, V, logp_out, ws, kStaticScratchBytes, stream);
}

extern "C" grpo_status grpo_noalloc_check_status(void* stream) {
  void* ws = static_scratch();
  if (!ws) return GRPO_ERR_CUDA;
  return grpo_check_device_status(ws, stream);
}
