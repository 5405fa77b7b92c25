// dz_rows.cuh — dZ rows of one vocabulary chunk from the kept logits.
//
// dZ = g (onehot(y) - softmax(z)) (Eq. 1 differentiated through the
// log-softmax), formed element-wise from the fp32 logits that the forward GEMM
// stored (kEpiLseZ) with dz_value, the same arithmetic as the kEpiDz GEMM
// epilogue, so that from the same logits the same bits come out.
#pragma once

#include <stdint.h>

#include "ptx.cuh"

namespace grpo {

// Columns c0 .. c0 + width of z [rows x ldz] (fp32) -> dz [rows x vc] (bf16),
// rows r0, r0 + rstride, ... by threads tid = 0 .. nthr - 1 of a group.  What
// the kEpiDz epilogue's tiles write as 0 is written as 0 here too: rows from
// N_valid up to the next 256-row tile edge (at most rows_cap) and columns from
// width up to the next 256-column edge (at most vc); the dH and dW GEMMs read
// those padding entries against zero operands.  A thread takes 8 consecutive
// columns four times per pass (8 streaming 16-byte loads in flight: the logits
// are read once), then writes four 16-byte groups of bf16.
__device__ __forceinline__ void dz_rows(const float* __restrict__ z, int64_t ldz, const float* __restrict__ lse,
                                        const float* __restrict__ gcoef, const int* __restrict__ yc, int nv,
                                        int64_t rows_cap, int64_t c0, int width, int vc,
                                        uint16_t* __restrict__ dz, int64_t r0, int64_t rstride, int tid, int nthr) {
  constexpr int kGroups = 4;
  const float kLog2e = 1.4426950408889634f;
  const int64_t rows = min(rows_cap, (static_cast<int64_t>(nv) + 255) / 256 * 256);
  const int cols = min(vc, (width + 255) / 256 * 256);  // a multiple of 8, as vc is
  const int step = nthr * 8;
  for (int64_t r = r0; r < rows; r += rstride) {
    uint16_t* out = dz + r * vc;
    if (r >= nv) {
      for (int c = tid * 8; c < cols; c += step)
        *reinterpret_cast<uint4*>(out + c) = make_uint4(0u, 0u, 0u, 0u);
      continue;
    }
    const float lse2 = lse[r] * kLog2e;
    const float g = gcoef[r];
    const int64_t ty = yc[r] - c0;  // the target's column within the chunk
    const float* src = z + r * ldz + c0;
    for (int cb = tid * 8; cb < cols; cb += kGroups * step) {
      float v[kGroups][8];
#pragma unroll
      for (int k = 0; k < kGroups; ++k) {
        const int c = cb + k * step;
        if (c + 8 <= width) {
          const float4 a = __ldcs(reinterpret_cast<const float4*>(src + c));
          const float4 b = __ldcs(reinterpret_cast<const float4*>(src + c) + 1);
          v[k][0] = a.x, v[k][1] = a.y, v[k][2] = a.z, v[k][3] = a.w;
          v[k][4] = b.x, v[k][5] = b.y, v[k][6] = b.z, v[k][7] = b.w;
        } else {
#pragma unroll
          for (int j = 0; j < 8; ++j) v[k][j] = c + j < width ? src[c + j] : 0.f;
        }
      }
#pragma unroll
      for (int k = 0; k < kGroups; ++k) {
        const int c = cb + k * step;
        if (c >= cols) break;
        uint32_t w[4];
#pragma unroll
        for (int j = 0; j < 8; j += 2) {
          const float d0 = c + j < width ? dz_value(v[k][j], lse2, g, c + j == ty) : 0.f;
          const float d1 = c + j + 1 < width ? dz_value(v[k][j + 1], lse2, g, c + j + 1 == ty) : 0.f;
          w[j / 2] = pack_bf16x2(d0, d1);
        }
        *reinterpret_cast<uint4*>(out + c) = make_uint4(w[0], w[1], w[2], w[3]);
      }
    }
  }
}

}  // namespace grpo
