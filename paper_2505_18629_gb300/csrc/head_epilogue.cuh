// Online log-softmax epilogue of the LM head (Alg. 1 / Eq. 2), shared by the
// tcgen05 kernel and the fp32 kernel.
//
// Thread layout: a warp holds 32 consecutive vocab rows v of a tile, one per
// lane.  For each pair (original row, reflective row) the lane has o = o_i[v]
// and r = o'_i[v]; it forms the fused logit z = (1-alpha) o + alpha r (Eq. 2)
// and the warp reduces, across its 32 rows, the max and sum-exp of o, r and z
// and the argmax of z over v != x_i.  The lane that owns the pair (pair % 32)
// folds the tile's result into the warp's running statistics in shared memory.
// The lane whose row equals the draft x_i stores o, r, z at x_i (unique writer).
#pragma once

#include <climits>

#include "rv_device.cuh"
#include "rv_kernels.h"

namespace rv {

__device__ __forceinline__ void head_stats_init(float* stats, int n_entries, int tid,
                                                int nthreads) {
  for (int e = tid; e < n_entries; e += nthreads) {
    float* s = stats + e * HEAD_STAT_FIELDS;
    s[ST_M_O] = NEG_INF;
    s[ST_S_O] = 0.f;
    s[ST_M_R] = NEG_INF;
    s[ST_S_R] = 0.f;
    s[ST_M_Z] = NEG_INF;
    s[ST_S_Z] = 0.f;
    s[ST_BEST_V] = NEG_INF;
    s[ST_BEST_I] = __int_as_float(INT_MAX);
  }
}

// Eight pairs g8..g8+7 of one tile.  o[j], r[j]: this lane's logits of pair
// g8+j at vocab row v.  `warp_stats` points at this warp's [128][FIELDS] table;
// `gathered` at the chunk's first pair.
__device__ __forceinline__ void head_tile_pairs8(const float (&o)[8], const float (&r)[8], int g8,
                                                 int npairs, int v, bool valid, float alpha,
                                                 const int* s_drafts, float* warp_stats,
                                                 float* gathered, int lane) {
  const float beta = 1.f - alpha;
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const int pj = g8 + j;
    if (pj >= npairs) break;  // uniform across the warp
    const int x = s_drafts[pj];
    const float ov = valid ? o[j] : NEG_INF;
    const float rv = valid ? r[j] : NEG_INF;
    const float zv = valid ? fmaf(alpha, r[j], beta * o[j]) : NEG_INF;
    if (valid && v == x) {
      float* gx = gathered + pj * GATHER_FIELDS;
      gx[0] = ov;
      gx[1] = rv;
      gx[2] = zv;
    }
    float bv = (v == x) ? NEG_INF : zv;
    int bi = (bv == NEG_INF) ? INT_MAX : v;
    const float Mo = warp_max(ov);
    const float Mr = warp_max(rv);
    const float Mz = warp_max(zv);
    const float So = warp_sum(exp_shifted(ov, Mo));
    const float Sr = warp_sum(exp_shifted(rv, Mr));
    const float Sz = warp_sum(exp_shifted(zv, Mz));
    warp_argmax(bv, bi);
    if (lane == (pj & 31)) {
      float* s = warp_stats + pj * HEAD_STAT_FIELDS;
      lse_merge(s[ST_M_O], s[ST_S_O], Mo, So);
      lse_merge(s[ST_M_R], s[ST_S_R], Mr, Sr);
      lse_merge(s[ST_M_Z], s[ST_S_Z], Mz, Sz);
      const int si = __float_as_int(s[ST_BEST_I]);
      if (bv > s[ST_BEST_V] || (bv == s[ST_BEST_V] && bi < si)) {
        s[ST_BEST_V] = bv;
        s[ST_BEST_I] = __int_as_float(bi);
      }
    }
  }
}

// Combine the warps' tables into one partial per pair and store it.
// `out` points at partials[slot][chunk's first pair].
__device__ __forceinline__ void head_stats_finish(const float* stats, int nwarps, int npairs,
                                                  float* out, int tid, int nthreads) {
  for (int pj = tid; pj < npairs; pj += nthreads) {
    float mo = NEG_INF, so = 0.f, mr = NEG_INF, sr = 0.f, mz = NEG_INF, sz = 0.f;
    float bv = NEG_INF;
    int bi = INT_MAX;
    for (int w = 0; w < nwarps; ++w) {
      const float* s = stats + (w * MAX_PAIRS_PER_CHUNK + pj) * HEAD_STAT_FIELDS;
      lse_merge(mo, so, s[ST_M_O], s[ST_S_O]);
      lse_merge(mr, sr, s[ST_M_R], s[ST_S_R]);
      lse_merge(mz, sz, s[ST_M_Z], s[ST_S_Z]);
      const float v = s[ST_BEST_V];
      const int i = __float_as_int(s[ST_BEST_I]);
      if (v > bv || (v == bv && i < bi)) {
        bv = v;
        bi = i;
      }
    }
    float* d = out + pj * HEAD_STAT_FIELDS;
    d[ST_M_O] = mo;
    d[ST_S_O] = so;
    d[ST_M_R] = mr;
    d[ST_S_R] = sr;
    d[ST_M_Z] = mz;
    d[ST_S_Z] = sz;
    d[ST_BEST_V] = bv;
    d[ST_BEST_I] = __int_as_float(bi);
  }
}

// Draft id scored by pair `pair` (-1 for the last position of a sequence).
__device__ __forceinline__ int pair_draft(const int32_t* drafts, int pair, int gamma) {
  const int b = pair / (gamma + 1), i = pair % (gamma + 1);
  return i < gamma ? drafts[b * gamma + i] : -1;
}

}  // namespace rv
