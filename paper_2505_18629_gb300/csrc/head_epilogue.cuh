// Online log-softmax epilogue of the LM head (Alg. 1 / Eq. 2), shared by the
// tcgen05 kernel and the fp32 kernel.
//
// Thread layout: a warp holds 32 consecutive vocab rows v of a tile, one per
// lane.  For each pair (original row, reflective row) the lane has o = o_i[v]
// and r = o'_i[v]; it forms the fused logit z = (1-alpha) o + alpha r (Eq. 2)
// and the warp reduces, across its 32 rows, the max and sum-exp of o, r and z
// and the argmax of z over v != x_i.  Lane j of the warp folds the tile result
// of the j-th pair of a group of eight into the warp's running statistics in
// shared memory.
// The lane whose row equals the draft x_i stores o, r, z at x_i (unique writer).
#pragma once

#include <climits>

#include "rv_device.cuh"
#include "rv_kernels.h"

namespace rv {

// Shared-memory statistics tables use a stride of 10 floats per pair (the 9
// fields used + 1): eight lanes updating consecutive pairs then hit different
// banks.
constexpr int HEAD_STAT_STRIDE = HEAD_STAT_USED + 1;

// Merge running (m, s, t) with another (M, S, T), where s = sum exp(x - m) and
// t = sum exp(x - m) (x - m): both are re-based to the larger maximum.  The
// entropy of softmax(x) is then log(s) - t / s.
__device__ __forceinline__ void lse_merge3(float& m, float& s, float& t, float M, float S,
                                           float T) {
  const float mn = fmaxf(m, M);
  if (mn == NEG_INF) return;
  const float a = (m == NEG_INF) ? 0.f : exp2f(__fmul_rn(m - mn, LOG2E));
  const float c = (M == NEG_INF) ? 0.f : exp2f(__fmul_rn(M - mn, LOG2E));
  t = (a == 0.f ? 0.f : a * (t + (m - mn) * s)) + (c == 0.f ? 0.f : c * (T + (M - mn) * S));
  s = lse_rescale_sum(s, a, S, c);  // the update of lse_merge, bit for bit
  m = mn;
}

__device__ __forceinline__ void head_stats_init(float* stats, int n_entries, int tid,
                                                int nthreads) {
  for (int e = tid; e < n_entries; e += nthreads) {
    float* s = stats + e * HEAD_STAT_STRIDE;
    s[ST_M_O] = NEG_INF;
    s[ST_S_O] = 0.f;
    s[ST_M_R] = NEG_INF;
    s[ST_S_R] = 0.f;
    s[ST_M_Z] = NEG_INF;
    s[ST_S_Z] = 0.f;
    s[ST_BEST_V] = NEG_INF;
    s[ST_BEST_I] = __int_as_float(INT_MAX);
    s[ST_T_O] = 0.f;
  }
}

// Eight pairs g8..g8+7 of one tile.  o[j], r[j]: this lane's logits of pair
// g8+j at vocab row v (pairs at or beyond `npairs` are padding: computed, never
// stored).  The eight pairs' warp reductions run interleaved so that their
// shuffle chains overlap.  `warp_stats` points at this warp's [pairs][FIELDS]
// table; `gathered` at the chunk's first pair.
__device__ __forceinline__ void head_tile_pairs8(const float (&o)[8], const float (&r)[8], int g8,
                                                 int npairs, int v, bool valid, float alpha,
                                                 const int* s_drafts, float* warp_stats,
                                                 float* gathered, int lane, float* zout = nullptr,
                                                 int V = 0) {
  const float beta = 1.f - alpha;
  float ov[8], rv[8], zv[8], Mo[8], Mr[8], Mz[8], bv[8];
  int bi[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const int pj = g8 + j;
    const int x = s_drafts[pj];
    ov[j] = valid ? o[j] : NEG_INF;
    rv[j] = valid ? r[j] : NEG_INF;
    zv[j] = valid ? fmaf(alpha, r[j], beta * o[j]) : NEG_INF;
    if (zout != nullptr && valid && pj < npairs) zout[static_cast<long long>(pj) * V + v] = zv[j];
    if (valid && v == x && pj < npairs) {
      float* gx = gathered + pj * GATHER_FIELDS;
      gx[0] = ov[j];
      gx[1] = rv[j];
      gx[2] = zv[j];
    }
    bv[j] = (v == x) ? NEG_INF : zv[j];
    bi[j] = (bv[j] == NEG_INF) ? INT_MAX : v;
    Mo[j] = ov[j];
    Mr[j] = rv[j];
    Mz[j] = zv[j];
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      Mo[j] = fmaxf(Mo[j], __shfl_xor_sync(0xffffffffu, Mo[j], off));
      Mr[j] = fmaxf(Mr[j], __shfl_xor_sync(0xffffffffu, Mr[j], off));
      Mz[j] = fmaxf(Mz[j], __shfl_xor_sync(0xffffffffu, Mz[j], off));
    }
  }
  float So[8], Sr[8], Sz[8], To[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    So[j] = exp_shifted(ov[j], Mo[j]);
    To[j] = So[j] == 0.f ? 0.f : So[j] * (ov[j] - Mo[j]);
    Sr[j] = exp_shifted(rv[j], Mr[j]);
    Sz[j] = exp_shifted(zv[j], Mz[j]);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      So[j] += __shfl_xor_sync(0xffffffffu, So[j], off);
      To[j] += __shfl_xor_sync(0xffffffffu, To[j], off);
      Sr[j] += __shfl_xor_sync(0xffffffffu, Sr[j], off);
      Sz[j] += __shfl_xor_sync(0xffffffffu, Sz[j], off);
      const float ov2 = __shfl_xor_sync(0xffffffffu, bv[j], off);
      const int oi2 = __shfl_xor_sync(0xffffffffu, bi[j], off);
      if (ov2 > bv[j] || (ov2 == bv[j] && oi2 < bi[j])) {
        bv[j] = ov2;
        bi[j] = oi2;
      }
    }
  }
  // Every lane now holds the tile results of all eight pairs; lane j < 8
  // folds pair g8+j into the running statistics (one SIMT pass, no divergence
  // between the pairs).
  float cMo = Mo[0], cSo = So[0], cTo = To[0], cMr = Mr[0], cSr = Sr[0], cMz = Mz[0], cSz = Sz[0],
        cbv = bv[0];
  int cbi = bi[0];
#pragma unroll
  for (int j = 1; j < 8; ++j) {
    const bool me = lane == j;
    cMo = me ? Mo[j] : cMo;
    cSo = me ? So[j] : cSo;
    cTo = me ? To[j] : cTo;
    cMr = me ? Mr[j] : cMr;
    cSr = me ? Sr[j] : cSr;
    cMz = me ? Mz[j] : cMz;
    cSz = me ? Sz[j] : cSz;
    cbv = me ? bv[j] : cbv;
    cbi = me ? bi[j] : cbi;
  }
  const int pj = g8 + lane;
  if (lane < 8 && pj < npairs) {
    float* s = warp_stats + pj * HEAD_STAT_STRIDE;
    lse_merge3(s[ST_M_O], s[ST_S_O], s[ST_T_O], cMo, cSo, cTo);
    lse_merge(s[ST_M_R], s[ST_S_R], cMr, cSr);
    lse_merge(s[ST_M_Z], s[ST_S_Z], cMz, cSz);
    const int si = __float_as_int(s[ST_BEST_I]);
    if (cbv > s[ST_BEST_V] || (cbv == s[ST_BEST_V] && cbi < si)) {
      s[ST_BEST_V] = cbv;
      s[ST_BEST_I] = __int_as_float(cbi);
    }
  }
}

// Transposed variant of head_tile_pairs8 for the tensor-core kernels: the
// warp stages its 32 rows x (o, r, z) of the eight pairs in shared memory
// (`scr`: HEAD_SCR_FLOATS per warp), and lane c < 24 reduces column c (pair
// c % 8; o, r or z for c / 8) over the 32 rows with plain loads - no shuffle
// trees - then folds the result into the warp's running statistics.  Same
// results as the shuffle version up to the order of the sums.
// sum over the 32 staged rows of exp((x - m) / T); rows at -inf add 0.
__device__ __forceinline__ float subtile_sum_t(const float (&val)[32], float m, float inv_t) {
  float s2[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int i = 0; i < 32; ++i) s2[i & 3] += __expf((val[i] - m) * inv_t);
  return (s2[0] + s2[1]) + (s2[2] + s2[3]);
}

constexpr int HEAD_SCR_STRIDE = 24;  // floats per staged row (16-byte aligned rows)
constexpr int HEAD_SCR_FLOATS = 32 * HEAD_SCR_STRIDE;

__device__ __forceinline__ void head_tile_pairs8_t(const float (&o)[8], const float (&r)[8], int g8,
                                                   int npairs, int v, bool valid, float alpha,
                                                   const int* s_drafts, float* warp_stats,
                                                   float* gathered, float* scr, int lane,
                                                   float* zout = nullptr, int V = 0,
                                                   float2* zsub = nullptr, int n_sub = 0,
                                                   float inv_t = 1.f) {
  const float beta = 1.f - alpha;
  float zr[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const int pj = g8 + j;
    zr[j] = fmaf(alpha, r[j], beta * o[j]);
    // fused logits for the residual draw of speculative sampling (Alg. 1):
    // a warp store covers 32 consecutive vocab rows of one pair
    if (zout != nullptr && valid && pj < npairs) zout[static_cast<long long>(pj) * V + v] = zr[j];
    if (valid && v == s_drafts[pj] && pj < npairs) {
      float* gx = gathered + pj * GATHER_FIELDS;
      gx[0] = o[j];
      gx[1] = r[j];
      gx[2] = zr[j];
    }
  }
  // 16-byte slot k of staged row l sits at slot k ^ ((l >> 2) & 1): rows l and
  // l + 4 of an eight-lane store wavefront then fall on different banks
  float4* const row = reinterpret_cast<float4*>(scr + lane * HEAD_SCR_STRIDE);
  const int sw = (lane >> 2) & 1;
  const float ninf = NEG_INF;
  row[0 ^ sw] = valid ? make_float4(o[0], o[1], o[2], o[3]) : make_float4(ninf, ninf, ninf, ninf);
  row[1 ^ sw] = valid ? make_float4(o[4], o[5], o[6], o[7]) : make_float4(ninf, ninf, ninf, ninf);
  row[2 ^ sw] = valid ? make_float4(r[0], r[1], r[2], r[3]) : make_float4(ninf, ninf, ninf, ninf);
  row[3 ^ sw] = valid ? make_float4(r[4], r[5], r[6], r[7]) : make_float4(ninf, ninf, ninf, ninf);
  row[4 ^ sw] = valid ? make_float4(zr[0], zr[1], zr[2], zr[3]) : make_float4(ninf, ninf, ninf, ninf);
  row[5 ^ sw] = valid ? make_float4(zr[4], zr[5], zr[6], zr[7]) : make_float4(ninf, ninf, ninf, ninf);
  __syncwarp();
  if (lane < 24) {
    const int j = lane & 7, kind = lane >> 3;  // 0: o, 1: r, 2: z
    const int pj = g8 + j;
    float val[32];
    float m = NEG_INF;
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      val[i] = scr[i * HEAD_SCR_STRIDE + (((i >> 2) & 1) ? (lane ^ 4) : lane)];
      m = fmaxf(m, val[i]);
    }
    float sum = 0.f, tsum = 0.f;  // tsum: sum exp(x - m) (x - m), for the entropy of o
    if (m != NEG_INF) {
      float s2[4] = {0.f, 0.f, 0.f, 0.f}, t2[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        const float d = val[i] - m;
        const float e = __expf(d);
        s2[i & 3] += e;
        t2[i & 3] += e == 0.f ? 0.f : e * d;
      }
      sum = (s2[0] + s2[1]) + (s2[2] + s2[3]);
      tsum = (t2[0] + t2[1]) + (t2[2] + t2[3]);
    }
    if (pj < npairs) {
      float* st = warp_stats + pj * HEAD_STAT_STRIDE;
      if (kind == 0) {
        lse_merge3(st[ST_M_O], st[ST_S_O], st[ST_T_O], m, sum, tsum);
      } else if (kind == 1) {
        lse_merge(st[ST_M_R], st[ST_S_R], m, sum);
      } else {
        lse_merge(st[ST_M_Z], st[ST_S_Z], m, sum);
        const int v0 = v - lane;  // vocab row of staged row 0
        if (zsub != nullptr && m != NEG_INF)  // sampled exact match: this subtile's sums at T
          zsub[static_cast<long long>(pj) * n_sub + (v0 >> 5)] =
              make_float2(m, inv_t == 1.f ? sum : subtile_sum_t(val, m, inv_t));
        // best z over the rows v != x_i (lowest row on ties)
        const int x = s_drafts[pj];
        float bv = NEG_INF;
        int bi = INT_MAX;
#pragma unroll
        for (int i = 0; i < 32; ++i)
          if (val[i] > bv && v0 + i != x) {
            bv = val[i];
            bi = v0 + i;
          }
        const int si = __float_as_int(st[ST_BEST_I]);
        if (bv > st[ST_BEST_V] || (bv == st[ST_BEST_V] && bi < si)) {
          st[ST_BEST_V] = bv;
          st[ST_BEST_I] = __int_as_float(bi);
        }
      }
    }
  }
  __syncwarp();  // the staging rows are reused by the next group
}

// Variant of head_tile_pairs8_t for the pre-blended head: the accumulator
// columns are the fused logits z themselves (z = W b, b the blended hidden
// state), so only the z statistics are kept: lane j < 8 reduces pair g8+j over
// the warp's 32 rows (max, sum-exp, best z over v != x_i) and folds it into
// the running statistics; the lane at v == x_i stores z there.
__device__ __forceinline__ void head_tile_z8_t(const float (&z)[8], int g8, int npairs, int v,
                                               bool valid, const int* s_drafts, float* warp_stats,
                                               float* gathered, float* scr, int lane,
                                               float* zout = nullptr, int V = 0,
                                               float2* zsub = nullptr, int n_sub = 0,
                                               float inv_t = 1.f) {
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const int pj = g8 + j;
    if (zout != nullptr && valid && pj < npairs) zout[static_cast<long long>(pj) * V + v] = z[j];
    if (valid && v == s_drafts[pj] && pj < npairs) gathered[pj * GATHER_FIELDS + 2] = z[j];
  }
  float4* const row = reinterpret_cast<float4*>(scr + lane * HEAD_SCR_STRIDE);
  const int sw = (lane >> 2) & 1;  // the swizzle of head_tile_pairs8_t
  const float ninf = NEG_INF;
  row[0 ^ sw] = valid ? make_float4(z[0], z[1], z[2], z[3]) : make_float4(ninf, ninf, ninf, ninf);
  row[1 ^ sw] = valid ? make_float4(z[4], z[5], z[6], z[7]) : make_float4(ninf, ninf, ninf, ninf);
  __syncwarp();
  if (lane < 8) {
    const int pj = g8 + lane;
    float val[32];
    float m = NEG_INF;
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      val[i] = scr[i * HEAD_SCR_STRIDE + (((i >> 2) & 1) ? (lane ^ 4) : lane)];
      m = fmaxf(m, val[i]);
    }
    float sum = 0.f;
    if (m != NEG_INF) {
      float s2[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int i = 0; i < 32; ++i) s2[i & 3] += __expf(val[i] - m);
      sum = (s2[0] + s2[1]) + (s2[2] + s2[3]);
    }
    if (pj < npairs) {
      float* st = warp_stats + pj * HEAD_STAT_STRIDE;
      lse_merge(st[ST_M_Z], st[ST_S_Z], m, sum);
      const int x = s_drafts[pj];
      const int v0 = v - lane;  // vocab row of staged row 0
      if (zsub != nullptr && m != NEG_INF)  // sampled exact match: this subtile's sums at T
        zsub[static_cast<long long>(pj) * n_sub + (v0 >> 5)] =
            make_float2(m, inv_t == 1.f ? sum : subtile_sum_t(val, m, inv_t));
      float bv = NEG_INF;
      int bi = INT_MAX;
#pragma unroll
      for (int i = 0; i < 32; ++i)
        if (val[i] > bv && v0 + i != x) {
          bv = val[i];
          bi = v0 + i;
        }
      const int si = __float_as_int(st[ST_BEST_I]);
      if (bv > st[ST_BEST_V] || (bv == st[ST_BEST_V] && bi < si)) {
        st[ST_BEST_V] = bv;
        st[ST_BEST_I] = __int_as_float(bi);
      }
    }
  }
  __syncwarp();  // the staging rows are reused by the next group
}

// Combine the warps' tables (each `tab` pairs long) into one partial per pair
// and store it.  `out` points at partials[slot][chunk's first pair].
__device__ __forceinline__ void head_stats_finish(const float* stats, int nwarps, int tab,
                                                  int npairs, float* out, int tid, int nthreads) {
  for (int pj = tid; pj < npairs; pj += nthreads) {
    float mo = NEG_INF, so = 0.f, to = 0.f, mr = NEG_INF, sr = 0.f, mz = NEG_INF, sz = 0.f;
    float bv = NEG_INF;
    int bi = INT_MAX;
    for (int w = 0; w < nwarps; ++w) {
      const float* s = stats + (w * tab + pj) * HEAD_STAT_STRIDE;
      lse_merge3(mo, so, to, s[ST_M_O], s[ST_S_O], s[ST_T_O]);
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
    d[ST_T_O] = to;
#pragma unroll
    for (int f = HEAD_STAT_USED; f < HEAD_STAT_FIELDS; ++f) d[f] = 0.f;
  }
}

// Merge the slots' partial statistics of every pair and finish the
// per-position outputs (one warp per pair), then, if asked, the exact-match
// acceptance of every sequence (Alg. 2).  Run by every thread of one CTA, the
// last LM-head CTA to finish; partials are read past L1 (other CTAs wrote
// them).  Each lane issues the loads of all its slots before merging them, and
// the choices go through shared memory (`s_choice`, P ints), so the tail costs
// about one L2 round trip.
constexpr int MERGE_SLOTS_PER_LANE = 6;

// Acceptance test of one position from its fused log-probability, entropy
// and greedy choice: exact match (Alg. 2) or the typical threshold (Alg. 3).
__device__ __forceinline__ bool position_kept(const AcceptArgs& acc, int x, int choice,
                                              float logp_fused, float ent_orig) {
  if (acc.mode == RV_ACCEPT_TYPICAL)
    return logp_fused > fminf(acc.log_eps, acc.log_delta - ent_orig);  // false for NaN
  return x == choice;
}

// s_draft[p]: the draft scored by pair p (-1 for none), in shared memory;
// s_choice: 2P ints of shared memory (choices, then kept flags).
__device__ __forceinline__ void head_merge_all(const float* partials, const float* gathered,
                                               const int* s_draft, int B, int gamma, int V,
                                               int P, int slots, const HeadFinal& f,
                                               unsigned* status, int* s_choice, int tid,
                                               int nthreads) {
  const int lane = tid & 31, warp = tid >> 5, nw = nthreads >> 5;
  const float nan = __int_as_float(0x7fc00000);
  int* const s_kept = s_choice + P;
  for (int p = warp; p < P; p += nw) {
    float mo = NEG_INF, so = 0.f, to = 0.f, mr = NEG_INF, sr = 0.f, mz = NEG_INF, sz = 0.f;
    float bv = NEG_INF;
    int bi = INT_MAX;
    for (int g0 = lane; g0 < slots; g0 += 32 * MERGE_SLOTS_PER_LANE) {
      float4 lo[MERGE_SLOTS_PER_LANE], hi[MERGE_SLOTS_PER_LANE];
      float tt[MERGE_SLOTS_PER_LANE];
#pragma unroll
      for (int k = 0; k < MERGE_SLOTS_PER_LANE; ++k) {
        const int g = g0 + 32 * k;
        if (g < slots) {
          const float* q = partials + (static_cast<long long>(g) * P + p) * HEAD_STAT_FIELDS;
          lo[k] = __ldcg(reinterpret_cast<const float4*>(q));
          hi[k] = __ldcg(reinterpret_cast<const float4*>(q) + 1);
          tt[k] = __ldcg(q + ST_T_O);
        }
      }
#pragma unroll
      for (int k = 0; k < MERGE_SLOTS_PER_LANE; ++k) {
        if (g0 + 32 * k < slots) {
          lse_merge3(mo, so, to, lo[k].x, lo[k].y, tt[k]);
          lse_merge(mr, sr, lo[k].z, lo[k].w);
          lse_merge(mz, sz, hi[k].x, hi[k].y);
          const int i = __float_as_int(hi[k].w);
          if (hi[k].z > bv || (hi[k].z == bv && i < bi)) {
            bv = hi[k].z;
            bi = i;
          }
        }
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      lse_merge3(mo, so, to, __shfl_xor_sync(0xffffffffu, mo, o), __shfl_xor_sync(0xffffffffu, so, o),
                 __shfl_xor_sync(0xffffffffu, to, o));
      lse_merge(mr, sr, __shfl_xor_sync(0xffffffffu, mr, o), __shfl_xor_sync(0xffffffffu, sr, o));
      lse_merge(mz, sz, __shfl_xor_sync(0xffffffffu, mz, o), __shfl_xor_sync(0xffffffffu, sz, o));
    }
    warp_argmax(bv, bi);
    if (lane == 0) {
      const int b = p / (gamma + 1), i = p % (gamma + 1);
      // (the pre-blended head has no separate original / reflective logits)
      const float lse_o = f.zonly ? nan : mo + logf(so), lse_r = f.zonly ? nan : mr + logf(sr);
      const float lse_z = mz + logf(sz);
      const float ent = f.zonly ? nan : logf(so) - to / so;
      float* sc = f.scores + static_cast<long long>(p) * RV_NSCORES;
      sc[RV_SCORE_LSE_ORIG] = lse_o;
      sc[RV_SCORE_LSE_REFL] = lse_r;
      sc[RV_SCORE_LSE_FUSED] = lse_z;
      sc[RV_SCORE_ENT_ORIG] = ent;
      int choice = bi;
      float lp_z = nan, lp_o = nan, lp_r = nan;
      int x = -1;
      if (i < gamma) {
        x = s_draft[p];
        if (x >= 0 && x < V) {
          const float4 gx = __ldcg(reinterpret_cast<const float4*>(gathered) + p);
          lp_z = gx.z - lse_z;
          lp_o = f.zonly ? nan : gx.x - lse_o;
          lp_r = f.zonly ? nan : gx.y - lse_r;
          if (gx.z > bv || (gx.z == bv && x < bi)) choice = x;
          f.margin[b * gamma + i] = fabsf(gx.z - bv);
        } else {
          raise_status(status, RV_DEV_DRAFT_RANGE);
          f.margin[b * gamma + i] = nan;
        }
      }
      sc[RV_SCORE_LOGP_FUSED] = lp_z;
      sc[RV_SCORE_LOGP_ORIG] = lp_o;
      sc[RV_SCORE_LOGP_REFL] = lp_r;
      f.argmax[p] = choice;
      s_choice[p] = choice;
      s_kept[p] = position_kept(f.acc, x, choice, lp_z, ent) ? 1 : 0;
    }
  }
  if (f.acc.accepted_len == nullptr) return;
  __syncthreads();  // every choice of this CTA is in s_choice
  for (int b = tid; b < B; b += nthreads) {
    int n = gamma;
    for (int i = 0; i < gamma; ++i) {
      const bool ok = s_kept[b * (gamma + 1) + i] != 0;
      f.acc.accept_mask[b * gamma + i] = ok ? 1 : 0;
      if (!ok && n == gamma) n = i;
    }
    f.acc.accepted_len[b] = n;
    f.acc.next_token[b] = s_choice[b * (gamma + 1) + n];
    f.acc.ctx_out[b] = f.acc.ctx_in[b] + n + f.acc.ctx_extra;
  }
}

// Draft id scored by pair `pair` (-1 for the last position of a sequence).
__device__ __forceinline__ int pair_draft(const int32_t* drafts, int pair, int gamma) {
  const int b = pair / (gamma + 1), i = pair % (gamma + 1);
  return i < gamma ? drafts[b * gamma + i] : -1;
}

}  // namespace rv
