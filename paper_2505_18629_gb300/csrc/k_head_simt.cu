// LM head of the verify step for fp32 models (CUDA cores, fp32 FMA).
//
// Same decomposition and output as the tcgen05 kernel: each CTA (slot, chunk)
// walks its vocab tiles of 128 rows; per tile and per group of 8 pairs every
// thread forms the dot products of its vocab row with the 8 original and the 8
// reflective hidden rows (k staged through shared memory 32 at a time), then
// runs the shared online log-softmax epilogue.  Used for RV_DTYPE_F32, where
// TF32 tensor cores would round the operands.
#include "head_epilogue.cuh"
#include "rv_device.cuh"
#include "rv_kernels.h"

namespace rv {

constexpr int HS_BM = 128;
constexpr int HS_BK = 32;

struct HeadSimtParams {
  const float* hidden;
  const float* w;
  int V, H, Lh, gamma, R, P, Pc, n_vtiles, slots;
  float alpha;
  const int32_t* drafts;
  float* partials;
  float* gathered;
  float* zout;  // [P][V] fused logits, or null
};

__global__ void __launch_bounds__(HS_BM) head_simt_kernel(const HeadSimtParams p) {
  __shared__ float ws[HS_BM][HS_BK + 1];
  __shared__ float hs[16][HS_BK];
  __shared__ int s_drafts[MAX_PAIRS_PER_CHUNK];
  __shared__ float stats[4 * MAX_PAIRS_PER_CHUNK * HEAD_STAT_STRIDE];

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int slot_id = blockIdx.x, chunk = blockIdx.y;
  const int pair0 = chunk * p.Pc;
  const int npairs = min(p.Pc, p.P - pair0);
  const int t0 = static_cast<int>(static_cast<long long>(slot_id) * p.n_vtiles / p.slots);
  const int t1 = static_cast<int>(static_cast<long long>(slot_id + 1) * p.n_vtiles / p.slots);

  for (int j = tid; j < MAX_PAIRS_PER_CHUNK; j += HS_BM)
    s_drafts[j] = (j < npairs) ? pair_draft(p.drafts, pair0 + j, p.gamma) : -1;
  head_stats_init(stats, 4 * MAX_PAIRS_PER_CHUNK, tid, HS_BM);
  __syncthreads();

  float* const wstats = stats + warp * MAX_PAIRS_PER_CHUNK * HEAD_STAT_STRIDE;
  float* const gathered = p.gathered + static_cast<long long>(pair0) * GATHER_FIELDS;

  for (int t = t0; t < t1; ++t) {
    const int v = t * HS_BM + tid;
    const bool valid = v < p.V;
    for (int g8 = 0; g8 < npairs; g8 += 8) {
      float o[8], r[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) o[j] = r[j] = 0.f;
      for (int k0 = 0; k0 < p.H; k0 += HS_BK) {
        __syncthreads();
        for (int e = tid; e < HS_BM * HS_BK; e += HS_BM) {
          const int rr = e / HS_BK, kk = e % HS_BK;
          const int vv = t * HS_BM + rr, k = k0 + kk;
          ws[rr][kk] = (vv < p.V && k < p.H) ? p.w[static_cast<long long>(vv) * p.H + k] : 0.f;
        }
        for (int e = tid; e < 16 * HS_BK; e += HS_BM) {
          const int rr = e / HS_BK, kk = e % HS_BK;
          const int j = rr & 7, pair = pair0 + g8 + j, k = k0 + kk;
          float val = 0.f;
          if (g8 + j < npairs && k < p.H) {
            const int b = pair / (p.gamma + 1), i = pair % (p.gamma + 1);
            const int row = rr < 8 ? i : i + p.gamma + p.R;  // shift_len = gamma + R
            val = p.hidden[(static_cast<long long>(b) * p.Lh + row) * p.H + k];
          }
          hs[rr][kk] = val;
        }
        __syncthreads();
#pragma unroll 4
        for (int kk = 0; kk < HS_BK; ++kk) {
          const float wv = ws[tid][kk];
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            o[j] = fmaf(wv, hs[j][kk], o[j]);
            r[j] = fmaf(wv, hs[8 + j][kk], r[j]);
          }
        }
      }
      head_tile_pairs8(o, r, g8, npairs, v, valid, p.alpha, s_drafts, wstats, gathered, lane,
                       p.zout ? p.zout + static_cast<long long>(pair0) * p.V : nullptr, p.V);
    }
  }
  __syncthreads();
  head_stats_finish(stats, 4, MAX_PAIRS_PER_CHUNK, npairs,
                    p.partials + (static_cast<long long>(slot_id) * p.P + pair0) * HEAD_STAT_FIELDS,
                    tid, HS_BM);
}

cudaError_t launch_head_simt(const HeadArgs& a, const HeadPlan& pl, cudaStream_t s) {
  HeadSimtParams p;
  p.hidden = static_cast<const float*>(a.hidden);
  p.w = static_cast<const float*>(a.w);
  p.V = a.V;
  p.H = a.H;
  p.Lh = 2 * a.gamma + a.R + 1;
  p.gamma = a.gamma;
  p.R = a.R;
  p.P = pl.P;
  p.Pc = pl.pairs_per_chunk;
  p.n_vtiles = pl.n_vtiles;
  p.slots = pl.slots;
  p.alpha = a.alpha;
  p.drafts = a.drafts;
  p.partials = a.partials;
  p.gathered = a.gathered;
  p.zout = a.zout;
  dim3 grid(pl.slots, pl.n_chunks);
  head_simt_kernel<<<grid, HS_BM, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace rv
