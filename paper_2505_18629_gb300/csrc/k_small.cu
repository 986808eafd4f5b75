// Small kernels of the verify step: block packing (Eq. 1), gathering of the
// original / reflective hidden rows for the LM head, the merge of the head's
// per-CTA statistics into per-position scores (Eq. 2), and exact-match
// acceptance with the longest accepted prefix (Alg. 2).
#include <cfloat>
#include <climits>

#include "rv_device.cuh"
#include "rv_kernels.h"

namespace rv {

// ---------------------------------------------------------------- pack (Eq. 1)
// block[b] = [x_1..x_gamma, prompt, prefix_b, x_1..x_gamma]; pos = ctx_b + j.
__global__ void pack_block_kernel(const int32_t* __restrict__ drafts,
                                  const int32_t* __restrict__ prompt,
                                  const int32_t* __restrict__ prefix,
                                  const int32_t* __restrict__ ctx, int B, int gamma,
                                  int n_prompt, int n_prefix, int32_t* __restrict__ block,
                                  int32_t* __restrict__ pos) {
  const int Lb = 2 * gamma + n_prompt + n_prefix;
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= B * Lb) return;
  const int b = idx / Lb, j = idx % Lb;
  int tok;
  if (j < gamma) {
    tok = drafts[b * gamma + j];
  } else if (j < gamma + n_prompt) {
    tok = prompt[j - gamma];
  } else if (j < gamma + n_prompt + n_prefix) {
    tok = prefix[b * n_prefix + (j - gamma - n_prompt)];
  } else {
    tok = drafts[b * gamma + (j - gamma - n_prompt - n_prefix)];
  }
  block[idx] = tok;
  pos[idx] = ctx[b] + j;
}

cudaError_t launch_pack_block(const int32_t* drafts, const int32_t* prompt, const int32_t* prefix,
                              const int32_t* ctx, int B, int gamma, int n_prompt, int n_prefix,
                              int32_t* block_ids, int32_t* pos_ids, cudaStream_t s) {
  const int n = B * (2 * gamma + n_prompt + n_prefix);
  if (n == 0) return cudaSuccess;
  pack_block_kernel<<<(n + 255) / 256, 256, 0, s>>>(drafts, prompt, prefix, ctx, B, gamma,
                                                     n_prompt, n_prefix, block_ids, pos_ids);
  return cudaGetLastError();
}

// ---------------------------------------------------------------- gather rows
// hsel row (c*N + j)        = hidden[b][i]            (original row of pair c*Pc+j)
// hsel row (c*N + Pcp + j)  = hidden[b][gamma+R+i]    (reflective row, shift_len = gamma+R)
// padding rows are zero.  One 16-byte vector per thread.
__global__ void gather_rows_kernel(const uint4* __restrict__ hidden, uint4* __restrict__ hsel,
                                   int P, int gamma, int R, int Lh, int Hv, int Pc, int Pcp,
                                   int N, int n_chunks) {
  const long long total = static_cast<long long>(n_chunks) * N * Hv;
  for (long long idx = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; idx < total;
       idx += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int col = static_cast<int>(idx % Hv);
    const int row = static_cast<int>(idx / Hv);
    const int c = row / N, r = row % N;
    const bool refl = r >= Pcp;
    const int j = refl ? r - Pcp : r;
    const int p = c * Pc + j;
    uint4 v = make_uint4(0, 0, 0, 0);
    if (j < Pc && p < P) {
      const int b = p / (gamma + 1), i = p % (gamma + 1);
      const int hrow = refl ? i + gamma + R : i;
      v = hidden[(static_cast<long long>(b) * Lh + hrow) * Hv + col];
    }
    hsel[idx] = v;
  }
}

cudaError_t launch_gather_rows(const HeadArgs& a, const HeadPlan& p, void* hsel, cudaStream_t s) {
  const int Hv = a.H / 8;  // 8 bf16 per 16-byte vector
  const int Lh = 2 * a.gamma + a.R + 1;
  const long long total = static_cast<long long>(p.n_chunks) * p.N * Hv;
  const int threads = 256;
  const int blocks = static_cast<int>(std::min<long long>((total + threads - 1) / threads, 4096));
  gather_rows_kernel<<<blocks, threads, 0, s>>>(static_cast<const uint4*>(a.hidden),
                                                static_cast<uint4*>(hsel), p.P, a.gamma, a.R, Lh,
                                                Hv, p.pairs_per_chunk, p.pad_pairs, p.N,
                                                p.n_chunks);
  return cudaGetLastError();
}

// ---------------------------------------------------------------- head merge
// One warp per pair: merge the slots' (max, sum) triples and argmax, then
// finish the per-position scores.
__global__ void head_merge_kernel(const float* __restrict__ partials,
                                  const float* __restrict__ gathered,
                                  const int32_t* __restrict__ drafts, int P, int gamma, int V,
                                  int slots, float* __restrict__ scores,
                                  int32_t* __restrict__ argmax_out, float* __restrict__ margin,
                                  unsigned* status) {
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= P) return;
  const int p = warp;
  float mo = NEG_INF, so = 0.f, mr = NEG_INF, sr = 0.f, mz = NEG_INF, sz = 0.f;
  float bv = NEG_INF;
  int bi = INT_MAX;
  for (int g = lane; g < slots; g += 32) {
    const float* st = partials + (static_cast<long long>(g) * P + p) * HEAD_STAT_FIELDS;
    lse_merge(mo, so, st[ST_M_O], st[ST_S_O]);
    lse_merge(mr, sr, st[ST_M_R], st[ST_S_R]);
    lse_merge(mz, sz, st[ST_M_Z], st[ST_S_Z]);
    const float v = st[ST_BEST_V];
    const int i = __float_as_int(st[ST_BEST_I]);
    if (v > bv || (v == bv && i < bi)) {
      bv = v;
      bi = i;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    lse_merge(mo, so, __shfl_xor_sync(0xffffffffu, mo, o), __shfl_xor_sync(0xffffffffu, so, o));
    lse_merge(mr, sr, __shfl_xor_sync(0xffffffffu, mr, o), __shfl_xor_sync(0xffffffffu, sr, o));
    lse_merge(mz, sz, __shfl_xor_sync(0xffffffffu, mz, o), __shfl_xor_sync(0xffffffffu, sz, o));
  }
  warp_argmax(bv, bi);
  if (lane != 0) return;
  const int b = p / (gamma + 1), i = p % (gamma + 1);
  const float lse_o = mo + logf(so);
  const float lse_r = mr + logf(sr);
  const float lse_z = mz + logf(sz);
  float* sc = scores + static_cast<long long>(p) * RV_NSCORES;
  sc[RV_SCORE_LSE_ORIG] = lse_o;
  sc[RV_SCORE_LSE_REFL] = lse_r;
  sc[RV_SCORE_LSE_FUSED] = lse_z;
  const float nan = __int_as_float(0x7fc00000);
  int choice = bi;
  if (i < gamma) {
    const int x = drafts[b * gamma + i];
    if (x >= 0 && x < V) {
      const float* gx = gathered + static_cast<long long>(p) * GATHER_FIELDS;
      const float zx = gx[2];
      sc[RV_SCORE_LOGP_FUSED] = zx - lse_z;
      sc[RV_SCORE_LOGP_ORIG] = gx[0] - lse_o;
      sc[RV_SCORE_LOGP_REFL] = gx[1] - lse_r;
      if (zx > bv || (zx == bv && x < bi)) choice = x;
      margin[b * gamma + i] = fabsf(zx - bv);
    } else {
      raise_status(status, RV_DEV_DRAFT_RANGE);
      sc[RV_SCORE_LOGP_FUSED] = nan;
      sc[RV_SCORE_LOGP_ORIG] = nan;
      sc[RV_SCORE_LOGP_REFL] = nan;
      margin[b * gamma + i] = nan;
    }
  } else {
    sc[RV_SCORE_LOGP_FUSED] = nan;
    sc[RV_SCORE_LOGP_ORIG] = nan;
    sc[RV_SCORE_LOGP_REFL] = nan;
  }
  argmax_out[p] = choice;
}

cudaError_t launch_head_merge(const HeadArgs& a, const HeadPlan& p, float* scores,
                              int32_t* argmax, float* margin, cudaStream_t s) {
  const int threads = 128;
  const int blocks = (p.P * 32 + threads - 1) / threads;
  head_merge_kernel<<<blocks, threads, 0, s>>>(a.partials, a.gathered, a.drafts, p.P, a.gamma,
                                               a.V, p.slots, scores, argmax, margin, a.status);
  return cudaGetLastError();
}

// ---------------------------------------------------------------- accept (Alg. 2)
__global__ void accept_kernel(const int32_t* __restrict__ drafts,
                              const int32_t* __restrict__ argmax, int B, int gamma,
                              uint8_t* __restrict__ accept_mask, int32_t* __restrict__ accepted_len,
                              int32_t* __restrict__ next_token, const int32_t* ctx_in,
                              int32_t* ctx_out) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  int n = gamma;
  for (int i = 0; i < gamma; ++i) {
    const bool acc = drafts[b * gamma + i] == argmax[b * (gamma + 1) + i];
    accept_mask[b * gamma + i] = acc ? 1 : 0;
    if (!acc && n == gamma) n = i;
  }
  accepted_len[b] = n;
  next_token[b] = argmax[b * (gamma + 1) + n];
  ctx_out[b] = ctx_in[b] + n;
}

cudaError_t launch_accept(const int32_t* drafts, const int32_t* argmax, int B, int gamma,
                          uint8_t* accept_mask, int32_t* accepted_len, int32_t* next_token,
                          const int32_t* ctx_in, int32_t* ctx_out, cudaStream_t s) {
  accept_kernel<<<(B + 127) / 128, 128, 0, s>>>(drafts, argmax, B, gamma, accept_mask,
                                                accepted_len, next_token, ctx_in, ctx_out);
  return cudaGetLastError();
}

}  // namespace rv
