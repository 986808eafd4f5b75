// Small kernels of the verify step: block packing (Eq. 1); the prep kernel
// that gathers the original / reflective hidden rows for the LM head (and
// packs the block in the same launch); the finalize kernel that merges the
// head's per-CTA statistics into per-position scores (Eq. 2) and, inside
// rv_verify_step, runs the acceptance (exact match, Alg. 2, or the typical
// threshold, Alg. 3) with the longest accepted prefix; the stand-alone
// acceptance kernels of rv_accept and rv_accept_typical.
#include <cfloat>
#include <climits>

#include "head_epilogue.cuh"
#include "rv_device.cuh"
#include "rv_kernels.h"

namespace rv {

// ---------------------------------------------------------------- pack (Eq. 1)
// block[b] = [x_1..x_gamma, prompt, prefix_b, x_1..x_gamma]; pos = ctx_b + j.
// With `pending`, the pending-token block [t_b, x_1..x_gamma, prompt, prefix_b,
// x_1..x_gamma]: the last emitted token goes first.  copy == 0: standard
// verification's block, [x_1..x_gamma] (or [t_b, x_1..x_gamma]), no template.
__global__ void pack_block_kernel(const int32_t* __restrict__ drafts,
                                  const int32_t* __restrict__ prompt,
                                  const int32_t* __restrict__ prefix,
                                  const int32_t* __restrict__ ctx, int B, int gamma,
                                  int n_prompt, int n_prefix, int32_t* __restrict__ block,
                                  int32_t* __restrict__ pos, const int32_t* __restrict__ pending,
                                  int copy) {
  const int lead = pending ? 1 : 0;
  const int Lb = (1 + copy) * gamma + n_prompt + n_prefix + lead;
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= B * Lb) return;
  const int b = idx / Lb, jj = idx % Lb, j = jj - lead;
  int tok;
  if (j < 0) {
    tok = pending[b];
  } else if (j < gamma) {
    tok = drafts[b * gamma + j];
  } else if (j < gamma + n_prompt) {
    tok = prompt[j - gamma];
  } else if (j < gamma + n_prompt + n_prefix) {
    tok = prefix[b * n_prefix + (j - gamma - n_prompt)];
  } else {
    tok = drafts[b * gamma + (j - gamma - n_prompt - n_prefix)];
  }
  block[idx] = tok;
  pos[idx] = ctx[b] + jj;
}

cudaError_t launch_pack_block(const int32_t* drafts, const int32_t* prompt, const int32_t* prefix,
                              const int32_t* ctx, int B, int gamma, int n_prompt, int n_prefix,
                              int32_t* block_ids, int32_t* pos_ids, cudaStream_t s,
                              const int32_t* pending, int copy) {
  const int n = B * ((1 + copy) * gamma + n_prompt + n_prefix + (pending ? 1 : 0));
  if (n == 0) return cudaSuccess;
  pack_block_kernel<<<(n + 255) / 256, 256, 0, s>>>(drafts, prompt, prefix, ctx, B, gamma,
                                                     n_prompt, n_prefix, block_ids, pos_ids,
                                                     pending, copy);
  return cudaGetLastError();
}

// ---------------------------------------------------------------- prep: gather rows (+ pack)
// hsel row (c*N + j)        = hidden[b][i]            (original row of pair c*Pc+j)
// hsel row (c*N + Pcp + j)  = hidden[b][gamma+R+i]    (reflective row, shift_len = gamma+R)
// or, for the pre-blended head (N = Pcp), the blended state of Eq. 2's
// linearity, each element rounded once to bf16:
// hsel row (c*N + j)        = bf16(fl((1-a) h[b][i]) + fl(a h[b][gamma+R+i]))
// or, for standard verification (zonly == 2, N = Pcp, hidden [B, gamma+1, H]):
// hsel row (c*N + j)        = h[b][i]
// padding rows are zero.  One 16-byte vector per thread and step.  When the
// block is to be packed too, the first B*Lb threads of the grid also do that.
__device__ __forceinline__ uint32_t blend_bf16x2(uint32_t o, uint32_t r, float alpha, float beta) {
  const float o0 = __uint_as_float(o << 16), o1 = __uint_as_float(o & 0xFFFF0000u);
  const float r0 = __uint_as_float(r << 16), r1 = __uint_as_float(r & 0xFFFF0000u);
  const float b0 = __fadd_rn(__fmul_rn(beta, o0), __fmul_rn(alpha, r0));
  const float b1 = __fadd_rn(__fmul_rn(beta, o1), __fmul_rn(alpha, r1));
  return pack_bf16(b0, b1);
}

__global__ void prep_kernel(const uint4* __restrict__ hidden, uint4* __restrict__ hsel, int P,
                            int gamma, int R, int Lh, int Hv, int Pc, int Pcp, int N, int n_chunks,
                            int zonly, float alpha, float beta, const PackArgs pk,
                            unsigned* tile_counter, unsigned* done_counter) {
  // The LM-head kernel that follows may start now (programmatic dependent
  // launch); it waits for this grid before it reads anything written here.
  asm volatile("griddepcontrol.launch_dependents;");
  const long long tid0 = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x;
  if (tid0 == 0 && tile_counter) *tile_counter = 0u;  // the LM head that follows claims tiles from 0
  if (tid0 == 0 && done_counter) *done_counter = 0u;
  if (pk.block != nullptr) {
    const int lead = pk.pending ? 1 : 0;  // the pending-token block [t, x, prompt, prefix, x]
    const int Lb = (1 + pk.copy) * pk.gamma + pk.n_prompt + pk.n_prefix + lead;
    for (long long idx = tid0; idx < static_cast<long long>(pk.B) * Lb;
         idx += static_cast<long long>(gridDim.x) * blockDim.x) {
      const int b = static_cast<int>(idx / Lb), jj = static_cast<int>(idx % Lb), j = jj - lead;
      int tok;
      if (j < 0)
        tok = pk.pending[b];
      else if (j < pk.gamma)
        tok = pk.drafts[b * pk.gamma + j];
      else if (j < pk.gamma + pk.n_prompt)
        tok = pk.prompt[j - pk.gamma];
      else if (j < pk.gamma + pk.n_prompt + pk.n_prefix)
        tok = pk.prefix[b * pk.n_prefix + (j - pk.gamma - pk.n_prompt)];
      else
        tok = pk.drafts[b * pk.gamma + (j - pk.gamma - pk.n_prompt - pk.n_prefix)];
      pk.block[idx] = tok;
      pk.pos[idx] = pk.ctx[b] + jj;
    }
  }
  if (hsel == nullptr) return;
  const long long total = static_cast<long long>(n_chunks) * N * Hv;
  for (long long idx = tid0; idx < total; idx += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int col = static_cast<int>(idx % Hv);
    const int row = static_cast<int>(idx / Hv);
    const int c = row / N, r = row % N;
    const bool refl = !zonly && r >= Pcp;
    const int j = refl ? r - Pcp : r;
    const int p = c * Pc + j;
    uint4 v = make_uint4(0, 0, 0, 0);
    if (j < Pc && p < P) {
      const int b = p / (gamma + 1), i = p % (gamma + 1);
      const long long orow = (static_cast<long long>(b) * Lh + i) * Hv + col;
      const long long rrow = (static_cast<long long>(b) * Lh + i + gamma + R) * Hv + col;
      if (zonly == 2) {
        v = hidden[orow];
      } else if (zonly) {
        const uint4 o = hidden[orow], rr = hidden[rrow];
        v = make_uint4(blend_bf16x2(o.x, rr.x, alpha, beta), blend_bf16x2(o.y, rr.y, alpha, beta),
                       blend_bf16x2(o.z, rr.z, alpha, beta), blend_bf16x2(o.w, rr.w, alpha, beta));
      } else {
        v = hidden[refl ? rrow : orow];
      }
    }
    hsel[idx] = v;
  }
}

cudaError_t launch_prep(const HeadArgs& a, const HeadPlan& p, void* hsel, const PackArgs* pack,
                        cudaStream_t s) {
  PackArgs pk = {};
  long long work = 0;
  if (pack) {
    pk = *pack;
    work = static_cast<long long>(pk.B) *
           ((1 + pk.copy) * pk.gamma + pk.n_prompt + pk.n_prefix + (pk.pending ? 1 : 0));
  }
  const int Hv = a.H / 8;  // 8 bf16 per 16-byte vector
  // hidden rows per sequence: the block's positions plus the state before it
  const int Lh = p.standard ? a.gamma + 1 : 2 * a.gamma + a.R + 1;
  if (hsel) work = std::max(work, static_cast<long long>(p.n_chunks) * p.N * Hv);
  if (a.tile_counter) work = std::max(work, 1LL);
  if (work == 0) return cudaSuccess;
  const int threads = 256;
  const int blocks = static_cast<int>(std::min<long long>((work + threads - 1) / threads, 4096));
  prep_kernel<<<blocks, threads, 0, s>>>(static_cast<const uint4*>(a.hidden),
                                         static_cast<uint4*>(hsel), p.P, a.gamma, a.R, Lh, Hv,
                                         p.pairs_per_chunk, p.pad_pairs, p.N, p.n_chunks,
                                         p.standard ? 2 : (p.zonly ? 1 : 0), a.alpha,
                                         1.0f - a.alpha, pk,
                                         a.tile_counter, a.done_counter);
  return cudaGetLastError();
}

// ---------------------------------------------------------------- head finalize
// One CTA per position p = b*(gamma+1) + i: its threads merge the slots'
// (max, sum) triples and argmax candidates (16-byte loads, a few slots per
// thread), then thread 0 finishes the position's scores.  Inside
// rv_verify_step each sequence's acceptance follows: the last of its
// positions' CTAs to finish (a ticket per sequence, re-armed by that CTA)
// reads the positions' choices and scores back and runs Alg. 2 (or Alg. 3).
constexpr int FIN_THREADS = 128;

struct MergeStat {
  float mo, so, to, mr, sr, mz, sz, bv;
  int bi;
};

__device__ __forceinline__ void merge_into(MergeStat& a, const MergeStat& b) {
  lse_merge3(a.mo, a.so, a.to, b.mo, b.so, b.to);
  lse_merge(a.mr, a.sr, b.mr, b.sr);
  lse_merge(a.mz, a.sz, b.mz, b.sz);
  if (b.bv > a.bv || (b.bv == a.bv && b.bi < a.bi)) {
    a.bv = b.bv;
    a.bi = b.bi;
  }
}

__device__ __forceinline__ MergeStat shfl_stat(const MergeStat& s, int o) {
  MergeStat r;
  r.mo = __shfl_xor_sync(0xffffffffu, s.mo, o);
  r.so = __shfl_xor_sync(0xffffffffu, s.so, o);
  r.to = __shfl_xor_sync(0xffffffffu, s.to, o);
  r.mr = __shfl_xor_sync(0xffffffffu, s.mr, o);
  r.sr = __shfl_xor_sync(0xffffffffu, s.sr, o);
  r.mz = __shfl_xor_sync(0xffffffffu, s.mz, o);
  r.sz = __shfl_xor_sync(0xffffffffu, s.sz, o);
  r.bv = __shfl_xor_sync(0xffffffffu, s.bv, o);
  r.bi = __shfl_xor_sync(0xffffffffu, s.bi, o);
  return r;
}

__global__ void __launch_bounds__(FIN_THREADS)
    head_finalize_kernel(const float* __restrict__ partials, const float* __restrict__ gathered,
                         const int32_t* __restrict__ drafts, int P, int gamma, int V, int slots,
                         float* scores, int32_t* argmax_out, float* __restrict__ margin,
                         unsigned* status, AcceptArgs acc, int zonly, unsigned* seq_tickets) {
  // launched as a programmatic dependent of the LM head: wait for its results
  asm volatile("griddepcontrol.wait;" ::: "memory");
  __shared__ MergeStat red[FIN_THREADS / 32];
  __shared__ int s_last;
  const int p = blockIdx.x;
  const int npos = gamma + 1, b = p / npos, i = p % npos;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const float nan = __int_as_float(0x7fc00000);
  MergeStat st{NEG_INF, 0.f, 0.f, NEG_INF, 0.f, NEG_INF, 0.f, NEG_INF, INT_MAX};
  for (int g = threadIdx.x; g < slots; g += FIN_THREADS) {
    // fields 0..3: o and o' (max, sum); 4..7: z (max, sum), best z and its row; 8: entropy term
    const float4* q =
        reinterpret_cast<const float4*>(partials + (static_cast<long long>(g) * P + p) * HEAD_STAT_FIELDS);
    const float4 lo = __ldcg(q), hi = __ldcg(q + 1);
    const float t = __ldcg(reinterpret_cast<const float*>(q) + ST_T_O);
    merge_into(st, MergeStat{lo.x, lo.y, t, lo.z, lo.w, hi.x, hi.y, hi.z, __float_as_int(hi.w)});
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) merge_into(st, shfl_stat(st, o));
  if (lane == 0) red[warp] = st;
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int w = 1; w < FIN_THREADS / 32; ++w) merge_into(st, red[w]);
    // (the pre-blended head has no separate original / reflective logits)
    const float lse_o = zonly ? nan : st.mo + logf(st.so);
    const float lse_r = zonly ? nan : st.mr + logf(st.sr);
    const float lse_z = st.mz + logf(st.sz);
    const float ent = zonly ? nan : logf(st.so) - st.to / st.so;
    float* sc = scores + static_cast<long long>(p) * RV_NSCORES;
    sc[RV_SCORE_ENT_ORIG] = ent;
    sc[RV_SCORE_LSE_ORIG] = lse_o;
    sc[RV_SCORE_LSE_REFL] = lse_r;
    sc[RV_SCORE_LSE_FUSED] = lse_z;
    int choice = st.bi;
    float lp_z = nan, lp_o = nan, lp_r = nan;
    if (i < gamma) {
      const int x = drafts[b * gamma + i];
      if (x >= 0 && x < V) {
        const float* gx = gathered + static_cast<long long>(p) * GATHER_FIELDS;
        const float zx = gx[2];
        lp_z = zx - lse_z;
        lp_o = zonly ? nan : gx[0] - lse_o;
        lp_r = zonly ? nan : gx[1] - lse_r;
        if (zx > st.bv || (zx == st.bv && x < st.bi)) choice = x;
        margin[b * gamma + i] = fabsf(zx - st.bv);
      } else {
        raise_status(status, RV_DEV_DRAFT_RANGE);
        margin[b * gamma + i] = nan;
      }
    }
    sc[RV_SCORE_LOGP_FUSED] = lp_z;
    sc[RV_SCORE_LOGP_ORIG] = lp_o;
    sc[RV_SCORE_LOGP_REFL] = lp_r;
    argmax_out[p] = choice;
    s_last = 0;
    if (acc.accepted_len != nullptr) {
      __threadfence();  // this position's outputs before the ticket
      s_last = atomicAdd(seq_tickets + b, 1u) == static_cast<unsigned>(npos - 1) ? 1 : 0;
    }
  }
  __syncthreads();
  if (!s_last || threadIdx.x != 0) return;
  // the sequence's last position: every other position's outputs are visible
  __threadfence();
  seq_tickets[b] = 0u;  // re-armed for the next launch
  int n = gamma;
  for (int k = 0; k < gamma; ++k) {
    const int pk = b * npos + k;
    const int x = drafts[b * gamma + k];
    const int choice = __ldcg(argmax_out + pk);
    const float lp = __ldcg(scores + static_cast<long long>(pk) * RV_NSCORES + RV_SCORE_LOGP_FUSED);
    const float ent = __ldcg(scores + static_cast<long long>(pk) * RV_NSCORES + RV_SCORE_ENT_ORIG);
    const bool ok = position_kept(acc, x, choice, lp, ent);
    acc.accept_mask[b * gamma + k] = ok ? 1 : 0;
    if (!ok && n == gamma) n = k;
  }
  acc.accepted_len[b] = n;
  acc.next_token[b] = __ldcg(argmax_out + b * npos + n);
  acc.ctx_out[b] = acc.ctx_in[b] + n + acc.ctx_extra;
}

cudaError_t launch_head_finalize(const HeadArgs& a, const HeadPlan& p, float* scores,
                                 int32_t* argmax, float* margin, const AcceptArgs* acc,
                                 cudaStream_t s) {
  AcceptArgs ac = {};
  if (acc) ac = *acc;
  if (acc && a.seq_tickets == nullptr) return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.P, 1, 1);
  cfg.blockDim = dim3(FIN_THREADS, 1, 1);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, head_finalize_kernel, a.partials, a.gathered, a.drafts, p.P,
                            a.gamma, a.V, p.slots, scores, argmax, margin, a.status, ac,
                            p.zonly ? 1 : 0, a.seq_tickets);
}

// ---------------------------------------------------------------- accept (Alg. 2)
__global__ void accept_kernel(const int32_t* __restrict__ drafts,
                              const int32_t* __restrict__ argmax, int B, int gamma,
                              uint8_t* __restrict__ accept_mask, int32_t* __restrict__ accepted_len,
                              int32_t* __restrict__ next_token, const int32_t* ctx_in,
                              int32_t* ctx_out, int ctx_extra) {
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
  ctx_out[b] = ctx_in[b] + n + ctx_extra;
}

// ---------------------------------------------------------------- speculative accept (Alg. 1)
// A cluster of SPC_CL CTAs per sequence.  The first warp of every CTA runs the
// ratio test (one lane per draft): draft i is kept while
// log r_i <= log p_i(x_i) - log q_i(x_i) (p_i from the head's fused log-prob),
// n = the number of leading kept drafts.  Then the cluster draws t from
//   p' = norm(max(0, p_{n+1} - q_{n+1}))  (n < gamma)   or   p_{gamma+1}
// by inverse CDF with u.  CTA c owns the c-th of SPC_CL equal slices of the
// vocabulary; it scans the weights of its slice in vocabulary order (warp w
// owns SPC_WARP consecutive tokens, lane l the ones at 32 j + l: the loads
// coalesce) and sends its total to every CTA of the cluster.  Every CTA forms
// the same prefix of the slice totals, so all agree on the slice that holds
// u * sum(w); that CTA finds the token.  Each range's upper end and the next
// range's lower end are the same expression of the same values, within a
// slice as between slices, so the ranges tile [0, sum(w)) exactly in floating
// point.  If every residual weight is zero (p_{n+1} <= q_{n+1} everywhere, only
// through rounding) the draw is from p_{n+1} itself.
constexpr int SPC_CL = 16;
constexpr int SPC_THREADS = 512;
constexpr int SPC_E = 16;                        // tokens per lane and round
constexpr int SPC_WARP = 32 * SPC_E;
constexpr int SPC_ROUND = SPC_THREADS * SPC_E;

__device__ __forceinline__ float spec_weight(float zv, float qv, float lse, bool resid) {
  const float p = __expf(zv - lse);
  return resid ? fmaxf(0.f, p - qv) : p;
}

// One round of a slice: the lane's weights and their warp scans (see
// sub_round_weights); returns the warp's total.
__device__ __forceinline__ float spc_round(const float* zrow, const float* qrow, float lse,
                                           bool resid, int base, int v_hi, int lane,
                                           float (&w)[SPC_E], float (&incl)[SPC_E], int& last) {
  float zv[SPC_E], qv[SPC_E];
#pragma unroll
  for (int j = 0; j < SPC_E; ++j) {
    const int v = base + 32 * j;
    zv[j] = v < v_hi ? __ldg(zrow + v) : NEG_INF;
    qv[j] = (resid && v < v_hi) ? __ldg(qrow + v) : 0.f;
  }
#pragma unroll
  for (int j = 0; j < SPC_E; ++j) {
    w[j] = zv[j] == NEG_INF ? 0.f : spec_weight(zv[j], qv[j], lse, resid);
    incl[j] = w[j];
    if (w[j] > 0.f) last = base + 32 * j;
  }
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
#pragma unroll
    for (int j = 0; j < SPC_E; ++j) {
      const float y = __shfl_up_sync(0xffffffffu, incl[j], o);
      if (lane >= o) incl[j] += y;
    }
  }
  float carry = 0.f;
#pragma unroll
  for (int j = 0; j < SPC_E; ++j) carry = carry + __shfl_sync(0xffffffffu, incl[j], 31);
  return carry;
}

__global__ void __launch_bounds__(SPC_THREADS)
    accept_speculative_kernel(const int32_t* __restrict__ drafts, const float* __restrict__ q,
                              const float* __restrict__ r, const float* __restrict__ u,
                              const float* __restrict__ scores, const float* __restrict__ z,
                              int gamma, int V, AcceptArgs a, unsigned* status) {
  constexpr int NW = SPC_THREADS / 32;
  __shared__ float s_wc[2][SPC_CL];  // every slice's total, per pass (written by its CTA)
  __shared__ int s_lastc[2][SPC_CL];  // every slice's last token of positive weight
  __shared__ float s_wtot[NW];
  __shared__ int s_n, s_last;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint32_t rank;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(rank));
  const int b = blockIdx.x / SPC_CL;
  // (other CTAs' shared memory is written only after every CTA has started)
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
  if (warp == 0) {  // the ratio test, 32 drafts per round
    int n = gamma;
    for (int i0 = 0; i0 < gamma; i0 += 32) {
      const int i = i0 + lane;
      bool keep = true;
      if (i < gamma) {
        const int x = drafts[b * gamma + i];
        const float logp = scores[(static_cast<long long>(b) * (gamma + 1) + i) * RV_NSCORES +
                                  RV_SCORE_LOGP_FUSED];
        keep = false;
        if (x >= 0 && x < V) {
          const float qx = q[(static_cast<long long>(b) * gamma + i) * V + x];
          // log r <= log p - log q; q(x) = 0 makes the ratio infinite (kept)
          keep = qx > 0.f ? logf(r[b * gamma + i]) <= logp - logf(qx) : logp > NEG_INF;
        } else if (rank == 0) {
          raise_status(status, RV_DEV_DRAFT_RANGE);
        }
        if (rank == 0) a.accept_mask[b * gamma + i] = keep ? 1 : 0;
      }
      const unsigned bad = __ballot_sync(0xffffffffu, !keep);
      if (bad != 0u && n == gamma) n = i0 + __ffs(bad) - 1;
    }
    if (lane == 0) s_n = n;
  }
  __syncthreads();
  const int n = s_n;
  const long long prow = static_cast<long long>(b) * (gamma + 1) + n;
  const float lse = scores[prow * RV_NSCORES + RV_SCORE_LSE_FUSED];
  const float* const zrow = z + prow * V;
  const float* const qrow = q + (static_cast<long long>(b) * gamma + min(n, gamma - 1)) * V;
  const int Vc = (V + SPC_CL - 1) / SPC_CL;
  const int v_lo = min(V, static_cast<int>(rank) * Vc), v_hi = min(V, v_lo + Vc);
  const int base0 = v_lo + SPC_WARP * warp + lane;
  const bool one_round = v_hi - v_lo <= SPC_ROUND;
  float w[SPC_E], incl[SPC_E];
  for (int pass = 0; pass < 2; ++pass) {
    const bool resid = pass == 0 && n < gamma;
    // this slice's total, in the scan's own arithmetic
    float run = 0.f, wt_first = 0.f;
    int last = -1;
    for (int r0 = 0; r0 < v_hi - v_lo; r0 += SPC_ROUND) {
      const float wt = spc_round(zrow, qrow, lse, resid, base0 + r0, v_hi, lane, w, incl, last);
      if (r0 == 0) wt_first = wt;
      __syncthreads();
      if (lane == 0) s_wtot[warp] = wt;
      __syncthreads();
      float total = 0.f;
      for (int k = 0; k < NW; ++k) total = total + s_wtot[k];
      run = run + total;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) last = max(last, __shfl_xor_sync(0xffffffffu, last, o));
    if (tid == 0) s_last = -1;
    __syncthreads();
    if (lane == 0 && last >= 0) atomicMax(&s_last, last);
    __syncthreads();
    // to every CTA of the cluster: this slice's total and last weighted token
    if (pass == 0) asm volatile("barrier.cluster.wait.aligned;" ::: "memory");
    if (tid < SPC_CL) {
      uint32_t d0, d1;
      asm volatile("mapa.shared::cluster.u32 %0, %1, %2;"
                   : "=r"(d0) : "r"(smem_u32(&s_wc[pass][rank])), "r"(tid));
      asm volatile("mapa.shared::cluster.u32 %0, %1, %2;"
                   : "=r"(d1) : "r"(smem_u32(&s_lastc[pass][rank])), "r"(tid));
      asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(d0), "f"(run) : "memory");
      asm volatile("st.shared::cluster.s32 [%0], %1;" ::"r"(d1), "r"(s_last) : "memory");
    }
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::
                     : "memory");
    float W = 0.f;
    for (int c = 0; c < SPC_CL; ++c) W = W + s_wc[pass][c];
    if (!(W > 0.f)) {  // (the same in every CTA of the cluster)
      if (pass == 0) continue;
      if (rank == 0 && tid == 0) a.next_token[b] = 0;  // no weight at all: non-finite logits
      break;
    }
    const float target = u[b] * W;
    float P = 0.f;
    int owner = -1, last_c = -1;
    float P_owner = 0.f;
    for (int c = 0; c < SPC_CL; ++c) {
      const float Pn = P + s_wc[pass][c];
      if (owner < 0 && target >= P && target < Pn) {
        owner = c;
        P_owner = P;
      }
      if (s_wc[pass][c] > 0.f) last_c = c;
      P = Pn;
    }
    if (owner < 0) {  // u * W at or past the rounded total: the last token with weight
      if (static_cast<int>(rank) == last_c && tid == 0) a.next_token[b] = s_lastc[pass][last_c];
      break;
    }
    if (static_cast<int>(rank) != owner) break;
    // the owner: the token whose range holds the target
    run = 0.f;
    if (tid == 0) s_last = -1;  // reused: the token found
    for (int r0 = 0; r0 < v_hi - v_lo; r0 += SPC_ROUND) {
      int dummy = -1;
      const float wt = one_round ? wt_first
                                 : spc_round(zrow, qrow, lse, resid, base0 + r0, v_hi, lane, w,
                                             incl, dummy);
      __syncthreads();
      if (lane == 0) s_wtot[warp] = wt;
      __syncthreads();
      float woff = 0.f, total = 0.f;
      for (int k = 0; k < NW; ++k) {
        if (k == warp) woff = total;
        total = total + s_wtot[k];
      }
      float carry = 0.f;
#pragma unroll
      for (int j = 0; j < SPC_E; ++j) {
        const float ex = __shfl_up_sync(0xffffffffu, incl[j], 1);
        const float tj = __shfl_sync(0xffffffffu, incl[j], 31);
        const float lo = P_owner + (run + (woff + (carry + (lane == 0 ? 0.f : ex))));
        const float hi = P_owner + (run + (woff + (carry + incl[j])));
        if (target >= lo && target < hi) s_last = base0 + r0 + 32 * j;
        carry = carry + tj;
      }
      run = run + total;
      __syncthreads();
      if (s_last >= 0) break;
    }
    if (tid == 0) a.next_token[b] = s_last >= 0 ? s_last : s_lastc[pass][owner];
    break;
  }
  if (rank == 0 && tid == 0) {
    a.accepted_len[b] = n;
    a.ctx_out[b] = a.ctx_in[b] + n + a.ctx_extra;
  }
}

cudaError_t launch_accept_speculative(const int32_t* drafts, const float* q, const float* r,
                                      const float* u, const float* scores, const float* z, int B,
                                      int gamma, int V, uint8_t* accept_mask,
                                      int32_t* accepted_len, int32_t* next_token,
                                      const int32_t* ctx_in, int32_t* ctx_out, unsigned* status,
                                      cudaStream_t s, int ctx_extra) {
  static bool configured = false;
  if (!configured) {
    const cudaError_t e = cudaFuncSetAttribute(accept_speculative_kernel,
                                               cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  AcceptArgs a{accept_mask, accepted_len, next_token, ctx_in, ctx_out, 0, 0.f, 0.f, ctx_extra};
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(B * SPC_CL, 1, 1);
  cfg.blockDim = dim3(SPC_THREADS, 1, 1);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = SPC_CL;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, accept_speculative_kernel, drafts, q, r, u, scores, z, gamma, V,
                            a, status);
}

// ---------------------------------------------------------------- sampled target tokens (Alg. 2)
// A cluster of CL CTAs per position (b, i), i = 1..gamma+1: the target's
// token at temperature T, x^_i ~ softmax(z_i / T), drawn by inverse CDF with
// the position's uniform u: the smallest v whose cumulative weight
// w_v = exp((z_i[v] - max z_i) / T) exceeds u * sum(w).  CTA c owns the c-th
// of CL slices of the row, as in accept_speculative_kernel: the slices'
// maxima are exchanged first (every CTA then holds max z_i), then their
// totals, and the CTA whose slice holds the target finds the token.
__device__ __forceinline__ float samp_round(const float* zrow, float M, float inv_t, int base,
                                            int v_hi, int lane, float (&w)[SPC_E],
                                            float (&incl)[SPC_E], int& last) {
  float zv[SPC_E];
#pragma unroll
  for (int j = 0; j < SPC_E; ++j) {
    const int v = base + 32 * j;
    zv[j] = v < v_hi ? __ldg(zrow + v) : NEG_INF;
  }
#pragma unroll
  for (int j = 0; j < SPC_E; ++j) {
    w[j] = zv[j] == NEG_INF ? 0.f : expf((zv[j] - M) * inv_t);
    incl[j] = w[j];
    if (w[j] > 0.f) last = base + 32 * j;
  }
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
#pragma unroll
    for (int j = 0; j < SPC_E; ++j) {
      const float y = __shfl_up_sync(0xffffffffu, incl[j], o);
      if (lane >= o) incl[j] += y;
    }
  }
  float carry = 0.f;
#pragma unroll
  for (int j = 0; j < SPC_E; ++j) carry = carry + __shfl_sync(0xffffffffu, incl[j], 31);
  return carry;
}

template <int CL>
__global__ void __launch_bounds__(SPC_THREADS)
    sample_fused_kernel(const float* __restrict__ z, const float* __restrict__ u, int V,
                        float inv_t, int32_t* __restrict__ xhat) {
  constexpr int NW = SPC_THREADS / 32;
  __shared__ float s_max[CL];   // every slice's max z (written by its CTA)
  __shared__ float s_wc[CL];    // every slice's total weight
  __shared__ int s_lastc[CL];   // every slice's last token of positive weight
  __shared__ float s_wtot[NW];
  __shared__ int s_last;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint32_t rank;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(rank));
  const long long prow = blockIdx.x / CL;
  const float* const row = z + prow * V;
  // (other CTAs' shared memory is written only after every CTA has started)
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
  const int Vc = (V + CL - 1) / CL;
  const int v_lo = min(V, static_cast<int>(rank) * Vc), v_hi = min(V, v_lo + Vc);
  const int base0 = v_lo + SPC_WARP * warp + lane;
  // this slice's max, to every CTA of the cluster
  float m = NEG_INF;
  for (int r0 = 0; r0 < v_hi - v_lo; r0 += SPC_ROUND)
#pragma unroll
    for (int j = 0; j < SPC_E; ++j) {
      const int v = base0 + r0 + 32 * j;
      if (v < v_hi) m = fmaxf(m, __ldg(row + v));
    }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
  if (lane == 0) s_wtot[warp] = m;
  __syncthreads();
  if (tid == 0) {
    for (int k = 1; k < NW; ++k) m = fmaxf(m, s_wtot[k]);
    s_wtot[0] = m;
  }
  __syncthreads();
  m = s_wtot[0];
  asm volatile("barrier.cluster.wait.aligned;" ::: "memory");
  if (tid < CL) {
    uint32_t d0;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;"
                 : "=r"(d0) : "r"(smem_u32(&s_max[rank])), "r"(tid));
    asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(d0), "f"(m) : "memory");
  }
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::
                   : "memory");
  float M = s_max[0];
  for (int c = 1; c < CL; ++c) M = fmaxf(M, s_max[c]);
  // this slice's weights and total, in the scan's own arithmetic
  float w[SPC_E], incl[SPC_E];
  float run = 0.f, wt_first = 0.f;
  int last = -1;
  const bool one_round = v_hi - v_lo <= SPC_ROUND;
  for (int r0 = 0; r0 < v_hi - v_lo; r0 += SPC_ROUND) {
    const float wt = samp_round(row, M, inv_t, base0 + r0, v_hi, lane, w, incl, last);
    if (r0 == 0) wt_first = wt;
    __syncthreads();
    if (lane == 0) s_wtot[warp] = wt;
    __syncthreads();
    float total = 0.f;
    for (int k = 0; k < NW; ++k) total = total + s_wtot[k];
    run = run + total;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) last = max(last, __shfl_xor_sync(0xffffffffu, last, o));
  if (tid == 0) s_last = -1;
  __syncthreads();
  if (lane == 0 && last >= 0) atomicMax(&s_last, last);
  __syncthreads();
  if (tid < CL) {
    uint32_t d0, d1;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;"
                 : "=r"(d0) : "r"(smem_u32(&s_wc[rank])), "r"(tid));
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;"
                 : "=r"(d1) : "r"(smem_u32(&s_lastc[rank])), "r"(tid));
    asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(d0), "f"(run) : "memory");
    asm volatile("st.shared::cluster.s32 [%0], %1;" ::"r"(d1), "r"(s_last) : "memory");
  }
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::
                   : "memory");
  float W = 0.f;
  for (int c = 0; c < CL; ++c) W = W + s_wc[c];
  const float target = u[prow] * W;
  float P = 0.f, P_owner = 0.f;
  int owner = -1, last_c = -1;
  for (int c = 0; c < CL; ++c) {
    const float Pn = P + s_wc[c];
    if (owner < 0 && target >= P && target < Pn) {
      owner = c;
      P_owner = P;
    }
    if (s_wc[c] > 0.f) last_c = c;
    P = Pn;
  }
  if (owner < 0) {  // u * W at or past the rounded total: the last token with weight
    if (static_cast<int>(rank) == max(last_c, 0) && tid == 0)
      xhat[prow] = last_c >= 0 ? s_lastc[last_c] : 0;
    return;
  }
  if (static_cast<int>(rank) != owner) return;
  run = 0.f;
  if (tid == 0) s_last = -1;  // reused: the token found
  for (int r0 = 0; r0 < v_hi - v_lo; r0 += SPC_ROUND) {
    int dummy = -1;
    const float wt = one_round ? wt_first
                               : samp_round(row, M, inv_t, base0 + r0, v_hi, lane, w, incl, dummy);
    __syncthreads();
    if (lane == 0) s_wtot[warp] = wt;
    __syncthreads();
    float woff = 0.f, total = 0.f;
    for (int k = 0; k < NW; ++k) {
      if (k == warp) woff = total;
      total = total + s_wtot[k];
    }
    float carry = 0.f;
#pragma unroll
    for (int j = 0; j < SPC_E; ++j) {
      const float ex = __shfl_up_sync(0xffffffffu, incl[j], 1);
      const float tj = __shfl_sync(0xffffffffu, incl[j], 31);
      const float lo = P_owner + (run + (woff + (carry + (lane == 0 ? 0.f : ex))));
      const float hi = P_owner + (run + (woff + (carry + incl[j])));
      if (target >= lo && target < hi) s_last = base0 + r0 + 32 * j;
      carry = carry + tj;
    }
    run = run + total;
    __syncthreads();
    if (s_last >= 0) break;
  }
  if (tid == 0) xhat[prow] = s_last >= 0 ? s_last : s_lastc[owner];
}

template <int CL>
static cudaError_t launch_sample_fused_cl(const float* z, const float* u, int P, int V,
                                          float temperature, int32_t* xhat, cudaStream_t s) {
  static bool configured = false;
  if (!configured) {
    const cudaError_t e = cudaFuncSetAttribute(sample_fused_kernel<CL>,
                                               cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(P * CL, 1, 1);
  cfg.blockDim = dim3(SPC_THREADS, 1, 1);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = CL;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, sample_fused_kernel<CL>, z, u, V, 1.f / temperature, xhat);
}

// A few positions: 16 CTAs each (the shortest chain per position); many: 4,
// so that the clusters of all positions fit the GPU at once.
cudaError_t launch_sample_fused(const float* z, const float* u, int P, int V, float temperature,
                                int32_t* xhat, cudaStream_t s) {
  if (P <= 0) return cudaSuccess;
  return P <= 16 ? launch_sample_fused_cl<16>(z, u, P, V, temperature, xhat, s)
                 : launch_sample_fused_cl<4>(z, u, P, V, temperature, xhat, s);
}

// ---------------------------------------------------------------- draws from subtile sums (Alg. 2)
// One CTA of 32 warps per position p.  The inverse CDF of softmax(z_p / T)
// at u_p, in two levels: the head left per 32-row subtile k the pair
// (m_k, s_k) with s_k = sum exp((z - m_k) / T), so the subtile weights are
// w_k = s_k exp((m_k - M) / T) (M = max m_k).  The CTA scans the w_k in
// vocabulary order to the subtile k* whose range holds u S (S = sum w_k),
// with the fraction f of w_k* below the target.  Warp r then recomputes row r
// of that subtile's fused logits from the head's own operands (the w row
// times the position's hsel rows, fp32 sums; z = (1-a) o + a o' as the head
// forms it), and the first warp picks the first row whose cumulative weight
// within the subtile exceeds f times the subtile's total.  Up to the rounding of the sums this is the
// smallest v whose cumulative weight exceeds u * sum(w); a target at or past
// the rounded total takes the last row of positive weight.
//
// The scan: a round covers SUB_ROUND entries; warp w owns SUB_WARP
// consecutive ones, entry 32 j + lane of them in register j of the lane (the
// loads coalesce).  Each entry's range [lo, hi) is formed so that one
// entry's hi and the next entry's lo are the same expression of the same
// values (the shuffled neighbour, the carried register total, the warp
// offset), so the ranges tile [0, S) without gaps or overlaps in floating
// point: a target below S falls in exactly one of them.
constexpr int SUB_THREADS = 1024;          // one warp per row of a subtile
constexpr int SUB_REG = 4;                 // subtile entries per lane and round
constexpr int SUB_WARP = 32 * SUB_REG;
constexpr int SUB_ROUND = SUB_THREADS * SUB_REG;
constexpr int SUB_LD = 8;                  // 16-byte weight loads per lane and batch

// A 16-byte read-only load the compiler keeps in program order with the
// others of its kind (volatile), so that a batch of them is in flight at once.
// D += A B, m16n8k16, bf16 operands, fp32 accumulators (register order of
// the PTX fragment layout: a0 / a1 rows g / g+8 at k 2q..2q+1, a2 / a3 the
// same rows at k 2q+8..2q+9; b0 / b1 column g at k 2q.. / 2q+8..).
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                               uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint4 ldg_batch(const uint4* p) {
  uint4 v;
  asm volatile("ld.global.nc.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

// One round of the scan: the lane's weights w[], their in-register inclusive
// scans across the warp (incl[]) and the warp's total; nothing is shared yet.
// k2 = log2(e) / T: w = s exp2((m - M) k2).
__device__ __forceinline__ float sub_round_weights(const float2* sub, int n_sub, int base, float M,
                                                   float k2, int lane, float (&w)[SUB_REG],
                                                   float (&incl)[SUB_REG], int& last) {
  float2 e[SUB_REG];  // every load in flight before the first is used
#pragma unroll
  for (int j = 0; j < SUB_REG; ++j)
    e[j] = base + 32 * j < n_sub ? __ldg(sub + base + 32 * j) : make_float2(NEG_INF, 0.f);
#pragma unroll
  for (int j = 0; j < SUB_REG; ++j) {
    const float x = e[j].x == NEG_INF ? 0.f : e[j].y * ex2_approx((e[j].x - M) * k2);
    w[j] = x;
    incl[j] = x;
    if (x > 0.f) last = base + 32 * j;
  }
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
#pragma unroll
    for (int j = 0; j < SUB_REG; ++j) {
      const float y = __shfl_up_sync(0xffffffffu, incl[j], o);
      if (lane >= o) incl[j] += y;
    }
  }
  float carry = 0.f;
#pragma unroll
  for (int j = 0; j < SUB_REG; ++j) carry = carry + __shfl_sync(0xffffffffu, incl[j], 31);
  return carry;
}

__global__ void __launch_bounds__(SUB_THREADS, 1)
    sample_subtiles_kernel(const SubtileDraw d, AcceptArgs acc) {
  constexpr int NW = SUB_THREADS / 32;
  static_assert(NW == 32, "one warp per row of a 32-row subtile");
  __shared__ float s_red[NW];
  __shared__ float s_wtot[NW];
  __shared__ float2 s_part[16][32];  // per chunk group: (o, o') of each subtile row
  __shared__ float s_frac;
  __shared__ int s_k, s_last;
  extern __shared__ uint4 s_h[];  // the position's hsel rows: o (and o')
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int p = blockIdx.x;
  const int nvec = d.H / 8;
  const float k2 = LOG2E * d.inv_t;
  const float2* const sub = d.zsub + static_cast<long long>(p) * d.n_sub;
  if (tid == 0) {
    s_k = -1;
    s_last = -1;
    s_frac = 1.f;
  }
  // launched as a programmatic dependent of the LM head: its outputs first
  asm volatile("griddepcontrol.wait;" ::: "memory");
  // M = max m_k, with the position's hsel rows staged meanwhile
  const int base0 = SUB_WARP * warp + lane;
  float m = NEG_INF;
  for (int r0 = 0; r0 < d.n_sub; r0 += SUB_ROUND) {
    float mk[SUB_REG];
#pragma unroll
    for (int j = 0; j < SUB_REG; ++j) {
      const int k = r0 + base0 + 32 * j;
      mk[j] = k < d.n_sub ? __ldg(&sub[k].x) : NEG_INF;
    }
    if (r0 == 0) {
      const int pc = p / d.Pc, pj = p % d.Pc;
      const uint4* const h_o =
          static_cast<const uint4*>(d.hsel) + static_cast<long long>(pc * d.N + pj) * nvec;
      const uint4* const h_r = h_o + static_cast<long long>(d.Pcp) * nvec;
      for (int c = tid; c < nvec; c += SUB_THREADS) {
        const uint4 a = __ldg(h_o + c);
        const uint4 b = d.zonly ? a : __ldg(h_r + c);
        s_h[c] = a;
        if (!d.zonly) s_h[nvec + c] = b;
      }
    }
#pragma unroll
    for (int j = 0; j < SUB_REG; ++j) m = fmaxf(m, mk[j]);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
  if (lane == 0) s_red[warp] = m;
  __syncthreads();
  float M = s_red[0];
#pragma unroll
  for (int k = 1; k < NW; ++k) M = fmaxf(M, s_red[k]);
  // S: with several rounds, a first pass of the same arithmetic
  const bool one_round = d.n_sub <= SUB_ROUND;
  float S = 0.f;
  float w[SUB_REG], incl[SUB_REG];
  if (!one_round) {
    float run = 0.f;
    for (int r0 = 0; r0 < d.n_sub; r0 += SUB_ROUND) {
      int dummy = -1;
      const float wt = sub_round_weights(sub, d.n_sub, r0 + base0, M, k2, lane, w, incl, dummy);
      __syncthreads();
      if (lane == 0) s_wtot[warp] = wt;
      __syncthreads();
      float woff = 0.f;
      for (int k = 0; k < NW; ++k) woff = woff + s_wtot[k];
      run = run + woff;
    }
    S = run;
  }
  float run = 0.f;
  for (int r0 = 0; r0 < d.n_sub; r0 += SUB_ROUND) {
    int last = -1;
    const float wt = sub_round_weights(sub, d.n_sub, r0 + base0, M, k2, lane, w, incl, last);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) last = max(last, __shfl_xor_sync(0xffffffffu, last, o));
    if (r0 > 0) __syncthreads();  // s_wtot of the previous round has been read
    if (lane == 0) {
      s_wtot[warp] = wt;
      if (last >= 0) atomicMax(&s_last, last);
    }
    __syncthreads();
    float woff = 0.f, total = 0.f;
    for (int k = 0; k < NW; ++k) {
      if (k == warp) woff = total;
      total = total + s_wtot[k];
    }
    if (one_round) S = total;
    const float target = d.u[p] * S;
    // the lane's entries: lo = run + (woff + (carry_j + excl_j)), hi likewise
    // with incl_j (the shuffles first, all independent; then the carries)
    float excl[SUB_REG], tot[SUB_REG];
#pragma unroll
    for (int j = 0; j < SUB_REG; ++j) {
      excl[j] = __shfl_up_sync(0xffffffffu, incl[j], 1);
      tot[j] = __shfl_sync(0xffffffffu, incl[j], 31);
    }
    float carry = 0.f;
    int hit = -1;
    float hit_lo = 0.f;
#pragma unroll
    for (int j = 0; j < SUB_REG; ++j) {
      const float lo = run + (woff + (carry + (lane == 0 ? 0.f : excl[j])));
      const float hi = run + (woff + (carry + incl[j]));
      if (target >= lo && target < hi) {
        hit = j;
        hit_lo = lo;
      }
      carry = carry + tot[j];
    }
    if (hit >= 0) {  // one entry of the whole CTA at most
#pragma unroll
      for (int j = 0; j < SUB_REG; ++j)
        if (j == hit) s_frac = (target - hit_lo) / w[j];
      s_k = r0 + base0 + 32 * hit;
    }
    run = run + total;
    __syncthreads();
    if (s_k >= 0) break;
  }
  // (clamped: a defect upstream must not turn into reads outside w)
  const int ks = min(max(s_k >= 0 ? s_k : s_last, 0), d.n_sub - 1);
  const float frac = s_k >= 0 ? fminf(fmaxf(s_frac, 0.f), 1.f) : 1.f;
  // The subtile's 32 rows times the position's rows on the tensor cores
  // (mma.sync m16n8k16, bf16 operands, fp32 sums): warp w takes rows
  // 16 (w & 1) .. + 15 and every 16th 32-element chunk of the hidden
  // dimension from w >> 1.  A chunk is read as one 16-byte vector per thread
  // and row (8 consecutive k): thread (g, q) = (lane / 4, lane % 4) holds
  // k = 32 c + 8 q .. + 7 of rows g and g + 8, and its fragments use them as
  // the k slots it owns in two consecutive k16 steps (2q, 2q+1 | 2q+8, 2q+9);
  // the fragment of column g (0: o, 1: o', the others zero) takes the same k
  // of the position's rows from shared memory.  Both operands see one
  // permutation of k, so the sums are the dot products.
  {
    const int g = lane >> 2, q = lane & 3;
    const int mt = warp & 1, cw = warp >> 1;
    const int nch = d.H / 32;
    const int r0 = 16 * mt + g, r1 = r0 + 8;  // rows within the subtile
    // (rows at or past V read row V - 1: in bounds; their z is discarded)
    const uint4* const w0 = static_cast<const uint4*>(d.w) +
                            static_cast<long long>(min(ks * 32 + r0, d.V - 1)) * nvec + q;
    const uint4* const w1 = static_cast<const uint4*>(d.w) +
                            static_cast<long long>(min(ks * 32 + r1, d.V - 1)) * nvec + q;
    const uint4* const hq = s_h + (g == 1 ? nvec : 0) + q;
    const bool hcol = g == 0 || (g == 1 && !d.zonly);
    for (int c = cw; c < nch; c += 16) {  // every chunk of this warp toward L2 first
      asm volatile("prefetch.global.L2 [%0];" ::"l"(w0 + 4 * c));
      asm volatile("prefetch.global.L2 [%0];" ::"l"(w1 + 4 * c));
    }
    float acc4[4] = {0.f, 0.f, 0.f, 0.f};
    constexpr int NB = SUB_LD / 2;  // chunks per batch
    for (int c0 = cw; c0 < nch; c0 += 16 * NB) {
      uint4 a0[NB], a1[NB];
#pragma unroll
      for (int u = 0; u < NB; ++u) {
        const int c = c0 + 16 * u;
        a0[u] = c < nch ? ldg_batch(w0 + 4 * c) : make_uint4(0, 0, 0, 0);
        a1[u] = c < nch ? ldg_batch(w1 + 4 * c) : make_uint4(0, 0, 0, 0);
      }
#pragma unroll
      for (int u = 0; u < NB; ++u) {
        const int c = c0 + 16 * u;
        if (c < nch) {  // warp-uniform
          const uint4 h = hcol ? hq[4 * c] : make_uint4(0, 0, 0, 0);
          mma_bf16_16816(acc4, a0[u].x, a1[u].x, a0[u].y, a1[u].y, h.x, h.y);
          mma_bf16_16816(acc4, a0[u].z, a1[u].z, a0[u].w, a1[u].w, h.z, h.w);
        }
      }
    }
    if (q == 0) {  // columns 0 and 1 of rows r0 and r1
      s_part[cw][r0] = make_float2(acc4[0], acc4[1]);
      s_part[cw][r1] = make_float2(acc4[2], acc4[3]);
    }
  }
  __syncthreads();
  if (warp != 0) return;
  const int npos = d.gamma + 1, b = p / npos;
  int last_pos;
  {
    float so = 0.f, sr = 0.f;  // row `lane` of the subtile: the 16 partials in order
#pragma unroll
    for (int k = 0; k < 16; ++k) {
      so += s_part[k][lane].x;
      sr += s_part[k][lane].y;
    }
    const float z = ks * 32 + lane < d.V ? (d.zonly ? so : fmaf(d.alpha, sr, (1.f - d.alpha) * so))
                                         : NEG_INF;
    float zmax = z;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) zmax = fmaxf(zmax, __shfl_xor_sync(0xffffffffu, zmax, o));
    const float ew = z == NEG_INF ? 0.f : ex2_approx((z - zmax) * k2);
    float cum = ew;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float y = __shfl_up_sync(0xffffffffu, cum, o);
      if (lane >= o) cum += y;
    }
    const float tgt = frac * __shfl_sync(0xffffffffu, cum, 31);
    const unsigned over = __ballot_sync(0xffffffffu, ew > 0.f && cum > tgt);
    const unsigned pos = __ballot_sync(0xffffffffu, ew > 0.f);
    const int r = over != 0u ? __ffs(over) - 1 : (pos != 0u ? 31 - __clz(pos) : 0);
    unsigned t = 0u;
    if (lane == 0) {
      d.xhat[p] = ks * 32 + r;
      if (acc.accepted_len != nullptr)  // release: this position's draw before the ticket;
        asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;"  // acquire: the others'
                     : "=r"(t) : "l"(d.tickets + b) : "memory");
    }
    last_pos = acc.accepted_len != nullptr &&
               __shfl_sync(0xffffffffu, t, 0) == static_cast<unsigned>(npos - 1);
  }
  if (!last_pos) return;
  // the sequence's last position: the acceptance against every draw (Alg. 2 or 3),
  // 32 drafts per round (the ticket's acquire made the other draws visible to
  // lane 0; the warp barrier below passes that on to the warp)
  __syncwarp();
  if (lane == 0) d.tickets[b] = 0u;  // re-armed for the next launch
  int n = d.gamma, t = 0;
  for (int i0 = 0; i0 <= d.gamma; i0 += 32) {  // the draws x^_1..x^_{gamma+1}
    const int i = i0 + lane;
    const int xh = i <= d.gamma ? __ldcg(d.xhat + b * npos + i) : 0;
    bool ok = true;
    if (i < d.gamma) {
      const int x = d.drafts[b * d.gamma + i];
      if (acc.mode == RV_ACCEPT_TYPICAL) {  // Alg. 3: the threshold, t still the draw at n+1
        const float* sc = d.scores + static_cast<long long>(b * npos + i) * RV_NSCORES;
        ok = position_kept(acc, x, xh, __ldcg(sc + RV_SCORE_LOGP_FUSED),
                           __ldcg(sc + RV_SCORE_ENT_ORIG));
      } else {
        ok = x == xh;
      }
    }
    if (i < d.gamma) acc.accept_mask[b * d.gamma + i] = ok ? 1 : 0;
    const unsigned bad = __ballot_sync(0xffffffffu, !ok);
    if (bad != 0u && n == d.gamma) n = i0 + __ffs(bad) - 1;
    const int tn = __shfl_sync(0xffffffffu, xh, (n - i0) & 31);
    if (n >= i0 && n < i0 + 32) t = tn;
  }
  if (lane == 0) {
    acc.accepted_len[b] = n;
    acc.next_token[b] = t;
    acc.ctx_out[b] = acc.ctx_in[b] + n + acc.ctx_extra;
  }
}

cudaError_t launch_sample_subtiles(const SubtileDraw& d, const AcceptArgs* acc, cudaStream_t s) {
  if (d.P <= 0) return cudaSuccess;
  if (d.H % 32 != 0 || (acc && d.tickets == nullptr)) return cudaErrorInvalidValue;
  AcceptArgs a = {};
  if (acc) a = *acc;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(d.P, 1, 1);
  cfg.blockDim = dim3(SUB_THREADS, 1, 1);
  cfg.dynamicSmemBytes = static_cast<size_t>(d.zonly ? 1 : 2) * d.H * 2;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (cfg.dynamicSmemBytes > 48 * 1024) {  // hidden sizes above 12288
    const cudaError_t e = cudaFuncSetAttribute(sample_subtiles_kernel,
                                               cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               static_cast<int>(cfg.dynamicSmemBytes));
    if (e != cudaSuccess) return e;
  }
  return cudaLaunchKernelEx(&cfg, sample_subtiles_kernel, d, a);
}

// ---------------------------------------------------------------- typical accept (Alg. 3)
__global__ void accept_typical_kernel(const int32_t* __restrict__ drafts,
                                      const float* __restrict__ scores,
                                      const int32_t* __restrict__ argmax, int B, int gamma,
                                      AcceptArgs a) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  int n = gamma;
  for (int i = 0; i < gamma; ++i) {
    const float* sc = scores + (static_cast<long long>(b) * (gamma + 1) + i) * RV_NSCORES;
    const bool ok = position_kept(a, drafts[b * gamma + i], argmax[b * (gamma + 1) + i],
                                  sc[RV_SCORE_LOGP_FUSED], sc[RV_SCORE_ENT_ORIG]);
    a.accept_mask[b * gamma + i] = ok ? 1 : 0;
    if (!ok && n == gamma) n = i;
  }
  a.accepted_len[b] = n;
  a.next_token[b] = argmax[b * (gamma + 1) + n];
  a.ctx_out[b] = a.ctx_in[b] + n + a.ctx_extra;
}

cudaError_t launch_accept_typical(const int32_t* drafts, const float* scores,
                                  const int32_t* argmax, int B, int gamma, float log_eps,
                                  float log_delta, uint8_t* accept_mask, int32_t* accepted_len,
                                  int32_t* next_token, const int32_t* ctx_in, int32_t* ctx_out,
                                  cudaStream_t s, int ctx_extra) {
  AcceptArgs a{accept_mask, accepted_len, next_token, ctx_in, ctx_out, RV_ACCEPT_TYPICAL, log_eps,
               log_delta, ctx_extra};
  accept_typical_kernel<<<(B + 127) / 128, 128, 0, s>>>(drafts, scores, argmax, B, gamma, a);
  return cudaGetLastError();
}

cudaError_t launch_accept(const int32_t* drafts, const int32_t* argmax, int B, int gamma,
                          uint8_t* accept_mask, int32_t* accepted_len, int32_t* next_token,
                          const int32_t* ctx_in, int32_t* ctx_out, cudaStream_t s,
                          int ctx_extra) {
  accept_kernel<<<(B + 127) / 128, 128, 0, s>>>(drafts, argmax, B, gamma, accept_mask,
                                                accepted_len, next_token, ctx_in, ctx_out,
                                                ctx_extra);
  return cudaGetLastError();
}

}  // namespace rv
