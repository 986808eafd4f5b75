// Launch interface between the C-ABI host code (rv_host.cpp) and the CUDA
// translation units.  Plain structs of sizes and device pointers; every
// launcher enqueues on `stream` and returns the cudaGetLastError() of the launch.
#pragma once

#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

namespace rv {

// Per-pair partial statistics written by each head CTA, merged by head_merge.
// Layout [slot][pair][HEAD_STAT_FIELDS] (three 16-byte vectors per pair).
enum HeadStat : int {
  ST_M_O = 0,  // running max of o_i over the CTA's vocab rows
  ST_S_O,      // sum exp(o_i - m)
  ST_M_R,      // same for the reflective logits o'_i
  ST_S_R,
  ST_M_Z,      // same for the fused logits z_i
  ST_S_Z,
  ST_BEST_V,   // max of z_i over rows v != x_i
  ST_BEST_I,   // its row (int bits; smallest on ties)
  ST_T_O,      // sum exp(o_i - m) (o_i - m): with ST_S_O, the entropy of softmax(o_i)
  HEAD_STAT_USED,
  HEAD_STAT_FIELDS = 12
};
constexpr int GATHER_FIELDS = 4;  // o_i[x_i], o'_i[x_i], z_i[x_i], unused

// Pair p = b * (gamma + 1) + i scores x_{i+1} (none for i = gamma).  Pairs are
// split into chunks of at most MAX_PAIRS_PER_CHUNK; chunk c holds pairs
// [c*pairs_per_chunk, ...).  Its gathered hidden rows form a block of
// 2*pad_pairs rows: original rows first, reflective rows after pad_pairs.
constexpr int MAX_PAIRS_PER_CHUNK = 128;
// The pre-blended head gathers one row per pair (the blended hidden state), so
// its chunks take up to 256 pairs (pad_pairs rows, one accumulator column each).
constexpr int MAX_ZPAIRS_PER_CHUNK = 256;

struct HeadPlan {
  int P;               // total pairs B*(gamma+1)
  int n_chunks;
  int pairs_per_chunk; // Pc
  int pad_pairs;       // Pcp = round_up(Pc, 8) (pre-blended: round_up(Pc, 16))
  int N;               // MMA N (columns of the TMEM accumulator): 2*Pcp (pre-blended: Pcp)
  int n_vtiles;        // ceil(V / 128)
  int slots;           // CTAs per chunk (= partial slots)
  bool pair;           // CTA-pair kernel (k_head_tc2.cu): slots = 2 * pairs
  // CTA-pair kernel: the chunk's pairs in `sub` sub-groups of `sub_pairs`
  // (pad_pairs = sub * sub_pairs), one accumulator each; 1 and pad_pairs otherwise
  int sub = 1;
  int sub_pairs = 0;
  bool zonly = false;  // pre-blended head: one blended row per pair, z statistics only
  bool standard = false;  // standard verification: z-only on the original rows (Lh = gamma+1)
};

// Optional acceptance fused into the head merge (rv_verify_step).
// mode RV_ACCEPT_EXACT: x_i == argmax p_i (Alg. 2); RV_ACCEPT_TYPICAL:
// log p_i(x_i) > min(log_eps, log_delta - H(softmax(o_i))) (Alg. 3).
struct AcceptArgs {
  uint8_t* accept_mask;
  int32_t* accepted_len;
  int32_t* next_token;
  const int32_t* ctx_in;
  int32_t* ctx_out;
  int mode;
  float log_eps, log_delta;
  int ctx_extra = 0;  // 1 with the pending-token block: t stays in the context too
};

// Outputs of the merge when the LM-head kernel finishes it itself (its last
// CTA), instead of the separate finalize launch.
struct HeadFinal {
  float* scores;
  int32_t* argmax;
  float* margin;
  AcceptArgs acc;  // acc.accepted_len == nullptr: no acceptance
  int zonly = 0;   // pre-blended head: the original / reflective fields are NaN
};
// Largest pair count whose merge the head kernel's last CTA finishes itself.
#ifndef RV_HEAD_FUSED_FINAL_MAX_PAIRS
#define RV_HEAD_FUSED_FINAL_MAX_PAIRS 64
#endif
constexpr int HEAD_FUSED_FINAL_MAX_PAIRS = RV_HEAD_FUSED_FINAL_MAX_PAIRS;

struct HeadArgs {
  const void* hidden;      // [B, Lb+1, H]
  const void* w;           // [V, H]
  const int32_t* drafts;   // [B, gamma]
  int B, gamma, R, V, H;
  float alpha;
  float* partials;         // [slots][P][HEAD_STAT_FIELDS]
  float* gathered;         // [P][GATHER_FIELDS]
  unsigned* status;
  unsigned* tile_counter;  // LM-head tile counter, zeroed by the prep kernel
  unsigned* done_counter;  // finished LM-head CTAs (fused merge), zeroed by the prep kernel
  float* zout = nullptr;   // [P][V] fused logits z_i (speculative sampling), or none
  // [B] per-sequence tickets of the finalize launch's acceptance (zero between
  // launches; needed when the finalize runs the acceptance)
  unsigned* seq_tickets = nullptr;
  // Sampled exact match (Alg. 2, temperature T): per position and 32-row
  // subtile k (vocab rows [32k, 32k+32) below V) the pair (max z, sum exp((z -
  // max) / T)), [P][ceil(V / 32)]; or none.  The bf16 tensor-core heads only.
  float2* zsub = nullptr;
  float inv_t = 1.f;       // 1 / T for zsub
};

// ---- small kernels (k_small.cu)
// pending != nullptr: the pending-token block [t, x, prompt, prefix, x] (Lb + 1 positions).
cudaError_t launch_pack_block(const int32_t* drafts, const int32_t* prompt, const int32_t* prefix,
                              const int32_t* ctx, int B, int gamma, int n_prompt, int n_prefix,
                              int32_t* block_ids, int32_t* pos_ids, cudaStream_t s,
                              const int32_t* pending = nullptr, int copy = 1);
// Optional block packing (Eq. 1) for rv_verify_step: pack.block == nullptr skips it.
struct PackArgs {
  const int32_t* drafts;
  const int32_t* prompt;
  const int32_t* prefix;
  const int32_t* ctx;
  int B, gamma, n_prompt, n_prefix;
  int32_t* block;
  int32_t* pos;
  const int32_t* pending = nullptr;  // [B]: the pending-token block [t, x, prompt, prefix, x]
  int copy = 1;  // 0: standard verification's block, the drafts alone (no template, no copy)
};
// hidden rows of every chunk into hsel [n_chunks * N, H] (bf16), pads zeroed;
// also packs the block when `pack` is given (one launch for both).
cudaError_t launch_prep(const HeadArgs& a, const HeadPlan& p, void* hsel, const PackArgs* pack,
                        cudaStream_t s);
// Merge the head's per-CTA statistics into scores / argmax / margin, and run
// the acceptance of each sequence when `acc` is given.
cudaError_t launch_head_finalize(const HeadArgs& a, const HeadPlan& p, float* scores,
                                 int32_t* argmax, float* margin, const AcceptArgs* acc,
                                 cudaStream_t s);
cudaError_t launch_accept(const int32_t* drafts, const int32_t* argmax, int B, int gamma,
                          uint8_t* accept_mask, int32_t* accepted_len, int32_t* next_token,
                          const int32_t* ctx_in, int32_t* ctx_out, cudaStream_t s,
                          int ctx_extra = 0);
// Speculative-sampling acceptance (Alg. 1) from the head's scores and the
// fused logits it wrote (z [P][V]), the draft distributions q [B][gamma][V],
// uniforms r [B][gamma] and u [B].  One CTA per sequence.
cudaError_t launch_accept_speculative(const int32_t* drafts, const float* q, const float* r,
                                      const float* u, const float* scores, const float* z, int B,
                                      int gamma, int V, uint8_t* accept_mask,
                                      int32_t* accepted_len, int32_t* next_token,
                                      const int32_t* ctx_in, int32_t* ctx_out, unsigned* status,
                                      cudaStream_t s, int ctx_extra = 0);
// Target tokens at temperature T (Alg. 2 with sampling): for each of the P
// positions, xhat[p] ~ softmax(z[p] / T) by inverse CDF with u[p]; z [P][V]
// are the fused logits the head wrote.  One CTA per position.
cudaError_t launch_sample_fused(const float* z, const float* u, int P, int V, float temperature,
                                int32_t* xhat, cudaStream_t s);
// Target tokens at temperature T from the head's subtile sums (zsub above):
// for each of the P positions the inverse CDF of softmax(z / T) at u[p] picks
// the 32-row subtile from the sums, then the row inside it from that
// subtile's fused logits, recomputed from the head's operands (w rows, the
// position's hsel rows as `launch_prep` laid them out for plan `pl`).  With
// `acc`, the last of a sequence's positions to finish runs the acceptance: exact
// match against the draws, or with acc->mode == RV_ACCEPT_TYPICAL the typical
// rule on `scores`, with t the draw at n+1 (a ticket per sequence in `tickets`, zero between
// launches).  One CTA per position.
struct SubtileDraw {
  const float2* zsub;
  int n_sub;
  const float* u;       // [P]
  float inv_t;
  const void* w;        // [V][H] bf16
  const void* hsel;     // prep's rows
  int V, H, P, gamma;
  int Pc, Pcp, N;       // the head plan's chunking of hsel
  int zonly;            // 1: one row per position (z = w . row)
  float alpha;
  int32_t* xhat;        // [P]
  const int32_t* drafts;
  unsigned* tickets;
  const float* scores;  // [P][RV_NSCORES] (the typical rule's log-probability and entropy)
};
cudaError_t launch_sample_subtiles(const SubtileDraw& d, const AcceptArgs* acc, cudaStream_t s);
// Typical acceptance (Alg. 3) from the head's scores and argmax.
cudaError_t launch_accept_typical(const int32_t* drafts, const float* scores,
                                  const int32_t* argmax, int B, int gamma, float log_eps,
                                  float log_delta, uint8_t* accept_mask, int32_t* accepted_len,
                                  int32_t* next_token, const int32_t* ctx_in, int32_t* ctx_out,
                                  cudaStream_t s, int ctx_extra = 0);

// ---- LM head (k_head_tc.cu: bf16 tcgen05; k_head_simt.cu: fp32)
// Vocab rows per TMA box of the weight: full tiles use HEAD_TILE_ROWS, the
// partial last tile of a CTA HEAD_W_BOX_ROWS; the tensor maps (host) and the
// kernel's transaction byte counts (device) both use them.
constexpr int HEAD_TILE_ROWS = 128;
constexpr int HEAD_W_BOX_ROWS = 16;
struct HeadTcLaunch {
  CUtensorMap tm_w;    // W [V, H] bf16, box {64, 128}, 128B swizzle
  CUtensorMap tm_w16;  // W [V, H] bf16, box {64, 16}, 128B swizzle
  CUtensorMap tm_h;    // hsel [n_chunks*N, H] bf16, box {64, N}, 128B swizzle
  int stages;
  int unit_rows;       // vocab split granularity across CTAs (multiple of 16, <= 128)
  size_t smem_bytes;
};
// `pairs` = pad_pairs of the plan (the statistics tables' length)
size_t head_tc_smem_bytes(int N, int pairs, int stages);
int head_tc_max_stages(int N, int pairs, size_t smem_limit);
int head_tc_stages(int N, int pairs, size_t smem_limit);  // the depth the launcher uses
cudaError_t head_tc_configure(size_t smem_bytes);  // cudaFuncSetAttribute
// fin != nullptr: the kernel's last CTA merges the statistics and writes the
// outputs (P <= HEAD_FUSED_FINAL_MAX_PAIRS).  The launch uses programmatic
// dependent launch: it must directly follow the prep launch on `s`.
cudaError_t launch_head_tc(const HeadArgs& a, const HeadPlan& p, const HeadTcLaunch& l,
                           const HeadFinal* fin, cudaStream_t s);
cudaError_t launch_head_simt(const HeadArgs& a, const HeadPlan& p, cudaStream_t s);
// CTA-pair LM head (k_head_tc2.cu, tcgen05 cta_group::2): 256-row vocab tiles,
// each CTA of a pair stages its 128 weight rows and half of the N hidden rows
// (tm_h box {64, N/2}); the grid is p.slots (= 2 * pairs) x n_chunks in
// clusters of 2.
#ifndef RV_HEAD_PAIR_MIN_N
#define RV_HEAD_PAIR_MIN_N 96
#endif
constexpr int HEAD_PAIR_MIN_N = RV_HEAD_PAIR_MIN_N;  // N from which pairs are used
// Chunks of the CTA-pair head: at most HEAD_PAIR_MAX_CHUNK pairs per chunk; a
// chunk of more than MAX_PAIRS_PER_CHUNK pairs is split into two sub-groups.
#ifndef RV_HEAD_PAIR_MAX_CHUNK
#define RV_HEAD_PAIR_MAX_CHUNK 160
#endif
constexpr int HEAD_PAIR_MAX_CHUNK = RV_HEAD_PAIR_MAX_CHUNK;
void head_pair_chunks(int P, int* n_chunks, int* pairs_per_chunk, int* sub, int* sub_pairs);
size_t head_tc2_smem_bytes(int N, int pairs, int stages);
int head_tc2_stages(int N, int pairs, size_t smem_limit);
cudaError_t head_tc2_configure(size_t smem_bytes);
// co-resident CTA pairs (occupancy query)
int head_tc2_max_pairs(int N, int pairs, int stages);

// whether the kernel takes the plan (its sub-groups fit an accumulator slot layout)
bool head_tc2_supports(const HeadPlan& p);
cudaError_t launch_head_tc2(const HeadArgs& a, const HeadPlan& p, const HeadTcLaunch& l,
                            const HeadFinal* fin, cudaStream_t s);

// ---- attention (k_attention.cu)
struct AttnArgs {
  const void* q;      // [B, Lb, Hq, D]
  const void* k_blk;  // [B, Lb, Hkv, D]
  const void* v_blk;
  void* k_cache;      // [B, Hkv, Cmax, D]
  void* v_cache;
  const int32_t* ctx;
  void* out;          // [B, Lb, Hq, D]
  int B, Lb, Hq, Hkv, D, Cmax;
  unsigned* status;
};
struct AttnPlan {
  int rows;        // query rows per KV head: Lb * G
  int row_groups;  // CTAs along the rows (<= 128 rows each)
  int splits;      // key splits
  int warps;       // warps per CTA (mma.sync kernel)
  bool tc;         // tcgen05 kernel (head_dim 128, larger batches)
};
// max_cluster: largest thread-block cluster the attention kernel can use (<= 16)
// allow_tc: the tcgen05 kernel may be chosen (its shapes and shared memory fit)
AttnPlan attn_plan(int B, int Lb, int Hq, int Hkv, int Cmax, int num_sms, bool bf16,
                   int max_cluster, int D, bool allow_tc);
size_t attn_bf16_smem_bytes(int D, int warps);
cudaError_t attn_configure(int* max_cluster);
cudaError_t launch_attention_bf16(const AttnArgs& a, const AttnPlan& p, cudaStream_t s);
cudaError_t launch_attention_f32(const AttnArgs& a, cudaStream_t s);
// tcgen05 attention (k_attention_tc.cu), head_dim 128: persistent CTAs that
// claim (sequence, KV head, row group, key chunk) items, then (when a
// sequence spans several chunks) a merge launch.
struct AttnTcPlan {
  int rows;        // query rows per KV head: Lb * G
  int n_rg;        // row groups of 128
  int chunk;       // cached keys per item
  int max_chunks;  // chunks of a sequence at capacity
  int slots;       // partial-result slots used: groups * max_chunks
  int grid;        // CTAs
  size_t smem_bytes;
};
struct AttnTcMaps {
  CUtensorMap kc, vc;  // [B*Hkv*Cmax][D], box {64, 128}
  CUtensorMap kb, vb;  // [B*Lb][Hkv][D], box {64, 1, 128}
  CUtensorMap q;       // [B*Lb][Hq][D], box {64, G, 128 / G}
};
struct AttnTcScratch {
  float* part_o;       // [slots][128][128]
  float* part_ml;      // [slots][128][2]
  unsigned* counters;  // [2], zero between launches
  int max_slots = 0;   // slots allocated; a plan needing more is not launched
};
AttnTcPlan attn_tc_plan(int B, int Lb, int Hq, int Hkv, int Cmax, int num_sms);
bool attn_tc_supported(int Hq, int Hkv, int D);
size_t attn_tc_smem_max(int max_batch);
// partial-result slots any launch within these maxima may use
int attn_tc_max_slots(int max_batch, int Lb_max, int Hq, int Hkv, int num_sms);
cudaError_t attn_tc_configure(size_t smem_bytes);
bool attn_tc_encode(PFN_cuTensorMapEncodeTiled_v12000 enc, const AttnArgs& x, AttnTcMaps* m);
cudaError_t launch_attention_tc(const AttnArgs& x, const AttnTcPlan& p, const AttnTcMaps& m,
                                const AttnTcScratch& sc, cudaStream_t s);

}  // namespace rv
