// LM head of the verify step on the 5th-generation tensor cores (sm_103a):
//
//   acc[v][c] = sum_k W[v][k] * hsel[c][k]   for 128 vocab rows v per tile and
//   the N gathered hidden rows c of one pair chunk (original rows 0..Pcp-1,
//   reflective rows Pcp..2Pcp-1), i.e. o_i and o_{m+i-1} of Alg. 1,
//
// followed by the online log-softmax / fusion epilogue (Eq. 2) so that no
// logit is ever written to memory.  Swap-AB orientation: the vocab is the MMA
// M dimension (128 TMEM lanes), the few hidden rows are N (16..256 columns).
//
// Vocab tiles of 128 rows: with one pair chunk the producer warp claims them
// from a shared counter (dynamic: a CTA slowed by other work on its SM takes
// fewer), and passes each tile to the MMA and epilogue warps through a small
// mbarrier-guarded ring.  With several chunks each CTA takes a static range
// (units of `unit_rows` rows) so the chunk CTAs of a cluster stay in step.
// Full tiles arrive as one 128-row TMA box; a partial tile as 16-row boxes
// (its missing rows are never loaded and their accumulator lanes are masked).
//
// Persistent CTA per SM, warp-specialised:
//   warp 0      TMA producer: W tile [128 x 64] + hsel tile [N x 64] per stage
//               into a ring of `stages` 128B-swizzled shared-memory buffers
//   warp 1      allocates TMEM (2 accumulator slots of N columns) and issues
//               tcgen05.mma (M=128, N, K=16) from one thread
//   warps 2..    epilogue (4 warps, or 8 above 32 pairs per chunk): tcgen05.ld of
//               the finished accumulator slot, fusion, warp-shuffle
//               max/sum/argmax, running statistics in shared memory; with 8,
//               the two warps of a lane quadrant take alternate groups of 8 pairs
// When the pairs need several chunks, the chunk CTAs of one vocab range form a
// cluster: they stream the same weight tiles together, so the second read of
// each tile is served by L2.
// The weight streams from HBM exactly once per step (evict-first); the small
// hidden operand is re-read from L2 per tile (evict-last).
#include <cfloat>

#include "head_epilogue.cuh"
#include "rv_device.cuh"
#include "rv_kernels.h"

namespace rv {

constexpr int HT_BM = HEAD_TILE_ROWS;
constexpr int HT_BK = 64;
// Epilogue warps: 4 (one per TMEM lane quadrant) for up to 32 pairs per chunk,
// else 8 (two per quadrant, taking alternate groups of 8 pairs).
constexpr int HT_SMALL_PAIRS = 32;
__host__ __device__ constexpr int ht_threads(int epi_warps) { return 64 + epi_warps * 32; }
constexpr int HT_WBOX = HEAD_W_BOX_ROWS;             // vocab rows per TMA box of W
constexpr uint32_t HT_A_BYTES = HT_BM * HT_BK * 2;  // 16 KB
constexpr uint32_t HT_BOX_BYTES = HT_WBOX * HT_BK * 2;  // 2 KB

constexpr int HT_TRING = 4;  // tile-index ring between the producer and the consumers

struct HeadTcParams {
  int V, n_kb, N, Pcp, Pc, P, slots, stages, gamma;
  int n_vtiles;              // ceil(V / 128): tiles handed out by the counter
  unsigned* tile_counter;    // one chunk: shared tile counter (zeroed before launch); else null
  unsigned* done_counter;    // finished CTAs, for the fused merge (zeroed before launch)
  int B, fused;              // fused != 0: the last CTA merges and writes `fin`
  HeadFinal fin;
  int unit_rows;  // the vocab is split across CTAs in multiples of this (16..128)
  int units;      // ceil(V / unit_rows)
  uint32_t tmem_cols;
  float alpha;
  const int32_t* drafts;
  float* partials;
  float* gathered;
  float* zout;  // [P][V] fused logits, or null
  float2* zsub;  // [P][n_sub] subtile (max z, sum exp((z - max) / T)), or null
  int n_sub;
  float inv_t;
  unsigned* status;
  int zonly;    // pre-blended head: column j of the accumulator is z of pair j
};

static int ht_epi_warps(int pairs) { return pairs <= HT_SMALL_PAIRS ? 4 : 8; }

static size_t ht_fixed_bytes(int pairs) {
  // alignment slack + barriers/tile ring/misc + drafts + per-warp statistics (`pairs`
  // entries per lane quadrant) + per-warp staging rows of the tile reduction
  return 1024 + 512 + MAX_ZPAIRS_PER_CHUNK * 4 +
         static_cast<size_t>(4) * pairs * HEAD_STAT_STRIDE * 4 + 16 +
         static_cast<size_t>(ht_epi_warps(pairs)) * HEAD_SCR_FLOATS * 4;
}

size_t head_tc_smem_bytes(int N, int pairs, int stages) {
  return ht_fixed_bytes(pairs) + static_cast<size_t>(stages) * (HT_A_BYTES + N * 128);
}

int head_tc_max_stages(int N, int pairs, size_t smem_limit) {
  const size_t per = HT_A_BYTES + N * 128;
  if (smem_limit <= ht_fixed_bytes(pairs)) return 0;
  const int s = static_cast<int>((smem_limit - ht_fixed_bytes(pairs)) / per);
  return s > 12 ? 12 : s;
}

// Pipeline depth: about 128 KB of tiles in flight per SM streams the weight at
// full HBM bandwidth (measured on GB300: 7-8 stages of 18 KB beat both 4-6 and
// 11), and a CTA of at most ~150 KB leaves room on the SM for the concurrent
// small-batch attention kernel (75 KB).
#ifndef RV_HEAD_SMEM_TARGET_KB
#define RV_HEAD_SMEM_TARGET_KB 151
#endif
int head_tc_stages(int N, int pairs, size_t smem_limit) {
  const int per = static_cast<int>(HT_A_BYTES) + N * 128;
  const int room = RV_HEAD_SMEM_TARGET_KB * 1024 - static_cast<int>(ht_fixed_bytes(pairs));
  const int want = room > 0 ? room / per : 0;
  return std::max(2, std::min(head_tc_max_stages(N, pairs, smem_limit), std::max(4, want)));
}

// SUB: the epilogue also stores the subtile sums of sampled exact match (its
// own instantiation, so that the other modes carry none of its registers: the
// batch-1 attention CTA shares the SM with this one only within a register budget).
template <int EPI, bool SUB>
__global__ void __launch_bounds__(ht_threads(EPI), 1)
    head_tc_kernel(const __grid_constant__ CUtensorMap tm_w,
                   const __grid_constant__ CUtensorMap tm_w16,
                   const __grid_constant__ CUtensorMap tm_h, const HeadTcParams p) {
  // the merge launch that follows (programmatic dependent launch) may be
  // scheduled now; it waits for this grid before it reads anything
  asm volatile("griddepcontrol.launch_dependents;");
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* const gbase = smem_raw + (base - raw);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int slot_id = blockIdx.x;  // partial slot within the chunk
  const int chunk = blockIdx.y;
  const int S = p.stages;
  const uint32_t b_bytes = static_cast<uint32_t>(p.N) * 128u;

  const uint32_t a_tiles = base;
  const uint32_t b_tiles = base + S * HT_A_BYTES;
  const uint32_t bars = b_tiles + S * b_bytes;
  auto full_bar = [&](int s) { return bars + 8u * s; };
  auto empty_bar = [&](int s) { return bars + 8u * (S + s); };
  const uint32_t accf0 = bars + 8u * (2 * S);
  const uint32_t acce0 = accf0 + 16u;
  const uint32_t drain_bar = acce0 + 16u;
  const uint32_t tfull0 = drain_bar + 8u;            // tile ring: HT_TRING full barriers
  const uint32_t tempty0 = tfull0 + 8u * HT_TRING;   //            and HT_TRING empty barriers
  const uint32_t misc = (tempty0 + 8u * HT_TRING + 15u) & ~15u;
  uint32_t* const tmem_slot = reinterpret_cast<uint32_t*>(gbase + (misc - base));
  volatile int* const abort_flag = reinterpret_cast<volatile int*>(gbase + (misc - base) + 4);
  int2* const tring = reinterpret_cast<int2*>(gbase + (misc - base) + 16);  // (v0, v_end) or v0 < 0
  int* const s_drafts = reinterpret_cast<int*>(gbase + (misc - base) + 16 + 8 * HT_TRING);
  float* const stats =
      reinterpret_cast<float*>(gbase + (misc - base) + 16 + 8 * HT_TRING + MAX_ZPAIRS_PER_CHUNK * 4);
  const int tab = p.Pcp;  // pairs per statistics table
  // per-warp staging rows of the transposed tile reduction (16-byte aligned)
  float* const scr_base = reinterpret_cast<float*>(
      (reinterpret_cast<uintptr_t>(stats + 4 * tab * HEAD_STAT_STRIDE) + 15) & ~uintptr_t(15));

  const int pair0 = chunk * p.Pc;
  const int npairs = min(p.Pc, p.P - pair0);
  // Static split (several chunks): vocab rows [v_lo, v_hi) of this CTA.
  const int v_lo = p.unit_rows * static_cast<int>(static_cast<long long>(slot_id) * p.units / p.slots);
  const int v_hi = min(p.V, p.unit_rows * static_cast<int>(static_cast<long long>(slot_id + 1) *
                                                            p.units / p.slots));

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    mbar_init(accf0, 1);
    mbar_init(accf0 + 8, 1);
    mbar_init(acce0, EPI);
    mbar_init(acce0 + 8, EPI);
    mbar_init(drain_bar, 1);
    for (int k = 0; k < HT_TRING; ++k) {
      mbar_init(tfull0 + 8u * k, 1);
      mbar_init(tempty0 + 8u * k, 1 + EPI);  // the MMA thread + one lane per epilogue warp
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tm_w);
    tma_prefetch_desc(&tm_w16);
    tma_prefetch_desc(&tm_h);
  }
  if (warp == 1) tmem_alloc(smem_u32(tmem_slot), p.tmem_cols);
  if (warp >= 2) {
    const int e = threadIdx.x - 64;
    for (int j = e; j < MAX_ZPAIRS_PER_CHUNK; j += EPI * 32)
      s_drafts[j] = (j < npairs) ? pair_draft(p.drafts, pair0 + j, p.gamma) : -1;
    head_stats_init(stats, 4 * tab, e, EPI * 32);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      const uint64_t pol_w = policy_evict_first();
      const uint64_t pol_h = policy_evict_last();
      // The prep launch before this kernel (programmatic dependent launch)
      // gathers the hidden rows and zeroes the counters: wait for it here.
      asm volatile("griddepcontrol.wait;" ::: "memory");
      int s = 0, issued = 0;
      uint32_t ph = 0;
      bool ok = true;
      // Tile source: the shared counter (one chunk: CTAs slowed by other work
      // on their SM simply take fewer tiles) or this CTA's static range.
      int t_next = p.tile_counter ? static_cast<int>(atomicAdd(p.tile_counter, 1u)) : 0;
      for (int lt = 0; ok; ++lt) {
        int v0, v_end;
        if (p.tile_counter) {
          const int t = t_next;
          v0 = t < p.n_vtiles ? t * HT_BM : -1;
          v_end = v0 >= 0 ? min(p.V, v0 + HT_BM) : 0;
          if (v0 >= 0) t_next = static_cast<int>(atomicAdd(p.tile_counter, 1u));
        } else {
          v0 = v_lo + lt * HT_BM < v_hi ? v_lo + lt * HT_BM : -1;
          v_end = v0 >= 0 ? min(v_hi, v0 + HT_BM) : 0;
        }
        const int k = lt % HT_TRING;
        if (!mbar_wait(tempty0 + 8u * k, ((lt / HT_TRING) & 1) ^ 1u, abort_flag, p.status)) {
          ok = false;
          break;
        }
        tring[k] = make_int2(v0, v_end);
        mbar_arrive(tfull0 + 8u * k);
        if (v0 < 0) break;
        const int rows = v_end - v0;
        const int nbox = rows == HT_BM ? 0 : (rows + HT_WBOX - 1) / HT_WBOX;  // 0: one full box
        const uint32_t a_bytes = nbox == 0 ? HT_A_BYTES : nbox * HT_BOX_BYTES;
        for (int kb = 0; kb < p.n_kb; ++kb) {
          if (!mbar_wait(empty_bar(s), ph ^ 1u, abort_flag, p.status)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(full_bar(s), a_bytes + b_bytes);
          if (nbox == 0)
            tma_load_2d(a_tiles + s * HT_A_BYTES, &tm_w, kb * HT_BK, v0, full_bar(s), pol_w);
          for (int j = 0; j < nbox; ++j)
            tma_load_2d(a_tiles + s * HT_A_BYTES + j * HT_BOX_BYTES, &tm_w16, kb * HT_BK,
                        v0 + j * HT_WBOX, full_bar(s), pol_w);
          tma_load_2d(b_tiles + s * b_bytes, &tm_h, kb * HT_BK, chunk * p.N, full_bar(s), pol_h);
          ++issued;
          if (++s == S) {
            s = 0;
            ph ^= 1u;
          }
        }
      }
      if (!ok) {  // let every copy still in flight land before the CTA exits
        for (int j = max(0, issued - S); j < issued; ++j)
          drain_wait(full_bar(j % S), static_cast<uint32_t>((j / S) & 1));
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_f32(HT_BM, p.N);
      int s = 0;
      uint32_t ph = 0;
      bool ok = true;
      for (int lt = 0; ok; ++lt) {
        const int k = lt % HT_TRING;
        if (!mbar_wait(tfull0 + 8u * k, (lt / HT_TRING) & 1, abort_flag, p.status)) break;
        const int v0 = tring[k].x;
        mbar_arrive(tempty0 + 8u * k);
        if (v0 < 0) break;
        const int slot = lt & 1;
        const uint32_t aph = (lt >> 1) & 1;
        if (!mbar_wait(acce0 + 8u * slot, aph ^ 1u, abort_flag, p.status)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(slot * p.N);
        for (int kb = 0; kb < p.n_kb; ++kb) {
          if (!mbar_wait(full_bar(s), ph, abort_flag, p.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t ad = sw128_kmajor_desc(a_tiles + s * HT_A_BYTES);
          const uint64_t bd = sw128_kmajor_desc(b_tiles + s * b_bytes);
          static_assert(HT_BK == 64, "one 64-wide box per stage: four MMAs");
          tc_mma_stage4(d_tmem, ad, bd, idesc, kb != 0 ? 1u : 0u);
          tc_commit(empty_bar(s));
          if (++s == S) {
            s = 0;
            ph ^= 1u;
          }
        }
        if (ok) tc_commit(accf0 + 8u * slot);
      }
      // every MMA issued must be complete before TMEM is released
      tc_commit(drain_bar);
      drain_wait(drain_bar, 0);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ epilogue
    const int q = warp & 3;       // TMEM lane quadrant this warp may access
    const int ew = warp - 2;      // statistics table of this warp
    const int half = ew >> 2;     // which alternate groups of 8 pairs it takes
    // the two warps of a quadrant take disjoint pairs: they share one table
    float* const wstats = stats + q * tab * HEAD_STAT_STRIDE;
    float* const gathered = p.gathered + static_cast<long long>(pair0) * GATHER_FIELDS;
    for (int lt = 0;; ++lt) {
      const int k = lt % HT_TRING;
      bool ok = mbar_wait(tfull0 + 8u * k, (lt / HT_TRING) & 1, abort_flag, p.status);
      if (!__all_sync(0xffffffffu, ok)) break;
      const int2 tile = tring[k];
      __syncwarp();
      if (lane == 0) mbar_arrive(tempty0 + 8u * k);
      if (tile.x < 0) break;
      const int slot = lt & 1;
      const uint32_t aph = (lt >> 1) & 1;
      ok = mbar_wait(accf0 + 8u * slot, aph, abort_flag, p.status);
      if (!__all_sync(0xffffffffu, ok)) break;
      tc_fence_after();
      const int v = tile.x + q * 32 + lane;
      const bool valid = v < tile.y;
      const uint32_t trow =
          tmem_base + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>(slot * p.N);
      float* const zout = p.zout ? p.zout + static_cast<long long>(pair0) * p.V : nullptr;
      float2* const zsub = SUB ? p.zsub + static_cast<long long>(pair0) * p.n_sub : nullptr;
      for (int g8 = 8 * half; g8 < npairs; g8 += 8 * (EPI / 4)) {
        if (p.zonly) {
          float z[8];
          tmem_ld8(trow + g8, z);
          tmem_ld_wait();
          head_tile_z8_t(z, g8, npairs, v, valid, s_drafts, wstats, gathered,
                         scr_base + ew * HEAD_SCR_FLOATS, lane, zout, p.V, zsub, p.n_sub, p.inv_t);
          continue;
        }
        float o[8], r[8];
        tmem_ld8(trow + g8, o);
        tmem_ld8(trow + p.Pcp + g8, r);
        tmem_ld_wait();
        head_tile_pairs8_t(o, r, g8, npairs, v, valid, p.alpha, s_drafts, wstats, gathered,
                           scr_base + ew * HEAD_SCR_FLOATS, lane, zout, p.V, zsub, p.n_sub,
                           p.inv_t);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(acce0 + 8u * slot);
    }
    named_bar_sync(1, EPI * 32);
    head_stats_finish(stats, 4, tab, npairs,
                      p.partials + (static_cast<long long>(slot_id) * p.P + pair0) * HEAD_STAT_FIELDS,
                      threadIdx.x - 64, EPI * 32);
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, p.tmem_cols);
  }
  if (!p.fused) return;
  // Fused merge: the last CTA to finish (a ticket, no waiting) reads every
  // CTA's partial statistics and writes the per-position outputs.
  volatile int* const last = abort_flag + 1;
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0)
    *last = atomicAdd(p.done_counter, 1u) == gridDim.x * gridDim.y - 1 ? 1 : 0;
  __syncthreads();
  if (*last) {
    __threadfence();
    // the statistics tables are free now: reuse them for the choices
    head_merge_all(p.partials, p.gathered, s_drafts, p.B, p.gamma, p.V, p.P, p.slots, p.fin,
                   p.status, reinterpret_cast<int*>(stats), threadIdx.x, blockDim.x);
    if (threadIdx.x == 0) *p.done_counter = 0u;
  }
}

// The maximum shared-memory carveout lets the attention kernel's CTAs share an
// SM with this kernel's (the SM is otherwise configured just large enough for
// whichever kernel arrives first).
template <int EPI, bool SUB>
static cudaError_t head_tc_configure_one(size_t smem_bytes) {
  cudaError_t e = cudaFuncSetAttribute(head_tc_kernel<EPI, SUB>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem_bytes));
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(head_tc_kernel<EPI, SUB>,
                              cudaFuncAttributePreferredSharedMemoryCarveout,
                              cudaSharedmemCarveoutMaxShared);
}

cudaError_t head_tc_configure(size_t smem_bytes) {
  cudaError_t e = head_tc_configure_one<4, false>(smem_bytes);
  if (e == cudaSuccess) e = head_tc_configure_one<8, false>(smem_bytes);
  if (e == cudaSuccess) e = head_tc_configure_one<4, true>(smem_bytes);
  if (e == cudaSuccess) e = head_tc_configure_one<8, true>(smem_bytes);
  return e;
}

static uint32_t tmem_cols_for(int N) {
  uint32_t need = static_cast<uint32_t>(2 * N), c = 32;
  while (c < need) c <<= 1;
  return c;
}

cudaError_t launch_head_tc(const HeadArgs& a, const HeadPlan& pl, const HeadTcLaunch& l,
                           const HeadFinal* fin, cudaStream_t s) {
  HeadTcParams p;
  p.V = a.V;
  p.n_kb = (a.H + HT_BK - 1) / HT_BK;
  p.N = pl.N;
  p.Pcp = pl.pad_pairs;
  p.Pc = pl.pairs_per_chunk;
  p.P = pl.P;
  p.unit_rows = l.unit_rows;
  p.units = (a.V + l.unit_rows - 1) / l.unit_rows;
  p.n_vtiles = (a.V + HT_BM - 1) / HT_BM;
  p.tile_counter = pl.n_chunks == 1 ? a.tile_counter : nullptr;
  p.done_counter = a.done_counter;
  p.B = a.B;
  p.fused = fin != nullptr ? 1 : 0;
  if (fin) p.fin = *fin;
  p.slots = pl.slots;
  p.stages = l.stages;
  p.gamma = a.gamma;
  p.tmem_cols = tmem_cols_for(pl.N);
  p.alpha = a.alpha;
  p.drafts = a.drafts;
  p.partials = a.partials;
  p.gathered = a.gathered;
  p.zout = a.zout;
  p.zsub = a.zsub;
  p.n_sub = (a.V + 31) / 32;
  p.inv_t = a.inv_t;
  p.status = a.status;
  p.zonly = pl.zonly ? 1 : 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(pl.slots, pl.n_chunks, 1);
  const int epi = ht_epi_warps(pl.pad_pairs);
  cfg.blockDim = dim3(ht_threads(epi), 1, 1);
  cfg.dynamicSmemBytes = l.smem_bytes;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  int na = 0;
  attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[na].val.programmaticStreamSerializationAllowed = 1;
  ++na;
  if (pl.n_chunks >= 2 && pl.n_chunks <= 8) {
    attr[na].id = cudaLaunchAttributeClusterDimension;
    attr[na].val.clusterDim.x = 1;
    attr[na].val.clusterDim.y = pl.n_chunks;
    attr[na].val.clusterDim.z = 1;
    ++na;
  }
  cfg.attrs = attr;
  cfg.numAttrs = na;
  if (a.zsub != nullptr) {
    if (epi == 4)
      return cudaLaunchKernelEx(&cfg, head_tc_kernel<4, true>, l.tm_w, l.tm_w16, l.tm_h, p);
    return cudaLaunchKernelEx(&cfg, head_tc_kernel<8, true>, l.tm_w, l.tm_w16, l.tm_h, p);
  }
  if (epi == 4) return cudaLaunchKernelEx(&cfg, head_tc_kernel<4, false>, l.tm_w, l.tm_w16, l.tm_h, p);
  return cudaLaunchKernelEx(&cfg, head_tc_kernel<8, false>, l.tm_w, l.tm_w16, l.tm_h, p);
}

}  // namespace rv
