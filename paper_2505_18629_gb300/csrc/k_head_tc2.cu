// LM head of the verify step on CTA pairs (tcgen05 cta_group::2), for the
// larger pair counts where one SM per vocab tile is limited by its shared
// memory rather than by HBM:
//
//   acc[v][c] = sum_k W[v][k] * hsel[c][k]   over 256 vocab rows v per pair tile
//   (128 per CTA) and the N gathered hidden rows c of one pair chunk (original
//   rows 0..Pcp-1, reflective rows Pcp..2Pcp-1: o_i and o_{m+i-1} of Alg. 1),
//
// followed by the same online log-softmax / fusion epilogue (Eq. 2) as the
// one-CTA kernel, so that no logit is written to memory.  One MMA of the pair
// (M = 256, issued by the even CTA) reads the A operand from each CTA's own
// shared memory (its 128 weight rows) and the B operand split across the two
// (the even CTA holds the original rows, the odd CTA the reflective rows), so
// each SM stages its weight rows and only half of the hidden rows; every CTA
// gets its own 128 x N accumulator in its TMEM.
//
// Per CTA, warp-specialised:
//   warp 0      TMA producer: weight tile [128 x 128] + half hidden tile
//               [Pcp x 128] per stage (each as two 64-wide boxes); both CTAs'
//               copies complete on the even CTA's full barrier
//   warp 1      TMEM owner (both CTAs, 2 accumulator slots of N columns); in
//               the even CTA it also issues the pair's MMAs from one thread,
//               and its commits release the stage and fill the accumulator
//               slot in both CTAs
//   warps 2..   epilogue over this CTA's 128 rows; the slot is free again once
//               the epilogue warps of both CTAs have arrived on the even CTA's
//               empty-accumulator barrier
// The pair streams a static range of 256-row vocab tiles; the weight streams
// from HBM once per chunk (evict-first), the hidden rows are re-read from L2.
#include <cfloat>

#include "head_epilogue.cuh"
#include "rv_device.cuh"
#include "rv_kernels.h"

namespace rv {

namespace {

constexpr int H2_BM = 128;  // vocab rows per CTA per pair tile
constexpr int H2_BK = 128;  // K per stage: two 64-wide swizzled halves, 8 MMAs
constexpr uint32_t H2_A_HALF = H2_BM * 64 * 2;      // 16 KB
constexpr uint32_t H2_A_BYTES = 2 * H2_A_HALF;      // 32 KB
__host__ __device__ constexpr int h2_threads(int epi_warps) { return 64 + epi_warps * 32; }

struct Head2Params {
  int V, n_kb, N, Pcp, Pc, P, stages, gamma;
  int pair_slots;  // CTA pairs per chunk
  int n_ptiles;    // ceil(V / 256)
  unsigned* done_counter;
  int B, fused, slots;
  HeadFinal fin;
  uint32_t tmem_cols;
  float alpha;
  const int32_t* drafts;
  float* partials;
  float* gathered;
  float* zout;  // [P][V] fused logits, or null
  unsigned* status;
  int zonly;    // pre-blended head: column j of the accumulator is z of pair j
};

__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

// shared::cluster address of `addr` (a shared::cta address) in CTA `rank`
__device__ __forceinline__ uint32_t mapa_shared(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}

__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::
                   : "memory");
}

__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr)
               : "memory");
}

// 2-D TMA load into this CTA's shared memory whose completion (tx bytes) is
// signalled on a barrier of either CTA of the pair.
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const CUtensorMap* tm, int32_t x,
                                                 int32_t y, uint32_t bar_cluster, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
      ".L2::cache_hint [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tm)), "r"(x), "r"(y), "r"(bar_cluster), "l"(policy)
      : "memory");
}

// The 8 MMAs of one 128-wide K stage of the pair (two 64-wide boxes of A and
// of B, `a_half` / `b_half` descriptor units apart) from one asm block; only
// the first reads the accumulate flag (see tc_mma_stage4 for why).
__device__ __forceinline__ void tc2_mma_stage8(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                               uint32_t a_half, uint32_t b_half, uint32_t idesc,
                                               uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t.reg .b64 a<8>, b<8>, ha, hb;\n\t"
      "setp.ne.b32 p, %6, 0;\n\t"
      "cvt.u64.u32 ha, %4;\n\tcvt.u64.u32 hb, %5;\n\t"
      "add.s64 a1, %1, 2;\n\tadd.s64 a2, %1, 4;\n\tadd.s64 a3, %1, 6;\n\t"
      "add.s64 a4, %1, ha;\n\tadd.s64 a5, a4, 2;\n\tadd.s64 a6, a4, 4;\n\tadd.s64 a7, a4, 6;\n\t"
      "add.s64 b1, %2, 2;\n\tadd.s64 b2, %2, 4;\n\tadd.s64 b3, %2, 6;\n\t"
      "add.s64 b4, %2, hb;\n\tadd.s64 b5, b4, 2;\n\tadd.s64 b6, b4, 4;\n\tadd.s64 b7, b4, 6;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], a1, b1, %3, 1;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], a2, b2, %3, 1;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], a3, b3, %3, 1;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], a4, b4, %3, 1;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], a5, b5, %3, 1;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], a6, b6, %3, 1;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], a7, b7, %3, 1;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(a_half), "r"(b_half), "r"(accumulate)
      : "memory");
}

// Arrive on the barrier at `bar` in every CTA of `mask` once the MMAs issued
// so far by this thread are complete.
__device__ __forceinline__ void tc2_commit(uint32_t bar, uint16_t mask) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
      " [%0], %1;" ::"r"(bar),
      "h"(mask)
      : "memory");
}

}  // namespace

template <int EPI>
__global__ void __launch_bounds__(h2_threads(EPI), 1)
    head_tc2_kernel(const __grid_constant__ CUtensorMap tm_w,
                    const __grid_constant__ CUtensorMap tm_h, const Head2Params p) {
  // the merge launch that follows (programmatic dependent launch) may be
  // scheduled now; it waits for this grid before it reads anything
  asm volatile("griddepcontrol.launch_dependents;");
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* const gbase = smem_raw + (base - raw);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t crank = cluster_ctarank();
  const uint32_t rank = crank & 1u;  // 0: the pair's MMA issuer
  const bool leader = rank == 0;
  // commit mask: this pair's two CTAs (the stage release and the accumulator)
  const uint16_t pair_mask = static_cast<uint16_t>(3u << (crank & ~1u));
  const int pair = blockIdx.x >> 1;
  const int chunk = blockIdx.y;
  const int slot_id = blockIdx.x;  // partial slot within the chunk
  const int S = p.stages;
  // this CTA's half of the B rows (the original or the reflective rows; or, for
  // the pre-blended head, the first or second half of the blended rows)
  const uint32_t b_half = static_cast<uint32_t>(p.N / 2) * 128u;  // one 64-wide half of B
  const uint32_t b_bytes = 2u * b_half;                          // this CTA's part of B

  const uint32_t a_tiles = base;
  const uint32_t b_tiles = base + S * H2_A_BYTES;
  const uint32_t bars = b_tiles + S * b_bytes;
  auto full_bar = [&](int s) { return bars + 8u * s; };
  auto empty_bar = [&](int s) { return bars + 8u * (S + s); };
  const uint32_t accf0 = bars + 8u * (2 * S);
  const uint32_t acce0 = accf0 + 16u;
  const uint32_t drain_bar = acce0 + 16u;
  const uint32_t misc = (drain_bar + 8u + 15u) & ~15u;
  uint32_t* const tmem_slot = reinterpret_cast<uint32_t*>(gbase + (misc - base));
  volatile int* const abort_flag = reinterpret_cast<volatile int*>(gbase + (misc - base) + 4);
  int* const s_drafts = reinterpret_cast<int*>(gbase + (misc - base) + 16);
  float* const stats =
      reinterpret_cast<float*>(gbase + (misc - base) + 16 + MAX_ZPAIRS_PER_CHUNK * 4);
  const int tab = p.Pcp;
  // per-warp staging rows of the transposed tile reduction (16-byte aligned)
  float* const scr_base = reinterpret_cast<float*>(
      (reinterpret_cast<uintptr_t>(stats + 4 * tab * HEAD_STAT_STRIDE) + 15) & ~uintptr_t(15));

  const int pair0 = chunk * p.Pc;
  const int npairs = min(p.Pc, p.P - pair0);
  const int pt0 = static_cast<int>(static_cast<long long>(pair) * p.n_ptiles / p.pair_slots);
  const int pt1 = static_cast<int>(static_cast<long long>(pair + 1) * p.n_ptiles / p.pair_slots);

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(full_bar(s), 1);   // the even CTA's expect-tx; both CTAs' bytes
      mbar_init(empty_bar(s), 1);  // the pair's MMA commit
    }
    mbar_init(accf0, 1);
    mbar_init(accf0 + 8, 1);
    mbar_init(acce0, 2 * EPI);  // the epilogue warps of both CTAs
    mbar_init(acce0 + 8, 2 * EPI);
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tm_w);
    tma_prefetch_desc(&tm_h);
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_slot)),
                 "r"(p.tmem_cols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
  }
  if (warp >= 2) {
    const int e = threadIdx.x - 64;
    for (int j = e; j < MAX_ZPAIRS_PER_CHUNK; j += EPI * 32)
      s_drafts[j] = (j < npairs) ? pair_draft(p.drafts, pair0 + j, p.gamma) : -1;
    head_stats_init(stats, 4 * tab, e, EPI * 32);
  }
  // both CTAs: barriers initialised and TMEM allocated before any cross-CTA use
  tc_fence_before();
  cluster_sync();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const uint32_t leader_rank = cluster_ctarank() & ~1u;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      const uint64_t pol_w = policy_evict_first();
      const uint64_t pol_h = policy_evict_last();
      asm volatile("griddepcontrol.wait;" ::: "memory");  // the row gather before this launch
      int s = 0, issued = 0;
      uint32_t ph = 0;
      bool ok = true;
      for (int pt = pt0; pt < pt1 && ok; ++pt) {
        const int v0 = pt * 2 * H2_BM + static_cast<int>(rank) * H2_BM;
        for (int kb = 0; kb < p.n_kb; ++kb) {
          if (!mbar_wait(empty_bar(s), ph ^ 1u, abort_flag, p.status)) {
            ok = false;
            break;
          }
          if (leader) mbar_arrive_expect_tx(full_bar(s), 2u * (H2_A_BYTES + b_bytes));
          const uint32_t fb = mapa_shared(full_bar(s), leader_rank);
          const int hrow = chunk * p.N + static_cast<int>(rank) * (p.N / 2);
#pragma unroll
          for (int hf = 0; hf < 2; ++hf) {
            tma_load_2d_pair(a_tiles + s * H2_A_BYTES + hf * H2_A_HALF, &tm_w, kb * H2_BK + 64 * hf,
                             v0, fb, pol_w);
            tma_load_2d_pair(b_tiles + s * b_bytes + hf * b_half, &tm_h, kb * H2_BK + 64 * hf, hrow,
                             fb, pol_h);
          }
          ++issued;
          if (++s == S) {
            s = 0;
            ph ^= 1u;
          }
        }
      }
      // after an abort the even CTA lets every copy of the pair still in flight
      // land (its full barriers count both CTAs' bytes) before the final
      // cluster barrier releases the odd CTA
      if (!ok && leader) {
        for (int j = max(0, issued - S); j < issued; ++j)
          drain_wait(full_bar(j % S), static_cast<uint32_t>((j / S) & 1));
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer (even CTA)
    if (leader && lane == 0) {
      const uint32_t idesc = idesc_bf16_f32(2 * H2_BM, p.N);
      // descriptors of stage 0; stage s adds s * bytes / 16 to the start field
      const uint64_t ad0 = sw128_kmajor_desc(a_tiles), bd0 = sw128_kmajor_desc(b_tiles);
      const uint32_t a_step = H2_A_BYTES >> 4, b_step = b_bytes >> 4;
      const uint32_t a_hstep = H2_A_HALF >> 4, b_hstep = b_half >> 4;
      int s = 0;
      uint32_t ph = 0;
      bool ok = true;
      for (int pt = pt0, lt = 0; pt < pt1 && ok; ++pt, ++lt) {
        const int slot = lt & 1;
        if (!mbar_wait(acce0 + 8u * slot, ((lt >> 1) & 1) ^ 1u, abort_flag, p.status)) {
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
          const uint64_t ad = ad0 + static_cast<uint32_t>(s) * a_step;
          const uint64_t bd = bd0 + static_cast<uint32_t>(s) * b_step;
          tc2_mma_stage8(d_tmem, ad, bd, a_hstep, b_hstep, idesc, kb != 0 ? 1u : 0u);
          tc2_commit(empty_bar(s), pair_mask);
          if (++s == S) {
            s = 0;
            ph ^= 1u;
          }
        }
        if (ok) tc2_commit(accf0 + 8u * slot, pair_mask);
      }
      // every MMA issued must be complete before TMEM is released
      tc2_commit(drain_bar, static_cast<uint16_t>(1u << crank));
      drain_wait(drain_bar, 0);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ epilogue (both CTAs)
    const int q = warp & 3;    // TMEM lane quadrant this warp may access
    const int ew = warp - 2;   // statistics table of this warp
    const int half = ew >> 2;  // which alternate groups of 8 pairs it takes
    // the two warps of a quadrant take disjoint pairs: they share one table
    float* const wstats = stats + q * tab * HEAD_STAT_STRIDE;
    float* const gathered = p.gathered + static_cast<long long>(pair0) * GATHER_FIELDS;
    for (int pt = pt0, lt = 0; pt < pt1; ++pt, ++lt) {
      const int slot = lt & 1;
      const bool ok = mbar_wait(accf0 + 8u * slot, (lt >> 1) & 1, abort_flag, p.status);
      if (!__all_sync(0xffffffffu, ok)) break;
      tc_fence_after();
      const int v = pt * 2 * H2_BM + static_cast<int>(rank) * H2_BM + q * 32 + lane;
      const bool valid = v < p.V;
      const uint32_t trow =
          tmem_base + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>(slot * p.N);
      float* const zout = p.zout ? p.zout + static_cast<long long>(pair0) * p.V : nullptr;
      for (int g8 = 8 * half; g8 < npairs; g8 += 8 * (EPI / 4)) {
        if (p.zonly) {
          float z[8];
          tmem_ld8(trow + g8, z);
          tmem_ld_wait();
          head_tile_z8_t(z, g8, npairs, v, valid, s_drafts, wstats, gathered,
                         scr_base + ew * HEAD_SCR_FLOATS, lane, zout, p.V);
          continue;
        }
        float o[8], r[8];
        tmem_ld8(trow + g8, o);
        tmem_ld8(trow + p.Pcp + g8, r);
        tmem_ld_wait();
        head_tile_pairs8_t(o, r, g8, npairs, v, valid, p.alpha, s_drafts, wstats, gathered,
                           scr_base + ew * HEAD_SCR_FLOATS, lane, zout, p.V);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(mapa_shared(acce0 + 8u * slot, leader_rank));
    }
    named_bar_sync(1, EPI * 32);
    head_stats_finish(stats, 4, tab, npairs,
                      p.partials + (static_cast<long long>(slot_id) * p.P + pair0) * HEAD_STAT_FIELDS,
                      threadIdx.x - 64, EPI * 32);
  }

  tc_fence_before();
  __syncthreads();
  // the pair's MMAs are drained (and, after an abort, its copies): neither CTA
  // may release TMEM or exit while the other still reads its shared memory
  cluster_sync();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem_base),
                 "r"(p.tmem_cols)
                 : "memory");
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
    head_merge_all(p.partials, p.gathered, s_drafts, p.B, p.gamma, p.V, p.P, p.slots, p.fin,
                   p.status, reinterpret_cast<int*>(stats), threadIdx.x, blockDim.x);
    if (threadIdx.x == 0) *p.done_counter = 0u;
  }
}


// ---------------------------------------------------------------- host side

namespace {
#ifndef RV_HEAD2_EPI4_MAX_PAIRS
#define RV_HEAD2_EPI4_MAX_PAIRS 72
#endif
// epilogue warps: four (one per TMEM lane quadrant) up to this many pairs, else
// eight.  At 72 pairs (8B, B=16) four warps leave room for a fourth pipeline
// stage: 264 -> 254 us for the head.
int h2_epi_warps(int pairs) { return pairs <= RV_HEAD2_EPI4_MAX_PAIRS ? 4 : 8; }
size_t h2_fixed_bytes(int pairs) {
  return 1024 + 256 + 16 + MAX_ZPAIRS_PER_CHUNK * 4 +
         static_cast<size_t>(4) * pairs * HEAD_STAT_STRIDE * 4 + 64 + 16 +
         static_cast<size_t>(h2_epi_warps(pairs)) * HEAD_SCR_FLOATS * 4;
}
uint32_t h2_tmem_cols(int N) {
  uint32_t need = static_cast<uint32_t>(2 * N), c = 32;
  while (c < need) c <<= 1;
  return c;
}
}  // namespace

size_t head_tc2_smem_bytes(int N, int pairs, int stages) {
  return h2_fixed_bytes(pairs) + static_cast<size_t>(stages) * (H2_A_BYTES + (N / 2) * 256);
}

#ifndef RV_HEAD2_STAGE_TARGET_KB
#define RV_HEAD2_STAGE_TARGET_KB 200
#endif
int head_tc2_stages(int N, int pairs, size_t smem_limit) {
  const size_t per = H2_A_BYTES + (N / 2) * 256;
  if (smem_limit <= h2_fixed_bytes(pairs)) return 0;
  const int most = static_cast<int>((smem_limit - h2_fixed_bytes(pairs)) / per);
  const int want = static_cast<int>((RV_HEAD2_STAGE_TARGET_KB * 1024 + per - 1) / per);
  return std::max(0, std::min(std::min(most, 8), std::max(3, want)));
}

template <int EPI>
static cudaError_t head_tc2_configure_one(size_t smem_bytes) {
  cudaError_t e = cudaFuncSetAttribute(head_tc2_kernel<EPI>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem_bytes));
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(head_tc2_kernel<EPI>,
                           cudaFuncAttributePreferredSharedMemoryCarveout,
                           cudaSharedmemCarveoutMaxShared);
  return e;
}

cudaError_t head_tc2_configure(size_t smem_bytes) {
  cudaError_t e = head_tc2_configure_one<4>(smem_bytes);
  if (e == cudaSuccess) e = head_tc2_configure_one<8>(smem_bytes);
  return e;
}

int head_tc2_max_pairs(int N, int pairs, int stages) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2, 1, 1);
  cfg.blockDim = dim3(h2_threads(h2_epi_warps(pairs)), 1, 1);
  cfg.dynamicSmemBytes = head_tc2_smem_bytes(N, pairs, stages);
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  const bool e4 = h2_epi_warps(pairs) == 4;
  cudaError_t e = e4 ? cudaOccupancyMaxActiveClusters(&n, head_tc2_kernel<4>, &cfg)
                     : cudaOccupancyMaxActiveClusters(&n, head_tc2_kernel<8>, &cfg);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

cudaError_t launch_head_tc2(const HeadArgs& a, const HeadPlan& pl, const HeadTcLaunch& l,
                            const HeadFinal* fin, cudaStream_t s) {
  Head2Params p;
  p.V = a.V;
  p.n_kb = (a.H + H2_BK - 1) / H2_BK;
  p.N = pl.N;
  p.Pcp = pl.pad_pairs;
  p.Pc = pl.pairs_per_chunk;
  p.P = pl.P;
  p.stages = l.stages;
  p.gamma = a.gamma;
  p.pair_slots = pl.slots / 2;
  p.n_ptiles = (a.V + 2 * H2_BM - 1) / (2 * H2_BM);
  p.done_counter = a.done_counter;
  p.B = a.B;
  p.fused = fin != nullptr ? 1 : 0;
  if (fin) p.fin = *fin;
  p.slots = pl.slots;
  p.tmem_cols = h2_tmem_cols(pl.N);
  p.alpha = a.alpha;
  p.drafts = a.drafts;
  p.partials = a.partials;
  p.gathered = a.gathered;
  p.zout = a.zout;
  p.status = a.status;
  p.zonly = pl.zonly ? 1 : 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(pl.slots, pl.n_chunks, 1);
  const int epi = h2_epi_warps(pl.pad_pairs);
  cfg.blockDim = dim3(h2_threads(epi), 1, 1);
  cfg.dynamicSmemBytes = l.smem_bytes;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = 2;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  if (epi == 4) return cudaLaunchKernelEx(&cfg, head_tc2_kernel<4>, l.tm_w, l.tm_h, p);
  return cudaLaunchKernelEx(&cfg, head_tc2_kernel<8>, l.tm_w, l.tm_h, p);
}

}  // namespace rv
