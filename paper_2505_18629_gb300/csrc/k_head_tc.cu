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
// The vocab is split across the CTAs of a chunk in units of `unit_rows` rows
// (a multiple of 16, at most 128).  Full tiles arrive as one 128-row TMA box;
// a partial tile as 16-row boxes (its missing rows are never loaded and their
// accumulator lanes are masked).
//
// Persistent CTA per SM, warp-specialised:
//   warp 0      TMA producer: W tile [128 x 64] + hsel tile [N x 64] per stage
//               into a ring of `stages` 128B-swizzled shared-memory buffers
//   warp 1      allocates TMEM (2 accumulator slots of N columns) and issues
//               tcgen05.mma (M=128, N, K=16) from one thread
//   warps 2..5  epilogue: tcgen05.ld of the finished accumulator slot, fusion,
//               warp-shuffle max/sum/argmax, running statistics in shared memory
// The weight streams from HBM exactly once per step (evict-first); the small
// hidden operand is re-read from L2 per tile (evict-last).
#include <cfloat>

#include "head_epilogue.cuh"
#include "rv_device.cuh"
#include "rv_kernels.h"

namespace rv {

constexpr int HT_BM = HEAD_TILE_ROWS;
constexpr int HT_BK = 64;
constexpr int HT_THREADS = 192;
constexpr int HT_EPI_WARPS = 4;
constexpr int HT_WBOX = HEAD_W_BOX_ROWS;             // vocab rows per TMA box of W
constexpr uint32_t HT_A_BYTES = HT_BM * HT_BK * 2;  // 16 KB
constexpr uint32_t HT_BOX_BYTES = HT_WBOX * HT_BK * 2;  // 2 KB

struct HeadTcParams {
  int V, n_kb, N, Pcp, Pc, P, slots, stages, gamma;
  int unit_rows;  // the vocab is split across CTAs in multiples of this (16..128)
  int units;      // ceil(V / unit_rows)
  uint32_t tmem_cols;
  float alpha;
  const int32_t* drafts;
  float* partials;
  float* gathered;
  unsigned* status;
};

static size_t ht_fixed_bytes() {
  // alignment slack + barriers/misc + drafts + per-warp statistics
  return 1024 + 512 + MAX_PAIRS_PER_CHUNK * 4 +
         HT_EPI_WARPS * MAX_PAIRS_PER_CHUNK * HEAD_STAT_FIELDS * 4;
}

size_t head_tc_smem_bytes(int N, int stages) {
  return ht_fixed_bytes() + static_cast<size_t>(stages) * (HT_A_BYTES + N * 128);
}

int head_tc_max_stages(int N, size_t smem_limit) {
  const size_t per = HT_A_BYTES + N * 128;
  if (smem_limit <= ht_fixed_bytes()) return 0;
  const int s = static_cast<int>((smem_limit - ht_fixed_bytes()) / per);
  return s > 12 ? 12 : s;
}

// Pipeline depth: about 144 KB of tiles in flight per SM streams the weight at
// full HBM bandwidth (measured on GB300: 8 stages of 18 KB beat both 6 and 11).
int head_tc_stages(int N, size_t smem_limit) {
  const int per = static_cast<int>(HT_A_BYTES) + N * 128;
  const int want = (144 * 1024 + per - 1) / per;
  return std::max(2, std::min(head_tc_max_stages(N, smem_limit), std::max(4, want)));
}

// Wait used while draining after an abort: ignores the abort flag.
__device__ __forceinline__ void drain_wait(uint32_t bar, uint32_t parity) {
  const unsigned long long t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (globaltimer_ns() - t0 > RV_WAIT_TIMEOUT_NS / 4) return;
  }
}

__global__ void __launch_bounds__(HT_THREADS, 1)
    head_tc_kernel(const __grid_constant__ CUtensorMap tm_w,
                   const __grid_constant__ CUtensorMap tm_w16,
                   const __grid_constant__ CUtensorMap tm_h, const HeadTcParams p) {
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
  const uint32_t misc = (drain_bar + 8u + 15u) & ~15u;
  uint32_t* const tmem_slot = reinterpret_cast<uint32_t*>(gbase + (misc - base));
  volatile int* const abort_flag = reinterpret_cast<volatile int*>(gbase + (misc - base) + 4);
  int* const s_drafts = reinterpret_cast<int*>(gbase + (misc - base) + 16);
  float* const stats = reinterpret_cast<float*>(gbase + (misc - base) + 16 + MAX_PAIRS_PER_CHUNK * 4);

  const int pair0 = chunk * p.Pc;
  const int npairs = min(p.Pc, p.P - pair0);
  // vocab rows [v_lo, v_hi) of this CTA, in tiles of 128 rows
  const int v_lo = p.unit_rows * static_cast<int>(static_cast<long long>(slot_id) * p.units / p.slots);
  const int v_hi = min(p.V, p.unit_rows * static_cast<int>(static_cast<long long>(slot_id + 1) *
                                                            p.units / p.slots));
  const int t0 = 0;
  const int t1 = v_hi > v_lo ? (v_hi - v_lo + HT_BM - 1) / HT_BM : 0;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    mbar_init(accf0, 1);
    mbar_init(accf0 + 8, 1);
    mbar_init(acce0, HT_EPI_WARPS);
    mbar_init(acce0 + 8, HT_EPI_WARPS);
    mbar_init(drain_bar, 1);
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
    for (int j = e; j < MAX_PAIRS_PER_CHUNK; j += 128)
      s_drafts[j] = (j < npairs) ? pair_draft(p.drafts, pair0 + j, p.gamma) : -1;
    head_stats_init(stats, HT_EPI_WARPS * MAX_PAIRS_PER_CHUNK, e, 128);
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
      int s = 0, issued = 0;
      uint32_t ph = 0;
      bool ok = true;
      for (int t = t0; t < t1 && ok; ++t) {
        const int v0 = v_lo + t * HT_BM;
        const int rows = min(HT_BM, v_hi - v0);
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
      for (int t = t0, lt = 0; t < t1 && ok; ++t, ++lt) {
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
#pragma unroll
          for (int k = 0; k < HT_BK / 16; ++k)
            tc_mma_bf16(d_tmem, ad + 2u * k, bd + 2u * k, idesc, (kb | k) != 0 ? 1u : 0u);
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
    float* const wstats = stats + ew * MAX_PAIRS_PER_CHUNK * HEAD_STAT_FIELDS;
    float* const gathered = p.gathered + static_cast<long long>(pair0) * GATHER_FIELDS;
    for (int t = t0, lt = 0; t < t1; ++t, ++lt) {
      const int slot = lt & 1;
      const uint32_t aph = (lt >> 1) & 1;
      bool ok = mbar_wait(accf0 + 8u * slot, aph, abort_flag, p.status);
      if (!__all_sync(0xffffffffu, ok)) break;
      tc_fence_after();
      const int v = v_lo + t * HT_BM + q * 32 + lane;
      const bool valid = v < v_hi;
      const uint32_t trow =
          tmem_base + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>(slot * p.N);
      for (int g8 = 0; g8 < npairs; g8 += 8) {
        float o[8], r[8];
        tmem_ld8(trow + g8, o);
        tmem_ld8(trow + p.Pcp + g8, r);
        tmem_ld_wait();
        head_tile_pairs8(o, r, g8, npairs, v, valid, p.alpha, s_drafts, wstats, gathered, lane);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(acce0 + 8u * slot);
    }
    named_bar_sync(1, 128);
    head_stats_finish(stats, HT_EPI_WARPS, npairs,
                      p.partials + (static_cast<long long>(slot_id) * p.P + pair0) * HEAD_STAT_FIELDS,
                      threadIdx.x - 64, 128);
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, p.tmem_cols);
  }
}

cudaError_t head_tc_configure(size_t smem_bytes) {
  return cudaFuncSetAttribute(head_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(smem_bytes));
}

static uint32_t tmem_cols_for(int N) {
  uint32_t need = static_cast<uint32_t>(2 * N), c = 32;
  while (c < need) c <<= 1;
  return c;
}

cudaError_t launch_head_tc(const HeadArgs& a, const HeadPlan& pl, const HeadTcLaunch& l,
                           cudaStream_t s) {
  HeadTcParams p;
  p.V = a.V;
  p.n_kb = (a.H + HT_BK - 1) / HT_BK;
  p.N = pl.N;
  p.Pcp = pl.pad_pairs;
  p.Pc = pl.pairs_per_chunk;
  p.P = pl.P;
  p.unit_rows = l.unit_rows;
  p.units = (a.V + l.unit_rows - 1) / l.unit_rows;
  p.slots = pl.slots;
  p.stages = l.stages;
  p.gamma = a.gamma;
  p.tmem_cols = tmem_cols_for(pl.N);
  p.alpha = a.alpha;
  p.drafts = a.drafts;
  p.partials = a.partials;
  p.gathered = a.gathered;
  p.status = a.status;
  dim3 grid(pl.slots, pl.n_chunks);
  head_tc_kernel<<<grid, HT_THREADS, l.smem_bytes, s>>>(l.tm_w, l.tm_w16, l.tm_h, p);
  return cudaGetLastError();
}

}  // namespace rv
