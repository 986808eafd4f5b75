// Verify-block attention (Sec. 3.1) on the 5th-generation tensor cores, for
// head_dim 128 (bf16): every query row of the packed block attends causally to
// the cached context and to the block positions up to its own.
//
// Work items.  The Lb*G query rows that share a KV head (G = Hq / Hkv) form one
// MMA tile of M = 128 rows (row groups of 128 when there are more).  The keys
// of a sequence are cut into chunks of `chunk` cached keys; the block's own
// keys belong to the last chunk.  An item is (sequence, KV head, row group,
// chunk); persistent CTAs (at most one per SM) claim items from a counter, so
// sequences of different lengths balance across the SMs.  An item that covers
// the whole sequence writes its rows directly; otherwise it writes its
// normalised partial O (bf16) with (max, sum), and a second small kernel
// merges the chunks (one thread per row).
//
// Per CTA, warp-specialised:
//   warp 0     claims items and loads with TMA the item's 128 query rows
//              (3-D box over q [B*Lb][Hq][D]) into a shared-memory buffer,
//              then, per tile of 128 keys, the K and V tiles from the cache
//              ([B*Hkv*Cmax][D]) or, for the block's keys, from k_blk / v_blk
//              (3-D box over [B*Lb][Hkv][D]) into a ring of stages.  Items are
//              claimed full key chunks first and the sequences' last chunks
//              (shorter, with the block's keys) after them, so that the small
//              items fill the end of the launch
//   warp 1     allocates TMEM and issues the MMAs from one thread:
//                S_t  = Q K_t^T   (M 128, N 128, K 128) into S[t % 2]; Q is
//                                 read from TMEM
//                O   += P_t V_t   (M 128, N 128, K 128); P_t (bf16) is read from
//                                 TMEM, where the softmax wrote it over the
//                                 first half of S[t % 2]; V is used as stored,
//                                 an MN-major operand
//              QK of tile t+1 is issued before PV of tile t, so the tensor core
//              computes the next scores while the softmax runs; the MMAs of a
//              CTA execute in issue order, so QK of tile t+2 overwrites S[t % 2]
//              only after PV of tile t has read P_t
//   warps 2-5  one thread per query row (its TMEM lane): copies its Q row from
//              the shared-memory buffer into TMEM (which frees the buffer for
//              the next item's rows), runs the online softmax of S_t (base-2, the 1/sqrt(D)
//              scale folded into the exponent), rescales its O row lazily
//              (only when its max rises by more than 2^8), and at the end of
//              the item stores the O row (output or partial).  The next item's
//              Q is written before this item's O is read out, so the tensor
//              core starts the next item meanwhile.
// Every wait is bounded (a timeout is reported in the status word).  The CTA
// that handles the last chunk of (sequence, KV head) in row group 0 appends
// the block's keys and values to the cache.
#include <cfloat>

#include "rv_device.cuh"
#include "rv_kernels.h"

namespace rv {

namespace {

constexpr int TC_D = 128;
constexpr int TC_M = 128;        // query rows per MMA tile
constexpr int TC_KT = 128;       // keys per tile
constexpr int TC_STAGES = 3;     // K/V ring depth
constexpr int TC_THREADS = 192;  // producer, MMA, 4 softmax warps
constexpr int TC_IRING = 4;      // item ring between the producer and the consumers
constexpr float TC_RESCALE_LOG2 = 8.f;
// Key chunks are sized for about this many items per SM at capacity; the
// partial-result slots of the workspace (attn_tc_max_slots) are sized from the
// same number, so the two cannot disagree.
constexpr int TC_ITEMS_PER_SM = 4;

constexpr uint32_t TC_KV_BYTES = TC_KT * TC_D * 2;  // 32 KB: two halves of [128 keys][128 B]
constexpr uint32_t TC_Q_BYTES = TC_M * TC_D * 2;    // 32 KB: two halves of [128 rows][128 B]
constexpr uint32_t TC_K_OFF = 0;
constexpr uint32_t TC_V_OFF = TC_K_OFF + TC_STAGES * TC_KV_BYTES;
constexpr uint32_t TC_QS_OFF = TC_V_OFF + TC_STAGES * TC_KV_BYTES;  // staged query rows
constexpr uint32_t TC_BAR_OFF = TC_QS_OFF + TC_Q_BYTES;
constexpr uint32_t TC_MISC_OFF = TC_BAR_OFF + 256;
constexpr uint32_t TC_RING_OFF = TC_MISC_OFF + 16;  // TC_IRING items of 8 ints
constexpr uint32_t TC_SCAN_OFF = TC_RING_OFF + TC_IRING * 32;
// TMEM columns: S[0] [0, 128), S[1] [128, 256) (P_t over the first 64 columns
// of S[t % 2], two bf16 per column), O [256, 384), Q [384, 448) (bf16 pairs)
constexpr uint32_t TC_TMEM_COLS = 512;
constexpr uint32_t TC_O_COL = 256;
constexpr uint32_t TC_Q_COL = 384;

struct TcArgs {
  const __nv_bfloat16* q;
  const int32_t* ctx;
  __nv_bfloat16* k_cache;
  __nv_bfloat16* v_cache;
  const __nv_bfloat16* k_blk;
  const __nv_bfloat16* v_blk;
  __nv_bfloat16* out;
  // normalised partial O, chunk-major: [slot][32 chunks of 4 dims][128 rows] x 16 B,
  // so that a warp's 32 rows store one chunk as 512 contiguous bytes
  float* part_o;
  float* part_ml;      // [slot][128][2]   (max in log2 units, sum)
  unsigned* counters;  // [0] item counter, [1] CTAs finished
  unsigned* status;
  int B, Lb, Hq, Hkv, G, Cmax, rows, n_rg, chunk, max_chunks;
  float scale_log2;
  int kv_evict_first;
};

struct Item {
  int b, kvh, rg, c;  // b < 0: no more items
  int ctx;            // -1: context length out of range (no tiles)
  int kc_lo, kc_hi;   // cached keys of this chunk
  int nch;            // chunks of the sequence
};

__device__ __forceinline__ int item_cache_tiles(const Item& it) {
  return it.kc_hi > it.kc_lo ? (it.kc_hi - it.kc_lo + TC_KT - 1) / TC_KT : 0;
}
__device__ __forceinline__ int item_tiles(const Item& it, int Lb) {
  if (it.b < 0 || it.ctx < 0) return 0;
  return item_cache_tiles(it) + (it.c == it.nch - 1 ? (Lb + TC_KT - 1) / TC_KT : 0);
}

// Chunks of a sequence (an invalid context length still gets one, empty, item).
__device__ __forceinline__ int seq_chunks(int ctx, int Lb, int Cmax, int chunk) {
  if (ctx < 0 || ctx + Lb > Cmax) return 1;
  return ctx > 0 ? (ctx + chunk - 1) / chunk : 1;
}

}  // namespace

__global__ void __launch_bounds__(TC_THREADS, 1)
    attention_tc_kernel(const __grid_constant__ CUtensorMap tm_kc,
                        const __grid_constant__ CUtensorMap tm_vc,
                        const __grid_constant__ CUtensorMap tm_kb,
                        const __grid_constant__ CUtensorMap tm_vb,
                        const __grid_constant__ CUtensorMap tm_q, const TcArgs a) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* const smem = smem_raw + (base - raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  const uint32_t bars = base + TC_BAR_OFF;
  const uint32_t q_full = bars;  // Q of the next item is in TMEM (4 softmax warps)
  auto kv_full = [&](int i) { return bars + 32u + 8u * i; };  // TC_STAGES each
  auto kv_empty = [&](int i) { return bars + 32u + 8u * (TC_STAGES + i); };
  const uint32_t b2 = bars + 32u + 16u * TC_STAGES;
  auto s_full = [&](int i) { return b2 + 8u * i; };  // 2 each
  auto p_full = [&](int i) { return b2 + 16u + 8u * i; };
  auto o_done = [&](int i) { return b2 + 32u + 8u * i; };
  const uint32_t o_free = b2 + 48u;
  const uint32_t drain_bar = b2 + 56u;
  auto r_full = [&](int i) { return b2 + 64u + 8u * i; };  // TC_IRING each
  auto r_empty = [&](int i) { return b2 + 64u + 8u * (TC_IRING + i); };
  const uint32_t qs_full = b2 + 64u + 16u * TC_IRING;  // an item's rows are staged (TMA)
  const uint32_t qs_empty = qs_full + 8u;              // the softmax warps copied them to TMEM
  static_assert(32 + 16 * TC_STAGES + 64 + 16 * TC_IRING + 16 <= 256, "barrier block");
  uint32_t* const tmem_slot = reinterpret_cast<uint32_t*>(smem + TC_MISC_OFF);
  volatile int* const abort_flag = reinterpret_cast<volatile int*>(smem + TC_MISC_OFF + 4);
  Item* const ring = reinterpret_cast<Item*>(smem + TC_RING_OFF);
  int* const scan = reinterpret_cast<int*>(smem + TC_SCAN_OFF);  // [B + 1] first item of b
  int* const order = scan + a.B + 1;  // [B] sequences by the size of their last chunk, largest first

  if (threadIdx.x == 0) {
    mbar_init(q_full, 4);
    for (int i = 0; i < 2; ++i) {
      mbar_init(s_full(i), 1);
      mbar_init(p_full(i), 4);
      mbar_init(o_done(i), 1);
    }
    for (int i = 0; i < TC_STAGES; ++i) {
      mbar_init(kv_full(i), 1);
      mbar_init(kv_empty(i), 1);
    }
    mbar_init(o_free, 4);
    mbar_init(drain_bar, 1);
    mbar_init(qs_full, 1);
    mbar_init(qs_empty, 4);
    for (int i = 0; i < TC_IRING; ++i) {
      mbar_init(r_full(i), 1);
      mbar_init(r_empty(i), 5);  // the MMA thread + one lane per softmax warp
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0) {
    // Items: first the full chunks (all chunks but the last) of every sequence,
    // numbered sequence by sequence (scan[b] = the first of sequence b), then
    // the last chunk of every (sequence, KV head, row group), the sequences in
    // decreasing order of that chunk's tiles (ties: lower b first), so that
    // the smallest items end the launch.
    const int per_seq = a.Hkv * a.n_rg;
    int carry = 0;
    for (int b0 = 0; b0 < a.B; b0 += 32) {
      const int b = b0 + lane;
      const int n = b < a.B ? per_seq * (seq_chunks(a.ctx[b], a.Lb, a.Cmax, a.chunk) - 1) : 0;
      int incl = n;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
      }
      if (b < a.B) scan[b] = carry + incl - n;
      carry += __shfl_sync(0xffffffffu, incl, 31);
    }
    auto last_tiles = [&](int b) {
      const int ctx = a.ctx[b];
      if (ctx < 0 || ctx + a.Lb > a.Cmax) return 0;
      const int nch = seq_chunks(ctx, a.Lb, a.Cmax, a.chunk);
      const int kc = ctx - min(ctx, (nch - 1) * a.chunk);
      return (kc + TC_KT - 1) / TC_KT + (a.Lb + TC_KT - 1) / TC_KT;
    };
    for (int b = lane; b < a.B; b += 32) {
      const int tb = last_tiles(b);
      int rank = 0;
      for (int o = 0; o < a.B; ++o) {
        const int to = last_tiles(o);
        rank += (to > tb || (to == tb && o < b)) ? 1 : 0;
      }
      order[rank] = b;
    }
    if (lane == 0) {
      scan[a.B] = carry;
      tma_prefetch_desc(&tm_q);
      tma_prefetch_desc(&tm_kc);
      tma_prefetch_desc(&tm_vc);
      tma_prefetch_desc(&tm_kb);
      tma_prefetch_desc(&tm_vb);
    }
  }
  if (warp == 1) tmem_alloc(smem_u32(tmem_slot), TC_TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // the merge launch that follows may start (it waits for this grid's results)
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const uint64_t pol_blk = policy_evict_last();
      const uint64_t pol_kv = a.kv_evict_first ? policy_evict_first() : policy_evict_normal();
      const int per_seq = a.Hkv * a.n_rg;
      const int n_full = scan[a.B];
      const int total = n_full + a.B * per_seq;
      int u = 0, nq = 0;
      bool ok = true;
      for (int lt = 0; ok; ++lt) {
        const int i = static_cast<int>(atomicAdd(&a.counters[0], 1u));
        Item item;
        item.b = -1;
        item.kvh = item.rg = item.c = item.ctx = item.kc_lo = item.kc_hi = 0;
        item.nch = 1;
        if (i < total) {
          int b, rem, c_last = 0;
          if (i < n_full) {
            int lo = 0, hi = a.B - 1;  // the last b with scan[b] <= i
            while (lo < hi) {
              const int mid = (lo + hi + 1) >> 1;
              if (scan[mid] <= i)
                lo = mid;
              else
                hi = mid - 1;
            }
            b = lo;
            rem = i - scan[b];
          } else {
            b = order[(i - n_full) / per_seq];
            rem = (i - n_full) % per_seq;
            c_last = 1;
          }
          const int ctx = a.ctx[b];
          const int nch = seq_chunks(ctx, a.Lb, a.Cmax, a.chunk);
          item.b = b;
          item.rg = rem % a.n_rg;
          rem /= a.n_rg;
          if (c_last) {
            item.c = nch - 1;
            item.kvh = rem;
          } else {
            item.c = rem % (nch - 1);
            item.kvh = rem / (nch - 1);
          }
          item.nch = nch;
          const bool valid = ctx >= 0 && ctx + a.Lb <= a.Cmax;
          item.ctx = valid ? ctx : -1;
          if (!valid && item.kvh == 0 && item.rg == 0) raise_status(a.status, RV_DEV_CTX_RANGE);
          item.kc_lo = valid ? min(ctx, item.c * a.chunk) : 0;
          item.kc_hi = valid ? min(ctx, item.kc_lo + a.chunk) : 0;
        }
        const int k = lt % TC_IRING;
        if (!mbar_wait(r_empty(k), ((lt / TC_IRING) & 1) ^ 1u, abort_flag, a.status)) {
          ok = false;
          break;
        }
        ring[k] = item;
        mbar_arrive(r_full(k));
        if (item.b < 0) break;
        const int n = item_tiles(item, a.Lb);
        if (n == 0) continue;
        // the item's query rows: (j, g) for j from rg * 128 / G, one box per 64 dims
        if (!mbar_wait(qs_empty, (nq & 1) ^ 1u, abort_flag, a.status)) {
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(qs_full, TC_Q_BYTES);
        {
          const int z = item.b * a.Lb + item.rg * (TC_M / a.G);
          tma_load_3d(base + TC_QS_OFF, &tm_q, 0, item.kvh * a.G, z, qs_full, pol_blk);
          tma_load_3d(base + TC_QS_OFF + TC_Q_BYTES / 2, &tm_q, 64, item.kvh * a.G, z, qs_full,
                      pol_blk);
        }
        ++nq;
        const int n_cache = item_cache_tiles(item);
        const int row_c = (item.b * a.Hkv + item.kvh) * a.Cmax;
        for (int j = 0; j < n; ++j) {
          const int st = u % TC_STAGES;
          if (!mbar_wait(kv_empty(st), ((u / TC_STAGES) & 1) ^ 1u, abort_flag, a.status)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(kv_full(st), 2 * TC_KV_BYTES);
          const uint32_t kd = base + TC_K_OFF + st * TC_KV_BYTES;
          const uint32_t vd = base + TC_V_OFF + st * TC_KV_BYTES;
          if (j < n_cache) {
            const int y = row_c + item.kc_lo + j * TC_KT;
            tma_load_2d(kd, &tm_kc, 0, y, kv_full(st), pol_kv);
            tma_load_2d(kd + TC_KV_BYTES / 2, &tm_kc, 64, y, kv_full(st), pol_kv);
            tma_load_2d(vd, &tm_vc, 0, y, kv_full(st), pol_kv);
            tma_load_2d(vd + TC_KV_BYTES / 2, &tm_vc, 64, y, kv_full(st), pol_kv);
          } else {
            const int z = item.b * a.Lb + (j - n_cache) * TC_KT;
            tma_load_3d(kd, &tm_kb, 0, item.kvh, z, kv_full(st), pol_blk);
            tma_load_3d(kd + TC_KV_BYTES / 2, &tm_kb, 64, item.kvh, z, kv_full(st), pol_blk);
            tma_load_3d(vd, &tm_vb, 0, item.kvh, z, kv_full(st), pol_blk);
            tma_load_3d(vd + TC_KV_BYTES / 2, &tm_vb, 64, item.kvh, z, kv_full(st), pol_blk);
          }
          ++u;
        }
      }
      if (!ok) {  // let the copies still in flight land before the CTA exits
        for (int v = max(0, u - TC_STAGES); v < u; ++v)
          drain_wait(kv_full(v % TC_STAGES), static_cast<uint32_t>((v / TC_STAGES) & 1));
        if (nq > 0) drain_wait(qs_full, static_cast<uint32_t>((nq - 1) & 1));
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc_s = idesc_bf16_f32(TC_M, TC_KT);
      const uint32_t idesc_o = idesc_bf16_f32_bmn(TC_M, TC_D);
      int u = 0, it = 0;
      bool ok = true;
      // O += P_v V_v for tile v; the first tile of an item overwrites O, once
      // the softmax warps have read the previous item's O
      auto issue_pv = [&](int v, bool first) -> bool {
        const int pb = v & 1;
        if (!mbar_wait(p_full(pb), (v >> 1) & 1, abort_flag, a.status)) return false;
        if (first && it > 0 && !mbar_wait(o_free, (it - 1) & 1, abort_flag, a.status)) return false;
        tc_fence_after();
        const uint32_t pcol = tmem + static_cast<uint32_t>(pb * TC_KT);
        const uint32_t vb = base + TC_V_OFF + (v % TC_STAGES) * TC_KV_BYTES;
        // K-slice kk of V (16 keys x 128 B rows) starts 16 * 128 bytes after slice kk - 1
        static_assert(TC_KT == 128, "eight K-slices of 16 keys per tile");
        tc_mma_stage8_tmem_a_mn(tmem + TC_O_COL, pcol,
                                sw128_mnmajor_desc(vb, TC_KV_BYTES / 2, 1024), (16 * 128) >> 4,
                                idesc_o, first ? 0u : 1u);
        tc_commit(o_done(pb));
        tc_commit(kv_empty(v % TC_STAGES));
        return true;
      };
      for (int lt = 0; ok; ++lt) {
        const int k = lt % TC_IRING;
        if (!mbar_wait(r_full(k), (lt / TC_IRING) & 1, abort_flag, a.status)) break;
        const Item item = ring[k];
        mbar_arrive(r_empty(k));
        if (item.b < 0) break;
        const int n = item_tiles(item, a.Lb);
        if (n == 0) continue;
        if (!mbar_wait(q_full, it & 1, abort_flag, a.status)) break;
        tc_fence_after();
        for (int j = 0; j < n && ok; ++j) {
          const int v = u + j;
          const int st = v % TC_STAGES;
          if (!mbar_wait(kv_full(st), (v / TC_STAGES) & 1, abort_flag, a.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t kb = base + TC_K_OFF + st * TC_KV_BYTES;
          static_assert(TC_D == 128, "eight K-slices of 16 head dims");
          tc_mma_stage8_tmem_a(tmem + static_cast<uint32_t>((v & 1) * TC_KT), tmem + TC_Q_COL,
                               sw128_kmajor_desc(kb), (TC_KV_BYTES / 2) >> 4, idesc_s, 0u);
          tc_commit(s_full(v & 1));
          if (j > 0 && !issue_pv(v - 1, j == 1)) ok = false;
        }
        if (ok && !issue_pv(u + n - 1, n == 1)) ok = false;
        u += n;
        ++it;
      }
      // every MMA issued must be complete before TMEM is released
      tc_commit(drain_bar);
      drain_wait(drain_bar, 0);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ softmax warps
    const int q = warp & 3;       // TMEM lane quadrant
    const int r = q * 32 + lane;  // query row within the row group (TMEM lane)
    const int st_tid = threadIdx.x - 64;
    const uint32_t t_row = tmem + (static_cast<uint32_t>(q * 32) << 16);
    int lt = 0;
    bool live = true;
    // next ring entry with tiles (or the end); every entry is acknowledged
    auto next_item = [&](Item& it) -> bool {
      for (;;) {
        const int k = lt % TC_IRING;
        const bool ok = mbar_wait(r_full(k), (lt / TC_IRING) & 1, abort_flag, a.status);
        if (!__all_sync(0xffffffffu, ok)) return false;
        it = ring[k];
        __syncwarp();
        if (lane == 0) mbar_arrive(r_empty(k));
        ++lt;
        if (it.b < 0 || item_tiles(it, a.Lb) > 0) return true;
      }
    };
    // this row of the item's Q: the staged rows (TMA, 128-byte swizzle: chunk c
    // of row r at c ^ (r & 7)) -> registers -> TMEM; the buffer is released as
    // soon as every row has been read.  Rows past the item's (another
    // sequence's, or zeros) are read too; their scores are masked.
    uint4 qv[16];
    int nq = 0;
    auto q_fetch = [&](const Item& it) -> bool {
      (void)it;
      const bool w = mbar_wait(qs_full, nq & 1, abort_flag, a.status);
      if (!__all_sync(0xffffffffu, w)) return false;
      ++nq;
#pragma unroll
      for (int c = 0; c < 16; ++c)
        qv[c] = *reinterpret_cast<const uint4*>(smem + TC_QS_OFF + (c >> 3) * (TC_Q_BYTES / 2) +
                                                r * 128 + (((c & 7) ^ (r & 7)) << 4));
      __syncwarp();
      if (lane == 0) mbar_arrive(qs_empty);
      return true;
    };
    auto q_store = [&]() {
#pragma unroll
      for (int h = 0; h < 4; ++h) {
        uint32_t w[16];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          w[4 * c] = qv[4 * h + c].x;
          w[4 * c + 1] = qv[4 * h + c].y;
          w[4 * c + 2] = qv[4 * h + c].z;
          w[4 * c + 3] = qv[4 * h + c].w;
        }
        tmem_st16(t_row + TC_Q_COL + 16 * h, w);
      }
      tmem_st_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(q_full);
    };

    Item item;
    live = next_item(item);
    if (live && item.b >= 0) {
      live = q_fetch(item);
      if (live) q_store();
    }
    int u = 0;
    while (live && item.b >= 0) {
      const int n = item_tiles(item, a.Lb);
      const int n_cache = item_cache_tiles(item);
      const int ctx = item.ctx;
      const int gr = item.rg * TC_M + r;  // row among the Lb*G rows of (sequence, KV head)
      const bool rvalid = gr < a.rows;
      const int lim = rvalid ? ctx + gr / a.G : -1;  // last key this row may see

      // append the block's keys/values to the cache, once per (sequence, KV head)
      if (item.c == item.nch - 1 && item.rg == 0) {
        for (int e = st_tid; e < a.Lb * 16; e += 128) {
          const int j = e >> 4, c16 = e & 15;
          const long long src =
              ((static_cast<long long>(item.b) * a.Lb + j) * a.Hkv + item.kvh) * TC_D + c16 * 8;
          const long long dst =
              ((static_cast<long long>(item.b) * a.Hkv + item.kvh) * a.Cmax + ctx + j) * TC_D +
              c16 * 8;
          *reinterpret_cast<uint4*>(a.k_cache + dst) = *reinterpret_cast<const uint4*>(a.k_blk + src);
          *reinterpret_cast<uint4*>(a.v_cache + dst) = *reinterpret_cast<const uint4*>(a.v_blk + src);
        }
      }

      float m_used = NEG_INF, l = 0.f;  // running max (log2 units) and sum of this row
      for (int j = 0; j < n && live; ++j) {
        const int v = u + j;
        const int sb = v & 1;
        const uint32_t s_col = t_row + static_cast<uint32_t>(sb * TC_KT);
        bool ok = mbar_wait(s_full(sb), (v >> 1) & 1, abort_flag, a.status);
        if (!__all_sync(0xffffffffu, ok)) {
          live = false;
          break;
        }
        tc_fence_after();
        float sv[4][32];
#pragma unroll
        for (int c = 0; c < 4; ++c) tmem_ld32(s_col + 32 * c, sv[c]);
        tmem_ld_wait();
        int kb, kend;
        if (j < n_cache) {
          kb = item.kc_lo + j * TC_KT;
          kend = item.kc_hi;
        } else {
          kb = ctx + (j - n_cache) * TC_KT;
          kend = ctx + a.Lb;
        }
        const int kmax = min(kend - 1, lim);  // last key of the tile this row sees
        if (kb + TC_KT - 1 > kmax) {          // a partial tile for this row: mask
#pragma unroll
          for (int c = 0; c < 4; ++c)
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if (kb + 32 * c + i > kmax) sv[c][i] = NEG_INF;
        }
        // row max: eight chains of three-input maxima (16 scores each)
        float mx[8];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            float m = fmaxf(sv[c][e], sv[c][e + 2]);
#pragma unroll
            for (int i = e + 4; i < 32; i += 4) m = max3f(m, sv[c][i], sv[c][i + 2]);
            mx[2 * c + e] = m;
          }
        }
        const float mt = max3f(max3f(mx[0], mx[1], mx[2]), max3f(mx[3], mx[4], mx[5]),
                               fmaxf(mx[6], mx[7])) *
                         a.scale_log2;
        float fac = 1.f;
        const bool rise = mt > m_used + TC_RESCALE_LOG2 || (m_used == NEG_INF && mt != NEG_INF);
        if (rise) {
          fac = (m_used == NEG_INF) ? 0.f : exp2f(m_used - mt);
          m_used = mt;
        }
        // O holds this item's earlier tiles: rescale this warp's rows if any rose
        if (j > 0 && __any_sync(0xffffffffu, rise && fac != 1.f)) {
          ok = mbar_wait(o_done((v - 1) & 1), ((v - 1) >> 1) & 1, abort_flag, a.status);
          if (!__all_sync(0xffffffffu, ok)) {
            live = false;
            break;
          }
          tc_fence_after();
#pragma unroll
          for (int c = 0; c < TC_D; c += 32) {
            float ov[32];
            tmem_ld32(t_row + TC_O_COL + c, ov);
            tmem_ld_wait();
#pragma unroll
            for (int i = 0; i < 32; ++i) ov[i] *= fac;
            tmem_st32(t_row + TC_O_COL + c, ov);
          }
          tmem_st_wait();
        }
        // P = 2^(s * scale - m), bf16, over the first half of S[sb]; the
        // exponent arguments and the row sum two scores per instruction
        const float neg_m = (m_used == NEG_INF) ? 0.f : -m_used;
        const uint64_t sc2 = f32x2(a.scale_log2, a.scale_log2), nm2 = f32x2(neg_m, neg_m);
        uint64_t ls2[2] = {f32x2(0.f, 0.f), f32x2(0.f, 0.f)};
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          uint32_t pk[16];
#pragma unroll
          for (int i = 0; i < 32; i += 2) {
            float x0, x1;
            f32x2_split(fma_f32x2(f32x2(sv[c][i], sv[c][i + 1]), sc2, nm2), x0, x1);
            const float p0 = ex2_approx(x0);
            const float p1 = ex2_approx(x1);
            ls2[c & 1] = add_f32x2(ls2[c & 1], f32x2(p0, p1));
            pk[i >> 1] = pack_bf16(p0, p1);
          }
          tmem_st16(s_col + 16 * c, pk);
        }
        float ls[4];
        f32x2_split(ls2[0], ls[0], ls[1]);
        f32x2_split(ls2[1], ls[2], ls[3]);
        l = l * fac + ((ls[0] + ls[1]) + (ls[2] + ls[3]));
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(p_full(sb));
      }
      if (!live) break;

      // ---- the next item's Q goes to TMEM first (every QK of this item is
      // complete), so its first scores are computed during this item's end
      Item nxt;
      live = next_item(nxt);
      if (!live) break;
      if (nxt.b >= 0) {
        live = q_fetch(nxt);
        if (!live) break;
        q_store();
      }

      // ---- item end: this row's O
      const int vl = u + n - 1;
      bool ok = mbar_wait(o_done(vl & 1), (vl >> 1) & 1, abort_flag, a.status);
      if (!__all_sync(0xffffffffu, ok)) break;
      tc_fence_after();
      u += n;
      float ov[4][32];
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld32(t_row + TC_O_COL + 32 * c, ov[c]);
      tmem_ld_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(o_free);
      const float inv = (l > 0.f) ? 1.f / l : 0.f;
      const int group = (item.b * a.Hkv + item.kvh) * a.n_rg + item.rg;
      const int slot = group * a.max_chunks + item.c;
      if (rvalid) {
        if (item.nch == 1) {
          const long long orow = (static_cast<long long>(item.b) * a.Lb + gr / a.G) * a.Hq +
                                 item.kvh * a.G + gr % a.G;
          __nv_bfloat16* dst = a.out + orow * TC_D;
#pragma unroll
          for (int c = 0; c < 4; ++c)
#pragma unroll
            for (int i = 0; i < 32; i += 8) {
              uint4 pk;
              pk.x = pack_bf16(ov[c][i] * inv, ov[c][i + 1] * inv);
              pk.y = pack_bf16(ov[c][i + 2] * inv, ov[c][i + 3] * inv);
              pk.z = pack_bf16(ov[c][i + 4] * inv, ov[c][i + 5] * inv);
              pk.w = pack_bf16(ov[c][i + 6] * inv, ov[c][i + 7] * inv);
              *reinterpret_cast<uint4*>(dst + 32 * c + i) = pk;
            }
        } else {
          float4* const po =
              reinterpret_cast<float4*>(a.part_o) + static_cast<long long>(slot) * 32 * TC_M + r;
#pragma unroll
          for (int c = 0; c < 32; ++c) {
            const float* v = &ov[c >> 3][(c & 7) * 4];
            __stcg(po + c * TC_M, make_float4(v[0] * inv, v[1] * inv, v[2] * inv, v[3] * inv));
          }
          __stcg(reinterpret_cast<float2*>(a.part_ml) + static_cast<long long>(slot) * TC_M + r,
                 make_float2(m_used, l));
        }
      }
      item = nxt;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, TC_TMEM_COLS);
  }
  // the last CTA to finish re-arms the item counter for the next launch
  if (threadIdx.x == 0) {
    __threadfence();
    if (atomicAdd(&a.counters[1], 1u) == gridDim.x - 1) {
      a.counters[0] = 0u;
      a.counters[1] = 0u;
      __threadfence();
    }
  }
}

// Merge of the chunks of each (sequence, KV head, row group) whose sequence
// needed several: one CTA per (group, 8 dims), one thread per query row, so
// that the CTA's threads read consecutive rows of the chunk-major partials.
// out = sum_c w_c O_c / sum_c w_c with w_c = l_c 2^(m_c - max_c m_c).
struct MergeArgs {
  const int32_t* ctx;
  const float* part_o;
  const float* part_ml;
  __nv_bfloat16* out;
  int Lb, Hq, Hkv, G, Cmax, rows, n_rg, chunk, max_chunks;
};

__global__ void __launch_bounds__(TC_M) attention_merge_kernel(const MergeArgs a) {
  asm volatile("griddepcontrol.wait;" ::: "memory");  // the attention grid's results
  const int group = blockIdx.x;
  const int rg = group % a.n_rg, t = group / a.n_rg;
  const int kvh = t % a.Hkv, b = t / a.Hkv;
  const int rr = threadIdx.x;  // row within the row group
  const int gr = rg * TC_M + rr;
  if (gr >= a.rows) return;
  const int ctx = a.ctx[b];
  if (ctx < 0 || ctx + a.Lb > a.Cmax) return;
  const int nch = seq_chunks(ctx, a.Lb, a.Cmax, a.chunk);
  if (nch == 1) return;
  const long long slot0 = static_cast<long long>(group) * a.max_chunks;
  const float2* ml = reinterpret_cast<const float2*>(a.part_ml);
  float M = NEG_INF;
  for (int c = 0; c < nch; ++c) {
    const float2 v = __ldcg(ml + (slot0 + c) * TC_M + rr);
    if (v.y > 0.f) M = fmaxf(M, v.x);
  }
  float den = 0.f;
  for (int c = 0; c < nch; ++c) {
    const float2 v = __ldcg(ml + (slot0 + c) * TC_M + rr);
    den += v.y > 0.f ? v.y * exp2f(v.x - M) : 0.f;
  }
  const float id = den > 0.f ? 1.f / den : 0.f;
  const long long orow =
      (static_cast<long long>(b) * a.Lb + gr / a.G) * a.Hq + kvh * a.G + gr % a.G;
  const float4* part = reinterpret_cast<const float4*>(a.part_o);
  {
    const int ch = blockIdx.y;  // 8 dims: chunks 2 ch and 2 ch + 1
    float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    for (int c = 0; c < nch; ++c) {
      const float2 v = __ldcg(ml + (slot0 + c) * TC_M + rr);
      const float w = v.y > 0.f ? v.y * exp2f(v.x - M) * id : 0.f;
      const float4 lo = __ldcg(part + ((slot0 + c) * 32 + 2 * ch) * TC_M + rr);
      const float4 hi = __ldcg(part + ((slot0 + c) * 32 + 2 * ch + 1) * TC_M + rr);
      acc[0] = fmaf(w, lo.x, acc[0]);
      acc[1] = fmaf(w, lo.y, acc[1]);
      acc[2] = fmaf(w, lo.z, acc[2]);
      acc[3] = fmaf(w, lo.w, acc[3]);
      acc[4] = fmaf(w, hi.x, acc[4]);
      acc[5] = fmaf(w, hi.y, acc[5]);
      acc[6] = fmaf(w, hi.z, acc[6]);
      acc[7] = fmaf(w, hi.w, acc[7]);
    }
    uint4 o;
    o.x = pack_bf16(acc[0], acc[1]);
    o.y = pack_bf16(acc[2], acc[3]);
    o.z = pack_bf16(acc[4], acc[5]);
    o.w = pack_bf16(acc[6], acc[7]);
    *reinterpret_cast<uint4*>(a.out + orow * TC_D + ch * 8) = o;
  }
}

// ---------------------------------------------------------------- planning / launch

AttnTcPlan attn_tc_plan(int B, int Lb, int Hq, int Hkv, int Cmax, int num_sms) {
  AttnTcPlan p;
  const int G = Hq / Hkv;
  p.rows = Lb * G;
  p.n_rg = (p.rows + TC_M - 1) / TC_M;
  const long long groups = static_cast<long long>(B) * Hkv * p.n_rg;
  // chunks sized for about four items per SM when every sequence is full.
  // Fewer, longer items run faster alone where there are many groups and
  // short caches (70B B=32: 160.8 us at two items per SM against 167.8 us), but
  // in the step, where the attention takes SMs as the LM head's CTAs finish,
  // the finer items balance the late-starting CTAs (70B B=32 step 805-815 us
  // at four against 870 us at two).
  const long long per_sm = static_cast<long long>(TC_ITEMS_PER_SM) * num_sms;
  long long ch = (groups * Cmax + per_sm - 1) / per_sm;
  ch = std::max<long long>(256, (ch + TC_KT - 1) / TC_KT * TC_KT);
  ch = std::min<long long>(ch, (Cmax + TC_KT - 1) / TC_KT * TC_KT + TC_KT);
  p.chunk = static_cast<int>(ch);
  p.max_chunks = std::max(1, (Cmax + p.chunk - 1) / p.chunk);
  p.slots = static_cast<int>(groups) * p.max_chunks;
  p.grid = static_cast<int>(std::min<long long>(num_sms, p.slots));
  // scan [B + 1], order [B] (+ 1024 for alignment)
  p.smem_bytes = TC_SCAN_OFF + static_cast<size_t>(2 * B + 1) * 4 + 1024;
  return p;
}

bool attn_tc_supported(int Hq, int Hkv, int D) {
  return D == TC_D && Hkv > 0 && Hq % Hkv == 0 && TC_M % (Hq / Hkv) == 0;
}

size_t attn_tc_smem_max(int max_batch) {
  return TC_SCAN_OFF + static_cast<size_t>(2 * max_batch + 1) * 4 + 1024;
}

int attn_tc_max_slots(int max_batch, int Lb_max, int Hq, int Hkv, int num_sms) {
  // chunk >= groups * Cmax / (TC_ITEMS_PER_SM * SMs), or one chunk per group:
  // slots <= TC_ITEMS_PER_SM * SMs + groups
  const int n_rg = (Lb_max * (Hq / Hkv) + TC_M - 1) / TC_M;
  return TC_ITEMS_PER_SM * num_sms + max_batch * Hkv * n_rg;
}

cudaError_t attn_tc_configure(size_t smem_bytes) {
  cudaError_t e = cudaFuncSetAttribute(attention_tc_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem_bytes));
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(attention_tc_kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                             cudaSharedmemCarveoutMaxShared);
  return e;
}

namespace {
bool encode(PFN_cuTensorMapEncodeTiled_v12000 enc, CUtensorMap* m, const void* ptr,
            cuuint32_t rank, const cuuint64_t* dims, const cuuint64_t* strides,
            const cuuint32_t* box) {
  const cuuint32_t es[3] = {1, 1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, const_cast<void*>(ptr), dims, strides, box,
             es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}
}  // namespace

// The block K/V as 3-D [B*Lb][Hkv][D], the caches as 2-D [B*Hkv*Cmax][D];
// boxes of 64 dims x 128 keys, 128-byte swizzled.
bool attn_tc_encode(PFN_cuTensorMapEncodeTiled_v12000 enc, const AttnArgs& x, AttnTcMaps* m) {
  const cuuint64_t rs = static_cast<cuuint64_t>(TC_D) * 2;
  {  // q [B*Lb][Hq][D]: boxes of 64 dims x G heads x 128/G block positions
    const int G = x.Hq / x.Hkv;
    const cuuint64_t dims[3] = {TC_D, static_cast<cuuint64_t>(x.Hq),
                                static_cast<cuuint64_t>(x.B) * x.Lb};
    const cuuint64_t str[2] = {rs, rs * x.Hq};
    const cuuint32_t box[3] = {64, static_cast<cuuint32_t>(G), static_cast<cuuint32_t>(TC_M / G)};
    if (!encode(enc, &m->q, x.q, 3, dims, str, box)) return false;
  }
  {
    const cuuint64_t dims[3] = {TC_D, static_cast<cuuint64_t>(x.Hkv),
                                static_cast<cuuint64_t>(x.B) * x.Lb};
    const cuuint64_t str[2] = {rs, rs * x.Hkv};
    const cuuint32_t box[3] = {64, 1, TC_KT};
    if (!encode(enc, &m->kb, x.k_blk, 3, dims, str, box)) return false;
    if (!encode(enc, &m->vb, x.v_blk, 3, dims, str, box)) return false;
  }
  {
    const cuuint64_t dims[2] = {TC_D, static_cast<cuuint64_t>(x.B) * x.Hkv * x.Cmax};
    const cuuint64_t str[1] = {rs};
    const cuuint32_t box[2] = {64, TC_KT};
    if (!encode(enc, &m->kc, x.k_cache, 2, dims, str, box)) return false;
    if (!encode(enc, &m->vc, x.v_cache, 2, dims, str, box)) return false;
  }
  return true;
}

cudaError_t launch_attention_tc(const AttnArgs& x, const AttnTcPlan& p, const AttnTcMaps& m,
                                const AttnTcScratch& sc, cudaStream_t s) {
  if (p.slots > sc.max_slots) return cudaErrorInvalidValue;  // the partials would not fit
  TcArgs a;
  a.q = static_cast<const __nv_bfloat16*>(x.q);
  a.ctx = x.ctx;
  a.k_cache = static_cast<__nv_bfloat16*>(x.k_cache);
  a.v_cache = static_cast<__nv_bfloat16*>(x.v_cache);
  a.k_blk = static_cast<const __nv_bfloat16*>(x.k_blk);
  a.v_blk = static_cast<const __nv_bfloat16*>(x.v_blk);
  a.out = static_cast<__nv_bfloat16*>(x.out);
  a.part_o = sc.part_o;
  a.part_ml = sc.part_ml;
  a.counters = sc.counters;
  a.status = x.status;
  a.B = x.B;
  a.Lb = x.Lb;
  a.Hq = x.Hq;
  a.Hkv = x.Hkv;
  a.G = x.Hq / x.Hkv;
  a.Cmax = x.Cmax;
  a.rows = p.rows;
  a.n_rg = p.n_rg;
  a.chunk = p.chunk;
  a.max_chunks = p.max_chunks;
  a.scale_log2 = LOG2E / sqrtf(static_cast<float>(x.D));
  a.kv_evict_first = p.n_rg == 1;  // with several row groups each K/V tile is read again
  attention_tc_kernel<<<p.grid, TC_THREADS, p.smem_bytes, s>>>(m.kc, m.vc, m.kb, m.vb, m.q, a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess || p.max_chunks == 1) return e;

  MergeArgs g;
  g.ctx = x.ctx;
  g.part_o = sc.part_o;
  g.part_ml = sc.part_ml;
  g.out = a.out;
  g.Lb = x.Lb;
  g.Hq = x.Hq;
  g.Hkv = x.Hkv;
  g.G = a.G;
  g.Cmax = x.Cmax;
  g.rows = p.rows;
  g.n_rg = p.n_rg;
  g.chunk = p.chunk;
  g.max_chunks = p.max_chunks;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(x.B * x.Hkv * p.n_rg, TC_D / 8, 1);
  cfg.blockDim = dim3(TC_M, 1, 1);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, attention_merge_kernel, g);
}

}  // namespace rv
