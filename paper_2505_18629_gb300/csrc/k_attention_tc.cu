// Verify-block attention (Sec. 3.1) on the 5th-generation tensor cores, for
// head_dim 128 (bf16).  Same decomposition and split-KV cluster merge as the
// mma.sync kernel in k_attention.cu; the two products run as tcgen05.mma with
// the accumulators in TMEM:
//
//   S  = Q K^T   M = 128 query rows (the Lb*G rows that share a KV head, zero
//                padded), N = KT keys, K = 128 (head dim); Q and the K tile are
//                K-major, 128-byte swizzled (two 64-column halves each)
//   O += P V     M = 128, N = 128 (head dim), K = KT keys; P (bf16, written by
//                the softmax) is K-major, V is used as stored ([key][dim]) as an
//                MN-major operand
//
// Thread t of the 4 warps owns query row t (TMEM lane t): it reads its S row
// with tcgen05.ld, keeps the row max / sum, writes its P row to shared memory
// and, when its max rises by more than 2^8, rescales its O row in TMEM.  K/V
// tiles stream through a cp.async ring (XOR-swizzled into the 128-byte
// pattern the MMA expects); the block's own keys/values are read from
// k_blk/v_blk and appended to the cache by split 0.  Every mbarrier wait is
// bounded.
#include <cfloat>

#include <cooperative_groups.h>

#include "rv_device.cuh"
#include "rv_kernels.h"

namespace rv {

namespace cg = cooperative_groups;

namespace {

constexpr int TC_D = 128;
constexpr int TC_ROWS = 128;           // MMA M: query rows per CTA
constexpr int TC_THREADS = 128;        // one thread per row
constexpr int TC_MAX_SPLITS = 16;
constexpr int TC_Q_BYTES = TC_ROWS * TC_D * 2;  // 32 KB, two 16 KB halves
constexpr float TC_RESCALE_LOG2 = 8.f;  // rescale O only when the max rises by > 2^8

struct TcArgs {
  const __nv_bfloat16* q;
  const __nv_bfloat16* k_blk;
  const __nv_bfloat16* v_blk;
  __nv_bfloat16* k_cache;
  __nv_bfloat16* v_cache;
  const int32_t* ctx;
  __nv_bfloat16* out;
  int B, Lb, Hq, Hkv, Cmax, G, rows, splits;
  float scale_log2;
  unsigned* status;
};

template <int KT, int STAGES>
struct TcLayout {
  static constexpr int KV_TILE = KT * TC_D * 2;              // one K (or V) tile
  static constexpr int P_ROW = KT < 64 ? 128 : KT * 2;       // bytes per P row (>= one 128 B atom row)
  static constexpr int P_BYTES = TC_ROWS * P_ROW;
  static constexpr int Q_OFF = 0;
  static constexpr int K_OFF = TC_Q_BYTES;
  static constexpr int V_OFF = K_OFF + STAGES * KV_TILE;
  static constexpr int P_OFF = V_OFF + STAGES * KV_TILE;
  static constexpr int BAR_OFF = P_OFF + P_BYTES;             // mbar_s, mbar_o, tmem slot, abort
  static constexpr int W_OFF = BAR_OFF + 64;                  // merge weights [128][16]
  static constexpr int ML_OFF = W_OFF + TC_ROWS * TC_MAX_SPLITS * 4;  // (m, l) [128][2]
  static constexpr int BYTES = ML_OFF + TC_ROWS * 2 * 4;
  // the fp32 partial [128][128] of the merge (64 KB) overlays Q and the K/V rings
  static_assert(TC_ROWS * TC_D * 4 <= P_OFF, "merge buffer must fit in Q + K/V");
};

// byte offset of 16-byte chunk c (of 16) of row r in a [rows][128 dims] tile
// stored as two 128B-swizzled halves of 64 dims
__device__ __forceinline__ uint32_t tc_swz(int r, int c, int half_bytes) {
  return static_cast<uint32_t>((c >> 3) * half_bytes + r * 128 + (((c & 7) ^ (r & 7)) << 4));
}

}  // namespace

template <int KT, int STAGES>
__global__ void __launch_bounds__(TC_THREADS, 1) attention_tc_kernel(const TcArgs a) {
  using L = TcLayout<KT, STAGES>;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* const smem = smem_raw + (base - raw);

  const int split = blockIdx.x, kvh = blockIdx.y;
  const int n_rg = (a.rows + TC_ROWS - 1) / TC_ROWS;
  const int b = blockIdx.z / n_rg, rg = blockIdx.z % n_rg;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  const int ctx = a.ctx[b];
  if (ctx < 0 || ctx + a.Lb > a.Cmax) {
    if (split == 0 && kvh == 0 && rg == 0 && tid == 0) raise_status(a.status, RV_DEV_CTX_RANGE);
    return;
  }
  const int T = ctx + a.Lb;
  const int per = ((T + a.splits - 1) / a.splits + 15) / 16 * 16;
  const int k_lo = min(T, split * per);
  const int k_hi = min(T, k_lo + per);
  const int n_tiles = (k_hi - k_lo + KT - 1) / KT;

  const int row0 = rg * TC_ROWS;
  const int r = row0 + tid;  // this thread's query row
  const bool rvalid = r < a.rows;
  const int lim = rvalid ? ctx + r / a.G : -1;  // last key this row may see

  const uint32_t bar_s = base + L::BAR_OFF, bar_o = bar_s + 8, bar_d = bar_s + 16;
  uint32_t* const tmem_slot = reinterpret_cast<uint32_t*>(smem + L::BAR_OFF + 24);
  volatile int* const abort_flag = reinterpret_cast<volatile int*>(smem + L::BAR_OFF + 28);
  if (tid == 0) {
    mbar_init(bar_s, 1);
    mbar_init(bar_o, 1);
    mbar_init(bar_d, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0) tmem_alloc(smem_u32(tmem_slot), 256);  // S: cols [0, KT); O: [128, 256)

  // ---- Q rows and the first K/V tiles (cp.async, swizzled)
  for (int e = tid; e < TC_ROWS * 16; e += TC_THREADS) {
    const int rr = e >> 4, c = e & 15;
    const int qr = row0 + rr;
    const bool ok = qr < a.rows;
    const int j = ok ? qr / a.G : 0, hh = ok ? kvh * a.G + qr % a.G : 0;
    const __nv_bfloat16* src = a.q + ((static_cast<long long>(b) * a.Lb + j) * a.Hq + hh) * TC_D + c * 8;
    cp_async16(base + L::Q_OFF + tc_swz(rr, c, TC_ROWS * 128), src, ok);
  }
  auto load_kv = [&](int tile, int buf) {
    const int k0 = k_lo + tile * KT;
    const uint32_t kd = base + L::K_OFF + buf * L::KV_TILE;
    const uint32_t vd = base + L::V_OFF + buf * L::KV_TILE;
    for (int e = tid; e < KT * 16; e += TC_THREADS) {
      const int rr = e >> 4, c = e & 15;
      const int kk = k0 + rr;
      const bool ok = kk < k_hi;
      const __nv_bfloat16 *ks, *vs;
      if (kk < ctx) {
        const long long off = ((static_cast<long long>(b) * a.Hkv + kvh) * a.Cmax + kk) * TC_D + c * 8;
        ks = a.k_cache + off;
        vs = a.v_cache + off;
      } else {
        const int j = ok ? kk - ctx : 0;
        const long long off = ((static_cast<long long>(b) * a.Lb + j) * a.Hkv + kvh) * TC_D + c * 8;
        ks = a.k_blk + off;
        vs = a.v_blk + off;
      }
      cp_async16(kd + tc_swz(rr, c, KT * 128), ks, ok);
      cp_async16(vd + tc_swz(rr, c, KT * 128), vs, ok);
    }
  };
  if (n_tiles > 0) load_kv(0, 0);
  cp_async_commit();  // group: Q + tile 0
#pragma unroll
  for (int t = 1; t < STAGES - 1; ++t) {
    if (t < n_tiles) load_kv(t, t);
    cp_async_commit();
  }

  // Append the block's keys/values (positions ctx..ctx+Lb-1) once per (b, kvh).
  if (split == 0 && rg == 0) {
    for (int e = tid; e < a.Lb * 16; e += TC_THREADS) {
      const int j = e >> 4, c = e & 15;
      const long long src = ((static_cast<long long>(b) * a.Lb + j) * a.Hkv + kvh) * TC_D + c * 8;
      const long long dst =
          ((static_cast<long long>(b) * a.Hkv + kvh) * a.Cmax + ctx + j) * TC_D + c * 8;
      *reinterpret_cast<uint4*>(a.k_cache + dst) = *reinterpret_cast<const uint4*>(a.k_blk + src);
      *reinterpret_cast<uint4*>(a.v_cache + dst) = *reinterpret_cast<const uint4*>(a.v_blk + src);
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t t_row = tmem + (static_cast<uint32_t>(warp * 32) << 16);  // this warp's lanes
  const uint32_t s_cols = t_row, o_cols = t_row + 128u;

  const uint32_t idesc_s = idesc_bf16_f32(TC_ROWS, KT);
  const uint32_t idesc_o = idesc_bf16_f32_bmn(TC_ROWS, TC_D);
  float m_used = NEG_INF, l = 0.f;
  bool ok_all = true;

  for (int t = 0; t < n_tiles && ok_all; ++t) {
    const int buf = t % STAGES;
    cp_async_wait<STAGES - 2>();  // Q and tile t have landed
    fence_proxy_async_smem();
    __syncthreads();
    if (tid == 0) {
      tc_fence_after();
      const uint32_t kb = base + L::K_OFF + buf * L::KV_TILE;
#pragma unroll
      for (int kk = 0; kk < TC_D / 16; ++kk) {
        const uint32_t half = static_cast<uint32_t>(kk >> 2), off = static_cast<uint32_t>((kk & 3) * 32);
        tc_mma_bf16(tmem, sw128_kmajor_desc(base + L::Q_OFF + half * (TC_ROWS * 128) + off),
                    sw128_kmajor_desc(kb + half * (KT * 128) + off), idesc_s, kk > 0 ? 1u : 0u);
      }
      tc_commit(bar_s);
    }
    bool ok = mbar_wait(bar_s, t & 1, abort_flag, a.status);
    if (ok && t > 0) ok = mbar_wait(bar_o, (t - 1) & 1, abort_flag, a.status);  // PV(t-1) done
    if (!__syncthreads_and(ok)) {
      ok_all = false;
      break;
    }
    tc_fence_after();

    // ---- online softmax of this row over the tile's KT keys
    float sv[KT];
#pragma unroll
    for (int c = 0; c < KT; c += 32) {
      float tmp[32];
      tmem_ld32(s_cols + c, tmp);
#pragma unroll
      for (int i = 0; i < 32; ++i) sv[c + i] = tmp[i];
    }
    tmem_ld_wait();
    const int kbase = k_lo + t * KT;
    float mt = NEG_INF;
#pragma unroll
    for (int j = 0; j < KT; ++j) {
      const int key = kbase + j;
      sv[j] = (key < k_hi && key <= lim) ? sv[j] * a.scale_log2 : NEG_INF;
      mt = fmaxf(mt, sv[j]);
    }
    float fac = 1.f;
    const bool rise = mt > m_used + TC_RESCALE_LOG2 || (m_used == NEG_INF && mt != NEG_INF);
    if (rise) {
      fac = (m_used == NEG_INF) ? 0.f : exp2f(m_used - mt);
      m_used = mt;
    }
    // O already holds earlier tiles (t > 0): rescale this warp's rows if any rose
    if (t > 0 && __any_sync(0xffffffffu, rise && fac != 1.f)) {
#pragma unroll
      for (int c = 0; c < TC_D; c += 32) {
        float ov[32];
        tmem_ld32(o_cols + c, ov);
        tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 32; ++i) ov[i] *= fac;
        tmem_st32(o_cols + c, ov);
      }
      tmem_st_wait();
    }
    l *= fac;
    // P row (bf16) into the K-major swizzled P tile
    uint8_t* const prow = smem + L::P_OFF + tid * 128;
#pragma unroll
    for (int c = 0; c < KT / 8; ++c) {
      float p[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        p[i] = (m_used == NEG_INF) ? 0.f : exp2f(sv[c * 8 + i] - m_used);
        l += p[i];
      }
      uint4 pk;
      pk.x = pack_bf16(p[0], p[1]);
      pk.y = pack_bf16(p[2], p[3]);
      pk.z = pack_bf16(p[4], p[5]);
      pk.w = pack_bf16(p[6], p[7]);
      const int half = c >> 3, cc = c & 7;
      *reinterpret_cast<uint4*>(prow + half * (TC_ROWS * 128) + ((cc ^ (tid & 7)) << 4)) = pk;
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    if (tid == 0) {
      tc_fence_after();
      const uint32_t vb = base + L::V_OFF + buf * L::KV_TILE;
#pragma unroll
      for (int kk = 0; kk < KT / 16; ++kk) {
        const uint32_t half = static_cast<uint32_t>(kk >> 2), off = static_cast<uint32_t>((kk & 3) * 32);
        tc_mma_bf16(tmem + 128u,
                    sw128_kmajor_desc(base + L::P_OFF + half * (TC_ROWS * 128) + off),
                    sw128_mnmajor_desc(vb + kk * 16 * 128, KT * 128, 1024), idesc_o,
                    (t > 0 || kk > 0) ? 1u : 0u);
      }
      tc_commit(bar_o);
    }
    // refill: tile t+STAGES-1 into the buffer of tile t-1 (its PV is complete)
    if (t + STAGES - 1 < n_tiles) load_kv(t + STAGES - 1, (t + STAGES - 1) % STAGES);
    cp_async_commit();
  }
  cp_async_wait_all();
  if (ok_all && n_tiles > 0) {
    const bool ok = mbar_wait(bar_o, (n_tiles - 1) & 1, abort_flag, a.status);
    ok_all = __syncthreads_and(ok);
  } else {
    ok_all = __syncthreads_and(ok_all) && ok_all;
  }
  tc_fence_after();

  // ---- this row's O/l (zeros when the row saw no key)
  const float inv = (l > 0.f) ? 1.f / l : 0.f;
  auto row_index = [&](int rr) {
    const int j = rr / a.G, hh = kvh * a.G + rr % a.G;
    return (static_cast<long long>(b) * a.Lb + j) * a.Hq + hh;
  };
  float* const part = reinterpret_cast<float*>(smem);  // [128][128], overlays Q and K/V
  __syncthreads();  // every thread is done with Q / K / V before the overlay is written
#pragma unroll
  for (int c = 0; c < TC_D; c += 32) {
    float ov[32];
    tmem_ld32(o_cols + c, ov);
    tmem_ld_wait();
#pragma unroll
    for (int i = 0; i < 32; ++i) ov[i] = (n_tiles > 0 && l > 0.f) ? ov[i] * inv : 0.f;
    if (a.splits == 1) {
      if (rvalid) {
        __nv_bfloat16* dst = a.out + row_index(r) * TC_D + c;
#pragma unroll
        for (int i = 0; i < 32; i += 8) {
          uint4 pk;
          pk.x = pack_bf16(ov[i], ov[i + 1]);
          pk.y = pack_bf16(ov[i + 2], ov[i + 3]);
          pk.z = pack_bf16(ov[i + 4], ov[i + 5]);
          pk.w = pack_bf16(ov[i + 6], ov[i + 7]);
          *reinterpret_cast<uint4*>(dst + i) = pk;
        }
      }
    } else {
#pragma unroll
      for (int i = 0; i < 32; i += 4) {
        const int i2 = (i + 4 * (tid & 7)) & 31;  // rotate to spread banks
        *reinterpret_cast<float4*>(part + tid * TC_D + c + i2) =
            make_float4(ov[i2], ov[i2 + 1], ov[i2 + 2], ov[i2 + 3]);
      }
    }
  }
  float* const wsm = reinterpret_cast<float*>(smem + L::W_OFF);
  float* const ml = reinterpret_cast<float*>(smem + L::ML_OFF);
  if (a.splits > 1) {
    ml[2 * tid] = m_used;
    ml[2 * tid + 1] = l;
  }
  // every MMA issued must be complete before TMEM is released (a no-op wait
  // unless a pipeline wait above gave up)
  if (tid == 0) {
    tc_commit(bar_d);
    const unsigned long long t0 = globaltimer_ns();
    while (!mbar_try_wait(bar_d, 0) && globaltimer_ns() - t0 < RV_WAIT_TIMEOUT_NS / 4) {
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, 256);
  }
  if (a.splits == 1) return;

  // ---- split-KV merge through distributed shared memory (as in k_attention.cu)
  cg::cluster_group cluster = cg::this_cluster();
  cluster.sync();
  const int S = a.splits;
  const int rank = static_cast<int>(cluster.block_rank());
  const int nrow = min(TC_ROWS, a.rows - row0);
  const int per_rank = (nrow + S - 1) / S;
  const int r_lo = min(nrow, rank * per_rank), r_hi = min(nrow, r_lo + per_rank);
  const int n_items = (r_hi - r_lo) * S;
  for (int b0 = 0; b0 < n_items; b0 += TC_THREADS) {
    const int it = b0 + tid;
    const bool act = it < n_items;
    const int rl = r_lo + (act ? it / S : 0), sp = it % S;
    float m = NEG_INF, lv = 0.f;
    if (act) {
      const float* rml = cluster.map_shared_rank(ml, sp);
      m = rml[2 * rl];
      lv = rml[2 * rl + 1];
    }
    float M = lv > 0.f ? m : NEG_INF;
    for (int o = 1; o < S; o <<= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
    const float w = lv > 0.f ? lv * exp2f(m - M) : 0.f;
    float den = w;
    for (int o = 1; o < S; o <<= 1) den += __shfl_xor_sync(0xffffffffu, den, o);
    if (act) wsm[rl * TC_MAX_SPLITS + sp] = den > 0.f ? w / den : 0.f;
  }
  __syncthreads();
  constexpr int D4 = TC_D / 4;
  for (int it = tid; it < (r_hi - r_lo) * D4; it += TC_THREADS) {
    const int rl = r_lo + it / D4, d = (it % D4) * 4;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int sp = 0; sp < TC_MAX_SPLITS; ++sp) {
      if (sp < S) {
        const float w = wsm[rl * TC_MAX_SPLITS + sp];
        const float4 v =
            *reinterpret_cast<const float4*>(cluster.map_shared_rank(part, sp) + rl * TC_D + d);
        acc.x = fmaf(w, v.x, acc.x);
        acc.y = fmaf(w, v.y, acc.y);
        acc.z = fmaf(w, v.z, acc.z);
        acc.w = fmaf(w, v.w, acc.w);
      }
    }
    uint2 pk;
    pk.x = pack_bf16(acc.x, acc.y);
    pk.y = pack_bf16(acc.z, acc.w);
    *reinterpret_cast<uint2*>(a.out + row_index(row0 + rl) * TC_D + d) = pk;
  }
  cluster.sync();
}

// ---------------------------------------------------------------- launch

namespace {
constexpr int TC_KT = 64;
constexpr int TC_STAGES = 3;
}  // namespace

size_t attn_tc_smem_bytes() { return TcLayout<TC_KT, TC_STAGES>::BYTES + 1024; }

cudaError_t attn_tc_configure() {
  auto k = attention_tc_kernel<TC_KT, TC_STAGES>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(attn_tc_smem_bytes()));
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(k, cudaFuncAttributePreferredSharedMemoryCarveout,
                             cudaSharedmemCarveoutMaxShared);
  if (e == cudaSuccess) e = cudaFuncSetAttribute(k, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  return e;
}

cudaError_t launch_attention_tc(const AttnArgs& x, const AttnPlan& p, cudaStream_t s) {
  TcArgs a;
  a.q = static_cast<const __nv_bfloat16*>(x.q);
  a.k_blk = static_cast<const __nv_bfloat16*>(x.k_blk);
  a.v_blk = static_cast<const __nv_bfloat16*>(x.v_blk);
  a.k_cache = static_cast<__nv_bfloat16*>(x.k_cache);
  a.v_cache = static_cast<__nv_bfloat16*>(x.v_cache);
  a.ctx = x.ctx;
  a.out = static_cast<__nv_bfloat16*>(x.out);
  a.B = x.B;
  a.Lb = x.Lb;
  a.Hq = x.Hq;
  a.Hkv = x.Hkv;
  a.Cmax = x.Cmax;
  a.G = x.Hq / x.Hkv;
  a.rows = p.rows;
  a.splits = p.splits;
  a.scale_log2 = LOG2E / sqrtf(static_cast<float>(x.D));
  a.status = x.status;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.splits, x.Hkv, x.B * ((p.rows + TC_ROWS - 1) / TC_ROWS));
  cfg.blockDim = dim3(TC_THREADS, 1, 1);
  cfg.dynamicSmemBytes = attn_tc_smem_bytes();
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = p.splits;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = p.splits > 1 ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, attention_tc_kernel<TC_KT, TC_STAGES>, a);
}

}  // namespace rv
