// One attention layer of the verify forward pass (Sec. 3.1): the packed block
// [x_1..x_gamma | template | x_1..x_gamma] attends causally to the KV cache and
// to itself.  Query j of sequence b (position ctx_b + j) sees cached keys
// [0, ctx_b) and block keys [0, j]; with GQA, query head h reads KV head h / G.
//
// bf16 path: split-KV flash-decoding.  One CTA per (key split, KV head,
// sequence, row group) stages its keys/values through shared memory in tiles
// of 32 with 16-byte cp.async loads (a ring of three, XOR-swizzled rows) and
// runs QK^T and PV on the tensor cores (mma.sync m16n8k16 bf16, fp32
// accumulate).  All G*Lb query rows that share a KV head live in one CTA
// (16 rows per warp), so each key/value byte is read once per head.  The
// splits of one (sequence, KV head, row group) form a thread-block cluster:
// each CTA leaves its partial (O/l, m, l) in its own shared memory and, after
// a cluster barrier, every CTA merges a slice of the rows by reading all the
// partials through distributed shared memory.  No partials touch global
// memory and no second kernel is launched.  The block's own
// keys/values are read from k_blk/v_blk and appended to the cache at
// [ctx_b, ctx_b + Lb) by one CTA per (sequence, KV head); no CTA reads those
// cache positions, so the append does not race.
//
// fp32 path: one warp per query row on the CUDA cores (tiny fp32 models).
#include <cfloat>

#include <cooperative_groups.h>

#include "rv_device.cuh"
#include "rv_kernels.h"

namespace rv {

namespace cg = cooperative_groups;

constexpr int AT_KT = 32;         // keys per shared-memory tile
constexpr int AT_STAGES = 3;      // K/V tiles in flight (cp.async ring)
constexpr int AT_MAX_WARPS = 8;   // 16 query rows per warp -> 128 rows per CTA
constexpr int AT_MAX_SPLITS = 16; // cluster size limit (non-portable above 8)

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ __forceinline__ void mma_bf16_16816(float (&c)[4], const uint32_t (&a)[4], uint32_t b0,
                                               uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}


// Byte offset of 16-byte chunk `c` of row `r` in a swizzled tile of rows of D bf16.
template <int D>
__device__ __forceinline__ uint32_t swz(int r, int c) {
  return static_cast<uint32_t>(r * (D * 2) + ((c ^ (r & 7)) << 4));
}

struct AttnKernelArgs {
  const __nv_bfloat16* q;
  const __nv_bfloat16* k_blk;
  const __nv_bfloat16* v_blk;
  __nv_bfloat16* k_cache;
  __nv_bfloat16* v_cache;
  const int32_t* ctx;
  __nv_bfloat16* out;
  int B, Lb, Hq, Hkv, Cmax, G, rows, splits;
  float scale_log2;  // log2(e) / sqrt(D)
  unsigned* status;
};

// 168 registers let two CTAs of up to 6 warps share an SM.
template <int D>
__global__ void __maxnreg__(168) attention_bf16_kernel(const AttnKernelArgs a) {
  constexpr int CH = D / 8;            // 16-byte chunks per row
  constexpr int TILE_BYTES = AT_KT * D * 2;
  const int WROWS = static_cast<int>(blockDim.x / 32) * 16;  // query rows of this CTA
  const int Q_BYTES = WROWS * D * 2;
  extern __shared__ __align__(128) uint8_t smem[];
  // [Q: WROWS rows][K/V ring: AT_STAGES x (K tile, V tile)][merge weights]
  // After the key loop the Q region holds (m, l) per row and the K/V region
  // the fp32 partial O/l of every row (read by the other CTAs of the cluster).
  const uint32_t s_base = smem_u32(smem);
  const uint32_t s_q = s_base;
  const uint32_t s_kv = s_base + Q_BYTES;

  const int split = blockIdx.x, kvh = blockIdx.y;
  const int n_rg = (a.rows + AT_MAX_WARPS * 16 - 1) / (AT_MAX_WARPS * 16);
  const int b = blockIdx.z / n_rg, rg = blockIdx.z % n_rg;
  const int tid = threadIdx.x, nthr = blockDim.x;
  const int warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, t4 = lane & 3;

  const int ctx = a.ctx[b];
  if (ctx < 0 || ctx + a.Lb > a.Cmax) {
    if (split == 0 && kvh == 0 && rg == 0 && tid == 0) raise_status(a.status, RV_DEV_CTX_RANGE);
    return;
  }
  const int T = ctx + a.Lb;
  // Key range of this split: near-equal shares in multiples of 16 keys.
  const int per = ((T + a.splits - 1) / a.splits + 15) / 16 * 16;
  const int k_lo = min(T, split * per);
  const int k_hi = min(T, k_lo + per);

  const int row0 = rg * AT_MAX_WARPS * 16;  // first query row of this CTA (within the KV head)
  // (a row group spans up to 128 rows; a CTA with fewer warps only exists when
  // there is a single row group, whose rows then all fit its warps)
  // Rows of this thread: r_a = row0 + warp*16 + g, r_b = r_a + 8.  Row r <-> (j = r / G, h = kvh*G + r % G).
  const int r_a = row0 + warp * 16 + g, r_b = r_a + 8;
  const bool va = r_a < a.rows, vb = r_b < a.rows;
  const int lim_a = va ? ctx + r_a / a.G : -1;  // last visible key
  const int lim_b = vb ? ctx + r_b / a.G : -1;

  // ---- Q rows -> shared memory (group 0)
  for (int e = tid; e < WROWS * CH; e += nthr) {
    const int r = e / CH, c = e % CH;
    const int rr = row0 + r;
    const bool ok = rr < a.rows;
    const int j = ok ? rr / a.G : 0, hh = ok ? kvh * a.G + rr % a.G : 0;
    const __nv_bfloat16* src = a.q + ((static_cast<long long>(b) * a.Lb + j) * a.Hq + hh) * D + c * 8;
    cp_async16(s_q + swz<D>(r, c), src, ok);
  }
  cp_async_commit();

  auto load_kv = [&](int tile_k0, int buf) {
    const uint32_t sk = s_kv + buf * 2 * TILE_BYTES, sv = sk + TILE_BYTES;
    for (int e = tid; e < AT_KT * CH; e += nthr) {
      const int r = e / CH, c = e % CH;
      const int kk = tile_k0 + r;
      const bool ok = kk < k_hi;
      const __nv_bfloat16 *ks, *vs;
      if (kk < ctx) {
        const long long off = ((static_cast<long long>(b) * a.Hkv + kvh) * a.Cmax + kk) * D + c * 8;
        ks = a.k_cache + off;
        vs = a.v_cache + off;
      } else {
        const int j = ok ? kk - ctx : 0;
        const long long off = ((static_cast<long long>(b) * a.Lb + j) * a.Hkv + kvh) * D + c * 8;
        ks = a.k_blk + off;
        vs = a.v_blk + off;
      }
      cp_async16(sk + swz<D>(r, c), ks, ok);
      cp_async16(sv + swz<D>(r, c), vs, ok);
    }
  };

  // AT_STAGES tiles in flight from the start (one commit group each; empty
  // groups are fine).
  const int n_tiles = (k_hi - k_lo + AT_KT - 1) / AT_KT;
#pragma unroll
  for (int t = 0; t < AT_STAGES; ++t) {
    if (t < n_tiles) load_kv(k_lo + t * AT_KT, t);
    cp_async_commit();
  }

  // Append the block's keys/values (positions ctx..ctx+Lb-1) once per (b, kvh).
  if (split == 0 && rg == 0) {
    for (int e = tid; e < a.Lb * CH; e += nthr) {
      const int j = e / CH, c = e % CH;
      const long long src = ((static_cast<long long>(b) * a.Lb + j) * a.Hkv + kvh) * D + c * 8;
      const long long dst = ((static_cast<long long>(b) * a.Hkv + kvh) * a.Cmax + ctx + j) * D + c * 8;
      *reinterpret_cast<uint4*>(a.k_cache + dst) = *reinterpret_cast<const uint4*>(a.k_blk + src);
      *reinterpret_cast<uint4*>(a.v_cache + dst) = *reinterpret_cast<const uint4*>(a.v_blk + src);
    }
  }

  float o[D / 8][4];
#pragma unroll
  for (int i = 0; i < D / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float m_a = NEG_INF, m_b = NEG_INF, l_a = 0.f, l_b = 0.f;

  for (int it = 0; it < n_tiles; ++it) {
    const int buf = it % AT_STAGES;
    cp_async_wait<AT_STAGES - 1>();  // Q and tile `it` have landed
    __syncthreads();
    const uint32_t sk = s_kv + buf * 2 * TILE_BYTES, sv = sk + TILE_BYTES;
    const int kbase = k_lo + it * AT_KT;

    // S = Q K^T for 16 rows x 64 keys (Q fragments re-read from shared memory)
    float s[AT_KT / 8][4];
#pragma unroll
    for (int nt = 0; nt < AT_KT / 8; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
#pragma unroll
    for (int ks = 0; ks < D / 16; ++ks) {
      const int mi = lane >> 3;
      uint32_t qf[4];
      ldsm_x4(s_q + swz<D>(warp * 16 + (mi & 1) * 8 + (lane & 7), 2 * ks + (mi >> 1)), qf[0], qf[1],
              qf[2], qf[3]);
#pragma unroll
      for (int nt = 0; nt < AT_KT / 8; nt += 2) {
        const int key = 8 * (nt + (mi >> 1)) + (lane & 7);
        uint32_t b0, b1, b2, b3;
        ldsm_x4(sk + swz<D>(key, 2 * ks + (mi & 1)), b0, b1, b2, b3);
        mma_bf16_16816(s[nt], qf, b0, b1);
        mma_bf16_16816(s[nt + 1], qf, b2, b3);
      }
    }
    // mask + online softmax (rows r_a: s[.][0..1], r_b: s[.][2..3])
    float mx_a = NEG_INF, mx_b = NEG_INF;
#pragma unroll
    for (int nt = 0; nt < AT_KT / 8; ++nt) {
      const int k0 = kbase + nt * 8 + 2 * t4;
      const bool in0 = k0 < k_hi, in1 = k0 + 1 < k_hi;
      s[nt][0] = (in0 && k0 <= lim_a) ? s[nt][0] : NEG_INF;
      s[nt][1] = (in1 && k0 + 1 <= lim_a) ? s[nt][1] : NEG_INF;
      s[nt][2] = (in0 && k0 <= lim_b) ? s[nt][2] : NEG_INF;
      s[nt][3] = (in1 && k0 + 1 <= lim_b) ? s[nt][3] : NEG_INF;
      mx_a = fmaxf(mx_a, fmaxf(s[nt][0], s[nt][1]));
      mx_b = fmaxf(mx_b, fmaxf(s[nt][2], s[nt][3]));
    }
    mx_a = fmaxf(mx_a, __shfl_xor_sync(0xffffffffu, mx_a, 1));
    mx_a = fmaxf(mx_a, __shfl_xor_sync(0xffffffffu, mx_a, 2));
    mx_b = fmaxf(mx_b, __shfl_xor_sync(0xffffffffu, mx_b, 1));
    mx_b = fmaxf(mx_b, __shfl_xor_sync(0xffffffffu, mx_b, 2));
    const float mn_a = fmaxf(m_a, mx_a), mn_b = fmaxf(m_b, mx_b);
    const float ca = (mn_a == NEG_INF) ? 1.f : exp2f((m_a - mn_a) * a.scale_log2);
    const float cb = (mn_b == NEG_INF) ? 1.f : exp2f((m_b - mn_b) * a.scale_log2);
    m_a = mn_a;
    m_b = mn_b;
    l_a *= ca;
    l_b *= cb;
#pragma unroll
    for (int dt = 0; dt < D / 8; ++dt) {
      o[dt][0] *= ca;
      o[dt][1] *= ca;
      o[dt][2] *= cb;
      o[dt][3] *= cb;
    }
    const float sa = m_a * a.scale_log2, sb = m_b * a.scale_log2;
#pragma unroll
    for (int nt = 0; nt < AT_KT / 8; ++nt) {
      s[nt][0] = (m_a == NEG_INF) ? 0.f : exp2f(s[nt][0] * a.scale_log2 - sa);
      s[nt][1] = (m_a == NEG_INF) ? 0.f : exp2f(s[nt][1] * a.scale_log2 - sa);
      s[nt][2] = (m_b == NEG_INF) ? 0.f : exp2f(s[nt][2] * a.scale_log2 - sb);
      s[nt][3] = (m_b == NEG_INF) ? 0.f : exp2f(s[nt][3] * a.scale_log2 - sb);
      l_a += s[nt][0] + s[nt][1];
      l_b += s[nt][2] + s[nt][3];
    }
    // O += P V
#pragma unroll
    for (int kk = 0; kk < AT_KT / 16; ++kk) {
      uint32_t pa[4];
      pa[0] = pack_bf16(s[2 * kk][0], s[2 * kk][1]);
      pa[1] = pack_bf16(s[2 * kk][2], s[2 * kk][3]);
      pa[2] = pack_bf16(s[2 * kk + 1][0], s[2 * kk + 1][1]);
      pa[3] = pack_bf16(s[2 * kk + 1][2], s[2 * kk + 1][3]);
#pragma unroll
      for (int dt = 0; dt < D / 8; dt += 2) {
        const int mi = lane >> 3;
        const int key = 16 * kk + (mi & 1) * 8 + (lane & 7);
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(sv + swz<D>(key, dt + (mi >> 1)), b0, b1, b2, b3);
        mma_bf16_16816(o[dt], pa, b0, b1);
        mma_bf16_16816(o[dt + 1], pa, b2, b3);
      }
    }
    __syncthreads();  // every warp is done with buffer `buf`
    if (it + AT_STAGES < n_tiles) load_kv(k_lo + (it + AT_STAGES) * AT_KT, buf);
    cp_async_commit();
  }
  cp_async_wait_all();

  l_a += __shfl_xor_sync(0xffffffffu, l_a, 1);
  l_a += __shfl_xor_sync(0xffffffffu, l_a, 2);
  l_b += __shfl_xor_sync(0xffffffffu, l_b, 1);
  l_b += __shfl_xor_sync(0xffffffffu, l_b, 2);
  const float ia = l_a > 0.f ? 1.f / l_a : 0.f, ib = l_b > 0.f ? 1.f / l_b : 0.f;

  auto row_index = [&](int r) {  // (b, j, h) flattened
    const int j = r / a.G, hh = kvh * a.G + r % a.G;
    return (static_cast<long long>(b) * a.Lb + j) * a.Hq + hh;
  };
  if (a.splits == 1) {
#pragma unroll
    for (int dt = 0; dt < D / 8; ++dt) {
      const int d = dt * 8 + 2 * t4;
      if (va)
        *reinterpret_cast<uint32_t*>(a.out + row_index(r_a) * D + d) =
            pack_bf16(o[dt][0] * ia, o[dt][1] * ia);
      if (vb)
        *reinterpret_cast<uint32_t*>(a.out + row_index(r_b) * D + d) =
            pack_bf16(o[dt][2] * ib, o[dt][3] * ib);
    }
    return;
  }

  // ---- split-KV merge through distributed shared memory
  __syncthreads();  // all warps done with Q and the K/V buffers
  // After the key loop: the fp32 partial O/l [WROWS][D] overwrites Q and the
  // K/V ring (WROWS*D*4 <= WROWS*D*2 + ring bytes for WROWS <= 128), the merge
  // weights [WROWS][16] and (m, l) [WROWS][2] follow the ring.
  static_assert(AT_MAX_WARPS * 16 <= 2 * AT_STAGES * AT_KT, "merge buffer exceeds Q + ring");
  float* const part = reinterpret_cast<float*>(smem);
  float* const wsm = reinterpret_cast<float*>(smem + Q_BYTES + 2 * AT_STAGES * TILE_BYTES);
  float* const ml = wsm + WROWS * AT_MAX_SPLITS;
  const int la = warp * 16 + g, lbr = la + 8;  // rows within the CTA window
#pragma unroll
  for (int dt = 0; dt < D / 8; ++dt) {
    const int d = dt * 8 + 2 * t4;
    *reinterpret_cast<float2*>(part + la * D + d) = make_float2(o[dt][0] * ia, o[dt][1] * ia);
    *reinterpret_cast<float2*>(part + lbr * D + d) = make_float2(o[dt][2] * ib, o[dt][3] * ib);
  }
  if (t4 == 0) {
    ml[2 * la] = m_a * a.scale_log2;
    ml[2 * la + 1] = l_a;
    ml[2 * lbr] = m_b * a.scale_log2;
    ml[2 * lbr + 1] = l_b;
  }
  cg::cluster_group cluster = cg::this_cluster();
  cluster.sync();
  const int S = a.splits;
  const int rank = static_cast<int>(cluster.block_rank());
  const int nrow = min(WROWS, a.rows - row0);
  const int per_rank = (nrow + S - 1) / S;
  const int r_lo = min(nrow, rank * per_rank), r_hi = min(nrow, r_lo + per_rank);
  // weights w_s = l_s 2^(m_s - M) / sum_s(...): one thread per (row, split);
  // S is a power of two <= 16, so a row's S threads are adjacent lanes of one warp.
  const int n_items = (r_hi - r_lo) * S;
  for (int base = 0; base < n_items; base += nthr) {
    const int it = base + tid;
    const bool act = it < n_items;
    const int rl = r_lo + (act ? it / S : 0), sp = it % S;
    float m = NEG_INF, l = 0.f;
    if (act) {
      const float* rml = cluster.map_shared_rank(ml, sp);
      m = rml[2 * rl];
      l = rml[2 * rl + 1];
    }
    float M = l > 0.f ? m : NEG_INF;
    for (int o = 1; o < S; o <<= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
    const float w = l > 0.f ? l * exp2f(m - M) : 0.f;
    float den = w;
    for (int o = 1; o < S; o <<= 1) den += __shfl_xor_sync(0xffffffffu, den, o);
    if (act) wsm[rl * AT_MAX_SPLITS + sp] = den > 0.f ? w / den : 0.f;
  }
  __syncthreads();
  constexpr int D4 = D / 4;
  for (int it = tid; it < (r_hi - r_lo) * D4; it += nthr) {
    const int rl = r_lo + it / D4, d = (it % D4) * 4;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int sp = 0; sp < AT_MAX_SPLITS; ++sp) {
      if (sp < S) {
        const float w = wsm[rl * AT_MAX_SPLITS + sp];
        const float4 v =
            *reinterpret_cast<const float4*>(cluster.map_shared_rank(part, sp) + rl * D + d);
        acc.x = fmaf(w, v.x, acc.x);
        acc.y = fmaf(w, v.y, acc.y);
        acc.z = fmaf(w, v.z, acc.z);
        acc.w = fmaf(w, v.w, acc.w);
      }
    }
    uint2 pk;
    pk.x = pack_bf16(acc.x, acc.y);
    pk.y = pack_bf16(acc.z, acc.w);
    *reinterpret_cast<uint2*>(a.out + row_index(row0 + rl) * D + d) = pk;
  }
  cluster.sync();  // partials stay alive until every CTA of the cluster has read them
}

// ---------------------------------------------------------------- fp32 path
// One warp per query row (b, j, h); keys in order, online softmax in fp32.
__global__ void attention_f32_kernel(const float* __restrict__ q, const float* __restrict__ k_blk,
                                     const float* __restrict__ v_blk, float* k_cache,
                                     float* v_cache, const int32_t* __restrict__ ctx_lens,
                                     float* __restrict__ out, int B, int Lb, int Hq, int Hkv,
                                     int D, int Cmax, float scale, unsigned* status) {
  const long long nrows = static_cast<long long>(B) * Lb * Hq;
  const long long row = (static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (row >= nrows) return;
  const int h = static_cast<int>(row % Hq);
  const int j = static_cast<int>((row / Hq) % Lb);
  const int b = static_cast<int>(row / (static_cast<long long>(Hq) * Lb));
  const int G = Hq / Hkv, kvh = h / G;
  const int ctx = ctx_lens[b];
  if (ctx < 0 || ctx + Lb > Cmax) {
    if (j == 0 && h == 0 && lane == 0) raise_status(status, RV_DEV_CTX_RANGE);
    return;
  }
  constexpr int MAXE = 8;  // D <= 256
  const int ne = D / 32;
  float qv[MAXE], acc[MAXE];
#pragma unroll
  for (int e = 0; e < MAXE; ++e) {
    qv[e] = e < ne ? q[row * D + lane + 32 * e] : 0.f;
    acc[e] = 0.f;
  }
  const float* kc = k_cache + (static_cast<long long>(b) * Hkv + kvh) * Cmax * D;
  const float* vc = v_cache + (static_cast<long long>(b) * Hkv + kvh) * Cmax * D;
  float m = NEG_INF, l = 0.f;
  const int last = ctx + j;  // inclusive
  for (int kk = 0; kk <= last; ++kk) {
    const float* kr;
    const float* vr;
    if (kk < ctx) {
      kr = kc + static_cast<long long>(kk) * D;
      vr = vc + static_cast<long long>(kk) * D;
    } else {
      const long long off = ((static_cast<long long>(b) * Lb + (kk - ctx)) * Hkv + kvh) * D;
      kr = k_blk + off;
      vr = v_blk + off;
    }
    float dot = 0.f;
#pragma unroll
    for (int e = 0; e < MAXE; ++e)
      if (e < ne) dot = fmaf(qv[e], kr[lane + 32 * e], dot);
    dot = warp_sum(dot) * scale;
    const float mn = fmaxf(m, dot);
    const float c = expf(m - mn), p = expf(dot - mn);
    l = l * c + p;
#pragma unroll
    for (int e = 0; e < MAXE; ++e)
      if (e < ne) acc[e] = acc[e] * c + p * vr[lane + 32 * e];
    m = mn;
  }
#pragma unroll
  for (int e = 0; e < MAXE; ++e)
    if (e < ne) out[row * D + lane + 32 * e] = acc[e] / l;
  // append the block's key/value of position ctx + j (first query head of the group)
  if (h % G == 0) {
    const long long src = ((static_cast<long long>(b) * Lb + j) * Hkv + kvh) * D;
    const long long dst = ((static_cast<long long>(b) * Hkv + kvh) * Cmax + ctx + j) * D;
    for (int d = lane; d < D; d += 32) {
      k_cache[dst + d] = k_blk[src + d];
      v_cache[dst + d] = v_blk[src + d];
    }
  }
}

// ---------------------------------------------------------------- planning / launch

#ifndef RV_ATTN_TC_MIN_UNITS
#define RV_ATTN_TC_MIN_UNITS 0  // (sequence, KV head) pairs that select tcgen05; 0: SMs / 4
#endif
AttnPlan attn_plan(int B, int Lb, int Hq, int Hkv, int Cmax, int num_sms, bool bf16,
                   int max_cluster, int D, bool allow_tc) {
  AttnPlan p;
  const int G = Hq / Hkv;
  p.rows = Lb * G;
  p.tc = false;
  if (!bf16) {
    p.row_groups = 1;
    p.splits = 1;
    p.warps = 0;
    return p;
  }
  // tcgen05 kernel (k_attention_tc.cu) once there are enough (sequence, KV
  // head) pairs to fill a quarter of the SMs; below that the step is
  // latency-bound and the small mma.sync kernel shares the SMs with the LM head.
  if (allow_tc && attn_tc_supported(Hq, Hkv, D) &&
      B * Hkv >= (RV_ATTN_TC_MIN_UNITS > 0 ? RV_ATTN_TC_MIN_UNITS : num_sms / 4)) {
    p.tc = true;
    p.row_groups = 0;
    p.splits = 0;
    p.warps = 0;
    return p;
  }
  p.row_groups = (p.rows + AT_MAX_WARPS * 16 - 1) / (AT_MAX_WARPS * 16);
  p.warps = std::min(AT_MAX_WARPS, (p.rows + 15) / 16);
  if (p.row_groups > 1) p.warps = AT_MAX_WARPS;
  const int base = B * Hkv * p.row_groups;
  int s = (2 * num_sms + base - 1) / base;          // about two CTAs per SM
  const int max_useful = (Cmax + 2 * AT_KT - 1) / (2 * AT_KT);  // >= 128 keys per split
  s = std::max(1, std::min(s, std::min(max_useful, std::min(max_cluster, AT_MAX_SPLITS))));
  int pow2 = 1;  // the merge groups a row's splits inside one warp: power of two
  while (pow2 * 2 <= s) pow2 *= 2;
  p.splits = pow2;
  return p;
}

// Q rows + the K/V ring + merge weights + (m, l).  The fp32 partial [rows][D]
// of the merge reuses the Q and K/V space (rows*D*4 <= Q + ring).
size_t attn_bf16_smem_bytes(int D, int warps) {
  return static_cast<size_t>(warps) * 16 * D * 2 + 2 * AT_STAGES * static_cast<size_t>(AT_KT) * D * 2 +
         static_cast<size_t>(warps) * 16 * (AT_MAX_SPLITS + 2) * 4;
}

template <int D>
static cudaError_t attn_configure_d() {
  auto k = attention_bf16_kernel<D>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(attn_bf16_smem_bytes(D, AT_MAX_WARPS)));
  if (e == cudaSuccess)  // share SMs with the concurrently running LM head
    e = cudaFuncSetAttribute(k, cudaFuncAttributePreferredSharedMemoryCarveout,
                             cudaSharedmemCarveoutMaxShared);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(k, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
}

// Largest cluster size (<= 16) for which clusters of the D=128 kernel can be resident.
static int max_cluster_for(int D) {
  for (int cs = AT_MAX_SPLITS; cs > 1; cs >>= 1) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(cs, 1, 1);
    cfg.blockDim = dim3(AT_MAX_WARPS * 32, 1, 1);
    cfg.dynamicSmemBytes = attn_bf16_smem_bytes(D, AT_MAX_WARPS);
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = cs;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    cudaError_t e = D == 128 ? cudaOccupancyMaxActiveClusters(&n, attention_bf16_kernel<128>, &cfg)
                             : cudaOccupancyMaxActiveClusters(&n, attention_bf16_kernel<64>, &cfg);
    if (e == cudaSuccess && n > 0) return cs;
    cudaGetLastError();
  }
  return 1;
}

cudaError_t attn_configure(int* max_cluster) {
  cudaError_t e = attn_configure_d<128>();
  if (e == cudaSuccess) e = attn_configure_d<64>();
  if (e != cudaSuccess) return e;
  *max_cluster = std::min(max_cluster_for(128), max_cluster_for(64));
  return cudaSuccess;
}

cudaError_t launch_attention_bf16(const AttnArgs& x, const AttnPlan& p, cudaStream_t s) {
  AttnKernelArgs a;
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
  cfg.gridDim = dim3(p.splits, x.Hkv, x.B * p.row_groups);
  cfg.blockDim = dim3(p.warps * 32, 1, 1);
  cfg.dynamicSmemBytes = attn_bf16_smem_bytes(x.D, p.warps);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = p.splits;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = p.splits > 1 ? 1 : 0;
  if (x.D == 128) return cudaLaunchKernelEx(&cfg, attention_bf16_kernel<128>, a);
  if (x.D == 64) return cudaLaunchKernelEx(&cfg, attention_bf16_kernel<64>, a);
  return cudaErrorInvalidValue;
}

cudaError_t launch_attention_f32(const AttnArgs& x, cudaStream_t s) {
  const long long nrows = static_cast<long long>(x.B) * x.Lb * x.Hq;
  const int threads = 128;
  const int blocks = static_cast<int>((nrows * 32 + threads - 1) / threads);
  attention_f32_kernel<<<blocks, threads, 0, s>>>(
      static_cast<const float*>(x.q), static_cast<const float*>(x.k_blk),
      static_cast<const float*>(x.v_blk), static_cast<float*>(x.k_cache),
      static_cast<float*>(x.v_cache), x.ctx, static_cast<float*>(x.out), x.B, x.Lb, x.Hq, x.Hkv,
      x.D, x.Cmax, 1.f / sqrtf(static_cast<float>(x.D)), x.status);
  return cudaGetLastError();
}

}  // namespace rv
