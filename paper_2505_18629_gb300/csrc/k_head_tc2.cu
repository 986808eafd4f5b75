// LM head of the verify step on CTA pairs (tcgen05 cta_group::2), for the
// larger pair counts where one SM per vocab tile is limited by its shared
// memory rather than by HBM:
//
//   acc[v][c] = sum_k W[v][k] * hsel[c][k]   over 256 vocab rows v per pair tile
//   (128 per CTA) and the gathered hidden rows c of one pair chunk: o_i and
//   o_{m+i-1} of Alg. 1,
//
// followed by the online log-softmax / fusion epilogue (Eq. 2), so that no
// logit is written to memory.  One MMA of the pair (M = 256, issued by the
// even CTA) reads the A operand from each CTA's own shared memory (its 128
// weight rows) and the B operand split across the two (the even CTA holds the
// original rows, the odd CTA the reflective rows), so each SM stages its
// weight rows and only half of the hidden rows; every CTA gets its own 128-row
// accumulator in its TMEM.
//
// Sub-groups.  The pairs of a chunk are split into H sub-groups of Ph[h]
// pairs; sub-group h has its own accumulator of 2 Ph[h] columns (o of its
// pairs, then o'), one MMA per 16-wide K step each.  Every sub-group reads the
// same weight stage, so a chunk of up to 160 pairs (H = 2) streams each weight
// tile into shared memory once.  Accumulator slots:
//   ring  (H = 1, up to 128 pairs): R equal slots in turn, R >= 2, so a tile
//         never waits for the epilogue of the tile before;
//   split (H = 2, 129..160 pairs): two tiles' 2 x 2 Pc columns exceed TMEM's
//         512, so sub-group 0 is small (Ph[0] = Pc - Ph[1], Ph[1] =
//         256 - Pc pairs) and sits in one fixed slot, sub-group 1 alternates
//         between two slots (2 Ph[0] + 4 Ph[1] = 512 columns).  The next
//         tile's sub-group 1 starts at once; its sub-group 0 waits only until
//         the epilogue has loaded this tile's sub-group 0 (at most three
//         groups per warp, freed as soon as they are in registers).
//
// Per CTA, warp-specialised:
//   warp 0      TMA producer: weight tile [128 x 128] + this CTA's hidden rows
//               of every sub-group per stage (each as two 64-wide boxes); both
//               CTAs' copies complete on the even CTA's full barrier
//   warp 1      TMEM owner (both CTAs); in the even CTA it also issues the
//               pair's MMAs from one thread, and its commits release the stage
//               and fill the accumulator slots in both CTAs
//   warps 2..   epilogue, H2_WPQ warps per TMEM lane quadrant
// The pair streams a static range of 256-row vocab tiles; the weight streams
// from HBM once per chunk (evict-first), the hidden rows are re-read from L2.
//
// Epilogue.  tcgen05.ld.16x256b gives lane l of a warp the rows l/4 + 8i
// (i = 0..3, two loads) and the columns 2(l%4), 2(l%4)+1 of an 8-column group,
// so a column's 32 rows lie in 4 registers of 8 lanes: the max / sum-exp /
// argmax reductions over the vocab rows take 3 register steps and 3 shuffle
// levels, with every lane busy.  The tile results are folded into running
// statistics that live in registers: in a group of 8 pairs, lane l keeps, for
// column 2(l%4) + ((l/4) & 1), the statistics of quantity l/8 (o with its
// entropy term, o', z, or the best z over v != x_i), one fold per lane and
// group.  At the end they go to per-quadrant tables in shared memory (over
// the drained pipeline stages) and are merged into the CTA's partials.
#include <cfloat>
#include <climits>

#include "head_epilogue.cuh"
#include "rv_device.cuh"
#include "rv_kernels.h"

namespace rv {

namespace {

constexpr int H2_BM = 128;  // vocab rows per CTA per pair tile
constexpr int H2_BK = 128;  // K per stage: two 64-wide swizzled halves, 8 MMAs per sub-group
constexpr uint32_t H2_A_HALF = H2_BM * 64 * 2;      // 16 KB
constexpr uint32_t H2_A_BYTES = 2 * H2_A_HALF;      // 32 KB
#ifndef RV_HEAD2_WPQ
#define RV_HEAD2_WPQ 3
#endif
constexpr int H2_WPQ = RV_HEAD2_WPQ;  // epilogue warps per TMEM lane quadrant (3: measured best at 8B B=16)
constexpr int H2_EPI = 4 * H2_WPQ;
constexpr int H2_THREADS = 64 + 32 * H2_EPI;
// groups one epilogue warp may own: of 2 sub-groups of up to 10 groups (160
// pairs), or of 1 of up to 16 groups (128 pairs, or 256 pre-blended pairs in
// groups of 16)
constexpr int h2_cdiv(int a, int b) { return (a + b - 1) / b; }
constexpr int H2_MAX_OWN = 2 * h2_cdiv(10, H2_WPQ) > h2_cdiv(16, H2_WPQ) ? 2 * h2_cdiv(10, H2_WPQ)
                                                                        : h2_cdiv(16, H2_WPQ);
constexpr int H2_MAX_H = 2;     // sub-groups per tile
constexpr int H2_MAX_R = 4;     // accumulator slots

struct Head2Params {
  int V, n_kb;
  int H, R, split;      // sub-groups per tile, slots, slot rule (0 ring, 1 split)
  int Ph[H2_MAX_H];     // pairs of sub-group h (its columns: 2 Ph, or Ph pre-blended)
  int pb[H2_MAX_H];     // its first pair (and first B row in each CTA) within the chunk
  int scol[H2_MAX_R];   // first TMEM column of each slot
  int b_rows;           // B rows per CTA per stage (the chunk's half)
  int Pcp, Pc, P, stages, gamma;
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
  float2* zsub;  // [P][n_sub] subtile (max z, sum exp((z - max) / T)), or null
  int n_sub;
  float inv_t;
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

// 16 lanes x 256 bit: lane l of the warp gets rows (base + l/4) and
// (base + 8 + l/4), columns 2(l%4) and 2(l%4)+1 of the 8 columns at `taddr`:
// v = {row l/4: col, col+1; row 8 + l/4: col, col+1}.
__device__ __forceinline__ void tmem_ld_16x256b(uint32_t taddr, uint32_t* v) {
  asm volatile("tcgen05.ld.sync.aligned.16x256b.x1.b32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3])
               : "r"(taddr));
}
// .x2: the same for columns 8..15 in v[4..7].
__device__ __forceinline__ void tmem_ld_16x256b_x2(uint32_t taddr, uint32_t* v) {
  asm volatile("tcgen05.ld.sync.aligned.16x256b.x2.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
               : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]),
                 "=r"(v[6]), "=r"(v[7])
               : "r"(taddr));
}

// After tcgen05.wait::ld: makes every later use of `v` depend on this point,
// so that no use of a loaded register is scheduled before the wait.
__device__ __forceinline__ void after_ld(uint32_t (&v)[16]) {
#pragma unroll
  for (int i = 0; i < 16; ++i) asm volatile("" : "+r"(v[i]));
}

__device__ __forceinline__ void shfl_best(float& bv, int& bi, int off) {
  const float ov = __shfl_xor_sync(0xffffffffu, bv, off);
  const int oi = __shfl_xor_sync(0xffffffffu, bi, off);
  if (ov > bv || (ov == bv && oi < bi)) {
    bv = ov;
    bi = oi;
  }
}

struct TileOut {
  float m, s, t;
};

// Where a group's fused logits go besides the statistics (sampling modes; the
// pointers are offset to the chunk's first pair, null when unused): every z
// (speculative sampling), or one (max z, sum exp((z - max) / T)) per pair and
// 32-row subtile (sampled exact match).
struct ZSink {
  float* z;
  float2* sub;
  int n_sub;
  float inv_t;
};

// Stores at the draft row of each of the lane's columns: `x[j]` (this lane's
// pair of column j) may fall on one of its rows rq + 8i; at most one (unique
// writer over the CTA).  Rows at or beyond V (a partial last tile) hold zeros;
// a draft there is out of range and its gathered values are never read.
template <int NC>
__device__ __forceinline__ void gather_draft_rows(const float* o, const float* r, const float* z,
                                                  const int* x, int row0, float* gathered,
                                                  int gpair_lane, const int* col_pair) {
#pragma unroll
  for (int j = 0; j < NC; ++j) {
    const int d = x[j] - row0;
    if (static_cast<unsigned>(d) < 32u && (d & 7) == 0) {
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        if (d == 8 * i) {
          float* gx = gathered + (gpair_lane + col_pair[j]) * GATHER_FIELDS;
          if (o != nullptr) {
            gx[0] = o[NC * i + j];
            gx[1] = r[NC * i + j];
          }
          gx[2] = z[NC * i + j];
        }
      }
    }
  }
}

// One group of eight pairs of the two-distribution head: lo = o and lr = o'
// as loaded by two tcgen05.ld.16x256b each (rows +0 / +16 of this warp's
// quadrant); x[j] the draft of the lane's column j (-1: none).  Rows at or
// beyond V count as -inf.  Forms z = (1-a) o + a o' (Eq. 2), stores o, o', z
// at the draft row of each pair and, when asked, z itself; returns this
// lane's tile statistics: quantity lane / 8 (o, o', z, best z over v != x_i)
// of column 2(lane%4) + ((lane/4)&1).
template <bool SUB>
__device__ __forceinline__ TileOut group8_fused(const uint32_t* lo, const uint32_t* lr,
                                                int v_row0, int V, float alpha, float beta,
                                                const int (&x)[2], int gpair, int npairs,
                                                float* gathered, const ZSink& zs, int lane) {
  const int c4 = lane & 3, rq = lane >> 2;
  const int row0 = v_row0 + rq;  // this lane's first row; the others are +8, +16, +24
  float o[8], r[8], z[8];
  // element 2i + j: row row0 + 8i, column 2 c4 + j
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    o[k] = __uint_as_float(lo[k]);
    r[k] = __uint_as_float(lr[k]);
    z[k] = fmaf(alpha, r[k], beta * o[k]);
  }
  if (v_row0 + 32 > V) {  // a partial last tile (warp-uniform)
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      if (row0 + 8 * i >= V) {
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          o[2 * i + j] = NEG_INF;
          r[2 * i + j] = NEG_INF;
          z[2 * i + j] = NEG_INF;
        }
      }
    }
  }
  {
    const int col_pair[2] = {2 * c4, 2 * c4 + 1};
    gather_draft_rows<2>(o, r, z, x, row0, gathered, gpair, col_pair);
  }
  if (zs.z != nullptr) {  // speculative sampling only (uniform)
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int v = row0 + 8 * i;
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        const int pj = gpair + 2 * c4 + j;
        if (v < V && pj < npairs) zs.z[static_cast<long long>(pj) * V + v] = z[2 * i + j];
      }
    }
  }
  float mo[2], mr[2], mz[2];
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    mo[j] = fmaxf(fmaxf(o[j], o[2 + j]), fmaxf(o[4 + j], o[6 + j]));
    mr[j] = fmaxf(fmaxf(r[j], r[2 + j]), fmaxf(r[4 + j], r[6 + j]));
    mz[j] = fmaxf(fmaxf(z[j], z[2 + j]), fmaxf(z[4 + j], z[6 + j]));
  }
#pragma unroll
  for (int off = 4; off < 32; off <<= 1) {
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      mo[j] = fmaxf(mo[j], __shfl_xor_sync(0xffffffffu, mo[j], off));
      mr[j] = fmaxf(mr[j], __shfl_xor_sync(0xffffffffu, mr[j], off));
      mz[j] = fmaxf(mz[j], __shfl_xor_sync(0xffffffffu, mz[j], off));
    }
  }
  float so[2], to[2], sr[2], sz[2], bv[2];
  int bi[2];
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    // all rows -inf (a tile past the vocab end): empty sums, no NaN
    const float nmo = mo[j] == NEG_INF ? 0.f : -mo[j] * LOG2E;
    const float nmr = mr[j] == NEG_INF ? 0.f : -mr[j] * LOG2E;
    const float nmz = mz[j] == NEG_INF ? 0.f : -mz[j] * LOG2E;
    so[j] = 0.f;
    to[j] = 0.f;
    sr[j] = 0.f;
    sz[j] = 0.f;
    bv[j] = NEG_INF;
    bi[j] = INT_MAX;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int k = 2 * i + j;
      const float eo = ex2_approx(fmaf(o[k], LOG2E, nmo));
      so[j] += eo;
      to[j] += eo == 0.f ? 0.f : eo * (o[k] - mo[j]);
      sr[j] += ex2_approx(fmaf(r[k], LOG2E, nmr));
      sz[j] += ex2_approx(fmaf(z[k], LOG2E, nmz));
      const int v = row0 + 8 * i;  // rows in increasing order: strict > keeps the lowest
      const bool better = v != x[j] && z[k] > bv[j];
      bv[j] = better ? z[k] : bv[j];
      bi[j] = better ? v : bi[j];
    }
  }
#pragma unroll
  for (int off = 4; off < 32; off <<= 1) {
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      so[j] += __shfl_xor_sync(0xffffffffu, so[j], off);
      to[j] += __shfl_xor_sync(0xffffffffu, to[j], off);
      sr[j] += __shfl_xor_sync(0xffffffffu, sr[j], off);
      sz[j] += __shfl_xor_sync(0xffffffffu, sz[j], off);
      shfl_best(bv[j], bi[j], off);
    }
  }
  if (SUB && v_row0 < V) {  // sampled exact match only (uniform)
    float sT[2] = {sz[0], sz[1]};         // T = 1: the sums above
    if (zs.inv_t != 1.f) {
      const float k2 = LOG2E * zs.inv_t;
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        sT[j] = 0.f;
#pragma unroll
        for (int i = 0; i < 4; ++i) sT[j] += ex2_approx((z[2 * i + j] - mz[j]) * k2);
      }
#pragma unroll
      for (int off = 4; off < 32; off <<= 1) {
#pragma unroll
        for (int j = 0; j < 2; ++j) sT[j] += __shfl_xor_sync(0xffffffffu, sT[j], off);
      }
    }
    if (rq == 0) {
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        const int pj = gpair + 2 * c4 + j;
        if (pj < npairs)
          zs.sub[static_cast<long long>(pj) * zs.n_sub + (v_row0 >> 5)] = make_float2(mz[j], sT[j]);
      }
    }
  }
  const int qn = rq >> 1;
  const bool j1 = (rq & 1) != 0;
  const float M_o = j1 ? mo[1] : mo[0], M_r = j1 ? mr[1] : mr[0], M_z = j1 ? mz[1] : mz[0];
  const float S_o = j1 ? so[1] : so[0], S_r = j1 ? sr[1] : sr[0], S_z = j1 ? sz[1] : sz[0];
  const float B_v = j1 ? bv[1] : bv[0];
  const int B_i = j1 ? bi[1] : bi[0];
  TileOut out;
  out.m = qn == 0 ? M_o : qn == 1 ? M_r : qn == 2 ? M_z : B_v;
  out.s = qn == 0 ? S_o : qn == 1 ? S_r : qn == 2 ? S_z : __int_as_float(B_i);
  out.t = j1 ? to[1] : to[0];
  return out;
}

// One group of sixteen pairs of the pre-blended head (the columns are z):
// la / lb as loaded by tcgen05.ld.16x256b.x2 at rows +0 / +16; lane l has
// rows l/4 + 8i and columns 2(l%4) + (jj & 1) + 8 (jj >> 1), jj = 0..3, with
// drafts x[jj].  Returns quantity l/16 (z statistics, best z over v != x_i)
// of column jj = (l/4) & 3.
template <bool SUB>
__device__ __forceinline__ TileOut group16_z(const uint32_t* la, const uint32_t* lb, int v_row0,
                                             int V, const int (&x)[4], int gpair, int npairs,
                                             float* gathered, const ZSink& zs, int lane) {
  const int c4 = lane & 3, rq = lane >> 2;
  const int row0 = v_row0 + rq;
  float z[16];  // element 4i + jj
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint32_t* src = i < 2 ? la : lb;
    const int ii = i & 1;  // .x2 registers: {row +0: c, c+1; row +8: c, c+1; the same 8 columns on}
#pragma unroll
    for (int jj = 0; jj < 4; ++jj) z[4 * i + jj] = __uint_as_float(src[4 * (jj >> 1) + 2 * ii + (jj & 1)]);
  }
  if (v_row0 + 32 > V) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      if (row0 + 8 * i >= V) {
#pragma unroll
        for (int jj = 0; jj < 4; ++jj) z[4 * i + jj] = NEG_INF;
      }
    }
  }
  {
    const int col_pair[4] = {2 * c4, 2 * c4 + 1, 8 + 2 * c4, 9 + 2 * c4};
    gather_draft_rows<4>(nullptr, nullptr, z, x, row0, gathered, gpair, col_pair);
  }
  if (zs.z != nullptr) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int v = row0 + 8 * i;
#pragma unroll
      for (int jj = 0; jj < 4; ++jj) {
        const int pj = gpair + 2 * c4 + (jj & 1) + 8 * (jj >> 1);
        if (v < V && pj < npairs) zs.z[static_cast<long long>(pj) * V + v] = z[4 * i + jj];
      }
    }
  }
  float mz[4], sz[4], bv[4];
  int bi[4];
#pragma unroll
  for (int jj = 0; jj < 4; ++jj)
    mz[jj] = fmaxf(fmaxf(z[jj], z[4 + jj]), fmaxf(z[8 + jj], z[12 + jj]));
#pragma unroll
  for (int off = 4; off < 32; off <<= 1) {
#pragma unroll
    for (int jj = 0; jj < 4; ++jj) mz[jj] = fmaxf(mz[jj], __shfl_xor_sync(0xffffffffu, mz[jj], off));
  }
#pragma unroll
  for (int jj = 0; jj < 4; ++jj) {
    const float nmz = mz[jj] == NEG_INF ? 0.f : -mz[jj] * LOG2E;
    sz[jj] = 0.f;
    bv[jj] = NEG_INF;
    bi[jj] = INT_MAX;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float zz = z[4 * i + jj];
      sz[jj] += ex2_approx(fmaf(zz, LOG2E, nmz));
      const int v = row0 + 8 * i;
      const bool better = v != x[jj] && zz > bv[jj];
      bv[jj] = better ? zz : bv[jj];
      bi[jj] = better ? v : bi[jj];
    }
  }
#pragma unroll
  for (int off = 4; off < 32; off <<= 1) {
#pragma unroll
    for (int jj = 0; jj < 4; ++jj) {
      sz[jj] += __shfl_xor_sync(0xffffffffu, sz[jj], off);
      shfl_best(bv[jj], bi[jj], off);
    }
  }
  if (SUB && v_row0 < V) {  // sampled exact match only (uniform)
    float sT[4] = {sz[0], sz[1], sz[2], sz[3]};
    if (zs.inv_t != 1.f) {
      const float k2 = LOG2E * zs.inv_t;
#pragma unroll
      for (int jj = 0; jj < 4; ++jj) {
        sT[jj] = 0.f;
#pragma unroll
        for (int i = 0; i < 4; ++i) sT[jj] += ex2_approx((z[4 * i + jj] - mz[jj]) * k2);
      }
#pragma unroll
      for (int off = 4; off < 32; off <<= 1) {
#pragma unroll
        for (int jj = 0; jj < 4; ++jj) sT[jj] += __shfl_xor_sync(0xffffffffu, sT[jj], off);
      }
    }
    if (rq == 0) {
#pragma unroll
      for (int jj = 0; jj < 4; ++jj) {
        const int pj = gpair + 2 * c4 + (jj & 1) + 8 * (jj >> 1);
        if (pj < npairs)
          zs.sub[static_cast<long long>(pj) * zs.n_sub + (v_row0 >> 5)] =
              make_float2(mz[jj], sT[jj]);
      }
    }
  }
  const int sel = rq & 3, qn = rq >> 2;
  float M = mz[0], S = sz[0], Bv = bv[0];
  int I = bi[0];
#pragma unroll
  for (int jj = 1; jj < 4; ++jj) {
    M = sel == jj ? mz[jj] : M;
    S = sel == jj ? sz[jj] : S;
    Bv = sel == jj ? bv[jj] : Bv;
    I = sel == jj ? bi[jj] : I;
  }
  TileOut out;
  out.m = qn == 0 ? M : Bv;
  out.s = qn == 0 ? S : __int_as_float(I);
  out.t = 0.f;
  return out;
}

}  // namespace

// Slot of sub-group h in the pair's t-th tile, and how many times that slot
// was used before (the parity of its barriers).  Ring: the R slots in turn;
// split: sub-group 0 in slot 0, sub-group 1 in slots 1 and 2 by turns.
__device__ __forceinline__ int h2_slot(const Head2Params& p, int t, int h, int& uses) {
  if (p.split) {
    if (h == 0) {
      uses = t;
      return 0;
    }
    uses = t >> 1;
    return 1 + (t & 1);
  }
  const int u = t * p.H + h;
  uses = u / p.R;
  return u - uses * p.R;
}

// Running statistics of the epilogue lane: one (m, s, t) per owned group, in
// registers.  The group loop stays rolled (unrolled over the groups, its body
// would not fit the instruction cache of the eight epilogue warps), so the
// state rotates: the current group's is always at index 0, and after a tile
// the ring has turned exactly once.
struct LaneStats {
  float m[H2_MAX_OWN], s[H2_MAX_OWN], t[H2_MAX_OWN];
  __device__ __forceinline__ void rotate() {
    const float m0 = m[0], s0 = s[0], t0 = t[0];
#pragma unroll
    for (int i = 0; i + 1 < H2_MAX_OWN; ++i) {
      m[i] = m[i + 1];
      s[i] = s[i + 1];
      t[i] = t[i + 1];
    }
    m[H2_MAX_OWN - 1] = m0;
    s[H2_MAX_OWN - 1] = s0;
    t[H2_MAX_OWN - 1] = t0;
  }
  // Fold the tile's (M, S, T) into entry 0 without branches.  Argmax lanes:
  // the larger value, the lower row on ties (rows kept as int bits in s).
  // The others: running (m, s, t) with s = sum exp(x - m) and
  // t = sum exp(x - m) (x - m) (t for o only; the entropy is log s - t / s),
  // merged with one exponential: the side whose maximum is kept is scaled
  // by exactly 1.
  __device__ __forceinline__ void fold0(bool best, const TileOut& o) {
    const float m0 = m[0], s0 = s[0], t0 = t[0];
    const bool take = o.m > m0 || (o.m == m0 && __float_as_int(o.s) < __float_as_int(s0));
    const float mn = fmaxf(m0, o.m);
    const bool keep = m0 >= o.m;
    const float f = ex2_approx(__fmul_rn(keep ? o.m - m0 : m0 - o.m, LOG2E));
    const float a = keep ? 1.f : f, c = keep ? f : 1.f;
    const float tn = (a == 0.f ? 0.f : a * (t0 + (m0 - mn) * s0)) +
                     (c == 0.f ? 0.f : c * (o.t + (o.m - mn) * o.s));
    const float sn = __fmaf_rn(s0, a, __fmul_rn(o.s, c));
    const bool empty = mn == NEG_INF;  // nothing seen yet on either side
    m[0] = best ? (take ? o.m : m0) : (empty ? m0 : mn);
    s[0] = best ? (take ? o.s : s0) : (empty ? s0 : sn);
    t[0] = best ? t0 : (empty ? t0 : tn);
  }
};

// SUB: the epilogue also stores the subtile sums of sampled exact match (its
// own instantiation, so that the other modes carry none of its registers).
template <bool ZONLY, bool SUB>
__global__ void __launch_bounds__(H2_THREADS, 1)
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
  // commit mask: this pair's two CTAs (the stage release and the accumulators)
  const uint16_t pair_mask = static_cast<uint16_t>(3u << (crank & ~1u));
  const int pair = blockIdx.x >> 1;
  const int chunk = blockIdx.y;
  const int slot_id = blockIdx.x;  // partial slot within the chunk
  const int S = p.stages, H = p.H;
  // this CTA's rows of B per stage: half of every sub-group's columns (the
  // original or the reflective rows; for the pre-blended head the first or
  // second half of the blended rows)
  const uint32_t b_rows = static_cast<uint32_t>(p.b_rows);
  const uint32_t b_half = b_rows * 128u;  // one 64-wide K half of this CTA's B
  const uint32_t b_bytes = 2u * b_half;

  const uint32_t a_tiles = base;
  const uint32_t b_tiles = base + S * H2_A_BYTES;
  const uint32_t bars = b_tiles + S * b_bytes;
  auto full_bar = [&](int s) { return bars + 8u * s; };
  auto empty_bar = [&](int s) { return bars + 8u * (S + s); };
  const uint32_t accf0 = bars + 8u * (2 * S);   // slot filled (MMA -> epilogue)
  const uint32_t acce0 = accf0 + 8u * H2_MAX_R;  // slot read (epilogue -> MMA)
  const uint32_t drain_bar = acce0 + 8u * H2_MAX_R;
  const uint32_t misc = (drain_bar + 8u + 15u) & ~15u;
  uint32_t* const tmem_slot = reinterpret_cast<uint32_t*>(gbase + (misc - base));
  volatile int* const abort_flag = reinterpret_cast<volatile int*>(gbase + (misc - base) + 4);
  int* const s_drafts = reinterpret_cast<int*>(gbase + (misc - base) + 16);
  // statistics tables [4 quadrants][Pcp][HEAD_STAT_STRIDE] over the drained
  // pipeline stages, written once at the end
  float* const stats = reinterpret_cast<float*>(gbase);

  const int pair0 = chunk * p.Pc;
  const int npairs = min(p.Pc, p.P - pair0);
  const int pt0 = static_cast<int>(static_cast<long long>(pair) * p.n_ptiles / p.pair_slots);
  const int pt1 = static_cast<int>(static_cast<long long>(pair + 1) * p.n_ptiles / p.pair_slots);

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(full_bar(s), 1);   // the even CTA's expect-tx; both CTAs' bytes
      mbar_init(empty_bar(s), 1);  // the pair's MMA commit
    }
    for (int k = 0; k < H2_MAX_R; ++k) {
      mbar_init(accf0 + 8u * k, 1);
      mbar_init(acce0 + 8u * k, 2 * H2_EPI);  // the epilogue warps of both CTAs
    }
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
    for (int j = e; j < MAX_ZPAIRS_PER_CHUNK; j += H2_EPI * 32)
      s_drafts[j] = (j < npairs) ? pair_draft(p.drafts, pair0 + j, p.gamma) : -1;
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
      const int hrow = (2 * chunk + static_cast<int>(rank)) * static_cast<int>(b_rows);
      for (int pt = pt0; pt < pt1 && ok; ++pt) {
        const int v0 = pt * 2 * H2_BM + static_cast<int>(rank) * H2_BM;
        for (int kb = 0; kb < p.n_kb; ++kb) {
          if (!mbar_wait(empty_bar(s), ph ^ 1u, abort_flag, p.status)) {
            ok = false;
            break;
          }
          if (leader) mbar_arrive_expect_tx(full_bar(s), 2u * (H2_A_BYTES + b_bytes));
          const uint32_t fb = mapa_shared(full_bar(s), leader_rank);
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
      const int cols0 = p.zonly ? p.Ph[0] : 2 * p.Ph[0];
      const int cols1 = p.zonly ? p.Ph[1] : 2 * p.Ph[1];
      const uint32_t idesc0 = idesc_bf16_f32(2 * H2_BM, cols0);
      const uint32_t idesc1 = H > 1 ? idesc_bf16_f32(2 * H2_BM, cols1) : idesc0;
      // descriptors of stage 0; stage s adds s * bytes / 16 to the start field
      const uint64_t ad0 = sw128_kmajor_desc(a_tiles), bd0 = sw128_kmajor_desc(b_tiles);
      const uint32_t a_step = H2_A_BYTES >> 4, b_step = b_bytes >> 4;
      const uint32_t a_hstep = H2_A_HALF >> 4, b_hstep = b_half >> 4;
      const uint32_t b_sub1 = (static_cast<uint32_t>(p.pb[1]) * 128u) >> 4;  // sub-group 1's rows
      int s = 0;
      uint32_t ph = 0;
      bool ok = true;
      for (int pt = pt0, t = 0; pt < pt1 && ok; ++pt, ++t) {
        uint32_t d0 = 0u, d1 = 0u;
        for (int kb = 0; kb < p.n_kb && ok; ++kb) {
          if (!mbar_wait(full_bar(s), ph, abort_flag, p.status)) {
            ok = false;
            break;
          }
          const uint64_t ad = ad0 + static_cast<uint32_t>(s) * a_step;
          const uint64_t bd = bd0 + static_cast<uint32_t>(s) * b_step;
#pragma unroll
          for (int i = 0; i < H2_MAX_H; ++i) {
            if (i >= H) break;
            // split: sub-group 1 first, its slot is free; sub-group 0's may
            // still be read by the epilogue of the tile before
            const int h = p.split ? H - 1 - i : i;
            if (kb == 0) {
              // the slot of this sub-group must have been read by the epilogue
              int uses;
              const int sl = h2_slot(p, t, h, uses);
              if (!mbar_wait(acce0 + 8u * sl, (uses & 1) ^ 1, abort_flag, p.status)) {
                ok = false;
                break;
              }
              tc_fence_after();
              const uint32_t d = tmem_base + static_cast<uint32_t>(p.scol[sl]);
              if (h == 0)
                d0 = d;
              else
                d1 = d;
            }
            tc2_mma_stage8(h == 0 ? d0 : d1, ad, h == 0 ? bd : bd + b_sub1, a_hstep, b_hstep,
                           h == 0 ? idesc0 : idesc1, kb != 0 ? 1u : 0u);
          }
          tc2_commit(empty_bar(s), pair_mask);
          if (++s == S) {
            s = 0;
            ph ^= 1u;
          }
        }
        if (ok) {
          for (int h = 0; h < H; ++h) {
            int uses;
            tc2_commit(accf0 + 8u * h2_slot(p, t, h, uses), pair_mask);
          }
        }
      }
      // every MMA issued must be complete before TMEM is released
      tc2_commit(drain_bar, static_cast<uint16_t>(1u << crank));
      drain_wait(drain_bar, 0);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ epilogue (both CTAs)
    const int q = warp & 3;          // TMEM lane quadrant this warp may access
    const int kq = (warp - 2) >> 2;  // this warp's index within its quadrant
    const float beta = 1.f - p.alpha;
    constexpr int gsz = ZONLY ? 16 : 8;  // pairs per group
    // this warp's groups: g = kq, kq + WPQ, ... of every sub-group, in order
    const int ng0 = p.Ph[0] / gsz, ng1 = H > 1 ? p.Ph[1] / gsz : 0;
    const int cnt0 = kq < ng0 ? (ng0 - kq + H2_WPQ - 1) / H2_WPQ : 0;
    const int cnt1 = kq < ng1 ? (ng1 - kq + H2_WPQ - 1) / H2_WPQ : 0;
    const int n_mine = cnt0 + cnt1;
    auto cnt_of = [&](int h) { return h == 0 ? cnt0 : cnt1; };
    LaneStats st;
    const int qn = ZONLY ? (lane >> 4) : (lane >> 3);
    const bool is_best = ZONLY ? qn == 1 : qn == 3;
#pragma unroll
    for (int i = 0; i < H2_MAX_OWN; ++i) {
      st.m[i] = NEG_INF;
      st.s[i] = is_best ? __int_as_float(INT_MAX) : 0.f;
      st.t[i] = 0.f;
    }
    const uint32_t lane_q = static_cast<uint32_t>(q * 32) << 16;
    float* const gathered = p.gathered + static_cast<long long>(pair0) * GATHER_FIELDS;
    const ZSink zs{p.zout ? p.zout + static_cast<long long>(pair0) * p.V : nullptr,
                   p.zsub ? p.zsub + static_cast<long long>(pair0) * p.n_sub : nullptr, p.n_sub,
                   p.inv_t};
    bool ok = true;
    int slot0 = 0, slot1 = 0, phase0 = 0, phase1 = 0;  // of sub-groups 0 and 1 this tile
    auto slot_of = [&](int h) { return h == 0 ? slot0 : slot1; };
    auto wait_slot = [&](int h) -> bool {
      const bool w = mbar_wait(accf0 + 8u * slot_of(h), h == 0 ? phase0 : phase1, abort_flag,
                               p.status);
      tc_fence_after();
      return __all_sync(0xffffffffu, w);
    };
    auto release_slot = [&](int h) {
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(mapa_shared(acce0 + 8u * slot_of(h), leader_rank));
    };
    // first TMEM column of group g of sub-group h of the current tile
    auto tcol = [&](int h, int g) -> uint32_t {
      return tmem_base + lane_q + static_cast<uint32_t>(p.scol[slot_of(h)] + g * gsz);
    };
    // o' of sub-group h starts Ph[h] columns after its o
    auto load_group = [&](uint32_t t0, int h, uint32_t* b) {
      if (ZONLY) {
        tmem_ld_16x256b_x2(t0, b);
        tmem_ld_16x256b_x2(t0 + (16u << 16), b + 8);
      } else {
        const uint32_t po = static_cast<uint32_t>(h == 0 ? p.Ph[0] : p.Ph[1]);
        tmem_ld_16x256b(t0, b);
        tmem_ld_16x256b(t0 + (16u << 16), b + 4);
        tmem_ld_16x256b(t0 + po, b + 8);
        tmem_ld_16x256b(t0 + po + (16u << 16), b + 12);
      }
    };
    // drafts of this lane's columns of group (h, g)
    constexpr int NC = ZONLY ? 4 : 2;
    auto load_drafts = [&](int h, int g, int (&x)[NC]) {
      const int c4 = lane & 3;
      const int gp = (h == 0 ? 0 : p.pb[1]) + g * gsz;
#pragma unroll
      for (int j = 0; j < NC; ++j)
        x[j] = s_drafts[gp + 2 * c4 + (j & 1) + 8 * (j >> 1)];  // -1: no draft (or padding)
    };
    for (int pt = pt0, t = 0; pt < pt1 && ok; ++pt, ++t) {
      // the slots and parities the MMA issuer uses for this tile
      {
        int u0, u1 = 0;
        slot0 = h2_slot(p, t, 0, u0);
        slot1 = H > 1 ? h2_slot(p, t, 1, u1) : 0;
        phase0 = u0 & 1;
        phase1 = u1 & 1;
      }
      const int v_row0 = pt * 2 * H2_BM + static_cast<int>(rank) * H2_BM + q * 32;
      // a sub-group with none of this warp's groups: its slot's barrier still
      // counts this warp, once the slot holds this tile's accumulator
      for (int h = 0; h < H && ok; ++h) {
        if (cnt_of(h) == 0) {
          ok = wait_slot(h);
          if (ok) release_slot(h);
        }
      }
      if (!ok) break;
      if (n_mine == 0) continue;
      uint32_t cb[16], nb[16];
      int cx[NC], nx[NC];
      int h = cnt0 > 0 ? 0 : 1, gi = 0;  // sub-group and index within it of group idx
      if (!wait_slot(h)) {
        ok = false;
        break;
      }
      load_group(tcol(h, kq), h, cb);
      load_drafts(h, kq, cx);
      tmem_ld_wait();
      after_ld(cb);
      bool freed = false;  // h's slot released already
#pragma unroll 1
      for (int idx = 0; idx < n_mine; ++idx) {
        const int g = gi * H2_WPQ + kq;
        // the next group
        int nh = h, ngi = gi + 1;
        if (ngi == cnt_of(h)) {
          ++nh;
          ngi = 0;
        }
        const bool more = idx + 1 < n_mine;
        // h's slot is released as soon as all of this warp's groups of h are
        // in registers, before they are reduced, so that the MMAs of the next
        // tile wait as little as possible: now, if this group is h's last ...
        if ((!more || nh != h) && !freed) release_slot(h);
        if (more && nh != h && !wait_slot(nh)) {
          ok = false;
          break;
        }
        if (more) {  // lands while this group is reduced
          load_group(tcol(nh, ngi * H2_WPQ + kq), nh, nb);
          load_drafts(nh, ngi * H2_WPQ + kq, nx);
        }
        // ... or once the next one, h's last, has landed
        if (more && nh == h && ngi + 1 == cnt_of(h)) {
          tmem_ld_wait();
          release_slot(h);
          freed = true;
        }
        const int gpair = (h == 0 ? 0 : p.pb[1]) + g * gsz;
        TileOut t;
        if constexpr (ZONLY)
          t = group16_z<SUB>(cb, cb + 8, v_row0, p.V, cx, gpair, npairs, gathered, zs, lane);
        else
          t = group8_fused<SUB>(cb, cb + 8, v_row0, p.V, p.alpha, beta, cx, gpair, npairs, gathered,
                           zs, lane);
        st.fold0(is_best, t);
        st.rotate();
        tmem_ld_wait();
        after_ld(nb);
#pragma unroll
        for (int k = 0; k < 16; ++k) cb[k] = nb[k];
#pragma unroll
        for (int j = 0; j < NC; ++j) cx[j] = nx[j];
        if (nh != h) freed = false;
        h = nh;
        gi = ngi;
      }
      // back to the tile-start alignment of the ring
#pragma unroll 1
      for (int k = n_mine; k < H2_MAX_OWN; ++k) st.rotate();
    }
    // every accumulator has been read (all MMAs of the pair complete), so the
    // pipeline stages of this CTA are no longer written or read: the tables go
    // over them
    named_bar_sync(1, H2_EPI * 32);
    const int c4 = lane & 3, rq = lane >> 2;
    const int tab = p.Pcp;
#pragma unroll
    for (int idx = 0; idx < H2_MAX_OWN; ++idx) {
      if (idx >= n_mine) break;
      const int h = idx < cnt0 ? 0 : 1;
      const int g = (idx < cnt0 ? idx : idx - cnt0) * H2_WPQ + kq;
      const int p0 = h == 0 ? 0 : p.pb[1];
      int pj;
      if (ZONLY) {
        const int jj = rq & 3;
        pj = p0 + g * 16 + 2 * c4 + (jj & 1) + 8 * (jj >> 1);
      } else {
        pj = p0 + g * 8 + 2 * c4 + (rq & 1);
      }
      if (pj < npairs) {
        float* d = stats + (q * tab + pj) * HEAD_STAT_STRIDE;
        if (is_best) {
          d[ST_BEST_V] = st.m[idx];
          d[ST_BEST_I] = st.s[idx];
        } else if (ZONLY) {
          d[ST_M_Z] = st.m[idx];
          d[ST_S_Z] = st.s[idx];
          d[ST_M_O] = NEG_INF;  // no separate o / o' in this head
          d[ST_S_O] = 0.f;
          d[ST_T_O] = 0.f;
          d[ST_M_R] = NEG_INF;
          d[ST_S_R] = 0.f;
        } else if (qn == 0) {
          d[ST_M_O] = st.m[idx];
          d[ST_S_O] = st.s[idx];
          d[ST_T_O] = st.t[idx];
        } else if (qn == 1) {
          d[ST_M_R] = st.m[idx];
          d[ST_S_R] = st.s[idx];
        } else {
          d[ST_M_Z] = st.m[idx];
          d[ST_S_Z] = st.s[idx];
        }
      }
    }
    named_bar_sync(1, H2_EPI * 32);
    head_stats_finish(stats, 4, tab, npairs,
                      p.partials + (static_cast<long long>(slot_id) * p.P + pair0) * HEAD_STAT_FIELDS,
                      threadIdx.x - 64, H2_EPI * 32);
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
size_t h2_fixed_bytes() { return 1024 + 256 + 16 + MAX_ZPAIRS_PER_CHUNK * 4 + 64; }
uint32_t h2_tmem_cols(int cols) {
  uint32_t c = 32;
  while (c < static_cast<uint32_t>(cols)) c <<= 1;
  return c;
}
size_t h2_stage_bytes(int N) { return H2_A_BYTES + static_cast<size_t>(N / 2) * 256; }
}  // namespace

size_t head_tc2_smem_bytes(int N, int pairs, int stages) {
  (void)pairs;
  return h2_fixed_bytes() + static_cast<size_t>(stages) * h2_stage_bytes(N);
}

#ifndef RV_HEAD2_STAGE_TARGET_KB
#define RV_HEAD2_STAGE_TARGET_KB 200
#endif
int head_tc2_stages(int N, int pairs, size_t smem_limit) {
  const size_t per = h2_stage_bytes(N);
  if (smem_limit <= h2_fixed_bytes()) return 0;
  const int most = static_cast<int>((smem_limit - h2_fixed_bytes()) / per);
  const int want = static_cast<int>((RV_HEAD2_STAGE_TARGET_KB * 1024 + per - 1) / per);
  int st = std::max(0, std::min(std::min(most, 8), std::max(3, want)));
  // the statistics tables written at the end go over the stages
  const size_t tables = static_cast<size_t>(4) * pairs * HEAD_STAT_STRIDE * 4;
  while (st > 0 && st < most && static_cast<size_t>(st) * per < tables) ++st;
  return static_cast<size_t>(st) * per >= tables ? st : 0;
}

template <bool ZONLY, bool SUB>
static cudaError_t head_tc2_configure_one(size_t smem_bytes) {
  cudaError_t e = cudaFuncSetAttribute(head_tc2_kernel<ZONLY, SUB>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem_bytes));
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(head_tc2_kernel<ZONLY, SUB>,
                             cudaFuncAttributePreferredSharedMemoryCarveout,
                             cudaSharedmemCarveoutMaxShared);
  return e;
}

cudaError_t head_tc2_configure(size_t smem_bytes) {
  cudaError_t e = head_tc2_configure_one<false, false>(smem_bytes);
  if (e == cudaSuccess) e = head_tc2_configure_one<true, false>(smem_bytes);
  if (e == cudaSuccess) e = head_tc2_configure_one<false, true>(smem_bytes);
  if (e == cudaSuccess) e = head_tc2_configure_one<true, true>(smem_bytes);
  return e;
}

int head_tc2_max_pairs(int N, int pairs, int stages) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2, 1, 1);
  cfg.blockDim = dim3(H2_THREADS, 1, 1);
  cfg.dynamicSmemBytes = head_tc2_smem_bytes(N, pairs, stages);
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  // both instantiations have the same block size and shared memory
  cudaError_t e = cudaOccupancyMaxActiveClusters(&n, head_tc2_kernel<false, false>, &cfg);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

void head_pair_chunks(int P, int* n_chunks, int* pairs_per_chunk, int* sub, int* sub_pairs) {
  const int n = std::max(1, (P + HEAD_PAIR_MAX_CHUNK - 1) / HEAD_PAIR_MAX_CHUNK);
  const int pc = (P + n - 1) / n;
  *n_chunks = n;
  *pairs_per_chunk = pc;
  *sub = pc > MAX_PAIRS_PER_CHUNK ? 2 : 1;
  const int per = (pc + *sub - 1) / *sub;
  *sub_pairs = (per + 7) / 8 * 8;
}

namespace {
// Sub-groups and accumulator slots of a chunk of pad_pairs (padded) pairs:
// the ring for one sub-group, the split layout for two (the kernel's header
// comment); false when the kernel cannot run the plan.
struct H2Layout {
  int H = 0, R = 0, split = 0;
  int Ph[H2_MAX_H] = {}, pb[H2_MAX_H] = {}, scol[H2_MAX_R] = {};
  int cols = 0;  // TMEM columns in use
};

bool h2_layout(const HeadPlan& pl, H2Layout* L) {
  const int gsz = pl.zonly ? 16 : 8;
  const int pad = pl.pad_pairs;
  *L = H2Layout{};
  if (pad < gsz || pad % gsz != 0) return false;
  if (pl.sub == 1) {
    const int ns = pl.zonly ? pad : 2 * pad;  // columns per slot
    L->H = 1;
    L->Ph[0] = pad;
    L->R = std::min(H2_MAX_R, 512 / ns);
    if (L->R < 2) return false;
    for (int k = 0; k < L->R; ++k) L->scol[k] = k * ns;
    L->cols = L->R * ns;
  } else if (pl.sub == 2 && !pl.zonly) {
    // 2 Ph[0] + 4 Ph[1] = 512 columns, Ph[0] + Ph[1] = pad
    const int p1 = std::min(128, 256 - pad), p0 = pad - p1;
    if (p0 < gsz || p1 < gsz || p0 > 128 || p1 % gsz != 0) return false;
    L->H = 2;
    L->split = 1;
    L->R = 3;
    L->Ph[0] = p0;
    L->Ph[1] = p1;
    L->pb[1] = p0;
    L->scol[1] = 2 * p0;
    L->scol[2] = 2 * p0 + 2 * p1;
    L->cols = 2 * p0 + 4 * p1;
  } else {
    return false;
  }
  int own = 0;  // groups one epilogue warp owns at most
  for (int h = 0; h < L->H; ++h) own += (L->Ph[h] / gsz + H2_WPQ - 1) / H2_WPQ;
  return own <= H2_MAX_OWN && L->cols <= 512;
}
}  // namespace

bool head_tc2_supports(const HeadPlan& pl) {
  H2Layout L;
  return h2_layout(pl, &L);
}

cudaError_t launch_head_tc2(const HeadArgs& a, const HeadPlan& pl, const HeadTcLaunch& l,
                            const HeadFinal* fin, cudaStream_t s) {
  H2Layout L;
  if (!h2_layout(pl, &L)) return cudaErrorInvalidValue;
  Head2Params p;
  p.V = a.V;
  p.n_kb = (a.H + H2_BK - 1) / H2_BK;
  p.H = L.H;
  p.R = L.R;
  p.split = L.split;
  for (int h = 0; h < H2_MAX_H; ++h) {
    p.Ph[h] = L.Ph[h];
    p.pb[h] = L.pb[h];
  }
  for (int k = 0; k < H2_MAX_R; ++k) p.scol[k] = L.scol[k];
  p.b_rows = pl.zonly ? pl.pad_pairs / 2 : pl.pad_pairs;
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
  p.tmem_cols = h2_tmem_cols(L.cols);
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
  cfg.blockDim = dim3(H2_THREADS, 1, 1);
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
  if (a.zsub != nullptr) {
    if (pl.zonly) return cudaLaunchKernelEx(&cfg, head_tc2_kernel<true, true>, l.tm_w, l.tm_h, p);
    return cudaLaunchKernelEx(&cfg, head_tc2_kernel<false, true>, l.tm_w, l.tm_h, p);
  }
  if (pl.zonly) return cudaLaunchKernelEx(&cfg, head_tc2_kernel<true, false>, l.tm_w, l.tm_h, p);
  return cudaLaunchKernelEx(&cfg, head_tc2_kernel<false, false>, l.tm_w, l.tm_h, p);
}

}  // namespace rv
