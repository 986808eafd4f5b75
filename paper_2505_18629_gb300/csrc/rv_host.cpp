// Host side of the C ABI declared in include/rv.h: argument validation,
// workspace ownership, launch planning, TMA descriptor encoding, device
// status, kernel timing.  Every compute step runs in the CUDA kernels.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <new>
#include <string>
#include <vector>

#include "rv.h"
#include "rv_kernels.h"

using namespace rv;

namespace {

thread_local std::string g_create_error;

struct ProfRegion {
  std::vector<cudaEvent_t> ev;  // pairs: [2i] start, [2i+1] stop
  int used = 0;
};
constexpr int PROF_PAIRS = 1024;

struct Workspace {
  void* base = nullptr;
  size_t bytes = 0;
  unsigned* status = nullptr;
  float* head_partials = nullptr;
  float* gathered = nullptr;
  void* hsel = nullptr;
  AttnTcScratch attn{};  // tcgen05 attention: partial results, tickets, counters
  unsigned* fin_tickets = nullptr;  // [max_batch], zero between launches (head finalize)
  // staging for rv_verify_step_host
  void* st_q = nullptr;
  void* st_kb = nullptr;
  void* st_vb = nullptr;
  void* st_hidden = nullptr;
  void* st_attn = nullptr;
  // rv_verify_step_host: sizes of the pinned regions holding the small per-step
  // inputs (ids, lengths) and all the per-step outputs but the attention
  size_t small_in_bytes = 0, small_out_bytes = 0;
};

}  // namespace

// Page-locked host memory (a stream capture cannot copy from pageable memory).
bool pinned(const void* p) {
  cudaPointerAttributes a{};
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeHost;
}

// Everything that determines the device work of one rv_verify_step_host call.
struct HostStepKey {
  const void* ptr[24];
  int32_t dims[5];  // B, gamma, n_prompt, n_prefix, hidden states read in place
  float alpha;
  int32_t accept_mode, head_mode;
  float log_eps, log_delta;
  void* stream;
  bool same(const HostStepKey& o) const {  // field by field (the struct has padding)
    return std::memcmp(ptr, o.ptr, sizeof(ptr)) == 0 &&
           std::memcmp(dims, o.dims, sizeof(dims)) == 0 && alpha == o.alpha &&
           accept_mode == o.accept_mode && head_mode == o.head_mode && log_eps == o.log_eps &&
           log_delta == o.log_delta && stream == o.stream;
  }
};

struct rv_handle {
  rv_config cfg;
  int device = 0;
  int num_sms = 0;
  size_t smem_optin = 0;
  int attn_max_cluster = 1;
  Workspace ws;
  std::string err;
  PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
  // cached tensor maps
  const void* tm_w_ptr = nullptr;
  CUtensorMap tm_w;
  CUtensorMap tm_w16;
  int tm_h_N = -1;
  int tm_h_rows = -1;
  CUtensorMap tm_h;
  // rv_verify_step runs the attention on this stream, concurrently with the
  // LM head on the caller's stream (fork / join through the two events).
  cudaStream_t side = nullptr;
  cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
  cudaEvent_t ev_copy_start = nullptr, ev_copy_done = nullptr;  // rv_verify_step_host
  // recorded after the row gather when `record_prep` is set (rv_verify_step_host:
  // the side stream's copies wait for it, so they do not share the host link
  // with the gather's reads of the hidden states)
  cudaEvent_t ev_prep = nullptr;
  bool record_prep = false;
  // pinned staging of rv_verify_step_host's small inputs / outputs, which the
  // kernels read / write in place (first rv_verify_step_host call)
  char* pin_in = nullptr;
  char* pin_out = nullptr;
  // rv_verify_step_host: the arguments of the last call, and the CUDA graph of
  // the device part of a call repeated with the same arguments
  HostStepKey last_key{};
  bool have_key = false;
  HostStepKey graph_key{};
  cudaGraphExec_t host_graph = nullptr;
  unsigned long long graph_launches = 0;  // our kernel launches in the graph
  bool graphs_off = false;                // capture failed once: direct calls only
  unsigned profiling = 0;  // bit mask of the regions being recorded
  ProfRegion prof[RV_PROF_COUNT];
  unsigned long long launches = 0;
  int head_mode = RV_HEAD_FUSED_LOGITS;  // rv_set_head_mode
  int head_tc_stages_cached_N = -1;     // keyed by 2 * N + pre-blended
  int head_tc_stages = 0;
  int head_pair_cached_N = -1;   // pair kernel: stages and co-resident pairs for this N
  int head_pair_stages = 0;
  int head_pair_max = 0;
  int tm_h_box = -1;
  bool attn_tc_ok = false;  // tcgen05 attention usable for this configuration
  // acceptance rule of rv_verify_step (rv_set_acceptance)
  int accept_mode = RV_ACCEPT_EXACT;
  float accept_log_eps = 0.f, accept_log_delta = 0.f;
  // fused logits z [max_batch * (max_gamma + 1)][vocab] written by the head in
  // speculative-sampling mode (allocated on the first rv_set_acceptance to it)
  float* zbuf = nullptr;
  // per position and 32-row subtile (max z, sum exp((z - max) / T)) for the
  // sampled-exact-match step of a bf16 handle [max_batch * (max_gamma + 1)]
  // [ceil(vocab / 32)] (allocated with zbuf)
  float2* zsub = nullptr;
  // tensor maps of the last tcgen05 attention call and what they were made for
  AttnTcMaps attn_maps;
  const void* attn_map_ptrs[5] = {nullptr, nullptr, nullptr, nullptr, nullptr};
  int attn_map_B = -1, attn_map_Lb = -1;
};

namespace {

int fail(rv_handle* h, int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  if (h)
    h->err = buf;
  else
    g_create_error = buf;
  return code;
}

int cuda_fail(rv_handle* h, cudaError_t e, const char* what) {
  return fail(h, RV_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

size_t esize(const rv_config& c) { return c.dtype == RV_DTYPE_BF16 ? 2 : 4; }
// Block positions: 2 gamma + R, plus one for the pending-token block.
int lb_max(const rv_config& c) { return 2 * c.max_gamma + c.max_template + 1; }

// zonly: the pre-blended head (one blended row per pair, N = pad_pairs,
// rounded to 16 for the MMA; up to MAX_ZPAIRS_PER_CHUNK pairs per chunk).
HeadPlan head_plan(int B, int gamma, int V, int num_sms, bool tc, bool zonly = false,
                   bool standard = false) {
  HeadPlan p;
  p.zonly = zonly;
  p.standard = standard;
  p.P = B * (gamma + 1);
  const int cap = zonly ? MAX_ZPAIRS_PER_CHUNK : MAX_PAIRS_PER_CHUNK;
  p.n_chunks = (p.P + cap - 1) / cap;
  p.pairs_per_chunk = (p.P + p.n_chunks - 1) / p.n_chunks;
  p.pad_pairs = zonly ? (p.pairs_per_chunk + 15) / 16 * 16 : (p.pairs_per_chunk + 7) / 8 * 8;
  p.N = zonly ? p.pad_pairs : 2 * p.pad_pairs;
  p.sub = 1;
  p.sub_pairs = p.pad_pairs;
  p.n_vtiles = (V + 127) / 128;
  p.pair = false;
  if (tc) {  // one persistent CTA per SM; the vocab is split in whole tiles
    p.slots = std::max(1, std::min(num_sms / p.n_chunks, p.n_vtiles));
  } else {
    p.slots = std::max(1, std::min(4 * num_sms / p.n_chunks, p.n_vtiles));
  }
  return p;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// The CTA-pair plan of the two-distribution head: chunks of up to
// HEAD_PAIR_MAX_CHUNK pairs, each one pass over the weight; a chunk of more
// than MAX_PAIRS_PER_CHUNK pairs (too many columns for two accumulators) is
// two sub-groups with accumulators of their own.
HeadPlan head_pair_plan(const HeadPlan& base) {
  HeadPlan p = base;
  head_pair_chunks(p.P, &p.n_chunks, &p.pairs_per_chunk, &p.sub, &p.sub_pairs);
  p.pad_pairs = p.sub * p.sub_pairs;
  p.N = 2 * p.pad_pairs;
  return p;
}

struct ProfScope {
  rv_handle* h;
  int region;
  cudaStream_t s;
  int idx = -1;
  ProfScope(rv_handle* h_, int r, cudaStream_t s_) : h(h_), region(r), s(s_) {
    if ((h->profiling & (1u << r)) && h->prof[r].used < PROF_PAIRS) {
      idx = h->prof[r].used++;
      cudaEventRecord(h->prof[r].ev[2 * idx], s);
    }
  }
  void close() {
    if (idx >= 0) cudaEventRecord(h->prof[region].ev[2 * idx + 1], s);
    idx = -1;
  }
  ~ProfScope() { close(); }
};

int validate_config(const rv_config* c) {
  if (!c) return fail(nullptr, RV_ERR_INVALID_ARG, "cfg is NULL");
  if (c->dtype != RV_DTYPE_BF16 && c->dtype != RV_DTYPE_F32)
    return fail(nullptr, RV_ERR_INVALID_ARG, "dtype %d is neither RV_DTYPE_BF16 nor RV_DTYPE_F32",
                c->dtype);
  if (c->hidden <= 0 || c->vocab <= 0 || c->n_q_heads <= 0 || c->n_kv_heads <= 0 ||
      c->head_dim <= 0 || c->max_batch <= 0 || c->max_gamma <= 0 || c->max_template < 0 ||
      c->max_ctx <= 0)
    return fail(nullptr, RV_ERR_INVALID_ARG, "config sizes must be positive (max_template >= 0)");
  if (c->hidden % 8 != 0)
    return fail(nullptr, RV_ERR_SHAPE, "hidden %d is not a multiple of 8", c->hidden);
  if (c->n_q_heads % c->n_kv_heads != 0)
    return fail(nullptr, RV_ERR_SHAPE, "n_q_heads %d is not a multiple of n_kv_heads %d",
                c->n_q_heads, c->n_kv_heads);
  if (c->dtype == RV_DTYPE_BF16 && c->head_dim != 64 && c->head_dim != 128)
    return fail(nullptr, RV_ERR_NOT_IMPLEMENTED, "bf16 attention is built for head_dim 64/128, not %d",
                c->head_dim);
  if (c->dtype == RV_DTYPE_F32 && (c->head_dim % 32 != 0 || c->head_dim > 256))
    return fail(nullptr, RV_ERR_NOT_IMPLEMENTED,
                "fp32 attention needs head_dim a multiple of 32 and <= 256, not %d", c->head_dim);
  if (c->max_gamma > 64 || c->max_template > 256)
    return fail(nullptr, RV_ERR_CAPACITY, "max_gamma <= 64 and max_template <= 256 are supported");
  if (static_cast<long long>(c->max_batch) * (c->max_gamma + 1) > (1 << 20))
    return fail(nullptr, RV_ERR_CAPACITY, "max_batch * (max_gamma + 1) too large");
  return RV_OK;
}

}  // namespace

// ============================================================================ create / destroy

extern "C" RV_API int rv_create(const rv_config* cfg, rv_handle** out) {
  g_create_error.clear();
  if (!out) return fail(nullptr, RV_ERR_INVALID_ARG, "out is NULL");
  int rc = validate_config(cfg);
  if (rc != RV_OK) return rc;

  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(nullptr, RV_ERR_CUDA, "no CUDA device: %s", cudaGetErrorString(e));
  cudaDeviceProp prop;
  e = cudaGetDeviceProperties(&prop, dev);
  if (e != cudaSuccess) return fail(nullptr, RV_ERR_CUDA, "cudaGetDeviceProperties: %s", cudaGetErrorString(e));
  if (!(prop.major == 10 && prop.minor == 3))
    return fail(nullptr, RV_ERR_UNSUPPORTED, "librv is built for sm_103a; device is sm_%d%d (%s)",
                prop.major, prop.minor, prop.name);

  rv_handle* h = new (std::nothrow) rv_handle();
  if (!h) return fail(nullptr, RV_ERR_CUDA, "out of host memory");
  h->cfg = *cfg;
  h->device = dev;
  h->num_sms = prop.multiProcessorCount;
  h->smem_optin = prop.sharedMemPerBlockOptin;
  const bool bf16 = cfg->dtype == RV_DTYPE_BF16;
  const rv_config& c = *cfg;
  const int Lbm = lb_max(c);

  // ---- workspace layout (every piece 256-byte aligned)
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off += (bytes + 255) / 256 * 256;
    return o;
  };
  const size_t o_status = take(256);
  const int Pmax = c.max_batch * (c.max_gamma + 1);
  const int slots_max = 4 * h->num_sms;
  const size_t o_part = take(static_cast<size_t>(slots_max) * Pmax * HEAD_STAT_FIELDS * 4);
  const size_t o_gath = take(static_cast<size_t>(Pmax) * GATHER_FIELDS * 4);
  size_t hsel_rows = 0;
  if (bf16) {
    for (int P = 1; P <= Pmax; ++P) {
      const int nch = (P + MAX_PAIRS_PER_CHUNK - 1) / MAX_PAIRS_PER_CHUNK;
      const int pc = (P + nch - 1) / nch;
      hsel_rows = std::max(hsel_rows, static_cast<size_t>(nch) * 2 * ((pc + 7) / 8 * 8));
      int pn = 0, ppc = 0, psub = 0, psp = 0;  // the CTA-pair plan's chunks
      head_pair_chunks(P, &pn, &ppc, &psub, &psp);
      hsel_rows = std::max(hsel_rows, static_cast<size_t>(pn) * 2 * psub * psp);
      // the pre-blended head's plan: one row per pair, 16-row aligned chunks
      const int nz = (P + MAX_ZPAIRS_PER_CHUNK - 1) / MAX_ZPAIRS_PER_CHUNK;
      const int pz = (P + nz - 1) / nz;
      hsel_rows = std::max(hsel_rows, static_cast<size_t>(nz) * ((pz + 15) / 16 * 16));
    }
  }
  const size_t o_hsel = take(hsel_rows * c.hidden * 2);
  const size_t es = esize(c);
  const size_t n_q = static_cast<size_t>(c.max_batch) * Lbm * c.n_q_heads * c.head_dim;
  const size_t n_kv = static_cast<size_t>(c.max_batch) * Lbm * c.n_kv_heads * c.head_dim;
  const size_t n_hid = static_cast<size_t>(c.max_batch) * (Lbm + 1) * c.hidden;
  const size_t o_q = take(n_q * es), o_kb = take(n_kv * es), o_vb = take(n_kv * es);
  const size_t o_hid = take(n_hid * es), o_ao = take(n_q * es);
  // the host-buffer step's contiguous small regions (layout: see small_layout)
  const size_t small_in = 4 * (static_cast<size_t>(c.max_batch) * (c.max_gamma + 1 + c.max_template) +
                               c.max_template) + 64;
  const size_t small_out =
      4 * (static_cast<size_t>(Pmax) * (RV_NSCORES + 1) + static_cast<size_t>(c.max_batch) *
                                                              (c.max_gamma + 3 + 2 * Lbm)) +
      static_cast<size_t>(c.max_batch) * c.max_gamma + 256;
  h->attn_tc_ok = bf16 && attn_tc_supported(c.n_q_heads, c.n_kv_heads, c.head_dim) &&
                  attn_tc_smem_max(c.max_batch) <= h->smem_optin;
  const int a_slots =
      h->attn_tc_ok ? attn_tc_max_slots(c.max_batch, Lbm, c.n_q_heads, c.n_kv_heads, h->num_sms) : 0;
  const size_t o_apo = take(static_cast<size_t>(a_slots) * 128 * 128 * 4);
  const size_t o_aml = take(static_cast<size_t>(a_slots) * 128 * 2 * 4);
  const size_t o_act = take(64);
  const size_t o_fin = take(static_cast<size_t>(c.max_batch) * 4);  // finalize tickets

  e = cudaMalloc(&h->ws.base, off);
  if (e != cudaSuccess) {
    delete h;
    return fail(nullptr, RV_ERR_CUDA, "workspace cudaMalloc(%zu): %s", off, cudaGetErrorString(e));
  }
  h->ws.bytes = off;
  char* b = static_cast<char*>(h->ws.base);
  h->ws.status = reinterpret_cast<unsigned*>(b + o_status);
  h->ws.head_partials = reinterpret_cast<float*>(b + o_part);
  h->ws.gathered = reinterpret_cast<float*>(b + o_gath);
  h->ws.hsel = b + o_hsel;
  h->ws.attn.part_o = reinterpret_cast<float*>(b + o_apo);
  h->ws.attn.part_ml = reinterpret_cast<float*>(b + o_aml);
  h->ws.attn.counters = reinterpret_cast<unsigned*>(b + o_act);
  h->ws.attn.max_slots = a_slots;
  h->ws.fin_tickets = reinterpret_cast<unsigned*>(b + o_fin);
  h->ws.st_q = b + o_q;
  h->ws.st_kb = b + o_kb;
  h->ws.st_vb = b + o_vb;
  h->ws.st_hidden = b + o_hid;
  h->ws.st_attn = b + o_ao;
  h->ws.small_in_bytes = small_in;
  h->ws.small_out_bytes = small_out;
  e = cudaMemset(h->ws.base, 0, off);
  if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&h->side, cudaStreamNonBlocking);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->ev_fork, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->ev_join, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->ev_copy_start, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->ev_copy_done, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->ev_prep, cudaEventDisableTiming);
  if (e == cudaSuccess && bf16) e = attn_configure(&h->attn_max_cluster);
  if (e == cudaSuccess && h->attn_tc_ok) e = attn_tc_configure(attn_tc_smem_max(c.max_batch));
  if (e == cudaSuccess && bf16) e = head_tc_configure(h->smem_optin);
  if (e == cudaSuccess && bf16) e = head_tc2_configure(h->smem_optin);
  if (e == cudaSuccess && bf16) {
    cudaDriverEntryPointQueryResult q;
    void* fn = nullptr;
    e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
    if (e == cudaSuccess && (q != cudaDriverEntryPointSuccess || !fn)) e = cudaErrorNotSupported;
    h->encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }
  if (e != cudaSuccess) {
    if (h->ev_prep) cudaEventDestroy(h->ev_prep);
    if (h->ev_copy_done) cudaEventDestroy(h->ev_copy_done);
    if (h->ev_copy_start) cudaEventDestroy(h->ev_copy_start);
    if (h->ev_join) cudaEventDestroy(h->ev_join);
    if (h->ev_fork) cudaEventDestroy(h->ev_fork);
    if (h->side) cudaStreamDestroy(h->side);
    cudaFree(h->ws.base);
    delete h;
    return fail(nullptr, RV_ERR_CUDA, "rv_create setup: %s", cudaGetErrorString(e));
  }
  *out = h;
  return RV_OK;
}

extern "C" RV_API int rv_destroy(rv_handle* h) {
  if (!h) return RV_OK;
  cudaDeviceSynchronize();
  for (auto& r : h->prof)
    for (auto ev : r.ev) cudaEventDestroy(ev);
  cudaEventDestroy(h->ev_join);
  cudaEventDestroy(h->ev_fork);
  cudaEventDestroy(h->ev_copy_start);
  cudaEventDestroy(h->ev_copy_done);
  cudaEventDestroy(h->ev_prep);
  cudaStreamDestroy(h->side);
  if (h->zbuf) cudaFree(h->zbuf);
  if (h->zsub) cudaFree(h->zsub);
  if (h->host_graph) cudaGraphExecDestroy(h->host_graph);
  if (h->pin_in) cudaFreeHost(h->pin_in);
  if (h->pin_out) cudaFreeHost(h->pin_out);
  cudaFree(h->ws.base);
  delete h;
  return RV_OK;
}

extern "C" RV_API const char* rv_last_error(const rv_handle* h) {
  return h ? h->err.c_str() : g_create_error.c_str();
}

extern "C" RV_API int rv_workspace_bytes(const rv_handle* h, uint64_t* bytes) {
  if (!h || !bytes) return RV_ERR_INVALID_ARG;
  *bytes = h->ws.bytes;
  return RV_OK;
}

// ============================================================================ pack

extern "C" RV_API int rv_pack_block(rv_handle* h, const int32_t* draft_ids, const int32_t* prompt_ids,
                                    const int32_t* prefix_ids, const int32_t* ctx_lens, int32_t B,
                                    int32_t gamma, int32_t n_prompt, int32_t n_prefix,
                                    int32_t* block_ids, int32_t* pos_ids, void* stream) {
  if (!h) return RV_ERR_INVALID_ARG;
  h->err.clear();
  if (B < 0 || gamma < 0 || n_prompt < 0 || n_prefix < 0)
    return fail(h, RV_ERR_SHAPE, "negative size");
  if (B > h->cfg.max_batch || gamma > h->cfg.max_gamma || n_prompt + n_prefix > h->cfg.max_template)
    return fail(h, RV_ERR_CAPACITY, "B/gamma/template above the handle's maxima");
  if (B == 0) return RV_OK;
  if (!draft_ids || !ctx_lens || !block_ids || !pos_ids || (n_prompt > 0 && !prompt_ids) ||
      (n_prefix > 0 && !prefix_ids))
    return fail(h, RV_ERR_INVALID_ARG, "NULL pointer argument");
  if (h->head_mode == RV_HEAD_STANDARD && n_prompt + n_prefix != 0)
    return fail(h, RV_ERR_SHAPE, "standard verification's block has no template");
  cudaError_t e = launch_pack_block(draft_ids, prompt_ids, prefix_ids, ctx_lens, B, gamma, n_prompt,
                                    n_prefix, block_ids, pos_ids, static_cast<cudaStream_t>(stream),
                                    nullptr, h->head_mode == RV_HEAD_STANDARD ? 0 : 1);
  h->launches += 1;
  return e == cudaSuccess ? RV_OK : cuda_fail(h, e, "pack_block launch");
}

extern "C" RV_API int rv_pack_block_pending(rv_handle* h, const int32_t* pending_ids,
                                            const int32_t* draft_ids, const int32_t* prompt_ids,
                                            const int32_t* prefix_ids, const int32_t* ctx_lens,
                                            int32_t B, int32_t gamma, int32_t n_prompt,
                                            int32_t n_prefix, int32_t* block_ids, int32_t* pos_ids,
                                            void* stream) {
  if (!h) return RV_ERR_INVALID_ARG;
  h->err.clear();
  if (B < 0 || gamma < 0 || n_prompt < 0 || n_prefix < 0)
    return fail(h, RV_ERR_SHAPE, "negative size");
  if (B > h->cfg.max_batch || gamma > h->cfg.max_gamma || n_prompt + n_prefix > h->cfg.max_template)
    return fail(h, RV_ERR_CAPACITY, "B/gamma/template above the handle's maxima");
  if (B == 0) return RV_OK;
  if (!pending_ids || !draft_ids || !ctx_lens || !block_ids || !pos_ids ||
      (n_prompt > 0 && !prompt_ids) || (n_prefix > 0 && !prefix_ids))
    return fail(h, RV_ERR_INVALID_ARG, "NULL pointer argument");
  if (h->head_mode == RV_HEAD_STANDARD && n_prompt + n_prefix != 0)
    return fail(h, RV_ERR_SHAPE, "standard verification's block has no template");
  cudaError_t e = launch_pack_block(draft_ids, prompt_ids, prefix_ids, ctx_lens, B, gamma, n_prompt,
                                    n_prefix, block_ids, pos_ids, static_cast<cudaStream_t>(stream),
                                    pending_ids, h->head_mode == RV_HEAD_STANDARD ? 0 : 1);
  h->launches += 1;
  return e == cudaSuccess ? RV_OK : cuda_fail(h, e, "pack_block launch");
}

// ============================================================================ attention

extern "C" RV_API int rv_verify_attention(rv_handle* h, const void* q, const void* k_blk,
                                          const void* v_blk, void* k_cache, void* v_cache,
                                          const int32_t* ctx_lens, int32_t B, int32_t Lb, void* out,
                                          void* stream) {
  if (!h) return RV_ERR_INVALID_ARG;
  h->err.clear();
  const rv_config& c = h->cfg;
  if (B < 0 || Lb < 0) return fail(h, RV_ERR_SHAPE, "negative B or Lb");
  if (B > c.max_batch || Lb > lb_max(c))
    return fail(h, RV_ERR_CAPACITY, "B %d / Lb %d above max_batch %d / 2*max_gamma+max_template %d",
                B, Lb, c.max_batch, lb_max(c));
  if (B == 0 || Lb == 0) return RV_OK;
  if (!q || !k_blk || !v_blk || !k_cache || !v_cache || !ctx_lens || !out)
    return fail(h, RV_ERR_INVALID_ARG, "NULL pointer argument");
  const bool bf16 = c.dtype == RV_DTYPE_BF16;
  if (!aligned16(q) || !aligned16(k_blk) || !aligned16(v_blk) || !aligned16(k_cache) ||
      !aligned16(v_cache) || !aligned16(out))
    return fail(h, RV_ERR_INVALID_ARG, "attention tensors must be 16-byte aligned");
  AttnArgs a{q, k_blk, v_blk, k_cache, v_cache, ctx_lens, out, B, Lb, c.n_q_heads, c.n_kv_heads,
             c.head_dim, c.max_ctx, h->ws.status};
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  ProfScope prof(h, RV_PROF_ATTENTION, s);
  cudaError_t e;
  if (bf16) {
    const AttnPlan p = attn_plan(B, Lb, c.n_q_heads, c.n_kv_heads, c.max_ctx, h->num_sms, true,
                                 h->attn_max_cluster, c.head_dim, h->attn_tc_ok);
    if (p.tc) {
      const void* ptrs[5] = {q, k_blk, v_blk, k_cache, v_cache};
      if (h->attn_map_B != B || h->attn_map_Lb != Lb ||
          !std::equal(ptrs, ptrs + 5, h->attn_map_ptrs)) {
        if (!attn_tc_encode(h->encode, a, &h->attn_maps)) {
          h->attn_map_B = -1;
          return fail(h, RV_ERR_CUDA, "cuTensorMapEncodeTiled(attention) failed");
        }
        std::copy(ptrs, ptrs + 5, h->attn_map_ptrs);
        h->attn_map_B = B;
        h->attn_map_Lb = Lb;
      }
      const AttnTcPlan tp = attn_tc_plan(B, Lb, c.n_q_heads, c.n_kv_heads, c.max_ctx, h->num_sms);
      e = launch_attention_tc(a, tp, h->attn_maps, h->ws.attn, s);
    } else {
      e = launch_attention_bf16(a, p, s);
    }
  } else {
    e = launch_attention_f32(a, s);
  }
  h->launches += 1;
  return e == cudaSuccess ? RV_OK : cuda_fail(h, e, "attention launch");
}

// ============================================================================ head

namespace {

int encode_maps(rv_handle* h, const void* w, const HeadPlan& pl, HeadTcLaunch& l) {
  const rv_config& c = h->cfg;
  if (h->tm_w_ptr != w) {
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(c.hidden), static_cast<cuuint64_t>(c.vocab)};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(c.hidden) * 2};
    const cuuint32_t es[2] = {1, 1};
    const cuuint32_t box[2] = {64, static_cast<cuuint32_t>(HEAD_TILE_ROWS)};
    const cuuint32_t box16[2] = {64, static_cast<cuuint32_t>(HEAD_W_BOX_ROWS)};
    CUresult r = h->encode(&h->tm_w, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(w), dims,
                           strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                           CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                           CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r == CUDA_SUCCESS)
      r = h->encode(&h->tm_w16, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(w), dims,
                    strides, box16, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
      h->tm_w_ptr = nullptr;
      return fail(h, RV_ERR_CUDA, "cuTensorMapEncodeTiled(W) failed: %d", static_cast<int>(r));
    }
    h->tm_w_ptr = w;
  }
  const int rows = pl.n_chunks * pl.N;
  const int box_rows = pl.pair ? pl.N / 2 : pl.N;
  if (h->tm_h_N != pl.N || h->tm_h_rows != rows || h->tm_h_box != box_rows) {
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(c.hidden), static_cast<cuuint64_t>(rows)};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(c.hidden) * 2};
    const cuuint32_t box[2] = {64, static_cast<cuuint32_t>(box_rows)};
    const cuuint32_t es[2] = {1, 1};
    CUresult r = h->encode(&h->tm_h, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, h->ws.hsel, dims, strides,
                           box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                           CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
      h->tm_h_N = -1;
      return fail(h, RV_ERR_CUDA, "cuTensorMapEncodeTiled(hidden rows) failed: %d", static_cast<int>(r));
    }
    h->tm_h_N = pl.N;
    h->tm_h_rows = rows;
    h->tm_h_box = box_rows;
  }
  l.tm_w = h->tm_w;
  l.tm_w16 = h->tm_w16;
  l.tm_h = h->tm_h;
  if (pl.pair) {
    l.stages = h->head_pair_stages;
    l.unit_rows = HEAD_TILE_ROWS;
    l.smem_bytes = head_tc2_smem_bytes(pl.N, pl.pad_pairs, l.stages);
    return RV_OK;
  }
  if (h->head_tc_stages_cached_N != 2 * pl.N + pl.zonly) {
    h->head_tc_stages = head_tc_stages(pl.N, pl.pad_pairs, h->smem_optin);
    h->head_tc_stages_cached_N = 2 * pl.N + pl.zonly;
  }
  l.stages = h->head_tc_stages;
  l.unit_rows = HEAD_TILE_ROWS;  // whole tiles: one TMA box per stage
  if (l.stages < 2) return fail(h, RV_ERR_UNSUPPORTED, "not enough shared memory for the head pipeline");
  l.smem_bytes = head_tc_smem_bytes(pl.N, pl.pad_pairs, l.stages);
  return RV_OK;
}

// Block positions of a step (without the pending token): [x, template, x], or
// the drafts alone for standard verification.
int block_len(const rv_handle* h, int gamma, int R) {
  return h->head_mode == RV_HEAD_STANDARD ? gamma : 2 * gamma + R;
}

int check_head_args(rv_handle* h, const void* hidden, const void* w_head, const int32_t* draft_ids,
                    int B, int gamma, int R, float alpha, const void* o1, const void* o2,
                    const void* o3) {
  const rv_config& c = h->cfg;
  if (B < 0 || gamma < 1 || R < 0) return fail(h, RV_ERR_SHAPE, "need B >= 0, gamma >= 1, R >= 0");
  if (B > c.max_batch || gamma > c.max_gamma || R > c.max_template)
    return fail(h, RV_ERR_CAPACITY, "B %d / gamma %d / R %d above the handle's maxima (%d/%d/%d)", B,
                gamma, R, c.max_batch, c.max_gamma, c.max_template);
  if (!std::isfinite(alpha)) return fail(h, RV_ERR_INVALID_ARG, "alpha is not finite");
  if (h->head_mode == RV_HEAD_STANDARD && R != 0)
    return fail(h, RV_ERR_SHAPE, "standard verification has no template: R must be 0 (got %d)", R);
  if (B == 0) return RV_OK;
  if (!hidden || !w_head || !draft_ids || !o1 || !o2 || !o3)
    return fail(h, RV_ERR_INVALID_ARG, "NULL pointer argument");
  if (!aligned16(hidden) || !aligned16(w_head))
    return fail(h, RV_ERR_INVALID_ARG, "hidden and w_head must be 16-byte aligned");
  return RV_OK;
}

// The head also writes the fused logits (speculative sampling, sampled exact match).
bool writes_z(const rv_handle* h) {
  return h->accept_mode == RV_ACCEPT_SPECULATIVE || h->accept_mode == RV_ACCEPT_SAMPLED ||
         h->accept_mode == RV_ACCEPT_TYPICAL_SAMPLED;
}

// Sampled exact match inside the step (bf16): the head leaves subtile sums at
// temperature 1 / inv_t instead of the fused logits, and the draws (and the
// acceptance on them) follow in one launch.
struct SubtileRequest {
  const float* u;
  float inv_t;
  int32_t* xhat;
  AcceptArgs acc;
};

int head_impl(rv_handle* h, const void* hidden, const void* w_head, const int32_t* draft_ids, int B,
              int gamma, int R, float alpha, float* scores, int32_t* argmax, float* margin,
              const PackArgs* pack, const AcceptArgs* acc, cudaStream_t s,
              const SubtileRequest* sub = nullptr) {
  const rv_config& c = h->cfg;
  const bool bf16 = c.dtype == RV_DTYPE_BF16;
  if (sub && (!bf16 || !h->zsub)) return fail(h, RV_ERR_INVALID_ARG, "no subtile-sum buffer");
  HeadArgs a{hidden, w_head, draft_ids, B, gamma, R, c.vocab, c.hidden, alpha,
             h->ws.head_partials, h->ws.gathered, h->ws.status,
             bf16 ? h->ws.status + 16 : nullptr,    // tile counter: its own 64-byte line
             bf16 ? h->ws.status + 32 : nullptr,    // finished-CTA counter
             writes_z(h) && !sub ? h->zbuf : nullptr, h->ws.fin_tickets};
  if (sub) {
    a.zsub = h->zsub;
    a.inv_t = sub->inv_t;
  }
  HeadPlan pl = head_plan(B, gamma, c.vocab, h->num_sms, bf16,
                          bf16 && h->head_mode != RV_HEAD_FUSED_LOGITS,
                          bf16 && h->head_mode == RV_HEAD_STANDARD);
  if (bf16 && pl.N >= HEAD_PAIR_MIN_N) {
    // CTA pairs: as many as fit at once (two CTAs of a pair share a GPC)
    HeadPlan pp = pl.zonly ? pl : head_pair_plan(pl);
    if (head_tc2_supports(pp)) {
      if (h->head_pair_cached_N != 2 * pp.N + pp.zonly) {
        h->head_pair_stages = head_tc2_stages(pp.N, pp.pad_pairs, h->smem_optin);
        h->head_pair_max = h->head_pair_stages >= 2
                               ? head_tc2_max_pairs(pp.N, pp.pad_pairs, h->head_pair_stages)
                               : 0;
        h->head_pair_cached_N = 2 * pp.N + pp.zonly;
      }
      const int n_pt = (c.vocab + 255) / 256;
      int pairs = std::min({h->num_sms / 2 / pp.n_chunks, h->head_pair_max / pp.n_chunks, n_pt});
      if (pairs >= 1) {
        // the fewest pairs whose busiest one runs as many vocab tiles: the
        // head ends no later, and the SMs left free run the attention of the
        // step from the start (8B: 501 tiles on 72 pairs instead of 76)
        const int most = (n_pt + pairs - 1) / pairs;
        pairs = (n_pt + most - 1) / most;
        pl = pp;
        pl.pair = true;
        pl.slots = 2 * pairs;
      }
    }
  }
  ProfScope prof_all(h, RV_PROF_HEAD, s);
  cudaError_t e = cudaSuccess;
  HeadTcLaunch l;
  if (bf16) {
    int rc = encode_maps(h, w_head, pl, l);
    if (rc != RV_OK) return rc;
  }
  if (bf16 || pack) {
    e = launch_prep(a, pl, bf16 ? h->ws.hsel : nullptr, pack, s);
    h->launches += 1;
    if (e != cudaSuccess) return cuda_fail(h, e, "prep launch");
  }
  if (h->record_prep) {
    e = cudaEventRecord(h->ev_prep, s);
    if (e != cudaSuccess) return cuda_fail(h, e, "event record");
  }
  // Small pair counts: the head kernel's last CTA finishes the merge itself.
  // (one chunk only: the merge reads each pair's draft from the CTA's chunk table)
  const bool fused = bf16 && pl.P <= HEAD_FUSED_FINAL_MAX_PAIRS && pl.n_chunks == 1;
  HeadFinal fin{scores, argmax, margin, acc ? *acc : AcceptArgs{}, pl.zonly ? 1 : 0};
  {
    ProfScope prof(h, RV_PROF_HEAD_GEMM, s);
    e = !bf16    ? launch_head_simt(a, pl, s)
        : pl.pair ? launch_head_tc2(a, pl, l, fused ? &fin : nullptr, s)
                  : launch_head_tc(a, pl, l, fused ? &fin : nullptr, s);
    h->launches += 1;
  }
  if (e != cudaSuccess) return cuda_fail(h, e, "LM head launch");
  if (!fused) {
    e = launch_head_finalize(a, pl, scores, argmax, margin, acc, s);
    h->launches += 1;
    if (e != cudaSuccess) return cuda_fail(h, e, "head finalize launch");
  }
  if (!sub) return RV_OK;
  prof_all.close();
  ProfScope prof(h, RV_PROF_ACCEPT, s);
  const SubtileDraw d{h->zsub,    (c.vocab + 31) / 32, sub->u,      sub->inv_t,      w_head,
                      h->ws.hsel, c.vocab,            c.hidden,    pl.P,            gamma,
                      pl.pairs_per_chunk, pl.pad_pairs, pl.N,      pl.zonly ? 1 : 0, alpha,
                      sub->xhat,  draft_ids,          h->ws.fin_tickets, scores};
  e = launch_sample_subtiles(d, &sub->acc, s);
  h->launches += 1;
  return e == cudaSuccess ? RV_OK : cuda_fail(h, e, "subtile draw launch");
}

int accept_impl(rv_handle* h, const int32_t* draft_ids, const int32_t* argmax, int B, int gamma,
                uint8_t* accept_mask, int32_t* accepted_len, int32_t* next_token,
                const int32_t* ctx_in, int32_t* ctx_out, cudaStream_t s) {
  ProfScope prof(h, RV_PROF_ACCEPT, s);
  cudaError_t e = launch_accept(draft_ids, argmax, B, gamma, accept_mask, accepted_len, next_token,
                                ctx_in, ctx_out, s);
  h->launches += 1;
  return e == cudaSuccess ? RV_OK : cuda_fail(h, e, "accept launch");
}

}  // namespace

extern "C" RV_API int rv_verify_head(rv_handle* h, const void* hidden, const void* w_head,
                                     const int32_t* draft_ids, int32_t B, int32_t gamma, int32_t R,
                                     float alpha, float* scores, int32_t* argmax, float* margin,
                                     void* stream) {
  if (!h) return RV_ERR_INVALID_ARG;
  h->err.clear();
  int rc = check_head_args(h, hidden, w_head, draft_ids, B, gamma, R, alpha, scores, argmax, margin);
  if (rc != RV_OK || B == 0) return rc;
  return head_impl(h, hidden, w_head, draft_ids, B, gamma, R, alpha, scores, argmax, margin,
                   nullptr, nullptr, static_cast<cudaStream_t>(stream));
}

extern "C" RV_API int rv_accept(rv_handle* h, const int32_t* draft_ids, const int32_t* argmax,
                                int32_t B, int32_t gamma, uint8_t* accept_mask,
                                int32_t* accepted_len, int32_t* next_token, const int32_t* ctx_in,
                                int32_t* ctx_out, void* stream) {
  if (!h) return RV_ERR_INVALID_ARG;
  h->err.clear();
  if (B < 0 || gamma < 1) return fail(h, RV_ERR_SHAPE, "need B >= 0 and gamma >= 1");
  if (B > h->cfg.max_batch || gamma > h->cfg.max_gamma)
    return fail(h, RV_ERR_CAPACITY, "B / gamma above the handle's maxima");
  if (B == 0) return RV_OK;
  if (!draft_ids || !argmax || !accept_mask || !accepted_len || !next_token || !ctx_in || !ctx_out)
    return fail(h, RV_ERR_INVALID_ARG, "NULL pointer argument");
  return accept_impl(h, draft_ids, argmax, B, gamma, accept_mask, accepted_len, next_token, ctx_in,
                     ctx_out, static_cast<cudaStream_t>(stream));
}

extern "C" RV_API int rv_accept_typical(rv_handle* h, const int32_t* draft_ids, const float* scores,
                                        const int32_t* argmax, int32_t B, int32_t gamma, float eps,
                                        float delta, uint8_t* accept_mask, int32_t* accepted_len,
                                        int32_t* next_token, const int32_t* ctx_in,
                                        int32_t* ctx_out, void* stream) {
  if (!h) return RV_ERR_INVALID_ARG;
  h->err.clear();
  if (B < 0 || gamma < 1) return fail(h, RV_ERR_SHAPE, "need B >= 0 and gamma >= 1");
  if (B > h->cfg.max_batch || gamma > h->cfg.max_gamma)
    return fail(h, RV_ERR_CAPACITY, "B / gamma above the handle's maxima");
  if (!(eps > 0.f) || !(delta > 0.f) || !std::isfinite(eps) || !std::isfinite(delta))
    return fail(h, RV_ERR_INVALID_ARG, "typical acceptance needs finite eps > 0 and delta > 0");
  if (B == 0) return RV_OK;
  if (!draft_ids || !scores || !argmax || !accept_mask || !accepted_len || !next_token || !ctx_in ||
      !ctx_out)
    return fail(h, RV_ERR_INVALID_ARG, "NULL pointer argument");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  ProfScope prof(h, RV_PROF_ACCEPT, s);
  cudaError_t e = launch_accept_typical(draft_ids, scores, argmax, B, gamma, logf(eps), logf(delta),
                                        accept_mask, accepted_len, next_token, ctx_in, ctx_out, s);
  h->launches += 1;
  return e == cudaSuccess ? RV_OK : cuda_fail(h, e, "typical accept launch");
}

extern "C" RV_API int rv_set_acceptance(rv_handle* h, int32_t mode, float eps, float delta) {
  if (!h) return RV_ERR_INVALID_ARG;
  h->err.clear();
  if (mode == RV_ACCEPT_EXACT) {
    h->accept_mode = mode;
    return RV_OK;
  }
  const bool typical = mode == RV_ACCEPT_TYPICAL || mode == RV_ACCEPT_TYPICAL_SAMPLED;
  if (typical) {
    if (h->head_mode != RV_HEAD_FUSED_LOGITS)
      return fail(h, RV_ERR_INVALID_ARG,
                  "typical acceptance needs the original distribution's entropy, which the "
                  "single-distribution heads do not form");
    if (!(eps > 0.f) || !(delta > 0.f) || !std::isfinite(eps) || !std::isfinite(delta))
      return fail(h, RV_ERR_INVALID_ARG, "typical acceptance needs finite eps > 0 and delta > 0");
  }
  if (mode == RV_ACCEPT_SPECULATIVE || mode == RV_ACCEPT_SAMPLED ||
      mode == RV_ACCEPT_TYPICAL_SAMPLED) {
    const rv_config& c = h->cfg;
    if (!h->zbuf) {
      const size_t bytes = static_cast<size_t>(c.max_batch) * (c.max_gamma + 1) * c.vocab * 4;
      cudaError_t e = cudaMalloc(&h->zbuf, bytes);
      if (e != cudaSuccess) {
        h->zbuf = nullptr;
        return fail(h, RV_ERR_CUDA, "fused-logit buffer cudaMalloc(%zu): %s", bytes,
                    cudaGetErrorString(e));
      }
    }
    if (mode != RV_ACCEPT_SPECULATIVE && c.dtype == RV_DTYPE_BF16 && !h->zsub) {
      const size_t bytes =
          static_cast<size_t>(c.max_batch) * (c.max_gamma + 1) * ((c.vocab + 31) / 32) * 8;
      cudaError_t e = cudaMalloc(&h->zsub, bytes);
      if (e != cudaSuccess) {
        h->zsub = nullptr;
        return fail(h, RV_ERR_CUDA, "subtile-sum buffer cudaMalloc(%zu): %s", bytes,
                    cudaGetErrorString(e));
      }
    }
    h->accept_mode = mode;
    if (typical) {
      h->accept_log_eps = logf(eps);
      h->accept_log_delta = logf(delta);
    }
    return RV_OK;
  }
  if (mode != RV_ACCEPT_TYPICAL) return fail(h, RV_ERR_INVALID_ARG, "unknown acceptance mode %d", mode);
  h->accept_mode = mode;
  h->accept_log_eps = logf(eps);
  h->accept_log_delta = logf(delta);
  return RV_OK;
}

extern "C" RV_API int rv_set_head_mode(rv_handle* h, int32_t mode) {
  if (!h) return RV_ERR_INVALID_ARG;
  h->err.clear();
  if (mode == RV_HEAD_FUSED_LOGITS) {
    h->head_mode = mode;
    return RV_OK;
  }
  if (mode != RV_HEAD_PREBLENDED && mode != RV_HEAD_STANDARD)
    return fail(h, RV_ERR_INVALID_ARG, "unknown head mode %d", mode);
  if (h->cfg.dtype != RV_DTYPE_BF16)
    return fail(h, RV_ERR_UNSUPPORTED, "the single-distribution heads are bf16 LM-head variants");
  if (h->accept_mode == RV_ACCEPT_TYPICAL || h->accept_mode == RV_ACCEPT_TYPICAL_SAMPLED)
    return fail(h, RV_ERR_INVALID_ARG,
                "typical acceptance needs the original distribution's entropy, which the "
                "single-distribution heads do not form");
  h->head_mode = mode;
  return RV_OK;
}

// ============================================================================ whole step

// The persistent tcgen05 attention also runs on the side stream, after the LM
// head is launched, when the KV capacity is at most this many positions: its
// CTAs take the SMs that the head's last tiles leave idle (8B B=16 step
// 318 -> 313 us, e2e 0.99 -> 1.07 M positions/s).  The two kernels cannot share
// an SM (their shared memory exceeds one SM's), and neither waits on the other.
// With long caches the attention is better run alone first (8B B=16 ctx 8192:
// 404 -> 383 us; B=64 ctx 8192: 887 -> 824 us); the context lengths
// themselves live on the device, so the capacity decides.
#ifndef RV_FORK_ATTENTION_MAX_CTX
#define RV_FORK_ATTENTION_MAX_CTX 4608
#endif

namespace {

// Whether the step runs the attention on the side stream, beside the LM head,
// or before it on the caller's stream.
bool attn_forks(const rv_handle* h, int B, int Lb) {
  const rv_config& c = h->cfg;
  if (c.max_ctx <= RV_FORK_ATTENTION_MAX_CTX) return true;
  return c.dtype != RV_DTYPE_BF16 ||
         !attn_plan(B, Lb, c.n_q_heads, c.n_kv_heads, c.max_ctx, h->num_sms, true,
                    h->attn_max_cluster, c.head_dim, h->attn_tc_ok)
              .tc;
}

// The whole step; `spec` != nullptr runs a sampling acceptance after the head
// instead of the rule fused into the head's merge: speculative sampling
// (Alg. 1; q, r, u) or exact match against sampled target tokens (Alg. 2;
// u, temperature, sampled).
struct SpecInputs {
  const float* q;
  const float* r;
  const float* u;
  bool sampled_exact = false;
  float temperature = 1.f;
  int32_t* sampled = nullptr;
};

// The draws from the fused logits the head wrote, then the acceptance: exact
// match against them, or (`typical_scores` given) the typical rule with t the
// draw at n+1.
int sampled_accept_launches(rv_handle* h, const int32_t* draft_ids, const float* u,
                            float temperature, int B, int gamma, int32_t* sampled,
                            uint8_t* accept_mask, int32_t* accepted_len, int32_t* next_token,
                            const int32_t* ctx_in, int32_t* ctx_out, cudaStream_t s,
                            int ctx_extra = 0, const float* typical_scores = nullptr) {
  ProfScope prof(h, RV_PROF_ACCEPT, s);
  cudaError_t e = launch_sample_fused(h->zbuf, u, B * (gamma + 1), h->cfg.vocab, temperature,
                                      sampled, s);
  h->launches += 1;
  if (e != cudaSuccess) return cuda_fail(h, e, "sampling launch");
  // (the typical kernel takes its t from the array in the argmax place)
  e = typical_scores
          ? launch_accept_typical(draft_ids, typical_scores, sampled, B, gamma, h->accept_log_eps,
                                  h->accept_log_delta, accept_mask, accepted_len, next_token,
                                  ctx_in, ctx_out, s, ctx_extra)
          : launch_accept(draft_ids, sampled, B, gamma, accept_mask, accepted_len, next_token,
                          ctx_in, ctx_out, s, ctx_extra);
  h->launches += 1;
  return e == cudaSuccess ? RV_OK : cuda_fail(h, e, "accept launch");
}

// Host-to-device copies of the attention's inputs that rv_verify_step_host
// leaves to the step: issued on the side stream once the row gather has run.
struct SideCopies {
  void* q;
  const void* q_src;
  void* k;
  const void* k_src;
  void* v;
  const void* v_src;
  size_t nq, nkv;
};

int step_impl(rv_handle* h, const void* q, const void* k_blk, const void* v_blk, void* k_cache,
              void* v_cache, const void* hidden, const void* w_head, const int32_t* draft_ids,
              const int32_t* prompt_ids, const int32_t* prefix_ids, const int32_t* ctx_in,
              int32_t B, int32_t gamma, int32_t n_prompt, int32_t n_prefix, float alpha,
              int32_t* block_ids, int32_t* pos_ids, void* attn_out, float* scores,
              int32_t* argmax, float* margin, uint8_t* accept_mask, int32_t* accepted_len,
              int32_t* next_token, int32_t* ctx_out, const SpecInputs* spec, void* stream,
              const int32_t* pending = nullptr, const SideCopies* copies = nullptr) {
  if (n_prompt < 0 || n_prefix < 0) return fail(h, RV_ERR_SHAPE, "negative template part");
  const int R = n_prompt + n_prefix;
  const int lead = pending ? 1 : 0;  // the pending-token block has one more position
  int rc = check_head_args(h, hidden, w_head, draft_ids, B, gamma, R, alpha, scores, argmax, margin);
  if (rc != RV_OK || B == 0) return rc;
  if (!ctx_in || !accept_mask || !accepted_len || !next_token || !ctx_out)
    return fail(h, RV_ERR_INVALID_ARG, "NULL pointer argument");
  const bool do_pack = block_ids != nullptr;
  if (do_pack && (!pos_ids || (n_prompt > 0 && !prompt_ids) || (n_prefix > 0 && !prefix_ids)))
    return fail(h, RV_ERR_INVALID_ARG, "NULL pointer argument for the block packing");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const rv_config& c = h->cfg;
  const int Lb = block_len(h, gamma, R) + lead;
  // The attention (independent of the LM head) runs on the side stream; join
  // before returning.  The head goes first (it is the long pole).  At small
  // batches the split-KV attention shares the SMs with the HBM-bound head; the
  // persistent tcgen05 attention of larger batches takes SMs as head CTAs finish.
  const bool fork = attn_forks(h, B, Lb);
  cudaError_t e = cudaSuccess;
  if (fork) {
    e = cudaEventRecord(h->ev_fork, s);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(h->side, h->ev_fork, 0);
    if (e != cudaSuccess) return cuda_fail(h, e, "stream fork");
  }
  auto run_head = [&]() -> int {
    PackArgs pk{draft_ids, prompt_ids, prefix_ids, ctx_in, B, gamma, n_prompt, n_prefix, block_ids,
                pos_ids, pending};
    pk.copy = h->head_mode == RV_HEAD_STANDARD ? 0 : 1;
    AcceptArgs ac{accept_mask, accepted_len,       next_token,         ctx_in,
                  ctx_out,     h->accept_mode,     h->accept_log_eps,  h->accept_log_delta,
                  lead};
    const bool typical_t = h->accept_mode == RV_ACCEPT_TYPICAL_SAMPLED;
    if (spec && spec->sampled_exact && h->zsub) {
      AcceptArgs sac = ac;  // the kept drafts: exact match with the draws, or typical
      sac.mode = typical_t ? RV_ACCEPT_TYPICAL : RV_ACCEPT_EXACT;
      const SubtileRequest sr{spec->u, 1.f / spec->temperature, spec->sampled, sac};
      return head_impl(h, hidden, w_head, draft_ids, B, gamma, R, alpha, scores, argmax, margin,
                       do_pack ? &pk : nullptr, nullptr, s, &sr);
    }
    int r = head_impl(h, hidden, w_head, draft_ids, B, gamma, R, alpha, scores, argmax, margin,
                      do_pack ? &pk : nullptr, spec ? nullptr : &ac, s);
    if (r == RV_OK && spec && spec->sampled_exact) {
      r = sampled_accept_launches(h, draft_ids, spec->u, spec->temperature, B, gamma,
                                  spec->sampled, accept_mask, accepted_len, next_token, ctx_in,
                                  ctx_out, s, lead, typical_t ? scores : nullptr);
    } else if (r == RV_OK && spec) {
      ProfScope prof(h, RV_PROF_ACCEPT, s);
      cudaError_t e2 = launch_accept_speculative(draft_ids, spec->q, spec->r, spec->u, scores,
                                                 h->zbuf, B, gamma, c.vocab, accept_mask,
                                                 accepted_len, next_token, ctx_in, ctx_out,
                                                 h->ws.status, s, lead);
      h->launches += 1;
      if (e2 != cudaSuccess) r = cuda_fail(h, e2, "speculative accept launch");
    }
    return r;
  };
  if (fork) {
    h->record_prep = copies != nullptr;
    rc = run_head();
    h->record_prep = false;
    if (rc == RV_OK && copies) {
      e = cudaStreamWaitEvent(h->side, h->ev_prep, 0);
      if (e == cudaSuccess)
        e = cudaMemcpyAsync(copies->q, copies->q_src, copies->nq, cudaMemcpyHostToDevice, h->side);
      if (e == cudaSuccess)
        e = cudaMemcpyAsync(copies->k, copies->k_src, copies->nkv, cudaMemcpyHostToDevice,
                            h->side);
      if (e == cudaSuccess)
        e = cudaMemcpyAsync(copies->v, copies->v_src, copies->nkv, cudaMemcpyHostToDevice,
                            h->side);
      if (e != cudaSuccess) rc = cuda_fail(h, e, "host->device copy");
    }
    if (rc == RV_OK)
      rc = rv_verify_attention(h, q, k_blk, v_blk, k_cache, v_cache, ctx_in, B, Lb, attn_out,
                               h->side);
  } else {
    rc = rv_verify_attention(h, q, k_blk, v_blk, k_cache, v_cache, ctx_in, B, Lb, attn_out, s);
    if (rc == RV_OK) rc = run_head();
  }
  if (fork) {
    e = cudaEventRecord(h->ev_join, h->side);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(s, h->ev_join, 0);
    if (e != cudaSuccess && rc == RV_OK) return cuda_fail(h, e, "stream join");
  }
  return rc;
}

}  // namespace

namespace {
// The acceptance modes rv_verify_step (and its host-buffer form) can run: the
// others need inputs of their own.
int plain_step_mode(rv_handle* h) {
  if (h->accept_mode == RV_ACCEPT_SPECULATIVE)
    return fail(h, RV_ERR_INVALID_ARG,
                "speculative sampling needs the draft distributions: use rv_verify_step_speculative");
  if (h->accept_mode == RV_ACCEPT_SAMPLED || h->accept_mode == RV_ACCEPT_TYPICAL_SAMPLED)
    return fail(h, RV_ERR_INVALID_ARG,
                "a sampled next token needs the uniforms: use rv_verify_step_sampled");
  return RV_OK;
}
}  // namespace

extern "C" RV_API int rv_verify_step(
    rv_handle* h, const void* q, const void* k_blk, const void* v_blk, void* k_cache, void* v_cache,
    const void* hidden, const void* w_head, const int32_t* draft_ids, const int32_t* prompt_ids,
    const int32_t* prefix_ids, const int32_t* ctx_in, int32_t B, int32_t gamma, int32_t n_prompt,
    int32_t n_prefix, float alpha, int32_t* block_ids, int32_t* pos_ids, void* attn_out,
    float* scores, int32_t* argmax, float* margin, uint8_t* accept_mask, int32_t* accepted_len,
    int32_t* next_token, int32_t* ctx_out, void* stream) {
  if (!h) return RV_ERR_INVALID_ARG;
  h->err.clear();
  const int mrc = plain_step_mode(h);
  if (mrc != RV_OK) return mrc;
  return step_impl(h, q, k_blk, v_blk, k_cache, v_cache, hidden, w_head, draft_ids, prompt_ids,
                   prefix_ids, ctx_in, B, gamma, n_prompt, n_prefix, alpha, block_ids, pos_ids,
                   attn_out, scores, argmax, margin, accept_mask, accepted_len, next_token, ctx_out,
                   nullptr, stream);
}

extern "C" RV_API int rv_verify_step_pending(
    rv_handle* h, const void* q, const void* k_blk, const void* v_blk, void* k_cache, void* v_cache,
    const void* hidden, const void* w_head, const int32_t* pending_ids, const int32_t* draft_ids,
    const int32_t* prompt_ids, const int32_t* prefix_ids, const int32_t* ctx_in, int32_t B,
    int32_t gamma, int32_t n_prompt, int32_t n_prefix, float alpha, int32_t* block_ids,
    int32_t* pos_ids, void* attn_out, float* scores, int32_t* argmax, float* margin,
    uint8_t* accept_mask, int32_t* accepted_len, int32_t* next_token, int32_t* ctx_out,
    void* stream) {
  if (!h) return RV_ERR_INVALID_ARG;
  h->err.clear();
  if (h->accept_mode == RV_ACCEPT_SPECULATIVE || h->accept_mode == RV_ACCEPT_SAMPLED ||
      h->accept_mode == RV_ACCEPT_TYPICAL_SAMPLED)
    return fail(h, RV_ERR_INVALID_ARG,
                "the pending-token step runs the exact-match or typical rule of the handle");
  if (B > 0 && !pending_ids)
    return fail(h, RV_ERR_INVALID_ARG, "NULL pending token ids");
  return step_impl(h, q, k_blk, v_blk, k_cache, v_cache, hidden, w_head, draft_ids, prompt_ids,
                   prefix_ids, ctx_in, B, gamma, n_prompt, n_prefix, alpha, block_ids, pos_ids,
                   attn_out, scores, argmax, margin, accept_mask, accepted_len, next_token, ctx_out,
                   nullptr, stream, pending_ids);
}

extern "C" RV_API int rv_verify_step_speculative(
    rv_handle* h, const void* q, const void* k_blk, const void* v_blk, void* k_cache, void* v_cache,
    const void* hidden, const void* w_head, const int32_t* draft_ids, const int32_t* prompt_ids,
    const int32_t* prefix_ids, const int32_t* ctx_in, int32_t B, int32_t gamma, int32_t n_prompt,
    int32_t n_prefix, float alpha, const float* q_draft, const float* r_uniform,
    const float* u_uniform, int32_t* block_ids, int32_t* pos_ids, void* attn_out, float* scores,
    int32_t* argmax, float* margin, uint8_t* accept_mask, int32_t* accepted_len,
    int32_t* next_token, int32_t* ctx_out, void* stream) {
  if (!h) return RV_ERR_INVALID_ARG;
  h->err.clear();
  if (h->accept_mode != RV_ACCEPT_SPECULATIVE || !h->zbuf)
    return fail(h, RV_ERR_INVALID_ARG,
                "call rv_set_acceptance(RV_ACCEPT_SPECULATIVE) on the handle first");
  if (B > 0 && (!q_draft || !r_uniform || !u_uniform))
    return fail(h, RV_ERR_INVALID_ARG, "NULL draft distribution or uniforms");
  const SpecInputs spec{q_draft, r_uniform, u_uniform};
  return step_impl(h, q, k_blk, v_blk, k_cache, v_cache, hidden, w_head, draft_ids, prompt_ids,
                   prefix_ids, ctx_in, B, gamma, n_prompt, n_prefix, alpha, block_ids, pos_ids,
                   attn_out, scores, argmax, margin, accept_mask, accepted_len, next_token, ctx_out,
                   &spec, stream);
}

extern "C" RV_API int rv_verify_step_sampled(
    rv_handle* h, const void* q, const void* k_blk, const void* v_blk, void* k_cache, void* v_cache,
    const void* hidden, const void* w_head, const int32_t* draft_ids, const int32_t* prompt_ids,
    const int32_t* prefix_ids, const int32_t* ctx_in, int32_t B, int32_t gamma, int32_t n_prompt,
    int32_t n_prefix, float alpha, float temperature, const float* u_uniform, int32_t* block_ids,
    int32_t* pos_ids, void* attn_out, float* scores, int32_t* argmax, float* margin,
    int32_t* sampled, uint8_t* accept_mask, int32_t* accepted_len, int32_t* next_token,
    int32_t* ctx_out, void* stream) {
  if (!h) return RV_ERR_INVALID_ARG;
  h->err.clear();
  if ((h->accept_mode != RV_ACCEPT_SAMPLED && h->accept_mode != RV_ACCEPT_TYPICAL_SAMPLED) ||
      !h->zbuf)
    return fail(h, RV_ERR_INVALID_ARG,
                "call rv_set_acceptance(RV_ACCEPT_SAMPLED or RV_ACCEPT_TYPICAL_SAMPLED) on the "
                "handle first");
  if (!(temperature > 0.f) || !std::isfinite(temperature))
    return fail(h, RV_ERR_INVALID_ARG, "temperature must be finite and > 0");
  if (B > 0 && (!u_uniform || !sampled))
    return fail(h, RV_ERR_INVALID_ARG, "NULL uniforms or sampled-token output");
  SpecInputs spec{nullptr, nullptr, u_uniform};
  spec.sampled_exact = true;
  spec.temperature = temperature;
  spec.sampled = sampled;
  return step_impl(h, q, k_blk, v_blk, k_cache, v_cache, hidden, w_head, draft_ids, prompt_ids,
                   prefix_ids, ctx_in, B, gamma, n_prompt, n_prefix, alpha, block_ids, pos_ids,
                   attn_out, scores, argmax, margin, accept_mask, accepted_len, next_token, ctx_out,
                   &spec, stream);
}

extern "C" RV_API int rv_accept_sampled(rv_handle* h, const int32_t* draft_ids,
                                        const float* u_uniform, float temperature, int32_t B,
                                        int32_t gamma, int32_t* sampled, uint8_t* accept_mask,
                                        int32_t* accepted_len, int32_t* next_token,
                                        const int32_t* ctx_in, int32_t* ctx_out, void* stream) {
  if (!h) return RV_ERR_INVALID_ARG;
  h->err.clear();
  if (h->accept_mode != RV_ACCEPT_SAMPLED || !h->zbuf)
    return fail(h, RV_ERR_INVALID_ARG,
                "call rv_set_acceptance(RV_ACCEPT_SAMPLED) before rv_verify_head");
  if (B < 0 || gamma < 1) return fail(h, RV_ERR_SHAPE, "need B >= 0 and gamma >= 1");
  if (B > h->cfg.max_batch || gamma > h->cfg.max_gamma)
    return fail(h, RV_ERR_CAPACITY, "B / gamma above the handle's maxima");
  if (!(temperature > 0.f) || !std::isfinite(temperature))
    return fail(h, RV_ERR_INVALID_ARG, "temperature must be finite and > 0");
  if (B == 0) return RV_OK;
  if (!draft_ids || !u_uniform || !sampled || !accept_mask || !accepted_len || !next_token ||
      !ctx_in || !ctx_out)
    return fail(h, RV_ERR_INVALID_ARG, "NULL pointer argument");
  return sampled_accept_launches(h, draft_ids, u_uniform, temperature, B, gamma, sampled,
                                 accept_mask, accepted_len, next_token, ctx_in, ctx_out,
                                 static_cast<cudaStream_t>(stream));
}

extern "C" RV_API int rv_accept_speculative(rv_handle* h, const int32_t* draft_ids,
                                            const float* q_draft, const float* r_uniform,
                                            const float* u_uniform, const float* scores,
                                            int32_t B, int32_t gamma, uint8_t* accept_mask,
                                            int32_t* accepted_len, int32_t* next_token,
                                            const int32_t* ctx_in, int32_t* ctx_out,
                                            void* stream) {
  if (!h) return RV_ERR_INVALID_ARG;
  h->err.clear();
  if (h->accept_mode != RV_ACCEPT_SPECULATIVE || !h->zbuf)
    return fail(h, RV_ERR_INVALID_ARG,
                "call rv_set_acceptance(RV_ACCEPT_SPECULATIVE) before rv_verify_head");
  if (B < 0 || gamma < 1) return fail(h, RV_ERR_SHAPE, "need B >= 0 and gamma >= 1");
  if (B > h->cfg.max_batch || gamma > h->cfg.max_gamma)
    return fail(h, RV_ERR_CAPACITY, "B / gamma above the handle's maxima");
  if (B == 0) return RV_OK;
  if (!draft_ids || !q_draft || !r_uniform || !u_uniform || !scores || !accept_mask ||
      !accepted_len || !next_token || !ctx_in || !ctx_out)
    return fail(h, RV_ERR_INVALID_ARG, "NULL pointer argument");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  ProfScope prof(h, RV_PROF_ACCEPT, s);
  cudaError_t e = launch_accept_speculative(draft_ids, q_draft, r_uniform, u_uniform, scores,
                                            h->zbuf, B, gamma, h->cfg.vocab, accept_mask,
                                            accepted_len, next_token, ctx_in, ctx_out,
                                            h->ws.status, s);
  h->launches += 1;
  return e == cudaSuccess ? RV_OK : cuda_fail(h, e, "speculative accept launch");
}

extern "C" RV_API int rv_verify_step_host(
    rv_handle* h, const void* q_host, const void* k_blk_host, const void* v_blk_host, void* k_cache,
    void* v_cache, const void* hidden_host, const void* w_head, const int32_t* draft_ids_host,
    const int32_t* prompt_ids_host, const int32_t* prefix_ids_host, const int32_t* ctx_in_host,
    int32_t B, int32_t gamma, int32_t n_prompt, int32_t n_prefix, float alpha,
    int32_t* block_ids_host, int32_t* pos_ids_host, void* attn_out_host, float* scores_host,
    int32_t* argmax_host, float* margin_host, uint8_t* accept_mask_host, int32_t* accepted_len_host,
    int32_t* next_token_host, int32_t* ctx_out_host, uint64_t* h2d_bytes, uint64_t* d2h_bytes,
    void* stream) {
  if (!h) return RV_ERR_INVALID_ARG;
  h->err.clear();
  const rv_config& c = h->cfg;
  if (B < 1 || gamma < 1 || n_prompt < 0 || n_prefix < 0)
    return fail(h, RV_ERR_SHAPE, "need B >= 1, gamma >= 1, template parts >= 0");
  const int R = n_prompt + n_prefix;
  if (B > c.max_batch || gamma > c.max_gamma || R > c.max_template)
    return fail(h, RV_ERR_CAPACITY, "B / gamma / R above the handle's maxima");
  if (!q_host || !k_blk_host || !v_blk_host || !k_cache || !v_cache || !hidden_host || !w_head ||
      !draft_ids_host || !ctx_in_host || !scores_host || !argmax_host || !margin_host ||
      !accept_mask_host || !accepted_len_host || !next_token_host || !ctx_out_host)
    return fail(h, RV_ERR_INVALID_ARG, "NULL pointer argument");
  const bool do_pack = block_ids_host != nullptr;
  if (do_pack && (!pos_ids_host || (n_prompt > 0 && !prompt_ids_host) ||
                  (n_prefix > 0 && !prefix_ids_host)))
    return fail(h, RV_ERR_INVALID_ARG, "NULL pointer argument for the block packing");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const size_t es = esize(c);
  if (h->head_mode == RV_HEAD_STANDARD && R != 0)
    return fail(h, RV_ERR_SHAPE, "standard verification has no template: R must be 0 (got %d)", R);
  const int Lb = block_len(h, gamma, R);
  const size_t nq = static_cast<size_t>(B) * Lb * c.n_q_heads * c.head_dim * es;
  const size_t nkv = static_cast<size_t>(B) * Lb * c.n_kv_heads * c.head_dim * es;
  const size_t nh = static_cast<size_t>(B) * (Lb + 1) * c.hidden * es;
  const size_t nd = static_cast<size_t>(B) * gamma * 4, nc = static_cast<size_t>(B) * 4;
  const size_t npr = static_cast<size_t>(n_prompt) * 4, npx = static_cast<size_t>(B) * n_prefix * 4;
  const size_t nbl = static_cast<size_t>(B) * Lb * 4;
  const size_t P = static_cast<size_t>(B) * (gamma + 1);
  Workspace& w = h->ws;
  cudaError_t e = cudaSuccess;
  if (!h->pin_in) {  // first call: pinned host mirrors of the small regions
    e = cudaHostAlloc(reinterpret_cast<void**>(&h->pin_in), w.small_in_bytes, cudaHostAllocDefault);
    if (e == cudaSuccess)
      e = cudaHostAlloc(reinterpret_cast<void**>(&h->pin_out), w.small_out_bytes,
                        cudaHostAllocDefault);
    if (e != cudaSuccess) {
      if (h->pin_in) cudaFreeHost(h->pin_in);
      h->pin_in = h->pin_out = nullptr;
      return cuda_fail(h, e, "pinned staging cudaHostAlloc");
    }
  }
  // Contiguous layouts of this call's small inputs and outputs (16-byte aligned parts).
  size_t off = 0;
  auto part = [&off](size_t n) {
    const size_t o = off;
    off += (n + 15) & ~size_t(15);
    return o;
  };
  const size_t i_dr = part(nd), i_ci = part(nc), i_pr = part(do_pack ? npr : 0),
               i_px = part(do_pack ? npx : 0);
  const size_t in_small = off;
  off = 0;
  const size_t o_sc = part(P * RV_NSCORES * 4), o_am = part(P * 4), o_mg = part(nd),
               o_al = part(nc), o_nt = part(nc), o_co = part(nc), o_bl = part(do_pack ? nbl : 0),
               o_ps = part(do_pack ? nbl : 0), o_ac = part(static_cast<size_t>(B) * gamma);
  const size_t out_small = off;
  char* const hi = h->pin_in;
  std::memcpy(hi + i_dr, draft_ids_host, nd);
  std::memcpy(hi + i_ci, ctx_in_host, nc);
  if (do_pack) {
    if (npr) std::memcpy(hi + i_pr, prompt_ids_host, npr);
    if (npx) std::memcpy(hi + i_px, prefix_ids_host, npx);
  }
  // The kernels read the small inputs from the pinned staging `hi` and write
  // the small outputs into the pinned staging `ho` themselves (mapped host
  // memory), and the row gather reads the hidden states from the caller's
  // buffer when it is page-locked: only q / k_blk / v_blk (and attn_out) go
  // through copies, on the side stream beside the LM head.
  // (asked on every call: a buffer at a known address may have been freed and
  // replaced by pageable memory)
  const bool zc_hidden = pinned(hidden_host);
  char* const di = hi;
  char* const dout = h->pin_out;
  const size_t in_bytes = in_small + nh + nq + 2 * nkv;
  const size_t out_bytes = out_small + (attn_out_host ? nq : 0);
  auto I32 = [](char* p) { return reinterpret_cast<int32_t*>(p); };
  // The device part: copies in, the step, copies out (all stream-ordered).
  auto issue = [&]() -> int {
    // The hidden states first (when they are not read in place), on `stream`.
    // With the attention beside the head, q / k_blk / v_blk go on the side
    // stream once the row gather has run (the gather's reads of the hidden
    // states then have the host link to themselves, and the attention follows
    // its copies in stream order); otherwise on the side stream at once, and
    // `stream` waits for them before the attention that opens the step.
    const bool fork = attn_forks(h, B, Lb);
    const SideCopies copies{w.st_q, q_host, w.st_kb, k_blk_host, w.st_vb, v_blk_host, nq, nkv};
    cudaError_t e = cudaSuccess;
    if (!zc_hidden) e = cudaMemcpyAsync(w.st_hidden, hidden_host, nh, cudaMemcpyHostToDevice, s);
    if (!fork) {
      if (e == cudaSuccess) e = cudaEventRecord(h->ev_copy_start, s);
      if (e == cudaSuccess) e = cudaStreamWaitEvent(h->side, h->ev_copy_start, 0);
      if (e == cudaSuccess)
        e = cudaMemcpyAsync(w.st_q, q_host, nq, cudaMemcpyHostToDevice, h->side);
      if (e == cudaSuccess)
        e = cudaMemcpyAsync(w.st_kb, k_blk_host, nkv, cudaMemcpyHostToDevice, h->side);
      if (e == cudaSuccess)
        e = cudaMemcpyAsync(w.st_vb, v_blk_host, nkv, cudaMemcpyHostToDevice, h->side);
      if (e == cudaSuccess) e = cudaEventRecord(h->ev_copy_done, h->side);
      if (e == cudaSuccess) e = cudaStreamWaitEvent(s, h->ev_copy_done, 0);
    }
    if (e != cudaSuccess) return cuda_fail(h, e, "host->device copy");
    int rc = plain_step_mode(h);
    if (rc != RV_OK) return rc;
    rc = step_impl(h, w.st_q, w.st_kb, w.st_vb, k_cache, v_cache,
                   zc_hidden ? hidden_host : w.st_hidden, w_head, I32(di + i_dr),
                   do_pack ? I32(di + i_pr) : nullptr, do_pack ? I32(di + i_px) : nullptr,
                   I32(di + i_ci), B, gamma, n_prompt, n_prefix, alpha,
                   do_pack ? I32(dout + o_bl) : nullptr, do_pack ? I32(dout + o_ps) : nullptr,
                   w.st_attn, reinterpret_cast<float*>(dout + o_sc), I32(dout + o_am),
                   reinterpret_cast<float*>(dout + o_mg), reinterpret_cast<uint8_t*>(dout + o_ac),
                   I32(dout + o_al), I32(dout + o_nt), I32(dout + o_co), nullptr, stream, nullptr,
                   fork ? &copies : nullptr);
    if (rc != RV_OK) return rc;
    if (attn_out_host) e = cudaMemcpyAsync(attn_out_host, w.st_attn, nq, cudaMemcpyDeviceToHost, s);
    return e == cudaSuccess ? RV_OK : cuda_fail(h, e, "device->host copy");
  };
  // A call repeated with the same arguments (a serving loop reusing its pinned
  // buffers) is captured once as a CUDA graph and then replayed: one launch
  // instead of about twenty API calls.  Profiling (event records inside the
  // step) keeps the direct path.
  HostStepKey key{};
  {
    const void* ptrs[24] = {q_host, k_blk_host, v_blk_host, k_cache, v_cache, hidden_host, w_head,
                            prompt_ids_host, prefix_ids_host, block_ids_host, pos_ids_host,
                            attn_out_host, scores_host, argmax_host, margin_host, accept_mask_host,
                            accepted_len_host, next_token_host, ctx_out_host, draft_ids_host,
                            ctx_in_host, nullptr, nullptr, nullptr};
    std::memcpy(key.ptr, ptrs, sizeof(ptrs));
    key.dims[0] = B;
    key.dims[1] = gamma;
    key.dims[2] = n_prompt;
    key.dims[3] = n_prefix;
    key.dims[4] = zc_hidden ? 1 : 0;
    key.alpha = alpha;
    key.accept_mode = h->accept_mode;
    key.head_mode = h->head_mode;
    key.log_eps = h->accept_log_eps;
    key.log_delta = h->accept_log_delta;
    key.stream = stream;
  }
  bool replay = false;
  if (!h->graphs_off && h->profiling == 0) {
    if (h->host_graph && key.same(h->graph_key)) {
      replay = true;
    } else if (h->have_key && key.same(h->last_key) && s != nullptr &&
               pinned(q_host) && pinned(k_blk_host) && pinned(v_blk_host) &&
               zc_hidden && (!attn_out_host || pinned(attn_out_host))) {
      if (h->host_graph) {
        cudaGraphExecDestroy(h->host_graph);
        h->host_graph = nullptr;
      }
      // (the legacy default stream cannot be captured, nor can copies from
      // pageable memory; a capture that fails all the same leaves the
      // handle on the direct path)
      const unsigned long long before = h->launches;
      cudaError_t e = s ? cudaStreamBeginCapture(s, cudaStreamCaptureModeThreadLocal)
                        : cudaErrorStreamCaptureUnsupported;
      int rc = e == cudaSuccess ? issue() : RV_OK;
      cudaGraph_t g = nullptr;
      if (e == cudaSuccess) e = cudaStreamEndCapture(s, &g);
      if (rc != RV_OK && rc != RV_ERR_CUDA) {  // an argument error: the direct call's too
        if (g) cudaGraphDestroy(g);
        h->launches = before;
        return rc;
      }
      if (rc == RV_OK && e == cudaSuccess) e = cudaGraphInstantiate(&h->host_graph, g, 0);
      if (g) cudaGraphDestroy(g);
      if (rc == RV_OK && e == cudaSuccess) {
        h->graph_key = key;
        h->graph_launches = h->launches - before;
        replay = true;
      } else {
        cudaGetLastError();
        h->err.clear();
        h->host_graph = nullptr;
        h->graphs_off = true;
      }
      h->launches = before;
    }
    h->last_key = key;
    h->have_key = true;
  }
  if (replay) {
    e = cudaGraphLaunch(h->host_graph, s);
    if (e != cudaSuccess) return cuda_fail(h, e, "graph launch");
    h->launches += h->graph_launches;
  } else {
    const int rc = issue();
    if (rc != RV_OK) return rc;
  }
  e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(h, e, "device->host copy");
  const char* const ho = h->pin_out;
  std::memcpy(scores_host, ho + o_sc, P * RV_NSCORES * 4);
  std::memcpy(argmax_host, ho + o_am, P * 4);
  std::memcpy(margin_host, ho + o_mg, nd);
  std::memcpy(accept_mask_host, ho + o_ac, static_cast<size_t>(B) * gamma);
  std::memcpy(accepted_len_host, ho + o_al, nc);
  std::memcpy(next_token_host, ho + o_nt, nc);
  std::memcpy(ctx_out_host, ho + o_co, nc);
  if (do_pack) {
    std::memcpy(block_ids_host, ho + o_bl, nbl);
    std::memcpy(pos_ids_host, ho + o_ps, nbl);
  }
  if (h2d_bytes) *h2d_bytes = in_bytes;
  if (d2h_bytes) *d2h_bytes = out_bytes;
  return RV_OK;
}

extern "C" RV_API int rv_host_step_graphed(const rv_handle* h, int32_t* active) {
  if (!h || !active) return RV_ERR_INVALID_ARG;
  *active = h->host_graph != nullptr ? 1 : 0;
  return RV_OK;
}

// ============================================================================ status / timing

extern "C" RV_API int rv_read_status(rv_handle* h, void* stream, uint32_t* status) {
  if (!h || !status) return RV_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  unsigned v = 0;
  cudaError_t e = cudaStreamSynchronize(s);
  if (e == cudaSuccess) e = cudaMemcpy(&v, h->ws.status, sizeof(v), cudaMemcpyDeviceToHost);
  if (e == cudaSuccess) e = cudaMemset(h->ws.status, 0, sizeof(unsigned));
  if (e != cudaSuccess) return cuda_fail(h, e, "rv_read_status");
  *status = v;
  if (v != 0) return fail(h, RV_ERR_DEVICE, "device status 0x%x", v);
  return RV_OK;
}

extern "C" RV_API int rv_profile_enable(rv_handle* h, int32_t mask) {
  if (!h) return RV_ERR_INVALID_ARG;
  if (mask) {
    for (auto& r : h->prof) {
      if (r.ev.empty()) {
        r.ev.resize(2 * PROF_PAIRS);
        for (auto& ev : r.ev) {
          cudaError_t e = cudaEventCreate(&ev);
          if (e != cudaSuccess) return cuda_fail(h, e, "cudaEventCreate");
        }
      }
    }
  }
  h->profiling = static_cast<unsigned>(mask) & ((1u << RV_PROF_COUNT) - 1u);
  return RV_OK;
}

extern "C" RV_API int rv_profile_read(rv_handle* h, int32_t region, double* total_ms,
                                      int32_t* count) {
  if (!h || !total_ms || !count || region < 0 || region >= RV_PROF_COUNT) return RV_ERR_INVALID_ARG;
  ProfRegion& r = h->prof[region];
  double sum = 0;
  for (int i = 0; i < r.used; ++i) {
    cudaError_t e = cudaEventSynchronize(r.ev[2 * i + 1]);
    float ms = 0.f;
    if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, r.ev[2 * i], r.ev[2 * i + 1]);
    if (e != cudaSuccess) return cuda_fail(h, e, "rv_profile_read");
    sum += ms;
  }
  *total_ms = sum;
  *count = r.used;
  r.used = 0;
  return RV_OK;
}

extern "C" RV_API int rv_launch_count(const rv_handle* h, uint64_t* count) {
  if (!h || !count) return RV_ERR_INVALID_ARG;
  *count = h->launches;
  return RV_OK;
}
