// rv_verify_head_static: the LM-head step (rv_verify_head) for callers that
// cannot allocate device memory -- for example code that runs where
// cudaMalloc is forbidden or unavailable (inside a host callback, under a
// memory allocator that owns the whole device, or in a plug-in whose host
// process forbids extra allocations).  It needs no handle: its scratch (the
// per-CTA partial statistics, the gathered hidden rows and a status word)
// lives in one file-scope __device__ array of fixed size that every GPU which
// loads this library holds until the process exits.
//
// The first call on a device (with that device current) looks up the array's
// device address with cudaGetSymbolAddress and configures the kernel; make
// that first call before any stream capture.  Later calls only launch.
// Calls share the array, so calls that overlap on the GPU (different streams
// without ordering) race; calls ordered on one stream are fine.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <mutex>

#include "rv.h"
#include "rv_kernels.h"

using namespace rv;

namespace {

constexpr size_t round256(size_t x) { return (x + 255) / 256 * 256; }
constexpr size_t ST_OFF_STATUS = 0;
constexpr size_t ST_OFF_GATHER = 256;
constexpr size_t ST_OFF_PART =
    ST_OFF_GATHER + round256(static_cast<size_t>(RV_STATIC_MAX_PAIRS) * GATHER_FIELDS * 4);
constexpr int ST_MAX_SLOTS = 256;
constexpr size_t ST_OFF_HSEL =
    ST_OFF_PART +
    round256(static_cast<size_t>(ST_MAX_SLOTS) * RV_STATIC_MAX_PAIRS * HEAD_STAT_FIELDS * 4);
// gathered rows: 2 * round_up(P, 8) <= 2 * RV_STATIC_MAX_PAIRS rows of H bf16
constexpr size_t ST_BYTES =
    ST_OFF_HSEL + static_cast<size_t>(2) * RV_STATIC_MAX_PAIRS * RV_STATIC_MAX_HIDDEN * 2;

constexpr int ST_MAX_DEVICES = 64;

struct DeviceState {
  bool ready = false;
  char* scratch = nullptr;  // device address of rv_static_scratch on this device
  int num_sms = 0;
  size_t smem_optin = 0;
  PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
};

std::mutex g_mu;
DeviceState g_dev[ST_MAX_DEVICES];

}  // namespace

static __device__ __align__(256) unsigned char rv_static_scratch[ST_BYTES];

namespace {

// Once per device: device check, symbol address, kernel attribute, encoder.
int device_setup(DeviceState** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= ST_MAX_DEVICES) return RV_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_mu);
  DeviceState& d = g_dev[dev];
  if (!d.ready) {
    cudaDeviceProp prop;
    if (cudaGetDeviceProperties(&prop, dev) != cudaSuccess) return RV_ERR_CUDA;
    if (!(prop.major == 10 && prop.minor == 3)) return RV_ERR_UNSUPPORTED;
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, rv_static_scratch) != cudaSuccess || ptr == nullptr) {
      cudaGetLastError();
      return RV_ERR_CUDA;
    }
    if (head_tc_configure(prop.sharedMemPerBlockOptin) != cudaSuccess) return RV_ERR_CUDA;
    cudaDriverEntryPointQueryResult q;
    void* fn = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || fn == nullptr)
      return RV_ERR_CUDA;
    d.scratch = static_cast<char*>(ptr);
    d.num_sms = prop.multiProcessorCount;
    d.smem_optin = prop.sharedMemPerBlockOptin;
    d.encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    d.ready = true;
  }
  *out = &d;
  return RV_OK;
}

bool encode_2d(PFN_cuTensorMapEncodeTiled_v12000 enc, CUtensorMap* m, const void* ptr,
               int inner, int outer, int box_inner, int box_outer) {
  const cuuint64_t dims[2] = {static_cast<cuuint64_t>(inner), static_cast<cuuint64_t>(outer)};
  const cuuint64_t strides[1] = {static_cast<cuuint64_t>(inner) * 2};
  const cuuint32_t box[2] = {static_cast<cuuint32_t>(box_inner), static_cast<cuuint32_t>(box_outer)};
  const cuuint32_t es[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

extern "C" RV_API int rv_verify_head_static(const void* hidden, const void* w_head,
                                            const int32_t* draft_ids, int32_t B, int32_t gamma,
                                            int32_t R, int32_t vocab, int32_t hidden_size,
                                            float alpha, float* scores, int32_t* argmax,
                                            float* margin, uint32_t* dev_status, void* stream) {
  if (B < 1 || gamma < 1 || R < 0 || vocab < 1 || hidden_size < 8 || hidden_size % 8 != 0)
    return RV_ERR_SHAPE;
  if (static_cast<long long>(B) * (gamma + 1) > RV_STATIC_MAX_PAIRS ||
      hidden_size > RV_STATIC_MAX_HIDDEN)
    return RV_ERR_CAPACITY;
  if (!std::isfinite(alpha)) return RV_ERR_INVALID_ARG;
  if (!hidden || !w_head || !draft_ids || !scores || !argmax || !margin)
    return RV_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(hidden) & 15u) || (reinterpret_cast<uintptr_t>(w_head) & 15u))
    return RV_ERR_INVALID_ARG;
  DeviceState* d = nullptr;
  int rc = device_setup(&d);
  if (rc != RV_OK) return rc;

  // One chunk of P <= RV_STATIC_MAX_PAIRS pairs; vocab split in whole tiles.
  HeadPlan pl;
  pl.pair = false;
  pl.P = B * (gamma + 1);
  pl.n_chunks = 1;
  pl.pairs_per_chunk = pl.P;
  pl.pad_pairs = (pl.P + 7) / 8 * 8;
  pl.N = 2 * pl.pad_pairs;
  pl.n_vtiles = (vocab + HEAD_TILE_ROWS - 1) / HEAD_TILE_ROWS;
  pl.slots = std::max(1, std::min({d->num_sms, pl.n_vtiles, ST_MAX_SLOTS}));

  char* s = d->scratch;
  unsigned* status = dev_status ? reinterpret_cast<unsigned*>(dev_status)
                                : reinterpret_cast<unsigned*>(s + ST_OFF_STATUS);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  // The shared array keeps the previous call's contents: the status word must
  // start at zero (the LM head's tile counter is zeroed by the prep launch).
  // Partials and gathered rows are fully rewritten each call.
  if (!dev_status && cudaMemsetAsync(s + ST_OFF_STATUS, 0, sizeof(unsigned), st) != cudaSuccess)
    return RV_ERR_CUDA;
  HeadArgs a{hidden, w_head, draft_ids, B, gamma, R, vocab, hidden_size, alpha,
             reinterpret_cast<float*>(s + ST_OFF_PART), reinterpret_cast<float*>(s + ST_OFF_GATHER),
             status, reinterpret_cast<unsigned*>(s + ST_OFF_STATUS + 64),
             reinterpret_cast<unsigned*>(s + ST_OFF_STATUS + 128)};
  HeadTcLaunch l;
  l.stages = head_tc_stages(pl.N, pl.pad_pairs, d->smem_optin);
  l.unit_rows = HEAD_TILE_ROWS;
  l.smem_bytes = head_tc_smem_bytes(pl.N, pl.pad_pairs, l.stages);
  if (l.stages < 2) return RV_ERR_UNSUPPORTED;
  if (!encode_2d(d->encode, &l.tm_w, w_head, hidden_size, vocab, 64, HEAD_TILE_ROWS) ||
      !encode_2d(d->encode, &l.tm_w16, w_head, hidden_size, vocab, 64, HEAD_W_BOX_ROWS) ||
      !encode_2d(d->encode, &l.tm_h, s + ST_OFF_HSEL, hidden_size, pl.N, 64, pl.N))
    return RV_ERR_CUDA;
  if (launch_prep(a, pl, s + ST_OFF_HSEL, nullptr, st) != cudaSuccess) return RV_ERR_CUDA;
  if (launch_head_tc(a, pl, l, nullptr, st) != cudaSuccess) return RV_ERR_CUDA;
  if (launch_head_finalize(a, pl, scores, argmax, margin, nullptr, st) != cudaSuccess)
    return RV_ERR_CUDA;
  return RV_OK;
}
