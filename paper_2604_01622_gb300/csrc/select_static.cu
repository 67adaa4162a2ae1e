// Expert-choice selection that allocates nothing, for callers that cannot call cudaMalloc.
//
// Some callers cannot allocate device memory at the point where they need a selection:
// code running under a fixed memory budget handed out by another runtime, code that must
// not grow the process's device footprint, or a runtime that forbids allocation calls once
// it is serving. ec_route needs a caller-sized workspace for its token->slot map and group
// tables. This variant keeps that scratch in one file-scope device array of fixed size
// instead, so the caller passes only the scores and the output buffers.
//
// The array is module memory: every GPU that loads this library holds it until the process
// exits. All calls share it, and it keeps the last call's contents: the group tables are
// rewritten by each call, and the slot map (the selection kernel's token->slot output, which
// this variant does not return) is only written, never read, so nothing has to start at
// zero or -1. Two calls whose work overlaps on the GPU (different streams,
// or different host threads) race on the array; order them.
#include <cuda.h>

#include <mutex>

#include "../../include/ecmoe.h"
#include "common.cuh"
#include "kernels.h"

namespace {

constexpr size_t kMaxScores = EC_STATIC_SELECT_MAX_SCORES;  // N * E
constexpr int kMaxGroups = EC_STATIC_SELECT_MAX_GROUPS;
constexpr size_t kTableInts = 3 * (size_t)(kMaxGroups + 1);   // group_off, k_g, k_off
constexpr size_t kScratchInts = kTableInts + kMaxScores;

// the three group tables (packed, see ec_select_static) and the slot map [N][E]
static __device__ __align__(256) int32_t g_select_scratch[kScratchInts];

// Device address of the array, looked up once per CUDA context (a device's primary context
// is replaced by cudaDeviceReset, and the module with the array is loaded into the new one
// at a new address). The key is the context's process-unique id, not its handle, which the
// driver may hand out again. In host code `g_select_scratch` names a host-side stand-in,
// never the device memory itself.
typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long*);

template <typename Fn>
Fn driver_fn(const char* name, int version) {
  void* p = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion(name, &p, version, cudaEnableDefault, &q) != cudaSuccess ||
      q != cudaDriverEntryPointSuccess)
    return nullptr;
  return reinterpret_cast<Fn>(p);
}

// id of the calling thread's current context, 0 if there is none yet
cudaError_t current_ctx_id(unsigned long long* id) {
  static CtxGetCurrentFn get_current = driver_fn<CtxGetCurrentFn>("cuCtxGetCurrent", 4000);
  static CtxGetIdFn get_id = driver_fn<CtxGetIdFn>("cuCtxGetId", 12000);
  *id = 0;
  if (!get_current || !get_id) return cudaErrorNotSupported;
  CUcontext ctx = nullptr;
  if (get_current(&ctx) != CUDA_SUCCESS) return cudaErrorInvalidValue;
  if (ctx && get_id(ctx, id) != CUDA_SUCCESS) return cudaErrorInvalidValue;
  return cudaSuccess;
}

constexpr int kMaxContexts = 64;
std::mutex g_mu;
unsigned long long g_ctx_id[kMaxContexts] = {};
int32_t* g_scratch_dev[kMaxContexts] = {};
int g_next = 0;

cudaError_t scratch_ptr(int32_t** out) {
  unsigned long long id = 0;
  cudaError_t e = current_ctx_id(&id);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(g_mu);
  if (id != 0)
    for (int i = 0; i < kMaxContexts; ++i)
      if (g_ctx_id[i] == id) {
        *out = g_scratch_dev[i];
        return cudaSuccess;
      }
  // first call in this context (the lookup also creates the device's primary context if the
  // thread has none yet)
  void* p = nullptr;
  e = cudaGetSymbolAddress(&p, g_select_scratch);
  if (e != cudaSuccess) return e;
  if (id == 0) {
    e = current_ctx_id(&id);
    if (e != cudaSuccess) return e;
  }
  if (id != 0) {
    g_ctx_id[g_next] = id;
    g_scratch_dev[g_next] = static_cast<int32_t*>(p);
    g_next = (g_next + 1) % kMaxContexts;
  }
  *out = static_cast<int32_t*>(p);
  return cudaSuccess;
}

}  // namespace

extern "C" ec_status ec_select_static(const float* S, int32_t N, int32_t E, int32_t G,
                                      const int32_t* group_off, const int32_t* k_g, int32_t* idx,
                                      float* gate, void* stream) {
  if (!S || !group_off || !k_g || !idx || !gate) return EC_ERR_INVALID_ARG;
  if (N < 0 || E <= 0 || G <= 0) return EC_ERR_SHAPE;
  if ((size_t)N * (size_t)E > kMaxScores || G > kMaxGroups) return EC_ERR_UNSUPPORTED;
  if (group_off[0] != 0 || group_off[G] != N) return EC_ERR_SHAPE;
  // The group tables are copied into this call's own host array (group_off, k_g and the
  // prefix sums k_off, packed), so the caller may reuse or free its arrays, pinned or not, as
  // soon as the call returns: the copy from this pageable array is staged by the driver
  // before cudaMemcpyAsync returns.
  int32_t tbl[3 * (kMaxGroups + 1)];
  int32_t* t_goff = tbl;
  int32_t* t_kg = tbl + (G + 1);
  int32_t* t_koff = tbl + (2 * G + 1);
  t_koff[0] = 0;
  int max_group = 0;
  for (int g = 0; g < G; ++g) {
    const int L = group_off[g + 1] - group_off[g];
    if (L < 0 || k_g[g] < 0 || k_g[g] > L) return EC_ERR_SHAPE;
    if ((int64_t)t_koff[g] + k_g[g] > INT32_MAX) return EC_ERR_UNSUPPORTED;
    t_goff[g] = group_off[g];
    t_kg[g] = k_g[g];
    t_koff[g + 1] = t_koff[g] + k_g[g];
    if (L > max_group) max_group = L;
  }
  t_goff[G] = group_off[G];
  const int M = t_koff[G];
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  // A stream capture would record the host table's address, which does not outlive this
  // call: refuse before anything is enqueued.
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  cudaError_t ce = cudaStreamIsCapturing(st, &cap);
  if (ce == cudaErrorStreamCaptureImplicit || (ce == cudaSuccess && cap != cudaStreamCaptureStatusNone)) {
    cudaGetLastError();   // leave no error behind for the caller's next launch check
    return EC_ERR_UNSUPPORTED;
  }
  if (ce != cudaSuccess) {
    cudaGetLastError();
    return EC_ERR_CUDA;
  }
  int32_t* base = nullptr;
  if (scratch_ptr(&base) != cudaSuccess) return EC_ERR_CUDA;
  int32_t* d_goff = base;
  int32_t* d_kg = base + (G + 1);
  int32_t* d_koff = base + (2 * G + 1);
  int32_t* d_slot = base + kTableInts;
  if (cudaMemcpyAsync(base, tbl, (size_t)(3 * G + 2) * sizeof(int32_t), cudaMemcpyHostToDevice,
                      st) != cudaSuccess)
    return EC_ERR_CUDA;
  if (ecmoe::launch_topk(S, N, E, G, d_goff, d_kg, d_koff, M, max_group, idx, gate, d_slot, st) !=
      cudaSuccess)
    return EC_ERR_CUDA;
  return EC_OK;
}
