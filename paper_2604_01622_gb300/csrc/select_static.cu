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
#include <mutex>

#include "../../include/ecmoe.h"
#include "common.cuh"
#include "kernels.h"

namespace {

constexpr size_t kMaxScores = EC_STATIC_SELECT_MAX_SCORES;  // N * E
constexpr int kMaxGroups = EC_STATIC_SELECT_MAX_GROUPS;
constexpr size_t kTableInts = 3 * (size_t)(kMaxGroups + 1);   // group_off, k_g, k_off
constexpr size_t kScratchInts = kTableInts + kMaxScores;

// slot map [N][E] and the three group tables
static __device__ __align__(256) int32_t g_select_scratch[kScratchInts];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
int32_t* g_scratch_dev[kMaxDevices] = {};

// Device address of the array on the current device, looked up once per device. In host
// code `g_select_scratch` names a host-side stand-in, never the device memory itself.
cudaError_t scratch_ptr(int32_t** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_scratch_dev[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_select_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_dev[dev] = static_cast<int32_t*>(p);
  }
  *out = g_scratch_dev[dev];
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
  int32_t koff[kMaxGroups + 1];
  koff[0] = 0;
  int max_group = 0;
  for (int g = 0; g < G; ++g) {
    const int L = group_off[g + 1] - group_off[g];
    if (L < 0 || k_g[g] < 0 || k_g[g] > L) return EC_ERR_SHAPE;
    if ((int64_t)koff[g] + k_g[g] > INT32_MAX) return EC_ERR_UNSUPPORTED;
    koff[g + 1] = koff[g] + k_g[g];
    if (L > max_group) max_group = L;
  }
  const int M = koff[G];
  int32_t* base = nullptr;
  if (scratch_ptr(&base) != cudaSuccess) return EC_ERR_CUDA;
  int32_t* d_goff = base;
  int32_t* d_kg = base + (kMaxGroups + 1);
  int32_t* d_koff = base + 2 * (kMaxGroups + 1);
  int32_t* d_slot = base + kTableInts;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (cudaMemcpyAsync(d_goff, group_off, (G + 1) * sizeof(int32_t), cudaMemcpyHostToDevice, st) !=
          cudaSuccess ||
      cudaMemcpyAsync(d_kg, k_g, G * sizeof(int32_t), cudaMemcpyHostToDevice, st) != cudaSuccess ||
      cudaMemcpyAsync(d_koff, koff, (G + 1) * sizeof(int32_t), cudaMemcpyHostToDevice, st) !=
          cudaSuccess)
    return EC_ERR_CUDA;
  if (ecmoe::launch_topk(S, N, E, G, d_goff, d_kg, d_koff, M, max_group, idx, gate, d_slot, st) !=
      cudaSuccess)
    return EC_ERR_CUDA;
  return EC_OK;
}
