// Router softmax and expert-choice top-k selection (arXiv 2604.01622, Sec. 2.2).
//
// Selection: for every expert e and group g (one sequence, Sec. 5.2) keep the k_g tokens
// with the largest S[t,e] (Sec. 2.2 TopC; capacity per group, Sec. 4.2). Ties go to the
// lower token index and the kept tokens are written in ascending index. One CTA per
// (e, g) runs an MSB-first radix select over order-preserving 32-bit keys of the fp32
// scores to find the k-th largest key, then compacts the column in index order with two
// block scans, which makes the result unique and independent of thread timing.
#include "common.cuh"
#include "kernels.h"

namespace ecmoe {

// ------------------------------------------------------------------ softmax over experts
// 32 tokens per CTA; the S^T tile is staged in shared memory so both layouts are written
// with coalesced stores.
__global__ void softmax_rows_kernel(const float* __restrict__ Z, const float* __restrict__ br,
                                    float* __restrict__ S, float* __restrict__ ST, int N, int E) {
  extern __shared__ float tile[];  // [32][E+1]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  const int t0 = blockIdx.x * 32;
  for (int r = warp; r < 32; r += nw) {
    const int t = t0 + r;
    if (t >= N) break;
    const float* z = Z + (size_t)t * E;
    float mx = -INFINITY;
    for (int e = lane; e < E; e += 32) {
      float v = z[e] + (br ? br[e] : 0.0f);
      tile[r * (E + 1) + e] = v;
      mx = fmaxf(mx, v);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    float sum = 0.f;
    for (int e = lane; e < E; e += 32) {
      float p = expf(tile[r * (E + 1) + e] - mx);
      tile[r * (E + 1) + e] = p;
      sum += p;
    }
    sum = warp_sum(sum);
    const float inv = 1.0f / sum;
    for (int e = lane; e < E; e += 32) {
      float p = tile[r * (E + 1) + e] * inv;
      tile[r * (E + 1) + e] = p;
      S[(size_t)t * E + e] = p;
    }
  }
  __syncthreads();
  for (int e = warp; e < E; e += nw) {
    const int t = t0 + lane;
    if (t < N) ST[(size_t)e * N + t] = tile[lane * (E + 1) + e];
  }
}

cudaError_t launch_softmax_rows(const float* Z, const float* br, float* S, float* ST, int N, int E,
                                cudaStream_t st) {
  if (N == 0) return cudaSuccess;
  size_t smem = (size_t)32 * (E + 1) * sizeof(float);
  if (smem > 48 * 1024)
    cudaFuncSetAttribute(softmax_rows_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  softmax_rows_kernel<<<(N + 31) / 32, 256, smem, st>>>(Z, br, S, ST, N, E);
  return cudaGetLastError();
}

__global__ void transpose_scores_kernel(const float* __restrict__ ST, float* __restrict__ S, int N,
                                        int E) {
  __shared__ float tile[32][33];
  const int t0 = blockIdx.x * 32, e0 = blockIdx.y * 32;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;  // 256 threads: 8 rows per pass
  for (int r = ty; r < 32; r += 8) {
    int e = e0 + r, t = t0 + tx;
    if (e < E && t < N) tile[r][tx] = ST[(size_t)e * N + t];
  }
  __syncthreads();
  for (int r = ty; r < 32; r += 8) {
    int t = t0 + r, e = e0 + tx;
    if (e < E && t < N) S[(size_t)t * E + e] = tile[tx][r];
  }
}

cudaError_t launch_transpose_scores(const float* ST, float* S, int N, int E, cudaStream_t st) {
  if (N == 0) return cudaSuccess;
  dim3 grid((N + 31) / 32, (E + 31) / 32);
  transpose_scores_kernel<<<grid, 256, 0, st>>>(ST, S, N, E);
  return cudaGetLastError();
}

// ------------------------------------------------------------------ top-k selection
// Order-preserving key: larger float -> larger unsigned key; -0.0 is folded onto +0.0.
__device__ __forceinline__ uint32_t score_key(float s) {
  uint32_t u = __float_as_uint(s);
  if (u == 0x80000000u) u = 0u;
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Exclusive scan of one int per thread across the block (blockDim multiple of 32).
__device__ __forceinline__ int block_excl_scan(int v, int* s_warp) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  int incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    int u = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += u;
  }
  if (lane == 31) s_warp[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    int w = lane < nw ? s_warp[lane] : 0;
    int wi = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      int u = __shfl_up_sync(0xffffffffu, wi, o);
      if (lane >= o) wi += u;
    }
    if (lane < nw) s_warp[lane] = wi - w;
  }
  __syncthreads();
  int r = incl - v + s_warp[warp];
  __syncthreads();
  return r;
}

template <bool SMEM>
__global__ void __launch_bounds__(512)
topk_kernel(const float* __restrict__ ST, int N, int E, const int* __restrict__ group_off,
            const int* __restrict__ k_g, const int* __restrict__ k_off, int M,
            int* __restrict__ idx, float* __restrict__ gate, int* __restrict__ slot) {
  extern __shared__ uint32_t skeys[];
  __shared__ int hist[256];
  __shared__ int s_warp[32];
  __shared__ uint32_t s_prefix;
  __shared__ int s_remaining;
  const int e = blockIdx.x, g = blockIdx.y;
  const int tid = threadIdx.x, nthr = blockDim.x, lane = tid & 31, warp = tid >> 5;
  const int lo = group_off[g];
  const int L = group_off[g + 1] - lo;
  const int k = k_g[g];
  const int base = k_off[g];
  const float* col = ST + (size_t)e * N + lo;

  if (SMEM) {
    for (int i = tid; i < L; i += nthr) skeys[i] = score_key(col[i]);
    __syncthreads();
  }
  auto key_at = [&](int i) -> uint32_t { return SMEM ? skeys[i] : score_key(col[i]); };

  // Radix select of the k-th largest key, 8 bits per pass from the top.
  uint32_t T = 0xFFFFFFFFu;
  int need_eq = 0;
  if (k > 0) {
    uint32_t prefix = 0u, mask = 0u;
    int remaining = k;
    for (int pass = 0; pass < 4; ++pass) {
      const int shift = 24 - 8 * pass;
      for (int i = tid; i < 256; i += nthr) hist[i] = 0;
      __syncthreads();
      for (int i = tid; i < L; i += nthr) {
        uint32_t key = key_at(i);
        if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1);
      }
      __syncthreads();
      if (warp == 0) {
        // lane l owns bins 255-8l .. 248-8l (descending); find the bin holding the
        // remaining-th largest key
        int c[8], local = 0;
#pragma unroll
        for (int j = 0; j < 8; ++j) { c[j] = hist[255 - (lane * 8 + j)]; local += c[j]; }
        int incl = local;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          int u = __shfl_up_sync(0xffffffffu, incl, o);
          if (lane >= o) incl += u;
        }
        int excl = incl - local;
        if (excl < remaining && remaining <= incl) {
          int run = excl;
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            if (run + c[j] >= remaining) {
              uint32_t bin = 255u - (uint32_t)(lane * 8 + j);
              s_prefix = prefix | (bin << shift);
              s_remaining = remaining - run;
              break;
            }
            run += c[j];
          }
        }
      }
      __syncthreads();
      prefix = s_prefix;
      remaining = s_remaining;
      mask |= 0xFFu << shift;
      __syncthreads();
    }
    T = prefix;
    need_eq = remaining;
  }
  const bool any = k > 0;

  // Compaction in token order: thread tid owns a contiguous chunk.
  const int chunk = (L + nthr - 1) / nthr;
  const int i0 = min(L, tid * chunk), i1 = min(L, i0 + chunk);
  int n_eq = 0;
  if (any)
    for (int i = i0; i < i1; ++i) n_eq += key_at(i) == T;
  const int eq_before = block_excl_scan(n_eq, s_warp);
  int n_sel = 0;
  {
    int r = eq_before;
    for (int i = i0; i < i1; ++i) {
      const uint32_t key = key_at(i);
      const bool eq = any && key == T;
      n_sel += any && (key > T || (eq && r < need_eq));
      r += eq;
    }
  }
  const int sel_before = block_excl_scan(n_sel, s_warp);
  int r = eq_before, pos = sel_before;
  int* idx_row = idx + (size_t)e * M + base;
  float* gate_row = gate + (size_t)e * M + base;
  for (int i = i0; i < i1; ++i) {
    const uint32_t key = key_at(i);
    const bool eq = any && key == T;
    const bool s = any && (key > T || (eq && r < need_eq));
    r += eq;
    const int t = lo + i;
    if (s) {
      idx_row[pos] = t;
      gate_row[pos] = col[i];
      slot[(size_t)t * E + e] = base + pos;
      ++pos;
    } else {
      slot[(size_t)t * E + e] = -1;
    }
  }
}

cudaError_t launch_topk(const float* ST, int N, int E, int G, const int* group_off, const int* k_g,
                        const int* k_off, int M, int max_group, int* idx, float* gate, int* slot,
                        cudaStream_t st) {
  if (G == 0 || E == 0) return cudaSuccess;
  dim3 grid(E, G);
  const int threads = max_group >= 4096 ? 512 : (max_group >= 1024 ? 256 : 128);
  const size_t smem = (size_t)max_group * sizeof(uint32_t);
  if (smem <= 200 * 1024) {
    if (smem > 48 * 1024)
      cudaFuncSetAttribute(topk_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)smem);
    topk_kernel<true><<<grid, threads, smem, st>>>(ST, N, E, group_off, k_g, k_off, M, idx, gate,
                                                   slot);
  } else {
    topk_kernel<false><<<grid, threads, 0, st>>>(ST, N, E, group_off, k_g, k_off, M, idx, gate,
                                                 slot);
  }
  return cudaGetLastError();
}

}  // namespace ecmoe
