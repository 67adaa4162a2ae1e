// Token-choice (TC) routing, the comparison baseline of arXiv 2604.01622 Sec. 2.2: each
// token takes its top-k experts (ties to the lower expert index) with gates normalised over
// those k; a capacity C caps each expert, keeping its tokens in ascending token order
// (C < 0: dropless). Experts then own variable numbers of rows; each expert's rows are laid
// out in a region padded to a multiple of PADR rows (zero rows in the padding) so the
// grouped GEMMs can tile them without straddling experts.
#include "common.cuh"
#include "kernels.h"

namespace ecmoe {

namespace {
constexpr int kPadRows = 256;   // must match the GEMM's variable-row padding unit

// Exclusive scan of one int per thread across the block (blockDim multiple of 32, <= 1024).
__device__ __forceinline__ int block_scan_excl(int v, int* s_warp, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  int incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int u = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += u;
  }
  if (lane == 31) s_warp[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    const int w = lane < nw ? s_warp[lane] : 0;
    int wi = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int u = __shfl_up_sync(0xffffffffu, wi, o);
      if (lane >= o) wi += u;
    }
    if (lane < nw) s_warp[lane] = wi - w;
    if (lane == nw - 1) s_warp[32] = wi;
  }
  __syncthreads();
  const int r = incl - v + s_warp[warp];
  *total = s_warp[32];
  __syncthreads();
  return r;
}
}  // namespace

// One warp per token: k rounds of a warp argmax over the E scores (larger score first, then
// lower expert index). Writes the choices best first, normalised gates and their sum Z.
__global__ void tc_topk_rows_kernel(const float* __restrict__ S, int N, int E, int k,
                                    int* __restrict__ choice, float* __restrict__ tgate,
                                    float* __restrict__ Z) {
  const int t = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (t >= N) return;
  const float* row = S + (size_t)t * E;
  uint32_t taken[16] = {};   // bit e%32 of word e/32: expert e already chosen (E <= 512)
  float sum = 0.f;
  int my_e = 0;              // lane r keeps the r-th choice
  for (int r = 0; r < k; ++r) {
    float best = -INFINITY;
    int bi = 0x7fffffff;
    for (int e = lane; e < E; e += 32) {
      if (taken[e >> 5] & (1u << (e & 31))) continue;
      float v = row[e] + 0.0f;
      if (v != v) v = -INFINITY;   // a NaN score ranks last, so every round finds an expert
      if (v > best || (v == best && e < bi)) { best = v; bi = e; }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, best, o);
      const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
      if (ov > best || (ov == best && oi < bi)) { best = ov; bi = oi; }
    }
    taken[bi >> 5] |= 1u << (bi & 31);   // every lane holds the same winner
    if (lane == r) my_e = bi;
    sum += row[bi];
  }
  if (lane < k) {
    choice[(size_t)t * k + lane] = my_e;
    tgate[(size_t)t * k + lane] = row[my_e] / sum;
  }
  if (lane == 0) Z[t] = sum;
}

// Per expert (one CTA): how many tokens chose it.
__global__ void tc_count_kernel(const int* __restrict__ choice, int N, int k,
                                int* __restrict__ count) {
  __shared__ int s_warp[33];
  __shared__ int s_total;
  const int e = blockIdx.x;
  int c = 0;
  for (int t = threadIdx.x; t < N; t += blockDim.x)
    for (int r = 0; r < k; ++r) c += choice[(size_t)t * k + r] == e;
  int tot;
  block_scan_excl(c, s_warp, &tot);
  if (threadIdx.x == 0) {
    s_total = tot;
    count[e] = s_total;
  }
}

// One thread: kept rows per expert (capped), padded region offsets in PADR-row blocks,
// and in count[E] the padded rows in use.
__global__ void tc_offsets_kernel(int E, int cap, int* __restrict__ count,
                                  int* __restrict__ tiles) {
  if (threadIdx.x != 0 || blockIdx.x != 0) return;
  int acc = 0;
  tiles[0] = 0;
  for (int e = 0; e < E; ++e) {
    int c = count[e];
    if (cap >= 0 && c > cap) c = cap;
    count[e] = c;
    acc += (c + kPadRows - 1) / kPadRows;
    tiles[e + 1] = acc;
  }
  count[E] = acc * kPadRows;
}

// Per expert (one CTA): walk tokens in order, give the first count[e] that chose e their rows
// (row-to-token map, gate, slot map), mark the rest dropped, zero-fill the padding rows.
__global__ void tc_fill_kernel(const int* __restrict__ choice, const float* __restrict__ tgate,
                               int N, int E, int k, const int* __restrict__ count,
                               const int* __restrict__ tiles, int* __restrict__ row_token,
                               float* __restrict__ row_gate, int* __restrict__ slot,
                               int* __restrict__ kept) {
  __shared__ int s_warp[33];
  const int e = blockIdx.x;
  const int kept_e = count[e];
  const int base = tiles[e] * kPadRows;
  const int end = tiles[e + 1] * kPadRows;
  int before = 0;   // tokens that chose e in earlier chunks
  for (int t0 = 0; t0 < N; t0 += blockDim.x) {
    const int t = t0 + threadIdx.x;
    int r_hit = -1;
    if (t < N)
      for (int r = 0; r < k; ++r)
        if (choice[(size_t)t * k + r] == e) r_hit = r;
    int chunk_total;
    const int pos = before + block_scan_excl(r_hit >= 0, s_warp, &chunk_total);
    if (r_hit >= 0) {
      const bool keep = pos < kept_e;
      kept[(size_t)t * k + r_hit] = keep;
      if (keep) {
        row_token[base + pos] = t;
        row_gate[base + pos] = tgate[(size_t)t * k + r_hit];
        slot[(size_t)t * E + e] = base + pos;
      }
    }
    before += chunk_total;
  }
  for (int row = base + kept_e + threadIdx.x; row < end; row += blockDim.x) {
    row_token[row] = -1;
    row_gate[row] = 0.f;
  }
}

cudaError_t launch_tc_route(const float* S, int N, int E, int k, int cap, int* choice,
                            float* tgate, float* Z, int* count, int* tiles, int* row_token,
                            float* row_gate, int* slot, int* kept, cudaStream_t st) {
  if (N == 0) return cudaSuccess;
  cudaError_t e = cudaMemsetAsync(slot, 0xFF, (size_t)N * E * sizeof(int), st);   // -1
  if (e != cudaSuccess) return e;
  tc_topk_rows_kernel<<<(N + 7) / 8, 256, 0, st>>>(S, N, E, k, choice, tgate, Z);
  tc_count_kernel<<<E, 512, 0, st>>>(choice, N, k, count);
  tc_offsets_kernel<<<1, 32, 0, st>>>(E, cap, count, tiles);
  tc_fill_kernel<<<E, 512, 0, st>>>(choice, tgate, N, E, k, count, tiles, row_token, row_gate,
                                    slot, kept);
  return cudaGetLastError();
}

// Gradient through the normalised gates and the softmax, one warp per token:
// dS_tj = (dg_tj - sum_{j' kept} dg_tj' g_tj') / Z_t for the k chosen j (dg = 0 if dropped),
// dZ = S * (dS - <dS, S>). dg comes from the per-row gate gradients through the slot map;
// lane r < k holds the token's r-th choice.
__global__ void tc_softmax_bwd_kernel(const float* __restrict__ S, const int* __restrict__ choice,
                                      const float* __restrict__ tgate, const float* __restrict__ Z,
                                      const int* __restrict__ slot,
                                      const float* __restrict__ row_dgate, float* __restrict__ dZ,
                                      bf16* __restrict__ dZb, int N, int E, int Ep, int k) {
  const int t = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (t >= N) return;
  int my_e = -1;
  float dg = 0.f, g = 0.f, s_e = 0.f;
  if (lane < k) {
    my_e = choice[(size_t)t * k + lane];
    const int row = slot[(size_t)t * E + my_e];
    dg = row >= 0 ? row_dgate[row] : 0.f;
    g = tgate[(size_t)t * k + lane];
    s_e = S[(size_t)t * E + my_e];
  }
  const float common = warp_sum(dg * g);
  const float my_ds = lane < k ? (dg - common) / Z[t] : 0.f;
  const float dot = warp_sum(my_ds * s_e);
  for (int e = lane; e < Ep; e += 32) {   // Ep is a multiple of 32: every lane iterates alike
    float ds = 0.f;
    for (int r = 0; r < k; ++r) {
      const int er = __shfl_sync(0xffffffffu, my_e, r);
      const float dr = __shfl_sync(0xffffffffu, my_ds, r);
      if (er == e) ds = dr;
    }
    float z = 0.f;
    if (e < E) {
      z = S[(size_t)t * E + e] * (ds - dot);
      dZ[(size_t)t * E + e] = z;
    }
    if (dZb) {
      const bf16 hi = __float2bfloat16_rn(z);
      dZb[(size_t)t * Ep + e] = hi;
      dZb[(size_t)N * Ep + (size_t)t * Ep + e] = __float2bfloat16_rn(z - __bfloat162float(hi));
    }
  }
}

cudaError_t launch_tc_softmax_bwd(const float* S, const int* choice, const float* tgate,
                                  const float* Z, const int* slot, const float* row_dgate,
                                  float* dZ, bf16* dZb, int N, int E, int Ep, int k,
                                  cudaStream_t st) {
  if (N == 0) return cudaSuccess;
  if (k > 32 || Ep % 32) return cudaErrorInvalidValue;
  tc_softmax_bwd_kernel<<<(N + 7) / 8, 256, 0, st>>>(S, choice, tgate, Z, slot, row_dgate, dZ, dZb,
                                                     N, E, Ep, k);
  return cudaGetLastError();
}

}  // namespace ecmoe
