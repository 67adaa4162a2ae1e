// Bandwidth kernels of the EC-MoE layer: token-major gather into expert rows, gated combine
// (arXiv 2604.01622, Sec. 2.2: y_t = sum_{e: t in T_e} g_te FFN_e(x_t)), and their
// backward (gate gradient, softmax Jacobian, scatter of the input gradient).
//
// The token->slot map slot[t][e] (row m of expert e, or -1) makes every per-token sum run
// over experts in ascending order with no atomics, so results are deterministic.
#include <algorithm>

#include <type_traits>

#include "common.cuh"
#include "kernels.h"

namespace ecmoe {

// Grid of 256-thread blocks for a grid-stride loop over n elements, capped at `cap` blocks.
static unsigned grid_for(int64_t n, int64_t cap) {
  const int64_t b = (n + 255) / 256;
  return (unsigned)(b < cap ? b : cap);
}

// ------------------------------------------------------------------ per-token pair lists
// Fills s_m/s_g (slot row, gate) of the experts that chose token t, ascending e. Returns count.
__device__ __forceinline__ int token_pairs(const int* __restrict__ slot, const float* __restrict__ gate,
                                           int t, int E, int M, int* s_e, int* s_m, float* s_g,
                                           int* s_cnt) {
  if (threadIdx.x < 32) {
    const int lane = threadIdx.x;
    int cnt = 0;
    for (int e0 = 0; e0 < E; e0 += 32) {
      const int e = e0 + lane;
      const int m = e < E ? slot[(size_t)t * E + e] : -1;
      const unsigned ball = __ballot_sync(0xffffffffu, m >= 0);
      if (m >= 0) {
        const int p = cnt + __popc(ball & ((1u << lane) - 1u));
        s_e[p] = e;
        s_m[p] = m;
        if (s_g) s_g[p] = gate ? gate[(size_t)e * M + m] : 1.0f;
      }
      cnt += __popc(ball);
    }
    if (lane == 0) *s_cnt = cnt;
  }
  __syncthreads();
  return *s_cnt;
}

// ------------------------------------------------------------------ combine Y_t = sum g * O
template <typename T>
__global__ void combine_kernel(const T* __restrict__ O, const float* __restrict__ gate,
                               const int* __restrict__ slot, const T* __restrict__ R,
                               const T* __restrict__ R2, T* __restrict__ Y, int N, int E, int M,
                               int d) {
  extern __shared__ int sh[];
  int* s_e = sh;
  int* s_m = sh + E;
  float* s_g = reinterpret_cast<float*>(sh + 2 * E);
  __shared__ int s_cnt;
  const int t = blockIdx.x;
  const int cnt = token_pairs(slot, gate, t, E, M, s_e, s_m, s_g, &s_cnt);
  constexpr int VN = 16 / sizeof(T);
  const int nv = d / VN;
  // each thread sums two 16-byte column groups of the row (v and v + blockDim), eight O loads
  // in flight; rows are summed in ascending expert order
  const uint4* ob = reinterpret_cast<const uint4*>(O);
  const int64_t rs = d / VN;   // uint4 per row
  for (int v0 = threadIdx.x; v0 < nv; v0 += 2 * blockDim.x) {
    const int v1 = v0 + blockDim.x;
    const bool two = v1 < nv;
    float acc0[VN], acc1[VN];
#pragma unroll
    for (int j = 0; j < VN; ++j) acc0[j] = acc1[j] = 0.f;
    if (R) {
      unpack16(__ldg(reinterpret_cast<const uint4*>(R + (size_t)t * d) + v0), acc0, T());
      if (two) unpack16(__ldg(reinterpret_cast<const uint4*>(R + (size_t)t * d) + v1), acc1, T());
    }
    if (R2) {
      float r[VN];
      unpack16(__ldg(reinterpret_cast<const uint4*>(R2 + (size_t)t * d) + v0), r, T());
#pragma unroll
      for (int j = 0; j < VN; ++j) acc0[j] += r[j];
      if (two) {
        unpack16(__ldg(reinterpret_cast<const uint4*>(R2 + (size_t)t * d) + v1), r, T());
#pragma unroll
        for (int j = 0; j < VN; ++j) acc1[j] += r[j];
      }
    }
    // up to four pairs per batch (the last batch partial), all their loads issued first
    for (int p = 0; p < cnt; p += 4) {
      const int nb = cnt - p < 4 ? cnt - p : 4;
      uint4 u0[4], u1[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        u0[q] = u1[q] = make_uint4(0, 0, 0, 0);
        if (q < nb) {
          const int64_t row = (int64_t)s_e[p + q] * M + s_m[p + q];
          u0[q] = __ldg(ob + row * rs + v0);
          if (two) u1[q] = __ldg(ob + row * rs + v1);
        }
      }
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        if (q < nb) {
          float o[VN];
          const float g = s_g[p + q];
          unpack16(u0[q], o, T());
#pragma unroll
          for (int j = 0; j < VN; ++j) acc0[j] = fmaf(g, o[j], acc0[j]);
          unpack16(u1[q], o, T());
#pragma unroll
          for (int j = 0; j < VN; ++j) acc1[j] = fmaf(g, o[j], acc1[j]);
        }
      }
    }
    reinterpret_cast<uint4*>(Y + (size_t)t * d)[v0] = pack16(acc0, T());
    if (two) reinterpret_cast<uint4*>(Y + (size_t)t * d)[v1] = pack16(acc1, T());
  }
}

template <typename T>
cudaError_t launch_combine(const T* O, const float* gate, const int* slot, const T* R, const T* R2,
                           T* Y, int N, int E, int M, int d, cudaStream_t st) {
  if (N == 0) return cudaSuccess;
  const size_t smem = (size_t)3 * E * sizeof(int);
  // two 16-byte column groups per thread: half a row's groups per CTA, 32 to 128 threads
  const int nv = d * (int)sizeof(T) / 16;
  const int threads = std::min(128, std::max(32, (nv / 2 + 31) / 32 * 32));
  combine_kernel<T><<<N, threads, smem, st>>>(O, gate, slot, R, R2, Y, N, E, M, d);
  return cudaGetLastError();
}

// ------------------------------------------------------------------ token-major scatter
// H[row] = X[t] for every (expert, row) that selected token t, one CTA per token: each X row
// is read once (an expert-major gather, row by row of H, would read it once per selecting
// expert, mostly from DRAM), and written to its rows in ascending expert order.
template <typename T>
__global__ void scatter_rows_kernel(const T* __restrict__ X, const int* __restrict__ slot,
                                    T* __restrict__ H, int N, int E, int M, int d) {
  extern __shared__ int sh[];
  int* s_e = sh;
  int* s_m = sh + E;
  __shared__ int s_cnt;
  const int t = blockIdx.x;
  const int cnt = token_pairs(slot, nullptr, t, E, M, s_e, s_m, nullptr, &s_cnt);
  if (cnt == 0) return;
  const int nv = d * (int)sizeof(T) / 16;
  const uint4* src = reinterpret_cast<const uint4*>(X + (size_t)t * d);
  for (int v = threadIdx.x; v < nv; v += blockDim.x) {
    const uint4 u = __ldg(src + v);
    for (int p = 0; p < cnt; ++p)
      reinterpret_cast<uint4*>(H + ((size_t)s_e[p] * M + s_m[p]) * d)[v] = u;
  }
}

template <typename T>
cudaError_t launch_scatter_rows(const T* X, const int* slot, T* H, int N, int E, int M, int d,
                                cudaStream_t st) {
  if (N == 0) return cudaSuccess;
  const size_t smem = (size_t)2 * E * sizeof(int);
  scatter_rows_kernel<T><<<N, 128, smem, st>>>(X, slot, H, N, E, M, d);
  return cudaGetLastError();
}

// Zero the padding rows of variable-row expert regions: rows count[e] .. 256*(tiles[e+1] -
// tiles[e]) - 1 of expert e's region (one warp per possible padding row).
template <typename T>
__global__ void zero_pad_rows_kernel(const int* __restrict__ count, const int* __restrict__ tiles,
                                     T* __restrict__ H, int E, int d) {
  const int64_t w = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  const int e = (int)(w / 256);
  if (e >= E) return;
  const int64_t row = (int64_t)tiles[e] * 256 + count[e] + (w % 256);
  if (row >= (int64_t)tiles[e + 1] * 256) return;
  uint4* dst = reinterpret_cast<uint4*>(H + row * d);
  const int nv = d * (int)sizeof(T) / 16;
  for (int v = lane; v < nv; v += 32) dst[v] = make_uint4(0, 0, 0, 0);
}

template <typename T>
cudaError_t launch_zero_pad_rows(const int* count, const int* tiles, T* H, int E, int d,
                                 cudaStream_t st) {
  const int64_t warps = (int64_t)E * 256;
  zero_pad_rows_kernel<T><<<(unsigned)((warps + 7) / 8), 256, 0, st>>>(count, tiles, H, E, d);
  return cudaGetLastError();
}

// ------------------------------------------------------------------ backward: dO = g dY_t, dgate = <dY_t, O>
template <typename T>
__global__ void bwd_gather_scale_kernel(const T* __restrict__ dY, const T* __restrict__ O,
                                        const int* __restrict__ idx, const float* __restrict__ gate,
                                        T* __restrict__ dO, float* __restrict__ dgate, int64_t P,
                                        int d) {
  const int64_t row = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= P) return;
  const int t = idx[row];
  const float g = gate[row];
  constexpr int VN = 16 / sizeof(T);
  const int nv = d / VN;
  if (t < 0) {   // padding row: zero gradient row, zero gate gradient
    uint4* out = reinterpret_cast<uint4*>(dO + (size_t)row * d);
    for (int v = lane; v < nv; v += 32) out[v] = make_uint4(0, 0, 0, 0);
    if (lane == 0) dgate[row] = 0.f;
    return;
  }
  const uint4* dy = reinterpret_cast<const uint4*>(dY + (size_t)t * d);
  const uint4* o = reinterpret_cast<const uint4*>(O + (size_t)row * d);
  uint4* out = reinterpret_cast<uint4*>(dO + (size_t)row * d);
  float dot = 0.f;
  for (int v = lane; v < nv; v += 32) {
    float a[VN], b[VN], c[VN];
    unpack16(__ldg(dy + v), a, T());
    unpack16(__ldg(o + v), b, T());
#pragma unroll
    for (int j = 0; j < VN; ++j) {
      dot = fmaf(a[j], b[j], dot);
      c[j] = g * a[j];
    }
    out[v] = pack16(c, T());
  }
  dot = warp_sum(dot);
  if (lane == 0) dgate[row] = dot;
}

template <typename T>
cudaError_t launch_bwd_gather_scale(const T* dY, const T* O, const int* idx, const float* gate,
                                    T* dO, float* dgate, int64_t P, int d, cudaStream_t st) {
  if (P == 0) return cudaSuccess;
  const int warps = 8;
  bwd_gather_scale_kernel<T><<<(unsigned)((P + warps - 1) / warps), warps * 32, 0, st>>>(
      dY, O, idx, gate, dO, dgate, P, d);
  return cudaGetLastError();
}

// ------------------------------------------------------------------ softmax Jacobian
// dS[t,e] = dgate of the pair (t chosen by e) else 0; dZ = S * (dS - <dS, S>).
// Optionally also writes dZ as two bf16 planes [2][N][Ep], hi = bf16(dZ) and
// lo = bf16(dZ - hi), zero in the padding columns E..Ep-1: the tensor-core operands of the
// router-gradient GEMMs, which sum the products of both planes (hi + lo carries dZ to
// about 16 significant bits, so the GEMMs keep near-fp32 accuracy).
// One warp per token; lane l holds experts l, l+32, ... (E <= 512) in registers.
__global__ void softmax_bwd_kernel(const float* __restrict__ S, const int* __restrict__ slot,
                                   const float* __restrict__ dgate, float* __restrict__ dZ,
                                   bf16* __restrict__ dZb, int N, int E, int Ep, int M) {
  constexpr int MAXC = 16;
  const int t = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (t >= N) return;
  float ds[MAXC], sv[MAXC];
  float dot = 0.f;
#pragma unroll
  for (int i = 0; i < MAXC; ++i) {
    const int e = lane + 32 * i;
    ds[i] = 0.f;
    sv[i] = 0.f;
    if (e < E) {
      const int m = slot[(size_t)t * E + e];
      ds[i] = m >= 0 ? dgate[(size_t)e * M + m] : 0.f;
      sv[i] = S[(size_t)t * E + e];
      dot = fmaf(ds[i], sv[i], dot);
    }
  }
  dot = warp_sum(dot);
#pragma unroll
  for (int i = 0; i < MAXC; ++i) {
    const int e = lane + 32 * i;
    if (e < E) {
      const float z = sv[i] * (ds[i] - dot);
      dZ[(size_t)t * E + e] = z;
      if (dZb) {
        const bf16 hi = __float2bfloat16_rn(z);
        dZb[(size_t)t * Ep + e] = hi;
        dZb[(size_t)N * Ep + (size_t)t * Ep + e] = __float2bfloat16_rn(z - __bfloat162float(hi));
      }
    }
  }
  if (dZb)
    for (int e = E + lane; e < Ep; e += 32) {
      dZb[(size_t)t * Ep + e] = __float2bfloat16_rn(0.f);
      dZb[(size_t)N * Ep + (size_t)t * Ep + e] = __float2bfloat16_rn(0.f);
    }
}

cudaError_t launch_softmax_bwd(const float* S, const int* slot, const float* dgate, float* dZ,
                               bf16* dZb, int N, int E, int Ep, int M, cudaStream_t st) {
  if (N == 0) return cudaSuccess;
  if (E > 512) return cudaErrorInvalidValue;
  softmax_bwd_kernel<<<(N + 7) / 8, 256, 0, st>>>(S, slot, dgate, dZ, dZb, N, E, Ep, M);
  return cudaGetLastError();
}

// Fused form. A group of LPT lanes owns a token (LPT = 16 up to 64 experts, 32 up to 128),
// each lane one 4-expert vector (16-byte loads of slot and S); a warp takes 32/LPT tokens at a
// time and kRbIter of them back to back, all loads issued first. The gate gradients of the
// selected pairs are gathered cooperatively: the warp lists its selected pairs in shared
// memory (ballot order), each lane sums the partials of list entries lane, lane+32, ... (two
// at a time, partials in order, as reduce_splits_kernel does), and every lane reads its own
// sums back. The column sums of dZ for the bias gradient are taken per CTA in a fixed order.
constexpr int kRbWarps = 8, kRbIter = 4;

template <int LPT, bool WDZ, bool BIAS>
__global__ void __launch_bounds__(kRbWarps * 32, 4)
router_softmax_bwd_kernel(const float* __restrict__ S, const int* __restrict__ slot,
                          const float* __restrict__ dg_part, int parts, int64_t P,
                          float* __restrict__ dZ, bf16* __restrict__ dZb,
                          float* __restrict__ bpart, int N, int E, int Ep, int M) {
  constexpr int TPW = 32 / LPT;                   // tokens per warp per step
  constexpr int TPB = kRbWarps * TPW * kRbIter;   // tokens per CTA
  constexpr int NC = kRbIter * 4;                 // (token, expert) candidates per lane
  __shared__ int s_list[kRbWarps][32 * NC];
  __shared__ float s_col[BIAS ? kRbWarps * TPW : 1][BIAS ? 4 * LPT : 1];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int sub = lane / LPT, v = lane % LPT;     // token of the warp, expert vector
  const bool vok = v < (E >> 2);
  const int t0 = blockIdx.x * TPB + (warp * TPW + sub) * kRbIter;
  int4 sl[kRbIter];
  float4 sv[kRbIter];
#pragma unroll
  for (int it = 0; it < kRbIter; ++it) {
    const int t = t0 + it;
    sl[it] = make_int4(-1, -1, -1, -1);
    sv[it] = make_float4(0.f, 0.f, 0.f, 0.f);
    if (t < N && vok) {
      sl[it] = reinterpret_cast<const int4*>(slot + (size_t)t * E)[v];
      sv[it] = reinterpret_cast<const float4*>(S + (size_t)t * E)[v];
    }
  }
  // list of the warp's selected pairs (offset of the pair in a partial plane)
  int* list = s_list[warp];
  int pos[NC];
  int cnt = 0;
  const unsigned below = (1u << lane) - 1u;
#pragma unroll
  for (int it = 0; it < kRbIter; ++it) {
    const int m[4] = {sl[it].x, sl[it].y, sl[it].z, sl[it].w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const bool sel = m[j] >= 0;
      const unsigned b = __ballot_sync(0xffffffffu, sel);
      const int p = cnt + __popc(b & below);
      pos[it * 4 + j] = sel ? p : -1;
      if (sel) list[p] = (4 * v + j) * M + m[j];
      cnt += __popc(b);
    }
  }
  __syncwarp();
  for (int i = lane; i < cnt; i += 64) {
    const int i2 = i + 32;
    const int o1 = list[i];
    const int o2 = i2 < cnt ? list[i2] : o1;
    float s1 = 0.f, s2 = 0.f;
    for (int k0 = 0; k0 < parts; k0 += 8) {
      float x1[8], x2[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const bool ok = k0 + j < parts;
        x1[j] = ok ? dg_part[(size_t)(k0 + j) * P + o1] : 0.f;
        x2[j] = ok ? dg_part[(size_t)(k0 + j) * P + o2] : 0.f;
      }
#pragma unroll
      for (int j = 0; j < 8; ++j)
        if (k0 + j < parts) { s1 += x1[j]; s2 += x2[j]; }
    }
    reinterpret_cast<float*>(list)[i] = s1;
    if (i2 < cnt) reinterpret_cast<float*>(list)[i2] = s2;
  }
  __syncwarp();
  float csum[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int it = 0; it < kRbIter; ++it) {
    float ds[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int p = pos[it * 4 + j];
      ds[j] = p >= 0 ? reinterpret_cast<const float*>(list)[p] : 0.f;
    }
    float dot = 0.f;
    dot = fmaf(ds[0], sv[it].x, dot);
    dot = fmaf(ds[1], sv[it].y, dot);
    dot = fmaf(ds[2], sv[it].z, dot);
    dot = fmaf(ds[3], sv[it].w, dot);
#pragma unroll
    for (int o = LPT / 2; o > 0; o >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, o);
    const int t = t0 + it;
    if (t >= N || !vok) continue;
    const float z[4] = {sv[it].x * (ds[0] - dot), sv[it].y * (ds[1] - dot),
                        sv[it].z * (ds[2] - dot), sv[it].w * (ds[3] - dot)};
    if (WDZ) reinterpret_cast<float4*>(dZ + (size_t)t * E)[v] = make_float4(z[0], z[1], z[2], z[3]);
    if (dZb) {
      uint32_t h[2], l[2];
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        const __nv_bfloat162 hh = __floats2bfloat162_rn(z[2 * j], z[2 * j + 1]);
        const float2 hf = __bfloat1622float2(hh);
        const __nv_bfloat162 ll = __floats2bfloat162_rn(z[2 * j] - hf.x, z[2 * j + 1] - hf.y);
        h[j] = *reinterpret_cast<const uint32_t*>(&hh);
        l[j] = *reinterpret_cast<const uint32_t*>(&ll);
      }
      reinterpret_cast<uint2*>(dZb + (size_t)t * Ep)[v] = make_uint2(h[0], h[1]);
      reinterpret_cast<uint2*>(dZb + (size_t)N * Ep + (size_t)t * Ep)[v] = make_uint2(l[0], l[1]);
    }
    if (BIAS)
#pragma unroll
      for (int j = 0; j < 4; ++j) csum[j] += z[j];
  }
  if (dZb && Ep > E)   // zero padding columns E..Ep-1 of both planes
    for (int it = 0; it < kRbIter; ++it) {
      const int t = t0 + it;
      if (t >= N) break;
      for (int c = E + 4 * v; c < Ep; c += 4 * LPT) {
        *reinterpret_cast<uint2*>(dZb + (size_t)t * Ep + c) = make_uint2(0u, 0u);
        *reinterpret_cast<uint2*>(dZb + (size_t)N * Ep + (size_t)t * Ep + c) = make_uint2(0u, 0u);
      }
    }
  if (BIAS) {
    // CTA column sums, rows in order; partials stored column-major [E][gridDim.x]
    const int row = warp * TPW + sub;
#pragma unroll
    for (int j = 0; j < 4; ++j) s_col[row][4 * v + j] = csum[j];
    __syncthreads();
    for (int c = threadIdx.x; c < E; c += blockDim.x) {
      float s = 0.f;
      for (int r = 0; r < kRbWarps * TPW; ++r) s += s_col[r][c];
      bpart[(size_t)c * gridDim.x + blockIdx.x] = s;
    }
  }
}

// out[c] = sum over b of part[c][b] (nblk partials per column): one warp per column, lanes
// over strided partials, then a fixed butterfly.
__global__ void colsum_rows_kernel(const float* __restrict__ part, int nblk, int E,
                                   float* __restrict__ out) {
  const int c = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (c >= E) return;
  float s = 0.f;
  for (int b = lane; b < nblk; b += 32) s += part[(size_t)c * nblk + b];
  s = warp_sum(s);
  if (lane == 0) out[c] = s;
}

bool router_bwd_fused(int E, int64_t P) {
  return E > 0 && E % 4 == 0 && E <= 128 && P <= INT32_MAX;   // pair offsets kept as int
}

static int router_bwd_tpb(int E) { return kRbWarps * (E <= 64 ? 2 : 1) * kRbIter; }

int64_t router_bwd_scratch_floats(int N, int E) {
  return (int64_t)E * ((N + router_bwd_tpb(E) - 1) / router_bwd_tpb(E));
}

template <int LPT, bool WDZ, bool BIAS>
static void router_bwd_go(int nblk, const float* S, const int* slot, const float* dg_part,
                          int parts, int64_t P, float* dZ, bf16* dZb, float* bpart, int N, int E,
                          int Ep, int M, cudaStream_t st) {
  router_softmax_bwd_kernel<LPT, WDZ, BIAS><<<nblk, kRbWarps * 32, 0, st>>>(
      S, slot, dg_part, parts, P, dZ, dZb, bpart, N, E, Ep, M);
}

template <int LPT>
static void router_bwd_pick(int nblk, const float* S, const int* slot, const float* dg_part,
                            int parts, int64_t P, float* dZ, bf16* dZb, float* bpart, int N,
                            int E, int Ep, int M, cudaStream_t st) {
  if (dZ) {
    if (bpart) router_bwd_go<LPT, true, true>(nblk, S, slot, dg_part, parts, P, dZ, dZb, bpart, N, E, Ep, M, st);
    else router_bwd_go<LPT, true, false>(nblk, S, slot, dg_part, parts, P, dZ, dZb, bpart, N, E, Ep, M, st);
  } else {
    if (bpart) router_bwd_go<LPT, false, true>(nblk, S, slot, dg_part, parts, P, dZ, dZb, bpart, N, E, Ep, M, st);
    else router_bwd_go<LPT, false, false>(nblk, S, slot, dg_part, parts, P, dZ, dZb, bpart, N, E, Ep, M, st);
  }
}

cudaError_t launch_router_softmax_bwd(const float* S, const int* slot, const float* dg_part,
                                      int parts, float* dZ, bf16* dZb, float* dbr,
                                      float* scratch, int N, int E, int Ep, int M,
                                      cudaStream_t st) {
  const int64_t P = (int64_t)E * M;
  if (!router_bwd_fused(E, P) || parts < 1 || (dZb && (Ep < E || Ep % 4)))
    return cudaErrorInvalidValue;
  if (N == 0) return dbr ? cudaMemsetAsync(dbr, 0, (size_t)E * sizeof(float), st) : cudaSuccess;
  const int nblk = (N + router_bwd_tpb(E) - 1) / router_bwd_tpb(E);
  float* bpart = dbr ? scratch : nullptr;
  if (E <= 64) router_bwd_pick<16>(nblk, S, slot, dg_part, parts, P, dZ, dZb, bpart, N, E, Ep, M, st);
  else router_bwd_pick<32>(nblk, S, slot, dg_part, parts, P, dZ, dZb, bpart, N, E, Ep, M, st);
  if (dbr) colsum_rows_kernel<<<(E + 7) / 8, 256, 0, st>>>(bpart, nblk, E, dbr);
  return cudaGetLastError();
}

// out[i][e] = sum_s part[s][i][e] for the first `cols` of `ld` columns.
// Each output is the sum of its `splits` partials in split order; the partials of a batch of
// sixteen splits are loaded before any of them is added, so sixteen loads are in flight per
// thread (the outputs are few: 2048 x 64 for the router's dWr, 128 CTAs of 256 threads). V = 4:
// four adjacent columns per thread with 16-byte loads (cols and ld multiples of 4).
template <int V>
__global__ void reduce_partials_kernel(const float* __restrict__ part, float* __restrict__ out,
                                       int rows, int cols, int ld, int splits) {
  typedef typename std::conditional<V == 4, float4, float>::type vec;
  const int cv = cols / V;
  const int64_t n = (int64_t)rows * cv;
  const int64_t plane = (int64_t)rows * ld;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = i / cv, c = (i % cv) * V;
    const float* src = part + r * ld + c;
    float s[V];
#pragma unroll
    for (int j = 0; j < V; ++j) s[j] = 0.f;
    int k = 0;
    for (; k + 16 <= splits; k += 16) {
      vec x[16];
#pragma unroll
      for (int u = 0; u < 16; ++u) x[u] = *reinterpret_cast<const vec*>(src + (k + u) * plane);
#pragma unroll
      for (int u = 0; u < 16; ++u) {
        const float* xf = reinterpret_cast<const float*>(&x[u]);
#pragma unroll
        for (int j = 0; j < V; ++j) s[j] += xf[j];
      }
    }
    for (; k < splits; ++k) {
      const vec x = *reinterpret_cast<const vec*>(src + k * plane);
      const float* xf = reinterpret_cast<const float*>(&x);
#pragma unroll
      for (int j = 0; j < V; ++j) s[j] += xf[j];
    }
    float* dst = out + r * cols + c;
    if constexpr (V == 4) *reinterpret_cast<float4*>(dst) = make_float4(s[0], s[1], s[2], s[3]);
    else dst[0] = s[0];
  }
}

cudaError_t launch_reduce_partials(const float* part, float* out, int rows, int cols, int ld,
                                   int splits, cudaStream_t st) {
  if (rows == 0 || cols == 0) return cudaSuccess;
  const bool v4 = cols % 4 == 0 && ld % 4 == 0 &&
                  (reinterpret_cast<uintptr_t>(part) & 15u) == 0 &&
                  (reinterpret_cast<uintptr_t>(out) & 15u) == 0;
  const int64_t n = (int64_t)rows * cols / (v4 ? 4 : 1);
  if (v4)
    reduce_partials_kernel<4><<<grid_for(n, 152 * 16), 256, 0, st>>>(part, out, rows, cols, ld,
                                                                       splits);
  else
    reduce_partials_kernel<1><<<grid_for(n, 152 * 16), 256, 0, st>>>(part, out, rows, cols, ld,
                                                                       splits);
  return cudaGetLastError();
}

// ------------------------------------------------------------------ dX_t = dXr_t + sum dH rows
template <typename T>
__global__ void dx_combine_kernel(const T* __restrict__ dH, const int* __restrict__ slot,
                                  const T* __restrict__ dXr, const T* __restrict__ R,
                                  const T* __restrict__ R2, T* __restrict__ dX, int N, int E,
                                  int M, int d) {
  extern __shared__ int sh[];
  int* s_e = sh;
  int* s_m = sh + E;
  __shared__ int s_cnt;
  const int t = blockIdx.x;
  const int cnt = token_pairs(slot, nullptr, t, E, M, s_e, s_m, nullptr, &s_cnt);
  constexpr int VN = 16 / sizeof(T);
  const int nv = d / VN;
  // as the combine: two 16-byte column groups per thread, up to four dH rows per batch with
  // all their loads issued first; rows added in ascending expert order
  const uint4* hb = reinterpret_cast<const uint4*>(dH);
  const int64_t rs = d / VN;
  for (int v0 = threadIdx.x; v0 < nv; v0 += 2 * blockDim.x) {
    const int v1 = v0 + blockDim.x;
    const bool two = v1 < nv;
    float acc0[VN], acc1[VN];
    auto init = [&](int v, float* acc) {
      if (dXr) {
        unpack16(__ldg(reinterpret_cast<const uint4*>(dXr + (size_t)t * d) + v), acc, T());
      } else {
#pragma unroll
        for (int j = 0; j < VN; ++j) acc[j] = 0.f;
      }
      float r[VN];
      if (R) {
        unpack16(__ldg(reinterpret_cast<const uint4*>(R + (size_t)t * d) + v), r, T());
#pragma unroll
        for (int j = 0; j < VN; ++j) acc[j] += r[j];
      }
      if (R2) {
        unpack16(__ldg(reinterpret_cast<const uint4*>(R2 + (size_t)t * d) + v), r, T());
#pragma unroll
        for (int j = 0; j < VN; ++j) acc[j] += r[j];
      }
    };
    init(v0, acc0);
    if (two) init(v1, acc1);
    for (int p = 0; p < cnt; p += 4) {
      const int nb = cnt - p < 4 ? cnt - p : 4;
      uint4 u0[4], u1[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        u0[q] = u1[q] = make_uint4(0, 0, 0, 0);
        if (q < nb) {
          const int64_t row = (int64_t)s_e[p + q] * M + s_m[p + q];
          u0[q] = __ldg(hb + row * rs + v0);
          if (two) u1[q] = __ldg(hb + row * rs + v1);
        }
      }
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        if (q < nb) {
          float h[VN];
          unpack16(u0[q], h, T());
#pragma unroll
          for (int j = 0; j < VN; ++j) acc0[j] += h[j];
          unpack16(u1[q], h, T());
#pragma unroll
          for (int j = 0; j < VN; ++j) acc1[j] += h[j];
        }
      }
    }
    reinterpret_cast<uint4*>(dX + (size_t)t * d)[v0] = pack16(acc0, T());
    if (two) reinterpret_cast<uint4*>(dX + (size_t)t * d)[v1] = pack16(acc1, T());
  }
}

template <typename T>
cudaError_t launch_dx_combine(const T* dH, const int* slot, const T* dXr, const T* R,
                              const T* R2, T* dX, int N, int E, int M, int d, cudaStream_t st) {
  if (N == 0) return cudaSuccess;
  const size_t smem = (size_t)2 * E * sizeof(int);
  const int nv = d * (int)sizeof(T) / 16;
  const int threads = std::min(128, std::max(32, (nv / 2 + 31) / 32 * 32));
  dx_combine_kernel<T><<<N, threads, smem, st>>>(dH, slot, dXr, R, R2, dX, N, E, M, d);
  return cudaGetLastError();
}

// ------------------------------------------------------------------ column sums of Z [N][E]
// Two passes, deterministic: partial sums over blocks of kColRows rows (32 columns per
// block, 8 warps over the rows), then the partials summed in block order.
constexpr int kColRows = 512;

__global__ void colsum_part_kernel(const float* __restrict__ Z, float* __restrict__ part, int N,
                                   int E) {
  __shared__ float sh[8][33];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int e = blockIdx.x * 32 + lane;
  const int r0 = blockIdx.y * kColRows;
  const int r1 = min(N, r0 + kColRows);
  float s = 0.f;
  if (e < E)
#pragma unroll 8
    for (int t = r0 + warp; t < r1; t += 8) s += Z[(size_t)t * E + e];
  sh[warp][lane] = s;
  __syncthreads();
  if (warp == 0 && e < E) {
    float r = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) r += sh[w][lane];
    part[(size_t)blockIdx.y * E + e] = r;
  }
}

__global__ void colsum_final_kernel(const float* __restrict__ part, int nrb, int E,
                                    float* __restrict__ out) {
  const int e = blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= E) return;
  float s = 0.f;
  for (int b = 0; b < nrb; ++b) s += part[(size_t)b * E + e];
  out[e] = s;
}

int64_t colsum_scratch_floats(int N, int E) {
  return (int64_t)((N + kColRows - 1) / kColRows) * E;
}

cudaError_t launch_colsum(const float* Z, float* out, int N, int E, float* scratch,
                          cudaStream_t st) {
  const int nrb = (N + kColRows - 1) / kColRows;
  if (nrb == 0) return cudaMemsetAsync(out, 0, (size_t)E * sizeof(float), st);
  colsum_part_kernel<<<dim3((E + 31) / 32, nrb), 256, 0, st>>>(Z, scratch, N, E);
  colsum_final_kernel<<<(E + 127) / 128, 128, 0, st>>>(scratch, nrb, E, out);
  return cudaGetLastError();
}

// ------------------------------------------------------------------ SwiGLU elementwise (SIMT path)
template <typename T>
__global__ void swiglu_fwd_ew_kernel(const float* __restrict__ Ag, const float* __restrict__ Bu,
                                     T* __restrict__ A, T* __restrict__ B, T* __restrict__ U,
                                     int64_t n) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    const float a = Ag[i], b = Bu[i];
    A[i] = from_f32<T>(a);
    B[i] = from_f32<T>(b);
    U[i] = from_f32<T>(a * sigmoidf_(a) * b);
  }
}

template <typename T>
cudaError_t launch_swiglu_fwd_ew(const float* Ag, const float* Bu, T* A, T* B, T* U, int64_t n,
                                 cudaStream_t st) {
  if (n == 0) return cudaSuccess;
  const unsigned blocks = grid_for(n, 152 * 64);
  swiglu_fwd_ew_kernel<T><<<blocks, 256, 0, st>>>(Ag, Bu, A, B, U, n);
  return cudaGetLastError();
}

template <typename T>
__global__ void swiglu_bwd_ew_kernel(const float* __restrict__ dU, const T* __restrict__ A,
                                     const T* __restrict__ B, T* __restrict__ dA,
                                     T* __restrict__ dB, int64_t n) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    const float a = to_f32(A[i]), b = to_f32(B[i]), du = dU[i];
    const float s = sigmoidf_(a);
    dA[i] = from_f32<T>(du * b * s * (1.0f + a * (1.0f - s)));
    dB[i] = from_f32<T>(du * a * s);
  }
}

template <typename T>
cudaError_t launch_swiglu_bwd_ew(const float* dU, const T* A, const T* B, T* dA, T* dB,
                                 int64_t n, cudaStream_t st) {
  if (n == 0) return cudaSuccess;
  const unsigned blocks = grid_for(n, 152 * 64);
  swiglu_bwd_ew_kernel<T><<<blocks, 256, 0, st>>>(dU, A, B, dA, dB, n);
  return cudaGetLastError();
}

template <typename T>
__global__ void convert_kernel(const float* __restrict__ in, T* __restrict__ out, int64_t n) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x)
    out[i] = from_f32<T>(in[i]);
}

template <typename T>
cudaError_t launch_convert(const float* in, T* out, int64_t n, cudaStream_t st) {
  if (n == 0) return cudaSuccess;
  const unsigned blocks = grid_for(n, 152 * 64);
  convert_kernel<T><<<blocks, 256, 0, st>>>(in, out, n);
  return cudaGetLastError();
}

__global__ void reduce_splits_kernel(const float* __restrict__ part, float* __restrict__ out,
                                     int64_t n, int splits) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    // split order, eight loads in flight before they are added
    float s = 0.f;
    int k = 0;
    for (; k + 8 <= splits; k += 8) {
      float x[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) x[u] = part[(size_t)(k + u) * n + i];
#pragma unroll
      for (int u = 0; u < 8; ++u) s += x[u];
    }
    for (; k < splits; ++k) s += part[(size_t)k * n + i];
    out[i] = s;
  }
}

cudaError_t launch_reduce_splits(const float* part, float* out, int64_t n, int splits,
                                 cudaStream_t st) {
  if (n == 0) return cudaSuccess;
  const unsigned blocks = grid_for(n, 152 * 16);
  reduce_splits_kernel<<<blocks, 256, 0, st>>>(part, out, n, splits);
  return cudaGetLastError();
}

#define ECMOE_INST(T)                                                                            \
  template cudaError_t launch_scatter_rows<T>(const T*, const int*, T*, int, int, int, int,       \
                                              cudaStream_t);                                      \
  template cudaError_t launch_zero_pad_rows<T>(const int*, const int*, T*, int, int, cudaStream_t); \
  template cudaError_t launch_combine<T>(const T*, const float*, const int*, const T*, const T*,  \
                                         T*, int, int, int, int, cudaStream_t);                   \
  template cudaError_t launch_bwd_gather_scale<T>(const T*, const T*, const int*, const float*,   \
                                                  T*, float*, int64_t, int, cudaStream_t);        \
  template cudaError_t launch_dx_combine<T>(const T*, const int*, const T*, const T*,             \
                                            const T*, T*, int, int, int, int, cudaStream_t);      \
  template cudaError_t launch_swiglu_fwd_ew<T>(const float*, const float*, T*, T*, T*, int64_t,   \
                                               cudaStream_t);                                     \
  template cudaError_t launch_swiglu_bwd_ew<T>(const float*, const T*, const T*, T*, T*,          \
                                               int64_t, cudaStream_t);                            \
  template cudaError_t launch_convert<T>(const float*, T*, int64_t, cudaStream_t);
ECMOE_INST(float)
ECMOE_INST(bf16)

}  // namespace ecmoe
