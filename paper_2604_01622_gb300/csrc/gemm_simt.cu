// Batched fp32 CUDA-core GEMM with arbitrary operand strides.
//
// Serves the fp32 path of the layer (where tensor-core TF32 would miss a 1e-4 relative
// error bound) and the small router-gradient products dZ.Wr^T and X^T.dZ. Tiles of
// 64x64 outputs, 16-deep K slices staged in shared memory, 4x4 outputs per thread; each
// operand tile is loaded along whichever of its two dimensions is contiguous.
#include "common.cuh"
#include "kernels.h"

namespace ecmoe {

namespace {
constexpr int BM = 64, BN = 64, BK = 16;

template <typename T>
__device__ __forceinline__ float ld(const void* p, int64_t i) {
  return to_f32(reinterpret_cast<const T*>(p)[i]);
}

template <typename TA, typename TB>
__global__ void __launch_bounds__(256) simt_gemm_kernel(SimtGemmArgs p) {
  __shared__ float As[BK][BM + 4];
  __shared__ float Bs[BK][BN + 4];
  const int tid = threadIdx.x;
  const int bz = blockIdx.z;
  const int b = bz / p.splits, s = bz % p.splits;
  const int m0 = blockIdx.y * BM, n0 = blockIdx.x * BN;
  const int kchunk = (p.K + p.splits - 1) / p.splits;
  const int kb = s * kchunk, ke = min(p.K, kb + kchunk);
  const int64_t a_off = (int64_t)b * p.a_bs, b_off = (int64_t)b * p.b_bs;
  const bool a_kfast = p.a_ks == 1, b_nfast = p.b_ns == 1;
  const int ty = tid >> 4, tx = tid & 15;
  float acc[4][4] = {};
  for (int k0 = kb; k0 < ke; k0 += BK) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int l = tid + i * 256;
      int mm, kk;
      if (a_kfast) { kk = l % BK; mm = l / BK; } else { mm = l % BM; kk = l / BM; }
      const int gm = m0 + mm, gk = k0 + kk;
      As[kk][mm] = (gm < p.M && gk < ke) ? ld<TA>(p.A, a_off + gm * p.a_ms + gk * p.a_ks) : 0.f;
      int nn, kk2;
      if (b_nfast) { nn = l % BN; kk2 = l / BN; } else { kk2 = l % BK; nn = l / BK; }
      const int gn = n0 + nn, gk2 = k0 + kk2;
      Bs[kk2][nn] = (gn < p.N && gk2 < ke) ? ld<TB>(p.B, b_off + gk2 * p.b_ks + gn * p.b_ns) : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < BK; ++kk) {
      float av[4], bv[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) av[i] = As[kk][ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) bv[j] = Bs[kk][tx * 4 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
    }
    __syncthreads();
  }
  float* C = p.C + (int64_t)b * p.c_bs + (p.splits > 1 ? (int64_t)s * p.c_split : 0);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int gm = m0 + ty * 4 + i;
    if (gm >= p.M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int gn = n0 + tx * 4 + j;
      if (gn >= p.N) continue;
      float v = acc[i][j];
      float* c = C + (int64_t)gm * p.c_ms + gn;
      if (p.splits == 1 && p.beta != 0.f) v += p.beta * *c;
      *c = v;
    }
  }
}
}  // namespace

cudaError_t launch_simt_gemm(const SimtGemmArgs& a, EType ta, EType tb, cudaStream_t st) {
  if (a.M == 0 || a.N == 0 || a.batch == 0) return cudaSuccess;
  dim3 grid((a.N + BN - 1) / BN, (a.M + BM - 1) / BM, a.batch * a.splits);
  if (ta == EType::F32 && tb == EType::F32)
    simt_gemm_kernel<float, float><<<grid, 256, 0, st>>>(a);
  else if (ta == EType::BF16 && tb == EType::BF16)
    simt_gemm_kernel<bf16, bf16><<<grid, 256, 0, st>>>(a);
  else if (ta == EType::F32 && tb == EType::BF16)
    simt_gemm_kernel<float, bf16><<<grid, 256, 0, st>>>(a);
  else
    simt_gemm_kernel<bf16, float><<<grid, 256, 0, st>>>(a);
  return cudaGetLastError();
}

}  // namespace ecmoe
