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

// Order-preserving unsigned key of a score (larger score, larger key; -0 == +0; NaN ranks
// with -inf). Key 0 is below every score: it marks an expert already taken.
__device__ __forceinline__ uint32_t score_key(float v) {
  v = v + 0.0f;
  if (v != v) v = -INFINITY;
  const uint32_t u = __float_as_uint(v);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// One warp per token, lane l holding experts l, l+32, ... (E <= 256) in registers: k rounds
// of a warp argmax (largest key by a max-reduction, then the lowest expert index holding
// it by a min-reduction). Writes the choices best first, the normalised gates and their
// sum Z (summed in choice order).
__global__ void tc_topk_rows_kernel(const float* __restrict__ S, int N, int E, int k,
                                    int* __restrict__ choice, float* __restrict__ tgate,
                                    float* __restrict__ Z) {
  constexpr int MAXC = 8;
  const int t = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (t >= N) return;
  const float* row = S + (size_t)t * E;
  float val[MAXC];
  uint32_t key[MAXC];
#pragma unroll
  for (int i = 0; i < MAXC; ++i) {
    const int e = lane + 32 * i;
    val[i] = e < E ? row[e] : 0.f;
    key[i] = e < E ? score_key(val[i]) : 0u;
  }
  float sum = 0.f, my_v = 0.f;
  int my_e = 0;   // lane r keeps the r-th choice
  for (int r = 0; r < k; ++r) {
    uint32_t best = 0u;
    int bi = 0x7fffffff;
#pragma unroll
    for (int i = 0; i < MAXC; ++i)          // ascending expert index: ties keep the first
      if (key[i] > best) { best = key[i]; bi = lane + 32 * i; }
    const uint32_t m = __reduce_max_sync(0xffffffffu, best);
    const int e = (int)__reduce_min_sync(0xffffffffu, best == m ? (uint32_t)bi : 0x7fffffffu);
    float v = 0.f;
#pragma unroll
    for (int i = 0; i < MAXC; ++i)
      if (lane + 32 * i == e) { v = val[i]; key[i] = 0u; }
    v = __shfl_sync(0xffffffffu, v, e & 31);
    if (lane == r) { my_e = e; my_v = v; }
    sum += v;
  }
  if (lane < k) {
    choice[(size_t)t * k + lane] = my_e;
    tgate[(size_t)t * k + lane] = my_v / sum;
  }
  if (lane == 0) Z[t] = sum;
}

// The same selection for up to 64 experts (E a multiple of 4) and k <= 8, four threads per
// token: thread j of the token holds scores 16 j .. 16 j + 15 and keeps its k best in a sorted
// register list of packed words (order-preserving key above, 255 - expert below, so equal
// scores order by lower expert index); k rounds take the largest head of the four lists. The
// choices, gates (normalised by the sum taken in choice order) and Z match the warp-per-token
// kernel exactly. The token's row of the slot map is set to -1 here as well.
constexpr int kTopkFastE = 64, kTopkFastK = 8;

__global__ void __launch_bounds__(256)
tc_topk_rows4_kernel(const float* __restrict__ S, int N, int E, int k, int* __restrict__ choice,
                     float* __restrict__ tgate, float* __restrict__ Z, int* __restrict__ slot) {
  const int64_t gt = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int t = (int)(gt >> 2), j = threadIdx.x & 3;
  const bool ok = t < N;                  // the token's four threads agree
  const int e0 = j * 16;
  const int ne = ok ? max(0, min(16, E - e0)) : 0;
  const float* row = S + (size_t)(ok ? t : 0) * E + e0;
  float val[16];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
    if (4 * q < ne) x = reinterpret_cast<const float4*>(row)[q];
    val[4 * q] = x.x; val[4 * q + 1] = x.y; val[4 * q + 2] = x.z; val[4 * q + 3] = x.w;
  }
  if (ok) {
    int4* sl = reinterpret_cast<int4*>(slot + (size_t)t * E + e0);
#pragma unroll
    for (int q = 0; q < 4; ++q)
      if (4 * q < ne) sl[q] = make_int4(-1, -1, -1, -1);
  }
  // this thread's best k, descending; 0 is below every packed score
  unsigned long long lst[kTopkFastK];
  float lv[kTopkFastK];
#pragma unroll
  for (int i = 0; i < kTopkFastK; ++i) { lst[i] = 0ull; lv[i] = 0.f; }
#pragma unroll
  for (int q = 0; q < 16; ++q) {
    if (q >= ne) break;
    unsigned long long x = ((unsigned long long)score_key(val[q]) << 32) |
                           (unsigned long long)(255 - (e0 + q));
    float xv = val[q];
#pragma unroll
    for (int i = 0; i < kTopkFastK; ++i) {
      if (x > lst[i]) {
        const unsigned long long tx = lst[i];
        const float tv = lv[i];
        lst[i] = x; lv[i] = xv;
        x = tx; xv = tv;
      }
    }
  }
  int my_e[2] = {0, 0};
  float my_v[2] = {0.f, 0.f};
  float sum = 0.f;
  for (int r = 0; r < k; ++r) {
    unsigned long long m = lst[0];
    m = max(m, __shfl_xor_sync(0xffffffffu, m, 1));
    m = max(m, __shfl_xor_sync(0xffffffffu, m, 2));
    const bool mine = lst[0] == m;                  // exactly one thread of the token
    float v = mine ? lv[0] : 0.f;
    v += __shfl_xor_sync(0xffffffffu, v, 1);
    v += __shfl_xor_sync(0xffffffffu, v, 2);
    if (mine) {
#pragma unroll
      for (int i = 0; i + 1 < kTopkFastK; ++i) { lst[i] = lst[i + 1]; lv[i] = lv[i + 1]; }
      lst[kTopkFastK - 1] = 0ull;
    }
    if ((r & 3) == j) {
      my_e[r >> 2] = 255 - (int)(uint32_t)(m & 0xFFFFFFFFull);
      my_v[r >> 2] = v;
    }
    sum += v;
  }
  if (!ok) return;
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int r = 4 * h + j;
    if (r < k) {
      choice[(size_t)t * k + r] = my_e[h];
      tgate[(size_t)t * k + r] = my_v[h] / sum;
    }
  }
  if (j == 0) Z[t] = sum;
}

// The position of token t in expert e's list is the number of tokens before t that chose
// e: an exclusive scan, in token order, of the 0/1 column "chose e". It is done in three
// levels: warp ballots within each 256-token block, warps within the block, blocks.
constexpr int kRankBlock = 256;   // tokens per ranking block (8 warps)
constexpr int kMaxE = 256;        // experts the ranking handles (8 mask words)

// Per 256-token block: hist[blk][e] = tokens of the block that chose e; for each chosen
// (t, e), slot[t][e] = rank of t among the block's tokens that chose e (made absolute by
// tc_fill_kernel). slot holds -1 elsewhere.
__global__ void __launch_bounds__(kRankBlock)
tc_rank_kernel(const int* __restrict__ choice, int N, int E, int k, int* __restrict__ slot,
               int* __restrict__ hist) {
  __shared__ int s_cnt[kRankBlock / 32][kMaxE];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t = blockIdx.x * kRankBlock + threadIdx.x;
  uint32_t mask[kMaxE / 32];
#pragma unroll
  for (int w = 0; w < kMaxE / 32; ++w) mask[w] = 0u;
  if (t < N)
    for (int r = 0; r < k; ++r) {
      const int e = choice[(size_t)t * k + r];
#pragma unroll
      for (int w = 0; w < kMaxE / 32; ++w)
        if ((e >> 5) == w) mask[w] |= 1u << (e & 31);
    }
  const uint32_t lt = (1u << lane) - 1u;
  // pass 1: per-warp counts
#pragma unroll
  for (int w = 0; w < kMaxE / 32; ++w) {
    const uint32_t m = mask[w];
    const int nb = min(32, E - 32 * w);   // experts in this mask word (<= 0: none)
    for (int b = 0; b < nb; ++b) {
      const uint32_t bal = __ballot_sync(0xffffffffu, (m >> b) & 1u);
      if (lane == 0) s_cnt[warp][32 * w + b] = __popc(bal);
    }
  }
  __syncthreads();
  // warp offsets within the block, block totals
  for (int e = threadIdx.x; e < E; e += kRankBlock) {
    int acc = 0;
#pragma unroll
    for (int w = 0; w < kRankBlock / 32; ++w) {
      const int c = s_cnt[w][e];
      s_cnt[w][e] = acc;
      acc += c;
    }
    hist[(size_t)blockIdx.x * E + e] = acc;
  }
  __syncthreads();
  // pass 2: ranks
#pragma unroll
  for (int w = 0; w < kMaxE / 32; ++w) {
    const uint32_t m = mask[w];
    const int nb = min(32, E - 32 * w);
    for (int b = 0; b < nb; ++b) {
      const bool mine = (m >> b) & 1u;
      const uint32_t bal = __ballot_sync(0xffffffffu, mine);
      if (mine) slot[(size_t)t * E + 32 * w + b] = s_cnt[warp][32 * w + b] + __popc(bal & lt);
    }
  }
}

// One CTA per expert: boff[blk][e] = tokens of earlier blocks that chose e (exclusive scan
// over the blocks), total[e] = all tokens that chose e.
__global__ void tc_block_scan_kernel(const int* __restrict__ hist, int nblk, int E,
                                     int* __restrict__ boff, int* __restrict__ total) {
  __shared__ int s_warp[33];
  const int e = blockIdx.x;
  int carry = 0;
  for (int b0 = 0; b0 < nblk; b0 += blockDim.x) {
    const int b = b0 + threadIdx.x;
    const int h = b < nblk ? hist[(size_t)b * E + e] : 0;
    int chunk;
    const int ex = block_scan_excl(h, s_warp, &chunk);
    if (b < nblk) boff[(size_t)b * E + e] = carry + ex;
    carry += chunk;
  }
  if (threadIdx.x == 0) total[e] = carry;
}

// One CTA (E <= blockDim): kept rows per expert count[e] = min(total, cap) (cap < 0: no cap),
// padded regions tiles[e] (cumulative 256-row blocks, tiles[E] the total) and in count[E]
// the padded rows in use.
__global__ void tc_offsets_kernel(int E, int cap, const int* __restrict__ total,
                                  int* __restrict__ count, int* __restrict__ tiles) {
  __shared__ int s_warp[33];
  const int e = threadIdx.x;
  int c = e < E ? total[e] : 0;
  if (cap >= 0 && c > cap) c = cap;
  const int nb = (c + kPadRows - 1) / kPadRows;
  int all;
  const int off = block_scan_excl(nb, s_warp, &all);
  if (e < E) {
    count[e] = c;
    tiles[e] = off;
  }
  if (threadIdx.x == 0) {
    tiles[E] = all;
    count[E] = all * kPadRows;
  }
}

// One thread per (token, choice) pair: absolute position, keep/drop, row maps; then one
// thread per possible padding row of each expert: row_token -1, gate 0.
__global__ void tc_fill_kernel(const int* __restrict__ choice, const float* __restrict__ tgate,
                               int N, int E, int k, const int* __restrict__ boff,
                               const int* __restrict__ count, const int* __restrict__ tiles,
                               int* __restrict__ row_token, float* __restrict__ row_gate,
                               int* __restrict__ slot, int* __restrict__ kept) {
  const int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t NK = (int64_t)N * k;
  if (j < NK) {
    const int t = (int)(j / k);
    const int e = choice[j];
    int* sl = slot + (size_t)t * E + e;
    const int pos = boff[(size_t)(t / kRankBlock) * E + e] + *sl;
    const bool keep = pos < count[e];
    kept[j] = keep;
    if (keep) {
      const int row = tiles[e] * kPadRows + pos;
      *sl = row;
      row_token[row] = t;
      row_gate[row] = tgate[j];
    } else {
      *sl = -1;
    }
    return;
  }
  const int64_t q = j - NK;
  const int e = (int)(q / kPadRows);
  if (e >= E) return;
  const int row = tiles[e] * kPadRows + count[e] + (int)(q % kPadRows);
  if (row < tiles[e + 1] * kPadRows) {
    row_token[row] = -1;
    row_gate[row] = 0.f;
  }
}

cudaError_t launch_tc_route(const float* S, int N, int E, int k, int cap, int* choice,
                            float* tgate, float* Z, int* count, int* tiles, int* row_token,
                            float* row_gate, int* slot, int* kept, int* scratch,
                            cudaStream_t st) {
  if (N == 0) return cudaSuccess;
  if (E > kMaxE || k > 32 || k > E) return cudaErrorInvalidValue;
  const int nblk = (N + kRankBlock - 1) / kRankBlock;
  int* hist = scratch;                          // [nblk][E]
  int* boff = scratch + (size_t)nblk * E;       // [nblk][E]
  int* total = boff + (size_t)nblk * E;         // [E]
  if (E % 4 == 0 && E <= kTopkFastE && k <= kTopkFastK) {
    // four threads per token; the slot map's -1 rows are written there too
    tc_topk_rows4_kernel<<<(unsigned)(((int64_t)N * 4 + 255) / 256), 256, 0, st>>>(
        S, N, E, k, choice, tgate, Z, slot);
  } else {
    cudaError_t err = cudaMemsetAsync(slot, 0xFF, (size_t)N * E * sizeof(int), st);   // -1
    if (err != cudaSuccess) return err;
    tc_topk_rows_kernel<<<(N + 7) / 8, 256, 0, st>>>(S, N, E, k, choice, tgate, Z);
  }
  tc_rank_kernel<<<nblk, kRankBlock, 0, st>>>(choice, N, E, k, slot, hist);
  tc_block_scan_kernel<<<E, 256, 0, st>>>(hist, nblk, E, boff, total);
  tc_offsets_kernel<<<1, kMaxE, 0, st>>>(E, cap, total, count, tiles);
  const int64_t threads = (int64_t)N * k + (int64_t)E * kPadRows;
  tc_fill_kernel<<<(unsigned)((threads + 255) / 256), 256, 0, st>>>(
      choice, tgate, N, E, k, boff, count, tiles, row_token, row_gate, slot, kept);
  return cudaGetLastError();
}

// Scratch ints launch_tc_route needs for N tokens and E experts.
int64_t tc_route_scratch_ints(int N, int E) {
  const int64_t nblk = (N + kRankBlock - 1) / kRankBlock;
  return 2 * nblk * E + E;
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
