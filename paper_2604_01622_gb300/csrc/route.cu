// Router softmax and expert-choice top-k selection (arXiv 2604.01622, Sec. 2.2).
//
// Selection: for every expert e and group g (one sequence, Sec. 5.2) keep the k_g tokens
// with the largest S[t,e] (Sec. 2.2 TopC; capacity per group, Sec. 4.2). Ties go to the
// lower token index and the kept tokens are written in ascending index. One CTA per
// (e, g) runs an MSB-first radix select over order-preserving 32-bit keys of the fp32
// scores to find the k-th largest key, then compacts the column in index order with one
// block scan, which makes the result unique and independent of thread timing.
#include "common.cuh"
#include "kernels.h"

namespace ecmoe {

// ------------------------------------------------------------------ softmax over experts
// 32 tokens per CTA; the S^T tile is staged in shared memory so both layouts are written
// with coalesced stores. The slot map [N][E] (same layout as S) is set to -1 beside S.
__global__ void softmax_rows_kernel(const float* __restrict__ Z, const float* __restrict__ br,
                                    float* __restrict__ S, float* __restrict__ ST,
                                    int* __restrict__ slot, int N, int E) {
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
      slot[(size_t)t * E + e] = -1;
    }
  }
  __syncthreads();
  for (int e = warp; e < E; e += nw) {
    const int t = t0 + lane;
    if (t < N) ST[(size_t)e * N + t] = tile[lane * (E + 1) + e];
  }
}

cudaError_t launch_softmax_rows(const float* Z, const float* br, float* S, float* ST, int* slot,
                                int N, int E, cudaStream_t st) {
  if (N == 0) return cudaSuccess;
  size_t smem = (size_t)32 * (E + 1) * sizeof(float);
  if (smem > 48 * 1024)
    cudaFuncSetAttribute(softmax_rows_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  softmax_rows_kernel<<<(N + 31) / 32, 256, smem, st>>>(Z, br, S, ST, slot, N, E);
  return cudaGetLastError();
}

// S = (S^T)^T through a 32 x 32 shared tile; the slot map is set to -1 beside S.
__global__ void transpose_scores_kernel(const float* __restrict__ ST, float* __restrict__ S,
                                        int* __restrict__ slot, int N, int E) {
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
    if (e < E && t < N) {
      S[(size_t)t * E + e] = tile[tx][r];
      slot[(size_t)t * E + e] = -1;
    }
  }
}

cudaError_t launch_transpose_scores(const float* ST, float* S, int* slot, int N, int E,
                                    cudaStream_t st) {
  if (N == 0) return cudaSuccess;
  dim3 grid((N + 31) / 32, (E + 31) / 32);
  transpose_scores_kernel<<<grid, 256, 0, st>>>(ST, S, slot, N, E);
  return cudaGetLastError();
}

// ------------------------------------------------------------------ top-k selection
// Order-preserving key: larger float -> larger unsigned key; -0.0 is folded onto +0.0.
__device__ __forceinline__ uint32_t score_key(float s) {
  uint32_t u = __float_as_uint(s);
  if (u == 0x80000000u) u = 0u;
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Exclusive scan of two counts per thread (packed as hi:lo 32-bit halves) across the block.
__device__ __forceinline__ unsigned long long block_excl_scan2(unsigned long long v,
                                                               unsigned long long* s_warp) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  unsigned long long incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned long long u = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += u;
  }
  if (lane == 31) s_warp[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    const unsigned long long w = lane < nw ? s_warp[lane] : 0ull;
    unsigned long long wi = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const unsigned long long u = __shfl_up_sync(0xffffffffu, wi, o);
      if (lane >= o) wi += u;
    }
    if (lane < nw) s_warp[lane] = wi - w;
  }
  __syncthreads();
  const unsigned long long r = incl - v + s_warp[warp];
  __syncthreads();
  return r;
}

// The k-th largest key is found by an MSB-first radix select over the offsets u = key - kmin
// of the column (kmin, kmax its smallest and largest key), 8 bits per pass starting at the top
// bit of kmax - kmin. Scores of one expert over a sequence span a narrow range, so digits of
// the raw key would put most of the column into a few bins of the first pass (and serialise
// its shared-memory atomics); digits of the offset spread it over the whole histogram. The
// select stops early once the bin that holds the k-th key is taken whole. The selected set
// is the one the (score desc, index asc) order defines, whatever the digit boundaries.
//
// The slot map is expected to hold -1 for every (token, expert) on entry (written by the
// kernel that produced S); only the selected entries are written here.
template <bool SMEM>
__global__ void __launch_bounds__(512, 4)
topk_kernel(const float* __restrict__ ST, int N, int E, const int* __restrict__ group_off,
            const int* __restrict__ k_g, const int* __restrict__ k_off, int M,
            int* __restrict__ idx, float* __restrict__ gate, int* __restrict__ slot) {
  extern __shared__ uint4 skeys4[];
  uint32_t* skeys = reinterpret_cast<uint32_t*>(skeys4);
  __shared__ int hist[256];
  __shared__ unsigned long long s_scan[32];
  __shared__ uint32_t s_mn[32], s_mx[32];
  __shared__ uint32_t s_prefix;
  __shared__ int s_remaining, s_done;
  const int e = blockIdx.x, g = blockIdx.y;
  const int tid = threadIdx.x, nthr = blockDim.x, lane = tid & 31, warp = tid >> 5;
  const int nw = nthr >> 5;
  const int lo = group_off[g];
  const int L = group_off[g + 1] - lo;
  const int k = k_g[g];
  const int base = k_off[g];
  const float* col = ST + (size_t)e * N + lo;

  uint32_t mn = 0xFFFFFFFFu, mx = 0u;
  for (int i = tid; i < L; i += nthr) {
    const uint32_t key = score_key(col[i]);
    if (SMEM) skeys[i] = key;
    mn = min(mn, key);
    mx = max(mx, key);
  }
  mn = __reduce_min_sync(0xffffffffu, mn);
  mx = __reduce_max_sync(0xffffffffu, mx);
  if (lane == 0) { s_mn[warp] = mn; s_mx[warp] = mx; }
  __syncthreads();
  if (warp == 0) {
    mn = __reduce_min_sync(0xffffffffu, lane < nw ? s_mn[lane] : 0xFFFFFFFFu);
    mx = __reduce_max_sync(0xffffffffu, lane < nw ? s_mx[lane] : 0u);
    if (lane == 0) { s_mn[0] = mn; s_mx[0] = mx; }
  }
  __syncthreads();
  mn = s_mn[0];
  mx = s_mx[0];
  auto off_at = [&](int i) -> uint32_t { return (SMEM ? skeys[i] : score_key(col[i])) - mn; };

  // threshold T (an offset) and how many keys equal to it are taken (in token order)
  uint32_t T = 0u;
  int need_eq = 0;
  if (k > 0) {
    int hi = mx == mn ? 0 : 32 - __clz(mx - mn);   // every offset lies in [0, 2^hi)
    uint32_t prefix = 0u, mask = hi == 32 ? 0u : ~((1u << hi) - 1u);
    int remaining = k;
    bool done = hi == 0;                           // all keys equal: the first k are taken
    while (!done && hi > 0) {
      const int shift = max(hi - 8, 0);
      const uint32_t dmask = (1u << (hi - shift)) - 1u;
      for (int i = tid; i < 256; i += nthr) hist[i] = 0;
      __syncthreads();
      for (int i = tid; i < L; i += nthr) {
        const uint32_t u = off_at(i);
        if ((u & mask) == prefix) atomicAdd(&hist[(u >> shift) & dmask], 1);
      }
      __syncthreads();
      if (warp == 0) {
        // lane l owns bins 255-8l .. 248-8l (descending); find the bin holding the
        // remaining-th largest offset
        int c[8], local = 0;
#pragma unroll
        for (int j = 0; j < 8; ++j) { c[j] = hist[255 - (lane * 8 + j)]; local += c[j]; }
        int incl = local;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int u = __shfl_up_sync(0xffffffffu, incl, o);
          if (lane >= o) incl += u;
        }
        const int excl = incl - local;
        if (excl < remaining && remaining <= incl) {
          int run = excl;
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            if (run + c[j] >= remaining) {
              const uint32_t bin = 255u - (uint32_t)(lane * 8 + j);
              s_prefix = prefix | (bin << shift);
              s_remaining = remaining - run;
              s_done = run + c[j] == remaining;   // the whole bin is taken
              break;
            }
            run += c[j];
          }
        }
      }
      __syncthreads();
      prefix = s_prefix;
      remaining = s_remaining;
      done = s_done;
      mask |= dmask << shift;
      hi = shift;
      __syncthreads();
    }
    T = prefix;
    // a bin taken whole: every offset >= T is selected
    need_eq = (done && hi > 0) ? 0x7FFFFFFF : remaining;
  }
  const bool any = k > 0;

  // Compaction in token order: thread tid owns a contiguous chunk (a multiple of 4 keys, read
  // 16 bytes at a time from shared memory); one scan gives both the keys above T and the keys
  // equal to T before the chunk.
  const int chunk = ((L + nthr - 1) / nthr + 3) & ~3;
  const int i0 = min(L, tid * chunk), i1 = min(L, i0 + chunk);
  auto load4 = [&](int i, uint32_t (&u)[4]) {
    if (SMEM && i + 4 <= i1) {
      const uint4 q = skeys4[i >> 2];
      u[0] = q.x - mn; u[1] = q.y - mn; u[2] = q.z - mn; u[3] = q.w - mn;
    } else {
#pragma unroll
      for (int j = 0; j < 4; ++j) u[j] = i + j < i1 ? off_at(i + j) : 0u;
    }
  };
  uint32_t n_gt = 0, n_eq = 0;
  if (any)
    for (int i = i0; i < i1; i += 4) {
      uint32_t u[4];
      load4(i, u);
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (i + j < i1) { n_gt += u[j] > T; n_eq += u[j] == T; }
    }
  const unsigned long long before =
      block_excl_scan2(((unsigned long long)n_gt << 32) | n_eq, s_scan);
  int r = (int)(before & 0xFFFFFFFFu);                 // keys equal to T before this one
  int pos = (int)(before >> 32) + min(r, need_eq);     // selected keys before this one
  if (!any) return;
  int* idx_row = idx + (size_t)e * M + base;
  float* gate_row = gate + (size_t)e * M + base;
  for (int i = i0; i < i1; i += 4) {
    uint32_t u[4];
    load4(i, u);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      if (i + j >= i1) break;
      const bool eq = u[j] == T;
      const bool s = u[j] > T || (eq && r < need_eq);
      r += eq;
      if (s) {
        const int t = lo + i + j;
        const uint32_t key = u[j] + mn;
        // the gate is the score the key encodes (-0.0 and +0.0 share a key: read it back)
        const float sv = key == 0x80000000u
                             ? col[i + j]
                             : __uint_as_float((key & 0x80000000u) ? (key & 0x7FFFFFFFu) : ~key);
        idx_row[pos] = t;
        gate_row[pos] = sv;
        slot[(size_t)t * E + e] = base + pos;
        ++pos;
      }
    }
  }
}

// The same selection with the column in registers: thread i owns the KPT consecutive scores
// [i KPT, i KPT + KPT) of the group (groups up to KPT * blockDim.x tokens), so every pass is an
// unrolled loop over registers (no shared-memory copy of the keys), and the two histogram
// buffers alternate between passes, so a pass needs two block barriers: one before the bin
// search and one after it.
template <int KPT, int NT, int MINB>
__global__ void __launch_bounds__(NT, MINB)
topk_reg_kernel(const float* __restrict__ ST, int N, int E, const int* __restrict__ group_off,
                const int* __restrict__ k_g, const int* __restrict__ k_off, int M,
                int* __restrict__ idx, float* __restrict__ gate, int* __restrict__ slot) {
  __shared__ int hist[2][256];
  __shared__ unsigned long long s_scan[32];
  __shared__ uint32_t s_mn[32], s_mx[32];
  __shared__ uint32_t s_prefix[2];
  __shared__ int s_remaining[2], s_done[2];
  const int e = blockIdx.x, g = blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  constexpr int nw = NT / 32;
  const int lo = group_off[g];
  const int L = group_off[g + 1] - lo;
  const int k = k_g[g];
  const int base = k_off[g];
  const float* col = ST + (size_t)e * N + lo;
  const int i0 = tid * KPT;
  const int nv = max(0, min(KPT, L - i0));        // keys this thread owns
  uint32_t key[KPT];
  if (nv == KPT && ((reinterpret_cast<uintptr_t>(col + i0) & 15u) == 0)) {
#pragma unroll
    for (int j = 0; j < KPT; j += 4) {
      const float4 q = *reinterpret_cast<const float4*>(col + i0 + j);
      key[j] = score_key(q.x); key[j + 1] = score_key(q.y);
      key[j + 2] = score_key(q.z); key[j + 3] = score_key(q.w);
    }
  } else {
#pragma unroll
    for (int j = 0; j < KPT; ++j) key[j] = j < nv ? score_key(col[i0 + j]) : 0u;
  }
  uint32_t mn = 0xFFFFFFFFu, mx = 0u;
#pragma unroll
  for (int j = 0; j < KPT; ++j)
    if (j < nv) { mn = min(mn, key[j]); mx = max(mx, key[j]); }
  mn = __reduce_min_sync(0xffffffffu, mn);
  mx = __reduce_max_sync(0xffffffffu, mx);
  if (lane == 0) { s_mn[warp] = mn; s_mx[warp] = mx; }
  for (int i = tid; i < 256; i += NT) hist[0][i] = 0;
  __syncthreads();
  mn = __reduce_min_sync(0xffffffffu, lane < nw ? s_mn[lane] : 0xFFFFFFFFu);
  mx = __reduce_max_sync(0xffffffffu, lane < nw ? s_mx[lane] : 0u);
  // keys become offsets from the column's smallest key (invalid slots are never read)
#pragma unroll
  for (int j = 0; j < KPT; ++j) key[j] -= mn;

  uint32_t T = 0u;
  int need_eq = 0;
  if (k > 0) {
    int hi = mx == mn ? 0 : 32 - __clz(mx - mn);   // every offset lies in [0, 2^hi)
    uint32_t prefix = 0u, mask = hi == 32 ? 0u : ~((1u << hi) - 1u);
    int remaining = k;
    bool done = hi == 0;                           // all keys equal: the first k are taken
    int b = 0;                                     // histogram buffer of this pass
    while (!done && hi > 0) {
      const int shift = max(hi - 8, 0);
      const uint32_t dmask = (1u << (hi - shift)) - 1u;
      // the other buffer was last read before the previous pass's second barrier
      for (int i = tid; i < 256; i += NT) hist[b ^ 1][i] = 0;
#pragma unroll
      for (int j = 0; j < KPT; ++j)
        if (j < nv && (key[j] & mask) == prefix) atomicAdd(&hist[b][(key[j] >> shift) & dmask], 1);
      __syncthreads();
      if (warp == 0) {
        int c[8], local = 0;
#pragma unroll
        for (int j = 0; j < 8; ++j) { c[j] = hist[b][255 - (lane * 8 + j)]; local += c[j]; }
        int incl = local;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int u = __shfl_up_sync(0xffffffffu, incl, o);
          if (lane >= o) incl += u;
        }
        const int excl = incl - local;
        if (excl < remaining && remaining <= incl) {
          int run = excl;
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            if (run + c[j] >= remaining) {
              const uint32_t bin = 255u - (uint32_t)(lane * 8 + j);
              s_prefix[b] = prefix | (bin << shift);
              s_remaining[b] = remaining - run;
              s_done[b] = run + c[j] == remaining;   // the whole bin is taken
              break;
            }
            run += c[j];
          }
        }
      }
      __syncthreads();
      prefix = s_prefix[b];
      remaining = s_remaining[b];
      done = s_done[b];
      mask |= dmask << shift;
      hi = shift;
      b ^= 1;
    }
    T = prefix;
    need_eq = (done && hi > 0) ? 0x7FFFFFFF : remaining;
  }
  // compaction in token order: this thread's keys follow those of lower threads
  uint32_t n_gt = 0, n_eq = 0;
  if (k > 0)
#pragma unroll
    for (int j = 0; j < KPT; ++j)
      if (j < nv) { n_gt += key[j] > T; n_eq += key[j] == T; }
  const unsigned long long before =
      block_excl_scan2(((unsigned long long)n_gt << 32) | n_eq, s_scan);
  if (k == 0) return;
  int r = (int)(before & 0xFFFFFFFFu);                 // keys equal to T before this one
  int pos = (int)(before >> 32) + min(r, need_eq);     // selected keys before this one
  int* idx_row = idx + (size_t)e * M + base;
  float* gate_row = gate + (size_t)e * M + base;
#pragma unroll
  for (int j = 0; j < KPT; ++j) {
    if (j >= nv) break;
    const bool eq = key[j] == T;
    const bool sel = key[j] > T || (eq && r < need_eq);
    r += eq;
    if (sel) {
      const int t = lo + i0 + j;
      const uint32_t kk = key[j] + mn;
      // the gate is the score the key encodes (-0.0 and +0.0 share a key: read it back)
      const float sv = kk == 0x80000000u
                           ? col[i0 + j]
                           : __uint_as_float((kk & 0x80000000u) ? (kk & 0x7FFFFFFFu) : ~kk);
      idx_row[pos] = t;
      gate_row[pos] = sv;
      slot[(size_t)t * E + e] = base + pos;
      ++pos;
    }
  }
}

cudaError_t launch_topk(const float* ST, int N, int E, int G, const int* group_off, const int* k_g,
                        const int* k_off, int M, int max_group, int* idx, float* gate, int* slot,
                        cudaStream_t st) {
  if (G == 0 || E == 0) return cudaSuccess;
  dim3 grid(E, G);
  // columns up to 8192 scores: in registers, 16 per thread (128 threads for up to 2048, so
  // that every column of a 16-sequence batch is resident at once; 256 up to 4096; 512)
  if (max_group <= 8192) {
    if (max_group <= 2048)
      topk_reg_kernel<16, 128, 8><<<grid, 128, 0, st>>>(ST, N, E, group_off, k_g, k_off, M, idx,
                                                        gate, slot);
    else if (max_group <= 4096)
      topk_reg_kernel<16, 256, 4><<<grid, 256, 0, st>>>(ST, N, E, group_off, k_g, k_off, M, idx,
                                                        gate, slot);
    else
      topk_reg_kernel<16, 512, 2><<<grid, 512, 0, st>>>(ST, N, E, group_off, k_g, k_off, M, idx,
                                                        gate, slot);
    return cudaGetLastError();
  }
  // measured per column (phase timestamps, 512 columns of 4096 and 2048 columns of 2048
  // scores): 256 threads beat 512 on 4096-score columns (13.0 vs 14.2 us for the launch), and
  // 128 threads let every column of 2048 scores be resident at once (19.8 vs 22.1 us)
  const int threads = max_group > 8192 ? 512 : (max_group > 2048 ? 256 : 128);
  const size_t smem = ((size_t)max_group + 3) / 4 * 16;
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

// ------------------------------------------------------------------ capacity update
// Per-sequence capacities that change every step (Sec. 4.2) without a host round trip: the
// new k_g is read from device memory, checked, and the group tables are rewritten in place.
// One CTA; thread i owns a contiguous chunk of groups.
__global__ void __launch_bounds__(1024) set_capacity_kernel(const int* __restrict__ k_new,
                                                            const int* __restrict__ group_off,
                                                            int G, int M, int* __restrict__ k_g,
                                                            int* __restrict__ k_off,
                                                            int* __restrict__ status) {
  __shared__ long long s_part[1024];
  __shared__ int s_bad;
  const int tid = threadIdx.x, nthr = blockDim.x;
  const int chunk = (G + nthr - 1) / nthr;
  const int g0 = min(G, tid * chunk), g1 = min(G, g0 + chunk);
  if (tid == 0) s_bad = 0;
  long long sum = 0;
  bool bad = false;
  for (int g = g0; g < g1; ++g) {
    const int k = k_new[g];
    bad |= k < 0 || k > group_off[g + 1] - group_off[g];
    sum += k;
  }
  s_part[tid] = sum;
  __syncthreads();
  if (bad) s_bad = 1;
  // inclusive scan of the chunk sums (Hillis-Steele over 1024 entries)
  for (int o = 1; o < nthr; o <<= 1) {
    const long long u = tid >= o ? s_part[tid - o] : 0;
    __syncthreads();
    s_part[tid] += u;
    __syncthreads();
  }
  const long long total = s_part[nthr - 1];
  if (s_bad || total != (long long)M) {
    if (tid == 0) atomicExch(status, DEV_BAD_CAPACITY);
    return;
  }
  long long run = s_part[tid] - sum;   // exclusive prefix of this chunk
  for (int g = g0; g < g1; ++g) {
    const int k = k_new[g];
    k_g[g] = k;
    k_off[g] = (int)run;
    run += k;
  }
  if (tid == nthr - 1) k_off[G] = (int)total;
}

cudaError_t launch_set_capacity(const int* k_new, const int* group_off, int G, int M, int* k_g,
                                int* k_off, int* status, cudaStream_t st) {
  if (G <= 0) return cudaSuccess;
  set_capacity_kernel<<<1, 1024, 0, st>>>(k_new, group_off, G, M, k_g, k_off, status);
  return cudaGetLastError();
}

}  // namespace ecmoe
