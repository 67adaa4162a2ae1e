// Persistent, warp-specialised tcgen05 GEMM for sm_103a with fused epilogues.
//
// Each CTA (or 2-CTA cluster, PAIR) walks a static list of output tiles over a batch of
// problems (one per expert: expert choice gives every expert the same M rows, arXiv
// 2604.01622 Sec. 2.2; token choice gives each expert its own padded row region, VARM).
// Roles:
//   warp 0      TMA producer: 3-D tensor-map loads of A and B k-slices (64 deep, 128-byte
//               swizzle) into a STAGES-deep shared-memory ring, one mbarrier per slot.
//   warp 1      allocates TMEM; one thread issues tcgen05.mma (kind::f16, bf16 in, fp32
//               accumulate; M = 256 across the pair's two CTAs) into one of two TMEM
//               accumulators (or, for 256 x 512 tiles, into the two halves of one that fills
//               TMEM) and commits slot releases and "accumulator full" to mbarriers.
//   warps 2..   epilogue (4 or 8 warps): tcgen05.ld of the accumulator (one TMEM lane = one
//               output row), fused math (router softmax, SwiGLU with the gate, SwiGLU
//               backward with the gate gradient, casts); outputs staged in swizzled shared
//               memory and written by TMA stores; then the accumulator is released so the
//               next tile's MMAs can reuse it.
// Operands may be K-major or MN-major in global memory (tensor-core transpose bits), so
// no operand is ever repacked. Every mbarrier wait is bounded in time: on expiry the CTA
// records DEV_TIMEOUT in the status word, all roles leave their loops, and TMEM is freed.
#include <cuda.h>
#include <cstdio>
#include "common.cuh"
#include "gemm_tc.h"

namespace ecmoe {
namespace {

constexpr int BM = 128;   // rows per tile = TMEM lanes
constexpr int BK = 64;    // k-slice per stage: one 128-byte swizzle atom of bf16
constexpr unsigned long long WAIT_LIMIT_NS = 2000000000ull;  // 2 s

enum Epi : int {
  EPI_ROUTER = 0,        // softmax over the (valid) columns, S [rows][E] and S^T [E][rows]
  EPI_SWIGLU_FWD = 1,    // cols [0,BN/2) gate, [BN/2,BN) up -> A, B, U bf16
  EPI_STORE_BF16 = 2,    // plain bf16 store
  EPI_SWIGLU_BWD = 3,    // acc = dU; reads A, B; writes dA, dB bf16
  EPI_STORE_F32 = 4,     // plain fp32 store
  EPI_STORE_F32_SPLIT = 5, // cols [0,BN/2) -> out0, [BN/2,BN) -> out1, fp32
  EPI_ROUTER_ST = 6      // the router softmax with S and S^T leaving by TMA stores (BN <= 128)
};

struct Args {
  int batch, M, N, K;           // C[b] is M x N (N per half for split-column epilogues)
  int m_tiles, n_tiles, k_blocks, k_blocks0;
  void* out0;
  void* out1;
  void* out2;
  const void* in0;
  const void* in1;
  const float* bias;
  int64_t ld;                   // output row stride (elements)
  int64_t bstride;              // output batch stride (elements)
  int n_valid;                  // router: number of experts (out2: int map set to -1 beside S)
  int* status;
  // Variable rows per expert (token-choice routing): expert e owns padded rows
  // vm_tiles[e]*PADR .. vm_tiles[e+1]*PADR of the row-major activations, of which the first
  // vm_count[e] are real (the rest are zero). Device arrays, read by the kernel.
  const int* vm_tiles;          // [vm_E + 1] cumulative PADR-row blocks
  const int* vm_count;          // [vm_E] rows per expert
  int vm_E;
  // Gate per row (row b*M + m of a uniform batch, the padded row of variable rows), or
  // NULL for 1. SWIGLU_FWD writes U scaled by it; SWIGLU_BWD scales its accumulator by it
  // and writes the row's gate gradient <acc, silu(A)*B> as partial sums (one per n-tile
  // and column part) to dgate_part[(nt*parts + part) * dgate_stride + row].
  const float* gate;
  float* dgate_part;
  int64_t dgate_stride;
};

constexpr int PADR = 256;       // row padding unit of variable-row expert regions

// ------------------------------------------------------------------ PTX wrappers
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ unsigned long long globaltimer() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
// Wait for the phase of `bar` with parity `parity`. Gives up after `limit` ns or when
// another role of the CTA has given up; on expiry records DEV_TIMEOUT.
__device__ __noinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                       int* status, unsigned long long limit = WAIT_LIMIT_NS) {
  const uint32_t a = smem_u32(bar);
  if (mbar_try_wait(a, parity)) return true;
  const unsigned long long t0 = globaltimer();
  while (true) {
    for (int i = 0; i < 32; ++i)
      if (mbar_try_wait(a, parity)) return true;
    if (*abort_flag) return false;
    if (globaltimer() - t0 > limit) {
      *abort_flag = 1;
      atomicExch(status, DEV_TIMEOUT);
      return false;
    }
  }
}
__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* map, uint64_t* bar,
                                            int c0, int c1, int c2) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4, %5}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(c0), "r"(c1), "r"(c2)
      : "memory");
}
__device__ __forceinline__ void prefetch_map(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tmem_alloc(uint32_t* holder, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(holder)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                         uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}
// ---- CTA-pair (cluster of 2) forms: one MMA spans the two SMs' tensor cores, M = 256
__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// Shared-memory address of the same variable in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t mapa_shared(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" :::
                   "memory");
}
// Arrive on an mbarrier of either CTA of the cluster. Release at CTA scope: the arrival only
// tells the MMA issuer that this warp's TMEM loads have completed (tcgen05.wait::ld ran
// before it), so the warp's earlier global stores need not be made visible cluster-wide
// first (a cluster-scope release would stall on them).
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.release.cta.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr)
               : "memory");
}
// TMA load whose completion is signalled on an mbarrier of either CTA of the pair.
__device__ __forceinline__ void tma_load_3d_pair(void* dst, const CUtensorMap* map, uint32_t bar,
                                                 int c0, int c1, int c2) {
  asm volatile(
      "cp.async.bulk.tensor.3d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4, %5}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(c0), "r"(c1), "r"(c2)
      : "memory");
}
__device__ __forceinline__ void tmem_alloc_pair(uint32_t* holder, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(holder)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void mma_bf16_pair(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                              uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrive on the mbarrier at this shared offset in every CTA of `mask` once the MMAs issued
// so far have completed.
__device__ __forceinline__ void mma_commit_pair(uint64_t* bar, uint16_t mask) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
      " [%0], %1;" ::"r"(smem_u32(bar)),
      "h"(mask)
      : "memory");
}

// 32 consecutive fp32 columns of this thread's TMEM lane.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t* v) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),
        "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]),
        "=r"(v[14]), "=r"(v[15]), "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]),
        "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]), "=r"(v[25]),
        "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_wait_ld() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Shared-memory matrix descriptor (tcgen05 format): start, leading/stride byte offsets,
// descriptor version 1, 128-byte swizzle.
__device__ __forceinline__ uint64_t smem_desc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr >> 4) & 0x3FFFu);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
  d |= (uint64_t)1u << 46;
  d |= (uint64_t)2u << 61;
  return d;
}

// Instruction descriptor of kind::f16: fp32 accumulator, bf16 A and B, M x BN (M = 128 for
// one CTA, 256 for a CTA pair).
template <int BN, bool A_MN, bool B_MN, int MMA_M>
__host__ __device__ constexpr uint32_t instr_desc() {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((A_MN ? 1u : 0u) << 15) |
         ((B_MN ? 1u : 0u) << 16) | ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(MMA_M >> 4) << 24);
}

template <int BN>
__host__ __device__ constexpr uint32_t tmem_cols() {
  return 2 * BN <= 32 ? 32 : 2 * BN <= 64 ? 64 : 2 * BN <= 128 ? 128 : 2 * BN <= 256 ? 256 : 512;
}

// Epilogue staging: one 4 KB buffer per epilogue warp (a 32 x 32 fp32 chunk, or two 32 x 32
// bf16 chunks), written by the warp and stored to global memory by TMA. The staged router
// epilogue passes a chunk of S and then the same chunk of S^T through it, and keeps the bias
// row (up to 128 fp32) behind the buffers.
constexpr uint32_t STAGE_BUF = 4096;

__host__ __device__ constexpr uint32_t stage_bytes(int EPI, int EPW) {
  // staged router: two buffers per warp, the bias row (128 floats) and the per-row partial
  // maxima and sums the two warps of a lane quarter exchange (2 x 2 x 128 floats)
  // SwiGLU backward: the staging buffers and two [128] float arrays in which the second warp
  // of a lane quarter leaves its gate-gradient partial for the first
  return EPI == EPI_ROUTER ? 0u
         : EPI == EPI_ROUTER_ST ? EPW * STAGE_BUF + 512u + (EPW > 4 ? 1024u : 0u)
         : EPI == EPI_SWIGLU_BWD ? EPW * STAGE_BUF + 1024u
                                 : EPW * STAGE_BUF;
}

template <int BN, int STAGES, bool PAIR, int EPW, int EPI>
__host__ __device__ constexpr uint32_t smem_bytes() {
  return 1024 /*align slack*/ + STAGES * (BM * BK * 2 + (PAIR ? BN / 2 : BN) * BK * 2) +
         stage_bytes(EPI, EPW) + 256 /*barriers*/;
}

__device__ __forceinline__ float f32(uint32_t u) { return __uint_as_float(u); }


// Paired fp32 arithmetic (one instruction on both lanes of a 64-bit register pair, each lane
// rounded as the scalar instruction would): the SwiGLU epilogues work on column pairs.
__device__ __forceinline__ uint64_t f2(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void f2_split(uint64_t r, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(r));
}
__device__ __forceinline__ uint64_t f2_fma(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t f2_mul(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
// Logistic sigmoid of both lanes from the identity sigma(a) = (1 + tanh(a/2)) / 2, with the
// hardware tanh approximation (relative error ~2^-11, below the 2^-8 of the bf16 values the
// epilogues write): one special-function op per lane and one paired FMA.
__device__ __forceinline__ uint64_t f2_sigmoid(uint64_t a) {
  const uint64_t half = f2(0.5f, 0.5f);
  float h0, h1, t0, t1;
  f2_split(f2_mul(a, half), h0, h1);
  asm("tanh.approx.f32 %0, %1;" : "=f"(t0) : "f"(h0));
  asm("tanh.approx.f32 %0, %1;" : "=f"(t1) : "f"(h1));
  return f2_fma(f2(t0, t1), half, half);
}

// Stage this thread's row (row r of the warp's 32) of a 32 x 32 chunk for a TMA store:
// fp32 rows of 128 bytes in the 128-byte swizzle, bf16 rows of 64 bytes in the 64-byte
// swizzle (16-byte unit j of row r at unit j ^ (row bits of the address)), so the warp's
// 16-byte shared stores are free of bank conflicts.
__device__ __forceinline__ void stage_f32(uint8_t* buf, int r, const float* v) {
#pragma unroll
  for (int j = 0; j < 8; ++j)
    *reinterpret_cast<float4*>(buf + r * 128 + ((j ^ (r & 7)) << 4)) =
        make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
}
__device__ __forceinline__ void stage_bf16(uint8_t* buf, int r, const float* v) {
#pragma unroll
  for (int j = 0; j < 4; ++j)
    *reinterpret_cast<uint4*>(buf + r * 64 + ((j ^ ((r >> 1) & 3)) << 4)) =
        make_uint4(pack_bf16x2(v[8 * j], v[8 * j + 1]), pack_bf16x2(v[8 * j + 2], v[8 * j + 3]),
                   pack_bf16x2(v[8 * j + 4], v[8 * j + 5]),
                   pack_bf16x2(v[8 * j + 6], v[8 * j + 7]));
}
// The same layouts from words already in their output format: 16 words of two bf16 columns
// each, or 32 fp32 words, in column order.
__device__ __forceinline__ void stage_bf16w(uint8_t* buf, int r, const uint32_t* w) {
#pragma unroll
  for (int j = 0; j < 4; ++j)
    *reinterpret_cast<uint4*>(buf + r * 64 + ((j ^ ((r >> 1) & 3)) << 4)) =
        make_uint4(w[4 * j], w[4 * j + 1], w[4 * j + 2], w[4 * j + 3]);
}
__device__ __forceinline__ void stage_f32w(uint8_t* buf, int r, const uint32_t* w) {
#pragma unroll
  for (int j = 0; j < 8; ++j)
    *reinterpret_cast<uint4*>(buf + r * 128 + ((j ^ (r & 7)) << 4)) =
        make_uint4(w[4 * j], w[4 * j + 1], w[4 * j + 2], w[4 * j + 3]);
}
__device__ __forceinline__ void fence_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void tma_store_3d(const CUtensorMap* map, uint32_t src, int c0, int c1,
                                             int c2) {
  asm volatile(
      "cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%2, %3, %4}], [%1];" ::"l"(
          reinterpret_cast<uint64_t>(map)),
      "r"(src), "r"(c0), "r"(c1), "r"(c2)
      : "memory");
  asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}
// Wait until at most N of this thread's bulk store groups still read shared memory.
template <int N>
__device__ __forceinline__ void bulk_wait_read() {
  asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void bulk_wait_all() {
  asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}

// ------------------------------------------------------------------ tile decode
// VARM: 0 uniform batch of equal-M problems; 1 variable rows per expert (the M dimension,
// rows are global padded rows, B is the expert's weights); 2 variable K per expert (weight
// gradients: K runs over the expert's padded rows); 3 one problem whose rows are split
// evenly over the CTAs in 32-row units (the router: every CTA streams its own contiguous
// block of tokens, in tiles of up to 128 rows, so no SM is left with a second wave of whole
// tiles while others idle).
struct Tile {
  int b, mt, nt;
  int row0;      // first row of this CTA in the A / output row space
  int valid;     // rows from row0 that are real (the rest are masked)
  int kbl;       // k-blocks of this tile
  int krow0;     // first K row (variable K)
};

template <int VARM, int TM>
__device__ __forceinline__ Tile tile_at(const Args& p, int tile, int tiles_per_b, uint32_t rank) {
  static_assert(VARM != 1 || TM == PADR, "variable-row tiles are one padding unit high");
  static_assert(VARM != 3 || TM == BM, "row-split tiles are one CTA high");
  Tile t;
  if constexpr (VARM == 3) {
    // CTA c owns the 32-row units [c U / G, (c+1) U / G) of the U = ceil(M / 32) units; its
    // j-th tile (tile = c + j G) starts 128 j rows into that block. valid <= 0: the CTA has
    // fewer tiles than the longest block (every role skips it).
    const int G = (int)gridDim.x;
    const int c = tile % G, j = tile / G;
    const int64_t units = (p.M + 31) / 32;
    const int r0 = (int)(32 * ((int64_t)c * units / G));
    const int r1 = (int)min((int64_t)p.M, 32 * (((int64_t)c + 1) * units / G));
    t.b = 0;
    t.mt = j;
    t.nt = 0;
    t.row0 = r0 + j * BM;
    t.valid = min(BM, r1 - t.row0);
    t.kbl = p.k_blocks;
    t.krow0 = 0;
  } else if constexpr (VARM == 1) {
    const int mtile = tile / p.n_tiles;
    t.nt = tile - mtile * p.n_tiles;
    int lo = 0, hi = p.vm_E;   // last expert whose first block is at or before mtile
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (__ldg(p.vm_tiles + mid) <= mtile) lo = mid; else hi = mid;
    }
    t.b = lo;
    t.mt = mtile - __ldg(p.vm_tiles + lo);
    t.row0 = mtile * TM + (int)rank * BM;
    t.valid = __ldg(p.vm_count + lo) - (t.mt * TM + (int)rank * BM);
    t.kbl = p.k_blocks;
    t.krow0 = 0;
  } else {
    t.b = tile / tiles_per_b;
    const int rem = tile - t.b * tiles_per_b;
    t.mt = rem / p.n_tiles;
    t.nt = rem - t.mt * p.n_tiles;
    t.row0 = t.mt * TM + (int)rank * BM;
    t.valid = p.M - t.row0;
    if constexpr (VARM == 2) {
      t.kbl = (__ldg(p.vm_count + t.b) + BK - 1) / BK;
      t.krow0 = __ldg(p.vm_tiles + t.b) * PADR;
    } else {
      t.kbl = p.k_blocks;
      t.krow0 = 0;
    }
  }
  return t;
}

// ------------------------------------------------------------------ the kernel
// PAIR: the CTAs of a 2-CTA cluster share each 256 x BN tile. Each CTA loads its own 128 rows
// of A and half (BN/2 columns) of B; the leader CTA (rank 0) issues M = 256 MMAs that read
// both CTAs' shared memory and write each CTA's 128 rows into that CTA's TMEM. Per SM this
// halves the B traffic into shared memory.
//
// Wide tiles (BN = 512, pairs only): each k-slice feeds two N = 256 MMAs from one A slice, so
// an SM takes in 48 KB of operands per 2 x 128 x 256 x 64 MMA work instead of 32 KB per half
// of it (25% fewer bytes per FLOP). The accumulator then fills all 512 TMEM columns, so the
// two 256-column halves are handed over separately: the last TAIL k-slices issue their
// half-1 MMAs after half 0 has completed (the epilogue drains half 0 while they run), and the
// next tile issues its half-0 MMAs as soon as half 0 is free, holding its k-slices for the
// half-1 MMAs until the epilogue has drained half 1.
template <int BN, bool A_MN, bool B_MN, bool B_SPLIT, bool K_SPLIT, int EPI, int STAGES, int EPW,
          bool PAIR, int VARM>
__global__ void __launch_bounds__(64 + 32 * EPW, 1)
tc_gemm_kernel(const __grid_constant__ CUtensorMap mA0, const __grid_constant__ CUtensorMap mA1,
               const __grid_constant__ CUtensorMap mB0, const __grid_constant__ CUtensorMap mB1,
               const __grid_constant__ CUtensorMap mO0, const __grid_constant__ CUtensorMap mO1,
               const __grid_constant__ CUtensorMap mO2, const Args p) {
  constexpr bool WIDE = BN == 512;            // single accumulator handed over in two halves
  constexpr int NH = WIDE ? 2 : 1;            // accumulator segments per tile
  constexpr int SEGW = BN / NH;               // columns per segment = N of one MMA
  constexpr int TAIL = 3;                     // wide: k-slices whose half-1 MMAs go last
  constexpr int BNL = PAIR ? BN / 2 : BN;     // B columns held by this CTA
  constexpr int TM = PAIR ? 2 * BM : BM;      // tile rows
  constexpr uint32_t A_BYTES = BM * BK * 2;
  constexpr uint32_t B_BYTES = BNL * BK * 2;
  constexpr uint32_t TCOLS = WIDE ? 512u : tmem_cols<BN>();
  constexpr uint32_t IDESC = instr_desc<SEGW, A_MN, B_MN, TM>();
  static_assert(BN % 64 == 0 && (BN <= 256 || (WIDE && PAIR)), "BN");
  static_assert(!PAIR || BN % 128 == 0, "pair tiles split B in two 64-column multiples");
  static_assert(!WIDE || (EPI != EPI_ROUTER && EPI != EPI_ROUTER_ST && STAGES > TAIL),
                "wide tiles: plain, split-column and SwiGLU epilogues");
  static_assert(EPW == 4 || EPW == 8, "epilogue warps: one or two per TMEM lane quarter");
  static_assert(EPI != EPI_ROUTER || EPW == 4, "the plain router keeps whole rows per thread");
  static_assert(EPI != EPI_ROUTER_ST || (BN <= 128 && !PAIR), "staged router: up to 128 experts");
  // every epilogue except the plain router's writes through shared memory and TMA stores
  constexpr bool STAGED = EPI != EPI_ROUTER;

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + STAGES * A_BYTES;
  uint8_t* sStage = sB + STAGES * B_BYTES;   // 1024-aligned: A_BYTES, B_BYTES are multiples
  uint64_t* bars = reinterpret_cast<uint64_t*>(sStage + stage_bytes(EPI, EPW));
  uint64_t* full = bars;
  uint64_t* empty = bars + STAGES;
  uint64_t* tfull = bars + 2 * STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* mma_done = tempty + 2;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(mma_done + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = PAIR ? cluster_ctarank() : 0u;
  const bool leader = rank == 0;
  const int cid = PAIR ? (int)(blockIdx.x >> 1) : (int)blockIdx.x;  // tile walker index
  const int nwalk = PAIR ? (int)(gridDim.x >> 1) : (int)gridDim.x;
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], PAIR ? 2 * EPW : EPW);
    }
    mbar_init(mma_done, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    prefetch_map(&mA0);
    prefetch_map(&mB0);
    if (K_SPLIT) prefetch_map(&mA1);
    if (K_SPLIT || B_SPLIT) prefetch_map(&mB1);
  }
  if (STAGED && warp >= 2 && lane == 0) {
    prefetch_map(&mO0);
    if (EPI == EPI_SWIGLU_FWD || EPI == EPI_SWIGLU_BWD || EPI == EPI_STORE_F32_SPLIT ||
        EPI == EPI_ROUTER_ST)
      prefetch_map(&mO1);
    if (EPI == EPI_SWIGLU_FWD) prefetch_map(&mO2);
  }
  if (warp == 1) {
    if constexpr (PAIR) tmem_alloc_pair(tmem_holder, TCOLS);
    else tmem_alloc(tmem_holder, TCOLS);
  }
  tc_fence_before();
  __syncthreads();
  if constexpr (PAIR) cluster_sync();   // the peer's barriers are initialised before use
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;

  const int tiles_per_b = p.m_tiles * p.n_tiles;
  const int total = VARM == 1 ? __ldg(p.vm_tiles + p.vm_E) * p.n_tiles : p.batch * tiles_per_b;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      int s = 0;
      uint32_t ph = 0;
      bool ok = true;
      for (int tile = cid; tile < total && ok; tile += nwalk) {
        const Tile T = tile_at<VARM, TM>(p, tile, tiles_per_b, rank);
        if (VARM == 3 && T.valid <= 0) continue;
        const int nt = T.nt;
        const int m0 = T.row0;
        const int ab = VARM ? 0 : T.b;          // batch coordinate of A
        const int bb = VARM == 2 ? 0 : T.b;     // batch coordinate of B
        for (int kb = 0; kb < T.kbl; ++kb) {
          if (!mbar_wait(&empty[s], ph ^ 1u, abort_flag, p.status)) { ok = false; break; }
          if (!PAIR || leader) mbar_arrive_expect_tx(&full[s], (A_BYTES + B_BYTES) * (PAIR ? 2 : 1));
          // completion goes to the leader's barrier: it gates the pair's MMAs
          const uint32_t fb = PAIR ? mapa_shared(smem_u32(&full[s]), 0) : smem_u32(&full[s]);
          auto load_b = [&](void* dst, const CUtensorMap* m, int c0, int c1, int bc) {
            if constexpr (PAIR) tma_load_3d_pair(dst, m, fb, c0, c1, bc);
            else tma_load_3d(dst, m, &full[s], c0, c1, bc);
          };
          auto load = [&](void* dst, const CUtensorMap* m, int c0, int c1) {
            load_b(dst, m, c0, c1, bb);
          };
          const bool second = K_SPLIT && kb >= p.k_blocks0;
          const CUtensorMap* mA = second ? &mA1 : &mA0;
          const CUtensorMap* mB = second ? &mB1 : &mB0;
          const int k0 = (second ? kb - p.k_blocks0 : kb) * BK + T.krow0;
          uint8_t* a_dst = sA + s * A_BYTES;
          uint8_t* b_dst = sB + s * B_BYTES;
          if (!A_MN) {
            load_b(a_dst, mA, k0, m0, ab);
          } else {
#pragma unroll
            for (int j = 0; j < BM / 64; ++j) load_b(a_dst + j * 8192, mA, m0 + 64 * j, k0, ab);
          }
          if constexpr (PAIR) {
            // this CTA's half of each segment's B columns: for split tiles the gate (rank 0)
            // or up half
            const CUtensorMap* mb = B_SPLIT ? (rank ? &mB1 : &mB0) : mB;
#pragma unroll
            for (int h = 0; h < NH; ++h) {
              uint8_t* bh = b_dst + h * (B_BYTES / NH);
              const int n0 = B_SPLIT ? nt * (BN / 2) + h * (SEGW / 2)
                                     : nt * BN + h * SEGW + (int)rank * (BNL / NH);
              if (!B_MN) {
                load(bh, mb, k0, n0);
              } else {
#pragma unroll
                for (int j = 0; j < BNL / NH / 64; ++j) load(bh + j * 8192, mb, n0 + 64 * j, k0);
              }
            }
          } else if (!B_MN) {
            if constexpr (B_SPLIT) {
              const int n0h = nt * (BN / 2);
              load(b_dst, &mB0, k0, n0h);
              load(b_dst + (BN / 2) * 128, &mB1, k0, n0h);
            } else {
              load(b_dst, mB, k0, nt * BN);
            }
          } else {
            constexpr int NB = BN / 64;
#pragma unroll
            for (int j = 0; j < NB; ++j) {
              if constexpr (B_SPLIT) {
                const int n0h = nt * (BN / 2);
                const CUtensorMap* m = j < NB / 2 ? &mB0 : &mB1;
                load(b_dst + j * 8192, m, n0h + 64 * (j % (NB / 2)), k0);
              } else {
                load(b_dst + j * 8192, mB, nt * BN + 64 * j, k0);
              }
            }
          }
          if (++s == STAGES) { s = 0; ph ^= 1u; }
        }
      }
      if (!ok) {
        // let copies already issued land before the CTA leaves
        const unsigned long long t0 = globaltimer();
        while (globaltimer() - t0 < 1000000ull) {}
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer (leader CTA)
    if (lane == 0 && leader) {
      int s = 0;
      uint32_t ph = 0;
      bool ok = true;
      int it = 0;
      // the BK/16 MMAs of ring slot `st` with B segment h into TMEM column `tcol`; `first`: the
      // tile's first k-slice (the accumulator starts from zero)
      auto issue = [&](int st, int h, uint32_t tcol, bool first) {
        const uint32_t sa = smem_u32(sA + st * A_BYTES);
        const uint32_t sb = smem_u32(sB + st * B_BYTES + h * (B_BYTES / NH));
#pragma unroll
        for (int j = 0; j < BK / 16; ++j) {
          const uint64_t ad = A_MN ? smem_desc(sa + j * 2048, 8192, 1024)
                                   : smem_desc(sa + j * 32, 16, 1024);
          const uint64_t bd = B_MN ? smem_desc(sb + j * 2048, 8192, 1024)
                                   : smem_desc(sb + j * 32, 16, 1024);
          const uint32_t acc = (!first || j != 0) ? 1u : 0u;
          if constexpr (PAIR) mma_bf16_pair(tcol, ad, bd, IDESC, acc);
          else mma_bf16(tcol, ad, bd, IDESC, acc);
        }
      };
      // arrive on `bar` (in both CTAs of a pair) once the MMAs issued so far have completed
      auto commit = [&](uint64_t* bar) {
        if constexpr (PAIR) mma_commit_pair(bar, 0x3);
        else mma_commit(bar);
      };
      for (int tile = cid; tile < total && ok; tile += nwalk, ++it) {
        const Tile T0 = tile_at<VARM, TM>(p, tile, tiles_per_b, 0);
        if (VARM == 3 && T0.valid <= 0) { --it; continue; }
        const int kbl = T0.kbl;
        if constexpr (!WIDE) {
          const int a = it & 1;
          const uint32_t use = (uint32_t)(it >> 1);
          if (!mbar_wait(&tempty[a], (use & 1u) ^ 1u, abort_flag, p.status)) { ok = false; break; }
          tc_fence_after();
          const uint32_t tacc = tmem_base + (uint32_t)(a * BN);
          for (int kb = 0; kb < kbl; ++kb) {
            if (!mbar_wait(&full[s], ph, abort_flag, p.status)) { ok = false; break; }
            tc_fence_after();
            issue(s, 0, tacc, kb == 0);
            commit(&empty[s]);
            if (++s == STAGES) { s = 0; ph ^= 1u; }
          }
          if (!ok) break;
          commit(&tfull[a]);
        } else {
          // segment h of the single accumulator: TMEM columns [h*SEGW, (h+1)*SEGW)
          const uint32_t par = ((uint32_t)it & 1u) ^ 1u;   // previous tile's release of a half
          if (!mbar_wait(&tempty[0], par, abort_flag, p.status)) { ok = false; break; }
          tc_fence_after();
          bool h1 = mbar_try_wait(smem_u32(&tempty[1]), par);
          if (h1) tc_fence_after();
          // k-slices whose half-1 MMAs are still to be issued: `held` consecutive ones from
          // k-slice pk in ring slot ps (their slots stay occupied until then)
          int held = 0, pk = 0, ps = s;
          auto flush = [&]() {
            int st = ps;
            for (int i = 0; i < held; ++i) {
              issue(st, 1, tmem_base + SEGW, pk + i == 0);
              commit(&empty[st]);
              if (++st == STAGES) st = 0;
            }
            held = 0;
          };
          for (int kb = 0; kb < kbl; ++kb) {
            if (!h1) {
              // every slot held: the producer is stalled, so wait for half 1 here
              if (held == STAGES) {
                if (!mbar_wait(&tempty[1], par, abort_flag, p.status)) { ok = false; break; }
                h1 = true;
              } else {
                h1 = mbar_try_wait(smem_u32(&tempty[1]), par);
              }
              if (h1) {
                tc_fence_after();
                flush();
              }
            }
            if (!mbar_wait(&full[s], ph, abort_flag, p.status)) { ok = false; break; }
            tc_fence_after();
            issue(s, 0, tmem_base, kb == 0);
            if (h1 && kb < kbl - TAIL) {
              issue(s, 1, tmem_base + SEGW, kb == 0);
              commit(&empty[s]);
            } else {
              if (held == 0) { pk = kb; ps = s; }
              ++held;
            }
            if (++s == STAGES) { s = 0; ph ^= 1u; }
          }
          if (!ok) break;
          commit(&tfull[0]);   // half 0 is final once the MMAs issued so far complete
          if (!h1) {
            if (!mbar_wait(&tempty[1], par, abort_flag, p.status)) { ok = false; break; }
            tc_fence_after();
          }
          flush();
          commit(&tfull[1]);
        }
      }
      if (!ok) {
        // wait for the MMAs already issued before TMEM is released
        if constexpr (PAIR) mma_commit_pair(mma_done, 0x1);
        else mma_commit(mma_done);
        volatile int keep_waiting = 0;
        mbar_wait(mma_done, 0, &keep_waiting, p.status, 100000000ull);
      }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ epilogue (warps 2..)
    const int q = warp & 3;             // TMEM lane quarter this warp may access
    const int r = q * 32 + lane;        // row within the tile
    constexpr int NPART = EPW / 4;      // warps sharing a lane quarter split the columns
    const int part = (warp - 2) / 4;
    int slot = 0;   // staging half of the next bf16 chunk (warp-uniform)
    int it = 0;
    bool stop = false;
    // staged router: the bias row goes to shared memory once (every row reads all of it)
    float* s_bias = reinterpret_cast<float*>(sStage + EPW * STAGE_BUF);
    if constexpr (EPI == EPI_ROUTER_ST) {
      const int t = (int)threadIdx.x - 64;   // over the epilogue warps
      if (t < 128) s_bias[t] = (p.bias && t < p.n_valid) ? __ldg(p.bias + t) : 0.f;
      asm volatile("bar.sync 1, %0;" ::"n"(32 * EPW) : "memory");
    }
    for (int tile = cid; tile < total && !stop; tile += nwalk, ++it) {
      const Tile T = tile_at<VARM, TM>(p, tile, tiles_per_b, rank);
      if (VARM == 3 && T.valid <= 0) { --it; continue; }
      const int nt = T.nt;
      const int gm = T.row0 + r;
      const bool row_ok = r < T.valid;
      // Variable rows: a 256-row tile never leaves its expert's padded region, and the
      // region's unused rows are written as zeros (the weight gradients run their K loop
      // over them). Uniform batches store only the valid rows.
      const int64_t row_off =
          VARM == 1 ? (int64_t)gm * p.ld : (int64_t)T.b * p.bstride + (int64_t)gm * p.ld;
      const int64_t grow = VARM == 1 ? (int64_t)gm : (int64_t)T.b * p.M + gm;   // gate row
      // zero output: an empty expert's weight gradient, or a padding row
      const bool no_k = (VARM == 2 && T.kbl == 0) || (VARM == 1 && !row_ok);
      uint32_t v[32];
      float f[32];

      // Outputs leave through the warp's staging buffer: the warp writes a 32-row x 32-column
      // chunk (thread = row) into shared memory and lane 0 stores it with one TMA copy, which
      // also clips the rows past the tensor's end (rows that are not valid in a uniform batch).
      const int srow = T.row0 + q * 32;                    // first row of the warp's block
      const int sbat = VARM == 1 ? 0 : T.b;                // batch coordinate of the output
      const bool st_any = VARM == 1 || T.valid > q * 32;   // the block has a row to store
      auto put_bf16 = [&](const CUtensorMap* m, int n, const float* vals) {
        if (lane == 0) bulk_wait_read<1>();   // this slot's previous store has read it
        __syncwarp();
        uint8_t* b = sStage + (warp - 2) * STAGE_BUF + slot * 2048;
        stage_bf16(b, lane, vals);
        fence_async_smem();
        __syncwarp();
        if (lane == 0) tma_store_3d(m, smem_u32(b), n, srow, sbat);
        slot ^= 1;
      };
      // two bf16 chunks at once (both halves of the buffer, one proxy fence): each store is
      // its own bulk group, the first one (half 0) the older
      auto put2_bf16 = [&](const CUtensorMap* m0, const CUtensorMap* m1, int n, const float* v0,
                           const float* v1) {
        if (lane == 0) bulk_wait_read<0>();
        __syncwarp();
        uint8_t* b = sStage + (warp - 2) * STAGE_BUF;
        stage_bf16(b, lane, v0);
        stage_bf16(b + 2048, lane, v1);
        fence_async_smem();
        __syncwarp();
        if (lane == 0) {
          tma_store_3d(m0, smem_u32(b), n, srow, sbat);
          tma_store_3d(m1, smem_u32(b + 2048), n, srow, sbat);
        }
        slot = 0;   // the next single chunk goes to half 0 once its store (the older) has read it
      };
      auto put_f32 = [&](const CUtensorMap* m, int n, const float* vals) {
        if (lane == 0) bulk_wait_read<0>();
        __syncwarp();
        uint8_t* b = sStage + (warp - 2) * STAGE_BUF;
        stage_f32(b, lane, vals);
        fence_async_smem();
        __syncwarp();
        if (lane == 0) tma_store_3d(m, smem_u32(b), n, srow, sbat);
      };
      // the same from words in the output format (wide tiles, whose segments are read into
      // registers before they are stored)
      auto put_bf16w = [&](const CUtensorMap* m, int n, const uint32_t* w) {
        if (lane == 0) bulk_wait_read<1>();
        __syncwarp();
        uint8_t* b = sStage + (warp - 2) * STAGE_BUF + slot * 2048;
        stage_bf16w(b, lane, w);
        fence_async_smem();
        __syncwarp();
        if (lane == 0) tma_store_3d(m, smem_u32(b), n, srow, sbat);
        slot ^= 1;
      };
      auto put_f32w = [&](const CUtensorMap* m, int n, const uint32_t* w) {
        if (lane == 0) bulk_wait_read<0>();
        __syncwarp();
        uint8_t* b = sStage + (warp - 2) * STAGE_BUF;
        stage_f32w(b, lane, w);
        fence_async_smem();
        __syncwarp();
        if (lane == 0) tma_store_3d(m, smem_u32(b), n, srow, sbat);
      };
      // hand accumulator segment a back to the MMA issuer (its TMEM loads have completed)
      auto release = [&](int a) {
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          if constexpr (PAIR) mbar_arrive_cluster(mapa_shared(smem_u32(&tempty[a]), 0));
          else mbar_arrive(&tempty[a]);
        }
      };

      // Staged router: the slot map's rows of this warp's tokens are one contiguous block set
      // to -1 throughout (split between the warps of the lane quarter); it does not depend on
      // the accumulator, so it is written while the tile's main loop runs.
      if constexpr (EPI == EPI_ROUTER_ST) {
        int* smap = reinterpret_cast<int*>(p.out2);
        if (smap && st_any) {
          const int E = p.n_valid;
          const int nrow = min(32, T.valid - q * 32);
          int4* blk = reinterpret_cast<int4*>(smap + (int64_t)srow * E);
          const int n4 = nrow * (E >> 2);
          for (int j = lane + part * 32; j < n4; j += 32 * NPART)
            blk[j] = make_int4(-1, -1, -1, -1);
        }
      }
      // The accumulator segments (one, or a wide tile's two halves, each released as soon
      // as it is drained): segment h holds tile columns [h*SEGW, (h+1)*SEGW).
      for (int h = 0; h < NH; ++h) {
        const int a = WIDE ? h : (it & 1);
        const uint32_t par = WIDE ? (uint32_t)(it & 1) : (uint32_t)((it >> 1) & 1);
        if (!mbar_wait(&tfull[a], par, abort_flag, p.status)) { stop = true; break; }
        tc_fence_after();
        const uint32_t tacc = tmem_base + (uint32_t)(WIDE ? h * SEGW : a * BN) +
                              ((uint32_t)(q * 32) << 16);
        const int cb = h * SEGW;                   // first tile column of the segment
        constexpr int NC32 = SEGW / 32 / NPART;    // 32-column chunks per warp
        const int c32 = part * NC32;
        if constexpr (EPI == EPI_SWIGLU_BWD) {
          // Both tile forms, segment by segment (columns cb.. of the tile). A and B of the next
          // chunk are requested before the current one is computed (not with variable rows,
          // whose tile decode leaves too few registers for the second set). The segment goes
          // back to the MMA issuer as soon as its last chunk has been read from TMEM.
          constexpr bool PREFETCH = VARM != 1;
          const bf16* pa = reinterpret_cast<const bf16*>(p.in0) + row_off + nt * BN + cb;
          const bf16* pb = reinterpret_cast<const bf16*>(p.in1) + row_off + nt * BN + cb;
          uint4 ra[4], rb[4], na[4], nb[4];
#pragma unroll
          for (int i = 0; i < 4; ++i) ra[i] = rb[i] = na[i] = nb[i] = make_uint4(0, 0, 0, 0);
          auto fetch = [&](int c, uint4* xa, uint4* xb) {
            const int n = nt * BN + cb + c * 32;
            if (row_ok && n < p.N) {
#pragma unroll
              for (int i = 0; i < 4; ++i) {
                xa[i] = __ldg(reinterpret_cast<const uint4*>(pa + c * 32) + i);
                xb[i] = __ldg(reinterpret_cast<const uint4*>(pb + c * 32) + i);
              }
            }
          };
          if (PREFETCH) fetch(c32, ra, rb);
          const float gs = (p.gate && row_ok) ? __ldg(p.gate + grow) : 1.0f;
          // <acc, silu(A) * B> over this warp's columns of the row: even and odd columns
          uint64_t dot2 = f2(0.f, 0.f);
#pragma unroll 1
          for (int c = c32; c < c32 + NC32; ++c) {
            if (!PREFETCH) fetch(c, ra, rb);
            else if (c + 1 < c32 + NC32) fetch(c + 1, na, nb);
            tmem_ld32(tacc + c * 32, v);
            tmem_wait_ld();
            if (c == c32 + NC32 - 1) release(a);   // the segment's last TMEM read has completed
            const int n = nt * BN + cb + c * 32;
            if (st_any && n < p.N) {
              float av[32], bv[32];   // av ends up holding dB
              if (no_k) {
#pragma unroll
                for (int i = 0; i < 32; ++i) f[i] = av[i] = 0.f;
              } else {
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                  unpack16(ra[i], av + 8 * i, bf16());
                  unpack16(rb[i], bv + 8 * i, bf16());
                }
                // two columns at a time: dU = gs acc, sg = sigma(a), dA = dU b sg (1 + a (1 - sg)),
                // dB = dU a sg, and the gate-gradient terms acc a sg b
                const uint64_t gs2 = f2(gs, gs), one2 = f2(1.f, 1.f), mone2 = f2(-1.f, -1.f);
#pragma unroll
                for (int i = 0; i < 32; i += 2) {
                  const uint64_t a2 = f2(av[i], av[i + 1]);
                  const uint64_t b2 = f2(bv[i], bv[i + 1]);
                  const uint64_t c2 = f2(f32(v[i]), f32(v[i + 1]));
                  const uint64_t sg2 = f2_sigmoid(a2);
                  const uint64_t das2 = f2_mul(f2_mul(gs2, c2), sg2);
                  dot2 = f2_fma(c2, f2_mul(f2_mul(a2, sg2), b2), dot2);
                  const uint64_t q2 = f2_fma(a2, f2_fma(sg2, mone2, one2), one2);
                  f2_split(f2_mul(f2_mul(das2, b2), q2), f[i], f[i + 1]);
                  f2_split(f2_mul(das2, a2), av[i], av[i + 1]);
                }
              }
              put2_bf16(&mO0, &mO1, n, f, av);
            }
            if (PREFETCH)
#pragma unroll
              for (int i = 0; i < 4; ++i) { ra[i] = na[i]; rb[i] = nb[i]; }
          }
          // Partial j of a row covers output columns [256 j, 256 j + 256) (the same partials
          // for both tile forms): the second warp of the lane quarter leaves its sum in shared
          // memory and the first adds it to its own (in that order). The two buffers alternate
          // between segments, so one barrier per segment keeps them apart.
          if (p.dgate_part) {
            float de, dd;
            f2_split(dot2, de, dd);
            float pd = de + dd;
            if constexpr (NPART > 1) {
              float* s_dg = reinterpret_cast<float*>(sStage + EPW * STAGE_BUF) +
                            (((it * NH + h) & 1) << 7);
              if (part == 1) s_dg[r] = pd;
              asm volatile("bar.sync %0, 64;" ::"r"(2 + q) : "memory");
              pd += s_dg[r];
            }
            if (part == 0 && row_ok)
              p.dgate_part[(int64_t)(nt * NH + h) * p.dgate_stride + grow] = pd;
          }
        } else if constexpr (WIDE) {
          // The segment's values go to registers first (packed to bf16 where the output is
          // bf16), the segment is handed back to the MMA issuer, and only then are the chunks
          // staged and stored: the next tile's MMAs wait for the TMEM reads alone.
          if constexpr (EPI == EPI_STORE_BF16) {
            uint32_t pk[NC32][16];
#pragma unroll
            for (int i = 0; i < NC32; ++i) {
              tmem_ld32(tacc + (c32 + i) * 32, v);
              tmem_wait_ld();
              if (i == NC32 - 1) release(a);   // the segment's last TMEM read has completed
#pragma unroll
              for (int j = 0; j < 16; ++j)
                pk[i][j] = no_k ? 0u : pack_bf16x2(f32(v[2 * j]), f32(v[2 * j + 1]));
            }
#pragma unroll
            for (int i = 0; i < NC32; ++i) {
              const int n = nt * BN + cb + (c32 + i) * 32;
              if (st_any && n < p.N) put_bf16w(&mO0, n, pk[i]);
            }
          } else if constexpr (EPI == EPI_STORE_F32 || EPI == EPI_STORE_F32_SPLIT) {
            uint32_t raw[NC32][32];
#pragma unroll
            for (int i = 0; i < NC32; ++i) tmem_ld32(tacc + (c32 + i) * 32, raw[i]);
            tmem_wait_ld();
            release(a);
#pragma unroll
            for (int i = 0; i < NC32; ++i) {
              const int c = c32 + i;
              if (no_k) {
#pragma unroll
                for (int j = 0; j < 32; ++j) raw[i][j] = 0u;
              }
              if constexpr (EPI == EPI_STORE_F32) {
                const int n = nt * BN + cb + c * 32;
                if (st_any && n < p.N) put_f32w(&mO0, n, raw[i]);
              } else {
                const int half = c >= SEGW / 64;
                const int n = nt * (BN / 2) + cb / 2 + (c % (SEGW / 64)) * 32;
                if (st_any && n < p.N) put_f32w(half ? &mO1 : &mO0, n, raw[i]);
              }
            }
          } else if constexpr (EPI == EPI_SWIGLU_FWD) {
            // column pairs (gate chunk, up chunk): a pair's A, B, U are packed while the next
            // pair's TMEM reads are in flight and stored once the segment is released
            constexpr int NC64 = SEGW / 64 / NPART;
            uint32_t pa[16], pb[16], pu[16];
            const float gs = (p.gate && row_ok) ? __ldg(p.gate + grow) : 1.0f;
            const uint64_t gs2 = f2(gs, gs);
            auto store_pair = [&](int c) {
              const int n = nt * (BN / 2) + cb / 2 + c * 32;
              if (st_any && n < p.N) {
                put_bf16w(&mO0, n, pa);
                put_bf16w(&mO1, n, pb);
                put_bf16w(&mO2, n, pu);
              }
            };
#pragma unroll
            for (int i = 0; i < NC64; ++i) {
              uint32_t w[32];
              const int c = part * NC64 + i;
              tmem_ld32(tacc + c * 32, v);
              tmem_ld32(tacc + SEGW / 2 + c * 32, w);
              tmem_wait_ld();
              if (i == NC64 - 1) release(a);   // the segment's last TMEM read has completed
              if (i > 0) store_pair(c - 1);
#pragma unroll
              for (int j = 0; j < 32; j += 2) {   // U = gs * silu(A) * B, two columns at a time
                const float a0 = no_k ? 0.f : f32(v[j]), a1 = no_k ? 0.f : f32(v[j + 1]);
                const float b0 = no_k ? 0.f : f32(w[j]), b1 = no_k ? 0.f : f32(w[j + 1]);
                const uint64_t a2 = f2(a0, a1);
                const uint64_t u2 = f2_mul(gs2, f2_mul(f2_mul(a2, f2_sigmoid(a2)), f2(b0, b1)));
                float u0, u1;
                f2_split(u2, u0, u1);
                pa[j / 2] = pack_bf16x2(a0, a1);
                pb[j / 2] = pack_bf16x2(b0, b1);
                pu[j / 2] = pack_bf16x2(u0, u1);
              }
            }
            store_pair(part * NC64 + NC64 - 1);
          }
        } else if constexpr (EPI == EPI_STORE_BF16 || EPI == EPI_STORE_F32) {
#pragma unroll 1
          for (int c = c32; c < c32 + NC32; ++c) {
            tmem_ld32(tacc + c * 32, v);
            tmem_wait_ld();
            const int n = nt * BN + cb + c * 32;
            if (st_any && n < p.N) {
#pragma unroll
              for (int i = 0; i < 32; ++i) f[i] = no_k ? 0.f : f32(v[i]);
              if constexpr (EPI == EPI_STORE_BF16) put_bf16(&mO0, n, f);
              else put_f32(&mO0, n, f);
            }
          }
        } else if constexpr (EPI == EPI_STORE_F32_SPLIT) {
#pragma unroll 1
          for (int c = c32; c < c32 + NC32; ++c) {
            tmem_ld32(tacc + c * 32, v);
            tmem_wait_ld();
            const int half = c >= SEGW / 64;
            const int n = nt * (BN / 2) + cb / 2 + (c % (SEGW / 64)) * 32;
            if (st_any && n < p.N) {
#pragma unroll
              for (int i = 0; i < 32; ++i) f[i] = no_k ? 0.f : f32(v[i]);
              put_f32(half ? &mO1 : &mO0, n, f);
            }
          }
        } else if constexpr (EPI == EPI_SWIGLU_FWD) {
          uint32_t w[32];
          constexpr int NC64 = SEGW / 64 / NPART;
          const float gs = (p.gate && row_ok) ? __ldg(p.gate + grow) : 1.0f;
#pragma unroll 1
          for (int c = part * NC64; c < (part + 1) * NC64; ++c) {
            tmem_ld32(tacc + c * 32, v);
            tmem_ld32(tacc + SEGW / 2 + c * 32, w);
            tmem_wait_ld();
            const int n = nt * (BN / 2) + cb / 2 + c * 32;
            if (st_any && n < p.N) {
              float g[32];
#pragma unroll
              for (int i = 0; i < 32; ++i) {
                f[i] = no_k ? 0.f : f32(v[i]);
                g[i] = no_k ? 0.f : f32(w[i]);
              }
              put2_bf16(&mO0, &mO1, n, f, g);
              const uint64_t gs2 = f2(gs, gs);
#pragma unroll
              for (int i = 0; i < 32; i += 2) {   // U = gs * silu(A) * B, two columns at a time
                const uint64_t a2 = f2(f[i], f[i + 1]);
                const uint64_t u2 =
                    f2_mul(gs2, f2_mul(f2_mul(a2, f2_sigmoid(a2)), f2(g[i], g[i + 1])));
                f2_split(u2, f[i], f[i + 1]);
              }
              put_bf16(&mO2, n, f);
            }
          }
        } else if constexpr ((EPI == EPI_ROUTER || EPI == EPI_ROUTER_ST) && BN <= 128) {
          // up to 128 experts the row's logits stay in registers: one TMEM read, exp once;
          // the staged form stores S and S^T as 32 x 32 chunks by TMA, the plain one writes
          // the row of S with 16-byte stores when E allows it. With two warps per lane quarter
          // (staged form) each takes half of the row's chunks and the pair exchanges its
          // partial maximum and sum through shared memory.
          const int E = p.n_valid;
          constexpr int NCH = BN / 32 / NPART;     // chunks of 32 experts per warp
          const int cb0 = part * NCH;              // first chunk of this warp
          float ev[NCH][32];
          float mx = -INFINITY;
#pragma unroll
          for (int c = 0; c < NCH; ++c) {
            tmem_ld32(tacc + (cb0 + c) * 32, v);
            tmem_wait_ld();
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const int e = (cb0 + c) * 32 + i;
              float bias = 0.f;
              if constexpr (EPI == EPI_ROUTER_ST) {
                if (e < E) bias = s_bias[e];
              } else {
                bias = p.bias && e < E ? __ldg(p.bias + e) : 0.f;
              }
              ev[c][i] = e < E ? f32(v[i]) + bias : -INFINITY;
              mx = fmaxf(mx, ev[c][i]);
            }
          }
          // [NPART][128]: slot `part` first holds this warp's maximum for the partner, then
          // (written by the partner once it has read that maximum) the partner's sum
          float* s_x = s_bias + 128;
          if constexpr (NPART > 1) {
            s_x[part * 128 + r] = mx;
            asm volatile("bar.sync %0, 64;" ::"r"(2 + q) : "memory");
            mx = fmaxf(mx, s_x[(1 - part) * 128 + r]);
          }
          // exp through the hardware exp2 approximation (relative error ~1e-7, far below the
          // bf16 inputs' rounding); four independent partial sums, added in a fixed order
          float ps[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
          for (int c = 0; c < NCH; ++c)
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              ev[c][i] = (cb0 + c) * 32 + i < E ? __expf(ev[c][i] - mx) : 0.f;
              ps[i & 3] += ev[c][i];
            }
          float sum = (ps[0] + ps[1]) + (ps[2] + ps[3]);
          if constexpr (NPART > 1) {
            s_x[(1 - part) * 128 + r] = sum;       // the partner's maximum was read above
            asm volatile("bar.sync %0, 64;" ::"r"(2 + q) : "memory");
            // the same order in both warps: part 0's sum first
            const float os = s_x[part * 128 + r];
            sum = part == 0 ? sum + os : os + sum;
          }
          const float inv = 1.0f / sum;
          int* smap = reinterpret_cast<int*>(p.out2);
          if constexpr (EPI == EPI_ROUTER_ST) {
            // chunk c through the warp's staging buffer: first the S rows of its 32 tokens
            // (128-byte swizzle, thread = row), then, once that store has read the buffer, the
            // same values as S^T rows of 32 experts (thread = column: each expert's row of 32
            // tokens is one 128-byte line of the buffer, so the stores are conflict-free)
            uint8_t* bS = sStage + (warp - 2) * STAGE_BUF;
#pragma unroll
            for (int c = 0; c < NCH; ++c) {
              const int cg = cb0 + c;
#pragma unroll
              for (int i = 0; i < 32; ++i) ev[c][i] *= inv;
              if (cg * 32 >= E || !st_any) continue;
              if (lane == 0) bulk_wait_read<0>();   // the buffer's last store has read it
              __syncwarp();
              stage_f32(bS, lane, ev[c]);
              fence_async_smem();
              __syncwarp();
              if (lane == 0) {
                tma_store_3d(&mO0, smem_u32(bS), cg * 32, srow, 0);
                bulk_wait_read<0>();
              }
              __syncwarp();
#pragma unroll
              for (int i = 0; i < 32; ++i)
                *reinterpret_cast<float*>(bS + i * 128 + ((((lane >> 2) ^ (i & 7)) << 4) |
                                                          ((lane & 3) << 2))) = ev[c][i];
              fence_async_smem();
              __syncwarp();
              if (lane == 0) tma_store_3d(&mO1, smem_u32(bS), srow, cg * 32, 0);
            }
          } else {
          float* S = reinterpret_cast<float*>(p.out0);
          float* ST = reinterpret_cast<float*>(p.out1);
          int* slot = smap;
          const bool vec = (E & 3) == 0;   // rows of S start on 16-byte boundaries
#pragma unroll
          for (int c = 0; c < NCH; ++c) {
#pragma unroll
            for (int i = 0; i < 32; ++i) ev[c][i] *= inv;
            if (row_ok) {
              float* srow = S + (int64_t)gm * E + c * 32;
              int* lrow = slot ? slot + (int64_t)gm * E + c * 32 : nullptr;
              if (vec && c * 32 + 32 <= E) {
#pragma unroll
                for (int j = 0; j < 8; ++j)
                  reinterpret_cast<float4*>(srow)[j] =
                      make_float4(ev[c][4 * j], ev[c][4 * j + 1], ev[c][4 * j + 2], ev[c][4 * j + 3]);
                if (lrow)
#pragma unroll
                  for (int j = 0; j < 8; ++j)
                    reinterpret_cast<int4*>(lrow)[j] = make_int4(-1, -1, -1, -1);
              } else {
#pragma unroll
                for (int i = 0; i < 32; ++i)
                  if (c * 32 + i < E) {
                    srow[i] = ev[c][i];
                    if (lrow) lrow[i] = -1;
                  }
              }
#pragma unroll
              for (int i = 0; i < 32; ++i)
                if (c * 32 + i < E) ST[(int64_t)(c * 32 + i) * p.M + gm] = ev[c][i];
            }
          }
          }
        } else if constexpr (EPI == EPI_ROUTER) {
          const int E = p.n_valid;
          float mx = -INFINITY;
#pragma unroll 1
          for (int c = 0; c < BN / 32; ++c) {
            tmem_ld32(tacc + c * 32, v);
            tmem_wait_ld();
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const int e = c * 32 + i;
              if (e < E) mx = fmaxf(mx, f32(v[i]) + (p.bias ? p.bias[e] : 0.f));
            }
          }
          float sum = 0.f;
#pragma unroll 1
          for (int c = 0; c < BN / 32; ++c) {
            tmem_ld32(tacc + c * 32, v);
            tmem_wait_ld();
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const int e = c * 32 + i;
              if (e < E) sum += __expf(f32(v[i]) + (p.bias ? p.bias[e] : 0.f) - mx);
            }
          }
          const float inv = 1.0f / sum;
          float* S = reinterpret_cast<float*>(p.out0);
          float* ST = reinterpret_cast<float*>(p.out1);
          int* slot = reinterpret_cast<int*>(p.out2);
#pragma unroll 1
          for (int c = 0; c < BN / 32; ++c) {
            tmem_ld32(tacc + c * 32, v);
            tmem_wait_ld();
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const int e = c * 32 + i;
              if (e < E && row_ok) {
                const float pr = __expf(f32(v[i]) + (p.bias ? p.bias[e] : 0.f) - mx) * inv;
                S[(int64_t)gm * E + e] = pr;
                ST[(int64_t)e * p.M + gm] = pr;
                if (slot) slot[(int64_t)gm * E + e] = -1;
              }
            }
          }
        }
        // the accumulator is free again: tell the CTA that issues the MMAs
        if constexpr (!WIDE && EPI != EPI_SWIGLU_BWD) release(a);
      }   // segments
    }
    // the TMA stores read the staging buffers until they complete
    if (STAGED && lane == 0) bulk_wait_all();
    __syncwarp();
  }
  tc_fence_before();
  __syncthreads();
  if constexpr (PAIR) cluster_sync();   // the pair's MMAs and remote arrivals are done
  if (warp == 1) {
    tc_fence_after();
    if constexpr (PAIR) tmem_dealloc_pair(tmem_base, TCOLS);
    else tmem_dealloc(tmem_base, TCOLS);
  }
}

// ------------------------------------------------------------------ host side
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  }
  return fn;
}

// 3-D bf16 tensor [batch][rows][cols] (cols contiguous), box {64, box_rows, 1}, 128B swizzle.
cudaError_t make_map(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows,
                     uint64_t batch, uint32_t box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return cudaErrorNotSupported;
  cuuint64_t dims[3] = {cols, rows, batch};
  cuuint64_t strides[2] = {cols * 2, cols * rows * 2};
  cuuint32_t box[3] = {64, box_rows, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

// 3-D output tensor [batch][rows][cols] for the epilogue's TMA stores: box of 32 rows x 32
// columns, bf16 with the 64-byte swizzle or fp32 with the 128-byte swizzle (one staged chunk).
cudaError_t make_out_map(CUtensorMap* m, const void* base, bool f32, uint64_t cols, uint64_t rows,
                         uint64_t batch) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return cudaErrorNotSupported;
  const uint64_t es = f32 ? 4 : 2;
  cuuint64_t dims[3] = {cols, rows, batch};
  cuuint64_t strides[2] = {cols * es, cols * rows * es};
  cuuint32_t box[3] = {32, 32, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = fn(m, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3,
                  const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                  f32 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B,
                  CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

int sm_count() {
  static int n = 0;
  if (!n) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 1;
  }
  return n;
}

template <int BN, bool A_MN, bool B_MN, bool B_SPLIT, bool K_SPLIT, int EPI, int STAGES,
          int EPW = 8, bool PAIR = false, int VARM = 0>
cudaError_t launch(const CUtensorMap& a0, const CUtensorMap& a1, const CUtensorMap& b0,
                   const CUtensorMap& b1, const CUtensorMap& o0, const CUtensorMap& o1,
                   const CUtensorMap& o2, Args p, cudaStream_t st) {
  auto kern = tc_gemm_kernel<BN, A_MN, B_MN, B_SPLIT, K_SPLIT, EPI, STAGES, EPW, PAIR, VARM>;
  constexpr uint32_t smem = smem_bytes<BN, STAGES, PAIR, EPW, EPI>();
  static_assert(smem <= 232448, "dynamic shared memory above the 227 KB per-block limit");
  constexpr int threads = 64 + 32 * EPW;
  static bool attr = false;
  static int max_clusters = 0;
  cudaLaunchAttribute cl[1];
  cl[0].id = cudaLaunchAttributeClusterDimension;
  cl[0].val.clusterDim.x = 2;
  cl[0].val.clusterDim.y = 1;
  cl[0].val.clusterDim.z = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(threads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  if (PAIR) {
    cfg.attrs = cl;
    cfg.numAttrs = 1;
  }
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    if (PAIR) {
      cfg.gridDim = dim3(2 * sm_count());
      e = cudaOccupancyMaxActiveClusters(&max_clusters, kern, &cfg);
      if (e != cudaSuccess) return e;
      if (max_clusters <= 0) return cudaErrorNotSupported;
    }
    attr = true;
  }
  // variable rows: p.M carries an upper bound of the padded rows, so `total` bounds the tiles
  if (PAIR) p.m_tiles = (p.M + 2 * BM - 1) / (2 * BM);
  if constexpr (VARM == 3) {
    // one CTA per SM (at most one per 32-row unit), each with the tiles of its row block
    static_assert(!PAIR, "row split: single-CTA tiles");
    const int64_t units = (p.M + 31) / 32;
    if (units == 0 || p.k_blocks == 0) return cudaSuccess;
    const int g = (int)(units < sm_count() ? units : sm_count());
    const int64_t max_rows = 32 * ((units + g - 1) / g);
    p.batch = 1;
    p.n_tiles = 1;
    p.m_tiles = g * (int)((max_rows + BM - 1) / BM);
    kern<<<g, threads, smem, st>>>(a0, a1, b0, b1, o0, o1, o2, p);
    return cudaGetLastError();
  }
  const int total = p.batch * p.m_tiles * p.n_tiles;
  if (total == 0 || (VARM != 2 && p.k_blocks == 0)) return cudaSuccess;
  if (PAIR) {
    const int clusters = total < max_clusters ? total : max_clusters;
    cfg.gridDim = dim3(2 * clusters);
    return cudaLaunchKernelEx(&cfg, kern, a0, a1, b0, b1, o0, o1, o2, p);
  }
  const int grid = total < sm_count() ? total : sm_count();
  kern<<<grid, threads, smem, st>>>(a0, a1, b0, b1, o0, o1, o2, p);
  return cudaGetLastError();
}

Args base_args(int batch, int M, int N, int K, int BN_tile, int* status) {
  Args p{};
  p.batch = batch;
  p.M = M;
  p.N = N;
  p.K = K;
  p.m_tiles = (M + BM - 1) / BM;
  p.n_tiles = (N + BN_tile - 1) / BN_tile;
  p.k_blocks = (K + BK - 1) / BK;
  p.k_blocks0 = p.k_blocks;
  p.status = status;
  return p;
}

__global__ void pad_router_weights(const bf16* __restrict__ Wr, bf16* __restrict__ Wp, int d,
                                   int E, int Ep) {
  const int64_t n = (int64_t)d * Ep;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int e = (int)(i % Ep);
    const int64_t k = i / Ep;
    Wp[i] = e < E ? Wr[k * E + e] : __float2bfloat16_rn(0.f);
  }
}

__global__ void wait_probe_kernel(int* status, unsigned long long limit) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) mbar_wait(&bar, 0, &abort_flag, status, limit);
}

}  // namespace

#define TC_TRY(x)                        \
  do {                                   \
    cudaError_t _e = (x);                \
    if (_e != cudaSuccess) return _e;    \
  } while (0)

bool router_needs_pad(int E) { return E % 64 != 0; }

cudaError_t tc_router_softmax(const void* X, const void* Wr, void* Wr_pad, const float* br,
                              float* S, float* ST, int* slot_init, int N, int d, int E,
                              int* status, cudaStream_t st) {
  if (N == 0) return cudaSuccess;
  const int Ep = (E + 63) / 64 * 64;
  // Wr [d][E] already has the padded layout when E is a multiple of 64
  const void* Wb = Wr;
  if (router_needs_pad(E)) {
    pad_router_weights<<<256, 256, 0, st>>>(static_cast<const bf16*>(Wr),
                                            static_cast<bf16*>(Wr_pad), d, E, Ep);
    TC_TRY(cudaGetLastError());
    Wb = Wr_pad;
  }
  CUtensorMap ma, mb;
  TC_TRY(make_map(&ma, X, d, N, 1, BM));
  TC_TRY(make_map(&mb, Wb, Ep, d, 1, 64));
  Args p = base_args(1, N, Ep, d, Ep, status);
  p.out0 = S;
  p.out1 = ST;
  p.out2 = slot_init;
  p.bias = br;
  p.n_valid = E;
  if (Ep <= 128 && E % 4 == 0 && N % 4 == 0) {
    // S [N][E] and S^T [E][N] leave through TMA stores (row strides of 16-byte multiples)
    CUtensorMap mo0, mo1;
    TC_TRY(make_out_map(&mo0, S, true, E, N, 1));
    TC_TRY(make_out_map(&mo1, ST, true, N, E, 1));
    // rows split evenly over the SMs; a 192 KB ring (the main loop streams X at the rate its
    // bytes in flight allow); 8 epilogue warps, two per TMEM lane quarter, each taking half of
    // a row's experts (the epilogue of a CTA's last tile is not hidden behind a main loop)
    if (Ep == 64)
      return launch<64, false, true, false, false, EPI_ROUTER_ST, 8, 8, false, 3>(
          ma, ma, mb, mb, mo0, mo1, ma, p, st);
    return launch<128, false, true, false, false, EPI_ROUTER_ST, 6, 8, false, 3>(
        ma, ma, mb, mb, mo0, mo1, ma, p, st);
  }
  switch (Ep) {
    // the router epilogue writes S and S^T itself: the output maps are unused
    case 64:
      return launch<64, false, true, false, false, EPI_ROUTER, 8, 4>(ma, ma, mb, mb, ma, ma, ma, p, st);
    case 128:
      return launch<128, false, true, false, false, EPI_ROUTER, 6, 4>(ma, ma, mb, mb, ma, ma, ma, p, st);
    case 192:
      return launch<192, false, true, false, false, EPI_ROUTER, 5, 4>(ma, ma, mb, mb, ma, ma, ma, p, st);
    case 256:
      return launch<256, false, true, false, false, EPI_ROUTER, 4, 4>(ma, ma, mb, mb, ma, ma, ma, p, st);
  }
  return cudaErrorInvalidValue;
}

// Activation maps and Args for the expert GEMMs: a uniform batch [E][M][cols], or with `vr`
// one [1][P][cols] tensor of padded variable-row expert regions (the tile decode finds the
// expert of each 256-row tile from vr->tiles).
static cudaError_t act_map(CUtensorMap* m, const void* base, int cols, int E, int M,
                           const VarRows* vr, uint32_t box_rows) {
  return vr ? make_map(m, base, cols, vr->P, 1, box_rows) : make_map(m, base, cols, M, E, box_rows);
}

// Output map of an expert activation tensor, laid out like the inputs of act_map.
static cudaError_t act_out_map(CUtensorMap* m, const void* base, int cols, int E, int M,
                               const VarRows* vr) {
  return vr ? make_out_map(m, base, false, cols, vr->P, 1) : make_out_map(m, base, false, cols, M, E);
}

static Args row_args(int E, int M, int N, int K, int BN_tile, int* status, const VarRows* vr) {
  Args p = vr ? base_args(1, vr->P, N, K, BN_tile, status) : base_args(E, M, N, K, BN_tile, status);
  if (vr) {
    p.vm_tiles = vr->tiles;
    p.vm_count = vr->count;
    p.vm_E = E;
  }
  return p;
}

constexpr int kDuStages = 5;
constexpr int kWideStages = 4;

// Wide (256 x 512) pair tiles where the output columns fill them exactly and the K loop is
// long enough (k rows) to cover the epilogue's hand-over of the two accumulator halves:
// measured, they gain 2-5% with k >= 1024 (k >= 2048 behind the SwiGLU epilogue, which
// writes three outputs; at 1024 it only breaks even) and lose about 3% at k = 512.
// `tiles`: 0 chooses so, 1 keeps 256-column tiles, 2 takes wide tiles wherever they fit.
static bool wide_cols(int tiles, int n, int k, int k_min = 1024) {
  if (tiles == 1 || n % 512 != 0) return false;
  return tiles == 2 || k >= k_min;
}

template <int BN, bool A_MN, bool B_MN, bool B_SPLIT, bool K_SPLIT, int EPI>
static cudaError_t launch_rows(const CUtensorMap& a0, const CUtensorMap& a1, const CUtensorMap& b0,
                               const CUtensorMap& b1, const CUtensorMap& o0, const CUtensorMap& o1,
                               const CUtensorMap& o2, const Args& p, const VarRows* vr,
                               cudaStream_t st) {
  // the dU GEMM's epilogue reads A and B through L1: a 5-deep ring leaves it 32 KB more;
  // wide tiles take 48 KB per k-slice
  constexpr int ST = BN == 512 ? kWideStages : EPI == EPI_SWIGLU_BWD ? kDuStages : 6;
  if (vr)
    return launch<BN, A_MN, B_MN, B_SPLIT, K_SPLIT, EPI, ST, 8, true, 1>(a0, a1, b0, b1, o0, o1, o2,
                                                                          p, st);
  return launch<BN, A_MN, B_MN, B_SPLIT, K_SPLIT, EPI, ST, 8, true, 0>(a0, a1, b0, b1, o0, o1, o2, p,
                                                                        st);
}

cudaError_t tc_expert_up(const void* H, const void* Wg, const void* Wu, void* A, void* B, void* U,
                         int E, int M, int d, int F, int* status, cudaStream_t st,
                         const VarRows* vr, const float* gate, int tiles) {
  CUtensorMap ma, mg, mu, oa, ob, ou;
  TC_TRY(act_map(&ma, H, d, E, M, vr, BM));
  TC_TRY(make_map(&mg, Wg, F, d, E, 64));
  TC_TRY(make_map(&mu, Wu, F, d, E, 64));
  TC_TRY(act_out_map(&oa, A, F, E, M, vr));
  TC_TRY(act_out_map(&ob, B, F, E, M, vr));
  TC_TRY(act_out_map(&ou, U, F, E, M, vr));
  const bool wide = wide_cols(tiles, 2 * F, d, 2048);   // gate and up columns side by side
  Args p = row_args(E, M, F, d, wide ? 256 : 128, status, vr);
  p.out0 = A;
  p.out1 = B;
  p.out2 = U;
  p.gate = gate;
  p.ld = F;
  p.bstride = (int64_t)M * F;
  if (wide)
    return launch_rows<512, false, true, true, false, EPI_SWIGLU_FWD>(ma, ma, mg, mu, oa, ob, ou, p,
                                                                      vr, st);
  return launch_rows<256, false, true, true, false, EPI_SWIGLU_FWD>(ma, ma, mg, mu, oa, ob, ou, p,
                                                                    vr, st);
}

cudaError_t tc_expert_down(const void* U, const void* Wd, void* O, int E, int M, int d, int F,
                           int* status, cudaStream_t st, const VarRows* vr, int tiles) {
  CUtensorMap ma, mb, mo;
  TC_TRY(act_map(&ma, U, F, E, M, vr, BM));
  TC_TRY(make_map(&mb, Wd, d, F, E, 64));
  TC_TRY(act_out_map(&mo, O, d, E, M, vr));
  const bool wide = wide_cols(tiles, d, F);
  Args p = row_args(E, M, d, F, wide ? 512 : 256, status, vr);
  p.out0 = O;
  p.ld = d;
  p.bstride = (int64_t)M * d;
  if (wide)
    return launch_rows<512, false, true, false, false, EPI_STORE_BF16>(ma, ma, mb, mb, mo, mo, mo,
                                                                       p, vr, st);
  return launch_rows<256, false, true, false, false, EPI_STORE_BF16>(ma, ma, mb, mb, mo, mo, mo, p,
                                                                     vr, st);
}

cudaError_t tc_expert_dgrad_up(const void* dO, const void* Wd, const void* A, const void* B,
                               void* dA, void* dB, int E, int M, int d, int F, int* status,
                               cudaStream_t st, const VarRows* vr, const float* gate,
                               float* dgate_part, int64_t dgate_stride, int tiles) {
  CUtensorMap ma, mb, oa, ob;
  TC_TRY(act_map(&ma, dO, d, E, M, vr, BM));
  TC_TRY(make_map(&mb, Wd, d, F, E, 128));   // B[n=f][k=i] = Wd[f][i]: K-major, half per CTA
  TC_TRY(act_out_map(&oa, dA, F, E, M, vr));
  TC_TRY(act_out_map(&ob, dB, F, E, M, vr));
  // 256 x 512 pair tiles only when forced (tile policy 2), for uniform batches: the epilogue
  // reads A and B per row, and draining an accumulator half that way takes longer than the
  // few k-slices of MMAs that can cover it (measured on the bench workload: 1.10 ms against
  // 0.83 ms with 256 x 256 tiles, whose double-buffered accumulators give the epilogue a
  // whole tile of MMAs)
  const bool wide = !vr && tiles == 2 && F % 512 == 0;
  Args p = row_args(E, M, F, d, wide ? 512 : 256, status, vr);
  p.in0 = A;
  p.in1 = B;
  p.out0 = dA;
  p.out1 = dB;
  p.gate = gate;
  p.dgate_part = dgate_part;
  p.dgate_stride = dgate_stride;
  p.ld = F;
  p.bstride = (int64_t)M * F;
  if (wide)
    return launch<512, false, false, false, false, EPI_SWIGLU_BWD, kWideStages, 8, true, 0>(
        ma, ma, mb, mb, oa, ob, ob, p, st);
  return launch_rows<256, false, false, false, false, EPI_SWIGLU_BWD>(ma, ma, mb, mb, oa, ob, ob, p,
                                                                      vr, st);
}

cudaError_t tc_expert_dgrad_h(const void* dA, const void* dB, const void* Wg, const void* Wu,
                              void* dH, int E, int M, int d, int F, int* status, cudaStream_t st,
                              const VarRows* vr, int tiles) {
  CUtensorMap ma0, ma1, mb0, mb1;
  TC_TRY(act_map(&ma0, dA, F, E, M, vr, BM));
  TC_TRY(act_map(&ma1, dB, F, E, M, vr, BM));
  TC_TRY(make_map(&mb0, Wg, F, d, E, 128));  // B[n=i][k=f] = Wg[i][f]: K-major, half per CTA
  TC_TRY(make_map(&mb1, Wu, F, d, E, 128));
  CUtensorMap mo;
  TC_TRY(act_out_map(&mo, dH, d, E, M, vr));
  const bool wide = wide_cols(tiles, d, 2 * F);
  Args p = row_args(E, M, d, 2 * F, wide ? 512 : 256, status, vr);
  p.k_blocks0 = F / BK;
  p.out0 = dH;
  p.ld = d;
  p.bstride = (int64_t)M * d;
  if (wide)
    return launch_rows<512, false, false, false, true, EPI_STORE_BF16>(ma0, ma1, mb0, mb1, mo, mo,
                                                                       mo, p, vr, st);
  return launch_rows<256, false, false, false, true, EPI_STORE_BF16>(ma0, ma1, mb0, mb1, mo, mo, mo,
                                                                     p, vr, st);
}

cudaError_t tc_expert_wgrad(const void* H, const void* U, const void* dO, const void* dA,
                            const void* dB, float* dWg, float* dWu, float* dWd, int E, int M,
                            int d, int F, int* status, cudaStream_t st, const VarRows* vr,
                            int tiles) {
  // Variable rows: the K loop of expert e runs over its own padded region (count rows,
  // rounded up to the 64-row k-step, the rest of which is zero in both operands).
  // K rows per expert (variable rows: on average)
  const int rows = vr ? vr->P / (E > 0 ? E : 1) : M;
  auto wg_args = [&](int Mo, int No, int BNt) {
    Args p = base_args(E, Mo, No, vr ? vr->P : M, BNt, status);
    if (vr) {
      p.vm_tiles = vr->tiles;
      p.vm_count = vr->count;
      p.vm_E = E;
    }
    return p;
  };
  if (dWd) {
    // dWd[e] [F][d] = U[e]^T . dO[e]: A[m=f][k=t] = U[t][f] (MN-major), B[k=t][n=i] = dO[t][i]
    CUtensorMap ma, mb, mo;
    TC_TRY(act_map(&ma, U, F, E, M, vr, 64));
    TC_TRY(act_map(&mb, dO, d, E, M, vr, 64));
    TC_TRY(make_out_map(&mo, dWd, true, d, F, E));
    const bool wide = wide_cols(tiles, d, rows);
    Args p = wg_args(F, d, wide ? 512 : 256);
    p.out0 = dWd;
    p.ld = d;
    p.bstride = (int64_t)F * d;
    constexpr int EP = EPI_STORE_F32, WS = kWideStages;
    if (wide && vr)
      TC_TRY((launch<512, true, true, false, false, EP, WS, 8, true, 2>(ma, ma, mb, mb, mo, mo, mo, p,
                                                                      st)));
    else if (wide)
      TC_TRY((launch<512, true, true, false, false, EP, WS, 8, true>(ma, ma, mb, mb, mo, mo, mo, p,
                                                                   st)));
    else if (vr)
      TC_TRY((launch<256, true, true, false, false, EP, 6, 8, true, 2>(ma, ma, mb, mb, mo, mo, mo, p,
                                                                     st)));
    else
      TC_TRY((launch<256, true, true, false, false, EP, 6, 8, true>(ma, ma, mb, mb, mo, mo, mo, p,
                                                                  st)));
  }
  if (dWg) {
    // [dWg | dWu][e] [d][F] = H[e]^T . [dA | dB][e]
    CUtensorMap ma, mb0, mb1, mo0, mo1;
    TC_TRY(act_map(&ma, H, d, E, M, vr, 64));
    TC_TRY(act_map(&mb0, dA, F, E, M, vr, 64));
    TC_TRY(act_map(&mb1, dB, F, E, M, vr, 64));
    TC_TRY(make_out_map(&mo0, dWg, true, F, d, E));
    TC_TRY(make_out_map(&mo1, dWu, true, F, d, E));
    const bool wide = wide_cols(tiles, 2 * F, rows);
    Args p = wg_args(d, F, wide ? 256 : 128);
    p.out0 = dWg;
    p.out1 = dWu;
    p.ld = F;
    p.bstride = (int64_t)d * F;
    constexpr int EP = EPI_STORE_F32_SPLIT, WS = kWideStages;
    if (wide && vr)
      TC_TRY((launch<512, true, true, true, false, EP, WS, 8, true, 2>(ma, ma, mb0, mb1, mo0, mo1, mo1,
                                                                     p, st)));
    else if (wide)
      TC_TRY((launch<512, true, true, true, false, EP, WS, 8, true>(ma, ma, mb0, mb1, mo0, mo1, mo1, p,
                                                                  st)));
    else if (vr)
      TC_TRY((launch<256, true, true, true, false, EP, 6, 8, true, 2>(ma, ma, mb0, mb1, mo0, mo1, mo1,
                                                                    p, st)));
    else
      TC_TRY((launch<256, true, true, true, false, EP, 6, 8, true>(ma, ma, mb0, mb1, mo0, mo1, mo1, p,
                                                                 st)));
  }
  return cudaSuccess;
}

cudaError_t tc_router_dgrad(const void* dZb, const void* Wr_pad, void* dXr, int N, int d, int Ep,
                            int* status, cudaStream_t st) {
  if (N == 0) return cudaSuccess;
  // dXr [N][d] = (dZ_hi + dZ_lo) [N][Ep] . Wr^T as one K loop over both planes;
  // B[n=i][k=e] = Wr_pad[i][e] is K-major
  const bf16* hi = static_cast<const bf16*>(dZb);
  CUtensorMap ma0, ma1, mb;
  TC_TRY(make_map(&ma0, hi, Ep, N, 1, BM));
  TC_TRY(make_map(&ma1, hi + (size_t)N * Ep, Ep, N, 1, BM));
  TC_TRY(make_map(&mb, Wr_pad, Ep, d, 1, 256));
  CUtensorMap mo;
  TC_TRY(make_out_map(&mo, dXr, false, d, N, 1));
  Args p = base_args(1, N, d, 2 * Ep, 256, status);
  p.k_blocks0 = Ep / BK;
  p.out0 = dXr;
  p.ld = d;
  p.bstride = 0;
  return launch<256, false, false, false, true, EPI_STORE_BF16, 4>(ma0, ma1, mb, mb, mo, mo, mo, p,
                                                                   st);
}

cudaError_t tc_router_wgrad(const void* X, const void* dZb, float* part, int N, int d, int Ep,
                            int splits, int* status, cudaStream_t st) {
  if (N == 0) return cudaSuccess;
  // part[h][s] [d][Ep] = X_s^T . dZ_h,s over the s-th block of N/splits tokens (split K as the
  // batch), h = hi / lo plane of dZ (the two column halves of each tile)
  const int rows = N / splits;
  const bf16* hi = static_cast<const bf16*>(dZb);
  CUtensorMap ma, mb0, mb1;
  TC_TRY(make_map(&ma, X, d, rows, splits, 64));
  TC_TRY(make_map(&mb0, hi, Ep, rows, splits, 64));
  TC_TRY(make_map(&mb1, hi + (size_t)N * Ep, Ep, rows, splits, 64));
  CUtensorMap mo0, mo1;
  TC_TRY(make_out_map(&mo0, part, true, Ep, d, splits));
  TC_TRY(make_out_map(&mo1, part + (size_t)splits * d * Ep, true, Ep, d, splits));
  const int BNt = Ep > 64 ? 256 : 128;
  Args p = base_args(splits, d, Ep, rows, BNt / 2, status);
  p.out0 = part;
  p.out1 = part + (size_t)splits * d * Ep;
  p.ld = Ep;
  p.bstride = (int64_t)d * Ep;
  if (BNt == 128)
    return launch<128, true, true, true, false, EPI_STORE_F32_SPLIT, 6>(ma, ma, mb0, mb1, mo0, mo1, mo1,
                                                                        p, st);
  return launch<256, true, true, true, false, EPI_STORE_F32_SPLIT, 4>(ma, ma, mb0, mb1, mo0, mo1, mo1,
                                                                      p, st);
}

cudaError_t tc_wait_probe(int* status, unsigned long long limit_ns, cudaStream_t st) {
  wait_probe_kernel<<<1, 32, 0, st>>>(status, limit_ns);
  return cudaGetLastError();
}

}  // namespace ecmoe
