// Tensor-core (tcgen05 + TMEM + TMA) GEMMs of the bf16 EC-MoE path. Internal.
//
// Expert choice gives every expert the same row count M (arXiv 2604.01622, Sec. 2.2:
// each expert processes exactly its capacity), so every expert GEMM is a uniform batch
// over E experts with 3-D TMA tensor maps [E][rows][cols].
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

namespace ecmoe {

// Variable rows per expert (token-choice routing): expert e owns the padded rows
// [256*tiles[e], 256*tiles[e+1]) of [P][cols] activation tensors, the first count[e] of them
// real. tiles [E+1] and count [E] are device arrays; P bounds the padded rows. The GEMMs
// write the unused rows of each region as zeros.
struct VarRows {
  const int* tiles;
  const int* count;
  int P;
};

// Tile shapes of the expert GEMMs (the `tiles` argument below): 0 chooses per GEMM (256 x 512
// pair tiles where the output columns fill them and the K loop is long enough to hide the
// hand-over of their two accumulator halves, else 256 x 256), 1 always 256 x 256, 2 wide
// tiles wherever the columns fill them. The dU GEMM takes 256 x 512 tiles only under
// policy 2 (and never with variable rows): its epilogue reads A and B per row and cannot
// drain an accumulator half within the MMAs that cover it.

// Router: Z = X.Wr (+br), S = row softmax over the E experts, written as S [N][E] and
// S^T [E][N]. X [N][d] bf16, Wr [d][E] bf16. Wr_pad: device scratch of d*round_up(E,64)
// bf16 (zero-padded copy of Wr made on the stream when E is not a multiple of 64,
// router_needs_pad; otherwise Wr itself is read and Wr_pad is untouched). slot_init
// (nullable): an int [N][E] map set to -1 beside S (the expert-choice slot map before
// selection).
bool router_needs_pad(int E);
cudaError_t tc_router_softmax(const void* X, const void* Wr, void* Wr_pad, const float* br,
                              float* S, float* ST, int* slot_init, int N, int d, int E,
                              int* status, cudaStream_t st);

// [A | B] = H.[Wg | Wu] per expert; U = g * silu(A) * B with g the row's gate (gate [E*M]
// or, with vr, [P]; NULL: g = 1). H [E][M][d]; Wg, Wu [E][d][F]; A, B, U [E][M][F] bf16.
cudaError_t tc_expert_up(const void* H, const void* Wg, const void* Wu, void* A, void* B, void* U,
                         int E, int M, int d, int F, int* status, cudaStream_t st,
                         const VarRows* vr = nullptr, const float* gate = nullptr,
                         int tiles = 0);

// O = U.Wd per expert. U [E][M][F]; Wd [E][F][d]; O [E][M][d] bf16.
cudaError_t tc_expert_down(const void* U, const void* Wd, void* O, int E, int M, int d, int F,
                           int* status, cudaStream_t st, const VarRows* vr = nullptr,
                           int tiles = 0);

// dU' = dO.Wd^T per expert, dU = g dU' (g the row's gate as in tc_expert_up, NULL: 1), then
// dA = dU * B * silu'(A), dB = dU * silu(A) (bf16 out). With dgate_part, also the row's
// gate gradient <dU', silu(A) * B> as ceil(F/256) partial sums (partial j over the columns
// [256 j, 256 j + 256)), partial j of row r at dgate_part[j * dgate_stride + r].
cudaError_t tc_expert_dgrad_up(const void* dO, const void* Wd, const void* A, const void* B,
                               void* dA, void* dB, int E, int M, int d, int F, int* status,
                               cudaStream_t st, const VarRows* vr = nullptr,
                               const float* gate = nullptr, float* dgate_part = nullptr,
                               int64_t dgate_stride = 0, int tiles = 0);

// dH = dA.Wg^T + dB.Wu^T per expert (one K loop over both halves). dH [E][M][d] bf16.
cudaError_t tc_expert_dgrad_h(const void* dA, const void* dB, const void* Wg, const void* Wu,
                              void* dH, int E, int M, int d, int F, int* status, cudaStream_t st,
                              const VarRows* vr = nullptr, int tiles = 0);

// Weight gradients per expert, fp32: dWd = U^T.dO, dWg = H^T.dA, dWu = H^T.dB (dWd NULL:
// only dWg and dWu; dWg NULL: only dWd). With `vr`, each expert sums over its own rows (an
// expert with none gets zeros).
cudaError_t tc_expert_wgrad(const void* H, const void* U, const void* dO, const void* dA,
                            const void* dB, float* dWg, float* dWu, float* dWd, int E, int M,
                            int d, int F, int* status, cudaStream_t st,
                            const VarRows* vr = nullptr, int tiles = 0);

// Router backward on the tensor cores. dZb [2][N][Ep] bf16: hi and lo planes of the
// zero-padded softmax gradient (dZ ~ hi + lo); Wr_pad [d][Ep] bf16 (the padded router
// weights of the forward pass). dXr [N][d] bf16 = dZ . Wr^T (summed in fp32, rounded once).
cudaError_t tc_router_dgrad(const void* dZb, const void* Wr_pad, void* dXr, int N, int d, int Ep,
                            int* status, cudaStream_t st);
// part [2][splits][d][Ep] fp32: X^T . dZ_plane over `splits` equal blocks of tokens
// (N % splits == 0); dWr is the sum of all 2*splits partials.
cudaError_t tc_router_wgrad(const void* X, const void* dZb, float* part, int N, int d, int Ep,
                            int splits, int* status, cudaStream_t st);

// Launch a kernel that waits, with the given limit, on an mbarrier nothing completes, so
// the bounded-wait path (status word, early return) can be exercised without a hang.
cudaError_t tc_wait_probe(int* status, unsigned long long limit_ns, cudaStream_t st);

}  // namespace ecmoe
