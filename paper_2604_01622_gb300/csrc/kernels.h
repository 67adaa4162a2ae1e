// Internal launchers of the EC-MoE library. Not part of the C ABI.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>
#include <cuda_bf16.h>

namespace ecmoe {

// ---------------------------------------------------------------- router + selection
// Row softmax of fp32 logits Z [N][E] (+ br) -> S [N][E] and S^T [E][N]; sets the slot map
// slot [N][E] to -1 (the state launch_topk expects).
cudaError_t launch_softmax_rows(const float* Z, const float* br, float* S, float* ST, int* slot,
                                int N, int E, cudaStream_t st);
// Transpose scores [E][N] -> [N][E] (used when the caller supplies S); sets slot [N][E] to -1.
cudaError_t launch_transpose_scores(const float* ST, float* S, int* slot, int N, int E,
                                    cudaStream_t st);
// Expert-choice top-k per (expert, group) over S^T [E][N]; writes idx/gate [E][M] and, for
// the selected pairs only, the token->slot map slot [N][E] (= m). The other entries of slot
// must already hold -1.
cudaError_t launch_topk(const float* ST, int N, int E, int G, const int* group_off, const int* k_g,
                        const int* k_off, int M, int max_group, int* idx, float* gate, int* slot,
                        cudaStream_t st);

// Capacity update from device memory (one CTA): if 0 <= k_new[g] <= L_g for every group and
// sum k_new == M, writes k_g [G] and its prefix sums k_off [G+1]; otherwise leaves both and
// records DEV_BAD_CAPACITY in the status word.
cudaError_t launch_set_capacity(const int* k_new, const int* group_off, int G, int M, int* k_g,
                                int* k_off, int* status, cudaStream_t st);

// ---------------------------------------------------------------- token-choice routing
// Row top-k of S [N][E] (k <= 32, E <= 512), per-expert counts capped at cap (cap < 0:
// dropless), padded expert regions (tiles[e] in 256-row blocks), row->token map (-1 in
// padding), row gates, slot map [N][E] (absolute row or -1) and kept flags [N][k].
// Token-choice routing of the scores S [N][E] (k <= 32, E <= 256; cap < 0: no cap):
// choice/tgate/kept [N][k] (experts best first, normalised gates, kept flags), Z [N] (sum of
// the k chosen scores), count [E+1] (kept rows per expert; count[E] = padded rows in use),
// tiles [E+1] (cumulative 256-row blocks), row_token/row_gate [P] per padded row (-1 / 0 in
// padding), slot [N][E] absolute padded row of each kept pair, else -1.
// scratch: tc_route_scratch_ints(N, E) ints. Five kernels (and a memset of slot).
cudaError_t launch_tc_route(const float* S, int N, int E, int k, int cap, int* choice,
                            float* tgate, float* Z, int* count, int* tiles, int* row_token,
                            float* row_gate, int* slot, int* kept, int* scratch,
                            cudaStream_t st);
int64_t tc_route_scratch_ints(int N, int E);
// Router gradient of token choice: dZ [N][E] (and optionally the bf16 hi/lo planes
// dZb [2][N][Ep]) from the per-row gate gradients row_dgate [P].
cudaError_t launch_tc_softmax_bwd(const float* S, const int* choice, const float* tgate,
                                  const float* Z, const int* slot, const float* row_dgate,
                                  float* dZ, __nv_bfloat16* dZb, int N, int E, int Ep, int k,
                                  cudaStream_t st);

// ---------------------------------------------------------------- data movement
// Token-major form of the gather: for each token t, X row t is copied to row e*M + slot[t][e]
// of H for every expert e with slot[t][e] >= 0 (M = 0: slot holds absolute rows).
template <typename T>
cudaError_t launch_scatter_rows(const T* X, const int* slot, T* H, int N, int E, int M, int d,
                                cudaStream_t st);
// Zeros the unused (padding) rows of variable-row expert regions (count [E], tiles [E+1] in
// 256-row blocks, device arrays).
template <typename T>
cudaError_t launch_zero_pad_rows(const int* count, const int* tiles, T* H, int E, int d,
                                 cudaStream_t st);
// Y_t = R_t + R2_t (each if given) + sum over the experts that chose t of gate * O row
// (gate NULL: 1, for O rows already scaled by their gates).
template <typename T>
cudaError_t launch_combine(const T* O, const float* gate, const int* slot, const T* R, const T* R2,
                           T* Y, int N, int E, int M, int d, cudaStream_t st);
// dO row r = gate[r] dY row idx[r], dgate[r] = <dY row idx[r], O row r> (zero rows where
// idx[r] < 0), for the P rows (fp32 path).
template <typename T>
cudaError_t launch_bwd_gather_scale(const T* dY, const T* O, const int* idx, const float* gate,
                                    T* dO, float* dgate, int64_t P, int d, cudaStream_t st);
// Router softmax Jacobian: dS[t][e] = dgate of the pair (t chosen by e) else 0,
// dZ = S (dS - <dS, S>_row). dgate [E*M] summed beforehand; writes dZ [N][E] and, with dZb,
// the bf16 hi/lo planes [2][N][Ep] (any E <= 512).
cudaError_t launch_softmax_bwd(const float* S, const int* slot, const float* dgate, float* dZ,
                               __nv_bfloat16* dZb, int N, int E, int Ep, int M, cudaStream_t st);
// The same, fused with the sum of the gate-gradient partials dg_part [parts][E*M] (in part
// order) and, with dbr, with the router bias gradient dbr[e] = sum_t dZ[t][e] (per-CTA
// column sums in scratch, then summed in a fixed order: deterministic). dZ and dZb are each
// optional. For E % 4 == 0, E <= 128 and E*M < 2^31 (router_bwd_fused); one kernel, two
// with dbr. scratch: router_bwd_scratch_floats(N, E) floats.
bool router_bwd_fused(int E, int64_t P);
int64_t router_bwd_scratch_floats(int N, int E);
cudaError_t launch_router_softmax_bwd(const float* S, const int* slot, const float* dg_part,
                                      int parts, float* dZ, __nv_bfloat16* dZb, float* dbr,
                                      float* scratch, int N, int E, int Ep, int M,
                                      cudaStream_t st);
cudaError_t launch_reduce_partials(const float* part, float* out, int rows, int cols, int ld,
                                   int splits, cudaStream_t st);
// dX_t = dXr_t + R_t + R2_t (each if given) + sum of the token's dH rows, summed in fp32;
// dXr (the router's part of the input gradient) is in the layer's dtype.
template <typename T>
cudaError_t launch_dx_combine(const T* dH, const int* slot, const T* dXr, const T* R,
                              const T* R2, T* dX, int N, int E, int M, int d, cudaStream_t st);
// out[e] = sum over the N rows of Z [N][E]; scratch: colsum_scratch_floats(N, E) floats.
// Two kernels.
cudaError_t launch_colsum(const float* Z, float* out, int N, int E, float* scratch,
                          cudaStream_t st);
int64_t colsum_scratch_floats(int N, int E);
template <typename T>
cudaError_t launch_swiglu_fwd_ew(const float* Ag, const float* Bu, T* A, T* B, T* U, int64_t n,
                                 cudaStream_t st);
template <typename T>
cudaError_t launch_swiglu_bwd_ew(const float* dU, const T* A, const T* B, T* dA, T* dB,
                                 int64_t n, cudaStream_t st);
template <typename T>
cudaError_t launch_convert(const float* in, T* out, int64_t n, cudaStream_t st);
cudaError_t launch_reduce_splits(const float* part, float* out, int64_t n, int splits,
                                 cudaStream_t st);

// ---------------------------------------------------------------- fp32 SIMT GEMM
// C[b] (+)= A[b] . B[b] with A logical [M][K], B logical [K][N], C [M][N] fp32 (unit column
// stride). Element strides per operand; TA/TB are float or bf16.
struct SimtGemmArgs {
  const void* A; int64_t a_bs, a_ms, a_ks;
  const void* B; int64_t b_bs, b_ks, b_ns;
  float* C; int64_t c_bs, c_ms;
  int M, N, K, batch;
  int splits;                 // >1: split s writes C + s * c_split (beta ignored)
  int64_t c_split;
  float beta;                 // C = A.B + beta*C (splits == 1 only)
};
enum class EType { F32, BF16 };
cudaError_t launch_simt_gemm(const SimtGemmArgs& a, EType ta, EType tb, cudaStream_t st);

}  // namespace ecmoe
