// C ABI of the EC-MoE layer: argument checks, workspace layout and the launch sequence of
// the forward and backward passes (arXiv 2604.01622, Sec. 2.2; per-sequence capacity,
// Sec. 4.2; one selection pool per sequence, Sec. 5.2).
#include <string>
#include <vector>
#include <cstdio>
#include <cmath>
#include <algorithm>
#include <cstring>
#include <cstdarg>

#include <nvtx3/nvToolsExt.h>

#include "../../include/ecmoe.h"
#include "common.cuh"
#include "kernels.h"
#include "gemm_tc.h"

using namespace ecmoe;

struct ec_ctx {
  int N = 0, d = 0, E = 0, F = 0, G = 0, dtype = 0;
  int M_cap = 0, M = 0, max_group = 0;
  std::vector<int32_t> group_off, k_g, k_off;
  char* ws = nullptr;
  size_t ws_bytes = 0;
  // workspace offsets (bytes)
  size_t o_status, o_goff, o_kg, o_koff, o_ST, o_S, o_idx, o_gate, o_slot, o_H, o_A, o_B, o_U,
      o_O, o_dO, o_dA, o_dB, o_dgate, o_dZ, o_dZb, o_wrpad, o_f32a, o_f32b, o_dXr, o_part, total;
  int wr_splits = 1;   // split-K factor of dWr = X^T dZ
  int dg_parts = 1;    // partial sums per gate gradient (tensor-core dU epilogue)
  size_t o_dgsum = 0;  // the gate gradients summed over their partials
  size_t o_colsum = 0; // partial column sums of dZ (router bias gradient)
  int Ep = 64;         // experts rounded up to 64 (tensor-core router operands)
  // per-kernel event timing (off by default) and kernel launch counter
  bool prof = false;
  std::vector<cudaEvent_t> ev;
  std::vector<const char*> ev_name;
  int ev_n = 0;
  bool nvtx_open = false;   // an NVTX range named after the current phase is open
  int64_t launches = 0;
  // state saved by the forward pass
  bool residual = false;   // Y = X + EC(X), dX = dY + EC input gradient
  int Fs = 0;              // shared experts: total hidden width (0 = none)
  size_t o_Ash = 0, o_Bsh = 0, o_Ush = 0, o_Osh = 0, o_dAsh = 0, o_dBsh = 0, o_shpart = 0;
  const void *Wgs = nullptr, *Wus = nullptr, *Wds = nullptr;
  float *dWgs = nullptr, *dWus = nullptr, *dWds = nullptr;
  bool have_fwd = false;
  const void *X = nullptr, *Wr = nullptr, *Wg = nullptr, *Wu = nullptr, *Wd = nullptr;
  const float* br = nullptr;
  // token choice (k > 0): k experts per token, per-expert cap (< 0: none), padded rows
  int tc_k = 0, tc_cap = -1;
  int64_t P_tc = 0;
  int tiles = EC_TILES_AUTO;   // expert-GEMM tile policy (ec_ctx_set_tiles)
  size_t o_choice = 0, o_tgate = 0, o_Zs = 0, o_count = 0, o_tiles = 0, o_kept = 0, o_tcscr = 0;
  std::string err;
  ec_status err_status = EC_OK;   // status of the last failed call (ec_get_last_error)
};

namespace {

ec_status fail(ec_ctx* c, ec_status s, const char* fmt, ...) {
  if (c) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    c->err = buf;
    c->err_status = s;
  }
  return s;
}

ec_status cuda_fail(ec_ctx* c, cudaError_t e, const char* where) {
  return fail(c, EC_ERR_CUDA, "%s: %s", where, cudaGetErrorString(e));
}

#define EC_CUDA(call, where)                         \
  do {                                               \
    cudaError_t _e = (call);                         \
    if (_e != cudaSuccess) return cuda_fail(c, _e, where); \
  } while (0)

// Phase marker: with profiling on, records an event named after the kernel about to be
// launched (or "end" after the last one) on the call's stream, and opens an NVTX range of
// the same name (closed at the next marker) for profilers that filter by range.
void mark(ec_ctx* c, const char* name, cudaStream_t st) {
  if (!c->prof) return;
  if (c->nvtx_open) nvtxRangePop();
  c->nvtx_open = std::strcmp(name, "end") != 0;
  if (c->nvtx_open) nvtxRangePushA(name);
  if (c->ev_n == (int)c->ev.size()) {
    cudaEvent_t e;
    if (cudaEventCreate(&e) != cudaSuccess) return;
    c->ev.push_back(e);
    c->ev_name.push_back(nullptr);
  }
  cudaEventRecord(c->ev[c->ev_n], st);
  c->ev_name[c->ev_n] = name;
  ++c->ev_n;
}

// Launch `nk` kernels through `call` as one named phase.
#define EC_KERNEL(name, nk, call)            \
  do {                                       \
    mark(c, name, st);                       \
    c->launches += (nk);                     \
    EC_CUDA(call, name);                     \
  } while (0)

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

size_t up256(size_t x) { return (x + 255) & ~size_t(255); }

template <typename P>
P* at(ec_ctx* c, size_t off) { return reinterpret_cast<P*>(c->ws + off); }

size_t esize(const ec_ctx* c) { return c->dtype == EC_BF16 ? 2 : 4; }

bool use_tc(const ec_ctx* c) { return c->dtype == EC_BF16; }

// SM pairs of the current device (the tensor-core GEMMs run one 2-CTA cluster per pair)
int sm_pairs(const ec_ctx*) {
  static int pairs = 0;
  if (!pairs) {
    int dev = 0, n = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    pairs = n > 1 ? n / 2 : 1;
  }
  return pairs;
}

void layout(ec_ctx* c) {
  const size_t N = c->N, d = c->d, E = c->E, F = c->F, M = c->M_cap, G = c->G, es = esize(c);
  // expert rows: E x M for expert choice; token choice keeps each expert's rows in a region
  // padded to 256 rows, at most N k + 255 E rows in all
  const size_t P = c->tc_k ? (size_t)c->P_tc : E * M;
  size_t o = 0;
  auto take = [&](size_t bytes) { size_t r = o; o = up256(o + bytes); return r; };
  c->o_status = take(256);
  const size_t NK = c->tc_k ? N * c->tc_k : 0;
  c->o_choice = take(NK * 4);
  c->o_tgate = take(NK * 4);
  c->o_kept = take(NK * 4);
  c->o_Zs = take(c->tc_k ? N * 4 : 0);
  c->o_count = take(c->tc_k ? (E + 1) * 4 : 0);
  c->o_tiles = take(c->tc_k ? (E + 1) * 4 : 0);
  c->o_tcscr = take(c->tc_k ? (size_t)tc_route_scratch_ints((int)N, (int)E) * 4 : 0);
  c->o_goff = take((G + 1) * 4);
  c->o_kg = take(G * 4);
  c->o_koff = take((G + 1) * 4);
  c->o_ST = take(E * N * 4);
  c->o_S = take(N * E * 4);
  c->o_idx = take(P * 4);
  c->o_gate = take(P * 4);
  c->o_slot = take(N * E * 4);
  c->o_H = take(P * d * es);
  c->o_A = take(P * F * es);
  c->o_B = take(P * F * es);
  c->o_U = take(P * F * es);
  c->o_O = take(P * d * es);   // also holds dH in the backward pass
  c->o_dO = take(P * d * es);
  c->o_dA = take(P * F * es);
  c->o_dB = take(P * F * es);
  // bf16: the dU GEMM's epilogue leaves one partial gate gradient per 256 columns of d_ff
  c->dg_parts = use_tc(c) ? (c->F + 255) / 256 : 1;
  c->o_dgate = take(c->dg_parts * P * 4);
  c->o_dgsum = use_tc(c) ? take(P * 4) : c->o_dgate;
  c->o_dZ = take(N * E * 4);
  c->Ep = (c->E + 63) / 64 * 64;
  c->o_dZb = take(use_tc(c) ? 2 * N * c->Ep * 2 : 0);
  c->o_wrpad = take(d * c->Ep * 2);
  // shared experts: one SwiGLU FFN of width Fs over all N tokens (Osh also holds its dH)
  const size_t Fs = c->Fs;
  c->o_Ash = take(N * Fs * es);
  c->o_Bsh = take(N * Fs * es);
  c->o_Ush = take(N * Fs * es);
  c->o_Osh = take(Fs ? N * d * es : 0);
  c->o_dAsh = take(N * Fs * es);
  c->o_dBsh = take(N * Fs * es);
  // the shared FFN's dWd as two split-K halves (tensor cores; see ffn_backward)
  c->o_shpart = take(use_tc(c) && Fs ? 2 * Fs * d * 4 : 0);
  // fp32 scratch: SIMT GEMM outputs (fp32 path) and router logits / router dX part
  const size_t big = std::max(std::max(P * F, P * d), std::max(N * Fs, Fs ? N * d : 0));
  const size_t f32n = use_tc(c) ? N * E : std::max(big, N * E);
  c->o_f32a = take(f32n * 4);
  c->o_f32b = take((use_tc(c) ? 0 : big) * 4);
  c->o_dXr = take(N * d * es);   // the router's part of dX, in the layer dtype
  c->o_colsum = take((size_t)std::max(colsum_scratch_floats((int)N, (int)E),
                                       router_bwd_scratch_floats((int)N, (int)E)) * 4);
  // split-K partials of dWr = X^T dZ (tensor cores: equal token blocks, so N % splits == 0)
  if (use_tc(c)) {
    c->wr_splits = 1;
    for (int s = 16; s > 1; s >>= 1)
      if (N % s == 0 && N / s >= 256) { c->wr_splits = s; break; }
    c->o_part = take((size_t)2 * c->wr_splits * d * c->Ep * 4);
  } else {
    c->wr_splits = (int)std::max<size_t>(1, std::min<size_t>(64, N / 512));
    c->o_part = take((size_t)c->wr_splits * d * E * 4);
  }
  c->total = o;
}

ec_status check_ready(ec_ctx* c) {
  if (!c) return EC_ERR_INVALID_ARG;
  if (!c->ws) return fail(c, EC_ERR_WORKSPACE, "no workspace attached (ec_ctx_set_workspace)");
  return EC_OK;
}

ec_status set_groups(ec_ctx* c, const int32_t* group_off, const int32_t* k_g, bool creating) {
  if (!group_off && creating) return fail(c, EC_ERR_INVALID_ARG, "group_off is NULL");
  if (!k_g) return fail(c, EC_ERR_INVALID_ARG, "k_g is NULL");
  const int G = c->G;
  if (creating) {
    if (group_off[0] != 0 || group_off[G] != c->N)
      return fail(c, EC_ERR_SHAPE, "group_off must start at 0 and end at N=%d", c->N);
    for (int g = 0; g < G; ++g)
      if (group_off[g + 1] < group_off[g])
        return fail(c, EC_ERR_SHAPE, "group_off must be non-decreasing (group %d)", g);
  }
  const int32_t* off = creating ? group_off : c->group_off.data();
  int64_t M = 0;
  int maxL = 0;
  for (int g = 0; g < G; ++g) {
    const int L = off[g + 1] - off[g];
    if (k_g[g] < 0 || k_g[g] > L)
      return fail(c, EC_ERR_SHAPE, "k_g[%d]=%d outside [0, %d]", g, k_g[g], L);
    M += k_g[g];
    maxL = std::max(maxL, L);
  }
  if (M > (int64_t)1 << 30) return fail(c, EC_ERR_UNSUPPORTED, "sum(k_g) too large");
  if (!creating && M > c->M_cap)
    return fail(c, EC_ERR_SHAPE, "sum(k_g)=%lld exceeds the context's capacity %d", (long long)M,
                c->M_cap);
  if (creating) {
    c->group_off.assign(group_off, group_off + G + 1);
    c->M_cap = (int)M;
    c->max_group = maxL;
  }
  c->k_g.assign(k_g, k_g + G);
  c->k_off.assign(G + 1, 0);
  for (int g = 0; g < G; ++g) c->k_off[g + 1] = c->k_off[g] + k_g[g];
  c->M = (int)M;
  c->have_fwd = false;
  return EC_OK;
}

ec_status upload_groups(ec_ctx* c) {
  if (!c->ws) return EC_OK;
  EC_CUDA(cudaMemcpy(at<int>(c, c->o_goff), c->group_off.data(), (c->G + 1) * 4,
                     cudaMemcpyHostToDevice), "upload group_off");
  EC_CUDA(cudaMemcpy(at<int>(c, c->o_kg), c->k_g.data(), c->G * 4, cudaMemcpyHostToDevice),
          "upload k_g");
  EC_CUDA(cudaMemcpy(at<int>(c, c->o_koff), c->k_off.data(), (c->G + 1) * 4,
                     cudaMemcpyHostToDevice), "upload k_off");
  return EC_OK;
}

// ---------------------------------------------------------------- SIMT GEMM helpers
// Batched over experts: C[e] = A[e] . B[e] (+ beta C[e]).
SimtGemmArgs sg(const void* A, int64_t a_bs, int64_t a_ms, int64_t a_ks, const void* B,
                int64_t b_bs, int64_t b_ks, int64_t b_ns, float* C, int64_t c_bs, int64_t c_ms,
                int M, int N, int K, int batch, float beta = 0.f) {
  SimtGemmArgs a;
  a.A = A; a.a_bs = a_bs; a.a_ms = a_ms; a.a_ks = a_ks;
  a.B = B; a.b_bs = b_bs; a.b_ks = b_ks; a.b_ns = b_ns;
  a.C = C; a.c_bs = c_bs; a.c_ms = c_ms;
  a.M = M; a.N = N; a.K = K; a.batch = batch; a.splits = 1; a.c_split = 0; a.beta = beta;
  return a;
}

EType et(const ec_ctx* c) { return c->dtype == EC_BF16 ? EType::BF16 : EType::F32; }

// The router weights as the tensor cores read them, [d][Ep] bf16: Wr itself when E is a
// multiple of 64, else the zero-padded copy the forward pass made.
const void* router_b(ec_ctx* c) {
  return router_needs_pad(c->E) ? at<void>(c, c->o_wrpad) : c->Wr;
}

// ---------------------------------------------------------------- router + selection
template <typename T>
ec_status run_route(ec_ctx* c, const void* X, const void* Wr, const float* br, const float* S_in,
                    cudaStream_t st) {
  const int N = c->N, E = c->E, d = c->d;
  float* ST = at<float>(c, c->o_ST);
  float* S = at<float>(c, c->o_S);
  const int nz = N > 0;
  // each of the three kernels that write S token-major also sets the slot map to -1, so the
  // top-k kernel writes only the selected entries
  int* slot = at<int>(c, c->o_slot);
  if (S_in) {
    EC_CUDA(cudaMemcpyAsync(ST, S_in, (size_t)E * N * 4, cudaMemcpyDeviceToDevice, st), "copy S_in");
    EC_KERNEL("transpose_scores", nz, launch_transpose_scores(ST, S, slot, N, E, st));
  } else if (use_tc(c)) {
    EC_KERNEL("router_gemm_softmax", (router_needs_pad(E) ? 2 : 1) * nz,
              tc_router_softmax(X, Wr, at<void>(c, c->o_wrpad), br, S, ST, slot, N, d, E,
                                at<int>(c, c->o_status), st));
  } else {
    float* Z = at<float>(c, c->o_f32a);
    EC_KERNEL("router_gemm", nz,
              launch_simt_gemm(sg(X, 0, d, 1, Wr, 0, E, 1, Z, 0, E, N, E, d, 1), et(c), et(c), st));
    EC_KERNEL("router_softmax", nz, launch_softmax_rows(Z, br, S, ST, slot, N, E, st));
  }
  EC_KERNEL("topk", 1,
            launch_topk(ST, N, E, c->G, at<int>(c, c->o_goff), at<int>(c, c->o_kg),
                        at<int>(c, c->o_koff), c->M, c->max_group, at<int>(c, c->o_idx),
                        at<float>(c, c->o_gate), slot, st));
  return EC_OK;
}

ec_status copy_out(ec_ctx* c, int32_t* idx, float* gate, float* S_out, cudaStream_t st) {
  const size_t P = (size_t)c->E * c->M;
  if (idx && P)
    EC_CUDA(cudaMemcpyAsync(idx, at<int>(c, c->o_idx), P * 4, cudaMemcpyDeviceToDevice, st), "idx out");
  if (gate && P)
    EC_CUDA(cudaMemcpyAsync(gate, at<float>(c, c->o_gate), P * 4, cudaMemcpyDeviceToDevice, st),
            "gate out");
  if (S_out)
    EC_CUDA(cudaMemcpyAsync(S_out, at<float>(c, c->o_ST), (size_t)c->E * c->N * 4,
                            cudaMemcpyDeviceToDevice, st), "S out");
  return EC_OK;
}

// ---------------------------------------------------------------- SwiGLU FFN building blocks
// One batch of E SwiGLU FFNs over M rows each: [A | B] = H.[Wg | Wu], U = silu(A) * B,
// O = U.Wd. Used for the routed experts (E experts, M selected rows each) and for the
// shared experts (one FFN of the concatenated width over all N tokens).
struct FfnNames {
  const char *up, *down, *dgrad_up, *dgrad_h, *wgrad;
};
const FfnNames kRouted = {"gemm_gate_up_swiglu", "gemm_down", "gemm_dgrad_up_swiglu",
                          "gemm_dgrad_h", "gemm_wgrad"};
const FfnNames kShared = {"shared_gate_up_swiglu", "shared_down", "shared_dgrad_up_swiglu",
                          "shared_dgrad_h", "shared_wgrad"};

// On the tensor-core path `gate` (per row, or NULL) scales U, so O rows come out gated.
template <typename T>
ec_status ffn_forward(ec_ctx* c, const FfnNames& nm, const T* H, const void* Wg, const void* Wu,
                      const void* Wd, T* A, T* B, T* U, T* O, int E, int M, int F,
                      cudaStream_t st, const float* gate = nullptr) {
  const int d = c->d;
  const int64_t P = (int64_t)E * M;
  if (P == 0) return EC_OK;
  int* status = at<int>(c, c->o_status);
  if (use_tc(c)) {
    EC_KERNEL(nm.up, 1,
              tc_expert_up(H, Wg, Wu, A, B, U, E, M, d, F, status, st, nullptr, gate, c->tiles));
    EC_KERNEL(nm.down, 1, tc_expert_down(U, Wd, O, E, M, d, F, status, st, nullptr, c->tiles));
  } else {
    float* Ag = at<float>(c, c->o_f32a);
    float* Bu = at<float>(c, c->o_f32b);
    const int64_t hs = (int64_t)M * d, ws = (int64_t)d * F, os = (int64_t)M * F;
    EC_KERNEL(nm.up, 1,
              launch_simt_gemm(sg(H, hs, d, 1, Wg, ws, F, 1, Ag, os, F, M, F, d, E), et(c), et(c), st));
    EC_KERNEL(nm.up, 1,
              launch_simt_gemm(sg(H, hs, d, 1, Wu, ws, F, 1, Bu, os, F, M, F, d, E), et(c), et(c), st));
    EC_KERNEL("swiglu", 1, launch_swiglu_fwd_ew<T>(Ag, Bu, A, B, U, P * F, st));
    float* O32 = at<float>(c, c->o_f32a);
    EC_KERNEL(nm.down, 1,
              launch_simt_gemm(sg(U, os, F, 1, Wd, (int64_t)F * d, d, 1, O32, hs, d, M, d, F, E),
                               et(c), et(c), st));
    EC_KERNEL("convert_o", 1, launch_convert<T>(O32, O, P * d, st));
  }
  return EC_OK;
}

// Backward of ffn_forward given dO: dU = dO.Wd^T, dA = dU*B*silu'(A), dB = dU*silu(A),
// dH = dA.Wg^T + dB.Wu^T, dWd = U^T.dO, dWg = H^T.dA, dWu = H^T.dB (fp32, overwritten).
// On the tensor-core path with `gate`, dO holds the ungated rows dY[idx] and U the gated
// ones (as ffn_forward wrote them): dU = gate * dO.Wd^T, dWd = U^T.dO, and the gate
// gradients <dO.Wd^T, silu(A) B> land in dgate_part (c->dg_parts partials, stride E*M).
// dwd_split: optional scratch of 2*F*d floats for the single-FFN case (E = 1, the shared
// experts), whose dWd = U^T.dO has few output tiles for the whole GPU and a K loop over all
// M rows: the rows are split into two halves computed as two batch entries at once and
// summed in order afterwards.
template <typename T>
ec_status ffn_backward(ec_ctx* c, const FfnNames& nm, const T* dO, const T* H, const T* A,
                       const T* B, const T* U, const void* Wg, const void* Wu, const void* Wd,
                       T* dA, T* dB, T* dH, float* dWg, float* dWu, float* dWd, int E, int M, int F,
                       cudaStream_t st, const float* gate = nullptr, float* dgate_part = nullptr,
                       float* dwd_split = nullptr) {
  const int d = c->d;
  const int64_t P = (int64_t)E * M;
  if (P == 0) {
    EC_CUDA(cudaMemsetAsync(dWg, 0, (size_t)E * d * F * 4, st), "zero dWg");
    EC_CUDA(cudaMemsetAsync(dWu, 0, (size_t)E * d * F * 4, st), "zero dWu");
    EC_CUDA(cudaMemsetAsync(dWd, 0, (size_t)E * d * F * 4, st), "zero dWd");
    return EC_OK;
  }
  int* status = at<int>(c, c->o_status);
  if (use_tc(c)) {
    EC_KERNEL(nm.dgrad_up, 1,
              tc_expert_dgrad_up(dO, Wd, A, B, dA, dB, E, M, d, F, status, st, nullptr, gate,
                                 dgate_part, P, c->tiles));
    EC_KERNEL(nm.dgrad_h, 1,
              tc_expert_dgrad_h(dA, dB, Wg, Wu, dH, E, M, d, F, status, st, nullptr, c->tiles));
    if (dwd_split && E == 1 && M % 2 == 0 && M >= 2048 &&
        2 * ((F + 255) / 256) * ((d + 511) / 512) <= sm_pairs(c)) {
      EC_KERNEL(nm.wgrad, 1,
                tc_expert_wgrad(H, U, dO, dA, dB, dWg, dWu, nullptr, 1, M, d, F, status, st,
                                nullptr, c->tiles));
      EC_KERNEL(nm.wgrad, 1,
                tc_expert_wgrad(H, U, dO, nullptr, nullptr, nullptr, nullptr, dwd_split, 2, M / 2,
                                d, F, status, st, nullptr, c->tiles));
      EC_KERNEL(nm.wgrad, 1,
                launch_reduce_splits(dwd_split, dWd, (int64_t)F * d, 2, st));
    } else {
      EC_KERNEL(nm.wgrad, 2,
                tc_expert_wgrad(H, U, dO, dA, dB, dWg, dWu, dWd, E, M, d, F, status, st, nullptr,
                                c->tiles));
    }
  } else {
    float* dU32 = at<float>(c, c->o_f32a);
    float* dH32 = at<float>(c, c->o_f32b);
    const int64_t hs = (int64_t)M * d, fs = (int64_t)M * F, wgs = (int64_t)d * F;
    // dU = dO . Wd^T : B[k=i][n=j] = Wd[j][i]
    EC_KERNEL(nm.dgrad_up, 1,
              launch_simt_gemm(sg(dO, hs, d, 1, Wd, (int64_t)F * d, 1, d, dU32, fs, F, M, F, d, E),
                               et(c), et(c), st));
    EC_KERNEL("swiglu_bwd", 1, launch_swiglu_bwd_ew<T>(dU32, A, B, dA, dB, P * F, st));
    // dH = dA . Wg^T + dB . Wu^T
    EC_KERNEL(nm.dgrad_h, 1,
              launch_simt_gemm(sg(dA, fs, F, 1, Wg, wgs, 1, F, dH32, hs, d, M, d, F, E),
                               et(c), et(c), st));
    EC_KERNEL(nm.dgrad_h, 1,
              launch_simt_gemm(sg(dB, fs, F, 1, Wu, wgs, 1, F, dH32, hs, d, M, d, F, E, 1.f),
                               et(c), et(c), st));
    EC_KERNEL("convert_dh", 1, launch_convert<T>(dH32, dH, P * d, st));
    // dWd = U^T dO ; dWg = H^T dA ; dWu = H^T dB   (A[m][k] = U[k][m])
    EC_KERNEL(nm.wgrad, 1,
              launch_simt_gemm(sg(U, fs, 1, F, dO, hs, d, 1, dWd, (int64_t)F * d, d, F, d, M, E),
                               et(c), et(c), st));
    EC_KERNEL(nm.wgrad, 1,
              launch_simt_gemm(sg(H, hs, 1, d, dA, fs, F, 1, dWg, wgs, F, d, F, M, E),
                               et(c), et(c), st));
    EC_KERNEL(nm.wgrad, 1,
              launch_simt_gemm(sg(H, hs, 1, d, dB, fs, F, 1, dWu, wgs, F, d, F, M, E),
                               et(c), et(c), st));
  }
  return EC_OK;
}

#define EC_TRY(call)                  \
  do {                                \
    ec_status _s = (call);            \
    if (_s != EC_OK) return _s;       \
  } while (0)

// ---------------------------------------------------------------- forward
// Shared experts (appendix "Token Coverage": they process every token) are one SwiGLU FFN
// of width Fs over all N tokens; their output is added in the combine.
template <typename T>
ec_status run_forward(ec_ctx* c, const void* X, const void* Wg, const void* Wu, const void* Wd,
                      const void* Wgs, const void* Wus, const void* Wds, void* Y,
                      cudaStream_t st) {
  const int N = c->N, d = c->d, E = c->E, F = c->F, M = c->M, Fs = c->Fs;
  const int64_t P = (int64_t)E * M;
  const int pz = P > 0;
  const T* Xt = static_cast<const T*>(X);
  T* H = at<T>(c, c->o_H);
  T* O = at<T>(c, c->o_O);
  const T* Osh = nullptr;
  if (Fs > 0) {
    T* o = at<T>(c, c->o_Osh);
    EC_TRY(ffn_forward<T>(c, kShared, Xt, Wgs, Wus, Wds, at<T>(c, c->o_Ash), at<T>(c, c->o_Bsh),
                          at<T>(c, c->o_Ush), o, 1, N, Fs, st));
    Osh = o;
  }
  const int* idx = at<int>(c, c->o_idx);
  const float* gate = at<float>(c, c->o_gate);
  // tensor cores: the gate is applied in the gate/up epilogue (O rows come out gated)
  const bool fused_gate = use_tc(c);
  // token-major: each X row is read once and written to the rows of the experts that chose it
  EC_KERNEL("gather", N > 0 && pz,
            launch_scatter_rows<T>(Xt, at<int>(c, c->o_slot), H, N, E, M, d, st));
  EC_TRY(ffn_forward<T>(c, kRouted, H, Wg, Wu, Wd, at<T>(c, c->o_A), at<T>(c, c->o_B),
                        at<T>(c, c->o_U), O, E, M, F, st, fused_gate ? gate : nullptr));
  EC_KERNEL("combine", N > 0,
            launch_combine<T>(O, fused_gate ? nullptr : gate, at<int>(c, c->o_slot),
                              c->residual ? Xt : nullptr, Osh, static_cast<T*>(Y), N, E, M, d,
                              st));
  return EC_OK;
}

// ---------------------------------------------------------------- backward
template <typename T>
ec_status run_backward(ec_ctx* c, const void* dY, void* dX, float* dWr, float* dbr, float* dWg,
                       float* dWu, float* dWd, float* dWgs, float* dWus, float* dWds,
                       cudaStream_t st) {
  const int N = c->N, d = c->d, E = c->E, F = c->F, M = c->M, Fs = c->Fs;
  const int64_t P = (int64_t)E * M;
  const int pz = P > 0, nz = N > 0;
  const T* dYt = static_cast<const T*>(dY);
  T* O = at<T>(c, c->o_O);
  T* dH = O;  // O is dead once dgate is formed
  T* dO = at<T>(c, c->o_dO);
  float* dgate = at<float>(c, c->o_dgate);
  float* dZ = at<float>(c, c->o_dZ);
  int* status = at<int>(c, c->o_status);
  const int* idx = at<int>(c, c->o_idx);
  const float* gate = at<float>(c, c->o_gate);
  const int* slot = at<int>(c, c->o_slot);

  if (use_tc(c)) {
    // dO holds dY[idx] ungated; the dU epilogue applies the gate and forms dgate
    EC_KERNEL("gather_dy", N > 0 && pz, launch_scatter_rows<T>(dYt, slot, dO, N, E, M, d, st));
    EC_TRY(ffn_backward<T>(c, kRouted, dO, at<T>(c, c->o_H), at<T>(c, c->o_A), at<T>(c, c->o_B),
                           at<T>(c, c->o_U), c->Wg, c->Wu, c->Wd, at<T>(c, c->o_dA),
                           at<T>(c, c->o_dB), dH, dWg, dWu, dWd, E, M, F, st, gate, dgate));
  } else {
    EC_KERNEL("bwd_gather_scale", pz,
              launch_bwd_gather_scale<T>(dYt, O, idx, gate, dO, dgate, P, d, st));
    EC_TRY(ffn_backward<T>(c, kRouted, dO, at<T>(c, c->o_H), at<T>(c, c->o_A), at<T>(c, c->o_B),
                           at<T>(c, c->o_U), c->Wg, c->Wu, c->Wd, at<T>(c, c->o_dA),
                           at<T>(c, c->o_dB), dH, dWg, dWu, dWd, E, M, F, st));
  }
  const T* dHsh = nullptr;
  if (Fs > 0) {
    // shared experts: dO is dY itself (no gate), the input gradient goes into the dX scatter
    T* dh = at<T>(c, c->o_Osh);
    EC_TRY(ffn_backward<T>(c, kShared, dYt, static_cast<const T*>(c->X), at<T>(c, c->o_Ash),
                           at<T>(c, c->o_Bsh), at<T>(c, c->o_Ush), c->Wgs, c->Wus, c->Wds,
                           at<T>(c, c->o_dAsh), at<T>(c, c->o_dBsh), dh, dWgs, dWus, dWds, 1, N,
                           Fs, st, nullptr, nullptr,
                           use_tc(c) ? at<float>(c, c->o_shpart) : nullptr));
    dHsh = dh;
  }
  // router: dZ = S (dS - <dS,S>), dX = dZ Wr^T + sum dH, dWr = X^T dZ, dbr = sum dZ
  T* dXr = at<T>(c, c->o_dXr);
  float* part = at<float>(c, c->o_part);
  const T* res = c->residual ? dYt : nullptr;
  // Up to 128 experts one kernel sums the gate-gradient partials, applies the softmax
  // Jacobian and takes the bias gradient's column sums (plus one kernel that adds those up).
  const float* S = at<float>(c, c->o_S);
  const bool fused = router_bwd_fused(E, (int64_t)P);
  float* colsum = at<float>(c, c->o_colsum);
  const int rb_launches = nz * (1 + (dbr ? 1 : 0));
  if (use_tc(c)) {
    bf16* dZb = at<bf16>(c, c->o_dZb);
    if (fused) {
      EC_KERNEL("softmax_bwd", rb_launches,
                launch_router_softmax_bwd(S, slot, dgate, c->dg_parts, nullptr, dZb, dbr, colsum,
                                          N, E, c->Ep, M, st));
    } else {
      float* dgsum = at<float>(c, c->o_dgsum);
      EC_KERNEL("dgate_reduce", pz, launch_reduce_splits(dgate, dgsum, P, c->dg_parts, st));
      EC_KERNEL("softmax_bwd", nz,
                launch_softmax_bwd(S, slot, dgsum, dZ, dZb, N, E, c->Ep, M, st));
    }
    EC_KERNEL("router_dgrad_gemm", nz,
              tc_router_dgrad(dZb, router_b(c), dXr, N, d, c->Ep, status, st));
    EC_KERNEL("dx_combine", nz,
              launch_dx_combine<T>(dH, slot, dXr, res, dHsh, static_cast<T*>(dX), N, E, M, d, st));
    EC_KERNEL("router_wgrad_gemm", nz,
              tc_router_wgrad(c->X, dZb, part, N, d, c->Ep, c->wr_splits, status, st));
    EC_KERNEL("router_wgrad_reduce", 1,
              launch_reduce_partials(part, dWr, d, E, c->Ep, 2 * c->wr_splits, st));
  } else {
    if (fused)
      EC_KERNEL("softmax_bwd", rb_launches,
                launch_router_softmax_bwd(S, slot, dgate, 1, dZ, nullptr, dbr, colsum, N, E, E, M,
                                          st));
    else
      EC_KERNEL("softmax_bwd", nz, launch_softmax_bwd(S, slot, dgate, dZ, nullptr, N, E, E, M, st));
    EC_KERNEL("router_dgrad_gemm", nz,
              launch_simt_gemm(sg(dZ, 0, E, 1, c->Wr, 0, 1, E, reinterpret_cast<float*>(dXr), 0, d,
                                  N, d, E, 1),
                               EType::F32,
                               et(c), st));
    EC_KERNEL("dx_combine", nz,
              launch_dx_combine<T>(dH, slot, dXr, res, dHsh, static_cast<T*>(dX), N, E, M, d, st));
    SimtGemmArgs a = sg(c->X, 0, 1, d, dZ, 0, E, 1, part, 0, E, d, E, N, 1);
    a.splits = c->wr_splits;
    a.c_split = (int64_t)d * E;
    EC_KERNEL("router_wgrad_gemm", 1, launch_simt_gemm(a, et(c), EType::F32, st));
    EC_KERNEL("router_wgrad_reduce", 1,
              launch_reduce_splits(part, dWr, (int64_t)d * E, c->wr_splits, st));
  }
  if (dbr && !fused) EC_KERNEL("router_dbias", 2, launch_colsum(dZ, dbr, N, E, colsum, st));
  return EC_OK;
}

// ---------------------------------------------------------------- token choice (bf16)
// Token-major copy of X (or dY) rows into the padded expert regions, padding rows zeroed.
cudaError_t tc_scatter(const bf16* X, const int* slot, const int* count, const int* tiles, bf16* H,
                       int N, int E, int d, cudaStream_t st) {
  cudaError_t e = launch_scatter_rows<bf16>(X, slot, H, N, E, 0, d, st);
  if (e != cudaSuccess) return e;
  return launch_zero_pad_rows<bf16>(count, tiles, H, E, d, st);
}

// Sec. 2.2 "Token-choice": router -> per-token top-k with renormalised gates and the
// per-expert cap -> gather into padded expert regions -> variable-row expert GEMMs ->
// gated combine through the token->row map.
ec_status run_tc_forward(ec_ctx* c, const void* X, const void* Wr, const float* br, const void* Wg,
                         const void* Wu, const void* Wd, void* Y, cudaStream_t st) {
  const int N = c->N, d = c->d, E = c->E, F = c->F, k = c->tc_k;
  const int nz = N > 0;
  int* status = at<int>(c, c->o_status);
  float* S = at<float>(c, c->o_S);
  int* count = at<int>(c, c->o_count);
  int* tiles = at<int>(c, c->o_tiles);
  int* row_token = at<int>(c, c->o_idx);
  float* row_gate = at<float>(c, c->o_gate);
  int* slot = at<int>(c, c->o_slot);
  const bf16* Xt = static_cast<const bf16*>(X);
  bf16* H = at<bf16>(c, c->o_H);
  bf16* U = at<bf16>(c, c->o_U);
  bf16* O = at<bf16>(c, c->o_O);
  if (!nz) return EC_OK;
  EC_KERNEL("router_gemm_softmax", router_needs_pad(E) ? 2 : 1,
            tc_router_softmax(X, Wr, at<void>(c, c->o_wrpad), br, S, at<float>(c, c->o_ST),
                              nullptr, N, d, E, status, st));
  EC_KERNEL("tc_route", 5,
            launch_tc_route(S, N, E, k, c->tc_cap, at<int>(c, c->o_choice),
                            at<float>(c, c->o_tgate), at<float>(c, c->o_Zs), count, tiles,
                            row_token, row_gate, slot, at<int>(c, c->o_kept),
                            at<int>(c, c->o_tcscr), st));
  const VarRows vr{tiles, count, (int)c->P_tc};
  EC_KERNEL("gather", 2, tc_scatter(Xt, slot, count, tiles, H, N, E, d, st));
  EC_KERNEL("gemm_gate_up_swiglu", 1,
            tc_expert_up(H, Wg, Wu, at<bf16>(c, c->o_A), at<bf16>(c, c->o_B), U, E, 0, d, F,
                         status, st, &vr, row_gate, c->tiles));
  EC_KERNEL("gemm_down", 1, tc_expert_down(U, Wd, O, E, 0, d, F, status, st, &vr, c->tiles));
  EC_KERNEL("combine", 1,
            launch_combine<bf16>(O, nullptr, slot, c->residual ? Xt : nullptr, nullptr,
                                 static_cast<bf16*>(Y), N, E, 0, d, st));
  return EC_OK;
}

ec_status run_tc_backward(ec_ctx* c, const void* dY, void* dX, float* dWr, float* dbr, float* dWg,
                          float* dWu, float* dWd, cudaStream_t st) {
  const int N = c->N, d = c->d, E = c->E, F = c->F, k = c->tc_k;
  if (N == 0) {
    const size_t w = (size_t)E * d * F * 4;
    EC_CUDA(cudaMemsetAsync(dWg, 0, w, st), "zero dWg");
    EC_CUDA(cudaMemsetAsync(dWu, 0, w, st), "zero dWu");
    EC_CUDA(cudaMemsetAsync(dWd, 0, w, st), "zero dWd");
    EC_CUDA(cudaMemsetAsync(dWr, 0, (size_t)d * E * 4, st), "zero dWr");
    if (dbr) EC_CUDA(cudaMemsetAsync(dbr, 0, (size_t)E * 4, st), "zero dbr");
    return EC_OK;
  }
  int* status = at<int>(c, c->o_status);
  const int* count = at<int>(c, c->o_count);
  const VarRows vr{at<int>(c, c->o_tiles), count, (int)c->P_tc};
  const bf16* dYt = static_cast<const bf16*>(dY);
  bf16* O = at<bf16>(c, c->o_O);
  bf16* dH = O;   // O is dead once the gate gradients are formed
  bf16* dO = at<bf16>(c, c->o_dO);
  bf16* dA = at<bf16>(c, c->o_dA);
  bf16* dB = at<bf16>(c, c->o_dB);
  float* row_dgate = at<float>(c, c->o_dgate);
  const int* slot = at<int>(c, c->o_slot);
  // dO = dY rows ungated; the dU epilogue applies the row gates and forms their gradients
  EC_KERNEL("gather_dy", 2, tc_scatter(dYt, slot, count, vr.tiles, dO, N, E, d, st));
  EC_KERNEL("gemm_dgrad_up_swiglu", 1,
            tc_expert_dgrad_up(dO, c->Wd, at<bf16>(c, c->o_A), at<bf16>(c, c->o_B), dA, dB, E, 0,
                               d, F, status, st, &vr, at<float>(c, c->o_gate), row_dgate,
                               c->P_tc));
  EC_KERNEL("gemm_dgrad_h", 1,
            tc_expert_dgrad_h(dA, dB, c->Wg, c->Wu, dH, E, 0, d, F, status, st, &vr, c->tiles));
  EC_KERNEL("gemm_wgrad", 2,
            tc_expert_wgrad(at<bf16>(c, c->o_H), at<bf16>(c, c->o_U), dO, dA, dB, dWg, dWu, dWd, E,
                            0, d, F, status, st, &vr, c->tiles));
  float* dZ = at<float>(c, c->o_dZ);
  bf16* dZb = at<bf16>(c, c->o_dZb);
  bf16* dXr = at<bf16>(c, c->o_dXr);
  float* part = at<float>(c, c->o_part);
  float* dgsum = at<float>(c, c->o_dgsum);
  EC_KERNEL("dgate_reduce", 1, launch_reduce_splits(row_dgate, dgsum, c->P_tc, c->dg_parts, st));
  EC_KERNEL("softmax_bwd", 1,
            launch_tc_softmax_bwd(at<float>(c, c->o_S), at<int>(c, c->o_choice),
                                  at<float>(c, c->o_tgate), at<float>(c, c->o_Zs), slot, dgsum, dZ,
                                  dZb, N, E, c->Ep, k, st));
  EC_KERNEL("router_dgrad_gemm", 1,
            tc_router_dgrad(dZb, router_b(c), dXr, N, d, c->Ep, status, st));
  EC_KERNEL("dx_combine", 1,
            launch_dx_combine<bf16>(dH, slot, dXr, c->residual ? dYt : nullptr, nullptr,
                                    static_cast<bf16*>(dX), N, E, 0, d, st));
  EC_KERNEL("router_wgrad_gemm", 1,
            tc_router_wgrad(c->X, dZb, part, N, d, c->Ep, c->wr_splits, status, st));
  EC_KERNEL("router_wgrad_reduce", 1,
            launch_reduce_partials(part, dWr, d, E, c->Ep, 2 * c->wr_splits, st));
  if (dbr)
    EC_KERNEL("router_dbias", 2, launch_colsum(dZ, dbr, N, E, at<float>(c, c->o_colsum), st));
  return EC_OK;
}

}  // namespace

// ====================================================================== C ABI
extern "C" {

const char* ec_status_string(ec_status s) {
  switch (s) {
    case EC_OK: return "EC_OK";
    case EC_ERR_INVALID_ARG: return "EC_ERR_INVALID_ARG";
    case EC_ERR_SHAPE: return "EC_ERR_SHAPE";
    case EC_ERR_UNSUPPORTED: return "EC_ERR_UNSUPPORTED";
    case EC_ERR_CUDA: return "EC_ERR_CUDA";
    case EC_ERR_TIMEOUT: return "EC_ERR_TIMEOUT";
    case EC_ERR_WORKSPACE: return "EC_ERR_WORKSPACE";
    case EC_ERR_STATE: return "EC_ERR_STATE";
  }
  return "EC_ERR_UNKNOWN";
}

ec_status ec_ctx_create(ec_ctx** out, int32_t N, int32_t d, int32_t E, int32_t d_ff, int32_t G,
                        const int32_t* group_off, const int32_t* k_g, int32_t dtype) {
  if (!out) return EC_ERR_INVALID_ARG;
  *out = nullptr;
  if (dtype != EC_F32 && dtype != EC_BF16) return EC_ERR_INVALID_ARG;
  if (N < 0 || d <= 0 || E <= 0 || d_ff <= 0 || G <= 0) return EC_ERR_SHAPE;
  if (E > 512) return EC_ERR_UNSUPPORTED;
  if (dtype == EC_BF16 && (d % 64 || d_ff % 64)) return EC_ERR_UNSUPPORTED;
  if (dtype == EC_F32 && (d % 4 || d_ff % 4)) return EC_ERR_UNSUPPORTED;
  if (dtype == EC_BF16 && E > 256) return EC_ERR_UNSUPPORTED;
  ec_ctx* c = new ec_ctx();
  c->N = N; c->d = d; c->E = E; c->F = d_ff; c->G = G; c->dtype = dtype;
  ec_status s = set_groups(c, group_off, k_g, true);
  if (s != EC_OK) { delete c; return s; }
  layout(c);
  *out = c;
  return EC_OK;
}

void ec_ctx_destroy(ec_ctx* c) {
  if (!c) return;
  for (cudaEvent_t e : c->ev) cudaEventDestroy(e);
  delete c;
}

ec_status ec_ctx_set_capacity(ec_ctx* c, const int32_t* k_g) {
  if (!c) return EC_ERR_INVALID_ARG;
  if (c && c->tc_k) return fail(c, EC_ERR_STATE, "token-choice context: use ec_tc_forward / ec_tc_backward");
  ec_status s = set_groups(c, nullptr, k_g, false);
  if (s != EC_OK) return s;
  // the group tables are rewritten in place: no kernel of an earlier call, on any stream, may
  // still be reading them
  if (c->ws) EC_CUDA(cudaDeviceSynchronize(), "wait for the device before the capacity update");
  return upload_groups(c);
}

ec_status ec_ctx_set_capacity_async(ec_ctx* c, const int32_t* k_g_dev, void* stream) {
  ec_status s = check_ready(c);
  if (s != EC_OK) return s;
  if (c->tc_k) return fail(c, EC_ERR_STATE, "token-choice context: use ec_tc_forward / ec_tc_backward");
  if (!k_g_dev) return fail(c, EC_ERR_INVALID_ARG, "k_g is NULL");
  if (reinterpret_cast<uintptr_t>(k_g_dev) & 3u)
    return fail(c, EC_ERR_INVALID_ARG, "k_g must be 4-byte aligned");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  c->have_fwd = false;
  EC_KERNEL("set_capacity", 1,
            launch_set_capacity(k_g_dev, at<int>(c, c->o_goff), c->G, c->M, at<int>(c, c->o_kg),
                                at<int>(c, c->o_koff), at<int>(c, c->o_status), st));
  mark(c, "end", st);
  return EC_OK;
}

int64_t ec_rows_per_expert(const ec_ctx* c) { return c ? c->M : -1; }

size_t ec_workspace_bytes(const ec_ctx* c) { return c ? c->total : 0; }

ec_status ec_ctx_set_workspace(ec_ctx* c, void* ws, size_t bytes) {
  if (!c) return EC_ERR_INVALID_ARG;
  if (!ws) return fail(c, EC_ERR_WORKSPACE, "workspace is NULL");
  if (reinterpret_cast<uintptr_t>(ws) & 255u)
    return fail(c, EC_ERR_WORKSPACE, "workspace must be 256-byte aligned");
  if (bytes < c->total)
    return fail(c, EC_ERR_WORKSPACE, "workspace has %zu bytes, needs %zu", bytes, c->total);
  c->ws = static_cast<char*>(ws);
  c->ws_bytes = bytes;
  c->have_fwd = false;
  EC_CUDA(cudaMemset(c->ws + c->o_status, 0, 256), "clear status");
  return upload_groups(c);
}

ec_status ec_route(ec_ctx* c, const void* X, const void* Wr, const float* br, const float* S_in,
                   float* S_out, int32_t* idx, float* gate, void* stream) {
  ec_status s = check_ready(c);
  if (s != EC_OK) return s;
  if (c && c->tc_k) return fail(c, EC_ERR_STATE, "token-choice context: use ec_tc_forward / ec_tc_backward");
  if (!S_in && (!X || !Wr)) return fail(c, EC_ERR_INVALID_ARG, "X and Wr are required without S_in");
  if (!idx || !gate) return fail(c, EC_ERR_INVALID_ARG, "idx and gate are required");
  if ((X && !aligned16(X)) || (Wr && !aligned16(Wr)) || (S_in && !aligned16(S_in)))
    return fail(c, EC_ERR_INVALID_ARG, "inputs must be 16-byte aligned");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  c->have_fwd = false;
  s = c->dtype == EC_BF16 ? run_route<bf16>(c, X, Wr, br, S_in, st)
                          : run_route<float>(c, X, Wr, br, S_in, st);
  if (s != EC_OK) return s;
  mark(c, "end", st);
  return copy_out(c, idx, gate, S_out, st);
}

static ec_status forward_impl(ec_ctx* c, const void* X, const void* Wr, const float* br,
                              const void* Wg, const void* Wu, const void* Wd, const void* Wgs,
                              const void* Wus, const void* Wds, void* Y, int32_t* idx,
                              float* gate, float* S_out, void* stream) {
  ec_status s = check_ready(c);
  if (s != EC_OK) return s;
  if (c && c->tc_k) return fail(c, EC_ERR_STATE, "token-choice context: use ec_tc_forward / ec_tc_backward");
  if (!X || !Wr || !Wg || !Wu || !Wd || !Y)
    return fail(c, EC_ERR_INVALID_ARG, "X, Wr, Wg, Wu, Wd and Y are required");
  for (const void* p : {X, Wr, Wg, Wu, Wd, (const void*)Y})
    if (!aligned16(p)) return fail(c, EC_ERR_INVALID_ARG, "tensors must be 16-byte aligned");
  if (c->Fs > 0 && (!Wgs || !Wus || !Wds || !aligned16(Wgs) || !aligned16(Wus) || !aligned16(Wds)))
    return fail(c, EC_ERR_INVALID_ARG, "shared-expert weights are required and 16-byte aligned");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  c->have_fwd = false;
  c->Wgs = Wgs; c->Wus = Wus; c->Wds = Wds;
  s = c->dtype == EC_BF16 ? run_route<bf16>(c, X, Wr, br, nullptr, st)
                          : run_route<float>(c, X, Wr, br, nullptr, st);
  if (s != EC_OK) return s;
  s = c->dtype == EC_BF16 ? run_forward<bf16>(c, X, Wg, Wu, Wd, Wgs, Wus, Wds, Y, st)
                          : run_forward<float>(c, X, Wg, Wu, Wd, Wgs, Wus, Wds, Y, st);
  if (s != EC_OK) return s;
  mark(c, "end", st);
  s = copy_out(c, idx, gate, S_out, st);
  if (s != EC_OK) return s;
  c->X = X; c->Wr = Wr; c->br = br; c->Wg = Wg; c->Wu = Wu; c->Wd = Wd;
  c->have_fwd = true;
  return EC_OK;
}

static ec_status backward_impl(ec_ctx* c, const void* dY, void* dX, float* dWr, float* dbr,
                               float* dWg, float* dWu, float* dWd, float* dWgs, float* dWus,
                               float* dWds, void* stream) {
  ec_status s = check_ready(c);
  if (s != EC_OK) return s;
  if (c && c->tc_k) return fail(c, EC_ERR_STATE, "token-choice context: use ec_tc_forward / ec_tc_backward");
  if (!c->have_fwd) return fail(c, EC_ERR_STATE, "the backward call needs a preceding forward");
  if (!dY || !dX || !dWr || !dWg || !dWu || !dWd)
    return fail(c, EC_ERR_INVALID_ARG, "dY, dX, dWr, dWg, dWu and dWd are required");
  for (const void* p : {dY, (const void*)dX, (const void*)dWr, (const void*)dWg, (const void*)dWu,
                        (const void*)dWd})
    if (!aligned16(p)) return fail(c, EC_ERR_INVALID_ARG, "tensors must be 16-byte aligned");
  if (c->Fs > 0 && (!dWgs || !dWus || !dWds || !aligned16(dWgs) || !aligned16(dWus) ||
                    !aligned16(dWds)))
    return fail(c, EC_ERR_INVALID_ARG, "shared-expert gradients are required and 16-byte aligned");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  c->dWgs = dWgs; c->dWus = dWus; c->dWds = dWds;
  s = c->dtype == EC_BF16
          ? run_backward<bf16>(c, dY, dX, dWr, dbr, dWg, dWu, dWd, dWgs, dWus, dWds, st)
          : run_backward<float>(c, dY, dX, dWr, dbr, dWg, dWu, dWd, dWgs, dWus, dWds, st);
  if (s != EC_OK) return s;
  mark(c, "end", st);
  return EC_OK;
}

ec_status ec_moe_forward(ec_ctx* c, const void* X, const void* Wr, const float* br, const void* Wg,
                         const void* Wu, const void* Wd, void* Y, int32_t* idx, float* gate,
                         float* S_out, void* stream) {
  if (c && c->Fs > 0)
    return fail(c, EC_ERR_STATE, "the context has shared experts: use ec_moe_forward_shared");
  return forward_impl(c, X, Wr, br, Wg, Wu, Wd, nullptr, nullptr, nullptr, Y, idx, gate, S_out,
                      stream);
}

ec_status ec_moe_backward(ec_ctx* c, const void* dY, void* dX, float* dWr, float* dbr, float* dWg,
                          float* dWu, float* dWd, void* stream) {
  if (c && c->Fs > 0)
    return fail(c, EC_ERR_STATE, "the context has shared experts: use ec_moe_backward_shared");
  return backward_impl(c, dY, dX, dWr, dbr, dWg, dWu, dWd, nullptr, nullptr, nullptr, stream);
}

ec_status ec_ctx_set_shared(ec_ctx* c, int32_t d_ff_shared) {
  if (!c) return EC_ERR_INVALID_ARG;
  if (c && c->tc_k) return fail(c, EC_ERR_STATE, "token-choice context: use ec_tc_forward / ec_tc_backward");
  if (c->ws) return fail(c, EC_ERR_STATE, "set shared experts before attaching the workspace");
  if (d_ff_shared < 0) return fail(c, EC_ERR_SHAPE, "negative shared width");
  if (c->dtype == EC_BF16 && d_ff_shared % 64)
    return fail(c, EC_ERR_UNSUPPORTED, "bf16 shared width must be a multiple of 64");
  if (c->dtype == EC_F32 && d_ff_shared % 4)
    return fail(c, EC_ERR_UNSUPPORTED, "fp32 shared width must be a multiple of 4");
  c->Fs = d_ff_shared;
  c->have_fwd = false;
  layout(c);
  return EC_OK;
}

ec_status ec_moe_forward_shared(ec_ctx* c, const void* X, const void* Wr, const float* br,
                                const void* Wg, const void* Wu, const void* Wd, const void* Wg_s,
                                const void* Wu_s, const void* Wd_s, void* Y, int32_t* idx,
                                float* gate, float* S_out, void* stream) {
  if (c && c->Fs == 0)
    return fail(c, EC_ERR_STATE, "no shared experts configured (ec_ctx_set_shared)");
  return forward_impl(c, X, Wr, br, Wg, Wu, Wd, Wg_s, Wu_s, Wd_s, Y, idx, gate, S_out, stream);
}

ec_status ec_moe_backward_shared(ec_ctx* c, const void* dY, void* dX, float* dWr, float* dbr,
                                 float* dWg, float* dWu, float* dWd, float* dWg_s, float* dWu_s,
                                 float* dWd_s, void* stream) {
  if (c && c->Fs == 0)
    return fail(c, EC_ERR_STATE, "no shared experts configured (ec_ctx_set_shared)");
  return backward_impl(c, dY, dX, dWr, dbr, dWg, dWu, dWd, dWg_s, dWu_s, dWd_s, stream);
}

ec_status ec_tc_ctx_create(ec_ctx** out, int32_t N, int32_t d, int32_t E, int32_t d_ff,
                           int32_t k, int32_t capacity, int32_t dtype) {
  if (!out) return EC_ERR_INVALID_ARG;
  *out = nullptr;
  if (dtype != EC_F32 && dtype != EC_BF16) return EC_ERR_INVALID_ARG;
  if (dtype != EC_BF16) return EC_ERR_UNSUPPORTED;
  if (N < 0 || d <= 0 || E <= 0 || d_ff <= 0) return EC_ERR_SHAPE;
  if (k < 1 || k > E || k > 32) return EC_ERR_SHAPE;
  if (E > 256 || d % 64 || d_ff % 64) return EC_ERR_UNSUPPORTED;
  const int64_t P = ((int64_t)N * k + 255 * (int64_t)E + 255) / 256 * 256;
  if (P > ((int64_t)1 << 30)) return EC_ERR_UNSUPPORTED;
  const int32_t off[2] = {0, N};
  const int32_t kg[1] = {0};
  ec_status s = ec_ctx_create(out, N, d, E, d_ff, 1, off, kg, dtype);
  if (s != EC_OK) return s;
  ec_ctx* c = *out;
  c->tc_k = k;
  c->tc_cap = capacity < 0 ? -1 : capacity;
  c->P_tc = P;
  layout(c);
  return EC_OK;
}

ec_status ec_tc_forward(ec_ctx* c, const void* X, const void* Wr, const float* br,
                        const void* Wg, const void* Wu, const void* Wd, void* Y, int32_t* choice,
                        float* gate, int32_t* kept, int32_t* load, float* S_out, void* stream) {
  ec_status s = check_ready(c);
  if (s != EC_OK) return s;
  if (!c->tc_k) return fail(c, EC_ERR_STATE, "not a token-choice context (ec_tc_ctx_create)");
  if (!X || !Wr || !Wg || !Wu || !Wd || !Y)
    return fail(c, EC_ERR_INVALID_ARG, "X, Wr, Wg, Wu, Wd and Y are required");
  for (const void* p : {X, Wr, Wg, Wu, Wd, (const void*)Y})
    if (!aligned16(p)) return fail(c, EC_ERR_INVALID_ARG, "tensors must be 16-byte aligned");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  c->have_fwd = false;
  s = run_tc_forward(c, X, Wr, br, Wg, Wu, Wd, Y, st);
  if (s != EC_OK) return s;
  mark(c, "end", st);
  const size_t NK = (size_t)c->N * c->tc_k;
  if (NK) {
    if (choice)
      EC_CUDA(cudaMemcpyAsync(choice, at<int>(c, c->o_choice), NK * 4, cudaMemcpyDeviceToDevice, st),
              "choice out");
    if (gate)
      EC_CUDA(cudaMemcpyAsync(gate, at<float>(c, c->o_tgate), NK * 4, cudaMemcpyDeviceToDevice, st),
              "gate out");
    if (kept)
      EC_CUDA(cudaMemcpyAsync(kept, at<int>(c, c->o_kept), NK * 4, cudaMemcpyDeviceToDevice, st),
              "kept out");
    if (load)
      EC_CUDA(cudaMemcpyAsync(load, at<int>(c, c->o_count), (size_t)c->E * 4,
                              cudaMemcpyDeviceToDevice, st), "load out");
    if (S_out)
      EC_CUDA(cudaMemcpyAsync(S_out, at<float>(c, c->o_S), (size_t)c->N * c->E * 4,
                              cudaMemcpyDeviceToDevice, st), "S out");
  } else if (load) {
    EC_CUDA(cudaMemsetAsync(load, 0, (size_t)c->E * 4, st), "load out");
  }
  c->X = X; c->Wr = Wr; c->br = br; c->Wg = Wg; c->Wu = Wu; c->Wd = Wd;
  c->have_fwd = true;
  return EC_OK;
}

ec_status ec_tc_backward(ec_ctx* c, const void* dY, void* dX, float* dWr, float* dbr,
                         float* dWg, float* dWu, float* dWd, void* stream) {
  ec_status s = check_ready(c);
  if (s != EC_OK) return s;
  if (!c->tc_k) return fail(c, EC_ERR_STATE, "not a token-choice context (ec_tc_ctx_create)");
  if (!c->have_fwd) return fail(c, EC_ERR_STATE, "the backward call needs a preceding forward");
  if (!dY || !dX || !dWr || !dWg || !dWu || !dWd)
    return fail(c, EC_ERR_INVALID_ARG, "dY, dX, dWr, dWg, dWu and dWd are required");
  for (const void* p : {dY, (const void*)dX, (const void*)dWr, (const void*)dWg, (const void*)dWu,
                        (const void*)dWd})
    if (!aligned16(p)) return fail(c, EC_ERR_INVALID_ARG, "tensors must be 16-byte aligned");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  s = run_tc_backward(c, dY, dX, dWr, dbr, dWg, dWu, dWd, st);
  if (s != EC_OK) return s;
  mark(c, "end", st);
  return EC_OK;
}

ec_status ec_ctx_set_residual(ec_ctx* c, int32_t on) {
  if (!c) return EC_ERR_INVALID_ARG;
  c->residual = on != 0;
  c->have_fwd = false;
  return EC_OK;
}

ec_status ec_ctx_set_tiles(ec_ctx* c, int32_t policy) {
  if (!c) return EC_ERR_INVALID_ARG;
  if (policy != EC_TILES_AUTO && policy != EC_TILES_256 && policy != EC_TILES_512)
    return fail(c, EC_ERR_INVALID_ARG, "tile policy %d is not one of 0, 1, 2", policy);
  c->tiles = policy;
  return EC_OK;
}

ec_status ec_ctx_set_profiling(ec_ctx* c, int32_t on) {
  if (!c) return EC_ERR_INVALID_ARG;
  c->prof = on != 0;
  c->ev_n = 0;
  return EC_OK;
}

int32_t ec_ctx_profile(ec_ctx* c, const char** names, float* ms, int32_t cap) {
  if (!c || c->ev_n == 0) return 0;
  if (cudaEventSynchronize(c->ev[c->ev_n - 1]) != cudaSuccess) return -1;
  int32_t n = 0;
  for (int i = 0; i + 1 < c->ev_n; ++i) {
    if (std::strcmp(c->ev_name[i], "end") == 0) continue;
    if (n < cap) {
      float t = 0.f;
      cudaEventElapsedTime(&t, c->ev[i], c->ev[i + 1]);
      if (names) names[n] = c->ev_name[i];
      if (ms) ms[n] = t;
    }
    ++n;
  }
  return n;
}

int64_t ec_kernel_launches(const ec_ctx* c) { return c ? c->launches : -1; }

ec_status ec_selftest_bounded_wait(ec_ctx* c, uint64_t limit_ns, void* stream) {
  ec_status s = check_ready(c);
  if (s != EC_OK) return s;
  if (limit_ns > 10000000000ull) return fail(c, EC_ERR_INVALID_ARG, "limit above 10 s");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  EC_KERNEL("wait_probe", 1, tc_wait_probe(at<int>(c, c->o_status), limit_ns, st));
  return EC_OK;
}

ec_status ec_check_device(ec_ctx* c, void* stream) {
  ec_status s = check_ready(c);
  if (s != EC_OK) return s;
  EC_CUDA(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)), "stream sync");
  int word = 0;
  EC_CUDA(cudaMemcpy(&word, c->ws + c->o_status, 4, cudaMemcpyDeviceToHost), "read status");
  if (word != DEV_OK) {
    EC_CUDA(cudaMemset(c->ws + c->o_status, 0, 256), "clear status");
    if (word == DEV_BAD_CAPACITY)
      return fail(c, EC_ERR_SHAPE,
                  "a capacity update from device memory was rejected (k_g outside [0, L_g] or "
                  "sum(k_g) != %d); the previous capacities stayed in force", c->M);
    return fail(c, EC_ERR_TIMEOUT, "a kernel gave up on a bounded wait (device status %d)", word);
  }
  return EC_OK;
}

const char* ec_last_error(const ec_ctx* c) { return c ? c->err.c_str() : ""; }

ec_status ec_get_last_error(const ec_ctx* c, char* buf, size_t n) {
  if (!c || (!buf && n > 0)) return EC_ERR_INVALID_ARG;
  if (n > 0) {
    const size_t len = std::min(c->err.size(), n - 1);
    std::memcpy(buf, c->err.data(), len);
    buf[len] = '\0';
  }
  return c->err_status;
}

int64_t ec_tc_capacity(double capacity_factor, int32_t k, int32_t N, int32_t E) {
  if (!(capacity_factor > 0.0)) return -1;   // dropless (also for NaN)
  if (k < 1 || N < 0 || E < 1) return -2;
  // Sec. 2.2: ceil(CF k N / E), evaluated left to right in double precision
  const double v = capacity_factor * (double)k * (double)N / (double)E;
  if (!(v < 9.0e18)) return -2;
  return (int64_t)std::ceil(v);
}

}  // extern "C"
