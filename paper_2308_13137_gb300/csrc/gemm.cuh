// Internal interface of the tcgen05 bf16 GEMM (gemm.cu).
#pragma once
#include "common.cuh"

struct GemmOperand {
  const void* ptr;   // bf16
  int64_t ld;        // elements between consecutive rows of the stored layout
  int64_t bs;        // elements between batches
  int kmajor;        // 1: element (m|n, k) at row m|n, column k; 0: at row k, column m|n
};

struct GemmEpilogue {
  float* Cf; __nv_bfloat16* Cb;   // outputs (either may be null)
  int64_t ldc, c_bs;
  float alpha;
  const float* bias;              // [N] or null
  const float* R; int64_t ldr;    // residual [M, N] (batch stride c_bs) or null
  float beta_acc;                 // C = ... + beta_acc * C (0 = overwrite)
};

// Straight-through LWC backward (Eq. 2) fused into the epilogue of the weight-gradient product
// dW_hat = dY^T X_hat [M = Cout, N = Cin]: dW_hat never leaves tensor memory.  Each epilogue
// thread owns one output row o of the tile and, per element, forms W~ = fl(fl(W s) r), its
// code decision, the STE gradient d = [0 <= code <= Q] dW_hat and the h-path term.  Outputs:
//  * per-channel (group == N): row partials of G_h = sum dW_hat dWhat/dh, G_bm = sum of dW_hat over
//    clamped elements and dr = sum d W s, one per half N tile ([3, M, ntn], ntn = 2 ceil(N / 256));
//    a finalize completes them;
//  * grouped (group | half N tile, no LET): dgamma_hat, dbeta_hat of every group directly;
//  * LET column partials per 32-row quadrant ([ceil(M/32), N]): sum_o d W r (for ds) and
//    sum_o dB~_o r_o W (for ddelta).
struct GemmLwcEpi {
  const __nv_bfloat16* W;         // [M, N] frozen weight, row stride N
  const float* s;                 // [N] LET column scale or null
  const float* r;                 // [M] row scale or null
  const float* h; const int32_t* z; const float* ga; const float* gb; const float* Mv; const float* mv;
  const float* dBt;               // [M] gradient of the LET bias or null
  float* rowpart;                 // per-channel: [3, M, ntn]
  float* part_s; float* part_d;   // [ceil(M/32), N] or null
  float* dgl; float* dbl;         // grouped: [M, N/group]
  int group, accumulate, ntn;
  float Q, eps;
  int want_dr;                    // the row sums for dr (rowpart[2]) are needed
};

// LWC fake quantization of the B operand inside the GEMM (Eq. 2 and Eq. 4 as operand preparation):
// B is the raw bf16 weight [N, K] (K-major); after each tile lands in shared memory, four warps
// replace every element by its fake-quantized value bf16((clamp(round(w~ / h), -z, Q - z)) h) with
// w~ = fl(fl(w s_k) r_n), exactly the value the LWC forward would have written to HBM.
struct GemmQuantB {
  const float* h; const int32_t* z;   // [N, ngroups] step and zero point (ngroups = K / group)
  const float* r;                     // [N] row scale or null
  const float* s;                     // [K] LET column scale or null
  int group;                          // group size along K (a multiple of 8); K = one group per row
  float Q;                            // 2^N - 1
};

// N-tile width the GEMM uses for a product with N columns
int gemm_n_tile(int64_t N);

// C[b] = alpha * A[b] B[b]^T (+bias)(+R)(+beta*C); causal modes as in omq_gemm_bf16
omq_status gemm_launch(cudaStream_t st, int64_t M, int64_t N, int64_t K, int64_t batch, const GemmOperand& A,
                       const GemmOperand& B, const GemmEpilogue& ep, int causal, int32_t* status);

// C = A B_hat^T with B_hat prepared from the raw weight B in shared memory (GemmQuantB); A, B K-major
omq_status gemm_launch_qb(cudaStream_t st, int64_t M, int64_t N, int64_t K, const GemmOperand& A, const GemmOperand& B,
                          const GemmEpilogue& ep, const GemmQuantB& qb, int32_t* status);

// dW_hat = A B^T (K-reduction over tokens) consumed by the fused LWC epilogue above; no C output
omq_status gemm_launch_lwc(cudaStream_t st, int64_t M, int64_t N, int64_t K, const GemmOperand& A,
                           const GemmOperand& B, const GemmLwcEpi& lw, int32_t* status);
