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

// C[b] = alpha * A[b] B[b]^T (+bias)(+R)(+beta*C); causal modes as in omq_gemm_bf16
omq_status gemm_launch(cudaStream_t st, int64_t M, int64_t N, int64_t K, int64_t batch, const GemmOperand& A,
                       const GemmOperand& B, const GemmEpilogue& ep, int causal, int32_t* status);
