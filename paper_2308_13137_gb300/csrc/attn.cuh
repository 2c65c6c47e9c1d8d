// Attention-side kernels of the block step (attn.cu).
#pragma once
#include "common.cuh"

// cos/sin table [T, hd/2] of RoPE (frequency theta^(-2j/hd)), evaluated in fp64
omq_status rope_table(cudaStream_t st, int T, int hd, float theta, float* cs /* [T, hd/2, 2] */);

struct QkvArgs {
  int T, H, Hkv, hd;
  const float* Y; int64_t ldy;           // [T, dq + 2 dkv] projection outputs (q | k | v)
  const float* cs;                       // rope table
  const float* sa_exp;                   // [dq] s_a broadcast to query heads (null = no LET)
  const float* sa;                       // [dkv]
  __nv_bfloat16 *Qh, *Kh, *Vh;           // [T, dq], [T, dkv], [T, dkv]
  float* h; int32_t* z; int32_t* imax; int32_t* imin;   // [3, T] (q, k, v)
  int abits; float eps;
  // backward only
  const float* dQKV; int64_t ldd;        // [T, dq + 2 dkv] gradients w.r.t. Qh | Kh | Vh
  float* dY; __nv_bfloat16* dYb;         // [T, dq + 2 dkv] gradients w.r.t. the projection outputs
  float* part_q; float* part_k;          // [nslab, dq], [nslab, dkv] partial sums of ds_a terms
  int rows_per_cta;
};
omq_status qkv_fwd_launch(cudaStream_t st, const QkvArgs& a);
omq_status qkv_bwd_launch(cudaStream_t st, const QkvArgs& a, int64_t* nslab);
int64_t qkv_bwd_nslab(int T);

// P = softmax(S) over keys j <= t (S already scaled); P bf16 [B, T, T], zero for t < j < the end of
// t's 128-row block.
omq_status softmax_fwd_launch(cudaStream_t st, int B, int T, const float* S, __nv_bfloat16* P);
// dS = scale * P (dP - sum_j P dP), bf16, same zero convention
omq_status softmax_bwd_launch(cudaStream_t st, int B, int T, const __nv_bfloat16* P, const float* dP, float scale,
                              __nv_bfloat16* dS);

// [v, out] LET pair vectors: r_qkv = [1 (q,k rows), 1/s_o (v rows)], shift_qkv = [0, delta_o]
omq_status qkv_row_vectors(cudaStream_t st, int dq, int dkv, const float* so, const float* do_, float* r, float* shift);
// ds_o (+)= -(dr_v + dBv * Bv * s_o) / s_o^2 ; ddo (+)= -dBv / s_o   (v rows of the stacked projection)
omq_status let_vo_finalize(cudaStream_t st, int dkv, const float* so, const float* dr_v, const float* dBv,
                           const float* Bv, float* dso, float* ddo, int accumulate);
