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

// Causal attention without a materialised score matrix (flash.cu).  Q [T, H*128], K and V
// [T, Hkv*128] bf16 (query head h reads kv head h / (H / Hkv)); O [T, H*128] fp32; lse [H, T] the
// base-2 log-sum-exp of the scaled logits.  Backward: dO bf16 like O; D [H, T] scratch;
// dQ [T, H*128], dK / dV [T, Hkv*128] fp32 (overwritten).
struct FlashArgs {
  int T, H, Hkv, hd;
  const __nv_bfloat16* Q; const __nv_bfloat16* K; const __nv_bfloat16* V;
  int64_t ldq, ldkv;
  float* O; int64_t ldo;
  float* lse;
  const __nv_bfloat16* dO; int64_t lddo;
  float* D;
  int d_ready;            // 1: D already holds rowsum(dO * O) (formed by the producer of dO)
  float* dQ; int64_t ldg;
  float* dK; float* dV; int64_t ldgkv;
  int32_t* status;
  // softmax-output quantization (pbits 2..8; 0 or 16 = off): per query row, MinMax over the
  // visible keys.  pqr [H, T, 8] quantizer state written by the forward, pqb [H, T, 4] backward
  // row statistics (scratch); both 16-byte aligned.
  int pbits; float eps;
  float* pqr; float* pqb;
  // row stride (in rows) of the per-row arrays lse, D, pqr, pqb: [H, ldl(, 8 | 4)]; 0 = T.  A
  // multiple of 4 at least T lets the backward fetch them with 16-byte bulk copies for any T.
  int ldl;
};
static inline bool flash_pq_on(int pbits) { return pbits >= 2 && pbits <= 8; }
omq_status flash_fwd_launch(cudaStream_t st, const FlashArgs& a);
omq_status flash_bwd_launch(cudaStream_t st, const FlashArgs& a);

// [v, out] LET pair vectors: r_qkv = [1 (q,k rows), 1/s_o (v rows)], shift_qkv = [0, delta_o]
omq_status qkv_row_vectors(cudaStream_t st, int dq, int dkv, const float* so, const float* do_, float* r, float* shift);
// ds_o (+)= -(dr_v + dBv * Bv * s_o) / s_o^2 ; ddo (+)= -dBv / s_o   (v rows of the stacked projection)
omq_status let_vo_finalize(cudaStream_t st, int dkv, const float* so, const float* dr_v, const float* dBv,
                           const float* Bv, float* dso, float* ddo, int accumulate);
