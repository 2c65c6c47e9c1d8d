// Internal launchers of the HBM-bound kernels (quant.cu), shared with the block step (block.cu).
#pragma once
#include "common.cuh"

// ---- LWC (Eq. 2) on W~ = r_o W_oi s_i --------------------------------------------------------
struct LwcFwdArgs {
  const __nv_bfloat16* W; int64_t Cout, Cin; int group;   // group = Cin for per-channel
  const float* s; const float* r;
  const float* gl; const float* bl;                        // logits [Cout, ngroups]
  int lwc;                                                 // 0 = gamma = beta = 1 (plain MinMax)
  __nv_bfloat16* Wq; uint8_t* codes;
  float* h; int32_t* z; int32_t* imax; int32_t* imin;
  const float* bias_delta; const float* bias_shift; float* Bt;
  float* ga_out; float* gb_out;                            // clipping strengths per group (nullable)
  float* M_out; float* m_out;                              // group max / min of W~ (nullable)
  int wbits; float eps;
  int32_t* status;
};
omq_status lwc_fwd_launch(cudaStream_t st, const LwcFwdArgs& a);

struct LwcBwdArgs {
  const __nv_bfloat16* W; int64_t Cout, Cin; int group;    // group = Cin for per-channel
  const float* s; const float* r;
  const float* gl; const float* bl; int lwc;
  const float* ga; const float* gb;                        // saved sigmoids (nullable: recomputed)
  const float* Mv; const float* mv;                        // saved group max / min (nullable: re-read)
  const float* h; const int32_t* z; const int32_t* imax; const int32_t* imin;
  const float* dWq; int64_t ld_dwq;
  float* dgl; float* dbl; float* dWt; float* dr;
  const float* dBt;
  float* ds; float* ddelta;                                // LET column sums (nullable)
  int wbits; float eps; int accumulate; int accumulate_sd; int accumulate_dr;
};
// scratch: partial column sums and per-row partials, carved from `scratch`
size_t lwc_bwd_scratch_bytes(int64_t Cout, int64_t Cin);
omq_status lwc_bwd_launch(cudaStream_t st, const LwcBwdArgs& a, void* scratch);
// Completion of the LWC backward whose per-element part ran inside the weight-gradient GEMM
// epilogue: per-channel row partials [3, Cout, ntn] -> dgamma, dbeta, max/min routing, dr (a.dWq and
// a.dWt unused); the routing's share of ds (staged in route [Cout, 4], 16-byte aligned) is added
// into the 32-row column partials part_s [nparts = ceil(Cout / 32), Cin] in a fixed order, which
// are then reduced to ds (and part_d to ddelta).
omq_status lwc_bwd_fused_finish(cudaStream_t st, const LwcBwdArgs& a, float* rowpart, int64_t ntn,
                                float* part_s, const float* part_d, int64_t nparts, float* route);

// ---- per-token activation quantizer Q_a with a fused producer ------------------------------
enum ActProducer { AP_PLAIN = 0, AP_LET = 1, AP_RMS_LET = 2, AP_SWIGLU = 3 };

struct ActFwdArgs {
  int producer;
  const float* X; int64_t ldx;       // PLAIN / LET / RMS input; SWIGLU gate
  const float* U; int64_t ldu;       // SWIGLU up
  const float* s; const float* delta;
  float rms_eps; float* rstd;        // RMS: rstd [T] written
  int64_t T, C;
  __nv_bfloat16* Xq; int64_t ldq;
  uint8_t* codes;
  float* h; int32_t* z; int32_t* imax; int32_t* imin;
  int abits; float eps;
  int32_t* status;                   // device status word (timeouts of the staged kernel), nullable
  int rows_per_cta;                  // set by the launcher
};
omq_status act_fwd_launch(cudaStream_t st, const ActFwdArgs& a);

struct ActBwdArgs {
  int producer;
  const float* X; int64_t ldx;
  const float* U; int64_t ldu;
  const float* s; const float* delta;
  const float* rstd;
  int64_t T, C;
  const float* h; const int32_t* z; const int32_t* imax; const int32_t* imin;
  const float* dXq; int64_t lddq;
  float* dX; int64_t lddx;           // PLAIN / LET: dL/dX; RMS: dL/d(norm input); SWIGLU: d gate
  __nv_bfloat16* dXb; int64_t lddxb; // bf16 copy of dX (nullable)
  float* dU; __nv_bfloat16* dUb;     // SWIGLU: d up (same ld as dX / dXb)
  const float* resid;                // RMS: residual gradient added to dX (nullable)
  float* part_s; float* part_d;      // [T / rows_per_cta, C] LET column partials (nullable)
  float* rowdot; int64_t ldrow;      // PLAIN over [T, heads x 128] rows: D[head, t] = sum of bf16(dX) X over
                                     // the head's 128 columns, row stride ldrow (nullable; needs dXb)
  int rows_per_cta;
  int abits; float eps;
};
omq_status act_bwd_launch(cudaStream_t st, const ActBwdArgs& a);

// ---- misc ------------------------------------------------------------------------------------
// out[n] (+)= scale * sum_t X[t, n] (two-stage, deterministic); part: [ceil(T/128), N] scratch
omq_status colsum_rows(cudaStream_t st, const float* X, int64_t T, int64_t N, int64_t ldx,
                       float* part, float* out, float scale, int accumulate);
int64_t colsum_rows_parts(int64_t T);
// the same over a bf16 array (each value widened exactly); N and ldx multiples of 8
omq_status colsum_rows_bf16(cudaStream_t st, const __nv_bfloat16* X, int64_t T, int64_t N, int64_t ldx, float* part,
                            float* out, float scale, int accumulate);

omq_status loss_launch(cudaStream_t st, int64_t n, const float* Yq, const float* Yfp, float* loss,
                       float* dY, __nv_bfloat16* dYb, float* part);
int64_t loss_parts(int64_t n);

// y[i] = f(x...) small vector kernels
omq_status vec_fill(cudaStream_t st, float* p, int64_t n, float v);
omq_status vec_copy(cudaStream_t st, float* dst, const float* src, int64_t n);
// expand a per-KV-channel vector [n_kv*hd] to [n_heads*hd]; op 0: copy, 1: reciprocal
omq_status gqa_expand(cudaStream_t st, const float* src, float* dst, int n_kv, int rep, int hd, int op);
// dst[c] (+)= sum over the rep query heads of src[h*hd + j] for c = kv*hd + j
omq_status gqa_fold(cudaStream_t st, const float* src, float* dst, int n_kv, int rep, int hd, int accumulate);

// ---- LET initialisation (letinit.cu) -------------------------------------------------------------
// column max|X| and sum of X over n rows (X optionally scaled per row by rstd); first: overwrite
omq_status let_colstats(cudaStream_t st, const float* X, int64_t n, int64_t C, int64_t ldx, const float* rstd,
                        float* absmax, float* sum, int first);
omq_status let_colstats_bf16(cudaStream_t st, const __nv_bfloat16* X, int64_t n, int64_t C, int64_t ldx,
                             float* absmax, int first);
// max over output rows of |W[:, c]|
omq_status let_weight_colmax(cudaStream_t st, const __nv_bfloat16* W, int64_t Cout, int64_t Cin, float* out, int first);
// s = max(xmax^alpha / wmax^(1-alpha), floor), delta = xsum / ntok
omq_status let_smooth_pair(cudaStream_t st, int64_t C, const float* xmax, const float* xsum, const float* wmax,
                           double ntok, float alpha, float floor, float* s, float* delta);
// [v, out] and [Q, K] pairs per value channel (query-head maxima / means over each kv group)
omq_status let_kv_pairs(cudaStream_t st, int Hkv, int rep, int hd, const float* omax, const float* osum,
                        const float* womax, const float* qmax, const float* kmax, double ntok, float alpha, float floor,
                        float* so, float* do_, float* sa);

// ---- fold & pack --------------------------------------------------------------------------------
omq_status pack_codes_launch(cudaStream_t st, const uint8_t* codes, int64_t Cout, int64_t Cin, int nbits, uint8_t* out);
// gain = 1 / s, bias = -delta / s
omq_status norm_fold_launch(cudaStream_t st, int64_t n, const float* s, const float* d, float* gain, float* bias);
