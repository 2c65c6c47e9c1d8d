// LET initialisation (Sec. 4.1 "Training": channel scales as in SmoothQuant, channel shifts as in
// Outlier Suppression+): column statistics of the full-precision block's activations over the
// calibration tokens, column maxima of the weights, and the initial s, delta, s_a from them.
// Every reduction has a fixed order (one CTA per column block, fixed row phases): deterministic.
#include "quant.cuh"

namespace {

constexpr int LI_THREADS = 256;          // 32 column lanes x 8 row phases

__device__ __forceinline__ float ldf(const float* p) { return __ldg(p); }
__device__ __forceinline__ float ldf(const __nv_bfloat16* p) { return __bfloat162float(*p); }

// absmax / sum over rows of X (optionally times rstd[row]) for 32 consecutive columns per CTA
template <typename TX>
__global__ void __launch_bounds__(LI_THREADS) colstats_kernel(const TX* __restrict__ X, int64_t n, int64_t C,
                                                              int64_t ldx, const float* __restrict__ rstd,
                                                              float* __restrict__ absmax, float* __restrict__ sum,
                                                              int first) {
  __shared__ float rm[8][33], rs[8][33];
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  const int64_t c = (int64_t)blockIdx.x * 32 + tx;
  float m = 0.f, s = 0.f;
  if (c < C)
    for (int64_t r = ty; r < n; r += 8) {
      float v = ldf(X + r * ldx + c);
      if (rstd) v *= rstd[r];
      m = fmaxf(m, fabsf(v));
      s += v;
    }
  rm[ty][tx] = m;
  rs[ty][tx] = s;
  __syncthreads();
  if (ty == 0 && c < C) {
    float M = rm[0][tx], S = rs[0][tx];
#pragma unroll
    for (int i = 1; i < 8; ++i) { M = fmaxf(M, rm[i][tx]); S += rs[i][tx]; }
    if (absmax) absmax[c] = first ? M : fmaxf(absmax[c], M);
    if (sum) sum[c] = first ? S : sum[c] + S;
  }
}

// max over output rows of |W[o, c]| for a bf16 [Cout, Cin] weight
__global__ void __launch_bounds__(LI_THREADS) weight_colmax_kernel(const __nv_bfloat16* __restrict__ W, int64_t Cout,
                                                                   int64_t Cin, float* __restrict__ out, int first) {
  __shared__ float rm[8][33];
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  const int64_t c = (int64_t)blockIdx.x * 32 + tx;
  float m = 0.f;
  if (c < Cin)
    for (int64_t o = ty; o < Cout; o += 8) m = fmaxf(m, fabsf(__bfloat162float(W[o * Cin + c])));
  rm[ty][tx] = m;
  __syncthreads();
  if (ty == 0 && c < Cin) {
    float M = rm[0][tx];
#pragma unroll
    for (int i = 1; i < 8; ++i) M = fmaxf(M, rm[i][tx]);
    out[c] = first ? M : fmaxf(out[c], M);
  }
}

__device__ __forceinline__ float smooth_scale(float xmax, float wmax, float alpha, float floor) {
  const float s = powf(xmax, alpha) / powf(wmax, 1.f - alpha);
  return s >= floor ? s : floor;          // a NaN (0 / 0) becomes the floor too
}

// s, delta of a [norm, linears] pair: one thread per channel
__global__ void smooth_pair_kernel(int64_t C, const float* xmax, const float* xsum, const float* wmax, double ntok,
                                   float alpha, float floor, float* s, float* delta) {
  const int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= C) return;
  s[c] = smooth_scale(xmax[c], wmax[c], alpha, floor);
  delta[c] = (float)((double)xsum[c] / ntok);
}

// [v, out] pair and [Q, K] pair, one thread per value channel (maxima / means over the rep query
// heads that share it)
__global__ void kv_pairs_kernel(int Hkv, int rep, int hd, const float* omax, const float* osum, const float* womax,
                                const float* qmax, const float* kmax, double ntok, float alpha, float floor,
                                float* so, float* do_, float* sa) {
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= Hkv * hd) return;
  const int g = c / hd, e = c % hd;
  float om = 0.f, wm = 0.f, qm = 0.f;
  double os = 0.0;
  for (int r = 0; r < rep; ++r) {
    const int qc = (g * rep + r) * hd + e;
    om = fmaxf(om, omax[qc]);
    wm = fmaxf(wm, womax[qc]);
    qm = fmaxf(qm, qmax[qc]);
    os += (double)osum[qc];
  }
  so[c] = smooth_scale(om, wm, alpha, floor);
  do_[c] = (float)(os / (ntok * rep));
  const float r = sqrtf(qm / kmax[c]);
  sa[c] = r >= floor ? r : floor;
}

}  // namespace

omq_status let_colstats(cudaStream_t st, const float* X, int64_t n, int64_t C, int64_t ldx, const float* rstd,
                        float* absmax, float* sum, int first) {
  colstats_kernel<float><<<(unsigned)((C + 31) / 32), LI_THREADS, 0, st>>>(X, n, C, ldx, rstd, absmax, sum, first);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

omq_status let_colstats_bf16(cudaStream_t st, const __nv_bfloat16* X, int64_t n, int64_t C, int64_t ldx,
                             float* absmax, int first) {
  colstats_kernel<__nv_bfloat16><<<(unsigned)((C + 31) / 32), LI_THREADS, 0, st>>>(X, n, C, ldx, nullptr, absmax,
                                                                                   nullptr, first);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

omq_status let_weight_colmax(cudaStream_t st, const __nv_bfloat16* W, int64_t Cout, int64_t Cin, float* out, int first) {
  weight_colmax_kernel<<<(unsigned)((Cin + 31) / 32), LI_THREADS, 0, st>>>(W, Cout, Cin, out, first);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

omq_status let_smooth_pair(cudaStream_t st, int64_t C, const float* xmax, const float* xsum, const float* wmax,
                           double ntok, float alpha, float floor, float* s, float* delta) {
  smooth_pair_kernel<<<(unsigned)((C + 255) / 256), 256, 0, st>>>(C, xmax, xsum, wmax, ntok, alpha, floor, s, delta);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

omq_status let_kv_pairs(cudaStream_t st, int Hkv, int rep, int hd, const float* omax, const float* osum,
                        const float* womax, const float* qmax, const float* kmax, double ntok, float alpha, float floor,
                        float* so, float* do_, float* sa) {
  const int n = Hkv * hd;
  kv_pairs_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(Hkv, rep, hd, omax, osum, womax, qmax, kmax, ntok, alpha,
                                                               floor, so, do_, sa);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}
