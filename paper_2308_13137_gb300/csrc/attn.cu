// Attention-side helpers: the RoPE table and the small finishers of the [v, out] LET pair
// gradients (the q/k/v row kernels live in rows.cu, the attention itself in flash.cu).
#include "attn.cuh"

#include <cmath>

// angle t * theta^(-2j/hd): the frequencies are formed on the host in double, the product and the
// reduction of the angle to [-pi, pi] in double on the device, and sin/cos of the reduced angle in
// float.  One thread per (position, frequency).
struct RopeFreq { double inv[128]; };

__global__ void rope_table_kernel(int T, int half, RopeFreq f, float* cs) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (int64_t)T * half) return;
  const int t = (int)(i / half), j = (int)(i % half);
  const double two_pi = 6.283185307179586476925286766559;
  const double inv_two_pi = 0.15915494309189533576888376337251;
  double ang = (double)t * f.inv[j];
  ang = fma(-two_pi, rint(ang * inv_two_pi), ang);
  float sv, cv;
  sincosf((float)ang, &sv, &cv);
  reinterpret_cast<float2*>(cs)[i] = make_float2(cv, sv);
}

omq_status rope_table(cudaStream_t st, int T, int hd, float theta, float* cs) {
  OMQ_REQUIRE(hd <= 256 && hd % 2 == 0, OMQ_ERR_UNSUPPORTED);
  OMQ_REQUIRE(omq_aligned16(cs), OMQ_ERR_ALIGN);
  RopeFreq f;
  const int half = hd / 2;
  for (int j = 0; j < half; ++j) f.inv[j] = std::pow((double)theta, -2.0 * (double)j / (double)hd);
  const int64_t n = (int64_t)T * half;
  rope_table_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(T, half, f, cs);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

// ------------------------------------------------------------------------------------------------
// [v, out] LET pair helpers
// ------------------------------------------------------------------------------------------------
__global__ void qkv_row_vectors_kernel(int dq, int dkv, const float* so, const float* do_, float* r, float* shift) {
  int i = blockIdx.x * blockDim.x + threadIdx.x;
  int n = dq + 2 * dkv;
  if (i >= n) return;
  int v = i - dq - dkv;
  r[i] = v >= 0 ? 1.0f / so[v] : 1.0f;
  shift[i] = v >= 0 ? do_[v] : 0.0f;
}

omq_status qkv_row_vectors(cudaStream_t st, int dq, int dkv, const float* so, const float* do_, float* r, float* shift) {
  int n = dq + 2 * dkv;
  qkv_row_vectors_kernel<<<(n + 255) / 256, 256, 0, st>>>(dq, dkv, so, do_, r, shift);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

__global__ void let_vo_finalize_kernel(int dkv, const float* so, const float* dr_v, const float* dBv, const float* Bv,
                                       float* dso, float* ddo, int accumulate) {
  int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= dkv) return;
  const float s = so[c];
  // W_v' = diag(r) W_v diag(s1) and B_v' = r (W_v d1 - d_o) with r = 1/s_o
  const float dr = dr_v[c] + dBv[c] * Bv[c] * s;     // B_v' / r = W_v d1 - d_o
  const float g_s = -dr / (s * s);
  const float g_d = -dBv[c] / s;
  dso[c] = accumulate ? dso[c] + g_s : g_s;
  ddo[c] = accumulate ? ddo[c] + g_d : g_d;
}

omq_status let_vo_finalize(cudaStream_t st, int dkv, const float* so, const float* dr_v, const float* dBv,
                           const float* Bv, float* dso, float* ddo, int accumulate) {
  let_vo_finalize_kernel<<<(dkv + 255) / 256, 256, 0, st>>>(dkv, so, dr_v, dBv, Bv, dso, ddo, accumulate);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}
