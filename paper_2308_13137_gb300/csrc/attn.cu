// Attention-side helpers: the RoPE table and the small finishers of the [v, out] LET pair
// gradients (the q/k/v row kernels live in rows.cu, the attention itself in flash.cu).
#include "attn.cuh"

// angle t * theta^(-2j/hd): the frequency and the product are formed in double, the angle is reduced
// to [-pi, pi] in double, and sin/cos of the reduced angle are taken in float.
__global__ void rope_table_kernel(int T, int hd, double theta, float* cs) {
  __shared__ double inv[128];
  const int half = hd / 2;
  for (int j = threadIdx.x; j < half; j += blockDim.x) inv[j] = pow(theta, -2.0 * (double)j / (double)hd);
  __syncthreads();
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= T * half) return;
  const int t = i / half, j = i % half;
  const double two_pi = 6.283185307179586476925286766559;
  double ang = (double)t * inv[j];
  ang -= two_pi * rint(ang / two_pi);
  float sv, cv;
  sincosf((float)ang, &sv, &cv);
  cs[2 * i] = cv;
  cs[2 * i + 1] = sv;
}

omq_status rope_table(cudaStream_t st, int T, int hd, float theta, float* cs) {
  OMQ_REQUIRE(hd <= 256, OMQ_ERR_UNSUPPORTED);
  int n = T * (hd / 2);
  rope_table_kernel<<<(n + 255) / 256, 256, 0, st>>>(T, hd, (double)theta, cs);
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
