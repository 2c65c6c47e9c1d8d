// Attention-side kernels: RoPE table, RoPE + [Q,K] LET (Eq. 5) + per-token Q_a of q, k, v and
// the straight-through backward of that chain, causal softmax forward/backward on materialised
// scores, and the small finishers of the [v, out] LET pair gradients.
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
// q, k, v producer: rotary embedding (rotate-half pairs), then Q~ = q / s_a, K~ = k * s_a
// ------------------------------------------------------------------------------------------------
struct QkvVal { float rot; float xt; };

__device__ __forceinline__ QkvVal qkv_value(const QkvArgs& a, int seg, int t, int i) {
  const int dq = a.H * a.hd, dkv = a.Hkv * a.hd;
  const float* base = a.Y + (int64_t)t * a.ldy + (seg == 0 ? 0 : (seg == 1 ? dq : dq + dkv));
  QkvVal r;
  if (seg == 2) { r.rot = base[i]; r.xt = r.rot; return r; }
  const int half = a.hd / 2;
  const int j = i % a.hd;
  const int jj = j % half;
  const float c = a.cs[((int64_t)t * half + jj) * 2], s = a.cs[((int64_t)t * half + jj) * 2 + 1];
  float v;
  if (j < half) v = base[i] * c - base[i + half] * s;
  else v = base[i] * c + base[i - half] * s;
  r.rot = v;
  if (a.sa_exp) r.xt = (seg == 0) ? __fdiv_rn(v, a.sa_exp[i]) : __fmul_rn(v, a.sa[i]);
  else r.xt = v;
  return r;
}

__global__ void __launch_bounds__(512) qkv_fwd_kernel(QkvArgs a) {
  extern __shared__ float row[];
  __shared__ MaxMin red_mm[32];
  const int t = blockIdx.x, tid = threadIdx.x, nt = blockDim.x;
  const int dq = a.H * a.hd, dkv = a.Hkv * a.hd;
  for (int seg = 0; seg < 3; ++seg) {
    const int W = seg == 0 ? dq : dkv;
    __nv_bfloat16* out = seg == 0 ? a.Qh + (int64_t)t * dq : (seg == 1 ? a.Kh + (int64_t)t * dkv : a.Vh + (int64_t)t * dkv);
    MaxMin r = mm_identity();
    #pragma unroll 4
    for (int i = tid; i < W; i += nt) {
      float v = qkv_value(a, seg, t, i).xt;
      row[i] = v;
      mm_push(r, v, i);
    }
    if (a.abits >= 16) {
      __syncthreads();
      #pragma unroll 4
      for (int i = tid; i < W; i += nt) out[i] = f_to_bf16(row[i]);
      __syncthreads();
      continue;
    }
    r = mm_block_reduce(r, red_mm);
    const float Q = (float)((1 << a.abits) - 1);
    QState qs = omq_qstate(r.M, r.m, 1.f, 1.f, Q, a.eps);
    const int64_t k = (int64_t)seg * a.T + t;
    if (tid == 0) { a.h[k] = qs.h; a.z[k] = (int32_t)qs.z; a.imax[k] = r.iM; a.imin[k] = r.im; }
    #pragma unroll 4
    for (int i = tid; i < W; i += nt) {
      float c;
      out[i] = f_to_bf16(omq_fakequant(row[i], qs, Q, &c));
    }
    __syncthreads();
  }
}

omq_status qkv_fwd_launch(cudaStream_t st, const QkvArgs& a) {
  const int dq = a.H * a.hd;
  size_t smem = (size_t)dq * sizeof(float);
  OMQ_REQUIRE(smem <= 200 * 1024, OMQ_ERR_UNSUPPORTED);
  if (smem + 2048 > 48 * 1024) cudaFuncSetAttribute(qkv_fwd_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  qkv_fwd_kernel<<<a.T, 512, smem, st>>>(a);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

int64_t qkv_bwd_nslab(int T) { return (T + 3) / 4; }

__global__ void __launch_bounds__(512) qkv_bwd_kernel(QkvArgs a) {
  extern __shared__ float sm[];
  const int dq = a.H * a.hd, dkv = a.Hkv * a.hd;
  float* row = sm;            // X~ of the segment
  float* dv = sm + dq;        // dL/dX~, then dL/d(rotated)
  float* acc_q = sm + 2 * dq;
  float* acc_k = acc_q + dq;
  __shared__ float red_f[64];
  const int tid = threadIdx.x, nt = blockDim.x;
  const bool sums = a.part_q != nullptr;
  if (sums) {
    #pragma unroll 4
    for (int i = tid; i < dq; i += nt) acc_q[i] = 0.f;
    #pragma unroll 4
    for (int i = tid; i < dkv; i += nt) acc_k[i] = 0.f;
  }
  const int t0 = blockIdx.x * a.rows_per_cta, t1 = min(a.T, t0 + a.rows_per_cta);
  const int half = a.hd / 2;
  for (int t = t0; t < t1; ++t) {
    for (int seg = 0; seg < 3; ++seg) {
      const int W = seg == 0 ? dq : dkv;
      const int off = seg == 0 ? 0 : (seg == 1 ? dq : dq + dkv);
      const float* g = a.dQKV + (int64_t)t * a.ldd + off;
      #pragma unroll 4
      for (int i = tid; i < W; i += nt) row[i] = qkv_value(a, seg, t, i).xt;
      __syncthreads();
      if (a.abits >= 16) {
        #pragma unroll 4
        for (int i = tid; i < W; i += nt) dv[i] = g[i];
      } else {
        const int64_t k = (int64_t)seg * a.T + t;
        const int iM = a.imax[k], im = a.imin[k];
        const float Q = (float)((1 << a.abits) - 1);
        QState qs = omq_qstate(row[iM], row[im], 1.f, 1.f, Q, a.eps);
        qs.h = a.h[k]; qs.z = (float)a.z[k]; qs.rh = __frcp_rn(qs.h); qs.u = __fmul_rn(row[im], qs.rh);
        float Gh = 0.f, Gbm = 0.f;
        #pragma unroll 4
        for (int i = tid; i < W; i += nt) {
          int inr;
          float gi = g[i];
          float dh = omq_ste_dh(row[i], qs, Q, &inr);
          Gh = fmaf(gi, dh, Gh);
          if (!inr) Gbm += gi;
          dv[i] = inr ? gi : 0.f;
        }
        float2 tot = block_sum2(Gh, Gbm, red_f);
        Gh = qs.floored ? 0.f : tot.x;
        Gbm = tot.y;
        if (tid == 0) { dv[iM] += Gh / Q; dv[im] += Gbm - Gh / Q; }
      }
      __syncthreads();
      float* dy = a.dY + (int64_t)t * a.ldy + off;
      __nv_bfloat16* dyb = a.dYb + (int64_t)t * a.ldy + off;
      if (seg == 2) {
        #pragma unroll 4
        for (int i = tid; i < W; i += nt) { dy[i] = dv[i]; dyb[i] = f_to_bf16(dv[i]); }
        __syncthreads();
        continue;
      }
      // [Q, K] LET: gradient w.r.t. the rotated projection and the s_a partial sums
      #pragma unroll 4
      for (int i = tid; i < W; i += nt) {
        float d = dv[i];
        if (a.sa_exp) {
          if (seg == 0) {
            if (sums) acc_q[i] -= d * row[i] / a.sa_exp[i];
            d = __fdiv_rn(d, a.sa_exp[i]);
          } else {
            if (sums) acc_k[i] += d * __fdiv_rn(row[i], a.sa[i]);
            d = __fmul_rn(d, a.sa[i]);
          }
        }
        dv[i] = d;
      }
      __syncthreads();
      // RoPE backward: the transpose of the rotation
      #pragma unroll 4
      for (int i = tid; i < W; i += nt) {
        const int j = i % a.hd, jj = j % half;
        const float c = a.cs[((int64_t)t * half + jj) * 2], s = a.cs[((int64_t)t * half + jj) * 2 + 1];
        float r = (j < half) ? dv[i] * c + dv[i + half] * s : dv[i] * c - dv[i - half] * s;
        dy[i] = r;
        dyb[i] = f_to_bf16(r);
      }
      __syncthreads();
    }
  }
  if (sums) {
    #pragma unroll 4
    for (int i = tid; i < dq; i += nt) a.part_q[(int64_t)blockIdx.x * dq + i] = acc_q[i];
    #pragma unroll 4
    for (int i = tid; i < dkv; i += nt) a.part_k[(int64_t)blockIdx.x * dkv + i] = acc_k[i];
  }
}

omq_status qkv_bwd_launch(cudaStream_t st, const QkvArgs& a0, int64_t* nslab) {
  QkvArgs a = a0;
  a.rows_per_cta = 4;
  const int dq = a.H * a.hd, dkv = a.Hkv * a.hd;
  size_t smem = (size_t)(2 * dq + (a.part_q ? dq + dkv : 0)) * sizeof(float);
  OMQ_REQUIRE(smem <= 200 * 1024, OMQ_ERR_UNSUPPORTED);
  if (smem + 2048 > 48 * 1024) cudaFuncSetAttribute(qkv_bwd_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  qkv_bwd_kernel<<<(unsigned)qkv_bwd_nslab(a.T), 512, smem, st>>>(a);
  OMQ_LAUNCH_CHECK();
  if (nslab) *nslab = qkv_bwd_nslab(a.T);
  return OMQ_OK;
}

// ------------------------------------------------------------------------------------------------
// causal softmax on materialised scores: one warp per query row
// ------------------------------------------------------------------------------------------------
__global__ void softmax_fwd_kernel(int B, int T, const float* __restrict__ S, __nv_bfloat16* __restrict__ P) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t r = (int64_t)blockIdx.x * (blockDim.x >> 5) + warp;
  if (r >= (int64_t)B * T) return;
  const int t = (int)(r % T);
  const float* s = S + r * T;
  __nv_bfloat16* p = P + r * T;
  float mx = -INFINITY;
  for (int j = lane; j <= t; j += 32) mx = fmaxf(mx, s[j]);
  for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
  float sum = 0.f;
  for (int j = lane; j <= t; j += 32) sum += expf(s[j] - mx);
  sum = warp_sum(sum);
  const float inv = 1.0f / sum;
  const int kend = min(T, (t / 128 + 1) * 128);
  for (int j = lane; j < kend; j += 32) p[j] = f_to_bf16(j <= t ? expf(s[j] - mx) * inv : 0.f);
}

omq_status softmax_fwd_launch(cudaStream_t st, int B, int T, const float* S, __nv_bfloat16* P) {
  int64_t rows = (int64_t)B * T;
  softmax_fwd_kernel<<<(unsigned)((rows + 7) / 8), 256, 0, st>>>(B, T, S, P);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

__global__ void softmax_bwd_kernel(int B, int T, const __nv_bfloat16* __restrict__ P, const float* __restrict__ dP,
                                   float scale, __nv_bfloat16* __restrict__ dS) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t r = (int64_t)blockIdx.x * (blockDim.x >> 5) + warp;
  if (r >= (int64_t)B * T) return;
  const int t = (int)(r % T);
  const __nv_bfloat16* p = P + r * T;
  const float* dp = dP + r * T;
  __nv_bfloat16* ds = dS + r * T;
  float D = 0.f;
  for (int j = lane; j <= t; j += 32) D = fmaf(bf16_to_f(p[j]), dp[j], D);
  D = warp_sum(D);
  const int kend = min(T, (t / 128 + 1) * 128);
  for (int j = lane; j < kend; j += 32) ds[j] = f_to_bf16(j <= t ? scale * bf16_to_f(p[j]) * (dp[j] - D) : 0.f);
}

omq_status softmax_bwd_launch(cudaStream_t st, int B, int T, const __nv_bfloat16* P, const float* dP, float scale,
                              __nv_bfloat16* dS) {
  int64_t rows = (int64_t)B * T;
  softmax_bwd_kernel<<<(unsigned)((rows + 7) / 8), 256, 0, st>>>(B, T, P, dP, scale, dS);
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
