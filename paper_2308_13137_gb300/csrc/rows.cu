// Per-token row kernels with the row held in registers: the activation quantizer Q_a (Eq. 2 with
// gamma = beta = 1, one group per token, Sec. 4.1) fused with its producers (LET of Eq. 3,
// RMSNorm, SwiGLU), the RoPE + [Q,K] LET (Eq. 5) + Q_a chain of q, k, v, and the straight-through
// backward of each.  One CTA walks one token row at a time; each thread owns fixed float4 vectors
// of the row (vector j*NT + tid), so a row needs no shared-memory staging, only its block
// reductions, and the LET column sums of a thread's columns accumulate in registers across rows.
#include "attn.cuh"
#include "quant.cuh"

namespace {

__device__ __forceinline__ float4 ld4(const float* p) { return __ldg(reinterpret_cast<const float4*>(p)); }
__device__ __forceinline__ float f4get(const float4& v, int e) { return e == 0 ? v.x : (e == 1 ? v.y : (e == 2 ? v.z : v.w)); }
__device__ __forceinline__ float silu(float g) { return g / (1.f + expf(-g)); }

// block-wide max and min of values; results in every thread.  smem >= 64 floats.
__device__ __forceinline__ void block_maxmin(float& M, float& m, float* smem) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = blockDim.x >> 5;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
    m = fminf(m, __shfl_xor_sync(0xffffffffu, m, off));
  }
  __syncthreads();
  if (lane == 0) { smem[wid] = M; smem[32 + wid] = m; }
  __syncthreads();
  M = lane < nw ? smem[lane] : -INFINITY;
  m = lane < nw ? smem[32 + lane] : INFINITY;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
    m = fminf(m, __shfl_xor_sync(0xffffffffu, m, off));
  }
}

// block-wide minimum of two ints; results in every thread.  smem >= 64 ints.
__device__ __forceinline__ void block_min2i(int& a, int& b, int* smem) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = blockDim.x >> 5;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    a = min(a, __shfl_xor_sync(0xffffffffu, a, off));
    b = min(b, __shfl_xor_sync(0xffffffffu, b, off));
  }
  __syncthreads();
  if (lane == 0) { smem[wid] = a; smem[32 + wid] = b; }
  __syncthreads();
  a = lane < nw ? smem[lane] : 0x7fffffff;
  b = lane < nw ? smem[32 + lane] : 0x7fffffff;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    a = min(a, __shfl_xor_sync(0xffffffffu, a, off));
    b = min(b, __shfl_xor_sync(0xffffffffu, b, off));
  }
}

__device__ __forceinline__ void st_bf16x4(__nv_bfloat16* p, const float* v) {
  uint2 u;
  __nv_bfloat162* q = reinterpret_cast<__nv_bfloat162*>(&u);
  q[0] = __floats2bfloat162_rn(v[0], v[1]);
  q[1] = __floats2bfloat162_rn(v[2], v[3]);
  *reinterpret_cast<uint2*>(p) = u;
}

// Q_a of one register-resident row: max/min values, first indices, state, fake quantization.
// val[k] holds element col[k] (col < 0: not owned).  Writes the quantized values back into val
// and the codes into cd; returns the state.
template <int NE>
__device__ __forceinline__ QState row_quantize(float (&val)[NE], const int (&col)[NE], float (&cd)[NE], float Q,
                                               float eps, int* iM_out, int* im_out, float* fsm, int* ism) {
  float M = -INFINITY, m = INFINITY;
#pragma unroll
  for (int k = 0; k < NE; ++k)
    if (col[k] >= 0) { M = fmaxf(M, val[k]); m = fminf(m, val[k]); }
  block_maxmin(M, m, fsm);
  int iM = 0x7fffffff, im = 0x7fffffff;
#pragma unroll
  for (int k = 0; k < NE; ++k)
    if (col[k] >= 0) {
      if (val[k] == M && col[k] < iM) iM = col[k];
      if (val[k] == m && col[k] < im) im = col[k];
    }
  block_min2i(iM, im, ism);
  const QState qs = omq_qstate(M, m, 1.f, 1.f, Q, eps);
#pragma unroll
  for (int k = 0; k < NE; ++k) val[k] = omq_fakequant(val[k], qs, Q, &cd[k]);
  *iM_out = iM;
  *im_out = im;
  return qs;
}

// STE pieces of one register-resident row given the saved state.  Returns the per-row routing
// amounts (added to d at the first max / min) in *GaM, *Gbt and the in-range mask in inr.
template <int NE>
__device__ __forceinline__ void row_ste(const float (&val)[NE], const int (&col)[NE], const float (&g)[NE],
                                        const QState& qs, float Q, bool (&inr)[NE], float* GaM, float* Gbt,
                                        float* fsm) {
  float Gh = 0.f, Gbm = 0.f;
#pragma unroll
  for (int k = 0; k < NE; ++k) {
    int in = 0;
    const float dh = omq_ste_dh(val[k], qs, Q, &in);
    inr[k] = in != 0;
    if (col[k] >= 0) {
      Gh = fmaf(g[k], dh, Gh);
      if (!in) Gbm += g[k];
    }
  }
  const float2 tot = block_sum2(Gh, Gbm, fsm);
  const float Gh_t = qs.floored ? 0.f : tot.x;
  *GaM = Gh_t / Q;
  *Gbt = tot.y - Gh_t / Q;
}

}  // namespace

// ================================================================================================
// activation quantizer forward: producer -> (LET) -> Q_a -> bf16
// ================================================================================================
template <int P, int NT, int VPT>
__global__ void __launch_bounds__(NT) act_fwd_rows(ActFwdArgs a) {
  constexpr int NE = 4 * VPT;
  __shared__ float fsm[64];
  __shared__ int ism[64];
  const int tid = threadIdx.x;
  const int64_t t = blockIdx.x;
  const int64_t nv = a.C / 4;
  float val[NE], cd[NE];
  int col[NE];
  const float* xr = a.X + t * a.ldx;
  float4 raw[VPT], raw2[VPT];
#pragma unroll
  for (int j = 0; j < VPT; ++j) {                     // every load of the row first
    const int64_t vi = (int64_t)j * NT + tid;
    const bool ok = vi < nv;
    raw[j] = ok ? ld4(xr + 4 * vi) : make_float4(0.f, 0.f, 0.f, 0.f);
    if (P == AP_SWIGLU) raw2[j] = ok ? ld4(a.U + t * a.ldu + 4 * vi) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int e = 0; e < 4; ++e) col[4 * j + e] = ok ? (int)(4 * vi + e) : -1;
  }
  float ss = 0.f;
#pragma unroll
  for (int j = 0; j < VPT; ++j)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      float x = f4get(raw[j], e);
      if (P == AP_SWIGLU) x = silu(x) * f4get(raw2[j], e);
      val[4 * j + e] = x;
      if (P == AP_RMS_LET) ss = fmaf(x, x, ss);
    }
  if (P == AP_RMS_LET) {
    const float2 tot = block_sum2(ss, 0.f, fsm);
    const float rstd = 1.0f / sqrtf(tot.x / (float)a.C + a.rms_eps);
    if (tid == 0 && a.rstd) a.rstd[t] = rstd;
#pragma unroll
    for (int k = 0; k < NE; ++k) val[k] = val[k] * rstd;
  }
  if (P == AP_LET || P == AP_RMS_LET) {
#pragma unroll
    for (int j = 0; j < VPT; ++j) {
      const int64_t vi = (int64_t)j * NT + tid;
      if (vi < nv) {
        const float4 dl = a.delta ? ld4(a.delta + 4 * vi) : make_float4(0.f, 0.f, 0.f, 0.f);
        const float4 sv = a.s ? ld4(a.s + 4 * vi) : make_float4(1.f, 1.f, 1.f, 1.f);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          float v = val[4 * j + e];
          if (a.delta) v = v - f4get(dl, e);
          if (a.s) v = __fdiv_rn(v, f4get(sv, e));
          val[4 * j + e] = v;
        }
      }
    }
  }
  __nv_bfloat16* qr = a.Xq + t * a.ldq;
  if (a.abits < 16) {
    const float Q = (float)((1 << a.abits) - 1);
    int iM, im;
    const QState qs = row_quantize<NE>(val, col, cd, Q, a.eps, &iM, &im, fsm, ism);
    if (tid == 0) { a.h[t] = qs.h; a.z[t] = (int32_t)qs.z; a.imax[t] = iM; a.imin[t] = im; }
  }
#pragma unroll
  for (int j = 0; j < VPT; ++j) {
    const int64_t vi = (int64_t)j * NT + tid;
    if (vi < nv) {
      st_bf16x4(qr + 4 * vi, &val[4 * j]);
      if (a.codes && a.abits < 16) {
        const uint32_t pk = (uint32_t)cd[4 * j] | ((uint32_t)cd[4 * j + 1] << 8) | ((uint32_t)cd[4 * j + 2] << 16) |
                            ((uint32_t)cd[4 * j + 3] << 24);
        *reinterpret_cast<uint32_t*>(a.codes + t * a.C + 4 * vi) = pk;
      }
    }
  }
}

// ================================================================================================
// activation quantizer backward: STE of Q_a, then the producer's backward
// ================================================================================================
template <int P, int NT, int VPT>
__global__ void __launch_bounds__(NT) act_bwd_rows(ActBwdArgs a) {
  constexpr int NE = 4 * VPT;
  __shared__ float fsm[64];
  const int tid = threadIdx.x;
  const int64_t nv = a.C / 4;
  const bool let_sums = (P != AP_SWIGLU) && a.part_s != nullptr;
  const bool quant = a.abits < 16;
  const float Q = (float)((1 << (quant ? a.abits : 1)) - 1);
  float acc_s[NE], acc_d[NE];
  int col[NE];
#pragma unroll
  for (int k = 0; k < NE; ++k) { acc_s[k] = 0.f; acc_d[k] = 0.f; }
#pragma unroll
  for (int j = 0; j < VPT; ++j) {
    const int64_t vi = (int64_t)j * NT + tid;
#pragma unroll
    for (int e = 0; e < 4; ++e) col[4 * j + e] = vi < nv ? (int)(4 * vi + e) : -1;
  }
  // X~ of one element exactly as the forward formed it
  auto xt_of = [&](int64_t t, int64_t i) -> float {
    const float* xr = a.X + t * a.ldx;
    float v;
    if (P == AP_SWIGLU) v = silu(xr[i]) * a.U[t * a.ldu + i];
    else if (P == AP_RMS_LET) v = xr[i] * a.rstd[t];
    else v = xr[i];
    if (P == AP_LET || P == AP_RMS_LET) {
      if (a.delta) v = v - a.delta[i];
      if (a.s) v = __fdiv_rn(v, a.s[i]);
    }
    return v;
  };
  const int64_t t0 = (int64_t)blockIdx.x * a.rows_per_cta;
  const int64_t t1 = min(a.T, t0 + a.rows_per_cta);
  for (int64_t t = t0; t < t1; ++t) {
    const float* xr = a.X + t * a.ldx;
    const float* gr = a.dXq + t * a.lddq;
    float val[NE], g[NE], xin[NE];
    float4 raw[VPT], graw[VPT];
#pragma unroll
    for (int j = 0; j < VPT; ++j) {                   // every load of the row first
      const int64_t vi = (int64_t)j * NT + tid;
      const bool ok = vi < nv;
      raw[j] = ok ? ld4(xr + 4 * vi) : make_float4(0.f, 0.f, 0.f, 0.f);
      graw[j] = ok ? ld4(gr + 4 * vi) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
    const float rstd = (P == AP_RMS_LET) ? a.rstd[t] : 1.f;
#pragma unroll
    for (int j = 0; j < VPT; ++j) {
      const int64_t vi = (int64_t)j * NT + tid;
      float4 uu = make_float4(0.f, 0.f, 0.f, 0.f), dl = uu, sv = make_float4(1.f, 1.f, 1.f, 1.f);
      if (vi < nv) {
        if (P == AP_SWIGLU) uu = ld4(a.U + t * a.ldu + 4 * vi);
        if ((P == AP_LET || P == AP_RMS_LET) && a.delta) dl = ld4(a.delta + 4 * vi);
        if ((P == AP_LET || P == AP_RMS_LET) && a.s) sv = ld4(a.s + 4 * vi);
      }
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int k = 4 * j + e;
        const float x = f4get(raw[j], e);
        xin[k] = x;
        float v;
        if (P == AP_SWIGLU) v = silu(x) * f4get(uu, e);
        else if (P == AP_RMS_LET) v = x * rstd;
        else v = x;
        if (P == AP_LET || P == AP_RMS_LET) {
          if (a.delta) v = v - f4get(dl, e);
          if (a.s) v = __fdiv_rn(v, f4get(sv, e));
        }
        val[k] = v;
        g[k] = f4get(graw[j], e);
      }
    }
    // STE of Q_a
    float d[NE];
    if (quant) {
      const int iM = a.imax[t], im = a.imin[t];
      const float M = xt_of(t, iM), m = xt_of(t, im);
      QState qs = omq_qstate(M, m, 1.f, 1.f, Q, a.eps);
      qs.h = a.h[t]; qs.z = (float)a.z[t]; qs.rh = __frcp_rn(qs.h); qs.u = __fmul_rn(m, qs.rh);
      bool inr[NE];
      float GaM, Gbt;
      row_ste<NE>(val, col, g, qs, Q, inr, &GaM, &Gbt, fsm);
#pragma unroll
      for (int k = 0; k < NE; ++k) {
        float dk = inr[k] ? g[k] : 0.f;
        if (col[k] == iM) dk += GaM;
        if (col[k] == im) dk += Gbt;
        d[k] = dk;
      }
    } else {
#pragma unroll
      for (int k = 0; k < NE; ++k) d[k] = g[k];
    }
    // producer backward
    float dn[NE];
    float dot = 0.f;
#pragma unroll
    for (int j = 0; j < VPT; ++j) {
      const int64_t vi = (int64_t)j * NT + tid;
      if (vi >= nv) continue;
      float sv[4] = {1.f, 1.f, 1.f, 1.f};
      if ((P == AP_LET || P == AP_RMS_LET) && a.s) {
        const float4 s4 = ld4(a.s + 4 * vi);
        sv[0] = s4.x; sv[1] = s4.y; sv[2] = s4.z; sv[3] = s4.w;
      }
      float o1[4], o2[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int k = 4 * j + e;
        if (P == AP_SWIGLU) {
          const float gg = xin[k], uu = a.U[t * a.ldu + 4 * vi + e];
          const float sg = 1.f / (1.f + expf(-gg));
          o1[e] = d[k] * uu * sg * (1.f + gg * (1.f - sg));
          o2[e] = d[k] * gg * sg;
        } else {
          if (let_sums) { acc_s[k] -= d[k] * val[k] / sv[e]; acc_d[k] -= d[k] / sv[e]; }
          const float v = (a.s && (P == AP_LET || P == AP_RMS_LET)) ? __fdiv_rn(d[k], sv[e]) : d[k];
          if (P == AP_RMS_LET) { dn[k] = v; dot = fmaf(v, xin[k] * rstd, dot); }
          o1[e] = v;
        }
      }
      if (P == AP_SWIGLU) {
        if (a.dX) {
          *reinterpret_cast<float4*>(a.dX + t * a.lddx + 4 * vi) = make_float4(o1[0], o1[1], o1[2], o1[3]);
          *reinterpret_cast<float4*>(a.dU + t * a.lddx + 4 * vi) = make_float4(o2[0], o2[1], o2[2], o2[3]);
        }
        if (a.dXb) { st_bf16x4(a.dXb + t * a.lddxb + 4 * vi, o1); st_bf16x4(a.dUb + t * a.lddxb + 4 * vi, o2); }
      } else if (P == AP_PLAIN || P == AP_LET) {
        if (a.dX) *reinterpret_cast<float4*>(a.dX + t * a.lddx + 4 * vi) = make_float4(o1[0], o1[1], o1[2], o1[3]);
        if (a.dXb) st_bf16x4(a.dXb + t * a.lddxb + 4 * vi, o1);
      }
    }
    if (P == AP_RMS_LET && (a.dX || a.dXb)) {        // RMSNorm backward
      const float2 tot = block_sum2(dot, 0.f, fsm);
      const float mean_dot = tot.x / (float)a.C;
#pragma unroll
      for (int j = 0; j < VPT; ++j) {
        const int64_t vi = (int64_t)j * NT + tid;
        if (vi >= nv) continue;
        float4 rs = make_float4(0.f, 0.f, 0.f, 0.f);
        if (a.resid) rs = ld4(a.resid + t * a.lddx + 4 * vi);
        float o[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int k = 4 * j + e;
          o[e] = rstd * (dn[k] - xin[k] * rstd * mean_dot) + f4get(rs, e);
        }
        if (a.dX) *reinterpret_cast<float4*>(a.dX + t * a.lddx + 4 * vi) = make_float4(o[0], o[1], o[2], o[3]);
        if (a.dXb) st_bf16x4(a.dXb + t * a.lddxb + 4 * vi, o);
      }
    }
  }
  if (let_sums) {
#pragma unroll
    for (int j = 0; j < VPT; ++j) {
      const int64_t vi = (int64_t)j * NT + tid;
      if (vi < nv) {
        float* ps = a.part_s + (int64_t)blockIdx.x * a.C + 4 * vi;
        float* pd = a.part_d + (int64_t)blockIdx.x * a.C + 4 * vi;
        *reinterpret_cast<float4*>(ps) = make_float4(acc_s[4 * j], acc_s[4 * j + 1], acc_s[4 * j + 2], acc_s[4 * j + 3]);
        *reinterpret_cast<float4*>(pd) = make_float4(acc_d[4 * j], acc_d[4 * j + 1], acc_d[4 * j + 2], acc_d[4 * j + 3]);
      }
    }
  }
}

// ---- launchers ---------------------------------------------------------------------------------
#define ACT_DISPATCH(KERNEL, ARGS, GRID, C)                                                          \
  do {                                                                                               \
    const int64_t nv_ = (C) / 4;                                                                     \
    if (nv_ <= 512 * 2) KERNEL<PRODUCER, 512, 2><<<(GRID), 512, 0, st>>>(ARGS);                      \
    else if (nv_ <= 512 * 4) KERNEL<PRODUCER, 512, 4><<<(GRID), 512, 0, st>>>(ARGS);                 \
    else if (nv_ <= 1024 * 4) KERNEL<PRODUCER, 1024, 4><<<(GRID), 1024, 0, st>>>(ARGS);              \
    else if (nv_ <= 1024 * 8) KERNEL<PRODUCER, 1024, 8><<<(GRID), 1024, 0, st>>>(ARGS);              \
    else return OMQ_ERR_UNSUPPORTED;                                                                 \
  } while (0)

template <int PRODUCER>
static omq_status act_fwd_dispatch(cudaStream_t st, const ActFwdArgs& a) {
  ACT_DISPATCH(act_fwd_rows, a, (unsigned)a.T, a.C);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

template <int PRODUCER>
static omq_status act_bwd_dispatch(cudaStream_t st, const ActBwdArgs& a) {
  const unsigned grid = (unsigned)((a.T + a.rows_per_cta - 1) / a.rows_per_cta);
  ACT_DISPATCH(act_bwd_rows, a, grid, a.C);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

omq_status act_fwd_launch(cudaStream_t st, const ActFwdArgs& a) {
  OMQ_REQUIRE(a.C % 8 == 0 && a.T > 0, OMQ_ERR_SHAPE);
  switch (a.producer) {
    case AP_PLAIN: return act_fwd_dispatch<AP_PLAIN>(st, a);
    case AP_LET: return act_fwd_dispatch<AP_LET>(st, a);
    case AP_RMS_LET: return act_fwd_dispatch<AP_RMS_LET>(st, a);
    case AP_SWIGLU: return act_fwd_dispatch<AP_SWIGLU>(st, a);
  }
  return OMQ_ERR_INVALID_ARG;
}

omq_status act_bwd_launch(cudaStream_t st, const ActBwdArgs& a0) {
  ActBwdArgs a = a0;
  OMQ_REQUIRE(a.C % 8 == 0 && a.T > 0, OMQ_ERR_SHAPE);
  if (a.rows_per_cta <= 0) a.rows_per_cta = 4;
  switch (a.producer) {
    case AP_PLAIN: return act_bwd_dispatch<AP_PLAIN>(st, a);
    case AP_LET: return act_bwd_dispatch<AP_LET>(st, a);
    case AP_RMS_LET: return act_bwd_dispatch<AP_RMS_LET>(st, a);
    case AP_SWIGLU: return act_bwd_dispatch<AP_SWIGLU>(st, a);
  }
  return OMQ_ERR_INVALID_ARG;
}

// ================================================================================================
// q, k, v: RoPE (rotate-half pairs), [Q, K] LET (Eq. 5: Q~ = q / s_a, K~ = k * s_a), per-token Q_a
// Each thread owns pairs p = j*NT + tid: head p/16, float4 q4 = p%16 of the first half-head and
// its partner 64 elements later, so the rotation and its transpose stay in registers.
// ================================================================================================
template <int PPT>
struct QkvRow {
  static constexpr int NE = 8 * PPT;
  float rot[NE];      // rotated projection (before s_a)
  float xt[NE];       // quantizer input
  int col[NE];        // element index in the segment (-1: not owned)
  float c[NE], sn[NE];
};

template <int NT, int PPT>
__device__ __forceinline__ void qkv_load(const QkvArgs& a, int seg, int t, QkvRow<PPT>& r) {
  const int dq = a.H * a.hd, dkv = a.Hkv * a.hd;
  const int Hs = seg == 0 ? a.H : a.Hkv;
  const int np = Hs * 16;
  const float* base = a.Y + (int64_t)t * a.ldy + (seg == 0 ? 0 : (seg == 1 ? dq : dq + dkv));
  float4 x1[PPT], x2[PPT], c4a[PPT], c4b[PPT];
#pragma unroll
  for (int j = 0; j < PPT; ++j) {                      // every load first
    const int p = j * NT + threadIdx.x;
    const bool ok = p < np;
    const int e1 = (p / 16) * 128 + 4 * (p % 16);
    const float4 z4 = make_float4(0.f, 0.f, 0.f, 0.f);
    x1[j] = ok ? ld4(base + e1) : z4;
    x2[j] = ok ? ld4(base + e1 + 64) : z4;
    const float* cs = a.cs + ((int64_t)t * 64 + 4 * (p % 16)) * 2;   // (cos, sin) of the 4 frequencies
    c4a[j] = (ok && seg < 2) ? ld4(cs) : z4;
    c4b[j] = (ok && seg < 2) ? ld4(cs + 4) : z4;
  }
#pragma unroll
  for (int j = 0; j < PPT; ++j) {
    const int p = j * NT + threadIdx.x;
    const bool ok = p < np;
    const int e1 = (p / 16) * 128 + 4 * (p % 16);
    const float cv[4] = {c4a[j].x, c4a[j].z, c4b[j].x, c4b[j].z};
    const float sv[4] = {c4a[j].y, c4a[j].w, c4b[j].y, c4b[j].w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int k1 = 8 * j + e, k2 = 8 * j + 4 + e;
      const float a1 = f4get(x1[j], e), a2 = f4get(x2[j], e);
      r.col[k1] = ok ? e1 + e : -1;
      r.col[k2] = ok ? e1 + 64 + e : -1;
      r.c[k1] = r.c[k2] = cv[e];
      r.sn[k1] = r.sn[k2] = sv[e];
      if (seg == 2) {
        r.rot[k1] = a1; r.rot[k2] = a2;
      } else {
        r.rot[k1] = a1 * cv[e] - a2 * sv[e];
        r.rot[k2] = a2 * cv[e] + a1 * sv[e];
      }
    }
  }
#pragma unroll
  for (int k = 0; k < QkvRow<PPT>::NE; ++k) {
    float v = r.rot[k];
    if (a.sa_exp && seg < 2 && r.col[k] >= 0)
      v = seg == 0 ? __fdiv_rn(v, a.sa_exp[r.col[k]]) : __fmul_rn(v, a.sa[r.col[k]]);
    r.xt[k] = v;
  }
}

template <int NT, int PPT>
__global__ void __launch_bounds__(NT) qkv_fwd_rows(QkvArgs a) {
  constexpr int NE = 8 * PPT;
  __shared__ float fsm[64];
  __shared__ int ism[64];
  const int t = blockIdx.x;
  const int dq = a.H * a.hd, dkv = a.Hkv * a.hd;
  for (int seg = 0; seg < 3; ++seg) {
    QkvRow<PPT> r;
    qkv_load<NT, PPT>(a, seg, t, r);
    const int W = seg == 0 ? dq : dkv;
    __nv_bfloat16* out = seg == 0 ? a.Qh + (int64_t)t * dq : (seg == 1 ? a.Kh + (int64_t)t * dkv : a.Vh + (int64_t)t * dkv);
    float cd[NE];
    if (a.abits < 16) {
      const float Q = (float)((1 << a.abits) - 1);
      int iM, im;
      const QState qs = row_quantize<NE>(r.xt, r.col, cd, Q, a.eps, &iM, &im, fsm, ism);
      const int64_t k = (int64_t)seg * a.T + t;
      if (threadIdx.x == 0) { a.h[k] = qs.h; a.z[k] = (int32_t)qs.z; a.imax[k] = iM; a.imin[k] = im; }
    }
#pragma unroll
    for (int j = 0; j < PPT; ++j) {
      if (r.col[8 * j] >= 0) {
        st_bf16x4(out + r.col[8 * j], &r.xt[8 * j]);
        st_bf16x4(out + r.col[8 * j + 4], &r.xt[8 * j + 4]);
      }
    }
    (void)W;
  }
}

template <int NT, int PPT>
__global__ void __launch_bounds__(NT) qkv_bwd_rows(QkvArgs a) {
  constexpr int NE = 8 * PPT;
  __shared__ float fsm[64];
  const int dq = a.H * a.hd, dkv = a.Hkv * a.hd;
  const bool sums = a.part_q != nullptr;
  float acc_q[NE], acc_k[NE];
#pragma unroll
  for (int k = 0; k < NE; ++k) { acc_q[k] = 0.f; acc_k[k] = 0.f; }
  int colq[NE], colk[NE];
  const int t0 = blockIdx.x * a.rows_per_cta, t1 = min(a.T, t0 + a.rows_per_cta);
  for (int t = t0; t < t1; ++t) {
    for (int seg = 0; seg < 3; ++seg) {
      QkvRow<PPT> r;
      qkv_load<NT, PPT>(a, seg, t, r);
      const int off = seg == 0 ? 0 : (seg == 1 ? dq : dq + dkv);
      const float* gsrc = a.dQKV + (int64_t)t * a.ldd + off;
      float g[NE], d[NE];
#pragma unroll
      for (int j = 0; j < PPT; ++j) {
        const bool ok = r.col[8 * j] >= 0;
        const float4 g1 = ok ? ld4(gsrc + r.col[8 * j]) : make_float4(0.f, 0.f, 0.f, 0.f);
        const float4 g2 = ok ? ld4(gsrc + r.col[8 * j + 4]) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int e = 0; e < 4; ++e) { g[8 * j + e] = f4get(g1, e); g[8 * j + 4 + e] = f4get(g2, e); }
      }
      if (a.abits < 16) {
        const int64_t k = (int64_t)seg * a.T + t;
        const int iM = a.imax[k], im = a.imin[k];
        const float Q = (float)((1 << a.abits) - 1);
        // the saved max / min of X~: recompute those two elements exactly as the forward did
        auto xt_at = [&](int i) -> float {
          const float* base = a.Y + (int64_t)t * a.ldy + off;
          if (seg == 2) return base[i];
          const int jj = (i % 128) % 64, first = (i % 128) < 64;
          const float cv = a.cs[((int64_t)t * 64 + jj) * 2], sv = a.cs[((int64_t)t * 64 + jj) * 2 + 1];
          const float v = first ? base[i] * cv - base[i + 64] * sv : base[i] * cv + base[i - 64] * sv;
          if (!a.sa_exp) return v;
          return seg == 0 ? __fdiv_rn(v, a.sa_exp[i]) : __fmul_rn(v, a.sa[i]);
        };
        const float M = xt_at(iM), m = xt_at(im);
        QState qs = omq_qstate(M, m, 1.f, 1.f, Q, a.eps);
        qs.h = a.h[k]; qs.z = (float)a.z[k]; qs.rh = __frcp_rn(qs.h); qs.u = __fmul_rn(m, qs.rh);
        bool inr[NE];
        float GaM, Gbt;
        row_ste<NE>(r.xt, r.col, g, qs, Q, inr, &GaM, &Gbt, fsm);
#pragma unroll
        for (int kk = 0; kk < NE; ++kk) {
          float dk = inr[kk] ? g[kk] : 0.f;
          if (r.col[kk] == iM) dk += GaM;
          if (r.col[kk] == im) dk += Gbt;
          d[kk] = dk;
        }
      } else {
#pragma unroll
        for (int kk = 0; kk < NE; ++kk) d[kk] = g[kk];
      }
      // [Q, K] LET backward and the s_a partial sums
      if (seg < 2 && a.sa_exp) {
#pragma unroll
        for (int kk = 0; kk < NE; ++kk) {
          if (r.col[kk] < 0) continue;
          if (seg == 0) {
            const float sa = a.sa_exp[r.col[kk]];
            if (sums) acc_q[kk] -= d[kk] * r.xt[kk] / sa;
            d[kk] = __fdiv_rn(d[kk], sa);
          } else {
            const float sa = a.sa[r.col[kk]];
            if (sums) acc_k[kk] += d[kk] * r.rot[kk];
            d[kk] = __fmul_rn(d[kk], sa);
          }
        }
      }
      if (seg == 0) {
#pragma unroll
        for (int kk = 0; kk < NE; ++kk) colq[kk] = r.col[kk];
      } else if (seg == 1) {
#pragma unroll
        for (int kk = 0; kk < NE; ++kk) colk[kk] = r.col[kk];
      }
      // RoPE backward: the transpose of the rotation, pair-local
      float o[NE];
#pragma unroll
      for (int j = 0; j < PPT; ++j)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int k1 = 8 * j + e, k2 = 8 * j + 4 + e;
          if (seg == 2) { o[k1] = d[k1]; o[k2] = d[k2]; }
          else {
            o[k1] = d[k1] * r.c[k1] + d[k2] * r.sn[k1];
            o[k2] = d[k2] * r.c[k1] - d[k1] * r.sn[k1];
          }
        }
      float* dy = a.dY + (int64_t)t * a.ldy + off;
      __nv_bfloat16* dyb = a.dYb + (int64_t)t * a.ldy + off;
#pragma unroll
      for (int j = 0; j < PPT; ++j) {
        if (r.col[8 * j] < 0) continue;
        const int e1 = r.col[8 * j], e2 = r.col[8 * j + 4];
        *reinterpret_cast<float4*>(dy + e1) = make_float4(o[8 * j], o[8 * j + 1], o[8 * j + 2], o[8 * j + 3]);
        *reinterpret_cast<float4*>(dy + e2) = make_float4(o[8 * j + 4], o[8 * j + 5], o[8 * j + 6], o[8 * j + 7]);
        st_bf16x4(dyb + e1, &o[8 * j]);
        st_bf16x4(dyb + e2, &o[8 * j + 4]);
      }
    }
  }
  if (sums) {
#pragma unroll
    for (int kk = 0; kk < NE; ++kk) {
      if (colq[kk] >= 0) a.part_q[(int64_t)blockIdx.x * dq + colq[kk]] = acc_q[kk];
      if (colk[kk] >= 0) a.part_k[(int64_t)blockIdx.x * dkv + colk[kk]] = acc_k[kk];
    }
  }
}

int64_t qkv_bwd_nslab(int T) { return (T + 3) / 4; }

omq_status qkv_fwd_launch(cudaStream_t st, const QkvArgs& a) {
  OMQ_REQUIRE(a.hd == 128, OMQ_ERR_UNSUPPORTED);
  const int np = a.H * 16;
  if (np <= 512) qkv_fwd_rows<512, 1><<<a.T, 512, 0, st>>>(a);
  else if (np <= 1024) qkv_fwd_rows<512, 2><<<a.T, 512, 0, st>>>(a);
  else if (np <= 2048) qkv_fwd_rows<512, 4><<<a.T, 512, 0, st>>>(a);
  else return OMQ_ERR_UNSUPPORTED;
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

omq_status qkv_bwd_launch(cudaStream_t st, const QkvArgs& a0, int64_t* nslab) {
  QkvArgs a = a0;
  OMQ_REQUIRE(a.hd == 128, OMQ_ERR_UNSUPPORTED);
  a.rows_per_cta = 4;
  const unsigned grid = (unsigned)qkv_bwd_nslab(a.T);
  const int np = a.H * 16;
  if (np <= 512) qkv_bwd_rows<512, 1><<<grid, 512, 0, st>>>(a);
  else if (np <= 1024) qkv_bwd_rows<512, 2><<<grid, 512, 0, st>>>(a);
  else if (np <= 2048) qkv_bwd_rows<512, 4><<<grid, 512, 0, st>>>(a);
  else return OMQ_ERR_UNSUPPORTED;
  OMQ_LAUNCH_CHECK();
  if (nslab) *nslab = qkv_bwd_nslab(a.T);
  return OMQ_OK;
}
