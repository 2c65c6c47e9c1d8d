// Per-token row kernels with the row held in registers: the activation quantizer Q_a (Eq. 2 with
// gamma = beta = 1, one group per token, Sec. 4.1) fused with its producers (LET of Eq. 3,
// RMSNorm, SwiGLU), the RoPE + [Q,K] LET (Eq. 5) + Q_a chain of q, k, v, and the straight-through
// backward of each.  One CTA walks one token row at a time; each thread owns fixed float4 vectors
// of the row (vector j*NT + tid), so a row needs no shared-memory staging, only its block
// reductions, and the LET column sums of a thread's columns accumulate in registers across rows.
#include "attn.cuh"
#include "quant.cuh"
#include "tc.cuh"

#include <algorithm>

namespace {

__device__ __forceinline__ float4 ld4(const float* p) { return __ldg(reinterpret_cast<const float4*>(p)); }
__device__ __forceinline__ float f4get(const float4& v, int e) { return e == 0 ? v.x : (e == 1 ? v.y : (e == 2 ? v.z : v.w)); }
// silu(g) = g sigmoid(g); the quotient by the correctly rounded reciprocal (one rounding more than
// an IEEE division: within 1 ulp of g / (1 + e^-g)); the forward and the backward's recomputation of
// the quantizer input both use this form
__device__ __forceinline__ float silu(float g) { return g * __frcp_rn(1.f + expf(-g)); }

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
  static_assert(NE % 2 == 0, "elements are quantized in pairs");
  float M = -INFINITY, m = INFINITY;
#pragma unroll
  for (int k = 0; k < NE; ++k)
    if (col[k] >= 0) { M = fmaxf(M, val[k]); m = fminf(m, val[k]); }
  const float lM = M, lm = m;                    // this thread's own extremes
  block_maxmin(M, m, fsm);
  int iM = 0x7fffffff, im = 0x7fffffff;
  if (lM == M || lm == m) {                      // only the holders of an extreme search its first index
#pragma unroll
    for (int k = 0; k < NE; ++k)
      if (col[k] >= 0) {
        if (val[k] == M && col[k] < iM) iM = col[k];
        if (val[k] == m && col[k] < im) im = col[k];
      }
  }
  block_min2i(iM, im, ism);
  const QState qs = omq_qstate(M, m, 1.f, 1.f, Q, eps);
#pragma unroll
  for (int k = 0; k < NE; k += 2) {
    float2 c2;
    const float2 v = omq_fakequant2(make_float2(val[k], val[k + 1]), qs, Q, &c2);
    val[k] = v.x; val[k + 1] = v.y; cd[k] = c2.x; cd[k + 1] = c2.y;
  }
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
// one token row t of the activation quantizer forward, held in registers
template <int P, int NT, int VPT>
__device__ __forceinline__ void act_fwd_row(const ActFwdArgs& a, const int64_t t, float* fsm, int* ism) {
  constexpr int NE = 4 * VPT;
  const int tid = threadIdx.x;
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


// token rows per CTA of the register-resident forward (rows of up to 4 K columns; the SwiGLU row)
// and of the q, k, v quantizer forward
constexpr int kFwdRows = 2, kFwdRowsSwiglu = 2, kQkvFwdRows = 1;

// rows blockIdx.x * R .. + R - 1 (R = a.rows_per_cta, at least 1); the CTA prefetches each next row's
// inputs into L2 while it works on the current one
template <int P, int NT, int VPT>
__global__ void __launch_bounds__(NT) act_fwd_rows(ActFwdArgs a) {
  __shared__ float fsm[64];
  __shared__ int ism[64];
  const int64_t R = a.rows_per_cta > 1 ? a.rows_per_cta : 1;
  const int64_t t0 = (int64_t)blockIdx.x * R, t1 = t0 + R < a.T ? t0 + R : a.T;
  for (int64_t t = t0; t < t1; ++t) {
    if (threadIdx.x == 0 && t + 1 < t1) {
      omq_l2_prefetch(a.X + (t + 1) * a.ldx, (uint64_t)a.C * 4);
      if (P == AP_SWIGLU) omq_l2_prefetch(a.U + (t + 1) * a.ldu, (uint64_t)a.C * 4);
    }
    act_fwd_row<P, NT, VPT>(a, t, fsm, ism);
    __syncthreads();                           // the reduction scratch is reused by the next row
  }
}
// ================================================================================================
// activation quantizer forward, staged: a persistent CTA walks the rows blockIdx.x, + gridDim.x, ...
// and the bulk-copy engine brings each row's inputs into a ring of `stages` shared-memory buffers
// (cp.async.bulk completing on one mbarrier per buffer) while the CTA works on earlier rows, so
// the row's HBM latency is hidden behind the compute and the block reductions of the rows before
// it.  The arithmetic on each element is act_fwd_rows's.  Waits are bounded: on expiry the status
// word is set, the CTA waits (again bounded) for the copies it issued and returns.
// ================================================================================================
template <int P, int NT, int VPT>
__global__ void __launch_bounds__(NT) act_fwd_staged(ActFwdArgs a, int stages) {
  constexpr int NE = 4 * VPT, NW = NT / 32, MAXS = 4;
  constexpr int NIN = P == AP_SWIGLU ? 2 : 1;
  extern __shared__ float4 stg4[];                 // [stages][NIN][C / 4]
  __shared__ uint64_t bar[MAXS];
  __shared__ float red[3][NW];
  __shared__ int sidx[2];
  __shared__ int abort_flag;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t nv = a.C / 4;
  const uint32_t row_bytes = (uint32_t)(a.C * 4);
  const bool quant = a.abits < 16;
  const float Q = (float)((1 << (quant ? a.abits : 1)) - 1);
  if (tid == 0) {
    for (int s = 0; s < stages; ++s) tc::mbar_init(&bar[s], 1);
    sidx[0] = 0x7fffffff; sidx[1] = 0x7fffffff;
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  int64_t issued = 0;                              // rows whose copies thread 0 has issued
  auto issue = [&](int64_t k) {
    const int64_t t = blockIdx.x + k * gridDim.x;
    if (t >= a.T) return;
    const int s = (int)(k % stages);
    float4* dst = stg4 + (size_t)s * NIN * nv;
    tc::mbar_expect_tx(&bar[s], NIN * row_bytes);
    tc::bulk_g2s(dst, a.X + t * a.ldx, row_bytes, &bar[s]);
    if (P == AP_SWIGLU) tc::bulk_g2s(dst + nv, a.U + t * a.ldu, row_bytes, &bar[s]);
    issued = k + 1;
  };
  if (tid == 0)
    for (int k = 0; k < stages; ++k) issue(k);
  int64_t k = 0;
  for (;; ++k) {
    const int64_t t = blockIdx.x + k * gridDim.x;
    if (t >= a.T) break;
    const int s = (int)(k % stages);
    if (!tc::mbar_wait(&bar[s], (uint32_t)((k / stages) & 1))) {
      omq_set_status(a.status, OMQ_ERR_TIMEOUT);
      abort_flag = 1;
    }
    const float4* xs = stg4 + (size_t)s * NIN * nv;
    float val[NE];
    float ss = 0.f;
#pragma unroll
    for (int j = 0; j < VPT; ++j) {
      const int64_t vi = (int64_t)j * NT + tid;
      const float4 xv = vi < nv ? xs[vi] : make_float4(0.f, 0.f, 0.f, 0.f);
      float4 uv = make_float4(0.f, 0.f, 0.f, 0.f);
      if (P == AP_SWIGLU && vi < nv) uv = xs[nv + vi];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        float x = f4get(xv, e);
        if (P == AP_SWIGLU) x = silu(x) * f4get(uv, e);
        val[4 * j + e] = x;
        if (P == AP_RMS_LET) ss = fmaf(x, x, ss);
      }
    }
    if (P == AP_RMS_LET) {                          // the summation tree of block_sum2
      ss = warp_sum(ss);
      if (lane == 0) red[0][warp] = ss;
      __syncthreads();
      const float tot = warp_sum(lane < NW ? red[0][lane] : 0.f);
      const float rstd = 1.0f / sqrtf(tot / (float)a.C + a.rms_eps);
      if (tid == 0 && a.rstd) a.rstd[t] = rstd;
#pragma unroll
      for (int k2 = 0; k2 < NE; ++k2) val[k2] = val[k2] * rstd;
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
    QState qs;
    if (quant) {
      float M = -INFINITY, m = INFINITY;
#pragma unroll
      for (int j = 0; j < VPT; ++j)
        if ((int64_t)j * NT + tid < nv)
#pragma unroll
          for (int e = 0; e < 4; ++e) { M = fmaxf(M, val[4 * j + e]); m = fminf(m, val[4 * j + e]); }
      float bM = M, bm = m;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        bM = fmaxf(bM, __shfl_xor_sync(0xffffffffu, bM, off));
        bm = fminf(bm, __shfl_xor_sync(0xffffffffu, bm, off));
      }
      if (lane == 0) { red[1][warp] = bM; red[2][warp] = bm; }
      __syncthreads();
      bM = red[1][0]; bm = red[2][0];
#pragma unroll
      for (int w = 1; w < NW; ++w) { bM = fmaxf(bM, red[1][w]); bm = fminf(bm, red[2][w]); }
      if (M == bM || m == bm) {                   // the first index, searched by the holders only
        int iM = 0x7fffffff, im = 0x7fffffff;
#pragma unroll
        for (int j = VPT - 1; j >= 0; --j) {
          const int64_t vi = (int64_t)j * NT + tid;
          if (vi < nv)
#pragma unroll
            for (int e = 3; e >= 0; --e) {
              if (val[4 * j + e] == bM) iM = (int)(4 * vi + e);
              if (val[4 * j + e] == bm) im = (int)(4 * vi + e);
            }
        }
        if (iM != 0x7fffffff) atomicMin(&sidx[0], iM);
        if (im != 0x7fffffff) atomicMin(&sidx[1], im);
      }
      qs = omq_qstate(bM, bm, 1.f, 1.f, Q, a.eps);
    }
    __nv_bfloat16* qr = a.Xq + t * a.ldq;
#pragma unroll
    for (int j = 0; j < VPT; ++j) {
      const int64_t vi = (int64_t)j * NT + tid;
      if (vi < nv) {
        float o[4], cd[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) o[e] = quant ? omq_fakequant(val[4 * j + e], qs, Q, &cd[e]) : val[4 * j + e];
        st_bf16x4(qr + 4 * vi, o);
        if (a.codes && quant) {
          const uint32_t pk = (uint32_t)cd[0] | ((uint32_t)cd[1] << 8) | ((uint32_t)cd[2] << 16) | ((uint32_t)cd[3] << 24);
          *reinterpret_cast<uint32_t*>(a.codes + t * a.C + 4 * vi) = pk;
        }
      }
    }
    __syncthreads();                               // buffer s read by every thread; first indices final
    if (tid == 0) {
      if (quant) {
        a.h[t] = qs.h; a.z[t] = (int32_t)qs.z; a.imax[t] = sidx[0]; a.imin[t] = sidx[1];
        sidx[0] = 0x7fffffff; sidx[1] = 0x7fffffff;
      }
      if (!abort_flag) {
        tc::fence_async_smem();                    // generic reads of buffer s before the copy engine refills it
        issue(k + stages);
      }
    }
    if (abort_flag) break;
  }
  if (tid == 0 && abort_flag)                      // rows k .. issued - 1 may still be in flight: let them land
    for (int64_t r = k; r < issued; ++r) tc::mbar_wait(&bar[r % stages], (uint32_t)((r / stages) & 1));
}

// ================================================================================================
// activation quantizer backward: STE of Q_a, then the producer's backward, streamed.
// The STE gradient of a token is the in-range mask times the incoming gradient everywhere except
// at the first max / min, which also receive the h-path routing (a row sum).  So one streaming
// pass writes every output with the masked gradient and accumulates the row sums; after one block
// reduction the owners of the two routed elements rewrite them.  Only RMSNorm, whose backward
// needs the row dot product of the final gradient, streams the row a second time (from L2).
// 256 threads, low register count: several CTAs (rows) per SM hide the load latency.  CTA p
// handles rows [p * rows_per_cta, ...) and writes LET column partial p.
// ================================================================================================
#define ACT_BWD_NT 256

__device__ __forceinline__ float3 block_sum3(float a, float b, float c, float* smem) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  a = warp_sum(a); b = warp_sum(b); c = warp_sum(c);
  __syncthreads();
  if (lane == 0) { smem[wid] = a; smem[32 + wid] = b; smem[64 + wid] = c; }
  __syncthreads();
  float x = lane < nw ? smem[lane] : 0.f, y = lane < nw ? smem[32 + lane] : 0.f, z = lane < nw ? smem[64 + lane] : 0.f;
  return make_float3(warp_sum(x), warp_sum(y), warp_sum(z));
}

// o . d over one float4 group, in the order of the attention backward's own row dot
__device__ __forceinline__ float rowdot4(const float4 o, const float (&d)[4]) {
  return o.x * d[0] + o.y * d[1] + o.z * d[2] + o.w * d[3];
}

template <int P>
struct ActBwdRow {
  const ActBwdArgs& a;
  int64_t t;
  float rstd;
  // X~ of one element from the producer's inputs (exactly as the forward formed it)
  __device__ __forceinline__ float xt(float x, float u, float dl, float sv) const {
    float v;
    if (P == AP_SWIGLU) v = silu(x) * u;
    else if (P == AP_RMS_LET) v = x * rstd;
    else v = x;
    if (P == AP_LET || P == AP_RMS_LET) {
      if (a.delta) v = v - dl;
      if (a.s) v = __fdiv_rn(v, sv);
    }
    return v;
  }
  __device__ __forceinline__ float xt_at(int64_t i) const {
    const float x = a.X[t * a.ldx + i];
    const float u = (P == AP_SWIGLU) ? a.U[t * a.ldu + i] : 0.f;
    const float dl = ((P == AP_LET || P == AP_RMS_LET) && a.delta) ? a.delta[i] : 0.f;
    const float sv = ((P == AP_LET || P == AP_RMS_LET) && a.s) ? a.s[i] : 1.f;
    return xt(x, u, dl, sv);
  }
};

template <int P, int VPT, int JB, int MINB, bool SUMS, bool RD = false>
__global__ void __launch_bounds__(ACT_BWD_NT, MINB) act_bwd_stream(ActBwdArgs a) {
  constexpr int NT = ACT_BWD_NT;
  constexpr bool LETP = (P == AP_LET || P == AP_RMS_LET);
  static_assert(!(SUMS && P == AP_SWIGLU), "SwiGLU has no LET column sums");
  constexpr int NE = SUMS ? 4 * VPT : 1;
  __shared__ float fsm[96];
  const int tid = threadIdx.x;
  const int64_t nv = a.C / 4;
  constexpr bool let_sums = SUMS;
  const bool quant = a.abits < 16;
  const float Q = (float)((1 << (quant ? a.abits : 1)) - 1);
  const bool want_out = a.dX != nullptr || a.dXb != nullptr;
  const int64_t nparts = (a.T + a.rows_per_cta - 1) / a.rows_per_cta;
  const float4 z4 = make_float4(0.f, 0.f, 0.f, 0.f), o4 = make_float4(1.f, 1.f, 1.f, 1.f);
  float acc_s[NE], acc_d[NE];
  // with column sums and rows of at most 8 K: 1/s of the thread's columns in shared memory (each
  // thread reads back only its own slots), computed once; the RMSNorm backward also keeps x * rstd
  // and the masked gradient of its elements in registers for pass 2
  constexpr bool RS = SUMS && VPT <= 8;
  constexpr bool KEEP = RS && P == AP_RMS_LET;
  // the plain form with a.rowdot: D[head, t] = the sum of bf16(dX) X over each 128-column head (the
  // attention backward's rowsum(dO * O)), taken while the row is here; the float4 group j of a warp
  // is one head (lane L holds its columns 4L .. 4L + 3)
  static_assert(!RD || (P == AP_PLAIN && !SUMS), "the row dot is a form of the plain producer");
  float dpart[RD ? VPT : 1];
  __shared__ float4 rs_sm[RS ? VPT * NT : 1];
  float xk[KEEP ? NE : 1], dk[KEEP ? NE : 1];
#pragma unroll
  for (int j = 0; j < (RS ? VPT : 0); ++j) {
    const int64_t vi = (int64_t)j * NT + tid;
    const float4 sv = (LETP && a.s && vi < nv) ? ld4(a.s + 4 * vi) : o4;
    rs_sm[j * NT + tid] = make_float4(__frcp_rn(sv.x), __frcp_rn(sv.y), __frcp_rn(sv.z), __frcp_rn(sv.w));
  }
  for (int64_t p = blockIdx.x; p < nparts; p += gridDim.x) {
#pragma unroll
    for (int k = 0; k < NE; ++k) { acc_s[k] = 0.f; acc_d[k] = 0.f; }
    const int64_t t0 = p * a.rows_per_cta, t1 = min(a.T, t0 + a.rows_per_cta);
    for (int64_t t = t0; t < t1; ++t) {
      if (tid == 0) {                          // the next row's inputs (and this row's residual) into L2
        const uint64_t rb = (uint64_t)a.C * 4;
        if (P == AP_RMS_LET && a.resid) omq_l2_prefetch(a.resid + t * a.lddx, rb);
        if (t + 1 < t1) {
          omq_l2_prefetch(a.X + (t + 1) * a.ldx, rb);
          omq_l2_prefetch(a.dXq + (t + 1) * a.lddq, rb);
          if (P == AP_SWIGLU) omq_l2_prefetch(a.U + (t + 1) * a.ldu, rb);
          if (P == AP_RMS_LET && a.resid) omq_l2_prefetch(a.resid + (t + 1) * a.lddx, rb);
        }
      }
      ActBwdRow<P> R{a, t, (P == AP_RMS_LET) ? a.rstd[t] : 1.f};
      const float* xr = a.X + t * a.ldx;
      const float* gr = a.dXq + t * a.lddq;
      const float* ur = (P == AP_SWIGLU) ? a.U + t * a.ldu : nullptr;
      QState qs;
      int iM = -1, im = -1;
      if (quant) {
        iM = a.imax[t]; im = a.imin[t];
        qs = omq_qstate(R.xt_at(iM), R.xt_at(im), 1.f, 1.f, Q, a.eps);
        qs.h = a.h[t]; qs.z = (float)a.z[t]; qs.rh = __frcp_rn(qs.h); qs.u = __fmul_rn(qs.m, qs.rh);
      }
      float Gh = 0.f, Gbm = 0.f, dot = 0.f;
      // ---- pass 1: masked gradient through the producer, row sums ----
#pragma unroll
      for (int jb = 0; jb < VPT; jb += JB) {
        float4 x4[JB], g4[JB], u4[JB];
#pragma unroll
        for (int jj = 0; jj < JB; ++jj) {               // every load of the batch first
          const int64_t vi = (int64_t)(jb + jj) * NT + tid;
          const bool ok = jb + jj < VPT && vi < nv;
          x4[jj] = ok ? ld4(xr + 4 * vi) : z4;
          g4[jj] = ok ? ld4(gr + 4 * vi) : z4;
          u4[jj] = (P == AP_SWIGLU && ok) ? ld4(ur + 4 * vi) : z4;
        }
#pragma unroll
        for (int jj = 0; jj < JB; ++jj) {
          const int j = jb + jj;
          const int64_t vi = (int64_t)j * NT + tid;
          if (j >= VPT || vi >= nv) continue;
          float4 dl = z4, sv = o4;
          if (LETP && a.delta) dl = ld4(a.delta + 4 * vi);
          if (LETP && a.s) sv = ld4(a.s + 4 * vi);
          const float4 rs4 = RS ? rs_sm[j * NT + tid] : o4;
          float o1[4], o2[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float x = f4get(x4[jj], e), g = f4get(g4[jj], e), se = f4get(sv, e);
            const float v = R.xt(x, f4get(u4[jj], e), f4get(dl, e), se);
            float d = g;
            if (quant) {
              int in = 0;
              const float dh = omq_ste_dh(v, qs, Q, &in);
              Gh = fmaf(g, dh, Gh);
              if (!in) { Gbm += g; d = 0.f; }
            }
            if (P == AP_SWIGLU) {
              const float uu = f4get(u4[jj], e);
              const float sg = 1.f / (1.f + expf(-x));
              o1[e] = d * uu * sg * (1.f + x * (1.f - sg));
              o2[e] = d * x * sg;
            } else {
              if (SUMS && let_sums) {            // divided by s once, when the partial is written
                const int k = 4 * j + e;
                acc_s[k] = fmaf(d, v, acc_s[k]);
                acc_d[k] += d;
              }
              const int k = (4 * j + e) % NE;
              const float rcp = RS ? f4get(rs4, e) : __frcp_rn(se);
              const float dn = (LETP && a.s) ? d * rcp : d;
              if (P == AP_RMS_LET) dot = fmaf(dn, x * R.rstd, dot);
              if (KEEP) { xk[k] = x * R.rstd; dk[k] = dn; }
              o1[e] = dn;
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
            if constexpr (RD) {   // C % 128 == 0: the whole warp is here
              float b4[4];
#pragma unroll
              for (int e = 0; e < 4; ++e) b4[e] = __bfloat162float(__float2bfloat16_rn(o1[e]));
              dpart[j] = rowdot4(x4[jj], b4);
            }
          }
        }
      }
      if constexpr (RD) {
#pragma unroll
        for (int j = 0; j < VPT; ++j) {
          const int64_t v0 = (int64_t)j * NT + (tid & ~31);   // the head's first float4 (warp-uniform)
          if (v0 >= nv) break;
          const float sd = warp_sum(dpart[j]);
          if ((tid & 31) == 0) a.rowdot[(v0 >> 5) * a.ldrow + t] = sd;
        }
      }
      if (!quant && !(P == AP_RMS_LET && want_out)) continue;
      const float3 tot = block_sum3(Gh, Gbm, dot, fsm);
      float GaM = 0.f, Gbt = 0.f;
      if (quant) {
        const float Gh_t = qs.floored ? 0.f : tot.x;
        GaM = Gh_t / Q;
        Gbt = tot.y - Gh_t / Q;
      }
      // ---- the routed elements: their owners rewrite them ----
      float dot_t = tot.z;
      if (quant) {
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          const int64_t c = r == 0 ? iM : im;
          if (r == 1 && im == iM) break;
          const float route = (im == iM) ? GaM + Gbt : (r == 0 ? GaM : Gbt);
          const float x = xr[c], g = gr[c];
          const float se = (LETP && a.s) ? a.s[c] : 1.f;
          const float v = R.xt_at(c);
          int in = 0;
          omq_ste_dh(v, qs, Q, &in);
          const float d = (in ? g : 0.f) + route;
          if (P == AP_RMS_LET) dot_t = fmaf((a.s ? __fdiv_rn(route, se) : route), x * R.rstd, dot_t);
          if ((c >> 2) % NT != tid) continue;
          if (P == AP_SWIGLU) {
            const float uu = ur[c];
            const float sg = 1.f / (1.f + expf(-x));
            const float v1 = d * uu * sg * (1.f + x * (1.f - sg)), v2 = d * x * sg;
            if (a.dX) { a.dX[t * a.lddx + c] = v1; a.dU[t * a.lddx + c] = v2; }
            if (a.dXb) { a.dXb[t * a.lddxb + c] = f_to_bf16(v1); a.dUb[t * a.lddxb + c] = f_to_bf16(v2); }
          } else {
            if (let_sums) {
#pragma unroll
              for (int k = 0; k < NE; ++k)
                if (4 * ((int64_t)(k >> 2) * NT + tid) + (k & 3) == c) {
                  acc_s[k] = fmaf(route, v, acc_s[k]);
                  acc_d[k] += route;
                }
            }
            if (P == AP_PLAIN || P == AP_LET) {
              const float dn = (LETP && a.s) ? __fdiv_rn(d, se) : d;
              if (a.dX) a.dX[t * a.lddx + c] = dn;
              if (a.dXb) a.dXb[t * a.lddxb + c] = f_to_bf16(dn);
            }
          }
        }
        if constexpr (RD) {     // the heads of the routed elements, summed again
          __syncwarp();                                  // the owner's rewrite, seen by its warp
#pragma unroll
          for (int r = 0; r < 2; ++r) {
            const int64_t c = r == 0 ? iM : im;
            if (r == 1 && (im >> 7) == (iM >> 7)) break;
            const int64_t v0 = (c >> 2) & ~(int64_t)31;    // the head's first float4
            if ((int)((v0 % NT) >> 5) != (tid >> 5)) continue;
            const int64_t vi = v0 + (tid & 31);
            const uint2 u = *reinterpret_cast<const uint2*>(a.dXb + t * a.lddxb + 4 * vi);
            const float2 b01 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.x));
            const float2 b23 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.y));
            const float b4[4] = {b01.x, b01.y, b23.x, b23.y};
            const float sd = warp_sum(rowdot4(ld4(xr + 4 * vi), b4));
            if ((tid & 31) == 0) a.rowdot[(v0 >> 5) * a.ldrow + t] = sd;
          }
        }
      }
      // ---- RMSNorm backward: second stream of the row ----
      if (KEEP && want_out) {                    // x * rstd and dn kept from pass 1: only resid is read
        const float mean_dot = dot_t / (float)a.C;
#pragma unroll
        for (int jb = 0; jb < VPT; jb += JB) {
          float4 r4[JB];
#pragma unroll
          for (int jj = 0; jj < JB; ++jj) {
            const int64_t vi = (int64_t)(jb + jj) * NT + tid;
            r4[jj] = (jb + jj < VPT && vi < nv && a.resid) ? ld4(a.resid + t * a.lddx + 4 * vi) : z4;
          }
#pragma unroll
          for (int jj = 0; jj < JB; ++jj) {
            const int j = jb + jj;
            const int64_t vi = (int64_t)j * NT + tid;
            if (j >= VPT || vi >= nv) continue;
            float o[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const int k = (4 * j + e) % NE;
              const int64_t c = 4 * vi + e;
              float dn = dk[k];
              if (c == iM || c == im) {
                const float rc = f4get(rs_sm[j * NT + tid], e);
                if (c == iM) dn = fmaf(GaM, rc, dn);
                if (c == im) dn = fmaf(Gbt, rc, dn);
              }
              o[e] = R.rstd * (dn - xk[k] * mean_dot) + f4get(r4[jj], e);
            }
            if (a.dX) *reinterpret_cast<float4*>(a.dX + t * a.lddx + 4 * vi) = make_float4(o[0], o[1], o[2], o[3]);
            if (a.dXb) st_bf16x4(a.dXb + t * a.lddxb + 4 * vi, o);
          }
        }
      } else if (P == AP_RMS_LET && want_out) {
        const float mean_dot = dot_t / (float)a.C;
#pragma unroll
        for (int jb = 0; jb < VPT; jb += JB) {
          float4 x4[JB], g4[JB], r4[JB];
#pragma unroll
          for (int jj = 0; jj < JB; ++jj) {
            const int64_t vi = (int64_t)(jb + jj) * NT + tid;
            const bool ok = jb + jj < VPT && vi < nv;
            x4[jj] = ok ? ld4(xr + 4 * vi) : z4;
            g4[jj] = ok ? ld4(gr + 4 * vi) : z4;
            r4[jj] = (ok && a.resid) ? ld4(a.resid + t * a.lddx + 4 * vi) : z4;
          }
#pragma unroll
          for (int jj = 0; jj < JB; ++jj) {
            const int j = jb + jj;
            const int64_t vi = (int64_t)j * NT + tid;
            if (j >= VPT || vi >= nv) continue;
            float4 dl = z4, sv = o4;
            if (a.delta) dl = ld4(a.delta + 4 * vi);
            if (a.s) sv = ld4(a.s + 4 * vi);
            float o[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const int64_t c = 4 * vi + e;
              const float x = f4get(x4[jj], e), g = f4get(g4[jj], e), se = f4get(sv, e);
              float d = g;
              if (quant) {
                const float v = R.xt(x, 0.f, f4get(dl, e), se);
                int in = 0;
                omq_ste_dh(v, qs, Q, &in);
                d = in ? g : 0.f;
                if (c == iM) d += GaM;
                if (c == im) d += Gbt;
              }
              const float dn = a.s ? __fdiv_rn(d, se) : d;
              o[e] = R.rstd * (dn - x * R.rstd * mean_dot) + f4get(r4[jj], e);
            }
            if (a.dX) *reinterpret_cast<float4*>(a.dX + t * a.lddx + 4 * vi) = make_float4(o[0], o[1], o[2], o[3]);
            if (a.dXb) st_bf16x4(a.dXb + t * a.lddxb + 4 * vi, o);
          }
        }
      }
    }
    if (let_sums) {                              // ds partial -sum(d X~) / s, ddelta partial -sum(d) / s
#pragma unroll
      for (int j = 0; j < VPT; ++j) {
        const int64_t vi = (int64_t)j * NT + tid;
        if (vi < nv) {
          const float4 sv = (LETP && a.s) ? ld4(a.s + 4 * vi) : o4;
          float* ps = a.part_s + p * a.C + 4 * vi;
          float* pd = a.part_d + p * a.C + 4 * vi;
          float os[4], od[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            os[e] = -acc_s[4 * j + e] / f4get(sv, e);
            od[e] = -acc_d[4 * j + e] / f4get(sv, e);
          }
          *reinterpret_cast<float4*>(ps) = make_float4(os[0], os[1], os[2], os[3]);
          *reinterpret_cast<float4*>(pd) = make_float4(od[0], od[1], od[2], od[3]);
        }
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

template <int P, int NT, int VPT>
static omq_status act_fwd_staged_go(cudaStream_t st, const ActFwdArgs& a, int stages, size_t smem) {
  auto kern = act_fwd_staged<P, NT, VPT>;
  static int per_sm = -1;
  static size_t smem_set = 0;
  if (smem > smem_set) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
      return OMQ_ERR_CUDA;
    smem_set = smem;
    per_sm = -1;
  }
  int bps = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&bps, kern, NT, smem) != cudaSuccess || bps < 1) return OMQ_ERR_CUDA;
  (void)per_sm;
  const int64_t grid = std::min<int64_t>(a.T, (int64_t)omq_num_sms() * bps);
  kern<<<(unsigned)grid, NT, smem, st>>>(a, stages);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

// Rows whose inputs fit two or more times in shared memory take the staged kernel; 16-byte aligned
// rows of up to 16 K columns.
template <int PRODUCER>
static omq_status act_fwd_dispatch(cudaStream_t st, const ActFwdArgs& a0) {
  ActFwdArgs a = a0;
  a.rows_per_cta = 1;
  const int nin = PRODUCER == AP_SWIGLU ? 2 : 1;
  const size_t row_bytes = (size_t)nin * a.C * 4;
  const int stages = (int)std::min<size_t>(3, (200 * 1024) / row_bytes);
  const bool aligned = a.ldx % 4 == 0 && omq_aligned16(a.X) &&
                       (PRODUCER != AP_SWIGLU || (a.ldu % 4 == 0 && omq_aligned16(a.U)));
  const int64_t nv = a.C / 4;
  if (nv <= 128 * 8) {                             // small rows: many CTAs per SM, 32 values per thread
    a.rows_per_cta = kFwdRows;
    act_fwd_rows<PRODUCER, 128, 8><<<(unsigned)((a.T + kFwdRows - 1) / kFwdRows), 128, 0, st>>>(a);
    OMQ_LAUNCH_CHECK();
    return OMQ_OK;
  }
  if (PRODUCER == AP_SWIGLU && nv <= 256 * 12) {
    a.rows_per_cta = kFwdRowsSwiglu;
    act_fwd_rows<PRODUCER, 256, 12><<<(unsigned)((a.T + kFwdRowsSwiglu - 1) / kFwdRowsSwiglu), 256, 0, st>>>(a);
    OMQ_LAUNCH_CHECK();
    return OMQ_OK;
  }
  if (stages >= 2 && aligned && nv <= 1024 * 4) {
    // the row-to-thread mapping of act_fwd_rows, so that the RMS sum (and every output) is the same
    const size_t smem = (size_t)stages * row_bytes;
    if (nv <= 512 * 2) return act_fwd_staged_go<PRODUCER, 512, 2>(st, a, stages, smem);
    if (nv <= 512 * 4) return act_fwd_staged_go<PRODUCER, 512, 4>(st, a, stages, smem);
    return act_fwd_staged_go<PRODUCER, 1024, 4>(st, a, stages, smem);
  }
  ACT_DISPATCH(act_fwd_rows, a, (unsigned)a.T, a.C);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

template <int PRODUCER, int VPT, int JB, int MINB, bool SUMS, bool RD = false>
static omq_status act_bwd_go(cudaStream_t st, const ActBwdArgs& a) {
  const int64_t nparts = (a.T + a.rows_per_cta - 1) / a.rows_per_cta;
  act_bwd_stream<PRODUCER, VPT, JB, MINB, SUMS, RD><<<(unsigned)nparts, ACT_BWD_NT, 0, st>>>(a);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

// Row length -> vectors per thread.  Without LET column sums any length up to 28 K streams in
// batches of four vectors; the column sums keep 8 VPT accumulators per thread in registers.
template <int PRODUCER>
static omq_status act_bwd_dispatch(cudaStream_t st, const ActBwdArgs& a) {
  const int64_t vpt = (a.C / 4 + ACT_BWD_NT - 1) / ACT_BWD_NT;
  const bool sums = PRODUCER != AP_SWIGLU && a.part_s != nullptr;
  if constexpr (PRODUCER == AP_PLAIN) {
    if (a.rowdot) {   // the row dot's partials take registers: loads in pairs to keep four CTAs per SM (two for longer rows)
      if (sums) return OMQ_ERR_UNSUPPORTED;
      if (vpt <= 4) return act_bwd_go<PRODUCER, 4, 2, 4, false, true>(st, a);
      if (vpt <= 8) return act_bwd_go<PRODUCER, 8, 4, 2, false, true>(st, a);
      if (vpt <= 16) return act_bwd_go<PRODUCER, 16, 4, 2, false, true>(st, a);
      if (vpt <= 28) return act_bwd_go<PRODUCER, 28, 4, 2, false, true>(st, a);
      return OMQ_ERR_UNSUPPORTED;
    }
  }
  if (!sums) {
    if (vpt <= 4) return act_bwd_go<PRODUCER, 4, 4, 4, false>(st, a);
    if (vpt <= 8) return act_bwd_go<PRODUCER, 8, 4, 4, false>(st, a);
    if (vpt <= 12) return act_bwd_go<PRODUCER, 12, 4, 4, false>(st, a);
    if (vpt <= 16) return act_bwd_go<PRODUCER, 16, 4, 4, false>(st, a);
    if (vpt <= 28) return act_bwd_go<PRODUCER, 28, 4, 4, false>(st, a);
    return OMQ_ERR_UNSUPPORTED;
  }
  if constexpr (PRODUCER != AP_SWIGLU) {
    if (vpt <= 4) return act_bwd_go<PRODUCER, 4, 4, 2, true>(st, a);
    if (vpt <= 8) return act_bwd_go<PRODUCER, 8, 4, 1, true>(st, a);
    if (vpt <= 16) return act_bwd_go<PRODUCER, 16, 4, 1, true>(st, a);
  }
  return OMQ_ERR_UNSUPPORTED;
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
  OMQ_REQUIRE(!a.rowdot || (a.producer == AP_PLAIN && a.dXb && a.C % 128 == 0 && a.ldrow >= a.T), OMQ_ERR_INVALID_ARG);
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
  const int dq = a.H * a.hd, dkv = a.Hkv * a.hd;
  const int t0 = blockIdx.x * kQkvFwdRows, t1 = t0 + kQkvFwdRows < a.T ? t0 + kQkvFwdRows : a.T;
  for (int t = t0; t < t1; ++t) {
  if (threadIdx.x == 0 && t + 1 < t1 && gridDim.y != 1) {   // the next row's segment into L2
    const int sg = (int)blockIdx.y;
    omq_l2_prefetch(a.Y + (int64_t)(t + 1) * a.ldy + (sg == 0 ? 0 : (sg == 1 ? dq : dq + dkv)),
                    (uint64_t)(sg == 0 ? dq : dkv) * 4);
  }
  for (int seg = blockIdx.y; seg < (gridDim.y == 1 ? 3 : (int)blockIdx.y + 1); ++seg) {   // y: one segment per CTA
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
  __syncthreads();                             // the reduction scratch is reused by the next row
  }
}

// Backward of the q, k, v chain, streamed like the activation quantizer backward: one pass writes
// the gradient with the in-range mask applied and accumulates the h-path row sums; after the
// block reduction the owner of each routed pair (the first max / min and its RoPE partner)
// recomputes that pair with the routing added and rewrites it.
#define QKV_BWD_NT 256

// SEG < 0: the three segments of every row in turn; SEG = 0, 1, 2: the q, k or v segment only (a
// CTA of each segment per row slab, so that the three run side by side).
template <int PPT, int SEG>
__device__ __forceinline__ void qkv_bwd_body(const QkvArgs& a, float* fsm) {
  constexpr int NT = QKV_BWD_NT;
  constexpr int NE = 8 * PPT;
  constexpr bool HAS_Q = SEG < 0 || SEG == 0, HAS_K = SEG < 0 || SEG == 1;
  const int tid = threadIdx.x;
  const int dq = a.H * a.hd, dkv = a.Hkv * a.hd;
  const bool sums = a.part_q != nullptr;
  const bool quant = a.abits < 16;
  const float Q = (float)((1 << (quant ? a.abits : 1)) - 1);
  const float4 z4 = make_float4(0.f, 0.f, 0.f, 0.f);
  float acc_q[NE], acc_k[NE], rq[NE];      // rq: 1/s_a of the thread's query columns, computed once
#pragma unroll
  for (int j = 0; j < (HAS_Q ? PPT : 0); ++j) {
    const int p = j * NT + tid;
    const int e1 = (p >> 4) * 128 + 4 * (p & 15);
    const bool ok = a.sa_exp != nullptr && p < a.H * 16;
    const float4 s1 = ok ? ld4(a.sa_exp + e1) : make_float4(1.f, 1.f, 1.f, 1.f);
    const float4 s2 = ok ? ld4(a.sa_exp + e1 + 64) : make_float4(1.f, 1.f, 1.f, 1.f);
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      rq[8 * j + e] = __frcp_rn(f4get(s1, e));
      rq[8 * j + 4 + e] = __frcp_rn(f4get(s2, e));
    }
  }
#pragma unroll
  for (int k = 0; k < NE; ++k) { acc_q[k] = 0.f; acc_k[k] = 0.f; }
  const int t0 = blockIdx.x * a.rows_per_cta, t1 = min(a.T, t0 + a.rows_per_cta);
  for (int t = t0; t < t1; ++t) {
    for (int seg = (SEG < 0 ? 0 : SEG); seg < (SEG < 0 ? 3 : SEG + 1); ++seg) {
      const int Hs = seg == 0 ? a.H : a.Hkv;
      const int np = Hs * 16;
      const int off = seg == 0 ? 0 : (seg == 1 ? dq : dq + dkv);
      if (tid == 0 && t + 1 < t1) {           // the next row's segment into L2
        omq_l2_prefetch(a.Y + (int64_t)(t + 1) * a.ldy + off, (uint64_t)Hs * a.hd * 4);
        omq_l2_prefetch(a.dQKV + (int64_t)(t + 1) * a.ldd + off, (uint64_t)Hs * a.hd * 4);
      }
      const float* base = a.Y + (int64_t)t * a.ldy + off;
      const float* gsrc = a.dQKV + (int64_t)t * a.ldd + off;
      float* dy = a.dY + (int64_t)t * a.ldy + off;
      __nv_bfloat16* dyb = a.dYb + (int64_t)t * a.ldy + off;
      const float* csr = a.cs + (int64_t)t * 128;
      const bool rope = seg < 2, let = seg < 2 && a.sa_exp != nullptr;
      // X~ of one element (the forward's exact operation order)
      auto xt_of = [&](float v, int i) -> float {
        if (!let) return v;
        return seg == 0 ? __fdiv_rn(v, a.sa_exp[i]) : __fmul_rn(v, a.sa[i]);
      };
      QState qs;
      int iM = -1, im = -1;
      const int64_t kq = (int64_t)seg * a.T + t;
      if (quant) {
        iM = a.imax[kq]; im = a.imin[kq];
        auto xt_at = [&](int i) -> float {
          if (!rope) return base[i];
          const int jj = (i % 128) % 64, first = (i % 128) < 64;
          const float cv = csr[2 * jj], sv = csr[2 * jj + 1];
          const float v = first ? base[i] * cv - base[i + 64] * sv : base[i] * cv + base[i - 64] * sv;
          return xt_of(v, i);
        };
        const float m = xt_at(im);
        qs = omq_qstate(xt_at(iM), m, 1.f, 1.f, Q, a.eps);
        qs.h = a.h[kq]; qs.z = (float)a.z[kq]; qs.rh = __frcp_rn(qs.h); qs.u = __fmul_rn(m, qs.rh);
      }
      float Gh = 0.f, Gbm = 0.f;
      // ---- pass 1 ----
      float4 x1[PPT], x2[PPT], g1[PPT], g2[PPT], ca[PPT], cb[PPT];
#pragma unroll
      for (int j = 0; j < PPT; ++j) {                   // every load of the segment first
        const int p = j * NT + tid;
        const bool ok = p < np;
        const int e1 = (p >> 4) * 128 + 4 * (p & 15);
        x1[j] = ok ? ld4(base + e1) : z4;
        x2[j] = ok ? ld4(base + e1 + 64) : z4;
        g1[j] = ok ? ld4(gsrc + e1) : z4;
        g2[j] = ok ? ld4(gsrc + e1 + 64) : z4;
        ca[j] = (ok && rope) ? ld4(csr + 8 * (p & 15)) : z4;
        cb[j] = (ok && rope) ? ld4(csr + 8 * (p & 15) + 4) : z4;
      }
#pragma unroll
      for (int j = 0; j < PPT; ++j) {
        const int p = j * NT + tid;
        if (p >= np) continue;
        const int e1 = (p >> 4) * 128 + 4 * (p & 15);
        const float cv[4] = {ca[j].x, ca[j].z, cb[j].x, cb[j].z};
        const float sv[4] = {ca[j].y, ca[j].w, cb[j].y, cb[j].w};
        float o1[4], o2[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float a1 = f4get(x1[j], e), a2 = f4get(x2[j], e);
          const float r1 = rope ? a1 * cv[e] - a2 * sv[e] : a1;
          const float r2 = rope ? a2 * cv[e] + a1 * sv[e] : a2;
          const float v1 = xt_of(r1, e1 + e), v2 = xt_of(r2, e1 + 64 + e);
          float d1 = f4get(g1[j], e), d2 = f4get(g2[j], e);
          if (quant) {
            int in1 = 0, in2 = 0;
            const float h1 = omq_ste_dh(v1, qs, Q, &in1), h2 = omq_ste_dh(v2, qs, Q, &in2);
            Gh = fmaf(d1, h1, Gh);
            Gh = fmaf(d2, h2, Gh);
            if (!in1) { Gbm += d1; d1 = 0.f; }
            if (!in2) { Gbm += d2; d2 = 0.f; }
          }
          if (let) {
            const int k1 = 8 * j + e, k2 = 8 * j + 4 + e;
            if (seg == 0) {                      // the 1/s_a of the ds_a terms is applied once, at the end
              if (sums) { acc_q[k1] = fmaf(-d1, v1, acc_q[k1]); acc_q[k2] = fmaf(-d2, v2, acc_q[k2]); }
              d1 *= rq[k1]; d2 *= rq[k2];
            } else {
              if (sums) { acc_k[k1] += d1 * r1; acc_k[k2] += d2 * r2; }
              d1 = __fmul_rn(d1, a.sa[e1 + e]); d2 = __fmul_rn(d2, a.sa[e1 + 64 + e]);
            }
          }
          o1[e] = rope ? d1 * cv[e] + d2 * sv[e] : d1;
          o2[e] = rope ? d2 * cv[e] - d1 * sv[e] : d2;
        }
        if (a.dY) {
          *reinterpret_cast<float4*>(dy + e1) = make_float4(o1[0], o1[1], o1[2], o1[3]);
          *reinterpret_cast<float4*>(dy + e1 + 64) = make_float4(o2[0], o2[1], o2[2], o2[3]);
        }
        st_bf16x4(dyb + e1, o1);
        st_bf16x4(dyb + e1 + 64, o2);
      }
      if (!quant) continue;
      const float3 tot = block_sum3(Gh, Gbm, 0.f, fsm);
      const float Gh_t = qs.floored ? 0.f : tot.x;
      const float GaM = Gh_t / Q, Gbt = tot.y - Gh_t / Q;
      // ---- the routed pairs: recomputed with the routing by their owners ----
#pragma unroll
      for (int r = 0; r < 2; ++r) {
        const int c = r == 0 ? iM : im;
        const int first = (c & ~127) + (c & 63);           // element of the pair in the first half
        if (r == 1 && ((iM & ~127) + (iM & 63)) == first) break;   // same pair: already done
        const int pp = (first >> 7) * 16 + ((first & 63) >> 2);
        if (pp % NT != tid) continue;
        const int j = pp / NT;
        const int e = first & 3;
        const int jj = first & 63;
        const float cv = rope ? csr[2 * jj] : 1.f, sv = rope ? csr[2 * jj + 1] : 0.f;
        const float a1 = base[first], a2 = base[first + 64];
        const float r1 = rope ? a1 * cv - a2 * sv : a1;
        const float r2 = rope ? a2 * cv + a1 * sv : a2;
        const float v1 = xt_of(r1, first), v2 = xt_of(r2, first + 64);
        const float g1s = gsrc[first], g2s = gsrc[first + 64];
        int in1 = 0, in2 = 0;
        omq_ste_dh(v1, qs, Q, &in1);
        omq_ste_dh(v2, qs, Q, &in2);
        float ro1 = 0.f, ro2 = 0.f;                        // routing of each element of the pair
        if (first == iM) ro1 += GaM;
        if (first == im) ro1 += Gbt;
        if (first + 64 == iM) ro2 += GaM;
        if (first + 64 == im) ro2 += Gbt;
        float d1 = (in1 ? g1s : 0.f) + ro1, d2 = (in2 ? g2s : 0.f) + ro2;
        if (let) {
#pragma unroll
          for (int jx = 0; jx < PPT; ++jx)
#pragma unroll
            for (int ex = 0; ex < 4; ++ex) {
              if (jx != j || ex != e) continue;
              const int k1 = 8 * jx + ex, k2 = 8 * jx + 4 + ex;
              if (seg == 0) {
                if (sums) { acc_q[k1] = fmaf(-ro1, v1, acc_q[k1]); acc_q[k2] = fmaf(-ro2, v2, acc_q[k2]); }
              } else {
                if (sums) { acc_k[k1] += ro1 * r1; acc_k[k2] += ro2 * r2; }
              }
            }
          if (seg == 0) { d1 = __fdiv_rn(d1, a.sa_exp[first]); d2 = __fdiv_rn(d2, a.sa_exp[first + 64]); }
          else { d1 = __fmul_rn(d1, a.sa[first]); d2 = __fmul_rn(d2, a.sa[first + 64]); }
        }
        const float o1 = rope ? d1 * cv + d2 * sv : d1;
        const float o2 = rope ? d2 * cv - d1 * sv : d2;
        if (a.dY) { dy[first] = o1; dy[first + 64] = o2; }
        dyb[first] = f_to_bf16(o1); dyb[first + 64] = f_to_bf16(o2);
      }
    }
  }
  if (sums) {
#pragma unroll
    for (int j = 0; j < PPT; ++j) {
      const int p = j * NT + tid;
      const int e1 = (p >> 4) * 128 + 4 * (p & 15);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        if (HAS_Q && p < a.H * 16) {
          a.part_q[(int64_t)blockIdx.x * dq + e1 + e] = acc_q[8 * j + e] * rq[8 * j + e];
          a.part_q[(int64_t)blockIdx.x * dq + e1 + 64 + e] = acc_q[8 * j + 4 + e] * rq[8 * j + 4 + e];
        }
        if (HAS_K && p < a.Hkv * 16) {
          a.part_k[(int64_t)blockIdx.x * dkv + e1 + e] = acc_k[8 * j + e];
          a.part_k[(int64_t)blockIdx.x * dkv + e1 + 64 + e] = acc_k[8 * j + 4 + e];
        }
      }
    }
  }
}

template <int PPT, int MINB>
__global__ void __launch_bounds__(QKV_BWD_NT, MINB) qkv_bwd_stream(QkvArgs a) {
  __shared__ float fsm[96];
  qkv_bwd_body<PPT, -1>(a, fsm);
}

// one CTA per (row slab, segment): blockIdx.y picks q, k or v
template <int PPT, int MINB>
__global__ void __launch_bounds__(QKV_BWD_NT, MINB) qkv_bwd_seg(QkvArgs a) {
  __shared__ float fsm[96];
  if (blockIdx.y == 0) qkv_bwd_body<PPT, 0>(a, fsm);
  else if (blockIdx.y == 1) qkv_bwd_body<PPT, 1>(a, fsm);
  else qkv_bwd_body<PPT, 2>(a, fsm);
}

// token rows per CTA of the q, k, v backward (each CTA prefetches its next row into L2); the ds_a
// partials have one row per CTA
constexpr int kQkvBwdRows = 7;
int64_t qkv_bwd_nslab(int T) { return (T + kQkvBwdRows - 1) / kQkvBwdRows; }

omq_status qkv_fwd_launch(cudaStream_t st, const QkvArgs& a) {
  OMQ_REQUIRE(a.hd == 128, OMQ_ERR_UNSUPPORTED);
  const int np = a.H * 16;
  const dim3 g3((unsigned)((a.T + kQkvFwdRows - 1) / kQkvFwdRows), 3);   // one CTA per (token rows, q | k | v)
  if (np <= 512) qkv_fwd_rows<128, 4><<<g3, 128, 0, st>>>(a);
  else if (np <= 1024) qkv_fwd_rows<512, 2><<<g3.x, 512, 0, st>>>(a);
  else if (np <= 2048) qkv_fwd_rows<512, 4><<<g3.x, 512, 0, st>>>(a);
  else return OMQ_ERR_UNSUPPORTED;
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

omq_status qkv_bwd_launch(cudaStream_t st, const QkvArgs& a0, int64_t* nslab) {
  QkvArgs a = a0;
  OMQ_REQUIRE(a.hd == 128, OMQ_ERR_UNSUPPORTED);
  a.rows_per_cta = kQkvBwdRows;
  const unsigned grid = (unsigned)qkv_bwd_nslab(a.T);
  const int np = a.H * 16;
  if (np <= 256) qkv_bwd_stream<1, 4><<<grid, QKV_BWD_NT, 0, st>>>(a);
  else if (np <= 512) qkv_bwd_seg<2, 2><<<dim3(grid, 3), QKV_BWD_NT, 0, st>>>(a);
  else if (np <= 1024) qkv_bwd_stream<4, 1><<<grid, QKV_BWD_NT, 0, st>>>(a);
  else if (np <= 2048) qkv_bwd_stream<8, 1><<<grid, QKV_BWD_NT, 0, st>>>(a);
  else return OMQ_ERR_UNSUPPORTED;
  OMQ_LAUNCH_CHECK();
  if (nslab) *nslab = qkv_bwd_nslab(a.T);
  return OMQ_OK;
}
