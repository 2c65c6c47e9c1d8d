// Shared device/host helpers of libomq (sm_103a).
#pragma once
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>
#include <math.h>

#include "omq.h"

#define OMQ_VERSION 1

// ------------------------------------------------------------------------------------------------
// host-side argument checks
// ------------------------------------------------------------------------------------------------
#define OMQ_REQUIRE(cond, code) do { if (!(cond)) return (code); } while (0)
// every kernel launch of the library is followed by this check, which also counts it
void omq_count_launch();
#define OMQ_LAUNCH_CHECK() do { omq_count_launch(); if (cudaPeekAtLastError() != cudaSuccess) { cudaGetLastError(); return OMQ_ERR_CUDA; } } while (0)
#define OMQ_TRY(expr) do { omq_status _s = (expr); if (_s != OMQ_OK) return _s; } while (0)

static inline bool omq_aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
static inline bool omq_bits_ok(int b) { return (b >= 2 && b <= 8) || b == 16; }

static inline omq_status omq_check_cfg(const omq_qcfg* cfg) {
  if (!cfg) return OMQ_ERR_INVALID_ARG;
  if (!omq_bits_ok(cfg->wbits) || !omq_bits_ok(cfg->abits)) return OMQ_ERR_UNSUPPORTED;
  if (cfg->group < 0) return OMQ_ERR_SHAPE;
  if (!(cfg->h_eps > 0.f)) return OMQ_ERR_INVALID_ARG;
  if (cfg->pbits != 0 && cfg->pbits != 16 && !(cfg->pbits >= 2 && cfg->pbits <= 8)) return OMQ_ERR_UNSUPPORTED;
  if (cfg->wprep != 0 && cfg->wprep != 1) return OMQ_ERR_INVALID_ARG;
  return OMQ_OK;
}

static inline int omq_num_sms() {
  static int n = 0;
  if (n == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 148;
  }
  return n;
}

// ------------------------------------------------------------------------------------------------
// device status word and bounded waits
// ------------------------------------------------------------------------------------------------
__device__ __forceinline__ void omq_set_status(int32_t* st, int32_t code) {
  if (st) atomicCAS(st, 0, code);
}

// Bulk prefetch of [p, p + bytes) into L2 (cp.async.bulk.prefetch: no data returned, no completion
// to wait for); p 16-byte aligned and bytes a multiple of 16, else nothing is issued
__device__ __forceinline__ void omq_l2_prefetch(const void* p, uint64_t bytes) {
  if (((uintptr_t)p & 15) != 0 || (bytes & 15) != 0 || bytes == 0) return;
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"((uint32_t)bytes) : "memory");
}

__device__ __forceinline__ uint64_t omq_globaltimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Upper bound of any single device-side wait: one second.
#define OMQ_WAIT_LIMIT_NS 1000000000ull

// ------------------------------------------------------------------------------------------------
// conversions
// ------------------------------------------------------------------------------------------------
__device__ __forceinline__ float bf16_to_f(__nv_bfloat16 v) { return __bfloat162float(v); }
__device__ __forceinline__ __nv_bfloat16 f_to_bf16(float v) { return __float2bfloat16_rn(v); }

__device__ __forceinline__ void unpack_bf16x8(const uint4& u, float* f) {
  const __nv_bfloat162* p = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    float2 t = __bfloat1622float2(p[i]);
    f[2 * i] = t.x;
    f[2 * i + 1] = t.y;
  }
}

__device__ __forceinline__ uint4 pack_bf16x8(const float* f) {
  uint4 u;
  __nv_bfloat162* p = reinterpret_cast<__nv_bfloat162*>(&u);
#pragma unroll
  for (int i = 0; i < 4; ++i) p[i] = __floats2bfloat162_rn(f[2 * i], f[2 * i + 1]);
  return u;
}

// ------------------------------------------------------------------------------------------------
// Eq. 2 on one element, given the group's h and z
// ------------------------------------------------------------------------------------------------
struct QState {          // per-group quantizer state
  float h;               // step, floored at eps
  float rh;              // 1/h, correctly rounded (a first guess of w/h is w * rh)
  float z;               // zero point (integer valued): -round(beta * min / h)
  float u;               // beta * min / h (its value; the rounding is taken exactly, -z)
  float a, b;            // clipping strengths
  float M, m;            // group max / min
  int floored;
};

// gamma = sigmoid(gamma_hat) in single precision with every operation rounded once (no fused
// multiply-add), so that the value is reproducible bit for bit on any IEEE machine:
// exp(-t) by Cody-Waite reduction, -t = n ln2 + r with |r| <= ln2/2 (ln2 split into a 15-bit head,
// whose product with n is exact, and a tail), a degree-7 Taylor polynomial for exp(r) in Horner
// form, and an exact scaling by 2^n; then 1 / (1 + exp(-t)).  |t| is clamped to 80.
__device__ __forceinline__ float omq_sigmoid(float t) {
  const float x = -fminf(fmaxf(t, -80.f), 80.f);
  const float n = rintf(__fmul_rn(x, 1.44269502162933349609375f));
  const float r = __fsub_rn(__fsub_rn(x, __fmul_rn(n, 0.693145751953125f)), __fmul_rn(n, 1.428606765330187e-06f));
  float p = 1.98412701138295233249664e-04f;
  p = __fadd_rn(__fmul_rn(p, r), 1.38888892251998186111450e-03f);
  p = __fadd_rn(__fmul_rn(p, r), 8.33333376795053482055664e-03f);
  p = __fadd_rn(__fmul_rn(p, r), 4.16666679084300994873047e-02f);
  p = __fadd_rn(__fmul_rn(p, r), 1.66666671633720397949219e-01f);
  p = __fadd_rn(__fmul_rn(p, r), 0.5f);
  p = __fadd_rn(__fmul_rn(p, r), 1.0f);
  p = __fadd_rn(__fmul_rn(p, r), 1.0f);
  const float e = __fmul_rn(p, __int_as_float((127 + (int)n) << 23));
  return __fdiv_rn(1.0f, __fadd_rn(1.0f, e));
}

// round(w / h) of Eq. 2 for the exact quotient of the two single-precision values (h > 0).
// A first guess k = rint(w * (1/h)) can land on the wrong side of a half when the quotient is
// within a few ulps of one.  The remainder r = w - k h is exact in single precision (a fused
// multiply-add; |r| is at most about h / 2 and lies on the grid of the smaller of the two
// exponents, so it fits in 24 bits), and k moves by rint(r / h), which is 0 or +-1.  The result
// equals the rounding of the exact quotient except for quotients within about 1e-7 of a half.
__device__ __forceinline__ float omq_round_quot(float w, float h, float rh) {
  const float k = rintf(__fmul_rn(w, rh));
  const float r = __fmaf_rn(-k, h, w);
  return __fadd_rn(k, rintf(__fmul_rn(r, rh)));
}

// h = (a*M - b*m)/Q floored at eps, its reciprocal, u = (b*m) / h and z = -round(u).
// The zero point rounds u written without the rounded h: Q (b m) / (a M - b m), or Q m / (M - m)
// when a = b (the clipping strengths cancel), or b m / eps when h is floored.  Such a quotient can
// be exactly a half, which then rounds to even, and often is: with gamma = beta and a group whose
// max and min are opposite (frequent among bf16 weights) u = -Q/2; rounding u = (b m) (1/h) from
// the rounded fp32 h would round it by noise instead.  The single-precision u decides unless it lies
// within its own error bound (eight roundings, times the cancellation factor of a M - b m) of a half;
// only then is the quotient formed in double precision, where the products by Q and the difference
// of single-precision values are exact and an exact half stays one.
__device__ __forceinline__ QState omq_qstate(float M, float m, float a, float b, float Q, float eps) {
  QState s;
  s.a = a; s.b = b; s.M = M; s.m = m;
  const float bm = __fmul_rn(b, m);
  const float aM = __fmul_rn(a, M);
  const float d = __fsub_rn(aM, bm);
  float hr = __fdiv_rn(d, Q);
  s.floored = !(hr >= eps);
  s.h = s.floored ? eps : hr;
  s.rh = __frcp_rn(s.h);
  s.u = __fmul_rn(bm, s.rh);
  float k = rintf(s.u);
  const float cancel = s.floored ? 1.f : (fabsf(aM) + fabsf(bm)) / fabsf(d);
  const float margin = 1e-6f + fabsf(s.u) * 4.76837158203125e-07f * (2.f + cancel);   // 2^-21 = eight ulps
  if (fabsf(fabsf(s.u - k) - 0.5f) <= margin) {
    double u64;
    if (s.floored) u64 = __ddiv_rn((double)bm, (double)eps);
    else if (a == b) u64 = __ddiv_rn((double)Q * (double)m, (double)M - (double)m);
    else u64 = __ddiv_rn((double)Q * (double)bm, (double)d);
    k = (float)rint(u64);
  }
  s.z = -k;
  return s;
}

// code c = round(w/h) + z before the clamp; *x_out = w/h (value, w * (1/h))
__device__ __forceinline__ float omq_code_raw(float w, const QState& s, float* x_out) {
  *x_out = __fmul_rn(w, s.rh);
  return omq_round_quot(w, s.h, s.rh) + s.z;
}

// clamp(round(w/h) + z, 0, Q) - z formed as clamp(round(w/h), -z, Q - z): every term is an
// integer below 2^24 after the clamp, so both forms give the same value
__device__ __forceinline__ float omq_fakequant(float w, const QState& s, float Q, float* code) {
  const float r = omq_round_quot(w, s.h, s.rh);
  const float qz = fminf(fmaxf(r, -s.z), Q - s.z);
  if (code) *code = qz + s.z;
  return __fmul_rn(qz, s.h);
}

// Paired f32 arithmetic (f32x2: one instruction for two lanes, each rounded to nearest exactly as
// __fmul_rn / __fmaf_rn / __fadd_rn round one)
__device__ __forceinline__ uint64_t omq_f2u(float2 v) {
  return ((uint64_t)__float_as_uint(v.y) << 32) | (uint64_t)__float_as_uint(v.x);
}
__device__ __forceinline__ float2 omq_u2f(uint64_t u) {
  return make_float2(__uint_as_float((uint32_t)u), __uint_as_float((uint32_t)(u >> 32)));
}
__device__ __forceinline__ float2 omq_mul2(float2 a, float2 b) {
  uint64_t d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(omq_f2u(a)), "l"(omq_f2u(b)));
  return omq_u2f(d);
}
__device__ __forceinline__ float2 omq_fma2(float2 a, float2 b, float2 c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(omq_f2u(a)), "l"(omq_f2u(b)), "l"(omq_f2u(c)));
  return omq_u2f(d);
}
__device__ __forceinline__ float2 omq_add2(float2 a, float2 b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(omq_f2u(a)), "l"(omq_f2u(b)));
  return omq_u2f(d);
}

// omq_fakequant of two elements with the paired operations: the same roundings in the same order,
// so each lane equals the scalar result bit for bit (w - k h as k (-h) + w: the same exact product)
__device__ __forceinline__ float2 omq_fakequant2(float2 w, const QState& s, float Q, float2* code) {
  const float2 rh = make_float2(s.rh, s.rh), h = make_float2(s.h, s.h), nh = make_float2(-s.h, -s.h);
  const float2 x = omq_mul2(w, rh);
  const float2 k = make_float2(rintf(x.x), rintf(x.y));
  const float2 r = omq_fma2(k, nh, w);
  const float2 y = omq_mul2(r, rh);
  const float2 q = omq_add2(k, make_float2(rintf(y.x), rintf(y.y)));
  const float2 qz = make_float2(fminf(fmaxf(q.x, -s.z), Q - s.z), fminf(fmaxf(q.y, -s.z), Q - s.z));
  if (code) *code = omq_add2(qz, make_float2(s.z, s.z));
  return omq_mul2(qz, h);
}

// STE pieces of one element: returns dwhat/dh; *inr = 1 when 0 <= c <= Q.  round(u) is -z, the
// zero point's own rounding.
__device__ __forceinline__ float omq_ste_dh(float w, const QState& s, float Q, int* inr) {
  const float x = __fmul_rn(w, s.rh);
  const float r = omq_round_quot(w, s.h, s.rh);
  const float c = r + s.z;
  if (c >= 0.f && c <= Q) { *inr = 1; return r - x; }
  *inr = 0;
  const float ru = -s.z - s.u;
  return (c < 0.f) ? ru : (Q + ru);
}

// omq_ste_dh of two elements with the paired operations (each lane equal to the scalar result)
__device__ __forceinline__ float2 omq_ste_dh2(float2 w, const QState& s, float Q, int* inr0, int* inr1) {
  const float2 rh = make_float2(s.rh, s.rh), nh = make_float2(-s.h, -s.h), m1 = make_float2(-1.f, -1.f);
  const float2 x = omq_mul2(w, rh);
  const float2 k = make_float2(rintf(x.x), rintf(x.y));
  const float2 y = omq_mul2(omq_fma2(k, nh, w), rh);
  const float2 r = omq_add2(k, make_float2(rintf(y.x), rintf(y.y)));
  const float2 c = omq_add2(r, make_float2(s.z, s.z));
  const float2 d = omq_fma2(x, m1, r);            // r - x
  const float ru = -s.z - s.u;
  const bool in0 = c.x >= 0.f && c.x <= Q, in1 = c.y >= 0.f && c.y <= Q;
  *inr0 = in0; *inr1 = in1;
  return make_float2(in0 ? d.x : (c.x < 0.f ? ru : Q + ru), in1 ? d.y : (c.y < 0.f ? ru : Q + ru));
}

// ------------------------------------------------------------------------------------------------
// (value, index) reductions with first-index tie break
// ------------------------------------------------------------------------------------------------
struct MaxMin { float M; int iM; float m; int im; };

__device__ __forceinline__ MaxMin mm_identity() { MaxMin r; r.M = -INFINITY; r.iM = 0x7fffffff; r.m = INFINITY; r.im = 0x7fffffff; return r; }

__device__ __forceinline__ void mm_push(MaxMin& r, float v, int i) {
  if (v > r.M || (v == r.M && i < r.iM)) { r.M = v; r.iM = i; }
  if (v < r.m || (v == r.m && i < r.im)) { r.m = v; r.im = i; }
}

__device__ __forceinline__ void mm_merge(MaxMin& r, const MaxMin& o) {
  if (o.M > r.M || (o.M == r.M && o.iM < r.iM)) { r.M = o.M; r.iM = o.iM; }
  if (o.m < r.m || (o.m == r.m && o.im < r.im)) { r.m = o.m; r.im = o.im; }
}

// reduction across `width` consecutive lanes (width power of two, <= 32)
__device__ __forceinline__ MaxMin mm_shfl_reduce(MaxMin r, int width) {
  for (int off = width >> 1; off > 0; off >>= 1) {
    MaxMin o;
    o.M = __shfl_xor_sync(0xffffffffu, r.M, off);
    o.iM = __shfl_xor_sync(0xffffffffu, r.iM, off);
    o.m = __shfl_xor_sync(0xffffffffu, r.m, off);
    o.im = __shfl_xor_sync(0xffffffffu, r.im, off);
    mm_merge(r, o);
  }
  return r;
}

// block-wide reduction; result valid in every thread.  smem: >= 32 MaxMin.
__device__ __forceinline__ MaxMin mm_block_reduce(MaxMin r, MaxMin* smem) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  r = mm_shfl_reduce(r, 32);
  __syncthreads();
  if (lane == 0) smem[wid] = r;
  __syncthreads();
  MaxMin t = mm_identity();
  if (lane < nw) t = smem[lane];
  t = mm_shfl_reduce(t, 32);
  return t;
}

__device__ __forceinline__ float warp_sum(float v, int width = 32) {
  for (int off = width >> 1; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  return v;
}

// block-wide sum of up to 2 values; results valid in every thread.  smem: >= 64 floats.
__device__ __forceinline__ float2 block_sum2(float a, float b, float* smem) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  a = warp_sum(a);
  b = warp_sum(b);
  __syncthreads();
  if (lane == 0) { smem[wid] = a; smem[32 + wid] = b; }
  __syncthreads();
  float x = lane < nw ? smem[lane] : 0.f;
  float y = lane < nw ? smem[32 + lane] : 0.f;
  x = warp_sum(x);
  y = warp_sum(y);
  return make_float2(x, y);
}

// deterministic column reduction: out[c] (+)= sum_p part[p, c]
__global__ void omq_colsum_partials_kernel(const float* __restrict__ part, int64_t P, int64_t C,
                                           float* __restrict__ out, float scale, int accumulate);

// one column reduction out[c] (+)= scale * sum_p part[p, c] of a [P, C] row-major array
struct ColsumJob {
  const float* part; int64_t P, C; float* out; float scale; int accumulate;
};
// two independent column reductions in one launch
omq_status omq_colsum_partials2(cudaStream_t st, const ColsumJob& a, const ColsumJob& b);
omq_status omq_colsum_partials(cudaStream_t st, const float* part, int64_t P, int64_t C, float* out,
                               float scale, int accumulate);
