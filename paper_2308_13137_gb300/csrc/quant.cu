// HBM-bound kernels of the calibration step: LWC (Eq. 2) forward/backward on the LET-scaled
// weight (Eq. 3), the per-token MinMax activation quantizer with fused producers (LET, RMSNorm,
// SwiGLU) and its straight-through backward, the block loss (Eq. 1), column reductions and AdamW.
#include "quant.cuh"

#include <atomic>
#include <cooperative_groups.h>

namespace cg = cooperative_groups;


static std::atomic<long long> g_launches{0};
void omq_count_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }
#define ACT_THREADS 256

// ================================================================================================
// LWC forward: one warp per output row, eight rows per CTA; reductions by shuffles only.
// ================================================================================================
__device__ __forceinline__ float lwc_wt(float w, const float* s, int64_t col, float rr) {
  float sv = s ? s[col] : 1.f;
  return __fmul_rn(__fmul_rn(w, sv), rr);
}

// eight consecutive entries of an optional vector (1 when absent)
__device__ __forceinline__ void load8(const float* v, int64_t c, float* out, float dflt) {
  if (!v) {
#pragma unroll
    for (int e = 0; e < 8; ++e) out[e] = dflt;
    return;
  }
  float4 x = __ldg(reinterpret_cast<const float4*>(v) + 2 * c);
  float4 y = __ldg(reinterpret_cast<const float4*>(v) + 2 * c + 1);
  out[0] = x.x; out[1] = x.y; out[2] = x.z; out[3] = x.w; out[4] = y.x; out[5] = y.y; out[6] = y.z; out[7] = y.w;
}

// W~ = fl32(fl32(W * s) * r) for one 8-element chunk
__device__ __forceinline__ void lwc_chunk(const uint4& raw, const float* s, int64_t c, float rr, float* wt) {
  float sv[8];
  unpack_bf16x8(raw, wt);
  load8(s, c, sv, 1.f);
#pragma unroll
  for (int e = 0; e < 8; ++e) wt[e] = __fmul_rn(__fmul_rn(wt[e], sv[e]), rr);
}

__device__ __forceinline__ void lwc_store(const LwcFwdArgs& a, int64_t o, int64_t c, const float* wt, const QState& qs,
                                          float Q) {
  float w[8], cd[8];
#pragma unroll
  for (int e = 0; e < 8; e += 2) {
    float2 c2;
    const float2 v = omq_fakequant2(make_float2(wt[e], wt[e + 1]), qs, Q, &c2);
    w[e] = v.x; w[e + 1] = v.y; cd[e] = c2.x; cd[e + 1] = c2.y;
  }
  if (a.Wq) reinterpret_cast<uint4*>(a.Wq + o * a.Cin)[c] = pack_bf16x8(w);
  if (a.codes) {
    uint2 pk;
    pk.x = (uint32_t)cd[0] | ((uint32_t)cd[1] << 8) | ((uint32_t)cd[2] << 16) | ((uint32_t)cd[3] << 24);
    pk.y = (uint32_t)cd[4] | ((uint32_t)cd[5] << 8) | ((uint32_t)cd[6] << 16) | ((uint32_t)cd[7] << 24);
    reinterpret_cast<uint2*>(a.codes + o * a.Cin)[c] = pk;
  }
}

__device__ __forceinline__ float dot8(const uint4& raw, const float* d, int64_t c) {
  float w[8], dv[8];
  unpack_bf16x8(raw, w);
  load8(d, c, dv, 0.f);
  float acc = 0.f;
#pragma unroll
  for (int e = 0; e < 8; ++e) acc = fmaf(w[e], dv[e], acc);
  return acc;
}

// MODE 0: quantization off; 1: one group per row; 2: groups of <= 256 columns
template <int MODE>
__global__ void __launch_bounds__(256, 4) lwc_fwd_kernel(LwcFwdArgs a) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t o = (int64_t)blockIdx.x * 8 + warp;
  if (o >= a.Cout) return;                       // whole warp leaves; no block-level barrier below
  const int64_t nchunk = a.Cin / 8;
  const int iters = (int)((nchunk + 31) / 32);
  const float Q = (float)((1 << (a.wbits >= 16 ? 1 : a.wbits)) - 1);
  const float rr = a.r ? a.r[o] : 1.f;
  const uint4* Wrow = reinterpret_cast<const uint4*>(a.W + o * a.Cin);
  const int gsz = a.group;
  const int64_t ngroups = a.Cin / gsz;
  const uint4 zero4 = make_uint4(0, 0, 0, 0);
  float dot = 0.f;

  if (MODE == 0) {                               // quantization off: W_hat = bf16(W~)
    for (int it0 = 0; it0 < iters; it0 += 4) {
      uint4 raw[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int64_t c = (int64_t)(it0 + j) * 32 + lane;
        raw[j] = (it0 + j < iters && c < nchunk) ? __ldg(Wrow + c) : zero4;
      }
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int64_t c = (int64_t)(it0 + j) * 32 + lane;
        if (it0 + j < iters && c < nchunk) {
          float wt[8];
          lwc_chunk(raw[j], a.s, c, rr, wt);
          if (a.Wq) reinterpret_cast<uint4*>(a.Wq + o * a.Cin)[c] = pack_bf16x8(wt);
          if (a.Bt) dot += dot8(raw[j], a.bias_delta, c);
        }
      }
    }
  } else if (MODE == 1) {
    // ---- one group per row.  Pass 1: values of max / min (and the LET bias dot).  Pass 2
    // (the row again, from L1/L2): quantize and store, and find the first index of max / min. ----
    float M = -INFINITY, m = INFINITY;
    for (int it0 = 0; it0 < iters; it0 += 4) {
      uint4 raw[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int64_t c = (int64_t)(it0 + j) * 32 + lane;
        raw[j] = (it0 + j < iters && c < nchunk) ? __ldg(Wrow + c) : zero4;
      }
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int64_t c = (int64_t)(it0 + j) * 32 + lane;
        if (it0 + j < iters && c < nchunk) {
          float wt[8];
          lwc_chunk(raw[j], a.s, c, rr, wt);
#pragma unroll
          for (int e = 0; e < 8; ++e) { M = fmaxf(M, wt[e]); m = fminf(m, wt[e]); }
          if (a.Bt) dot += dot8(raw[j], a.bias_delta, c);
        }
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
      m = fminf(m, __shfl_xor_sync(0xffffffffu, m, off));
    }
    float ga = 1.f, gb = 1.f;
    if (a.lwc) {                                 // one sigmoid per group, broadcast
      if (lane == 0) { ga = omq_sigmoid(a.gl[o]); gb = omq_sigmoid(a.bl[o]); }
      ga = __shfl_sync(0xffffffffu, ga, 0);
      gb = __shfl_sync(0xffffffffu, gb, 0);
    }
    const QState qs = omq_qstate(M, m, ga, gb, Q, a.eps);
    int iM = 0x7fffffff, im = 0x7fffffff;        // first index of the max / min held by this lane
    for (int it0 = 0; it0 < iters; it0 += 4) {
      uint4 raw[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int64_t c = (int64_t)(it0 + j) * 32 + lane;
        raw[j] = (it0 + j < iters && c < nchunk) ? __ldg(Wrow + c) : zero4;
      }
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int64_t c = (int64_t)(it0 + j) * 32 + lane;
        if (it0 + j < iters && c < nchunk) {
          float wt[8];
          lwc_chunk(raw[j], a.s, c, rr, wt);
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const int idx = (int)(c * 8 + e);
            if (wt[e] == M && idx < iM) iM = idx;
            if (wt[e] == m && idx < im) im = idx;
          }
          lwc_store(a, o, c, wt, qs, Q);
        }
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      iM = min(iM, __shfl_xor_sync(0xffffffffu, iM, off));
      im = min(im, __shfl_xor_sync(0xffffffffu, im, off));
    }
    if (lane == 0) {
      a.h[o] = qs.h; a.z[o] = (int32_t)qs.z; a.imax[o] = iM; a.imin[o] = im;
      if (a.ga_out) { a.ga_out[o] = ga; a.gb_out[o] = gb; }
      if (a.M_out) { a.M_out[o] = M; a.m_out[o] = m; }
    }
  } else {
    // ---- groups of lpg consecutive lanes (lpg a power of two <= 32), four chunks of loads ahead ----
    const int lpg = gsz / 8;
    const int leader = lane & ~(lpg - 1);
    for (int it0 = 0; it0 < iters; it0 += 4) {
      uint4 raw[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int64_t c = (int64_t)(it0 + j) * 32 + lane;
        raw[j] = (it0 + j < iters && c < nchunk) ? __ldg(Wrow + c) : zero4;
      }
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        if (it0 + j >= iters) break;                     // warp-uniform
        const int64_t c = (int64_t)(it0 + j) * 32 + lane;
        const bool valid = c < nchunk;
        float wt[8];
        MaxMin r = mm_identity();
        if (valid) {
          lwc_chunk(raw[j], a.s, c, rr, wt);
#pragma unroll
          for (int e = 0; e < 8; ++e) mm_push(r, wt[e], (int)(c * 8 + e));
          if (a.Bt) dot += dot8(raw[j], a.bias_delta, c);
        }
        r = mm_shfl_reduce(r, lpg);
        const int64_t gi = valid ? (c * 8) / gsz : 0;
        float ga = 1.f, gb = 1.f;
        if (a.lwc) {
          if (lane == leader && valid) { ga = omq_sigmoid(a.gl[o * ngroups + gi]); gb = omq_sigmoid(a.bl[o * ngroups + gi]); }
          ga = __shfl_sync(0xffffffffu, ga, leader);
          gb = __shfl_sync(0xffffffffu, gb, leader);
        }
        if (valid) {
          const QState qs = omq_qstate(r.M, r.m, ga, gb, Q, a.eps);
          if (lane == leader) {
            const int64_t k = o * ngroups + gi;
            a.h[k] = qs.h; a.z[k] = (int32_t)qs.z; a.imax[k] = r.iM; a.imin[k] = r.im;
            if (a.ga_out) { a.ga_out[k] = ga; a.gb_out[k] = gb; }
            if (a.M_out) { a.M_out[k] = r.M; a.m_out[k] = r.m; }
          }
          lwc_store(a, o, c, wt, qs, Q);
        }
      }
    }
  }
  if (a.Bt) {
    dot = warp_sum(dot);
    if (lane == 0) a.Bt[o] = rr * (dot - (a.bias_shift ? a.bias_shift[o] : 0.f));
  }
}

// One group per row, one CTA per row: the row lives in registers (CPT 8-column chunks per thread)
// between the block reduction of max / min (and the LET bias dot) and the quantize pass, so every
// weight is read from HBM once.  The weights are streamed with evict-first loads so that W_hat,
// which the next product reads, stays in L2.  The first index of the max / min is searched only by
// the threads whose own extreme equals the row's.  Every value matches lwc_fwd_kernel<1> bit for
// bit except the LET bias dot, whose summation order differs.
template <int NT, int CPT>
__global__ void __launch_bounds__(NT) lwc_fwd_row_kernel(LwcFwdArgs a) {
  constexpr int NW = NT / 32;
  __shared__ float red[3][NW];
  __shared__ int sidx[2];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t o = blockIdx.x;
  const int64_t nchunk = a.Cin / 8;
  const float Q = (float)((1 << a.wbits) - 1);
  const float rr = a.r ? a.r[o] : 1.f;
  const uint4* Wrow = reinterpret_cast<const uint4*>(a.W + o * a.Cin);
  uint4 raw[CPT];
#pragma unroll
  for (int j = 0; j < CPT; ++j) {
    const int64_t c = (int64_t)j * NT + tid;
    raw[j] = c < nchunk ? __ldcs(Wrow + c) : make_uint4(0, 0, 0, 0);
  }
  if (tid == 0) { sidx[0] = 0x7fffffff; sidx[1] = 0x7fffffff; }
  float wt[CPT][8];
  float M = -INFINITY, m = INFINITY, dot = 0.f;
#pragma unroll
  for (int j = 0; j < CPT; ++j) {
    const int64_t c = (int64_t)j * NT + tid;
    if (c < nchunk) {
      float w8[8], sv[8];
      unpack_bf16x8(raw[j], w8);
      // W~ = fl(fl(W s) r); a factor that is absent is 1 and its product is skipped (exact)
      if (a.s) {
        load8(a.s, c, sv, 1.f);
#pragma unroll
        for (int e = 0; e < 8; ++e) wt[j][e] = __fmul_rn(w8[e], sv[e]);
      } else {
#pragma unroll
        for (int e = 0; e < 8; ++e) wt[j][e] = w8[e];
      }
      if (a.r) {
#pragma unroll
        for (int e = 0; e < 8; ++e) wt[j][e] = __fmul_rn(wt[j][e], rr);
      }
#pragma unroll
      for (int e = 0; e < 8; ++e) { M = fmaxf(M, wt[j][e]); m = fminf(m, wt[j][e]); }
      if (a.Bt) {
        float dv[8];
        load8(a.bias_delta, c, dv, 0.f);
        float acc = 0.f;
#pragma unroll
        for (int e = 0; e < 8; ++e) acc = fmaf(w8[e], dv[e], acc);
        dot += acc;
      }
    }
  }
  float bM = M, bm = m, bd = dot;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    bM = fmaxf(bM, __shfl_xor_sync(0xffffffffu, bM, off));
    bm = fminf(bm, __shfl_xor_sync(0xffffffffu, bm, off));
    bd += __shfl_xor_sync(0xffffffffu, bd, off);
  }
  if (lane == 0) { red[0][warp] = bM; red[1][warp] = bm; red[2][warp] = bd; }
  __syncthreads();
  bM = red[0][0]; bm = red[1][0]; bd = red[2][0];
#pragma unroll
  for (int w = 1; w < NW; ++w) { bM = fmaxf(bM, red[0][w]); bm = fminf(bm, red[1][w]); bd += red[2][w]; }
  float ga = 1.f, gb = 1.f;
  if (a.lwc) { ga = omq_sigmoid(a.gl[o]); gb = omq_sigmoid(a.bl[o]); }
  const QState qs = omq_qstate(bM, bm, ga, gb, Q, a.eps);
  if (M == bM || m == bm) {
    int iM = 0x7fffffff, im = 0x7fffffff;
#pragma unroll
    for (int j = CPT - 1; j >= 0; --j) {
      const int64_t c = (int64_t)j * NT + tid;
      if (c < nchunk) {
#pragma unroll
        for (int e = 7; e >= 0; --e) {
          if (wt[j][e] == bM) iM = (int)(c * 8 + e);
          if (wt[j][e] == bm) im = (int)(c * 8 + e);
        }
      }
    }
    if (iM != 0x7fffffff) atomicMin(&sidx[0], iM);
    if (im != 0x7fffffff) atomicMin(&sidx[1], im);
  }
#pragma unroll
  for (int j = 0; j < CPT; ++j) {
    const int64_t c = (int64_t)j * NT + tid;
    if (c < nchunk) lwc_store(a, o, c, wt[j], qs, Q);
  }
  __syncthreads();
  if (tid == 0) {
    a.h[o] = qs.h; a.z[o] = (int32_t)qs.z; a.imax[o] = sidx[0]; a.imin[o] = sidx[1];
    if (a.ga_out) { a.ga_out[o] = ga; a.gb_out[o] = gb; }
    if (a.M_out) { a.M_out[o] = bM; a.m_out[o] = bm; }
    if (a.Bt) a.Bt[o] = rr * (bd - (a.bias_shift ? a.bias_shift[o] : 0.f));
  }
}

template <int NT>
static void lwc_fwd_row_go(cudaStream_t st, const LwcFwdArgs& a, int64_t cpt) {
  const unsigned grid = (unsigned)a.Cout;
  if (cpt <= 2) lwc_fwd_row_kernel<NT, 2><<<grid, NT, 0, st>>>(a);
  else if (cpt <= 4) lwc_fwd_row_kernel<NT, 4><<<grid, NT, 0, st>>>(a);
  else if (cpt <= 6) lwc_fwd_row_kernel<NT, 6><<<grid, NT, 0, st>>>(a);
  else lwc_fwd_row_kernel<NT, 8><<<grid, NT, 0, st>>>(a);
}

static bool lwc_group_ok(int64_t Cin, int g) {
  if (g == Cin) return Cin % 8 == 0;
  if (g < 8 || g > 256 || (g & (g - 1))) return false;
  return Cin % g == 0;
}


omq_status lwc_fwd_launch(cudaStream_t st, const LwcFwdArgs& a) {
  OMQ_REQUIRE(lwc_group_ok(a.Cin, a.group), OMQ_ERR_UNSUPPORTED);
  const unsigned grid = (unsigned)((a.Cout + 7) / 8);
  const int64_t nchunk = a.Cin / 8;
  if (a.wbits >= 16) lwc_fwd_kernel<0><<<grid, 256, 0, st>>>(a);
  else if (a.group == a.Cin && nchunk <= 128 * 8) lwc_fwd_row_go<128>(st, a, (nchunk + 127) / 128);
  else if (a.group == a.Cin && nchunk <= 256 * 8) lwc_fwd_row_go<256>(st, a, (nchunk + 255) / 256);
  else if (a.group == a.Cin && nchunk <= 512 * 8) lwc_fwd_row_go<512>(st, a, (nchunk + 511) / 512);
  else if (a.group == a.Cin) lwc_fwd_kernel<1><<<grid, 256, 0, st>>>(a);
  else lwc_fwd_kernel<2><<<grid, 256, 0, st>>>(a);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

// ================================================================================================
// LWC backward (straight-through, Eq. 2), streaming over [row tile x column tile] blocks.
// Each thread owns one 8-column chunk of a 2048-column tile and walks the rows of its row tile,
// keeping the LET column sums of its columns in registers.  Per-row reductions are warp
// shuffles: inside a group they complete in the warp (groups of <= 256 columns); for one group
// per row every warp writes its 256-column partial and a per-row finalize combines them.
// ================================================================================================
#define LWC_BWD_THREADS 256
#define LWC_BWD_TILE_COLS (LWC_BWD_THREADS * 8)

struct LwcBwdScratch {
  float* part_s;     // [nrt, Cin]
  float* part_d;     // [nrt, Cin]
  float* rowpart;    // [3, Cout, ncw]: G_h, G_bm, dr partials of every 256-column warp
  float* sig;        // [2, Cout, ng]: clipping strengths when the caller has none saved
  float* route;      // [Cout, 4]: max column, its ds term, min column, its ds term
  int64_t nrt, ncw, rows, ng;
};

static int64_t lwc_bwd_tile_rows(int64_t Cout, int64_t Cin) {
  const int64_t ncol = (Cin / 8 + LWC_BWD_THREADS - 1) / LWC_BWD_THREADS;
  int64_t rows = (Cout * ncol + 607) / 608;           // about four CTAs per SM of a 152-SM part
  if (rows < 8) rows = 8;
  if (rows > 64) rows = 64;
  return rows;
}

static LwcBwdScratch lwc_bwd_carve(void* base, int64_t Cout, int64_t Cin, int64_t ng, size_t* bytes) {
  LwcBwdScratch sc;
  sc.ng = ng;
  sc.rows = lwc_bwd_tile_rows(Cout, Cin);
  sc.nrt = (Cout + sc.rows - 1) / sc.rows;
  sc.ncw = (Cin / 8 + 31) / 32;
  size_t off = 0;
  auto take = [&](size_t n) { off = (off + 63) & ~size_t(63); float* p = base ? (float*)((char*)base + off * 4) : nullptr; off += n; return p; };
  sc.part_s = take((size_t)sc.nrt * Cin);
  sc.part_d = take((size_t)sc.nrt * Cin);
  sc.rowpart = take((size_t)3 * Cout * sc.ncw);
  sc.sig = take((size_t)2 * Cout * sc.ng);
  sc.route = take((size_t)4 * Cout);
  if (bytes) *bytes = off * 4 + 256;
  return sc;
}

size_t lwc_bwd_scratch_bytes(int64_t Cout, int64_t Cin) {
  size_t b = 0;
  lwc_bwd_carve(nullptr, Cout, Cin, Cin / 8, &b);      // groups of at least 8 columns
  return b;
}

__global__ void sigmoid_pair_kernel(const float* gl, const float* bl, int64_t n, float* ga, float* gb) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) { ga[i] = omq_sigmoid(gl[i]); gb[i] = omq_sigmoid(bl[i]); }
}

__device__ __forceinline__ float lwc_sig(const float* saved, const float* logit, int64_t k, int lwc) {
  if (!lwc) return 1.f;
  return saved ? saved[k] : omq_sigmoid(logit[k]);
}

#define LWC_BWD_RB 1          // rows whose loads are issued together

__global__ void __launch_bounds__(LWC_BWD_THREADS, 3) lwc_bwd_tile_kernel(LwcBwdArgs a, LwcBwdScratch sc) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t nchunk = a.Cin / 8;
  const int64_t c = (int64_t)blockIdx.x * LWC_BWD_THREADS + tid;     // this thread's chunk
  const bool valid = c < nchunk;
  const int64_t wglob = (int64_t)blockIdx.x * (LWC_BWD_THREADS / 32) + warp;
  const float Q = (float)((1 << a.wbits) - 1);
  const int gsz = a.group;
  const bool perch = gsz == a.Cin;
  const int64_t ngroups = a.Cin / gsz;
  const int lpg = perch ? 32 : gsz / 8;
  const int leader = lane & ~(lpg - 1);
  const int64_t gi = valid ? (c * 8) / gsz : 0;
  const bool want_s = a.ds != nullptr, want_d = a.ddelta != nullptr && a.dBt != nullptr;
  float sv[8];
  load8(a.s, valid ? c : 0, sv, 1.f);
  float acc_s[8], acc_d[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) { acc_s[e] = 0.f; acc_d[e] = 0.f; }
  const int64_t o0 = (int64_t)blockIdx.y * sc.rows;
  const int64_t o1 = min(a.Cout, o0 + sc.rows);
  const uint4 zero4 = make_uint4(0, 0, 0, 0);
  const float4 zf4 = make_float4(0.f, 0.f, 0.f, 0.f);

  for (int64_t ob = o0; ob < o1; ob += LWC_BWD_RB) {
    uint4 raw[LWC_BWD_RB];
    float4 ga4[LWC_BWD_RB], gb4[LWC_BWD_RB];
    float hv[LWC_BWD_RB], zv[LWC_BWD_RB], rv[LWC_BWD_RB], mv[LWC_BWD_RB], bv[LWC_BWD_RB], dbv[LWC_BWD_RB];
    int imv[LWC_BWD_RB], iMv[LWC_BWD_RB];
#pragma unroll
    for (int j = 0; j < LWC_BWD_RB; ++j) {      // every load of the batch first
      const int64_t o = ob + j;
      const bool rowok = o < o1;
      const bool ld = rowok && valid;
      const int64_t oo = rowok ? o : o0;
      raw[j] = ld ? __ldg(reinterpret_cast<const uint4*>(a.W + oo * a.Cin) + c) : zero4;
      ga4[j] = ld ? __ldg(reinterpret_cast<const float4*>(a.dWq + oo * a.ld_dwq) + 2 * c) : zf4;
      gb4[j] = ld ? __ldg(reinterpret_cast<const float4*>(a.dWq + oo * a.ld_dwq) + 2 * c + 1) : zf4;
      const int64_t k = perch ? oo : oo * ngroups + gi;
      hv[j] = a.h[k]; zv[j] = (float)a.z[k]; imv[j] = a.imin[k]; iMv[j] = a.imax[k];
      rv[j] = a.r ? a.r[oo] : 1.f;
      bv[j] = lwc_sig(a.gb, a.bl, k, a.lwc);
      mv[j] = a.mv ? a.mv[k] : lwc_wt(bf16_to_f(a.W[oo * a.Cin + imv[j]]), a.s, imv[j], rv[j]);
      dbv[j] = want_d ? a.dBt[oo] : 0.f;
    }
#pragma unroll
    for (int j = 0; j < LWC_BWD_RB; ++j) {
      const int64_t o = ob + j;
      if (o >= o1) break;                          // uniform across the CTA
      const float rr = rv[j];
      const int64_t k = perch ? o : o * ngroups + gi;
      float g[8] = {ga4[j].x, ga4[j].y, ga4[j].z, ga4[j].w, gb4[j].x, gb4[j].y, gb4[j].z, gb4[j].w};
      float w[8];
      unpack_bf16x8(raw[j], w);
      QState qs;
      qs.h = hv[j]; qs.z = zv[j]; qs.b = bv[j]; qs.m = mv[j];
      qs.rh = __frcp_rn(qs.h);
      qs.u = __fmul_rn(__fmul_rn(qs.b, qs.m), qs.rh);
      float Gh = 0.f, Gbm = 0.f, drm = 0.f;
      int inr_mask = 0;
      if (valid) {
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const float wt = __fmul_rn(__fmul_rn(w[e], sv[e]), rr);
          int inr;
          const float dh = omq_ste_dh(wt, qs, Q, &inr);
          Gh = fmaf(g[e], dh, Gh);
          if (!inr) Gbm += g[e];
          inr_mask |= inr << e;
        }
      }
      if (perch) {
        // warp partials of the row; routing to max/min is added by the per-row finalize
        Gh = warp_sum(Gh);
        Gbm = warp_sum(Gbm);
        if (valid) {
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const float d = ((inr_mask >> e) & 1) ? g[e] : 0.f;
            drm = fmaf(d * w[e], sv[e], drm);
            if (want_s) acc_s[e] = fmaf(d * w[e], rr, acc_s[e]);
            g[e] = d;
          }
          if (a.dWt) {
            float4* dst = reinterpret_cast<float4*>(a.dWt + o * a.Cin) + 2 * c;
            dst[0] = make_float4(g[0], g[1], g[2], g[3]);
            dst[1] = make_float4(g[4], g[5], g[6], g[7]);
          }
        }
        drm = warp_sum(drm);
        if (lane == 0 && wglob < sc.ncw) {
          sc.rowpart[(0 * a.Cout + o) * sc.ncw + wglob] = Gh;
          sc.rowpart[(1 * a.Cout + o) * sc.ncw + wglob] = Gbm;
          sc.rowpart[(2 * a.Cout + o) * sc.ncw + wglob] = drm;
        }
      } else {
        Gh = warp_sum(Gh, lpg);
        Gbm = warp_sum(Gbm, lpg);
        if (valid) {
          const int iM = iMv[j], im = imv[j];
          const float ga = lwc_sig(a.ga, a.gl, k, a.lwc), gb = qs.b;
          const float M = a.Mv ? a.Mv[k] : lwc_wt(bf16_to_f(a.W[o * a.Cin + iM]), a.s, iM, rr);
          const float m = qs.m;
          const float hr = __fdiv_rn(__fsub_rn(__fmul_rn(ga, M), __fmul_rn(gb, m)), Q);
          if (!(hr >= a.eps)) Gh = 0.f;                      // floored h: no gradient through h
          const float GaM = Gh / Q, Gbt = Gbm - Gh / Q;
          if (lane == leader && a.lwc) {
            const float dg = GaM * M * ga * (1.f - ga), db = Gbt * m * gb * (1.f - gb);
            if (a.accumulate) { a.dgl[k] += dg; a.dbl[k] += db; } else { a.dgl[k] = dg; a.dbl[k] = db; }
          }
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const int64_t col = c * 8 + e;
            float d = ((inr_mask >> e) & 1) ? g[e] : 0.f;
            if (col == iM) d += GaM * ga;
            if (col == im) d += Gbt * gb;
            drm = fmaf(d * w[e], sv[e], drm);
            if (want_s) acc_s[e] = fmaf(d * w[e], rr, acc_s[e]);
            g[e] = d;
          }
          if (a.dWt) {
            float4* dst = reinterpret_cast<float4*>(a.dWt + o * a.Cin) + 2 * c;
            dst[0] = make_float4(g[0], g[1], g[2], g[3]);
            dst[1] = make_float4(g[4], g[5], g[6], g[7]);
          }
        }
        if (a.dr) {
          drm = warp_sum(drm);
          if (lane == 0 && wglob < sc.ncw) sc.rowpart[(2 * a.Cout + o) * sc.ncw + wglob] = drm;
        }
      }
      if (want_d && valid) {
        const float f = dbv[j] * rr;
#pragma unroll
        for (int e = 0; e < 8; ++e) acc_d[e] = fmaf(f, w[e], acc_d[e]);
      }
    }
  }
  if (valid) {
    if (want_s) {
      float4* dst = reinterpret_cast<float4*>(sc.part_s + (int64_t)blockIdx.y * a.Cin) + 2 * c;
      dst[0] = make_float4(acc_s[0], acc_s[1], acc_s[2], acc_s[3]);
      dst[1] = make_float4(acc_s[4], acc_s[5], acc_s[6], acc_s[7]);
    }
    if (want_d) {
      float4* dst = reinterpret_cast<float4*>(sc.part_d + (int64_t)blockIdx.y * a.Cin) + 2 * c;
      dst[0] = make_float4(acc_d[0], acc_d[1], acc_d[2], acc_d[3]);
      dst[1] = make_float4(acc_d[4], acc_d[5], acc_d[6], acc_d[7]);
    }
  }
}

// Per-row completion of the LWC backward, one warp per weight row: the warp sums the row's warp
// partials (G_h, G_bm, dr); lane 0 forms dgamma, dbeta, dr and, for one group per row, the routing
// of dW~ to the row's max / min element.  The routing's share of ds is written to route[o] =
// (max column, value, min column, value) and added to the column partials by lwc_route_kernel.
__global__ void __launch_bounds__(256) lwc_bwd_finalize_kernel(LwcBwdArgs a, LwcBwdScratch sc, float4* route) {
  const int lane = threadIdx.x & 31;
  const int64_t o = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  if (o >= a.Cout) return;
  const bool perch = a.group == a.Cin;
  float Gh = 0.f, Gbm = 0.f, drm = 0.f;
  for (int64_t w = lane; w < sc.ncw; w += 32) {
    if (perch) {
      Gh += sc.rowpart[(0 * a.Cout + o) * sc.ncw + w];
      Gbm += sc.rowpart[(1 * a.Cout + o) * sc.ncw + w];
    }
    if (a.dr) drm += sc.rowpart[(2 * a.Cout + o) * sc.ncw + w];
  }
  Gh = warp_sum(Gh);
  Gbm = warp_sum(Gbm);
  drm = warp_sum(drm);
  if (lane != 0) return;
  const float rr = a.r ? a.r[o] : 1.f;
  if (perch) {
    const float Q = (float)((1 << a.wbits) - 1);
    const __nv_bfloat16* Wrow = a.W + o * a.Cin;
    const int iM = a.imax[o], im = a.imin[o];
    const float ga = lwc_sig(a.ga, a.gl, o, a.lwc), gb = lwc_sig(a.gb, a.bl, o, a.lwc);
    const float WM = bf16_to_f(Wrow[iM]), Wm = bf16_to_f(Wrow[im]);
    const float sM = a.s ? a.s[iM] : 1.f, sm = a.s ? a.s[im] : 1.f;
    const float M = a.Mv ? a.Mv[o] : __fmul_rn(__fmul_rn(WM, sM), rr);
    const float m = a.mv ? a.mv[o] : __fmul_rn(__fmul_rn(Wm, sm), rr);
    const float hr = __fdiv_rn(__fsub_rn(__fmul_rn(ga, M), __fmul_rn(gb, m)), Q);
    if (!(hr >= a.eps)) Gh = 0.f;
    const float GaM = Gh / Q, Gbt = Gbm - Gh / Q;
    if (a.lwc) {
      const float dg = GaM * M * ga * (1.f - ga), db = Gbt * m * gb * (1.f - gb);
      if (a.accumulate) { a.dgl[o] += dg; a.dbl[o] += db; } else { a.dgl[o] = dg; a.dbl[o] = db; }
    }
    const float rM = GaM * ga, rm = Gbt * gb;          // routing of dW~ to the max / min element
    drm += rM * WM * sM + rm * Wm * sm;
    if (a.ds) route[o] = make_float4((float)iM, rM * WM * rr, (float)im, rm * Wm * rr);
    if (a.dWt) {
      a.dWt[o * a.Cin + iM] += rM;
      a.dWt[o * a.Cin + im] += rm;
    }
  }
  if (a.dr) { if (a.accumulate_dr) a.dr[o] += drm; else a.dr[o] = drm; }
}

// Adds v to prow[col] for every lane's (col, v), col < 0 meaning none.  The lanes that share a
// column are summed in lane order and the first of them adds the sum: a fixed order, no atomics.
__device__ __forceinline__ void route_add(float* prow, int col, float v, int lane) {
  const unsigned m = __match_any_sync(0xffffffffu, col);           // lanes with this lane's column
  const unsigned dup = __ballot_sync(0xffffffffu, __popc(m) > 1);  // lanes in groups of two or more
  float sum = __popc(m) == 1 ? v : 0.f;
  for (unsigned u = dup; u; u &= u - 1) {                         // warp-uniform, increasing lanes
    const int l = __ffs(u) - 1;
    const float vl = __shfl_sync(0xffffffffu, v, l);
    if ((m >> l) & 1u) sum += vl;
  }
  if (col >= 0 && __ffs(m) - 1 == lane) prow[col] += sum;
}

// The max / min routing of ds (Eq. 2's max / min path) added into the LET column partials: one warp
// per partial row p (weight rows [p R, p R + R)), rows in chunks of 32 lanes, maxima before minima,
// so that ds does not depend on the order in which warps run.
__global__ void __launch_bounds__(256) lwc_route_kernel(const float4* __restrict__ route, int64_t Cout, int64_t R,
                                                        float* __restrict__ part_s, int64_t Cin) {
  const int lane = threadIdx.x & 31;
  const int64_t pidx = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  if (pidx * R >= Cout) return;                       // whole warp
  const int64_t r_end = min((pidx + 1) * R, Cout);
  float* prow = part_s + pidx * Cin;
  for (int64_t c0 = pidx * R; c0 < r_end; c0 += 32) {
    const int64_t o = c0 + lane;
    float4 e = make_float4(-1.f, 0.f, -1.f, 0.f);
    if (o < r_end) e = route[o];
    route_add(prow, (int)e.x, e.y, lane);
    __syncwarp();
    route_add(prow, (int)e.z, e.w, lane);
    __syncwarp();
  }
}

omq_status lwc_bwd_launch(cudaStream_t st, const LwcBwdArgs& a0, void* scratch) {
  OMQ_REQUIRE(lwc_group_ok(a0.Cin, a0.group), OMQ_ERR_UNSUPPORTED);
  OMQ_REQUIRE(scratch, OMQ_ERR_WORKSPACE);
  LwcBwdArgs a = a0;
  const bool perch = a.group == a.Cin;
  const int64_t ng = a.Cin / a.group;
  LwcBwdScratch sc = lwc_bwd_carve(scratch, a.Cout, a.Cin, ng, nullptr);
  if (a.lwc && (!a.ga || !a.gb)) {           // one sigmoid per group, not one per element
    const int64_t n = a.Cout * ng;
    sigmoid_pair_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(a.gl, a.bl, n, sc.sig, sc.sig + n);
    OMQ_LAUNCH_CHECK();
    a.ga = sc.sig;
    a.gb = sc.sig + n;
  }
  const int64_t ncol = (a.Cin / 8 + LWC_BWD_THREADS - 1) / LWC_BWD_THREADS;
  dim3 grid((unsigned)ncol, (unsigned)sc.nrt);
  lwc_bwd_tile_kernel<<<grid, LWC_BWD_THREADS, 0, st>>>(a, sc);
  OMQ_LAUNCH_CHECK();
  // the finalize and the routing of ds into the partial rows, then the partial rows are reduced
  if (perch || a.dr) {
    lwc_bwd_finalize_kernel<<<(unsigned)((a.Cout + 7) / 8), 256, 0, st>>>(a, sc, reinterpret_cast<float4*>(sc.route));
    OMQ_LAUNCH_CHECK();
  }
  if (perch && a.ds) {
    lwc_route_kernel<<<(unsigned)((sc.nrt + 7) / 8), 256, 0, st>>>(reinterpret_cast<const float4*>(sc.route), a.Cout,
                                                                    sc.rows, sc.part_s, a.Cin);
    OMQ_LAUNCH_CHECK();
  }
  if (a.ds) OMQ_TRY(omq_colsum_partials(st, sc.part_s, sc.nrt, a.Cin, a.ds, 1.f, a.accumulate_sd));
  if (a.ddelta && a.dBt) OMQ_TRY(omq_colsum_partials(st, sc.part_d, sc.nrt, a.Cin, a.ddelta, 1.f, a.accumulate_sd));
  return OMQ_OK;
}

omq_status lwc_bwd_fused_finish(cudaStream_t st, const LwcBwdArgs& a0, float* rowpart, int64_t ntn,
                                float* part_s, const float* part_d, int64_t nparts, float* route) {
  LwcBwdArgs a = a0;
  const bool perch = a.group == a.Cin;
  OMQ_REQUIRE(a.ga && a.gb, OMQ_ERR_INVALID_ARG);
  const bool want_s = a.ds != nullptr, want_d = a.ddelta && a.dBt;
  OMQ_REQUIRE((!want_s || part_s) && (!want_d || part_d), OMQ_ERR_INVALID_ARG);
  // the finalize and the routing of ds into the 32-row partials, then the partials are reduced
  if (perch || a.dr) {
    OMQ_REQUIRE(rowpart, OMQ_ERR_INVALID_ARG);
    OMQ_REQUIRE(!(perch && want_s) || (route && omq_aligned16(route) && nparts == (a.Cout + 31) / 32),
                OMQ_ERR_INVALID_ARG);
    LwcBwdScratch sc{};
    sc.rowpart = rowpart;
    sc.ncw = ntn;
    sc.ng = a.Cin / a.group;
    lwc_bwd_finalize_kernel<<<(unsigned)((a.Cout + 7) / 8), 256, 0, st>>>(a, sc, reinterpret_cast<float4*>(route));
    OMQ_LAUNCH_CHECK();
    if (perch && want_s) {
      lwc_route_kernel<<<(unsigned)((nparts + 7) / 8), 256, 0, st>>>(reinterpret_cast<const float4*>(route), a.Cout,
                                                                      32, part_s, a.Cin);
      OMQ_LAUNCH_CHECK();
    }
  }
  if (want_s && want_d) {
    OMQ_TRY(omq_colsum_partials2(st, ColsumJob{part_s, nparts, a.Cin, a.ds, 1.f, a.accumulate_sd},
                                 ColsumJob{part_d, nparts, a.Cin, a.ddelta, 1.f, a.accumulate_sd}));
  } else if (want_s) {
    OMQ_TRY(omq_colsum_partials(st, part_s, nparts, a.Cin, a.ds, 1.f, a.accumulate_sd));
  } else if (want_d) {
    OMQ_TRY(omq_colsum_partials(st, part_d, nparts, a.Cin, a.ddelta, 1.f, a.accumulate_sd));
  }
  return OMQ_OK;
}

// ================================================================================================
// packing of integer codes: code i of a row at bits [N i, N i + N) of its little-endian stream
// ================================================================================================
__global__ void pack_codes_kernel(const uint8_t* __restrict__ codes, int64_t Cout, int64_t Cin, int nbits,
                                  uint8_t* __restrict__ out) {
  const int64_t nchunk = Cin / 8;
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;     // one 8-code chunk
  if (i >= Cout * nchunk) return;
  const int64_t o = i / nchunk, c = i % nchunk;
  const uint2 raw = *reinterpret_cast<const uint2*>(codes + o * Cin + 8 * c);
  const uint32_t w[2] = {raw.x, raw.y};
  uint64_t acc = 0;
#pragma unroll
  for (int e = 0; e < 8; ++e) acc |= (uint64_t)((w[e >> 2] >> (8 * (e & 3))) & 0xffu) << (nbits * e);
  uint8_t* dst = out + o * (Cin * nbits / 8) + c * nbits;
  for (int b = 0; b < nbits; ++b) dst[b] = (uint8_t)(acc >> (8 * b));
}

omq_status pack_codes_launch(cudaStream_t st, const uint8_t* codes, int64_t Cout, int64_t Cin, int nbits, uint8_t* out) {
  OMQ_REQUIRE(Cin % 8 == 0 && nbits >= 1 && nbits <= 8, OMQ_ERR_SHAPE);
  const int64_t n = Cout * (Cin / 8);
  pack_codes_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(codes, Cout, Cin, nbits, out);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

__global__ void norm_fold_kernel(int64_t n, const float* s, const float* d, float* gain, float* bias) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  gain[i] = 1.0f / s[i];
  bias[i] = -d[i] / s[i];
}

omq_status norm_fold_launch(cudaStream_t st, int64_t n, const float* s, const float* d, float* gain, float* bias) {
  norm_fold_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(n, s, d, gain, bias);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

// ================================================================================================
// reductions, loss, small vector kernels
// ================================================================================================
// 32 columns per CTA, eight row phases per column; fixed summation order (deterministic).
// Used when the column count or a pointer does not allow 16-byte accesses.
__global__ void omq_colsum_partials_kernel(const float* __restrict__ part, int64_t P, int64_t C,
                                           float* __restrict__ out, float scale, int accumulate) {
  __shared__ float red[8][33];
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  const int64_t c = (int64_t)blockIdx.x * 32 + tx;
  float s = 0.f;
  if (c < C)
    for (int64_t p = ty; p < P; p += 8) s += part[p * C + c];
  red[ty][tx] = s;
  __syncthreads();
  if (ty == 0 && c < C) {
    float t = 0.f;
#pragma unroll
    for (int i = 0; i < 8; ++i) t += red[i][tx];
    t *= scale;
    out[c] = accumulate ? out[c] + t : t;
  }
}

// 128 columns per cluster of eight CTAs: CTA k of the cluster sums the k-th contiguous eighth of
// the P partial rows (its eight warps take every eighth row, four loads in flight per thread),
// and CTA 0 adds the eight CTA sums in rank order through distributed shared memory.  The
// summation order is fixed, so the result does not depend on scheduling.
#define COLSUM_CLUSTER 8
__device__ __forceinline__ void add4(float4& a, const float4 b) { a.x += b.x; a.y += b.y; a.z += b.z; a.w += b.w; }

// blockIdx.z selects one of two independent reductions of one launch
__global__ void __cluster_dims__(1, COLSUM_CLUSTER, 1) __launch_bounds__(256)
    colsum_cluster_kernel(ColsumJob j0, ColsumJob j1) {
  const ColsumJob& J = blockIdx.z == 0 ? j0 : j1;
  const float* __restrict__ part = J.part;
  const int64_t P = J.P, C = J.C;
  float* __restrict__ out = J.out;
  const float scale = J.scale;
  const int accumulate = J.accumulate;
  if ((int64_t)blockIdx.x * 128 >= C) return;     // the narrower job of a pair: whole cluster leaves
  __shared__ float4 red[8][32];
  __shared__ float4 cta_sum[32];
  cg::cluster_group cluster = cg::this_cluster();
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const unsigned rank = cluster.block_rank();
  const int64_t nc4 = C / 4;
  const int64_t c4 = (int64_t)blockIdx.x * 32 + lane;
  const int64_t rows_per = (P + COLSUM_CLUSTER - 1) / COLSUM_CLUSTER;
  const int64_t r0 = (int64_t)rank * rows_per, r1 = min(P, r0 + rows_per);
  float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
  if (c4 < nc4) {
    const float4* base = reinterpret_cast<const float4*>(part) + c4;
    int64_t r = r0 + w;
    for (; r + 24 < r1; r += 32) {
      const float4 v0 = __ldg(base + r * nc4), v1 = __ldg(base + (r + 8) * nc4);
      const float4 v2 = __ldg(base + (r + 16) * nc4), v3 = __ldg(base + (r + 24) * nc4);
      add4(s, v0); add4(s, v1); add4(s, v2); add4(s, v3);
    }
    for (; r < r1; r += 8) add4(s, __ldg(base + r * nc4));
  }
  red[w][lane] = s;
  __syncthreads();
  if (w == 0) {
    float4 t = red[0][lane];
#pragma unroll
    for (int k = 1; k < 8; ++k) add4(t, red[k][lane]);
    cta_sum[lane] = t;
  }
  cluster.sync();
  if (rank == 0 && w == 0 && c4 < nc4) {
    float4 t = cta_sum[lane];
#pragma unroll
    for (int k = 1; k < COLSUM_CLUSTER; ++k) add4(t, cluster.map_shared_rank(cta_sum, k)[lane]);
    t.x *= scale; t.y *= scale; t.z *= scale; t.w *= scale;
    float4* o = reinterpret_cast<float4*>(out) + c4;
    if (accumulate) add4(t, *o);
    *o = t;
  }
  cluster.sync();                  // keep every CTA's shared memory alive until CTA 0 has read it
}

static bool colsum_vec_ok(const ColsumJob& j) {
  return j.C % 4 == 0 && omq_aligned16(j.part) && omq_aligned16(j.out);
}

omq_status omq_colsum_partials2(cudaStream_t st, const ColsumJob& a, const ColsumJob& b) {
  if (!colsum_vec_ok(a) || !colsum_vec_ok(b)) {
    OMQ_TRY(omq_colsum_partials(st, a.part, a.P, a.C, a.out, a.scale, a.accumulate));
    return omq_colsum_partials(st, b.part, b.P, b.C, b.out, b.scale, b.accumulate);
  }
  const int64_t C = a.C > b.C ? a.C : b.C;
  dim3 grid((unsigned)((C / 4 + 31) / 32), COLSUM_CLUSTER, 2);
  colsum_cluster_kernel<<<grid, 256, 0, st>>>(a, b);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

omq_status omq_colsum_partials(cudaStream_t st, const float* part, int64_t P, int64_t C, float* out,
                               float scale, int accumulate) {
  ColsumJob j{part, P, C, out, scale, accumulate};
  if (colsum_vec_ok(j)) {
    dim3 grid((unsigned)((C / 4 + 31) / 32), COLSUM_CLUSTER);
    colsum_cluster_kernel<<<grid, 256, 0, st>>>(j, j);
  } else {
    omq_colsum_partials_kernel<<<(unsigned)((C + 31) / 32), 256, 0, st>>>(part, P, C, out, scale, accumulate);
  }
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

// stage 1 of a column sum over rows: part[blockIdx.y, n] = sum of X[t, n] over 128 rows
__global__ void colsum_rows_kernel(const float* __restrict__ X, int64_t T, int64_t N, int64_t ldx,
                                   float* __restrict__ part) {
  int64_t n = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (n >= N) return;
  int64_t t0 = (int64_t)blockIdx.y * 128, t1 = min(T, t0 + 128);
  float s = 0.f;
  for (int64_t t = t0; t < t1; ++t) s += X[t * ldx + n];
  part[(int64_t)blockIdx.y * N + n] = s;
}

// the same with 16-byte loads: a CTA covers 128 columns x 128 rows, lane l of warp w reads
// columns 4l .. 4l+3 of rows w, w + 8, ... (four loads in flight), and the eight warp sums are added
// in warp order
__global__ void __launch_bounds__(256) colsum_rows_vec_kernel(const float* __restrict__ X, int64_t T, int64_t N,
                                                              int64_t ldx, float* __restrict__ part) {
  __shared__ float4 red[8][32];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int64_t c = (int64_t)blockIdx.x * 128 + 4 * lane;
  const int64_t t0 = (int64_t)blockIdx.y * 128, t1 = min(T, t0 + 128);
  float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
  if (c < N) {
    int64_t t = t0 + w;
    for (; t + 24 < t1; t += 32) {
      const float4 v0 = __ldg(reinterpret_cast<const float4*>(X + t * ldx + c));
      const float4 v1 = __ldg(reinterpret_cast<const float4*>(X + (t + 8) * ldx + c));
      const float4 v2 = __ldg(reinterpret_cast<const float4*>(X + (t + 16) * ldx + c));
      const float4 v3 = __ldg(reinterpret_cast<const float4*>(X + (t + 24) * ldx + c));
      add4(s, v0); add4(s, v1); add4(s, v2); add4(s, v3);
    }
    for (; t < t1; t += 8) add4(s, __ldg(reinterpret_cast<const float4*>(X + t * ldx + c)));
  }
  red[w][lane] = s;
  __syncthreads();
  if (w == 0 && c < N) {
    float4 r = red[0][lane];
#pragma unroll
    for (int k = 1; k < 8; ++k) add4(r, red[k][lane]);
    *reinterpret_cast<float4*>(part + (int64_t)blockIdx.y * N + c) = r;
  }
}

int64_t colsum_rows_parts(int64_t T) { return (T + 127) / 128; }

// part[p, c] = sum of the bf16 X[t, c] (in fp32) over the 128 rows t of slab p; each thread sums 8
// columns (one 16-byte load per row), the eight warps of a CTA stride the slab's rows
__global__ void __launch_bounds__(256) colsum_rows_bf16_kernel(const __nv_bfloat16* __restrict__ X, int64_t T,
                                                               int64_t N, int64_t ldx, float* __restrict__ part) {
  __shared__ float red[8][32][9];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int64_t c = (int64_t)blockIdx.x * 256 + 8 * lane;
  const int64_t t0 = (int64_t)blockIdx.y * 128, t1 = min(T, t0 + 128);
  float s[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  if (c < N) {
    int64_t t = t0 + w;
    for (; t + 24 < t1; t += 32) {
      uint4 v[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) v[i] = __ldg(reinterpret_cast<const uint4*>(X + (t + 8 * i) * ldx + c));
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        float f[8];
        unpack_bf16x8(v[i], f);
#pragma unroll
        for (int e = 0; e < 8; ++e) s[e] += f[e];
      }
    }
    for (; t < t1; t += 8) {
      float f[8];
      unpack_bf16x8(__ldg(reinterpret_cast<const uint4*>(X + t * ldx + c)), f);
#pragma unroll
      for (int e = 0; e < 8; ++e) s[e] += f[e];
    }
  }
#pragma unroll
  for (int e = 0; e < 8; ++e) red[w][lane][e] = s[e];
  __syncthreads();
  if (w == 0 && c < N) {
    float r[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) r[e] = red[0][lane][e];
#pragma unroll
    for (int k = 1; k < 8; ++k)
#pragma unroll
      for (int e = 0; e < 8; ++e) r[e] += red[k][lane][e];
    float4* dst = reinterpret_cast<float4*>(part + (int64_t)blockIdx.y * N + c);
    dst[0] = make_float4(r[0], r[1], r[2], r[3]);
    dst[1] = make_float4(r[4], r[5], r[6], r[7]);
  }
}

omq_status colsum_rows_bf16(cudaStream_t st, const __nv_bfloat16* X, int64_t T, int64_t N, int64_t ldx, float* part,
                            float* out, float scale, int accumulate) {
  OMQ_REQUIRE(N % 8 == 0 && ldx % 8 == 0 && omq_aligned16(X) && omq_aligned16(part), OMQ_ERR_ALIGN);
  dim3 grid((unsigned)((N + 255) / 256), (unsigned)colsum_rows_parts(T));
  colsum_rows_bf16_kernel<<<grid, 256, 0, st>>>(X, T, N, ldx, part);
  OMQ_LAUNCH_CHECK();
  return omq_colsum_partials(st, part, colsum_rows_parts(T), N, out, scale, accumulate);
}

omq_status colsum_rows(cudaStream_t st, const float* X, int64_t T, int64_t N, int64_t ldx, float* part,
                       float* out, float scale, int accumulate) {
  if (N % 4 == 0 && ldx % 4 == 0 && omq_aligned16(X) && omq_aligned16(part)) {
    dim3 grid((unsigned)((N + 127) / 128), (unsigned)colsum_rows_parts(T));
    colsum_rows_vec_kernel<<<grid, 256, 0, st>>>(X, T, N, ldx, part);
  } else {
    dim3 grid((unsigned)((N + 255) / 256), (unsigned)colsum_rows_parts(T));
    colsum_rows_kernel<<<grid, 256, 0, st>>>(X, T, N, ldx, part);
  }
  OMQ_LAUNCH_CHECK();
  return omq_colsum_partials(st, part, colsum_rows_parts(T), N, out, scale, accumulate);
}

__global__ void loss_partial_kernel(int64_t n, const float* __restrict__ Yq, const float* __restrict__ Yfp,
                                    float* __restrict__ dY, __nv_bfloat16* __restrict__ dYb,
                                    float* __restrict__ part) {
  __shared__ float red_f[64];
  float s = 0.f;
  const float g = 2.0f / (float)n;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
    float d = Yq[i] - Yfp[i];
    s = fmaf(d, d, s);
    float gd = g * d;
    if (dY) dY[i] = gd;
    if (dYb) dYb[i] = f_to_bf16(gd);
  }
  float2 t = block_sum2(s, 0.f, red_f);
  if (threadIdx.x == 0) part[blockIdx.x] = t.x;
}

__global__ void loss_final_kernel(const float* __restrict__ part, int P, int64_t n, float* loss) {
  __shared__ float red_f[64];
  float s = 0.f;
  for (int i = threadIdx.x; i < P; i += blockDim.x) s += part[i];
  float2 t = block_sum2(s, 0.f, red_f);
  if (threadIdx.x == 0) *loss = t.x / (float)n;
}

int64_t loss_parts(int64_t n) {
  int64_t b = (n + 1023) / 1024;
  return b < 1024 ? b : 1024;
}

omq_status loss_launch(cudaStream_t st, int64_t n, const float* Yq, const float* Yfp, float* loss,
                       float* dY, __nv_bfloat16* dYb, float* part) {
  int P = (int)loss_parts(n);
  loss_partial_kernel<<<P, 256, 0, st>>>(n, Yq, Yfp, dY, dYb, part);
  OMQ_LAUNCH_CHECK();
  loss_final_kernel<<<1, 256, 0, st>>>(part, P, n, loss);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

__global__ void vec_fill_kernel(float* p, int64_t n, float v) {
  int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) p[i] = v;
}
omq_status vec_fill(cudaStream_t st, float* p, int64_t n, float v) {
  vec_fill_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(p, n, v);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

__global__ void vec_copy_kernel(float* d, const float* s, int64_t n) {
  int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) d[i] = s[i];
}
omq_status vec_copy(cudaStream_t st, float* dst, const float* src, int64_t n) {
  vec_copy_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(dst, src, n);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

__global__ void gqa_expand_kernel(const float* src, float* dst, int n_kv, int rep, int hd, int op) {
  int i = blockIdx.x * blockDim.x + threadIdx.x;
  int n = n_kv * rep * hd;
  if (i >= n) return;
  int h = i / hd, j = i % hd;
  float v = src[(h / rep) * hd + j];
  dst[i] = op == 1 ? 1.0f / v : v;
}
omq_status gqa_expand(cudaStream_t st, const float* src, float* dst, int n_kv, int rep, int hd, int op) {
  int n = n_kv * rep * hd;
  gqa_expand_kernel<<<(n + 255) / 256, 256, 0, st>>>(src, dst, n_kv, rep, hd, op);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

__global__ void gqa_fold_kernel(const float* src, float* dst, int n_kv, int rep, int hd, int accumulate) {
  int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= n_kv * hd) return;
  int kv = c / hd, j = c % hd;
  float s = 0.f;
  for (int r = 0; r < rep; ++r) s += src[(kv * rep + r) * hd + j];
  dst[c] = accumulate ? dst[c] + s : s;
}
omq_status gqa_fold(cudaStream_t st, const float* src, float* dst, int n_kv, int rep, int hd, int accumulate) {
  int n = n_kv * hd;
  gqa_fold_kernel<<<(n + 255) / 256, 256, 0, st>>>(src, dst, n_kv, rep, hd, accumulate);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

// ================================================================================================
// LET apply (Eq. 3) as a standalone operation
// ================================================================================================
__global__ void let_x_kernel(const float* X, int64_t T, int64_t C, const float* s, const float* d, float* Xt) {
  int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= T * C) return;
  int64_t c = i % C;
  Xt[i] = __fdiv_rn(X[i] - d[c], s[c]);
}

__global__ void let_w_kernel(const __nv_bfloat16* W, int64_t Cout, int64_t Cin, const float* s, float* Wt) {
  int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= Cout * Cin) return;
  Wt[i] = __fmul_rn(bf16_to_f(W[i]), s[i % Cin]);
}

__global__ void let_b_kernel(const __nv_bfloat16* W, int64_t Cout, int64_t Cin, const float* B, const float* d, float* Bt) {
  __shared__ float red_f[64];
  int64_t o = blockIdx.x;
  float acc = 0.f;
  for (int64_t i = threadIdx.x; i < Cin; i += blockDim.x) acc = fmaf(bf16_to_f(W[o * Cin + i]), d[i], acc);
  float2 t = block_sum2(acc, 0.f, red_f);
  if (threadIdx.x == 0) Bt[o] = (B ? B[o] : 0.f) + t.x;
}

// ================================================================================================
// AdamW (Sec. 4.1, weight decay 0 by default)
// ================================================================================================
__global__ void adamw_kernel(int64_t n, float* p, const float* g, float* m, float* v, float lr, float b1, float b2,
                             float eps, float wd, float bc1, float bc2) {
  int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  float gi = g[i];
  float mi = b1 * m[i] + (1.f - b1) * gi;
  float vi = b2 * v[i] + (1.f - b2) * gi * gi;
  m[i] = mi;
  v[i] = vi;
  float pi = p[i];
  p[i] = pi - lr * (mi / bc1) / (sqrtf(vi / bc2) + eps) - lr * wd * pi;
}

// the same, t read from device memory; bias corrections formed once per CTA
__global__ void adamw_dev_kernel(int64_t n, float* p, const float* g, float* m, float* v, float lr, float b1, float b2,
                                 float eps, float wd, const int32_t* step) {
  __shared__ float bc[2];
  if (threadIdx.x == 0) {
    const float t = (float)*step;
    bc[0] = 1.f - powf(b1, t);
    bc[1] = 1.f - powf(b2, t);
  }
  __syncthreads();
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const float gi = g[i];
  const float mi = b1 * m[i] + (1.f - b1) * gi;
  const float vi = b2 * v[i] + (1.f - b2) * gi * gi;
  m[i] = mi;
  v[i] = vi;
  const float pi = p[i];
  p[i] = pi - lr * (mi / bc[0]) / (sqrtf(vi / bc[1]) + eps) - lr * wd * pi;
}

__global__ void step_advance_kernel(int32_t* step) { *step += 1; }

// ================================================================================================
// C ABI: kernel-level entry points
// ================================================================================================
extern "C" {

omq_status omq_let_apply(omq_stream_t stream, int64_t T, int64_t Cin, int64_t Cout, const float* X,
                         const void* W, const float* B, const float* s, const float* delta, float* Xt,
                         float* Wt, float* Bt, const omq_qcfg* cfg) {
  (void)cfg;
  cudaStream_t st = (cudaStream_t)stream;
  OMQ_REQUIRE(T > 0 && Cin > 0 && Cout > 0, OMQ_ERR_SHAPE);
  OMQ_REQUIRE(s && delta, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(Cin % 8 == 0, OMQ_ERR_ALIGN);
  if (Xt) {
    OMQ_REQUIRE(X, OMQ_ERR_INVALID_ARG);
    let_x_kernel<<<(unsigned)((T * Cin + 255) / 256), 256, 0, st>>>(X, T, Cin, s, delta, Xt);
    OMQ_LAUNCH_CHECK();
  }
  if (Wt) {
    OMQ_REQUIRE(W, OMQ_ERR_INVALID_ARG);
    let_w_kernel<<<(unsigned)((Cout * Cin + 255) / 256), 256, 0, st>>>((const __nv_bfloat16*)W, Cout, Cin, s, Wt);
    OMQ_LAUNCH_CHECK();
  }
  if (Bt) {
    OMQ_REQUIRE(W, OMQ_ERR_INVALID_ARG);
    let_b_kernel<<<(unsigned)Cout, 256, 0, st>>>((const __nv_bfloat16*)W, Cout, Cin, B, delta, Bt);
    OMQ_LAUNCH_CHECK();
  }
  return OMQ_OK;
}

omq_status omq_lwc_fakequant_fwd(omq_stream_t stream, int64_t Cout, int64_t Cin, const void* W, const float* s,
                                 const float* r, const float* gamma_logit, const float* beta_logit, void* Wq,
                                 uint8_t* codes, float* h, int32_t* z, int32_t* argmax, int32_t* argmin,
                                 const float* bias_delta, const float* bias_shift, float* Bt, const omq_qcfg* cfg) {
  OMQ_TRY(omq_check_cfg(cfg));
  OMQ_REQUIRE(Cout > 0 && Cin > 0, OMQ_ERR_SHAPE);
  OMQ_REQUIRE(W, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(Cin % 8 == 0 && omq_aligned16(W) && (!Wq || omq_aligned16(Wq)), OMQ_ERR_ALIGN);
  OMQ_REQUIRE(!codes || ((uintptr_t)codes & 7) == 0, OMQ_ERR_ALIGN);
  const int g = cfg->group == 0 ? (int)Cin : cfg->group;
  OMQ_REQUIRE(Cin % g == 0, OMQ_ERR_SHAPE);
  if (cfg->wbits < 16) OMQ_REQUIRE(h && z && argmax && argmin && gamma_logit && beta_logit, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(!Bt || bias_delta, OMQ_ERR_INVALID_ARG);
  LwcFwdArgs a{};
  a.W = (const __nv_bfloat16*)W; a.Cout = Cout; a.Cin = Cin; a.group = g;
  a.s = s; a.r = r; a.gl = gamma_logit; a.bl = beta_logit; a.lwc = 1;
  a.Wq = (__nv_bfloat16*)Wq; a.codes = codes; a.h = h; a.z = z; a.imax = argmax; a.imin = argmin;
  a.bias_delta = bias_delta; a.bias_shift = bias_shift; a.Bt = Bt;
  a.wbits = cfg->wbits; a.eps = cfg->h_eps; a.status = cfg->dev_status;
  return lwc_fwd_launch((cudaStream_t)stream, a);
}

size_t omq_lwc_bwd_workspace_size(int64_t Cout, int64_t Cin) { return lwc_bwd_scratch_bytes(Cout, Cin); }

omq_status omq_lwc_fakequant_bwd(omq_stream_t stream, int64_t Cout, int64_t Cin, const void* W, const float* s,
                                 const float* r, const float* gamma_logit, const float* beta_logit, const float* h,
                                 const int32_t* z, const int32_t* argmax, const int32_t* argmin, const float* dWq,
                                 float* dgamma, float* dbeta, float* dWt, float* ds, float* dr, const float* dBt,
                                 float* ddelta, void* workspace, size_t ws_bytes, const omq_qcfg* cfg) {
  OMQ_TRY(omq_check_cfg(cfg));
  OMQ_REQUIRE(Cout > 0 && Cin > 0, OMQ_ERR_SHAPE);
  OMQ_REQUIRE(cfg->wbits < 16, OMQ_ERR_UNSUPPORTED);
  OMQ_REQUIRE(W && dWq && h && z && argmax && argmin && gamma_logit && beta_logit && dgamma && dbeta, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(Cin % 8 == 0 && omq_aligned16(W) && omq_aligned16(dWq) && (!dWt || omq_aligned16(dWt)), OMQ_ERR_ALIGN);
  OMQ_REQUIRE(!s || omq_aligned16(s), OMQ_ERR_ALIGN);
  const int g = cfg->group == 0 ? (int)Cin : cfg->group;
  OMQ_REQUIRE(Cin % g == 0, OMQ_ERR_SHAPE);
  OMQ_REQUIRE(!ddelta || dBt, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(workspace && ws_bytes >= omq_lwc_bwd_workspace_size(Cout, Cin), OMQ_ERR_WORKSPACE);
  OMQ_REQUIRE(omq_aligned16(workspace), OMQ_ERR_ALIGN);
  LwcBwdArgs a{};
  a.W = (const __nv_bfloat16*)W; a.Cout = Cout; a.Cin = Cin; a.group = g; a.s = s; a.r = r;
  a.gl = gamma_logit; a.bl = beta_logit; a.lwc = 1; a.ga = nullptr; a.gb = nullptr;
  a.h = h; a.z = z; a.imax = argmax; a.imin = argmin;
  a.dWq = dWq; a.ld_dwq = Cin; a.dgl = dgamma; a.dbl = dbeta; a.dWt = dWt; a.dr = dr; a.dBt = dBt;
  a.ds = ds; a.ddelta = ddelta;
  a.wbits = cfg->wbits; a.eps = cfg->h_eps; a.accumulate = cfg->accumulate; a.accumulate_sd = cfg->accumulate;
  a.accumulate_dr = cfg->accumulate;
  return lwc_bwd_launch((cudaStream_t)stream, a, workspace);
}

omq_status omq_act_quant_per_token(omq_stream_t stream, int64_t T, int64_t C, const float* X, const float* s,
                                   const float* delta, void* Xq, uint8_t* codes, float* h, int32_t* z,
                                   int32_t* argmax, int32_t* argmin, const omq_qcfg* cfg) {
  OMQ_TRY(omq_check_cfg(cfg));
  OMQ_REQUIRE(T > 0 && C > 0, OMQ_ERR_SHAPE);
  OMQ_REQUIRE(X && Xq, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(C % 8 == 0 && omq_aligned16(X) && omq_aligned16(Xq), OMQ_ERR_ALIGN);
  if (cfg->abits < 16) OMQ_REQUIRE(h && z && argmax && argmin, OMQ_ERR_INVALID_ARG);
  ActFwdArgs a{};
  a.producer = (s || delta) ? AP_LET : AP_PLAIN;
  a.X = X; a.ldx = C; a.s = s; a.delta = delta; a.T = T; a.C = C;
  a.Xq = (__nv_bfloat16*)Xq; a.ldq = C; a.codes = codes; a.h = h; a.z = z; a.imax = argmax; a.imin = argmin;
  a.abits = cfg->abits; a.eps = cfg->h_eps; a.status = cfg->dev_status;
  return act_fwd_launch((cudaStream_t)stream, a);
}

size_t omq_act_bwd_workspace_size(int64_t T, int64_t C) {
  return (size_t)(2 * ((T + 3) / 4) * C) * sizeof(float) + 256;
}

omq_status omq_act_quant_per_token_bwd(omq_stream_t stream, int64_t T, int64_t C, const float* X, const float* s,
                                       const float* delta, const float* h, const int32_t* z, const int32_t* argmax,
                                       const int32_t* argmin, const float* dXq, float* dX, float* ds, float* ddelta,
                                       void* workspace, size_t ws_bytes, const omq_qcfg* cfg) {
  OMQ_TRY(omq_check_cfg(cfg));
  OMQ_REQUIRE(T > 0 && C > 0, OMQ_ERR_SHAPE);
  OMQ_REQUIRE(X && dXq, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(C % 8 == 0 && omq_aligned16(X) && omq_aligned16(dXq), OMQ_ERR_ALIGN);
  if (cfg->abits < 16) OMQ_REQUIRE(h && z && argmax && argmin, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE((!ds && !ddelta) || (s && delta), OMQ_ERR_INVALID_ARG);
  const bool need_ws = ds || ddelta;
  const int64_t P = (T + 3) / 4;
  if (need_ws) OMQ_REQUIRE(workspace && ws_bytes >= omq_act_bwd_workspace_size(T, C), OMQ_ERR_WORKSPACE);
  cudaStream_t st = (cudaStream_t)stream;
  ActBwdArgs a{};
  a.producer = (s || delta) ? AP_LET : AP_PLAIN;
  a.X = X; a.ldx = C; a.s = s; a.delta = delta; a.T = T; a.C = C;
  a.h = h; a.z = z; a.imax = argmax; a.imin = argmin; a.dXq = dXq; a.lddq = C;
  a.dX = dX; a.lddx = C; a.rows_per_cta = 4;
  a.part_s = need_ws ? (float*)workspace : nullptr;
  a.part_d = need_ws ? (float*)workspace + P * C : nullptr;
  a.abits = cfg->abits; a.eps = cfg->h_eps;
  OMQ_TRY(act_bwd_launch(st, a));
  if (ds) OMQ_TRY(omq_colsum_partials(st, a.part_s, P, C, ds, 1.f, cfg->accumulate));
  if (ddelta) OMQ_TRY(omq_colsum_partials(st, a.part_d, P, C, ddelta, 1.f, cfg->accumulate));
  return OMQ_OK;
}

size_t omq_loss_workspace_size(int64_t n) { return (size_t)loss_parts(n) * sizeof(float) + 256; }

omq_status omq_block_loss(omq_stream_t stream, int64_t n, const float* Yq, const float* Yfp, float* loss, float* dY,
                          void* dY_bf16, void* workspace, size_t ws_bytes) {
  OMQ_REQUIRE(n > 0, OMQ_ERR_SHAPE);
  OMQ_REQUIRE(Yq && Yfp && loss, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(workspace && ws_bytes >= omq_loss_workspace_size(n), OMQ_ERR_WORKSPACE);
  return loss_launch((cudaStream_t)stream, n, Yq, Yfp, loss, dY, (__nv_bfloat16*)dY_bf16, (float*)workspace);
}

// ---- block loss without a caller workspace -------------------------------------------------------
// Some callers cannot allocate device memory for a workspace: code whose device memory is owned by
// another framework's fixed arena, plugin interfaces that pass only inputs and outputs, and code
// that must not call cudaMalloc/cudaFree while other work is in flight (both can synchronize the
// device).  This variant keeps the loss's partial sums in a file-scope device array instead.
#define OMQ_NOALLOC_LOSS_PARTS 1024                   // partial sums: 4 KB per device
#define OMQ_NOALLOC_MAX_DEVICES 64
static __device__ __align__(256) float g_noalloc_loss_part[OMQ_NOALLOC_LOSS_PARTS];
static std::atomic<float*> g_noalloc_loss_ptr[OMQ_NOALLOC_MAX_DEVICES];

omq_status omq_block_loss_noalloc(omq_stream_t stream, int64_t n, const float* Yq, const float* Yfp, float* loss,
                                  float* dY, void* dY_bf16) {
  OMQ_REQUIRE(n > 0 && n <= OMQ_NOALLOC_LOSS_MAX_N, OMQ_ERR_SHAPE);
  OMQ_REQUIRE(Yq && Yfp && loss, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(loss_parts(n) <= OMQ_NOALLOC_LOSS_PARTS, OMQ_ERR_SHAPE);
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return OMQ_ERR_CUDA;
  OMQ_REQUIRE(dev >= 0 && dev < OMQ_NOALLOC_MAX_DEVICES, OMQ_ERR_UNSUPPORTED);
  // The host-side name of the array is not a device address: ask the runtime for the array's
  // address on the current device whenever the stream is not being captured, so that a device
  // reset (which reloads the module) cannot leave a stale address behind; otherwise reuse the
  // address of the last lookup.
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing((cudaStream_t)stream, &cs) != cudaSuccess) {
    cudaGetLastError();
    cs = cudaStreamCaptureStatusActive;
  }
  float* part = g_noalloc_loss_ptr[dev].load();
  if (cs == cudaStreamCaptureStatusNone) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_loss_part) != cudaSuccess || !p) return OMQ_ERR_CUDA;
    part = static_cast<float*>(p);
    g_noalloc_loss_ptr[dev].store(part);
  }
  if (!part) return OMQ_ERR_CUDA;                 // first call on this device inside a capture
  // every partial the final reduction reads is written by this call, so nothing needs clearing
  return loss_launch((cudaStream_t)stream, n, Yq, Yfp, loss, dY, (__nv_bfloat16*)dY_bf16, part);
}

omq_status omq_adamw_update(omq_stream_t stream, int64_t n, float* p, const float* g, float* m, float* v, float lr,
                            float beta1, float beta2, float eps, float weight_decay, int32_t step) {
  OMQ_REQUIRE(n > 0, OMQ_ERR_SHAPE);
  OMQ_REQUIRE(p && g && m && v && step >= 1, OMQ_ERR_INVALID_ARG);
  float bc1 = 1.f - powf(beta1, (float)step), bc2 = 1.f - powf(beta2, (float)step);
  adamw_kernel<<<(unsigned)((n + 255) / 256), 256, 0, (cudaStream_t)stream>>>(n, p, g, m, v, lr, beta1, beta2, eps,
                                                                              weight_decay, bc1, bc2);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

omq_status omq_adamw_update_dev(omq_stream_t stream, int64_t n, float* p, const float* g, float* m, float* v,
                                float lr, float beta1, float beta2, float eps, float weight_decay,
                                const int32_t* step_dev) {
  OMQ_REQUIRE(n > 0, OMQ_ERR_SHAPE);
  OMQ_REQUIRE(p && g && m && v && step_dev, OMQ_ERR_INVALID_ARG);
  adamw_dev_kernel<<<(unsigned)((n + 255) / 256), 256, 0, (cudaStream_t)stream>>>(n, p, g, m, v, lr, beta1, beta2,
                                                                                  eps, weight_decay, step_dev);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

omq_status omq_step_advance(omq_stream_t stream, int32_t* step_dev) {
  OMQ_REQUIRE(step_dev, OMQ_ERR_INVALID_ARG);
  step_advance_kernel<<<1, 1, 0, (cudaStream_t)stream>>>(step_dev);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

omq_status omq_stream_status(omq_stream_t stream, const int32_t* dev_status, int32_t* host_out) {
  OMQ_REQUIRE(dev_status && host_out, OMQ_ERR_INVALID_ARG);
  if (cudaMemcpyAsync(host_out, dev_status, sizeof(int32_t), cudaMemcpyDeviceToHost, (cudaStream_t)stream) != cudaSuccess)
    return OMQ_ERR_CUDA;
  if (cudaStreamSynchronize((cudaStream_t)stream) != cudaSuccess) return OMQ_ERR_CUDA;
  return OMQ_OK;
}

const char* omq_status_string(omq_status s) {
  switch (s) {
    case OMQ_OK: return "ok";
    case OMQ_ERR_INVALID_ARG: return "invalid argument";
    case OMQ_ERR_SHAPE: return "bad shape";
    case OMQ_ERR_ALIGN: return "misaligned pointer or inner dimension";
    case OMQ_ERR_UNSUPPORTED: return "unsupported configuration";
    case OMQ_ERR_CUDA: return "CUDA launch failure";
    case OMQ_ERR_TIMEOUT: return "device wait timed out";
    case OMQ_ERR_WORKSPACE: return "workspace too small";
  }
  return "unknown status";
}

int32_t omq_version(void) { return OMQ_VERSION; }

int64_t omq_launch_count(void) { return (int64_t)g_launches.load(); }

}  // extern "C"
