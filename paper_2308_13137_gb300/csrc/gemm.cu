// Dense bf16 matrix product on the 5th-generation tensor cores (sm_103a):
// TMA (cp.async.bulk.tensor, 128-byte swizzle) -> shared-memory ring of STAGES slots guarded by
// mbarriers -> tcgen05.mma (M = 128, N = BN, K = 16, fp32 accumulator in tensor memory) ->
// tcgen05.ld epilogue (alpha, bias, residual, accumulate) -> fp32 output through TMA bulk tensor
// stores from swizzled shared-memory staging blocks, bf16 output through direct global stores.
//
// Warp roles (192 threads): warp 0 issues TMA loads, warp 1 owns tensor memory and issues the
// MMAs, warps 2..5 drain the accumulator (warp w reads TMEM lanes 32*(w%4) .. +31).
// Every wait on an mbarrier is bounded (OMQ_WAIT_LIMIT_NS); on expiry the kernel writes
// OMQ_ERR_TIMEOUT to the status word, stops issuing work, frees its tensor memory and exits.
#include "gemm.cuh"
#include "tc.cuh"
#include <cuda.h>
#include <cstring>
#include <vector>

namespace {

using namespace tc;

constexpr int BM = 128;
constexpr int BK = 64;          // one 128-byte swizzle row of bf16
constexpr int UMMA_K = 16;
constexpr int NUM_THREADS = 192;          // warp 0 TMA, warp 1 MMA, warps 2..5 epilogue
constexpr int NUM_THREADS_LWC = 320;      // LWC epilogue: warps 2..9, two per TMEM lane quadrant
// LWC = 4: the B operand is the raw weight and warps 6..9 form its fake-quantized bf16 values in
// shared memory (operand preparation of Eq. 4); warps 2..5 run the plain epilogue
constexpr int LWC_OPERAND = 4;

struct GemmParams {
  int M, N, K, batch;
  int a_mn, b_mn;            // 1 = MN-major operand
  int n_fast;                // tile order: 1 = n fastest (A streamed once), 0 = m fastest (B streamed once)
  int causal;
  GemmEpilogue ep;
  GemmLwcEpi lw;             // used by the LWC-epilogue instantiation only
  int32_t* status;
  GemmQuantB qb;             // used by the operand-preparation instantiation only
  int pair;                  // 1: CTA pairs, one 256-row tile per pair (cta_group::2)
  uint64_t wait_ns;          // limit of every mbarrier wait (OMQ_WAIT_LIMIT_NS unless a self-test sets it)
  int withhold;              // self-test only: the first operand load is never issued, so its wait expires
};

constexpr int EPI_TILE_BYTES = 32 * 32 * 4;      // one 32 x 32 fp32 block, 128-byte rows

template <int BN, int STAGES, bool PAIR = false>
struct SmemLayout {
  static constexpr int A_BYTES = BM * BK * 2;
  static constexpr int B_COLS = PAIR ? BN / 2 : BN;                 // a pair splits B's columns
  // room for whole 64-column boxes (MN-major B is staged in 64-wide swizzle atoms)
  static constexpr int B_BYTES = (B_COLS + 63) / 64 * 64 * BK * 2;
  static constexpr uint32_t TMEM_COLS = 2 * BN <= 256 ? 256 : 512;  // two accumulators, power of two
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int EPI_OFF = STAGES * STAGE_BYTES;           // 1024-aligned (swizzle atom)
  static constexpr int EPI_BYTES = 4 * 2 * EPI_TILE_BYTES;       // two staging blocks per epilogue warp
  static constexpr int BAR_OFF = EPI_OFF + EPI_BYTES;
  static constexpr int TOTAL = BAR_OFF + 256 + 1024;  // + barriers + alignment slack
  static_assert(EPI_OFF % 1024 == 0, "staging blocks must sit on the 1024-byte swizzle period");
  static_assert(TOTAL <= 227 * 1024, "shared memory per CTA");
};


// Tile t of the launch (m fastest, then n, then batch) and its K range.
struct TileInfo { int m0, n0, b, k_begin, nkb; bool skip; };

// With CTA pairs a tile is 2 BM rows; CTA `rank` of the pair owns rows m0 .. m0 + BM - 1.
__device__ __forceinline__ TileInfo tile_info(const GemmParams& p, int t, int bn, int rank = 0) {
  const int bm = p.pair ? 2 * BM : BM;
  const int mt = (p.M + bm - 1) / bm, nt = (p.N + bn - 1) / bn;
  TileInfo ti;
  if (p.n_fast) {
    ti.n0 = (t % nt) * bn;
    ti.m0 = ((t / nt) % mt) * bm;
  } else {
    ti.m0 = (t % mt) * bm;
    ti.n0 = ((t / mt) % nt) * bn;
  }
  ti.m0 += rank * BM;
  ti.b = t / (mt * nt);
  ti.skip = (p.causal == 1 && ti.n0 > ti.m0 + BM - 1);   // keys beyond every query of the tile
  int k_end = p.K;
  ti.k_begin = 0;
  if (p.causal == 2) k_end = min(p.K, ti.m0 + BM);
  if (p.causal == 3) ti.k_begin = ti.m0;
  ti.nkb = k_end > ti.k_begin ? (k_end - ti.k_begin + BK - 1) / BK : 0;
  return ti;
}

// Column sums of a warp's 32 x 32 block: on entry lane L holds row L's 32 values, on exit v[0]
// of lane L is the sum over the 32 rows of column L (five butterfly exchange stages, 31 shuffles).
__device__ __forceinline__ float colsum_warp32(float (&v)[32], int lane) {
#pragma unroll
  for (int k = 16; k >= 1; k >>= 1) {
    const bool up = (lane & k) != 0;
#pragma unroll
    for (int i = 0; i < k; ++i) {
      const float send = up ? v[i] : v[i + k];
      const float keep = up ? v[i + k] : v[i];
      v[i] = keep + __shfl_xor_sync(0xffffffffu, send, k);
    }
  }
  return v[0];
}

__device__ __forceinline__ void ldw32(const __nv_bfloat16* p, bool ok, uint4 (&r)[4]) {
#pragma unroll
  for (int i = 0; i < 4; ++i) r[i] = ok ? __ldg(reinterpret_cast<const uint4*>(p) + i) : make_uint4(0, 0, 0, 0);
}

// The per-element part of the LWC backward for one 32-column chunk of a row: W~ = fl(fl(W s) r),
// the code decision, the STE mask and h-path sums, and the LET column terms.  HS / HR: the column
// scale s / row scale r are present (an absent one is 1, its product skipped, exactly); DR: the row
// sum for dr is wanted; LET: the column terms for ds (cs) and ddelta (cd).
// the sums one element adds to, in element order: h path, clamped mass, dr, LET column terms
template <bool HS, bool HR, bool DR, bool LET>
__device__ __forceinline__ void lwc_elem(float g, float dh, int inr, float w, float sv, float rr, float dbr, float& Gh,
                                         float& Gbm, float& drm, float& cs, float& cd) {
  Gh = fmaf(g, dh, Gh);
  if (!inr) Gbm += g;
  const float d = inr ? g : 0.f;
  if (DR) drm = fmaf(d * w, sv, drm);
  if (LET) {
    cs = HR ? (d * w) * rr : d * w;
    cd = dbr * w;
  }
}

template <bool HS, bool HR, bool DR, bool LET>
__device__ __forceinline__ void lwc_elems(const uint4 (&wc)[4], const float* s_nb, float rr, float dbr, const QState& qs,
                                          float Q, const float (&g)[32], float& Gh, float& Gbm, float& drm,
                                          float (&cs)[32], float (&cd)[32]) {
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    float w8[8], s8[8];
    unpack_bf16x8(wc[i], w8);
    if (HS) {                                    // the tile's column scales, staged in shared memory
      const float4 a = reinterpret_cast<const float4*>(s_nb)[2 * i];
      const float4 b = reinterpret_cast<const float4*>(s_nb)[2 * i + 1];
      s8[0] = a.x; s8[1] = a.y; s8[2] = a.z; s8[3] = a.w; s8[4] = b.x; s8[5] = b.y; s8[6] = b.z; s8[7] = b.w;
    }
#pragma unroll
    for (int e = 0; e < 8; e += 2) {
      float2 wt = make_float2(w8[e], w8[e + 1]);
      if (HS) wt = omq_mul2(wt, make_float2(s8[e], s8[e + 1]));
      if (HR) wt = omq_mul2(wt, make_float2(rr, rr));
      int in0, in1;
      const float2 dh = omq_ste_dh2(wt, qs, Q, &in0, &in1);
      lwc_elem<HS, HR, DR, LET>(g[8 * i + e], dh.x, in0, w8[e], HS ? s8[e] : 1.f, rr, dbr, Gh, Gbm, drm,
                                cs[8 * i + e], cd[8 * i + e]);
      lwc_elem<HS, HR, DR, LET>(g[8 * i + e + 1], dh.y, in1, w8[e + 1], HS ? s8[e + 1] : 1.f, rr, dbr, Gh, Gbm, drm,
                                cs[8 * i + e + 1], cd[8 * i + e + 1]);
    }
  }
}

// Epilogue of the weight-gradient product with the straight-through LWC backward (Eq. 2) fused:
// the accumulator dW_hat is consumed from tensor memory 32 columns at a time and never stored.
// The weight row chunk of the next 32 columns is loaded while the current one is processed.
// hands accumulator buffer `buf` back to the MMA issuer (with CTA pairs: the leader CTA's barrier)
template <bool PAIR>
__device__ __forceinline__ void release_acc(uint64_t* acc_empty, uint32_t buf, int lane) {
  tc_fence_before();
  __syncwarp();
  if (lane == 0) {
    if (PAIR) mbar_arrive_cluster(mapa_shared(smem_u32(&acc_empty[buf]), 0));
    else mbar_arrive(&acc_empty[buf]);
  }
}

// Eight epilogue warps: warps w and w+4 drain the same 32 accumulator rows (lane quadrant w % 4),
// `half` 0 the first BN / 2 columns of the tile, 1 the others; each keeps its own row partials.
// Each warp stages the LET column scales of its half tile in its own 512 bytes of `s_stage` (the
// fp32 output staging area, unused here), and issues the loads of its rows' quantizer state and
// first weight chunk before it waits for the accumulator, so their latency overlaps the mainloop.
template <int BN, bool PAIR, int FORM>
__device__ __forceinline__ void lwc_epilogue(const GemmParams& p, uint32_t tmem, uint64_t* acc_full, uint64_t* acc_empty,
                                             volatile int* abort_flag, int q, int half, int lane, int total, int rank,
                                             float* s_stage) {
  constexpr int HB = BN / 2;                      // columns of a half
  const GemmLwcEpi& L = p.lw;
  const int N = p.N;
  const bool perch = L.group == N;
  const int ngroups = N / L.group;
  uint32_t acc_it = 0;
  const int t_first = PAIR ? (int)(blockIdx.x >> 1) : (int)blockIdx.x;
  const int t_step = PAIR ? (int)(gridDim.x >> 1) : (int)gridDim.x;
  for (int t = t_first; t < total; t += t_step) {
    const TileInfo ti = tile_info(p, t, BN, rank);
    if (ti.skip) continue;
    const bool has_acc = ti.nkb > 0;
    const uint32_t buf = acc_it & 1;
    bool ok = true;
    const int row0 = ti.m0 + q * 32;
    const int row = row0 + lane;
    const bool row_ok = row < p.M;
    const bool quad_ok = row0 < p.M;
    const float rr = (L.r && row_ok) ? L.r[row] : 1.f;
    const float dbr = (L.dBt && row_ok) ? __fmul_rn(L.dBt[row], rr) : 0.f;
    const __nv_bfloat16* wrow = L.W + (int64_t)(row_ok ? row : 0) * N;
    QState qs;
    qs.h = 1.f; qs.rh = 1.f; qs.z = 0.f; qs.u = 0.f; qs.b = 0.f; qs.m = 0.f; qs.a = 0.f; qs.M = 0.f; qs.floored = 0;
    int64_t gk = 0;                                // (row, group) index of the current group
    float Gh = 0.f, Gbm = 0.f, drm = 0.f;
    const int jb = half * HB;
    uint4 wcur[4], wnext[4];
    ldw32(wrow + ti.n0 + jb, row_ok && ti.n0 + jb < N, wcur);
    if (perch && row_ok) {                        // one quantizer state for the whole row
      gk = row;
      qs.h = L.h[gk];
      qs.z = (float)L.z[gk];
      qs.b = L.gb[gk];
      qs.m = L.mv[gk];
    }
    if (FORM != 2 && L.s) {                       // this half tile's column scales -> shared memory
      __syncwarp();                               // the previous tile's reads are done
      const int c = ti.n0 + jb + 4 * lane;
      const float4 sv = (4 * lane < HB && c < N) ? __ldg(reinterpret_cast<const float4*>(L.s + c))
                                                 : make_float4(1.f, 1.f, 1.f, 1.f);
      if (4 * lane < HB) reinterpret_cast<float4*>(s_stage)[lane] = sv;
      __syncwarp();
    }
    if (has_acc) {
      ok = __all_sync(0xffffffffu, mbar_wait(&acc_full[buf], (acc_it >> 1) & 1, p.wait_ns));
      if (!ok) { omq_set_status(p.status, OMQ_ERR_TIMEOUT); *abort_flag = 1; }
      tc_fence_after();
    }
    if (perch && row_ok) {
      qs.rh = __frcp_rn(qs.h);
      qs.u = __fmul_rn(__fmul_rn(qs.b, qs.m), qs.rh);
    }
#pragma unroll 1
    for (int j0 = jb; j0 < jb + HB; j0 += 32) {
      float g[32];
      if (has_acc && ok) {
        tmem_ld32(tmem + buf * BN + ((uint32_t)(q * 32) << 16) + (uint32_t)j0, g);
        if (j0 + 32 == jb + HB) release_acc<PAIR>(acc_empty, buf, lane);   // this warp's part drained
      } else {
#pragma unroll
        for (int i = 0; i < 32; ++i) g[i] = 0.f;
      }
      const int nb = ti.n0 + j0;
      if (j0 + 32 < jb + HB) ldw32(wrow + nb + 32, row_ok && nb + 32 < N, wnext);
      if (quad_ok && nb < N) {
        if (!perch && nb % L.group == 0 && row_ok) {   // quantizer state of the group starting here
          gk = (int64_t)row * ngroups + nb / L.group;
          qs.h = L.h[gk];
          qs.z = (float)L.z[gk];
          qs.b = L.gb[gk];
          qs.m = L.mv[gk];
          qs.rh = __frcp_rn(qs.h);
          qs.u = __fmul_rn(__fmul_rn(qs.b, qs.m), qs.rh);
          Gh = 0.f; Gbm = 0.f;
        }
        float cs[32], cd[32];
        // without LET only the STE part; with it every term (an absent s or r is 1: products by it
        // are exact)
        if (FORM == 2) lwc_elems<false, false, false, false>(wcur, nullptr, rr, dbr, qs, L.Q, g, Gh, Gbm, drm, cs, cd);
        else if (FORM == 3) lwc_elems<true, false, false, true>(wcur, s_stage + (j0 - jb), rr, dbr, qs, L.Q, g, Gh, Gbm, drm, cs, cd);
        else if (L.s) lwc_elems<true, true, true, true>(wcur, s_stage + (j0 - jb), rr, dbr, qs, L.Q, g, Gh, Gbm, drm, cs, cd);
        else lwc_elems<false, true, true, true>(wcur, nullptr, rr, dbr, qs, L.Q, g, Gh, Gbm, drm, cs, cd);
        const int64_t prow = (int64_t)(row0 >> 5) * N + nb + lane;
        if (L.part_s) {
          const float v = colsum_warp32(cs, lane);
          L.part_s[prow] = v;
        }
        if (L.part_d) {
          const float v = colsum_warp32(cd, lane);
          L.part_d[prow] = v;
        }
        if (!perch && (nb + 32) % L.group == 0 && row_ok) {   // group complete: dgamma, dbeta
          const float ga = L.ga[gk], gb = qs.b, M = L.Mv[gk], m = qs.m;
          const float hr = __fdiv_rn(__fsub_rn(__fmul_rn(ga, M), __fmul_rn(gb, m)), L.Q);
          const float Ghe = (hr >= L.eps) ? Gh : 0.f;           // floored h: no gradient through h
          const float GaM = Ghe / L.Q, Gbt = Gbm - Ghe / L.Q;
          const float dg = GaM * M * ga * (1.f - ga), db = Gbt * m * gb * (1.f - gb);
          if (L.accumulate) { L.dgl[gk] += dg; L.dbl[gk] += db; } else { L.dgl[gk] = dg; L.dbl[gk] = db; }
        }
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) wcur[i] = wnext[i];
    }
    if (perch && quad_ok && row_ok) {
      const int nt = 2 * (ti.n0 / BN) + half;     // one partial per (N tile, half)
      L.rowpart[((int64_t)0 * p.M + row) * L.ntn + nt] = Gh;
      L.rowpart[((int64_t)1 * p.M + row) * L.ntn + nt] = Gbm;
      L.rowpart[((int64_t)2 * p.M + row) * L.ntn + nt] = drm;
    }
    if (has_acc) ++acc_it;
    if (!ok) break;
  }
}

// Operand preparation (LWC = 4): warps 6..9 of each CTA turn the raw weight tile of every stage into
// its fake-quantized bf16 values in place.  The weight W is [rows, cols] with its quantizer state
// per (row, group of cols) (GemmQuantB); as a K-major B operand (Y = X W_hat^T) a B row is a weight
// row, as an MN-major one (dX = dY W_hat) a B row is a K index, i.e. again a weight row.  Either
// way the tile is a stack of 128-byte swizzled lines of 64 consecutive weight columns of one weight
// row (logical 16-byte chunk c of line l sits at chunk c ^ (l & 7); the conversion is elementwise,
// so each chunk is rewritten where it lies), and thread ct owns line ct.  It waits for the tile's
// own load barrier, converts, makes its writes visible to the tensor core's async proxy and arrives
// on the leader's `conv` barrier, which the MMA issuer waits for besides `full`.
template <int BN, int STAGES, bool PAIR>
__device__ __forceinline__ void operand_prep(const GemmParams& p, uint8_t* smem, uint64_t* bfull, uint64_t* conv,
                                             volatile int* abort_flag, int ct, int total, int rank) {
  using L = SmemLayout<BN, STAGES, PAIR>;
  constexpr int BNH = PAIR ? BN / 2 : BN;
  static_assert(BNH == 128, "one converter thread per 128-byte line of the B tile");
  const GemmQuantB& qb = p.qb;
  const bool mn = p.b_mn != 0;
  const int lane = ct & 31;
  const int t_first = PAIR ? (int)(blockIdx.x >> 1) : (int)blockIdx.x;
  const int t_step = PAIR ? (int)(gridDim.x >> 1) : (int)gridDim.x;
  const int wcols = mn ? p.N : p.K;                 // weight columns
  const int wrows = mn ? p.K : p.N;                 // weight rows
  const int ngroups = wcols / qb.group;
  uint32_t it = 0;
  for (int t = t_first; t < total && !*abort_flag; t += t_step) {
    const TileInfo ti = tile_info(p, t, BN, rank);
    if (ti.skip) continue;
    const int nb0 = ti.n0 + rank * BNH;
    QState qs;
    qs.h = 1.f; qs.rh = 1.f; qs.z = 0.f; qs.u = 0.f; qs.a = qs.b = qs.M = qs.m = 0.f; qs.floored = 0;
    int64_t gk_cur = -1;
    float rr = 1.f;
    int wr_cur = -1;
    for (int kb = 0; kb < ti.nkb; ++kb, ++it) {
      const int s = it % STAGES;
      if (!mbar_wait(&bfull[s], (it / STAGES) & 1, p.wait_ns)) {
        omq_set_status(p.status, OMQ_ERR_TIMEOUT); *abort_flag = 1; break;
      }
      const int k0 = ti.k_begin + kb * BK;
      // this thread's line: weight row wr, weight columns wc0 .. wc0 + 63
      int wr, wc0;
      uint32_t line;
      if (!mn) { wr = nb0 + ct; wc0 = k0; line = smem_u32(smem + s * L::STAGE_BYTES + L::A_BYTES) + ct * 128; }
      else { wr = k0 + (ct & 63); wc0 = nb0 + 64 * (ct >> 6);
             line = smem_u32(smem + s * L::STAGE_BYTES + L::A_BYTES) + (ct >> 6) * 64 * BK * 2 + (ct & 63) * 128; }
      if (wr < wrows) {
        if (wr != wr_cur) { wr_cur = wr; rr = qb.r ? __ldg(qb.r + wr) : 1.f; gk_cur = -1; }
        // all eight chunks first (logical chunk c sits at c ^ (line & 7): the eight lines of a
        // quarter-warp touch eight distinct 16-byte bank groups), then the arithmetic, then the stores
        uint4 raw[8];
#pragma unroll
        for (int c = 0; c < 8; ++c) raw[c] = lds128(line + ((c ^ (ct & 7)) << 4));
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          const int wc = wc0 + 8 * c;
          if (wc >= wcols) continue;                // beyond the weight the tile holds zeros
          const int64_t gk = (int64_t)wr * ngroups + wc / qb.group;
          if (gk != gk_cur) {
            gk_cur = gk;
            qs.h = __ldg(qb.h + gk);
            qs.z = (float)__ldg(qb.z + gk);
            qs.rh = __frcp_rn(qs.h);
          }
          float w[8], o[8];
          unpack_bf16x8(raw[c], w);
          if (qb.s) {
            const float4 s0 = __ldg(reinterpret_cast<const float4*>(qb.s + wc));
            const float4 s1 = __ldg(reinterpret_cast<const float4*>(qb.s + wc) + 1);
            const float sv[8] = {s0.x, s0.y, s0.z, s0.w, s1.x, s1.y, s1.z, s1.w};
#pragma unroll
            for (int e = 0; e < 8; ++e) w[e] = __fmul_rn(w[e], sv[e]);
          }
          if (qb.r) {
#pragma unroll
            for (int e = 0; e < 8; ++e) w[e] = __fmul_rn(w[e], rr);
          }
#pragma unroll
          for (int e = 0; e < 8; ++e) o[e] = omq_fakequant(w[e], qs, qb.Q, nullptr);
          raw[c] = pack_bf16x8(o);
        }
#pragma unroll
        for (int c = 0; c < 8; ++c) sts128(line + ((c ^ (ct & 7)) << 4), raw[c]);
      }
      fence_async_smem();                           // the converted tile -> visible to the tensor core
      __syncwarp();
      if (lane == 0) {
        if (PAIR) mbar_arrive_cluster(mapa_shared(smem_u32(&conv[s]), 0));
        else mbar_arrive(&conv[s]);
      }
    }
  }
}

// Persistent kernel: one CTA per SM walks tiles blockIdx.x, blockIdx.x + gridDim.x, ...
// The shared-memory ring runs continuously across tiles; the accumulator is double-buffered
// in tensor memory (2 x BN columns) so that the epilogue of one tile overlaps the MMAs of
// the next.
//
// PAIR: the grid is made of 2-CTA clusters; the pair computes one 2 BM x BN tile with one
// tcgen05.mma of cta_group::2 (M = 256): each CTA stages its BM rows of A and BN / 2 columns of B
// (both TMA loads complete on the leader CTA's mbarrier), the leader issues the MMAs, commits
// reach both CTAs' barriers, and each CTA drains its own BM rows of the accumulator.  Per CTA
// the shared-memory bytes per MMA flop halve for B, so six stages fit where four did.
// LWC: 0 plain product; LWC epilogue 1 general, 2 without LET terms, 3 with the LET column scale but
// neither row scale nor dr
template <int BN, int STAGES, int LWC, bool PAIR>
__global__ void __launch_bounds__(LWC ? NUM_THREADS_LWC : NUM_THREADS, 1)
    gemm_bf16_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                     const __grid_constant__ CUtensorMap tmC, const GemmParams p) {
  using L = SmemLayout<BN, STAGES, PAIR>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + L::BAR_OFF);
  uint64_t* empty = full + STAGES;
  uint64_t* acc_full = empty + STAGES;     // [2]
  uint64_t* acc_empty = acc_full + 2;      // [2]
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(acc_empty + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);
  uint64_t* drain = acc_empty + 3;         // after tmem_holder and abort_flag (8 bytes)
  constexpr bool QB = LWC == LWC_OPERAND;
  constexpr bool EPI_LWC = LWC != 0 && !QB;
  uint64_t* bfull = drain + 1;             // QB: [STAGES] this CTA's raw B tile landed
  uint64_t* conv = bfull + STAGES;         // QB: [STAGES] the pair's B tiles prepared (leader's)

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int bm_tile = PAIR ? 2 * BM : BM;
  const int mt = (p.M + bm_tile - 1) / bm_tile, nt = (p.N + BN - 1) / BN;
  const int total = mt * nt * p.batch;
  const int rank = PAIR ? (int)cluster_ctarank() : 0;
  const bool leader = rank == 0;
  const int t_first = PAIR ? (int)(blockIdx.x >> 1) : (int)blockIdx.x;
  const int t_step = PAIR ? (int)(gridDim.x >> 1) : (int)gridDim.x;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) { mbar_init(&full[s], 1); mbar_init(&empty[s], 1); }
    constexpr int EPI_WARPS = EPI_LWC ? 8 : 4;
    for (int b = 0; b < 2; ++b) { mbar_init(&acc_full[b], 1); mbar_init(&acc_empty[b], (PAIR ? 2 : 1) * EPI_WARPS); }
    *abort_flag = 0;
    mbar_init(drain, 1);
    if (QB)
      for (int s = 0; s < STAGES; ++s) { mbar_init(&bfull[s], 1); mbar_init(&conv[s], (PAIR ? 2 : 1) * 4); }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    if (PAIR) tmem_alloc_pair(tmem_holder, L::TMEM_COLS);
    else tmem_alloc(tmem_holder, L::TMEM_COLS);
  }
  tc_fence_before();
  __syncthreads();
  if (PAIR) cluster_sync();                 // both CTAs' barriers initialised before any remote use
  tc_fence_after();
  const uint32_t tmem = *tmem_holder;

  if (warp == 0 && lane == 0) {
    // ---------------- TMA producer ----------------
    uint32_t it = 0;
    constexpr int BNH = PAIR ? BN / 2 : BN;      // B columns staged by this CTA
    // bytes one stage of this CTA receives: A, and B as K-major rows or whole 64-column boxes
    const uint32_t stage_tx = L::A_BYTES + (p.b_mn ? (uint32_t)((BNH + 63) / 64 * 64 * BK * 2) : (uint32_t)(BNH * BK * 2));
    for (int t = t_first; t < total && !*abort_flag; t += t_step) {
      const TileInfo ti = tile_info(p, t, BN, rank);
      if (ti.skip) continue;
      const int nb0 = ti.n0 + rank * BNH;
      for (int kb = 0; kb < ti.nkb; ++kb, ++it) {
        const int s = it % STAGES;
        if (!mbar_wait(&empty[s], ((it / STAGES) & 1) ^ 1, p.wait_ns)) {
          omq_set_status(p.status, OMQ_ERR_TIMEOUT); *abort_flag = 1; break;
        }
        if (p.withhold && it == 0) continue;      // self-test: the stage's load is never issued
        uint8_t* sa = smem + s * L::STAGE_BYTES;
        uint8_t* sb = sa + L::A_BYTES;
        const int k0 = ti.k_begin + kb * BK;
        if (QB) {
          // A (both CTAs' halves) completes on the leader's full barrier, this CTA's raw B tile on its
          // own bfull barrier, which its converter warps wait for
          if (PAIR) {
            if (leader) mbar_expect_tx(&full[s], 2 * (uint32_t)L::A_BYTES);
            tma_load_3d_pair(&tmA, mapa_shared(smem_u32(&full[s]), 0), sa, k0, ti.m0, ti.b);
          } else {
            mbar_expect_tx(&full[s], (uint32_t)L::A_BYTES);
            tma_load_3d(&tmA, &full[s], sa, k0, ti.m0, ti.b);
          }
          mbar_expect_tx(&bfull[s], (uint32_t)(BNH * BK * 2));
          if (!p.b_mn) {
            tma_load_3d(&tmB, &bfull[s], sb, k0, nb0, ti.b);
          } else {
#pragma unroll
            for (int j = 0; j < BNH / 64; ++j) tma_load_3d(&tmB, &bfull[s], sb + j * 64 * BK * 2, nb0 + 64 * j, k0, ti.b);
          }
        } else if (PAIR) {
          // both CTAs' loads complete on the leader's barrier, which expects the pair's bytes
          const uint32_t fb = mapa_shared(smem_u32(&full[s]), 0);
          if (leader) mbar_expect_tx(&full[s], 2 * stage_tx);
          if (!p.a_mn) {
            tma_load_3d_pair(&tmA, fb, sa, k0, ti.m0, ti.b);
          } else {
            tma_load_3d_pair(&tmA, fb, sa, ti.m0, k0, ti.b);
            tma_load_3d_pair(&tmA, fb, sa + 64 * BK * 2, ti.m0 + 64, k0, ti.b);
          }
          if (!p.b_mn) {
            tma_load_3d_pair(&tmB, fb, sb, k0, nb0, ti.b);
          } else {
#pragma unroll
            for (int j = 0; j < (BNH + 63) / 64; ++j)
              tma_load_3d_pair(&tmB, fb, sb + j * 64 * BK * 2, nb0 + 64 * j, k0, ti.b);
          }
        } else {
          mbar_expect_tx(&full[s], stage_tx);
          if (!p.a_mn) {
            tma_load_3d(&tmA, &full[s], sa, k0, ti.m0, ti.b);
          } else {
            tma_load_3d(&tmA, &full[s], sa, ti.m0, k0, ti.b);
            tma_load_3d(&tmA, &full[s], sa + 64 * BK * 2, ti.m0 + 64, k0, ti.b);
          }
          if (!p.b_mn) {
            tma_load_3d(&tmB, &full[s], sb, k0, ti.n0, ti.b);
          } else {
#pragma unroll
            for (int j = 0; j < (BN + 63) / 64; ++j)
              tma_load_3d(&tmB, &full[s], sb + j * 64 * BK * 2, ti.n0 + 64 * j, k0, ti.b);
          }
        }
      }
    }
    // after an expired wait (or a withheld load) no copy this CTA issued may still be landing in its
    // shared memory when it exits: wait, bounded, for the last load of every stage (with CTA pairs
    // the leader's barrier counts both CTAs' bytes, and the peer leaves only after the leader)
    if ((*abort_flag || p.withhold) && leader) {
      const uint32_t first = it > (uint32_t)STAGES ? it - STAGES : 0u;
      for (uint32_t j = first; j < it; ++j)
        if (!(p.withhold && j == 0)) mbar_wait(&full[j % STAGES], (j / STAGES) & 1, p.wait_ns);
    }
    if (QB && *abort_flag) {                     // this CTA's own B loads
      const uint32_t first = it > (uint32_t)STAGES ? it - STAGES : 0u;
      for (uint32_t j = first; j < it; ++j) mbar_wait(&bfull[j % STAGES], (j / STAGES) & 1, p.wait_ns);
    }
  } else if (warp == 1 && lane == 0 && leader) {
    // ---------------- MMA issuer (with CTA pairs: the leader CTA only) ----------------
    constexpr uint32_t IDESC_KK = idesc_bf16(PAIR ? 2 * BM : BM, BN, 0, 0);
    const uint32_t idesc = IDESC_KK | ((uint32_t)p.a_mn << 15) | ((uint32_t)p.b_mn << 16);
    uint32_t it = 0, acc_it = 0;
    bool issued = false;
    for (int t = t_first; t < total && !*abort_flag; t += t_step) {
      const TileInfo ti = tile_info(p, t, BN, rank);
      if (ti.skip || ti.nkb == 0) continue;
      const uint32_t buf = acc_it & 1;
      if (!mbar_wait(&acc_empty[buf], ((acc_it >> 1) & 1) ^ 1, p.wait_ns)) {
        omq_set_status(p.status, OMQ_ERR_TIMEOUT); *abort_flag = 1; break;
      }
      tc_fence_after();
      const uint32_t d_tmem = tmem + buf * BN;
      bool ok = true;
      for (int kb = 0; kb < ti.nkb; ++kb, ++it) {
        const int s = it % STAGES;
        if (!mbar_wait(&full[s], (it / STAGES) & 1, p.wait_ns) ||
            (QB && !(PAIR ? mbar_wait_cluster(&conv[s], (it / STAGES) & 1, p.wait_ns)
                          : mbar_wait(&conv[s], (it / STAGES) & 1, p.wait_ns)))) {
          omq_set_status(p.status, OMQ_ERR_TIMEOUT); *abort_flag = 1; ok = false; break;
        }
        tc_fence_after();
        issued = true;
        const uint32_t sa = smem_u32(smem + s * L::STAGE_BYTES);
        const uint32_t sb = sa + L::A_BYTES;
#pragma unroll
        for (int k = 0; k < BK / UMMA_K; ++k) {
          // K-major: advance 32 bytes inside the swizzle row; MN-major: advance 16 K-rows (2 KB)
          const uint64_t ad = p.a_mn ? sdesc(sa + k * 2048, 64 * BK * 2, 1024) : sdesc(sa + k * 32, 16, 1024);
          const uint64_t bd = p.b_mn ? sdesc(sb + k * 2048, 64 * BK * 2, 1024) : sdesc(sb + k * 32, 16, 1024);
          if (PAIR) umma_bf16_pair(d_tmem, ad, bd, idesc, (kb | k) != 0);
          else umma_bf16(d_tmem, ad, bd, idesc, (kb | k) != 0);
        }
        if (PAIR) umma_commit_pair(&empty[s], 0x3);
        else umma_commit(&empty[s]);
      }
      if (PAIR) umma_commit_pair(&acc_full[buf], 0x3);
      else umma_commit(&acc_full[buf]);
      ++acc_it;
      if (!ok) break;
    }
    // after an expired wait, the products already issued must finish before the tensor memory is
    // released: one more commit, on a barrier of its own, tracks all of them (bounded wait)
    if (*abort_flag && issued) {
      if (PAIR) umma_commit_pair(drain, 0x1);
      else umma_commit(drain);
      mbar_wait(drain, 0, p.wait_ns);
    }
  } else if (QB && warp >= 6) {
    if constexpr (QB) operand_prep<BN, STAGES, PAIR>(p, smem, bfull, conv, abort_flag, threadIdx.x - 192, total, rank);
  } else if (EPI_LWC && warp >= 2) {
    lwc_epilogue<BN, PAIR, (EPI_LWC ? LWC : 1)>(p, tmem, acc_full, acc_empty, abort_flag, warp & 3, (warp - 2) >> 2, lane, total, rank,
                                reinterpret_cast<float*>(smem + L::EPI_OFF) + (warp - 2) * (BN / 2));
  } else if (warp >= 2) {
    // ---------------- epilogue ----------------
    // fp32 output leaves through TMA bulk stores: each warp stages its 32 x 32 block in one of two
    // 128-byte-swizzled shared-memory slots (16-byte chunk c of row r at chunk c ^ (r & 7), so the
    // eight rows of a quarter-warp hit distinct banks) and one lane issues the store.  bf16 output
    // is written directly from registers.
    const int q = warp & 3;                       // TMEM lane quadrant of this warp
    const GemmEpilogue& ep = p.ep;
    uint8_t* stage_base = smem + L::EPI_OFF + q * 2 * EPI_TILE_BYTES;
    uint32_t n_stores = 0;
    uint32_t acc_it = 0;
    for (int t = t_first; t < total; t += t_step) {
      const TileInfo ti = tile_info(p, t, BN, rank);
      if (ti.skip) continue;
      const bool has_acc = ti.nkb > 0;
      const uint32_t buf = acc_it & 1;
      bool ok = true;
      if (has_acc) {
        ok = __all_sync(0xffffffffu, mbar_wait(&acc_full[buf], (acc_it >> 1) & 1, p.wait_ns));  // tcgen05.ld is warp-wide
        if (!ok) { omq_set_status(p.status, OMQ_ERR_TIMEOUT); *abort_flag = 1; }
        tc_fence_after();
      }
      const int row0 = ti.m0 + q * 32;
      const int row = row0 + lane;
      const bool row_ok = row < p.M;
      const int64_t crow = (int64_t)ti.b * ep.c_bs + (int64_t)row * ep.ldc;
#pragma unroll 1
      for (int j0 = 0; j0 < BN; j0 += 32) {
        float v[32];
        if (has_acc && ok) {
          tmem_ld32(tmem + buf * BN + ((uint32_t)(q * 32) << 16) + (uint32_t)j0, v);
          if (j0 + 32 == BN) release_acc<PAIR>(acc_empty, buf, lane);   // accumulator drained
        } else {
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] = 0.f;
        }
        const int nb = ti.n0 + j0;
        if (row0 >= p.M || nb >= p.N) continue;   // warp-uniform: block wholly outside C
        const bool full_chunk = nb + 32 <= p.N;
#pragma unroll
        for (int i = 0; i < 32; ++i) v[i] *= ep.alpha;
        if (row_ok && full_chunk) {
          if (ep.bias) {
#pragma unroll
            for (int i = 0; i < 32; i += 4) {
              float4 bb = __ldg(reinterpret_cast<const float4*>(ep.bias + nb + i));
              v[i] += bb.x; v[i + 1] += bb.y; v[i + 2] += bb.z; v[i + 3] += bb.w;
            }
          }
          if (ep.R) {
            const float* rr = ep.R + (int64_t)ti.b * ep.c_bs + (int64_t)row * ep.ldr + nb;
#pragma unroll
            for (int i = 0; i < 32; i += 4) {
              float4 tt = __ldg(reinterpret_cast<const float4*>(rr + i));
              v[i] += tt.x; v[i + 1] += tt.y; v[i + 2] += tt.z; v[i + 3] += tt.w;
            }
          }
          if (ep.Cf && ep.beta_acc != 0.f) {
            const float* cp = ep.Cf + crow + nb;
#pragma unroll
            for (int i = 0; i < 32; i += 4) {
              float4 tt = *reinterpret_cast<const float4*>(cp + i);
              v[i] += ep.beta_acc * tt.x; v[i + 1] += ep.beta_acc * tt.y;
              v[i + 2] += ep.beta_acc * tt.z; v[i + 3] += ep.beta_acc * tt.w;
            }
          }
          if (ep.Cb) {
            __nv_bfloat16* cp = ep.Cb + crow + nb;
#pragma unroll
            for (int i = 0; i < 32; i += 8) *reinterpret_cast<uint4*>(cp + i) = pack_bf16x8(v + i);
          }
        } else if (row_ok) {                      // ragged last column block
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const int n = nb + i;
            if (n < p.N) {
              if (ep.bias) v[i] += ep.bias[n];
              if (ep.R) v[i] += ep.R[(int64_t)ti.b * ep.c_bs + (int64_t)row * ep.ldr + n];
              if (ep.Cf && ep.beta_acc != 0.f) v[i] += ep.beta_acc * ep.Cf[crow + n];
              if (ep.Cb) ep.Cb[crow + n] = f_to_bf16(v[i]);
            }
          }
        }
        if (ep.Cf) {
          uint8_t* stg = stage_base + (n_stores & 1) * EPI_TILE_BYTES;
          if (lane == 0) bulk_wait_read1();       // the store that last used this slot has read it
          __syncwarp();
          uint8_t* my_row = stg + lane * 128;
#pragma unroll
          for (int c = 0; c < 8; ++c)
            *reinterpret_cast<float4*>(my_row + ((c ^ (lane & 7)) << 4)) =
                make_float4(v[4 * c], v[4 * c + 1], v[4 * c + 2], v[4 * c + 3]);
          fence_async_smem();                     // generic-proxy writes -> visible to the copy engine
          __syncwarp();
          if (lane == 0) {
            tma_store_3d(&tmC, stg, nb, row0, ti.b);
            bulk_commit();
          }
          ++n_stores;
        }
      }
      if (has_acc) ++acc_it;
      if (!ok) break;
    }
    if (lane == 0) bulk_wait_all();
  }
  tc_fence_before();
  __syncthreads();
  if (PAIR) cluster_sync();                 // no CTA leaves while its peer may still signal it
  if (warp == 1) {
    tc_fence_after();
    if (PAIR) tmem_dealloc_pair(tmem, L::TMEM_COLS);
    else tmem_dealloc(tmem, L::TMEM_COLS);
  }
}

// ---------------------------------------------------------------------------------------------
// host side: tensor maps through the driver entry point (no link-time dependency on libcuda)
// ---------------------------------------------------------------------------------------------
typedef CUresult (*PFN_encodeTiled_t)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                      const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                      CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

PFN_encodeTiled_t get_encode() {
  static PFN_encodeTiled_t fn = nullptr;
  if (!fn) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_encodeTiled_t>(ptr);
  }
  return fn;
}

// 3-D bf16 map {inner, rows, batch} with a {64, box_rows, 1} box and 128-byte swizzle.
bool make_map(CUtensorMap* map, const void* ptr, int64_t inner, int64_t rows, int64_t batch, int64_t ld, int64_t bs,
              int box_rows) {
  PFN_encodeTiled_t enc = get_encode();
  if (!enc) return false;
  cuuint64_t dims[3] = {(cuuint64_t)inner, (cuuint64_t)rows, (cuuint64_t)batch};
  cuuint64_t strides[2] = {(cuuint64_t)(ld * 2), (cuuint64_t)((batch > 1 ? bs : ld * rows) * 2)};
  cuuint32_t box[3] = {64u, (cuuint32_t)box_rows, 1u};
  cuuint32_t estr[3] = {1u, 1u, 1u};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(ptr), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// 3-D fp32 map of the output {cols, rows, batch} with a {32, 32, 1} box and 128-byte swizzle
// (the layout of the epilogue's staging blocks).
bool make_map_c(CUtensorMap* map, float* ptr, int64_t N, int64_t M, int64_t batch, int64_t ldc, int64_t cbs) {
  PFN_encodeTiled_t enc = get_encode();
  if (!enc) return false;
  cuuint64_t dims[3] = {(cuuint64_t)N, (cuuint64_t)M, (cuuint64_t)batch};
  cuuint64_t strides[2] = {(cuuint64_t)(ldc * 4), (cuuint64_t)((batch > 1 ? cbs : ldc * M) * 4)};
  cuuint32_t box[3] = {32u, 32u, 1u};
  cuuint32_t estr[3] = {1u, 1u, 1u};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, ptr, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                   CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

template <int BN, int STAGES, int LWC = 0, bool PAIR = false>
omq_status launch_cfg(cudaStream_t st, const CUtensorMap& ta, const CUtensorMap& tb, const CUtensorMap& tc,
                      const GemmParams& p) {
  using L = SmemLayout<BN, STAGES, PAIR>;
  auto kern = gemm_bf16_kernel<BN, STAGES, LWC, PAIR>;
  static bool attr_set = false;
  if (!attr_set) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, L::TOTAL) != cudaSuccess)
      return OMQ_ERR_CUDA;
    attr_set = true;
  }
  const int bm_tile = PAIR ? 2 * BM : BM;
  const int64_t tiles = (int64_t)((p.M + bm_tile - 1) / bm_tile) * ((p.N + BN - 1) / BN) * p.batch;
  const int64_t sms = omq_num_sms();
  if (!PAIR) {
    const unsigned grid = (unsigned)(tiles < sms ? tiles : sms);
    kern<<<grid, LWC ? NUM_THREADS_LWC : NUM_THREADS, L::TOTAL, st>>>(ta, tb, tc, p);
  } else {
    const int64_t pairs = sms / 2;
    const unsigned grid = (unsigned)(2 * (tiles < pairs ? tiles : pairs));
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid, 1, 1);
    cfg.blockDim = dim3(LWC ? NUM_THREADS_LWC : NUM_THREADS, 1, 1);
    cfg.dynamicSmemBytes = L::TOTAL;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cudaLaunchKernelEx(&cfg, kern, ta, tb, tc, p) != cudaSuccess) return OMQ_ERR_CUDA;
  }
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

// ---- optional per-launch timing (CUDA events recorded on the launching stream) ----
struct GemmProfile {
  bool on = false;
  std::vector<cudaEvent_t> ev;     // pairs: start, stop
  size_t used = 0;                 // events in use
  double flops = 0.0;              // algorithmic flops of the recorded launches
};
GemmProfile g_prof;

// multiply-adds of the launch counted once each, times two; causal modes count the triangle only
double gemm_algorithmic_flops(int64_t M, int64_t N, int64_t K, int64_t batch, int causal) {
  double mnk;
  if (causal == 0) {
    mnk = (double)M * N * K;
  } else if (causal == 1) {         // keys n <= query m
    double pairs = 0;
    for (int64_t m = 0; m < M; ++m) pairs += (double)(m + 1 < N ? m + 1 : N);
    mnk = pairs * K;
  } else if (causal == 2) {         // k <= m
    double s = 0;
    for (int64_t m = 0; m < M; ++m) s += (double)(m + 1 < K ? m + 1 : K);
    mnk = s * N;
  } else {                          // k >= m
    double s = 0;
    for (int64_t m = 0; m < M; ++m) s += (double)(K - m > 0 ? K - m : 0);
    mnk = s * N;
  }
  return 2.0 * mnk * batch;
}

cudaEvent_t prof_event() {
  if (g_prof.used == g_prof.ev.size()) {
    cudaEvent_t e;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    g_prof.ev.push_back(e);
  }
  return g_prof.ev[g_prof.used++];
}

}  // namespace

omq_status gemm_launch(cudaStream_t st, int64_t M, int64_t N, int64_t K, int64_t batch, const GemmOperand& A,
                       const GemmOperand& B, const GemmEpilogue& ep, int causal, int32_t* status) {
  OMQ_REQUIRE(M > 0 && N > 0 && K > 0 && batch > 0, OMQ_ERR_SHAPE);
  OMQ_REQUIRE(M < (1ll << 31) && N < (1ll << 31) && K < (1ll << 31) && batch < 65536, OMQ_ERR_SHAPE);
  OMQ_REQUIRE(A.ptr && B.ptr && (ep.Cf || ep.Cb), OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(causal >= 0 && causal <= 3, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(omq_aligned16(A.ptr) && omq_aligned16(B.ptr), OMQ_ERR_ALIGN);
  OMQ_REQUIRE(A.ld % 8 == 0 && B.ld % 8 == 0 && (batch == 1 || (A.bs % 8 == 0 && B.bs % 8 == 0)), OMQ_ERR_ALIGN);
  OMQ_REQUIRE(ep.ldc % 8 == 0 && (batch == 1 || ep.c_bs % 8 == 0), OMQ_ERR_ALIGN);
  OMQ_REQUIRE(ep.ldc >= N, OMQ_ERR_SHAPE);
  OMQ_REQUIRE((!ep.Cf || omq_aligned16(ep.Cf)) && (!ep.Cb || omq_aligned16(ep.Cb)), OMQ_ERR_ALIGN);
  OMQ_REQUIRE(!ep.R || (omq_aligned16(ep.R) && ep.ldr % 4 == 0), OMQ_ERR_ALIGN);
  OMQ_REQUIRE(!ep.bias || omq_aligned16(ep.bias), OMQ_ERR_ALIGN);
  // the MN-major extents must cover whole 64-wide boxes inside the tensor (TMA zero-fills the rest)
  const bool wide = gemm_n_tile(N) == 256;
  // CTA pairs (one 256 x 256 tile per pair) for plain single products
  const bool pair = wide && batch == 1 && causal == 0 && M > BM;
  CUtensorMap ta, tb;
  const int bn = wide ? 256 : 128;
  bool ok = A.kmajor ? make_map(&ta, A.ptr, K, M, batch, A.ld, A.bs, BM) : make_map(&ta, A.ptr, M, K, batch, A.ld, A.bs, BK);
  ok = ok && (B.kmajor ? make_map(&tb, B.ptr, K, N, batch, B.ld, B.bs, pair ? bn / 2 : bn)
                       : make_map(&tb, B.ptr, N, K, batch, B.ld, B.bs, BK));
  CUtensorMap tc;
  memset(&tc, 0, sizeof(tc));
  if (ep.Cf) ok = ok && make_map_c(&tc, ep.Cf, N, M, batch, ep.ldc, ep.c_bs);
  if (!ok) return OMQ_ERR_UNSUPPORTED;
  GemmParams p;
  p.M = (int)M; p.N = (int)N; p.K = (int)K; p.batch = (int)batch;
  p.a_mn = A.kmajor ? 0 : 1; p.b_mn = B.kmajor ? 0 : 1;
  p.causal = causal; p.ep = ep; p.status = status; p.pair = pair ? 1 : 0;
  p.wait_ns = OMQ_WAIT_LIMIT_NS; p.withhold = 0;
  // stream the larger operand once and keep the smaller one L2-resident: with m fastest, the
  // CTAs working at one time share an N tile of B and sweep A; with n fastest, the reverse
  p.n_fast = ((double)M > 1.5 * (double)N) ? 1 : 0;
  cudaEvent_t e0 = nullptr, e1 = nullptr;
  if (g_prof.on) {
    e0 = prof_event();
    e1 = prof_event();
    if (e0 && e1) {
      cudaEventRecord(e0, st);
      g_prof.flops += gemm_algorithmic_flops(M, N, K, batch, causal);
    }
  }
  omq_status r = pair ? launch_cfg<256, 6, 0, true>(st, ta, tb, tc, p)
                      : (wide ? launch_cfg<256, 4>(st, ta, tb, tc, p) : launch_cfg<128, 6>(st, ta, tb, tc, p));
  if (e0 && e1) cudaEventRecord(e1, st);
  return r;
}

int gemm_n_tile(int64_t N) { return N % 256 == 0 ? 256 : 128; }

bool omq_make_map_f32_out(CUtensorMap* map, float* ptr, int64_t N, int64_t M, int64_t ld) {
  return make_map_c(map, ptr, N, M, 1, ld, 0);
}

bool omq_make_map_bf16(CUtensorMap* map, const void* ptr, int64_t inner, int64_t rows, int64_t batch, int64_t ld,
                       int64_t bs, int box_inner, int box_rows) {
  PFN_encodeTiled_t enc = get_encode();
  if (!enc) return false;
  cuuint64_t dims[3] = {(cuuint64_t)inner, (cuuint64_t)rows, (cuuint64_t)batch};
  cuuint64_t strides[2] = {(cuuint64_t)(ld * 2), (cuuint64_t)((batch > 1 ? bs : ld * rows) * 2)};
  cuuint32_t box[3] = {(cuuint32_t)box_inner, (cuuint32_t)box_rows, 1u};
  cuuint32_t estr[3] = {1u, 1u, 1u};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(ptr), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

omq_status gemm_launch_qb(cudaStream_t st, int64_t M, int64_t N, int64_t K, const GemmOperand& A, const GemmOperand& B,
                          const GemmEpilogue& ep, const GemmQuantB& qb, int32_t* status) {
  OMQ_REQUIRE(M > 0 && N > 0 && K > 0 && M < (1ll << 31) && N < (1ll << 31) && K < (1ll << 31), OMQ_ERR_SHAPE);
  OMQ_REQUIRE(A.ptr && B.ptr && (ep.Cf || ep.Cb) && qb.h && qb.z, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(A.kmajor, OMQ_ERR_UNSUPPORTED);
  const int64_t wcols = B.kmajor ? K : N;            // the weight's own column count
  OMQ_REQUIRE(qb.group > 0 && qb.group % 8 == 0 && wcols % qb.group == 0 && K % 8 == 0 && N % 8 == 0, OMQ_ERR_SHAPE);
  OMQ_REQUIRE(omq_aligned16(A.ptr) && omq_aligned16(B.ptr) && A.ld % 8 == 0 && B.ld % 8 == 0, OMQ_ERR_ALIGN);
  OMQ_REQUIRE(ep.ldc % 8 == 0 && ep.ldc >= N, OMQ_ERR_ALIGN);
  OMQ_REQUIRE((!ep.Cf || omq_aligned16(ep.Cf)) && (!ep.Cb || omq_aligned16(ep.Cb)), OMQ_ERR_ALIGN);
  OMQ_REQUIRE(!ep.R || (omq_aligned16(ep.R) && ep.ldr % 4 == 0), OMQ_ERR_ALIGN);
  OMQ_REQUIRE((!ep.bias || omq_aligned16(ep.bias)) && (!qb.s || omq_aligned16(qb.s)), OMQ_ERR_ALIGN);
  const bool pair = gemm_n_tile(N) == 256 && M > BM;   // pairs: 128 B rows per CTA; else BN = 128
  CUtensorMap ta, tb, tc;
  memset(&tc, 0, sizeof(tc));
  bool ok = make_map(&ta, A.ptr, K, M, 1, A.ld, 0, BM) &&
            (B.kmajor ? make_map(&tb, B.ptr, K, N, 1, B.ld, 0, 128) : make_map(&tb, B.ptr, N, K, 1, B.ld, 0, BK));
  if (ep.Cf) ok = ok && make_map_c(&tc, ep.Cf, N, M, 1, ep.ldc, 0);
  if (!ok) return OMQ_ERR_UNSUPPORTED;
  GemmParams p;
  memset(&p, 0, sizeof(p));
  p.M = (int)M; p.N = (int)N; p.K = (int)K; p.batch = 1;
  p.a_mn = 0; p.b_mn = B.kmajor ? 0 : 1; p.causal = 0; p.ep = ep; p.qb = qb; p.status = status; p.pair = pair ? 1 : 0;
  p.n_fast = ((double)M > 1.5 * (double)N) ? 1 : 0;
  p.wait_ns = OMQ_WAIT_LIMIT_NS; p.withhold = 0;
  cudaEvent_t e0 = nullptr, e1 = nullptr;
  if (g_prof.on) {
    e0 = prof_event();
    e1 = prof_event();
    if (e0 && e1) {
      cudaEventRecord(e0, st);
      g_prof.flops += gemm_algorithmic_flops(M, N, K, 1, 0);
    }
  }
  omq_status r = pair ? launch_cfg<256, 6, LWC_OPERAND, true>(st, ta, tb, tc, p)
                      : launch_cfg<128, 6, LWC_OPERAND>(st, ta, tb, tc, p);
  if (e0 && e1) cudaEventRecord(e1, st);
  return r;
}

omq_status gemm_launch_lwc(cudaStream_t st, int64_t M, int64_t N, int64_t K, const GemmOperand& A,
                           const GemmOperand& B, const GemmLwcEpi& lw, int32_t* status) {
  OMQ_REQUIRE(M > 0 && N > 0 && K > 0, OMQ_ERR_SHAPE);
  OMQ_REQUIRE(M < (1ll << 31) && N < (1ll << 31) && K < (1ll << 31), OMQ_ERR_SHAPE);
  OMQ_REQUIRE(A.ptr && B.ptr && lw.W && lw.h && lw.z && lw.gb && lw.mv, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(omq_aligned16(A.ptr) && omq_aligned16(B.ptr) && omq_aligned16(lw.W), OMQ_ERR_ALIGN);
  OMQ_REQUIRE(A.ld % 8 == 0 && B.ld % 8 == 0 && N % 32 == 0, OMQ_ERR_ALIGN);
  OMQ_REQUIRE(!lw.s || omq_aligned16(lw.s), OMQ_ERR_ALIGN);
  const int bn = gemm_n_tile(N);
  const bool perch = lw.group == N;
  // a group lies inside one 32-column chunk sequence of one tile; the grouped form carries no LET
  // a group lies inside one half of a tile (the part one epilogue warp drains)
  OMQ_REQUIRE(lw.group > 0 && (perch || (lw.group % 32 == 0 && (bn / 2) % lw.group == 0)), OMQ_ERR_UNSUPPORTED);
  OMQ_REQUIRE(perch || (!lw.s && !lw.r && !lw.dBt && !lw.part_s && !lw.part_d), OMQ_ERR_UNSUPPORTED);
  OMQ_REQUIRE(!perch || (lw.rowpart && lw.ntn == 2 * (int)((N + bn - 1) / bn)), OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(perch || (lw.dgl && lw.dbl && lw.ga && lw.Mv), OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(!lw.part_s || lw.s, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(!lw.part_d || lw.dBt, OMQ_ERR_INVALID_ARG);
  const bool pair = bn == 256 && M > BM;           // CTA pairs, one 256 x 256 tile per pair
  CUtensorMap ta, tb, tc;
  memset(&tc, 0, sizeof(tc));
  bool ok = A.kmajor ? make_map(&ta, A.ptr, K, M, 1, A.ld, 0, BM) : make_map(&ta, A.ptr, M, K, 1, A.ld, 0, BK);
  ok = ok && (B.kmajor ? make_map(&tb, B.ptr, K, N, 1, B.ld, 0, pair ? bn / 2 : bn)
                       : make_map(&tb, B.ptr, N, K, 1, B.ld, 0, BK));
  if (!ok) return OMQ_ERR_UNSUPPORTED;
  GemmParams p;
  memset(&p, 0, sizeof(p));
  p.M = (int)M; p.N = (int)N; p.K = (int)K; p.batch = 1;
  p.a_mn = A.kmajor ? 0 : 1; p.b_mn = B.kmajor ? 0 : 1;
  p.causal = 0; p.lw = lw; p.status = status; p.pair = pair ? 1 : 0;
  p.wait_ns = OMQ_WAIT_LIMIT_NS; p.withhold = 0;
  p.n_fast = ((double)M > 1.5 * (double)N) ? 1 : 0;
  cudaEvent_t e0 = nullptr, e1 = nullptr;
  if (g_prof.on) {
    e0 = prof_event();
    e1 = prof_event();
    if (e0 && e1) {
      cudaEventRecord(e0, st);
      g_prof.flops += gemm_algorithmic_flops(M, N, K, 1, 0);
    }
  }
  const bool nolet = !lw.s && !lw.r && !lw.want_dr && !lw.part_s && !lw.part_d;
  const bool scale_only = lw.s && !lw.r && !lw.want_dr;
  omq_status r = pair ? (nolet        ? launch_cfg<256, 6, 2, true>(st, ta, tb, tc, p)
                         : scale_only ? launch_cfg<256, 6, 3, true>(st, ta, tb, tc, p)
                                      : launch_cfg<256, 6, 1, true>(st, ta, tb, tc, p))
                      : (bn == 256 ? launch_cfg<256, 4, 1>(st, ta, tb, tc, p) : launch_cfg<128, 6, 1>(st, ta, tb, tc, p));
  if (e0 && e1) cudaEventRecord(e1, st);
  return r;
}

extern "C" void omq_profile_begin(void) {
  g_prof.on = true;
  g_prof.used = 0;
  g_prof.flops = 0.0;
}

extern "C" omq_status omq_profile_end(double* gemm_ms, double* gemm_flops, int64_t* gemm_launches) {
  g_prof.on = false;
  double ms = 0.0;
  for (size_t i = 0; i + 1 < g_prof.used; i += 2) {
    if (cudaEventSynchronize(g_prof.ev[i + 1]) != cudaSuccess) return OMQ_ERR_CUDA;
    float t = 0.f;
    if (cudaEventElapsedTime(&t, g_prof.ev[i], g_prof.ev[i + 1]) != cudaSuccess) return OMQ_ERR_CUDA;
    ms += t;
  }
  if (gemm_ms) *gemm_ms = ms;
  if (gemm_flops) *gemm_flops = g_prof.flops;
  if (gemm_launches) *gemm_launches = (int64_t)(g_prof.used / 2);
  g_prof.used = 0;
  return OMQ_OK;
}

extern "C" omq_status omq_gemm_bf16(omq_stream_t stream, int64_t M, int64_t N, int64_t K, int64_t batch, const void* A,
                                    int64_t a_ld, int64_t a_bs, int32_t a_kmajor, const void* B, int64_t b_ld,
                                    int64_t b_bs, int32_t b_kmajor, float* Cf, void* Cb, int64_t ldc, int64_t c_bs,
                                    float alpha, const float* bias, const float* R, int64_t ldr, float beta_acc,
                                    int32_t causal, int32_t* dev_status) {
  GemmOperand a{A, a_ld, a_bs, a_kmajor ? 1 : 0};
  GemmOperand b{B, b_ld, b_bs, b_kmajor ? 1 : 0};
  GemmEpilogue ep{Cf, (__nv_bfloat16*)Cb, ldc, c_bs, alpha, bias, R, ldr, beta_acc};
  return gemm_launch((cudaStream_t)stream, M, N, K, batch, a, b, ep, causal, dev_status);
}

// Failure-detection self-test: the product above on one CTA with every wait bounded by
// wait_limit_ns, and optionally without its first operand load, so that the wait for it expires.
extern "C" omq_status omq_selftest_bounded_wait(omq_stream_t stream, int64_t M, int64_t N, int64_t K, const void* A,
                                                const void* B, float* C, uint64_t wait_limit_ns, int32_t withhold,
                                                int32_t* dev_status) {
  OMQ_REQUIRE(M > 0 && M <= BM && N > 0 && N <= 128 && K > 0 && K <= 8192, OMQ_ERR_SHAPE);
  OMQ_REQUIRE(A && B && C, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(withhold == 0 || withhold == 1, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(wait_limit_ns >= 1000ull && wait_limit_ns <= OMQ_WAIT_LIMIT_NS, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(omq_aligned16(A) && omq_aligned16(B) && omq_aligned16(C), OMQ_ERR_ALIGN);
  OMQ_REQUIRE(K % 8 == 0 && N % 8 == 0, OMQ_ERR_ALIGN);
  CUtensorMap ta, tb, tc;
  bool ok = make_map(&ta, A, K, M, 1, K, 0, BM) && make_map(&tb, B, K, N, 1, K, 0, 128) &&
            make_map_c(&tc, C, N, M, 1, N, 0);
  if (!ok) return OMQ_ERR_UNSUPPORTED;
  GemmParams p;
  memset(&p, 0, sizeof(p));
  p.M = (int)M; p.N = (int)N; p.K = (int)K; p.batch = 1;
  p.a_mn = 0; p.b_mn = 0; p.n_fast = 0; p.causal = 0; p.pair = 0;
  p.ep = GemmEpilogue{C, nullptr, N, 0, 1.f, nullptr, nullptr, 0, 0.f};
  p.status = dev_status;
  p.wait_ns = wait_limit_ns;
  p.withhold = withhold;
  return launch_cfg<128, 6>((cudaStream_t)stream, ta, tb, tc, p);
}
