// Causal attention of the quantized block (Sec. 3.3 / Eq. 5: Q_a-quantized Q~, K~, V' in bf16)
// without materialising the score matrix.
//
// Forward (softmax output not quantized): one CTA per (128-query block, query head), one pass over
// the key blocks.  TMA streams 128-key blocks of K (three slots) and V (two slots); tcgen05.mma
// forms S = Q K^T in one of two tensor-memory buffers while the compute warps work on the previous
// one; each 64-key half of a row turns its scores into unnormalised probabilities 2^(c S - M)
// against its own integer reference M (moved up by whole powers of two, see flash_fwd1_kernel),
// writes them as bf16 into shared memory in the 128-byte-swizzled operand layout, and the MMA warp
// accumulates the half's O += P V in tensor memory; the halves are combined and divided by the
// row sum at the end.  The row log-sum-exp (base 2, scaled logits) is saved for the backward.
// With the softmax output quantized (flash_fwd_kernel<true>), the forward takes two passes: row
// max, sum and extremes first, then the normalised probabilities, quantized per row.
//
// Backward: dKV kernel per (128-key block, kv head) walks the 64-query blocks of every query head
// of its group: S^T = K Q^T and dP^T = V dO^T (double-buffered in tensor memory), P^T and
// dS^T = P^T (dP^T - D) scale formed by the compute warps (one key row per thread),
// dV += P^T dO and dK += dS^T Q accumulated in tensor memory.  dQ kernel per (128-query block,
// query head) recomputes S and dP for its keys and accumulates dQ += dS K.  D = rowsum(dO * O).
//
// Warp roles (320 threads): warp 0 TMA, warp 1 tensor memory + MMA issue, warps 2..9 compute
// (two warps per tensor-memory lane quadrant, each taking half of a block's columns).
// Every mbarrier wait is bounded; on expiry the status word gets OMQ_ERR_TIMEOUT and the kernel
// winds down (frees its tensor memory and returns).
#include "attn.cuh"
#include "tc.cuh"

#include <cstring>

namespace {

using namespace tc;

constexpr int FA_THREADS = 320;            // warp 0 TMA, warp 1 MMA, warps 2..9 compute
constexpr int HD = 128;                     // head dimension
constexpr int ROW_BYTES = 128;              // one swizzle row: 64 bf16

// K-major operand descriptor, k-step kk (16 columns), of a tile whose 64-column atoms are
// atom_bytes apart (atom = rows x 128 bytes)
__device__ __forceinline__ uint64_t desc_k(uint32_t tile, int kk, uint32_t atom_bytes) {
  return sdesc(tile + (kk >> 2) * atom_bytes + (kk & 3) * 32, 16, 1024);
}
// MN-major view of the same tile (rows = K, 64-column atoms = N chunks), k-step kk (16 rows)
__device__ __forceinline__ uint64_t desc_mn(uint32_t tile, int kk, uint32_t atom_bytes) {
  return sdesc(tile + kk * 2048, atom_bytes, 1024);
}

// columns c0 .. c0+31 (c0 a multiple of 32) of row r of a K-major, 128-byte-swizzled bf16 tile
__device__ __forceinline__ void st_row32(uint8_t* tile, uint32_t atom_bytes, int r, int c0, const float* v) {
  uint8_t* row = tile + (c0 >> 6) * atom_bytes + r * ROW_BYTES;
  const int ch0 = (c0 & 63) >> 3;
#pragma unroll
  for (int u = 0; u < 4; ++u) *reinterpret_cast<uint4*>(row + (((ch0 + u) ^ (r & 7)) << 4)) = pack_bf16x8(v + 8 * u);
}


// a [rows x 128] bf16 tile as two {64, rows} boxes (64-column atoms)
__device__ __forceinline__ void load_tile(const CUtensorMap* m, uint64_t* bar, uint8_t* dst, int col0, int row0,
                                          uint32_t atom_bytes) {
  tma_load_3d(m, bar, dst, col0, row0, 0);
  tma_load_3d(m, bar, dst + atom_bytes, col0 + 64, row0, 0);
}

struct Ctl {                 // barriers + tensor-memory holder + abort flag, after the tiles
  uint64_t bar[16];
  uint32_t tmem;
  int abort;
};

__device__ __forceinline__ bool waitb(uint64_t* b, uint32_t parity, int32_t* status, volatile int* abort_flag) {
  if (mbar_wait(b, parity)) return true;
  omq_set_status(status, OMQ_ERR_TIMEOUT);
  *abort_flag = 1;
  return false;
}

// warp-uniform wait of the compute warps (tcgen05.ld / st are warp-collective)
__device__ __forceinline__ bool waitw(uint64_t* b, uint32_t parity, int32_t* status, volatile int* abort_flag) {
  const bool ok = __all_sync(0xffffffffu, mbar_wait(b, parity));
  if (!ok) { omq_set_status(status, OMQ_ERR_TIMEOUT); *abort_flag = 1; }
  return ok;
}

// ================================================================================================
// forward
// ================================================================================================
struct FwdP {
  int T, H, rep;
  int ldl;                   // row stride of lse / pqr (>= T)
  float c;                   // log2(e) / sqrt(head_dim)
  float* O; int64_t ldo;     // [T, H*128] fp32
  float* lse;                // [H, T]: m + log2(l) of the scaled base-2 logits
  int32_t* status;
  float Q, eps;              // softmax-output quantizer: 2^bits - 1, floor of h
  float* pqr;                // [H, T, 8] quantizer state per query row (PQ only)
};

// Quantizer state of one query row of the softmax output (MinMax over the visible keys, Eq. 2
// with gamma = beta = 1): h, 1/h, z, the row's max and min probability M and m (u = m/h is
// m * (1/h)), floored (0/1), first index of the max and of the min (as exact floats).
enum { PQ_H = 0, PQ_RH, PQ_Z, PQ_PMAX, PQ_PMIN, PQ_FL, PQ_IMAX, PQ_IMIN, PQ_N = 8 };
// Backward statistics of one query row (PQ): D = sum_j P_j dP_j with dP the gradient reaching P
// through the quantizer, and the totals that reach the row's max and min (R7).
enum { PG_D = 0, PG_DM, PG_DMIN, PG_N = 4 };

constexpr int F_TILE = 128 * ROW_BYTES * 2;           // 32 KB: [128 x 128] bf16
constexpr int F_ATOM = 128 * ROW_BYTES;               // 16 KB
// K and V in separate rings: K (three slots) is free once S is formed, V (two slots) once P V is
constexpr int F_NK = 3, F_NV = 2;
constexpr int F_Q = 0, F_K = F_TILE, F_V = F_K + F_NK * F_TILE, F_P = F_V + F_NV * F_TILE;
constexpr int F_ST = F_P;                             // row statistics: in the P tile before P is written
constexpr int F_CTL = F_P + F_TILE;
constexpr int F_SMEM = F_CTL + 256 + 1024;            // + barriers + alignment slack
static_assert(F_SMEM <= 227 * 1024, "forward shared memory");

// PQ: the probabilities are quantized per query row before the P V product (softmax-output
// quantization); the statistics pass also finds the row's max and min score with first indices.
template <bool PQ>
__global__ void __launch_bounds__(FA_THREADS, 1)
    flash_fwd_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                     const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmO, const FwdP p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  Ctl* ctl = reinterpret_cast<Ctl*>(smem + F_CTL);
  uint64_t* q_full = &ctl->bar[0];
  uint64_t* k_full = &ctl->bar[1];        // [F_NK]
  uint64_t* k_empty = &ctl->bar[4];       // [F_NK]
  uint64_t* v_full = &ctl->bar[7];        // [F_NV]
  uint64_t* v_empty = &ctl->bar[9];       // [F_NV]
  uint64_t* s_full = &ctl->bar[11];       // [2]
  uint64_t* p_full = &ctl->bar[13];
  uint64_t* o_done = &ctl->bar[14];
  volatile int* abort_flag = &ctl->abort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nqb = (p.T + 127) / 128;
  // blocks launch in x-fastest order: every head's longest query block first
  const int qb = nqb - 1 - (int)blockIdx.y;
  const int h = blockIdx.x, g = h / p.rep;
  const int nkb = qb + 1;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int s = 0; s < F_NK; ++s) { mbar_init(&k_full[s], 1); mbar_init(&k_empty[s], 1); }
    for (int s = 0; s < F_NV; ++s) { mbar_init(&v_full[s], 1); mbar_init(&v_empty[s], 1); }
    for (int s = 0; s < 2; ++s) mbar_init(&s_full[s], 1);
    mbar_init(p_full, 8);
    mbar_init(o_done, 1);
    ctl->abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(&ctl->tmem, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = ctl->tmem;           // S buffers at columns 0 / 128, O at 256

  // iterations 0 .. nkb-1: statistics pass (S only: row max m, row sum l of exp2(c S - m));
  // iterations nkb .. 2 nkb-1: output pass (S again, P = bf16(exp2(c S - m) / l), O += P V)
  const int nit = 2 * nkb;
  if (warp == 0 && lane == 0) {
    mbar_expect_tx(q_full, F_TILE);
    load_tile(&tmQ, q_full, smem + F_Q, h * HD, qb * 128, F_ATOM);
    for (int it = 0; it < nit && !*abort_flag; ++it) {
      const int j = it < nkb ? it : it - nkb;
      const int sk = it % F_NK;
      if (!waitb(&k_empty[sk], ((it / F_NK) & 1) ^ 1, p.status, abort_flag)) break;
      mbar_expect_tx(&k_full[sk], F_TILE);
      load_tile(&tmK, &k_full[sk], smem + F_K + sk * F_TILE, g * HD, j * 128, F_ATOM);
      if (it >= nkb) {
        const int sv = j % F_NV;
        if (!waitb(&v_empty[sv], ((j / F_NV) & 1) ^ 1, p.status, abort_flag)) break;
        mbar_expect_tx(&v_full[sv], F_TILE);
        load_tile(&tmV, &v_full[sv], smem + F_V + sv * F_TILE, g * HD, j * 128, F_ATOM);
      }
    }
  } else if (warp == 1 && lane == 0) {
    constexpr uint32_t ID_S = idesc_bf16(128, 128, 0, 0), ID_O = idesc_bf16(128, 128, 0, 1);
    const uint32_t sq = smem_u32(smem + F_Q), sk = smem_u32(smem + F_K), sv = smem_u32(smem + F_V);
    const uint32_t sp = smem_u32(smem + F_P);
    bool ok = waitb(q_full, 0, p.status, abort_flag);
    auto issue_s = [&](int it) -> bool {
      const int s = it & 1, r = it % F_NK;
      if (!waitb(&k_full[r], (it / F_NK) & 1, p.status, abort_flag)) return false;
      tc_fence_after();
#pragma unroll
      for (int kk = 0; kk < 8; ++kk)
        umma_bf16(tmem + 128 * s, desc_k(sq, kk, F_ATOM), desc_k(sk + r * F_TILE, kk, F_ATOM), ID_S, kk > 0);
      umma_commit(&s_full[s]);
      umma_commit(&k_empty[r]);                       // K is free once S is formed
      return true;
    };
    if (ok) ok = issue_s(0);
    for (int it = 0; ok && it < nit; ++it) {
      // S buffer (it+1)&1 was last read at it-1, whose p_full was waited for below
      if (it + 1 < nit && !issue_s(it + 1)) break;
      if (!waitb(p_full, it & 1, p.status, abort_flag)) break;
      tc_fence_after();
      if (it >= nkb) {
        const int j = it - nkb, r = j % F_NV;
        if (!waitb(&v_full[r], (j / F_NV) & 1, p.status, abort_flag)) break;
        tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < 8; ++kk)
          umma_bf16(tmem + 256, desc_k(sp, kk, F_ATOM), desc_mn(sv + r * F_TILE, kk, F_ATOM), ID_O, (j | kk) != 0);
        umma_commit(o_done);
        umma_commit(&v_empty[r]);
      }
    }
  } else if (warp >= 2) {
    // eight compute warps: warps w and w+4 share TMEM lane quadrant w % 4 (rows), half 0 takes
    // columns 0..63 of each block, half 1 columns 64..127
    const int q = warp & 3, half = (warp - 2) >> 2;
    const int r = q * 32 + lane;                      // row of the block = TMEM lane
    const int row = qb * 128 + r;
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    uint8_t* ptile = smem + F_P;
    float* stat = reinterpret_cast<float*>(smem + F_ST);   // [2 halves][m | l (| PQ extremes)][128 rows]
    float m = -INFINITY, l = 0.f;
    float smax = -INFINITY, smin = INFINITY;        // PQ: raw extreme scores and their first keys
    int imx = 0x7fffffff, imn = 0x7fffffff;
    bool ok = true;
    for (int j = 0; j < nkb; ++j) {                   // pass 1: running max and rescaled sum
      if (!(ok = waitw(&s_full[j & 1], (j >> 1) & 1, p.status, abort_flag))) break;
      tc_fence_after();
      const uint32_t sb = tmem + 128 * (j & 1) + lane_off;
      const bool diag = (j == qb);                    // keys beyond the row exist only here
#pragma unroll 1
      for (int c = 2 * half; c < 2 * half + 2; ++c) {
        float v[32];
        tmem_ld32(sb + 32 * c, v);
        if constexpr (PQ) {                           // row minimum of the visible keys
          float u[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const float a = (diag && 32 * c + i > r) ? INFINITY : v[i];
            const float b = (diag && 32 * c + i + 16 > r) ? INFINITY : v[i + 16];
            u[i] = fminf(a, b);
          }
#pragma unroll
          for (int w = 8; w >= 1; w >>= 1)
#pragma unroll
            for (int i = 0; i < w; ++i) u[i] = fminf(u[i], u[i + w]);
          if (u[0] < smin) {                          // this thread's keys arrive in increasing order:
            smin = u[0];                              // a strict improvement keeps the first index
            int f = 0;
#pragma unroll
            for (int i = 31; i >= 0; --i)
              if (v[i] == smin && !(diag && 32 * c + i > r)) f = i;
            imn = j * 128 + 32 * c + f;
          }
        }
        if (diag) {
#pragma unroll
          for (int i = 0; i < 32; ++i) if (32 * c + i > r) v[i] = -INFINITY;
        }
        float t[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) t[i] = fmaxf(v[i], v[i + 16]);
#pragma unroll
        for (int w = 8; w >= 1; w >>= 1)
#pragma unroll
          for (int i = 0; i < w; ++i) t[i] = fmaxf(t[i], t[i + w]);
        if constexpr (PQ) {
          if (t[0] > smax) {
            smax = t[0];
            int f = 0;
#pragma unroll
            for (int i = 31; i >= 0; --i)
              if (v[i] == smax) f = i;
            imx = j * 128 + 32 * c + f;
          }
        }
        const float m_new = fmaxf(m, t[0] * p.c);
        if (m_new != -INFINITY) {                     // a chunk wholly above the diagonal adds nothing
          float s4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
          for (int i = 0; i < 32; ++i) s4[i & 3] += ex2(fmaf(v[i], p.c, -m_new));
          l = l * ex2(m - m_new) + ((s4[0] + s4[1]) + (s4[2] + s4[3]));
          m = m_new;
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(p_full);
    }
    // combine the two halves of every row (each compute thread reaches this barrier exactly once)
    constexpr int NS = PQ ? 6 : 2;                  // statistics per row and half
    stat[(half * NS + 0) * 128 + r] = m;
    stat[(half * NS + 1) * 128 + r] = l;
    if constexpr (PQ) {
      stat[(half * NS + 2) * 128 + r] = smax;
      stat[(half * NS + 3) * 128 + r] = smin;
      stat[(half * NS + 4) * 128 + r] = __int_as_float(imx);
      stat[(half * NS + 5) * 128 + r] = __int_as_float(imn);
    }
    asm volatile("bar.sync 1, 256;" ::: "memory");
    const int oh = 1 - half;
    const float mo = stat[(oh * NS + 0) * 128 + r], lo = stat[(oh * NS + 1) * 128 + r];
    if constexpr (PQ) {                               // extremes of both halves, first index on ties
      const float xo = stat[(oh * NS + 2) * 128 + r], no = stat[(oh * NS + 3) * 128 + r];
      const int ixo = __float_as_int(stat[(oh * NS + 4) * 128 + r]), ino = __float_as_int(stat[(oh * NS + 5) * 128 + r]);
      if (xo > smax || (xo == smax && ixo < imx)) { smax = xo; imx = ixo; }
      if (no < smin || (no == smin && ino < imn)) { smin = no; imn = ino; }
    }
    asm volatile("bar.sync 1, 256;" ::: "memory");   // statistics read before P overwrites them
    const float mt = fmaxf(m, mo);
    const float lt = (m == -INFINITY ? 0.f : l * ex2(m - mt)) + (mo == -INFINITY ? 0.f : lo * ex2(mo - mt));
    const float inv_l = 1.f / lt;
    // PQ: the row's quantizer from the probabilities of its max and min score (the map from a score
    // to its probability below is the one pass 2 applies to every key)
    QState qs{};
    float Mp = 0.f, mp = 0.f;
    if constexpr (PQ) {
      Mp = ex2(fmaf(smax, p.c, -mt)) * inv_l;
      mp = ex2(fmaf(smin, p.c, -mt)) * inv_l;
      qs = omq_qstate(Mp, mp, 1.f, 1.f, p.Q, p.eps);
    }
    for (int j = 0; ok && j < nkb; ++j) {             // pass 2: probabilities, O += P V
      const int it = nkb + j;
      if (!(ok = waitw(&s_full[it & 1], (it >> 1) & 1, p.status, abort_flag))) break;
      tc_fence_after();
      const uint32_t sb = tmem + 128 * (it & 1) + lane_off;
      const bool diag = (j == qb);
      float v[2][32];
#pragma unroll
      for (int cc = 0; cc < 2; ++cc) {
        const int c = 2 * half + cc;
        tmem_ld32(sb + 32 * c, v[cc]);
#pragma unroll
        for (int i = 0; i < 32; ++i) v[cc][i] = ex2(fmaf(v[cc][i], p.c, -mt)) * inv_l;
        if constexpr (PQ) {
#pragma unroll
          for (int i = 0; i < 32; ++i) v[cc][i] = omq_fakequant(v[cc][i], qs, p.Q, nullptr);
        }
        if (diag) {
#pragma unroll
          for (int i = 0; i < 32; ++i) if (32 * c + i > r) v[cc][i] = 0.f;
        }
      }
      if (j > 0) {                                    // the previous P V product has read P
        if (!(ok = waitw(o_done, (j - 1) & 1, p.status, abort_flag))) break;
        tc_fence_after();
      }
#pragma unroll
      for (int cc = 0; cc < 2; ++cc) st_row32(ptile, F_ATOM, r, 32 * (2 * half + cc), v[cc]);
      fence_async_smem();                             // P visible to the tensor core
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(p_full);
    }
    if (ok && waitw(o_done, (nkb - 1) & 1, p.status, abort_flag)) {
      // O through the copy engine, staged in the K ring (every product that read it has completed)
      tc_fence_after();
      uint8_t* slots = smem + F_K + (warp - 2) * 8192;
      int ns = 0;
#pragma unroll 1
      for (int c = 2 * half; c < 2 * half + 2; ++c) {
        float o[32];
        tmem_ld32(tmem + 256 + lane_off + 32 * c, o);
        store_block32(&tmO, slots + (ns++ & 1) * 4096, o, lane, h * HD + 32 * c, qb * 128 + q * 32);
      }
      if (lane == 0) bulk_wait_all();
      if (row < p.T && half == 0) p.lse[(int64_t)h * p.ldl + row] = mt + log2f(lt);
      if constexpr (PQ) {
        if (row < p.T && half == 0) {
          float4* d = reinterpret_cast<float4*>(p.pqr + ((int64_t)h * p.ldl + row) * PQ_N);
          d[0] = make_float4(qs.h, qs.rh, qs.z, Mp);
          d[1] = make_float4(mp, qs.floored ? 1.f : 0.f, (float)imx, (float)imn);
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// 2^k for an integer-valued k <= 0 (0 below the normal range), exact
__device__ __forceinline__ float pow2_int(float k) {
  return k < -126.f ? 0.f : __int_as_float((127 + (int)k) << 23);
}

// Single-pass forward (softmax output not quantized).  Each 64-key half of a row (one compute warp
// of the pair sharing the row's lane quadrant) keeps its own integer reference M of the scaled
// logits, its own row sum l and its own output accumulator in tensor memory (O_0, O_1): the
// probabilities 2^(c S - M) enter the P V product unnormalised, and when a block lifts the half's
// maximum more than F_TAU above M, M moves up to the ceiling of the new maximum and l and the
// half's accumulator rows are scaled by the exact power of two 2^(M_old - M_new).  Rounding to
// bf16 commutes with powers of two, so the product is exactly that of one common reference; the
// halves are combined and divided by l once, at the end.
constexpr float F_TAU = 8.f;                          // unnormalised probabilities stay below 2^8

__global__ void __launch_bounds__(FA_THREADS, 1)
    flash_fwd1_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                      const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmO, const FwdP p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  Ctl* ctl = reinterpret_cast<Ctl*>(smem + F_CTL);
  uint64_t* q_full = &ctl->bar[0];
  uint64_t* k_full = &ctl->bar[1];        // [F_NK]
  uint64_t* k_empty = &ctl->bar[4];       // [F_NK]
  uint64_t* v_full = &ctl->bar[7];        // [F_NV]
  uint64_t* v_empty = &ctl->bar[9];       // [F_NV]
  uint64_t* s_full = &ctl->bar[11];       // [2]
  uint64_t* p_full = &ctl->bar[13];
  uint64_t* o_done = &ctl->bar[14];
  volatile int* abort_flag = &ctl->abort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nqb = (p.T + 127) / 128;
  const int qb = nqb - 1 - (int)blockIdx.y;           // every head's longest query block first
  const int h = blockIdx.x, g = h / p.rep;
  const int nkb = qb + 1;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int s = 0; s < F_NK; ++s) { mbar_init(&k_full[s], 1); mbar_init(&k_empty[s], 1); }
    for (int s = 0; s < F_NV; ++s) { mbar_init(&v_full[s], 1); mbar_init(&v_empty[s], 1); }
    for (int s = 0; s < 2; ++s) mbar_init(&s_full[s], 1);
    mbar_init(p_full, 8);
    mbar_init(o_done, 1);
    ctl->abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(&ctl->tmem, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = ctl->tmem;           // S buffers at columns 0 / 128, O_0 at 256, O_1 at 384

  if (warp == 0 && lane == 0) {
    mbar_expect_tx(q_full, F_TILE);
    load_tile(&tmQ, q_full, smem + F_Q, h * HD, qb * 128, F_ATOM);
    for (int j = 0; j < nkb && !*abort_flag; ++j) {
      const int sk = j % F_NK, sv = j % F_NV;
      if (!waitb(&k_empty[sk], ((j / F_NK) & 1) ^ 1, p.status, abort_flag)) break;
      mbar_expect_tx(&k_full[sk], F_TILE);
      load_tile(&tmK, &k_full[sk], smem + F_K + sk * F_TILE, g * HD, j * 128, F_ATOM);
      if (!waitb(&v_empty[sv], ((j / F_NV) & 1) ^ 1, p.status, abort_flag)) break;
      mbar_expect_tx(&v_full[sv], F_TILE);
      load_tile(&tmV, &v_full[sv], smem + F_V + sv * F_TILE, g * HD, j * 128, F_ATOM);
    }
  } else if (warp == 1 && lane == 0) {
    constexpr uint32_t ID_S = idesc_bf16(128, 128, 0, 0), ID_O = idesc_bf16(128, 128, 0, 1);
    const uint32_t sq = smem_u32(smem + F_Q), sk = smem_u32(smem + F_K), sv = smem_u32(smem + F_V);
    const uint32_t sp = smem_u32(smem + F_P);
    bool ok = waitb(q_full, 0, p.status, abort_flag);
    auto issue_s = [&](int j) -> bool {
      const int s = j & 1, r = j % F_NK;
      if (!waitb(&k_full[r], (j / F_NK) & 1, p.status, abort_flag)) return false;
      tc_fence_after();
#pragma unroll
      for (int kk = 0; kk < 8; ++kk)
        umma_bf16(tmem + 128 * s, desc_k(sq, kk, F_ATOM), desc_k(sk + r * F_TILE, kk, F_ATOM), ID_S, kk > 0);
      umma_commit(&s_full[s]);
      umma_commit(&k_empty[r]);                       // K is free once S is formed
      return true;
    };
    if (ok) ok = issue_s(0);
    for (int j = 0; ok && j < nkb; ++j) {
      // S buffer (j+1)&1 was last read at j-1, whose p_full was waited for below
      if (j + 1 < nkb && !issue_s(j + 1)) break;
      if (!waitb(p_full, j & 1, p.status, abort_flag)) break;
      const int r = j % F_NV;
      if (!waitb(&v_full[r], (j / F_NV) & 1, p.status, abort_flag)) break;
      tc_fence_after();
      // keys 0..63 of the block (P atom 0, V rows 0..63) into O_0, keys 64..127 into O_1
#pragma unroll
      for (int kk = 0; kk < 8; ++kk)
        umma_bf16(tmem + 256 + 128 * (kk >> 2), desc_k(sp, kk, F_ATOM), desc_mn(sv + r * F_TILE, kk, F_ATOM), ID_O,
                  (j | (kk & 3)) != 0);
      umma_commit(o_done);
      umma_commit(&v_empty[r]);
    }
  } else if (warp >= 2) {
    // eight compute warps: warps w and w+4 share TMEM lane quadrant w % 4 (rows); half 0 takes
    // keys 0..63 of each block, half 1 keys 64..127, each with its own reference and accumulator
    const int q = warp & 3, half = (warp - 2) >> 2;
    const int r = q * 32 + lane;                      // row of the block = TMEM lane
    const int row = qb * 128 + r;
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    const uint32_t o_acc = tmem + 256 + 128 * half + lane_off;
    uint8_t* ptile = smem + F_P;
    float M = -INFINITY, l = 0.f;
    bool ok = true;
    for (int j = 0; j < nkb; ++j) {
      if (!(ok = waitw(&s_full[j & 1], (j >> 1) & 1, p.status, abort_flag))) break;
      tc_fence_after();
      const uint32_t sb = tmem + 128 * (j & 1) + lane_off;
      const bool diag = (j == qb);                    // keys beyond the row exist only here
      float v[2][32];
#pragma unroll
      for (int cc = 0; cc < 2; ++cc) {
        const int c = 2 * half + cc;
        tmem_ld32(sb + 32 * c, v[cc]);
        if (diag) {
#pragma unroll
          for (int i = 0; i < 32; ++i) if (32 * c + i > r) v[cc][i] = -INFINITY;
        }
      }
      float t[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) t[i] = fmaxf(fmaxf(v[0][i], v[0][i + 16]), fmaxf(v[1][i], v[1][i + 16]));
#pragma unroll
      for (int w = 8; w >= 1; w >>= 1)
#pragma unroll
        for (int i = 0; i < w; ++i) t[i] = fmaxf(t[i], t[i + w]);
      const float mb = t[0] * p.c;                    // c > 0: max of c S = c max S
      const bool lift = mb > M + F_TAU;               // false while the half has seen no key (mb = -inf)
      const float Mn = lift ? ceilf(mb) : M;
      const float fac = lift ? (M == -INFINITY ? 0.f : pow2_int(M - Mn)) : 1.f;
      float ls[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int cc = 0; cc < 2; ++cc) {
        const int c = 2 * half + cc;
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const float e = (Mn == -INFINITY || (diag && 32 * c + i > r)) ? 0.f : ex2(fmaf(v[cc][i], p.c, -Mn));
          v[cc][i] = e;
          ls[i & 3] += e;
        }
      }
      l = l * fac + ((ls[0] + ls[1]) + (ls[2] + ls[3]));
      M = Mn;
      if (j > 0) {                                    // the previous P V product has read P, written O
        if (!(ok = waitw(o_done, (j - 1) & 1, p.status, abort_flag))) break;
        tc_fence_after();
        if (__any_sync(0xffffffffu, fac != 1.f)) {    // rows whose reference moved: rescale their O rows
#pragma unroll 1
          for (int c = 0; c < 4; ++c) {
            float o[32];
            tmem_ld32(o_acc + 32 * c, o);
#pragma unroll
            for (int i = 0; i < 32; ++i) o[i] *= fac;
            tmem_st32(o_acc + 32 * c, o);
          }
        }
      }
#pragma unroll
      for (int cc = 0; cc < 2; ++cc) st_row32(ptile, F_ATOM, r, 32 * (2 * half + cc), v[cc]);
      fence_async_smem();                             // P visible to the tensor core
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(p_full);
    }
    // the last P V product has read P: its tile holds the halves' references and sums now
    if (ok) ok = waitw(o_done, (nkb - 1) & 1, p.status, abort_flag);
    float* stat = reinterpret_cast<float*>(smem + F_ST);   // [2 halves][M | l][128 rows]
    stat[(half * 2 + 0) * 128 + r] = M;
    stat[(half * 2 + 1) * 128 + r] = l;
    asm volatile("bar.sync 1, 256;" ::: "memory");   // every compute thread arrives exactly once
    const float M0 = stat[r], l0 = stat[128 + r], M1 = stat[256 + r], l1 = stat[384 + r];
    const float Mt = fmaxf(M0, M1);
    const float f0 = M0 == -INFINITY ? 0.f : pow2_int(M0 - Mt), f1 = M1 == -INFINITY ? 0.f : pow2_int(M1 - Mt);
    const float lt = l0 * f0 + l1 * f1;
    const float a0 = f0 / lt, a1 = f1 / lt;
    if (ok) {
      // O through the copy engine, staged in the K ring (every product that read it has completed)
      tc_fence_after();
      uint8_t* slots = smem + F_K + (warp - 2) * 8192;
      int ns = 0;
#pragma unroll 1
      for (int c = 2 * half; c < 2 * half + 2; ++c) {
        float o0[32], o1[32];
        tmem_ld32(tmem + 256 + lane_off + 32 * c, o0);
        tmem_ld32(tmem + 384 + lane_off + 32 * c, o1);
#pragma unroll
        for (int i = 0; i < 32; ++i) o0[i] = fmaf(o0[i], a0, o1[i] * a1);
        store_block32(&tmO, slots + (ns++ & 1) * 4096, o0, lane, h * HD + 32 * c, qb * 128 + q * 32);
      }
      if (lane == 0) bulk_wait_all();
      if (row < p.T && half == 0) p.lse[(int64_t)h * p.ldl + row] = Mt + log2f(lt);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// ================================================================================================
// backward: D = rowsum(dO * O) per (token, head)
// ================================================================================================
__global__ void attn_rowdot_kernel(int T, int H, const __nv_bfloat16* __restrict__ dO, int64_t lddo,
                                   const float* __restrict__ O, int64_t ldo, float* __restrict__ D, int ldl) {
  const int64_t w = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (w >= (int64_t)T * H) return;
  const int t = (int)(w / H), h = (int)(w % H);
  const float4 o = *reinterpret_cast<const float4*>(O + (int64_t)t * ldo + h * HD + 4 * lane);
  const uint2 u = *reinterpret_cast<const uint2*>(dO + (int64_t)t * lddo + h * HD + 4 * lane);
  const __nv_bfloat162* b = reinterpret_cast<const __nv_bfloat162*>(&u);
  const float2 d01 = __bfloat1622float2(b[0]), d23 = __bfloat1622float2(b[1]);
  const float s = warp_sum(o.x * d01.x + o.y * d01.y + o.z * d23.x + o.w * d23.y);
  if (lane == 0) D[(int64_t)h * ldl + t] = s;
}

// ================================================================================================
// backward, dK and dV: one CTA per (128-key block, kv head)
// ================================================================================================
struct BwdP {
  int T, H, rep;
  int ldl;                   // row stride of lse / D / pqr / pqb (>= T, a multiple of 4)
  float c;                   // log2(e) / sqrt(head_dim)
  float scale;               // 1 / sqrt(head_dim)
  const float* lse; const float* D;      // [H, T]
  float* dQ; int64_t ldq;    // [T, H*128]
  float* dK; float* dV; int64_t ldkv;    // [T, Hkv*128]
  int32_t* status;
  float Q;                   // PQ: 2^bits - 1 of the softmax-output quantizer
  const float* pqr;          // PQ: [H, T, PQ_N] forward quantizer state
  float* pqb;                // PQ: [H, T, PG_N] backward row statistics
};

constexpr int B_QATOM = 64 * ROW_BYTES;               // 8 KB: 64-row atom
constexpr int B_QTILE = 2 * B_QATOM;                  // [64 x 128] bf16

// dKV shared-memory layout.  Ring slots hold Q, dO and the row data of a 64-query block: lse and
// D (plain), or lse, the quantizer state and the backward row statistics (PQ, two slots).
template <bool PQ>
struct BL {
  static constexpr int NQD = PQ ? 2 : 3;              // slots of the Q / dO / row-data ring
  static constexpr int RD = PQ ? 64 * 4 * (1 + PQ_N + PG_N) : 512;   // row-data bytes per slot
  static constexpr int K = 0, V = F_TILE, Qo = 2 * F_TILE, DO = Qo + NQD * B_QTILE;
  static constexpr int PT = DO + NQD * B_QTILE;       // P^T [128 keys x 64 queries]: 16 KB, two buffers
  static constexpr int DST = PT + 2 * F_ATOM;         // dS^T, same shape, two buffers
  static constexpr int LD = DST + 2 * F_ATOM;         // [slot][row data]
  static constexpr int CTL = LD + NQD * RD;
  static constexpr int SMEM = CTL + 256 + 1024;       // + barriers + alignment slack
};
static_assert(sizeof(Ctl) <= 256 && BL<false>::SMEM <= 227 * 1024 && BL<true>::SMEM <= 227 * 1024,
              "dKV shared memory");

template <bool PQ>
__global__ void __launch_bounds__(FA_THREADS, 1)
    flash_bwd_dkv_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                         const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmdO,
                         const __grid_constant__ CUtensorMap tmdK, const __grid_constant__ CUtensorMap tmdV,
                         const BwdP p) {
  using L = BL<PQ>;
  constexpr int B_NQD = L::NQD;
  constexpr int B_K = L::K, B_V = L::V, B_Q = L::Qo, B_DO = L::DO, B_PT = L::PT, B_DST = L::DST, B_LD = L::LD;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  Ctl* ctl = reinterpret_cast<Ctl*>(smem + L::CTL);
  uint64_t* kv_full = &ctl->bar[0];
  uint64_t* qd_full = &ctl->bar[1];      // [B_NQD]
  uint64_t* qd_empty = &ctl->bar[1 + B_NQD];   // [B_NQD]
  uint64_t* s_full = &ctl->bar[1 + 2 * B_NQD];   // [2]: S^T and dP^T of a query block ready
  uint64_t* p_full = &ctl->bar[3 + 2 * B_NQD];   // P^T, dS^T written
  uint64_t* g_done = &ctl->bar[4 + 2 * B_NQD];   // [2]: dV / dK products that read P^T / dS^T buffer b done
  volatile int* abort_flag = &ctl->abort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int kb = blockIdx.y, g = blockIdx.x;           // key block 0 (most queries) of every head first
  const int nq64 = (p.T + 63) / 64;
  const int i0 = 2 * kb;                              // first 64-query block with a visible key
  const int niq = nq64 > i0 ? nq64 - i0 : 0;
  const int nit = niq * p.rep;                        // (head, query block) iterations

  if (threadIdx.x == 0) {
    mbar_init(kv_full, 1);
    for (int s = 0; s < B_NQD; ++s) { mbar_init(&qd_full[s], 1); mbar_init(&qd_empty[s], 1); }
    for (int s = 0; s < 2; ++s) mbar_init(&s_full[s], 1);
    mbar_init(p_full, 8);
    mbar_init(&g_done[0], 1);
    mbar_init(&g_done[1], 1);
    ctl->abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(&ctl->tmem, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // tensor memory: S^T at 0 / 64, dP^T at 128 / 192 (per buffer), dV at 256, dK at 384
  const uint32_t tmem = ctl->tmem;

  if (warp == 0 && lane == 0) {
    mbar_expect_tx(kv_full, 2 * F_TILE);
    load_tile(&tmK, kv_full, smem + B_K, g * HD, kb * 128, F_ATOM);
    load_tile(&tmV, kv_full, smem + B_V, g * HD, kb * 128, F_ATOM);
    for (int it = 0; it < nit && !*abort_flag; ++it) {
      const int s = it % B_NQD;
      const int h = g * p.rep + it / niq, qi = i0 + it % niq;
      if (!waitb(&qd_empty[s], ((it / B_NQD) & 1) ^ 1, p.status, abort_flag)) break;
      const uint32_t nb = (uint32_t)min(64, p.ldl - qi * 64) * 4;   // lse / D bytes inside [0, ldl)
      const int64_t r0 = (int64_t)h * p.ldl + qi * 64;
      float* ld = reinterpret_cast<float*>(smem + B_LD + s * L::RD);  // s: the ring slot
      if constexpr (PQ) {
        mbar_expect_tx(&qd_full[s], 2 * B_QTILE + (1 + PQ_N + PG_N) * nb);
        bulk_g2s(ld, p.lse + r0, nb, &qd_full[s]);
        bulk_g2s(ld + 64, p.pqr + r0 * PQ_N, PQ_N * nb, &qd_full[s]);
        bulk_g2s(ld + 64 * (1 + PQ_N), p.pqb + r0 * PG_N, PG_N * nb, &qd_full[s]);
      } else {
        mbar_expect_tx(&qd_full[s], 2 * B_QTILE + 2 * nb);
        bulk_g2s(ld, p.lse + r0, nb, &qd_full[s]);
        bulk_g2s(ld + 64, p.D + r0, nb, &qd_full[s]);
      }
      load_tile(&tmQ, &qd_full[s], smem + B_Q + s * B_QTILE, h * HD, qi * 64, B_QATOM);
      load_tile(&tmdO, &qd_full[s], smem + B_DO + s * B_QTILE, h * HD, qi * 64, B_QATOM);
    }
  } else if (warp == 1 && lane == 0) {
    constexpr uint32_t ID_S = idesc_bf16(128, 64, 0, 0), ID_G = idesc_bf16(128, 128, 0, 1);
    const uint32_t sk = smem_u32(smem + B_K), sv = smem_u32(smem + B_V);
    const uint32_t sq = smem_u32(smem + B_Q), sd = smem_u32(smem + B_DO);
    const uint32_t spt = smem_u32(smem + B_PT), sdst = smem_u32(smem + B_DST);
    bool ok = waitb(kv_full, 0, p.status, abort_flag);
    // ring slot r = it % B_NQD holds Q, dO of iteration it; S^T / dP^T (tensor memory) and P^T /
    // dS^T (shared memory) are double-buffered by b = it & 1
    auto issue_s = [&](int it) -> bool {
      const int r = it % B_NQD, b = it & 1;
      if (!waitb(&qd_full[r], (it / B_NQD) & 1, p.status, abort_flag)) return false;
      tc_fence_after();
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        umma_bf16(tmem + 64 * b, desc_k(sk, kk, F_ATOM), desc_k(sq + r * B_QTILE, kk, B_QATOM), ID_S, kk > 0);
        umma_bf16(tmem + 128 + 64 * b, desc_k(sv, kk, F_ATOM), desc_k(sd + r * B_QTILE, kk, B_QATOM), ID_S, kk > 0);
      }
      umma_commit(&s_full[b]);
      return true;
    };
    if (ok && nit > 0) ok = issue_s(0);
    for (int it = 0; ok && it < nit; ++it) {
      const int r = it % B_NQD, b = it & 1;
      if (it + 1 < nit && !issue_s(it + 1)) break;
      if (!waitb(p_full, it & 1, p.status, abort_flag)) break;
      tc_fence_after();
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {               // K = 64 queries
        umma_bf16(tmem + 256, desc_k(spt + b * F_ATOM, kk, F_ATOM), desc_mn(sd + r * B_QTILE, kk, B_QATOM), ID_G,
                  (it | kk) != 0);
        umma_bf16(tmem + 384, desc_k(sdst + b * F_ATOM, kk, F_ATOM), desc_mn(sq + r * B_QTILE, kk, B_QATOM), ID_G,
                  (it | kk) != 0);
      }
      umma_commit(&g_done[b]);
      umma_commit(&qd_empty[r]);
    }
  } else if (warp >= 2) {
    const int q = warp & 3, half = (warp - 2) >> 2;   // half: which 32 of the 64 query columns
    const int r = q * 32 + lane;                      // key row of the block = TMEM lane
    const int key = kb * 128 + r;
    const float fkey = (float)key;                    // PQ: compared with the rows' extreme indices
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    uint8_t* pt = smem + B_PT;
    uint8_t* dst = smem + B_DST;
    bool ok = true;
    for (int it = 0; it < nit; ++it) {
      const int s = it & 1;
      const int qi = i0 + it % niq;
      const float* Lr = reinterpret_cast<const float*>(smem + B_LD + (it % B_NQD) * L::RD);
      const float* Dq = Lr + 64;
      const float* R8 = Lr + 64;                      // PQ: quantizer state, then row statistics
      const float* G4 = Lr + 64 * (1 + PQ_N);
      // queries below the key block's last key, or past T, need the mask; the rest see every key
      const bool need_mask = qi * 64 < kb * 128 + 127 || qi * 64 + 64 > p.T;
      if (!(ok = waitw(&s_full[s], (it >> 1) & 1, p.status, abort_flag))) break;
      tc_fence_after();
      {
        const int c = half;
        float sv[32], dp[32];
        tmem_ld32(tmem + 64 * s + lane_off + 32 * c, sv);
        tmem_ld32(tmem + 128 + 64 * s + lane_off + 32 * c, dp);
        if constexpr (PQ) {
          // dV takes the quantized probabilities; dS = P (dP - D) with dP the gradient that reaches P
          // through the quantizer: straight through inside the clamp range, plus the totals of the
          // row's max and min at their first keys
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const int qc = 32 * c + i;
            const float4 s0 = reinterpret_cast<const float4*>(R8 + qc * PQ_N)[0];   // h, 1/h, z, M
            const float4 s1 = reinterpret_cast<const float4*>(R8 + qc * PQ_N)[1];   // m, fl, imax, imin
            const float4 gs = *reinterpret_cast<const float4*>(G4 + qc * PG_N);     // D, dM, dm
            const float pv = ex2(fmaf(sv[i], p.c, -Lr[qc]));
            const float rr = omq_round_quot(pv, s0.x, s0.y);
            const float cd = rr + s0.z;
            const bool inr = cd >= 0.f && cd <= p.Q;
            float g = inr ? dp[i] : 0.f;
            if (fkey == s1.z) g += gs.y;
            if (fkey == s1.w) g += gs.z;
            sv[i] = __fmul_rn(fminf(fmaxf(rr, -s0.z), p.Q - s0.z), s0.x);
            dp[i] = pv * (g - gs.x) * p.scale;
          }
        } else {
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const float pv = ex2(fmaf(sv[i], p.c, -Lr[32 * c + i]));
            sv[i] = pv;
            dp[i] = pv * (dp[i] - Dq[32 * c + i]) * p.scale;
          }
        }
        if (need_mask) {
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const int qrow = qi * 64 + 32 * c + i;
            if (key > qrow || qrow >= p.T) { sv[i] = 0.f; dp[i] = 0.f; }
          }
        }
        // buffer s was last read by the dV / dK products of it-2: phase (it >> 1) - 1 of g_done[s]
        // (each buffer's barrier is waited phase by phase, never more than one phase behind)
        if (it >= 2 && !(ok = waitw(&g_done[s], ((it >> 1) - 1) & 1, p.status, abort_flag))) break;
        tc_fence_after();
        st_row32(pt + s * F_ATOM, F_ATOM, r, 32 * c, sv);
        st_row32(dst + s * F_ATOM, F_ATOM, r, 32 * c, dp);
      }
      fence_async_smem();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(p_full);
    }
    for (int b = 0; ok && b < 2 && b < nit; ++b) {  // the last use of each buffer
      const int last = ((nit - 1 - b) & ~1) + b;
      ok = waitw(&g_done[b], (last >> 1) & 1, p.status, abort_flag);
    }
    if (ok && nit > 0) {
      // dV, dK leave through the copy engine: each warp stages its 32 x 32 blocks in two 4 KB slots
      // of the P^T / dS^T buffers (every product that read them has completed) and stores them
      // whole; rows past T are clipped by the copy
      tc_fence_after();
      uint8_t* slots = smem + B_PT + (warp - 2) * 8192;
      int ns = 0;
#pragma unroll 1
      for (int c = 2 * half; c < 2 * half + 2; ++c) {
        float dv[32], dk[32];
        tmem_ld32(tmem + 256 + lane_off + 32 * c, dv);
        tmem_ld32(tmem + 384 + lane_off + 32 * c, dk);
        store_block32(&tmdV, slots + (ns++ & 1) * 4096, dv, lane, g * HD + 32 * c, kb * 128 + q * 32);
        store_block32(&tmdK, slots + (ns++ & 1) * 4096, dk, lane, g * HD + 32 * c, kb * 128 + q * 32);
      }
      if (lane == 0) bulk_wait_all();
    } else if (ok && nit == 0 && key < p.T) {        // keys no query sees (cannot happen for T > 0)
      for (int c = 64 * half; c < 64 * half + 64; ++c) {
        p.dV[(int64_t)key * p.ldkv + g * HD + c] = 0.f;
        p.dK[(int64_t)key * p.ldkv + g * HD + c] = 0.f;
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// ================================================================================================
// backward, dQ: one CTA per (128-query block, query head), 64-key blocks, S / dP / dS double-buffered
// ================================================================================================
constexpr int Q_NKV = 4;                              // slots of the K / V ring
constexpr int Q_Q = 0, Q_DO = F_TILE, Q_K = 2 * F_TILE, Q_V = Q_K + Q_NKV * B_QTILE, Q_DS = Q_V + Q_NKV * B_QTILE;
constexpr int Q_CTL = Q_DS + 2 * F_ATOM;
constexpr int Q_SMEM = Q_CTL + 256 + 1024;            // + barriers + alignment slack
static_assert(Q_SMEM <= 227 * 1024, "dQ shared memory");

// MODE 0: dQ.  PQ (softmax-output quantization): MODE 1 is a statistics pass over the same products
// (no dQ) that writes each query row's backward statistics (PG_*); MODE 2 is dQ with dS formed as
// in the PQ dKV kernel.
template <int MODE>
__global__ void __launch_bounds__(FA_THREADS, 1)
    flash_bwd_dq_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                        const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmdO,
                        const __grid_constant__ CUtensorMap tmdQ, const BwdP p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  Ctl* ctl = reinterpret_cast<Ctl*>(smem + Q_CTL);
  uint64_t* q_full = &ctl->bar[0];
  uint64_t* kv_full = &ctl->bar[1];      // [Q_NKV]
  uint64_t* kv_empty = &ctl->bar[1 + Q_NKV];     // [Q_NKV]
  uint64_t* s_full = &ctl->bar[1 + 2 * Q_NKV];   // [2]: S and dP of a key block ready
  uint64_t* p_full = &ctl->bar[3 + 2 * Q_NKV];   // dS written
  uint64_t* g_done = &ctl->bar[4 + 2 * Q_NKV];   // [2]: dQ product that read dS buffer b done
  volatile int* abort_flag = &ctl->abort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nqb = (p.T + 127) / 128;
  const int qb = nqb - 1 - (int)blockIdx.y;           // longest query blocks of every head first
  const int h = blockIdx.x, g = h / p.rep;
  const int nkb = 2 * qb + 2;                         // 64-key blocks up to the block's last query

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int s = 0; s < Q_NKV; ++s) { mbar_init(&kv_full[s], 1); mbar_init(&kv_empty[s], 1); }
    for (int s = 0; s < 2; ++s) mbar_init(&s_full[s], 1);
    mbar_init(p_full, 8);
    mbar_init(&g_done[0], 1);
    mbar_init(&g_done[1], 1);
    ctl->abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(&ctl->tmem, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = ctl->tmem;       // S at 0 / 64, dP at 128 / 192, dQ at 256

  if (warp == 0 && lane == 0) {
    mbar_expect_tx(q_full, 2 * F_TILE);
    load_tile(&tmQ, q_full, smem + Q_Q, h * HD, qb * 128, F_ATOM);
    load_tile(&tmdO, q_full, smem + Q_DO, h * HD, qb * 128, F_ATOM);
    for (int j = 0; j < nkb && !*abort_flag; ++j) {
      const int s = j % Q_NKV;
      if (!waitb(&kv_empty[s], ((j / Q_NKV) & 1) ^ 1, p.status, abort_flag)) break;
      mbar_expect_tx(&kv_full[s], 2 * B_QTILE);
      load_tile(&tmK, &kv_full[s], smem + Q_K + s * B_QTILE, g * HD, j * 64, B_QATOM);
      load_tile(&tmV, &kv_full[s], smem + Q_V + s * B_QTILE, g * HD, j * 64, B_QATOM);
    }
  } else if (warp == 1 && lane == 0) {
    constexpr uint32_t ID_S = idesc_bf16(128, 64, 0, 0), ID_G = idesc_bf16(128, 128, 0, 1);
    const uint32_t sq = smem_u32(smem + Q_Q), sd = smem_u32(smem + Q_DO);
    const uint32_t sk = smem_u32(smem + Q_K), sv = smem_u32(smem + Q_V), sds = smem_u32(smem + Q_DS);
    bool ok = waitb(q_full, 0, p.status, abort_flag);
    // ring slot r = j % Q_NKV holds K, V of key block j; S / dP (tensor memory) and dS (shared
    // memory) are double-buffered by b = j & 1
    auto issue_s = [&](int j) -> bool {
      const int r = j % Q_NKV, b = j & 1;
      if (!waitb(&kv_full[r], (j / Q_NKV) & 1, p.status, abort_flag)) return false;
      tc_fence_after();
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        umma_bf16(tmem + 64 * b, desc_k(sq, kk, F_ATOM), desc_k(sk + r * B_QTILE, kk, B_QATOM), ID_S, kk > 0);
        umma_bf16(tmem + 128 + 64 * b, desc_k(sd, kk, F_ATOM), desc_k(sv + r * B_QTILE, kk, B_QATOM), ID_S, kk > 0);
      }
      umma_commit(&s_full[b]);
      return true;
    };
    if (ok) ok = issue_s(0);
    for (int j = 0; ok && j < nkb; ++j) {
      const int r = j % Q_NKV, b = j & 1;
      // S / dP buffer (j+1)&1 was last read at j-1, whose p_full was waited for below
      if (j + 1 < nkb && !issue_s(j + 1)) break;
      if (!waitb(p_full, j & 1, p.status, abort_flag)) break;
      tc_fence_after();
      if constexpr (MODE != 1) {
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)             // K = 64 keys
          umma_bf16(tmem + 256, desc_k(sds + b * F_ATOM, kk, F_ATOM), desc_mn(sk + r * B_QTILE, kk, B_QATOM), ID_G,
                    (j | kk) != 0);
      }
      umma_commit(&g_done[b]);
      umma_commit(&kv_empty[r]);
    }
  } else if (warp >= 2) {
    const int q = warp & 3, half = (warp - 2) >> 2;   // half: which 32 of the 64 key columns
    const int r = q * 32 + lane;
    const int row = qb * 128 + r;
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    const bool row_ok = row < p.T;
    const float Lr = row_ok ? p.lse[(int64_t)h * p.ldl + row] : 0.f;
    float Dr = (MODE == 0 && row_ok) ? p.D[(int64_t)h * p.ldl + row] : 0.f;
    // PQ: the row's quantizer state (and, for MODE 2, its backward statistics)
    float q_h = 1.f, q_rh = 0.f, q_z = 0.f, q_ru = 0.f, q_fl = 1.f, q_M = 0.f, q_m = 0.f;
    int q_imax = -1, q_imin = -1;
    float g_dM = 0.f, g_dm = 0.f;
    if (MODE != 0 && row_ok) {
      const float4* st = reinterpret_cast<const float4*>(p.pqr + ((int64_t)h * p.ldl + row) * PQ_N);
      const float4 a0 = st[0], a1 = st[1];
      const float u = __fmul_rn(a1.x, a0.y);        // m / h as the forward formed it
      q_h = a0.x; q_rh = a0.y; q_z = a0.z; q_M = a0.w; q_m = a1.x; q_ru = -a0.z - u; q_fl = a1.y;
      q_imax = (int)a1.z; q_imin = (int)a1.w;
      if (MODE == 2) {
        const float4 gs = *reinterpret_cast<const float4*>(p.pqb + ((int64_t)h * p.ldl + row) * PG_N);
        Dr = gs.x; g_dM = gs.y; g_dm = gs.z;
      }
    }
    // MODE 1 sums over the row's keys: sum of P dP inside the clamp range, the h-path total G_h and
    // the clamped total
    float a_E = 0.f, a_Gh = 0.f, a_Gc = 0.f;
    bool ok = true;
    for (int j = 0; j < nkb; ++j) {
      const int s = j & 1;
      if (!(ok = waitw(&s_full[s], (j >> 1) & 1, p.status, abort_flag))) break;
      tc_fence_after();
      // dS buffer s was last read by the dQ product of j-2: phase (j >> 1) - 1 of g_done[s]
      if (j >= 2 && !(ok = waitw(&g_done[s], ((j >> 1) - 1) & 1, p.status, abort_flag))) break;
      tc_fence_after();
      const bool need_mask = j * 64 + 63 > qb * 128 || !row_ok;
      uint8_t* dst = smem + Q_DS + s * F_ATOM;
      {
        const int c = half;
        float sv[32], dp[32];
        tmem_ld32(tmem + 64 * s + lane_off + 32 * c, sv);
        tmem_ld32(tmem + 128 + 64 * s + lane_off + 32 * c, dp);
        if constexpr (MODE == 0) {
#pragma unroll
          for (int i = 0; i < 32; ++i) dp[i] = ex2(fmaf(sv[i], p.c, -Lr)) * (dp[i] - Dr) * p.scale;
        } else {
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const int key = j * 64 + 32 * c + i;
            const bool vis = !need_mask || (key <= row && row_ok);
            const float pv = ex2(fmaf(sv[i], p.c, -Lr));
            const float x = __fmul_rn(pv, q_rh);
            const float rr = omq_round_quot(pv, q_h, q_rh);
            const float cd = rr + q_z;
            const bool inr = cd >= 0.f && cd <= p.Q;
            if constexpr (MODE == 1) {
              if (vis) {
                const float dh = inr ? rr - x : (cd < 0.f ? q_ru : p.Q + q_ru);
                if (inr) a_E = fmaf(pv, dp[i], a_E); else a_Gc += dp[i];
                a_Gh = fmaf(dp[i], dh, a_Gh);
              }
            } else {
              float g = inr ? dp[i] : 0.f;
              if (key == q_imax) g += g_dM;
              if (key == q_imin) g += g_dm;
              dp[i] = pv * (g - Dr) * p.scale;
            }
          }
        }
        if constexpr (MODE != 1) {
          if (need_mask) {
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if (j * 64 + 32 * c + i > row || !row_ok) dp[i] = 0.f;
          }
          st_row32(dst, F_ATOM, r, 32 * c, dp);
        }
      }
      fence_async_smem();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(p_full);
    }
    for (int b = 0; ok && b < 2 && b < nkb; ++b) {  // the last use of each buffer
      const int last = ((nkb - 1 - b) & ~1) + b;
      ok = waitw(&g_done[b], (last >> 1) & 1, p.status, abort_flag);
    }
    if constexpr (MODE == 1) {
      // combine the two halves of every row through the (unused) dS buffers; every compute thread
      // reaches this barrier exactly once
      float* x3 = reinterpret_cast<float*>(smem + Q_DS);              // [half][3][128]
      x3[(half * 3 + 0) * 128 + r] = a_E;
      x3[(half * 3 + 1) * 128 + r] = a_Gh;
      x3[(half * 3 + 2) * 128 + r] = a_Gc;
      asm volatile("bar.sync 1, 256;" ::: "memory");
      if (ok && half == 0 && row_ok) {
        float t[3];
#pragma unroll
        for (int k = 0; k < 3; ++k) t[k] = x3[k * 128 + r] + x3[(3 + k) * 128 + r];
        const float Gh = q_fl != 0.f ? 0.f : t[1];    // a floored step has no gradient
        const float dM = Gh / p.Q, dm = t[2] - Gh / p.Q;
        // sum_j P_j dP_j, dP including the totals that reach the max and the min (R7)
        *reinterpret_cast<float4*>(p.pqb + ((int64_t)h * p.ldl + row) * PG_N) =
            make_float4(t[0] + q_M * dM + q_m * dm, dM, dm, 0.f);
      }
    } else if (ok) {
      // dQ through the copy engine, staged in the Q / dO tiles (every product that read them has
      // completed): two 4 KB slots per warp, rows past T clipped by the copy
      tc_fence_after();
      uint8_t* slots = smem + Q_Q + (warp - 2) * 8192;
      int ns = 0;
#pragma unroll 1
      for (int c = 2 * half; c < 2 * half + 2; ++c) {
        float o[32];
        tmem_ld32(tmem + 256 + lane_off + 32 * c, o);
        store_block32(&tmdQ, slots + (ns++ & 1) * 4096, o, lane, h * HD + 32 * c, qb * 128 + q * 32);
      }
      if (lane == 0) bulk_wait_all();
      (void)row_ok;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

bool set_smem(const void* fn, int bytes) {
  return cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes) == cudaSuccess;
}

}  // namespace

omq_status flash_fwd_launch(cudaStream_t st, const FlashArgs& a) {
  OMQ_REQUIRE(a.T > 0 && a.H > 0 && a.Hkv > 0 && a.H % a.Hkv == 0 && a.hd == HD, OMQ_ERR_SHAPE);
  OMQ_REQUIRE(a.ldl == 0 || a.ldl >= a.T, OMQ_ERR_SHAPE);
  OMQ_REQUIRE(a.Q && a.K && a.V && a.O && a.lse, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(a.ldq % 8 == 0 && a.ldkv % 8 == 0 && a.ldo % 4 == 0, OMQ_ERR_ALIGN);
  OMQ_REQUIRE(omq_aligned16(a.Q) && omq_aligned16(a.K) && omq_aligned16(a.V) && omq_aligned16(a.O), OMQ_ERR_ALIGN);
  const bool pq = flash_pq_on(a.pbits);
  OMQ_REQUIRE(!pq || a.pqr, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(!pq || omq_aligned16(a.pqr), OMQ_ERR_ALIGN);
  CUtensorMap tq, tk, tv;
  bool ok = omq_make_map_bf16(&tq, a.Q, (int64_t)a.H * HD, a.T, 1, a.ldq, 0, 64, 128);
  ok = ok && omq_make_map_bf16(&tk, a.K, (int64_t)a.Hkv * HD, a.T, 1, a.ldkv, 0, 64, 128);
  ok = ok && omq_make_map_bf16(&tv, a.V, (int64_t)a.Hkv * HD, a.T, 1, a.ldkv, 0, 64, 128);
  CUtensorMap tk64, tv64;
  ok = ok && omq_make_map_bf16(&tk64, a.K, (int64_t)a.Hkv * HD, a.T, 1, a.ldkv, 0, 64, 64);
  ok = ok && omq_make_map_bf16(&tv64, a.V, (int64_t)a.Hkv * HD, a.T, 1, a.ldkv, 0, 64, 64);
  CUtensorMap to;                                   // fp32 O, 32 x 32 store boxes
  ok = ok && omq_make_map_f32_out(&to, a.O, (int64_t)a.H * HD, a.T, a.ldo);
  if (!ok) return OMQ_ERR_UNSUPPORTED;
  static bool attr = false;
  if (!attr) {
    if (!set_smem((const void*)flash_fwd1_kernel, F_SMEM) || !set_smem((const void*)flash_fwd_kernel<true>, F_SMEM))
      return OMQ_ERR_CUDA;
    attr = true;
  }
  FwdP p;
  p.T = a.T; p.H = a.H; p.rep = a.H / a.Hkv;
  p.ldl = a.ldl ? a.ldl : a.T;
  p.c = (float)(1.4426950408889634 / sqrt((double)HD));
  p.O = a.O; p.ldo = a.ldo; p.lse = a.lse; p.status = a.status;
  p.Q = pq ? (float)((1 << a.pbits) - 1) : 0.f; p.eps = a.eps; p.pqr = a.pqr;
  dim3 grid((unsigned)a.H, (unsigned)((a.T + 127) / 128));
  if (pq) flash_fwd_kernel<true><<<grid, FA_THREADS, F_SMEM, st>>>(tq, tk, tv, to, p);
  else flash_fwd1_kernel<<<grid, FA_THREADS, F_SMEM, st>>>(tq, tk, tv, to, p);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

omq_status flash_bwd_launch(cudaStream_t st, const FlashArgs& a) {
  OMQ_REQUIRE(a.T > 0 && a.H > 0 && a.Hkv > 0 && a.H % a.Hkv == 0 && a.hd == HD, OMQ_ERR_SHAPE);
  const bool pq = flash_pq_on(a.pbits);             // O and D are not used then
  OMQ_REQUIRE(a.Q && a.K && a.V && a.lse && a.dO && a.dQ && a.dK && a.dV && (pq || (a.O && a.D)), OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(a.ldq % 8 == 0 && a.ldkv % 8 == 0 && (pq || a.ldo % 4 == 0) && a.lddo % 8 == 0 && a.ldg % 4 == 0 &&
                  a.ldgkv % 4 == 0,
              OMQ_ERR_ALIGN);
  OMQ_REQUIRE(omq_aligned16(a.dO) && omq_aligned16(a.dQ) && omq_aligned16(a.dK) && omq_aligned16(a.dV), OMQ_ERR_ALIGN);
  // lse, D and the PQ row data are fetched by 16-byte bulk copies of whole groups of 4 rows
  const int ldl = a.ldl ? a.ldl : a.T;
  OMQ_REQUIRE(ldl >= a.T, OMQ_ERR_SHAPE);
  OMQ_REQUIRE(ldl % 4 == 0 && omq_aligned16(a.lse) && (pq || omq_aligned16(a.D)), OMQ_ERR_ALIGN);
  OMQ_REQUIRE(!pq || (a.pqr && a.pqb), OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(!pq || (omq_aligned16(a.pqr) && omq_aligned16(a.pqb)), OMQ_ERR_ALIGN);
  CUtensorMap tq64, tdo64, tk, tv, tq, tdo;
  bool ok = omq_make_map_bf16(&tq64, a.Q, (int64_t)a.H * HD, a.T, 1, a.ldq, 0, 64, 64);
  ok = ok && omq_make_map_bf16(&tdo64, a.dO, (int64_t)a.H * HD, a.T, 1, a.lddo, 0, 64, 64);
  ok = ok && omq_make_map_bf16(&tq, a.Q, (int64_t)a.H * HD, a.T, 1, a.ldq, 0, 64, 128);
  ok = ok && omq_make_map_bf16(&tdo, a.dO, (int64_t)a.H * HD, a.T, 1, a.lddo, 0, 64, 128);
  ok = ok && omq_make_map_bf16(&tk, a.K, (int64_t)a.Hkv * HD, a.T, 1, a.ldkv, 0, 64, 128);
  ok = ok && omq_make_map_bf16(&tv, a.V, (int64_t)a.Hkv * HD, a.T, 1, a.ldkv, 0, 64, 128);
  CUtensorMap tk64, tv64;
  ok = ok && omq_make_map_bf16(&tk64, a.K, (int64_t)a.Hkv * HD, a.T, 1, a.ldkv, 0, 64, 64);
  ok = ok && omq_make_map_bf16(&tv64, a.V, (int64_t)a.Hkv * HD, a.T, 1, a.ldkv, 0, 64, 64);
  CUtensorMap tdq, tdk, tdv;                       // fp32 outputs, 32 x 32 store boxes
  ok = ok && omq_make_map_f32_out(&tdq, a.dQ, (int64_t)a.H * HD, a.T, a.ldg);
  ok = ok && omq_make_map_f32_out(&tdk, a.dK, (int64_t)a.Hkv * HD, a.T, a.ldgkv);
  ok = ok && omq_make_map_f32_out(&tdv, a.dV, (int64_t)a.Hkv * HD, a.T, a.ldgkv);
  if (!ok) return OMQ_ERR_UNSUPPORTED;
  static bool attr = false;
  if (!attr) {
    if (!set_smem((const void*)flash_bwd_dkv_kernel<false>, BL<false>::SMEM) ||
        !set_smem((const void*)flash_bwd_dkv_kernel<true>, BL<true>::SMEM) ||
        !set_smem((const void*)flash_bwd_dq_kernel<0>, Q_SMEM) || !set_smem((const void*)flash_bwd_dq_kernel<1>, Q_SMEM) ||
        !set_smem((const void*)flash_bwd_dq_kernel<2>, Q_SMEM))
      return OMQ_ERR_CUDA;
    attr = true;
  }
  BwdP p;
  p.T = a.T; p.H = a.H; p.rep = a.H / a.Hkv;
  p.ldl = ldl;
  p.c = (float)(1.4426950408889634 / sqrt((double)HD));
  p.scale = (float)(1.0 / sqrt((double)HD));
  p.lse = a.lse; p.D = a.D;
  p.dQ = a.dQ; p.ldq = a.ldg; p.dK = a.dK; p.dV = a.dV; p.ldkv = a.ldgkv;
  p.status = a.status;
  p.Q = pq ? (float)((1 << a.pbits) - 1) : 0.f; p.pqr = a.pqr; p.pqb = a.pqb;
  dim3 g1((unsigned)a.Hkv, (unsigned)((a.T + 127) / 128));
  dim3 g2((unsigned)a.H, (unsigned)((a.T + 127) / 128));
  if (pq) {
    // row statistics first (they replace D = rowsum(dO * O), which no longer is sum_j P_j dP_j)
    flash_bwd_dq_kernel<1><<<g2, FA_THREADS, Q_SMEM, st>>>(tq, tk64, tv64, tdo, tdq, p);
    OMQ_LAUNCH_CHECK();
    flash_bwd_dkv_kernel<true><<<g1, FA_THREADS, BL<true>::SMEM, st>>>(tq64, tk, tv, tdo64, tdk, tdv, p);
    OMQ_LAUNCH_CHECK();
    flash_bwd_dq_kernel<2><<<g2, FA_THREADS, Q_SMEM, st>>>(tq, tk64, tv64, tdo, tdq, p);
    OMQ_LAUNCH_CHECK();
    return OMQ_OK;
  }
  if (!a.d_ready) {
    const int64_t rows = (int64_t)a.T * a.H;
    attn_rowdot_kernel<<<(unsigned)((rows + 7) / 8), 256, 0, st>>>(a.T, a.H, a.dO, a.lddo, a.O, a.ldo, a.D, ldl);
    OMQ_LAUNCH_CHECK();
  }
  flash_bwd_dkv_kernel<false><<<g1, FA_THREADS, BL<false>::SMEM, st>>>(tq64, tk, tv, tdo64, tdk, tdv, p);
  OMQ_LAUNCH_CHECK();
  flash_bwd_dq_kernel<0><<<g2, FA_THREADS, Q_SMEM, st>>>(tq, tk64, tv64, tdo, tdq, p);
  OMQ_LAUNCH_CHECK();
  return OMQ_OK;
}

extern "C" omq_status omq_attention_fwd(omq_stream_t stream, int32_t T, int32_t n_heads, int32_t n_kv, const void* Q,
                                        int64_t ldq, const void* K, const void* V, int64_t ldkv, float* O,
                                        int64_t ldo, float* lse, int32_t* dev_status) {
  FlashArgs a{};
  a.T = T; a.H = n_heads; a.Hkv = n_kv; a.hd = HD;
  a.Q = (const __nv_bfloat16*)Q; a.K = (const __nv_bfloat16*)K; a.V = (const __nv_bfloat16*)V;
  a.ldq = ldq; a.ldkv = ldkv; a.O = O; a.ldo = ldo; a.lse = lse; a.status = dev_status;
  return flash_fwd_launch((cudaStream_t)stream, a);
}

extern "C" omq_status omq_attention_bwd(omq_stream_t stream, int32_t T, int32_t n_heads, int32_t n_kv, const void* Q,
                                        int64_t ldq, const void* K, const void* V, int64_t ldkv, const float* O,
                                        int64_t ldo, const float* lse, const void* dO, int64_t lddo, float* D,
                                        float* dQ, int64_t ldg, float* dK, float* dV, int64_t ldgkv,
                                        int32_t* dev_status) {
  FlashArgs a{};
  a.T = T; a.H = n_heads; a.Hkv = n_kv; a.hd = HD;
  a.Q = (const __nv_bfloat16*)Q; a.K = (const __nv_bfloat16*)K; a.V = (const __nv_bfloat16*)V;
  a.ldq = ldq; a.ldkv = ldkv; a.O = const_cast<float*>(O); a.ldo = ldo; a.lse = const_cast<float*>(lse);
  a.dO = (const __nv_bfloat16*)dO; a.lddo = lddo; a.D = D;
  a.dQ = dQ; a.ldg = ldg; a.dK = dK; a.dV = dV; a.ldgkv = ldgkv; a.status = dev_status;
  return flash_bwd_launch((cudaStream_t)stream, a);
}

extern "C" omq_status omq_attention_pq_fwd(omq_stream_t stream, int32_t T, int32_t n_heads, int32_t n_kv,
                                           const void* Q, int64_t ldq, const void* K, const void* V, int64_t ldkv,
                                           float* O, int64_t ldo, float* lse, int32_t pbits, float h_eps,
                                           float* pq_rows, int32_t* dev_status) {
  OMQ_REQUIRE(flash_pq_on(pbits), OMQ_ERR_UNSUPPORTED);
  OMQ_REQUIRE(h_eps > 0.f, OMQ_ERR_INVALID_ARG);
  FlashArgs a{};
  a.T = T; a.H = n_heads; a.Hkv = n_kv; a.hd = HD;
  a.Q = (const __nv_bfloat16*)Q; a.K = (const __nv_bfloat16*)K; a.V = (const __nv_bfloat16*)V;
  a.ldq = ldq; a.ldkv = ldkv; a.O = O; a.ldo = ldo; a.lse = lse; a.status = dev_status;
  a.pbits = pbits; a.eps = h_eps; a.pqr = pq_rows;
  return flash_fwd_launch((cudaStream_t)stream, a);
}

extern "C" omq_status omq_attention_pq_bwd(omq_stream_t stream, int32_t T, int32_t n_heads, int32_t n_kv,
                                           const void* Q, int64_t ldq, const void* K, const void* V, int64_t ldkv,
                                           const float* lse, const void* dO, int64_t lddo, float* dQ, int64_t ldg,
                                           float* dK, float* dV, int64_t ldgkv, int32_t pbits, const float* pq_rows,
                                           float* pq_stats, int32_t* dev_status) {
  OMQ_REQUIRE(flash_pq_on(pbits), OMQ_ERR_UNSUPPORTED);
  FlashArgs a{};
  a.T = T; a.H = n_heads; a.Hkv = n_kv; a.hd = HD;
  a.Q = (const __nv_bfloat16*)Q; a.K = (const __nv_bfloat16*)K; a.V = (const __nv_bfloat16*)V;
  a.ldq = ldq; a.ldkv = ldkv; a.lse = const_cast<float*>(lse);
  a.dO = (const __nv_bfloat16*)dO; a.lddo = lddo;
  a.dQ = dQ; a.ldg = ldg; a.dK = dK; a.dV = dV; a.ldgkv = ldgkv; a.status = dev_status;
  a.pbits = pbits; a.pqr = const_cast<float*>(pq_rows); a.pqb = pq_stats;
  return flash_bwd_launch((cudaStream_t)stream, a);
}
