// One quantized decoder-block calibration step (Algorithm 1, inner loop) and the single quantized
// linear of Eq. 4, enqueued kernel by kernel on one stream.  All scratch lives in the caller's
// workspace, carved by the same routine that reports its size.
#include "attn.cuh"
#include "gemm.cuh"
#include "quant.cuh"

#include <mutex>

namespace {

struct Carve {
  uint8_t* base;
  size_t off;
  template <class T>
  T* take(size_t n) {
    off = (off + 255) & ~size_t(255);
    T* p = base ? reinterpret_cast<T*>(base + off) : nullptr;
    off += n * sizeof(T);
    return p;
  }
};

typedef __nv_bfloat16 bf16;

struct QState4 { float* h; int32_t* z; int32_t* imax; int32_t* imin; float* ga; float* gb; float* M; float* m; };

// Scratch (floats) of the fused weight-gradient + LWC backward of one [Cout, Cin] weight
int64_t lwc_fused_scratch_elems(int64_t Cout, int64_t Cin) {
  const int64_t ntn = 2 * ((Cin + gemm_n_tile(Cin) - 1) / gemm_n_tile(Cin));   // row partials per row
  return 2 * ((Cout + 31) / 32) * Cin + 3 * Cout * ntn + 4 * Cout + 64;
}

bool lwc_fused_ok(int64_t Cin, int group, bool let_terms) {
  if (Cin % 32 != 0) return false;
  if (group == Cin) return true;
  return !let_terms && group % 32 == 0 && (gemm_n_tile(Cin) / 2) % group == 0;
}

QState4 take_qstate(Carve& c, size_t n, bool saved = false) {
  QState4 q;
  q.h = c.take<float>(n); q.z = c.take<int32_t>(n); q.imax = c.take<int32_t>(n); q.imin = c.take<int32_t>(n);
  q.ga = saved ? c.take<float>(n) : nullptr;
  q.gb = saved ? c.take<float>(n) : nullptr;
  q.M = saved ? c.take<float>(n) : nullptr;
  q.m = saved ? c.take<float>(n) : nullptr;
  return q;
}

struct BlockWS {
  // fake-quantized weights and their per-group state
  bf16 *Wqkv_h, *Wo_h, *Wgu_h, *Wd_h;
  QState4 sq_qkv, sq_o, sq_gu, sq_d;
  float *B_qkv, *B_o, *B_gu;
  float *r_qkv, *shift_qkv, *so_exp, *do_exp, *sa_exp;
  float* cs;
  // forward activations
  bf16* a_h; float* rstd1; QState4 sa;
  float* Yqkv; bf16 *Qh, *Kh, *Vh; QState4 sqkv;
  float* lse;                       // [H, T] base-2 log-sum-exp of the attention rows
  float* pqr;                       // [H, T, 8] softmax-output quantizer rows (pbits on only)
  float* O; bf16* O_h; QState4 so;
  float* h1; bf16* b_h; float* rstd2; QState4 sb;
  float* Ygu; bf16* m_h; QState4 sm;
  float* y;
  // backward
  float* loss_part;
  float* dy; bf16* dy_b;
  float* dm;
  float* dW;
  bf16* dYgu_b;                     // dL/d(gate|up), bf16 (the products' operand; fp32 is not kept)
  float* db;
  bf16* dh1_b;
  float* dOh; bf16* dO_b;
  float* Drow;                      // [H, T] rowsum(dO * O)
  float* pqb;                       // [H, T, 4] softmax-output quantizer backward rows (pbits on only)
  float* dQKV; bf16* dYqkv_b;
  float* da;
  float *dB_qkv, *dB_o, *dB_gu, *dr_qkv;
  float *vtmp0, *vtmp1, *vtmp2;     // [max(d, dq)] scratch vectors
  float* part;                      // shared partial-sum scratch
  float* part_aux;                  // scratch of the launches on the auxiliary stream
  float* part2;                     // LET column partials of the second RMSNorm backward (reduced on the auxiliary stream)
  size_t part_elems;
};

int64_t imax64(int64_t a, int64_t b) { return a > b ? a : b; }

// Token rows per CTA of the step's activation-quantizer backward launches (each CTA prefetches its
// next row into L2 while it works on the current one); the RMSNorm backward's LET column partials
// have one row per CTA.
constexpr int kRowsRms = 7, kRowsSwiglu = 1, kRowsPlain = 4;
int64_t rms_parts(int64_t T) { return (T + kRowsRms - 1) / kRowsRms; }

void carve_block(Carve& c, const omq_block_shape& s, const omq_qcfg& cfg, BlockWS& w, bool with_bwd) {
  const int64_t T = s.T, d = s.d, hd = s.head_dim, H = s.n_heads, Hkv = s.n_kv, f = s.ffn;
  const int64_t dq = H * hd, dkv = Hkv * hd, nqkv = dq + 2 * dkv;
  auto ng = [&](int64_t cin) { return cfg.group == 0 ? (int64_t)1 : cin / cfg.group; };
  w.Wqkv_h = (cfg.wbits < 16 && cfg.wprep == 1) ? nullptr : c.take<bf16>(nqkv * d);   // wprep: never formed
  w.Wo_h = c.take<bf16>(d * dq);
  w.Wgu_h = c.take<bf16>(2 * f * d);
  w.Wd_h = c.take<bf16>(d * f);
  w.sq_qkv = take_qstate(c, nqkv * ng(d), true);
  w.sq_o = take_qstate(c, d * ng(dq), true);
  w.sq_gu = take_qstate(c, 2 * f * ng(d), true);
  w.sq_d = take_qstate(c, d * ng(f), true);
  w.B_qkv = c.take<float>(nqkv);
  w.B_o = c.take<float>(d);
  w.B_gu = c.take<float>(2 * f);
  w.r_qkv = c.take<float>(nqkv);
  w.shift_qkv = c.take<float>(nqkv);
  w.so_exp = c.take<float>(dq);
  w.do_exp = c.take<float>(dq);
  w.sa_exp = c.take<float>(dq);
  w.cs = c.take<float>(T * hd);
  w.a_h = c.take<bf16>(T * d);
  w.rstd1 = c.take<float>(T);
  w.sa = take_qstate(c, T);
  w.Yqkv = c.take<float>(T * nqkv);
  w.Qh = c.take<bf16>(T * dq);
  w.Kh = c.take<bf16>(T * dkv);
  w.Vh = c.take<bf16>(T * dkv);
  w.sqkv = take_qstate(c, 3 * T);
  const int64_t T4 = (T + 3) / 4 * 4;       // row stride of the attention's per-row arrays
  w.lse = c.take<float>(H * T4);
  w.pqr = flash_pq_on(cfg.pbits) ? c.take<float>(H * T4 * 8) : nullptr;
  w.O = c.take<float>(T * dq);
  w.O_h = c.take<bf16>(T * dq);
  w.so = take_qstate(c, T);
  w.h1 = c.take<float>(T * d);
  w.b_h = c.take<bf16>(T * d);
  w.rstd2 = c.take<float>(T);
  w.sb = take_qstate(c, T);
  w.Ygu = c.take<float>(T * 2 * f);
  w.m_h = c.take<bf16>(T * f);
  w.sm = take_qstate(c, T);
  w.y = c.take<float>(T * d);
  w.loss_part = c.take<float>(loss_parts(T * d) + 64);
  if (!with_bwd) return;
  w.dy = c.take<float>(T * d);
  w.dy_b = c.take<bf16>(T * d);
  w.dm = c.take<float>(T * f);
  w.dW = c.take<float>(imax64(imax64(nqkv * d, d * dq), imax64(2 * f * d, d * f)));
  w.dYgu_b = c.take<bf16>(T * 2 * f);
  w.db = c.take<float>(T * d);
  w.dh1_b = c.take<bf16>(T * d);
  w.dOh = c.take<float>(T * dq);
  w.dO_b = c.take<bf16>(T * dq);
  w.Drow = c.take<float>(H * T4);
  w.pqb = flash_pq_on(cfg.pbits) ? c.take<float>(H * T4 * 4) : nullptr;
  w.dQKV = c.take<float>(T * nqkv);
  w.dYqkv_b = c.take<bf16>(T * nqkv);
  w.da = c.take<float>(T * d);
  w.dB_qkv = c.take<float>(nqkv);
  w.dB_o = c.take<float>(d);
  w.dB_gu = c.take<float>(2 * f);
  w.dr_qkv = c.take<float>(nqkv);
  const int64_t vmax = imax64(d, dq);
  w.vtmp0 = c.take<float>(vmax);
  w.vtmp1 = c.take<float>(vmax);
  w.vtmp2 = c.take<float>(vmax);
  int64_t pe = 0;
  pe = imax64(pe, (int64_t)lwc_bwd_scratch_bytes(nqkv, d) / 4 + 64);
  pe = imax64(pe, (int64_t)lwc_bwd_scratch_bytes(d, dq) / 4 + 64);
  pe = imax64(pe, (int64_t)lwc_bwd_scratch_bytes(2 * f, d) / 4 + 64);
  pe = imax64(pe, (int64_t)lwc_bwd_scratch_bytes(d, f) / 4 + 64);
  pe = imax64(pe, lwc_fused_scratch_elems(nqkv, d));
  pe = imax64(pe, lwc_fused_scratch_elems(d, dq));
  pe = imax64(pe, lwc_fused_scratch_elems(2 * f, d));
  pe = imax64(pe, lwc_fused_scratch_elems(d, f));
  pe = imax64(pe, 2 * rms_parts(T) * imax64(d, dq));
  pe = imax64(pe, qkv_bwd_nslab((int)T) * (dq + dkv));
  pe = imax64(pe, colsum_rows_parts(T) * imax64(2 * f, nqkv));
  w.part_elems = (size_t)pe;
  w.part = c.take<float>(pe);
  int64_t pa = 0;
  const int64_t lin[4][2] = {{nqkv, d}, {d, dq}, {2 * f, d}, {d, f}};
  for (const auto& l : lin)
    pa = imax64(pa, imax64(lwc_fused_scratch_elems(l[0], l[1]), (int64_t)lwc_bwd_scratch_bytes(l[0], l[1]) / 4 + 64));
  pa = imax64(pa, colsum_rows_parts(T) * imax64(imax64(2 * f, nqkv), d));   // the LET bias column sums
  w.part_aux = c.take<float>(pa);
  w.part2 = c.take<float>(2 * rms_parts(T) * d);
}

omq_status check_block(const omq_block_shape* s, const omq_qcfg* cfg) {
  OMQ_REQUIRE(s, OMQ_ERR_INVALID_ARG);
  OMQ_TRY(omq_check_cfg(cfg));
  OMQ_REQUIRE(s->T > 0 && s->d > 0 && s->n_heads > 0 && s->n_kv > 0 && s->ffn > 0, OMQ_ERR_SHAPE);
  OMQ_REQUIRE(s->head_dim == 128, OMQ_ERR_UNSUPPORTED);
  OMQ_REQUIRE(s->n_heads % s->n_kv == 0, OMQ_ERR_SHAPE);
  OMQ_REQUIRE(s->d % 8 == 0 && s->ffn % 8 == 0, OMQ_ERR_ALIGN);
  if (cfg->group > 0) {
    OMQ_REQUIRE(s->d % cfg->group == 0 && s->ffn % cfg->group == 0 && ((int64_t)s->n_heads * 128) % cfg->group == 0,
                OMQ_ERR_SHAPE);
  }
  return OMQ_OK;
}

// C = alpha * A B^T with A [M, K] and B [N, K] both stored K-major
omq_status gemm_kk(cudaStream_t st, int64_t M, int64_t N, int64_t K, const bf16* A, int64_t lda, const bf16* B,
                   int64_t ldb, float* Cf, bf16* Cb, int64_t ldc, const float* bias, const float* R, int32_t* status) {
  GemmOperand a{A, lda, 0, 1}, b{B, ldb, 0, 1};
  GemmEpilogue ep{Cf, Cb, ldc, 0, 1.f, bias, R, ldc, 0.f};
  return gemm_launch(st, M, N, K, 1, a, b, ep, 0, status);
}

// dX = dY W  with dY [T, Cout] and W [Cout, Cin]: B[n = i, k = o] = W[o, i] is MN-major
omq_status gemm_dx(cudaStream_t st, int64_t T, int64_t Cout, int64_t Cin, const bf16* dY, const bf16* W, float* dX,
                   int32_t* status) {
  GemmOperand a{dY, Cout, 0, 1}, b{W, Cin, 0, 0};
  GemmEpilogue ep{dX, nullptr, Cin, 0, 1.f, nullptr, nullptr, 0, 0.f};
  return gemm_launch(st, T, Cin, Cout, 1, a, b, ep, 0, status);
}

// dW = dY^T X with dY [T, Cout], X [T, Cin]: both operands MN-major, K = T
omq_status gemm_dw(cudaStream_t st, int64_t T, int64_t Cout, int64_t Cin, const bf16* dY, const bf16* X, float* dW,
                   int32_t* status) {
  GemmOperand a{dY, Cout, 0, 0}, b{X, Cin, 0, 0};
  GemmEpilogue ep{dW, nullptr, Cin, 0, 1.f, nullptr, nullptr, 0, 0.f};
  return gemm_launch(st, Cout, Cin, T, 1, a, b, ep, 0, status);
}

// The q|k|v weight operand prepared inside the GEMM (omq_qcfg.wprep = 1): the raw weight with the
// quantizer state of its LWC forward and, with LET, the column scale s1 and the row scale of the
// v rows (1 / s_o, Eq. 5's [v, out] pair)
GemmQuantB qkv_operand(const QState4& q, const omq_qcfg& cfg, int64_t d, const float* s, const float* r) {
  GemmQuantB qb{};
  qb.h = q.h; qb.z = q.z; qb.r = r; qb.s = s;
  qb.group = cfg.group == 0 ? (int)d : cfg.group;
  qb.Q = (float)((1 << cfg.wbits) - 1);
  return qb;
}

LwcFwdArgs lwc_args(const bf16* W, int64_t Cout, int64_t Cin, const omq_qcfg& cfg, const float* s, const float* r,
                    const float* gl, const float* bl, bf16* Wq, const QState4& q, const float* bias_delta,
                    const float* bias_shift, float* Bt) {
  LwcFwdArgs a{};
  a.W = W; a.Cout = Cout; a.Cin = Cin; a.group = cfg.group == 0 ? (int)Cin : cfg.group;
  a.s = s; a.r = r; a.gl = gl; a.bl = bl; a.lwc = 1; a.Wq = Wq; a.codes = nullptr;
  a.h = q.h; a.z = q.z; a.imax = q.imax; a.imin = q.imin;
  a.bias_delta = bias_delta; a.bias_shift = bias_shift; a.Bt = Bt;
  a.ga_out = q.ga; a.gb_out = q.gb; a.M_out = q.M; a.m_out = q.m;
  a.wbits = cfg.wbits; a.eps = cfg.h_eps; a.status = cfg.dev_status;
  return a;
}

omq_status lwc_bwd_full(cudaStream_t st, const bf16* W, int64_t Cout, int64_t Cin, const omq_qcfg& cfg,
                        const float* s, const float* r, const float* gl, const float* bl, const QState4& q,
                        const float* dW, float* dgl, float* dbl, float* dr, const float* dBt, float* ds,
                        float* ddelta, int accumulate_sd, float* part) {
  LwcBwdArgs a{};
  a.W = W; a.Cout = Cout; a.Cin = Cin; a.group = cfg.group == 0 ? (int)Cin : cfg.group;
  a.s = s; a.r = r; a.gl = gl; a.bl = bl; a.lwc = 1; a.ga = q.ga; a.gb = q.gb; a.Mv = q.M; a.mv = q.m;
  a.h = q.h; a.z = q.z; a.imax = q.imax; a.imin = q.imin;
  a.dWq = dW; a.ld_dwq = Cin; a.dgl = dgl; a.dbl = dbl; a.dWt = nullptr; a.dr = dr; a.dBt = dBt;
  a.ds = ds; a.ddelta = ddelta;
  a.wbits = cfg.wbits; a.eps = cfg.h_eps;
  // dgamma/dbeta follow cfg.accumulate; the LET sums follow the caller; dr is scratch
  a.accumulate = cfg.accumulate; a.accumulate_sd = accumulate_sd; a.accumulate_dr = 0;
  return lwc_bwd_launch(st, a, part);
}

// dW_hat = dY^T X_hat and the straight-through LWC backward of W (Eq. 2, Eq. 3): the per-element
// part runs in the GEMM epilogue (dW_hat stays in tensor memory), the reductions finish after it.
// Falls back to the stored dW_hat + separate LWC backward for layouts the epilogue does not take.
omq_status lwc_bwd_dw(cudaStream_t st, int64_t T, const bf16* dY, const bf16* Xh, const bf16* W, int64_t Cout,
                      int64_t Cin, const omq_qcfg& cfg, const float* s, const float* r, const float* gl,
                      const float* bl, const QState4& q, float* dgl, float* dbl, float* dr, const float* dBt, float* ds,
                      float* ddelta, int accumulate_sd, float* part, float* dW_fallback, int32_t* status) {
  const int group = cfg.group == 0 ? (int)Cin : cfg.group;
  const bool let_terms = s || r || dBt || ds || ddelta || dr;
  if (!lwc_fused_ok(Cin, group, let_terms)) {
    OMQ_TRY(gemm_dw(st, T, Cout, Cin, dY, Xh, dW_fallback, status));
    return lwc_bwd_full(st, W, Cout, Cin, cfg, s, r, gl, bl, q, dW_fallback, dgl, dbl, dr, dBt, ds, ddelta,
                        accumulate_sd, part);
  }
  const int64_t P = (Cout + 31) / 32;
  const int ntn = 2 * (int)((Cin + gemm_n_tile(Cin) - 1) / gemm_n_tile(Cin));
  GemmLwcEpi lw{};
  lw.W = W; lw.s = s; lw.r = r; lw.h = q.h; lw.z = q.z; lw.ga = q.ga; lw.gb = q.gb; lw.Mv = q.M; lw.mv = q.m;
  lw.dBt = dBt;
  lw.part_s = ds ? part : nullptr;
  lw.part_d = (ddelta && dBt) ? part + P * Cin : nullptr;
  lw.rowpart = part + 2 * P * Cin;
  lw.want_dr = dr != nullptr;
  lw.dgl = dgl; lw.dbl = dbl;
  lw.group = group; lw.accumulate = cfg.accumulate; lw.ntn = ntn;
  lw.Q = (float)((1 << cfg.wbits) - 1); lw.eps = cfg.h_eps;
  GemmOperand a{dY, Cout, 0, 0}, b{Xh, Cin, 0, 0};
  OMQ_TRY(gemm_launch_lwc(st, Cout, Cin, T, a, b, lw, status));
  LwcBwdArgs la{};
  la.W = W; la.Cout = Cout; la.Cin = Cin; la.group = group;
  la.s = s; la.r = r; la.gl = gl; la.bl = bl; la.lwc = 1; la.ga = q.ga; la.gb = q.gb; la.Mv = q.M; la.mv = q.m;
  la.h = q.h; la.z = q.z; la.imax = q.imax; la.imin = q.imin;
  la.dgl = dgl; la.dbl = dbl; la.dWt = nullptr; la.dr = dr; la.dBt = dBt; la.ds = ds; la.ddelta = ddelta;
  la.wbits = cfg.wbits; la.eps = cfg.h_eps;
  la.accumulate = cfg.accumulate; la.accumulate_sd = accumulate_sd; la.accumulate_dr = 0;
  float* route = lw.rowpart + ((3 * Cout * ntn + 3) & ~int64_t(3));   // [Cout, 4], 16-byte aligned
  return lwc_bwd_fused_finish(st, la, lw.rowpart, ntn, lw.part_s, lw.part_d, P, route);
}

// Auxiliary stream of a device: work off the step's critical chain (the LWC forward of the later
// weights, the weight-gradient products with their LWC backward) runs there, concurrently with
// the caller's stream, and joins it through events.  One per device, created on first use; block
// calls of one device that overlap on the GPU share it and must not be issued concurrently.
struct Aux {
  cudaStream_t s = nullptr;
  cudaEvent_t ev[12] = {};
  bool ready = false;
};
std::mutex g_aux_mu;
Aux g_aux[64];

omq_status aux_get(Aux** out) {
  int dev = 0;
  OMQ_REQUIRE(cudaGetDevice(&dev) == cudaSuccess && dev >= 0 && dev < 64, OMQ_ERR_CUDA);
  std::lock_guard<std::mutex> lk(g_aux_mu);
  Aux& a = g_aux[dev];
  if (!a.ready) {
    OMQ_REQUIRE(cudaStreamCreateWithFlags(&a.s, cudaStreamNonBlocking) == cudaSuccess, OMQ_ERR_CUDA);
    for (auto& e : a.ev) OMQ_REQUIRE(cudaEventCreateWithFlags(&e, cudaEventDisableTiming) == cudaSuccess, OMQ_ERR_CUDA);
    a.ready = true;
  }
  *out = &a;
  return OMQ_OK;
}

// `to` waits for everything enqueued on `from` so far
omq_status join(cudaStream_t from, cudaStream_t to, cudaEvent_t e) {
  OMQ_REQUIRE(cudaEventRecord(e, from) == cudaSuccess, OMQ_ERR_CUDA);
  OMQ_REQUIRE(cudaStreamWaitEvent(to, e, 0) == cudaSuccess, OMQ_ERR_CUDA);
  return OMQ_OK;
}

struct Ctx {
  cudaStream_t st;
  Aux* aux;
  omq_block_shape s;
  omq_qcfg cfg;
  const omq_block_weights* w;
  const omq_block_params* th;
  BlockWS ws;
  int64_t T, d, hd, H, Hkv, rep, f, dq, dkv, nqkv;
  bool let, wq, aq, wprep;
};

// da = dY_qkv W_hat_qkv (the gradient reaching the quantized attention input), from W_hat in HBM or
// from the raw weight prepared tile by tile (omq_qcfg.wprep)
omq_status qkv_dx(Ctx& c, int32_t* status) {
  BlockWS& w = c.ws;
  if (!c.wprep) return gemm_dx(c.st, c.T, c.nqkv, c.d, w.dYqkv_b, w.Wqkv_h, w.da, status);
  GemmOperand a{w.dYqkv_b, c.nqkv, 0, 1}, b{c.w->wqkv, c.d, 0, 0};
  GemmEpilogue ep{w.da, nullptr, c.d, 0, 1.f, nullptr, nullptr, 0, 0.f};
  return gemm_launch_qb(c.st, c.T, c.d, c.nqkv, a, b, ep,
                        qkv_operand(w.sq_qkv, c.cfg, c.d, c.let ? c.th->s1 : nullptr, c.let ? w.r_qkv : nullptr),
                        status);
}

omq_status block_fwd(Ctx& c, const float* x, float* y) {
  cudaStream_t st = c.st;
  BlockWS& w = c.ws;
  const omq_qcfg& cfg = c.cfg;
  const omq_block_params* th = c.th;
  // s_o, delta_o, s_a per query channel (broadcast over the query heads of a kv head)
  const float* so_e = c.rep > 1 ? c.ws.so_exp : th->so;
  const float* do_e = c.rep > 1 ? c.ws.do_exp : th->do_;
  const float* sa_e = c.rep > 1 ? c.ws.sa_exp : th->sa;
  int32_t* status = cfg.dev_status;
  const bf16* Wqkv = (const bf16*)c.w->wqkv;
  const bf16* Wo = (const bf16*)c.w->wo;
  const bf16* Wgu = (const bf16*)c.w->wgu;
  const bf16* Wd = (const bf16*)c.w->wd;

  OMQ_TRY(rope_table(st, (int)c.T, (int)c.hd, c.s.rope_theta, w.cs));
  if (c.let) {
    OMQ_TRY(qkv_row_vectors(st, (int)c.dq, (int)c.dkv, th->so, th->do_, w.r_qkv, w.shift_qkv));
    if (c.rep > 1) {                            // one kv head per query head: the vectors serve as they are
      OMQ_TRY(gqa_expand(st, th->so, w.so_exp, (int)c.Hkv, (int)c.rep, (int)c.hd, 0));
      OMQ_TRY(gqa_expand(st, th->do_, w.do_exp, (int)c.Hkv, (int)c.rep, (int)c.hd, 0));
      OMQ_TRY(gqa_expand(st, th->sa, w.sa_exp, (int)c.Hkv, (int)c.rep, (int)c.hd, 0));
    }
  }
  // ---- LET (Eq. 3) + LWC (Eq. 2) on every weight: q|k|v here, the others on the auxiliary stream
  // while the attention half runs -------------------------------------------------------------------
  cudaStream_t ax = c.aux->s;
  cudaEvent_t* ev = c.aux->ev;
  OMQ_TRY(join(st, ax, ev[0]));
  OMQ_TRY(lwc_fwd_launch(st, lwc_args(Wqkv, c.nqkv, c.d, cfg, c.let ? th->s1 : nullptr, c.let ? w.r_qkv : nullptr,
                                      th->gamma_qkv, th->beta_qkv, c.wprep ? nullptr : w.Wqkv_h, w.sq_qkv,
                                      c.let ? th->d1 : nullptr,
                                      c.let ? w.shift_qkv : nullptr, c.let ? w.B_qkv : nullptr)));
  OMQ_TRY(lwc_fwd_launch(ax, lwc_args(Wo, c.d, c.dq, cfg, c.let ? so_e : nullptr, nullptr, th->gamma_o, th->beta_o,
                                      w.Wo_h, w.sq_o, c.let ? do_e : nullptr, nullptr, c.let ? w.B_o : nullptr)));
  OMQ_REQUIRE(cudaEventRecord(ev[1], ax) == cudaSuccess, OMQ_ERR_CUDA);
  OMQ_TRY(lwc_fwd_launch(ax, lwc_args(Wgu, 2 * c.f, c.d, cfg, c.let ? th->s2 : nullptr, nullptr, th->gamma_gu,
                                      th->beta_gu, w.Wgu_h, w.sq_gu, c.let ? th->d2 : nullptr, nullptr,
                                      c.let ? w.B_gu : nullptr)));
  OMQ_REQUIRE(cudaEventRecord(ev[2], ax) == cudaSuccess, OMQ_ERR_CUDA);
  OMQ_TRY(lwc_fwd_launch(ax, lwc_args(Wd, c.d, c.f, cfg, nullptr, nullptr, th->gamma_d, th->beta_d, w.Wd_h, w.sq_d,
                                      nullptr, nullptr, nullptr)));
  OMQ_REQUIRE(cudaEventRecord(ev[3], ax) == cudaSuccess, OMQ_ERR_CUDA);

  // ---- attention half ---------------------------------------------------------------------------
  ActFwdArgs af{};
  af.producer = AP_RMS_LET; af.X = x; af.ldx = c.d; af.s = c.let ? th->s1 : nullptr; af.delta = c.let ? th->d1 : nullptr;
  af.rms_eps = c.s.rms_eps; af.rstd = w.rstd1; af.T = c.T; af.C = c.d; af.Xq = w.a_h; af.ldq = c.d;
  af.h = w.sa.h; af.z = w.sa.z; af.imax = w.sa.imax; af.imin = w.sa.imin; af.abits = cfg.abits; af.eps = cfg.h_eps;
  af.status = status;
  OMQ_TRY(act_fwd_launch(st, af));
  if (c.wprep) {
    GemmOperand a{w.a_h, c.d, 0, 1}, b{Wqkv, c.d, 0, 1};
    GemmEpilogue ep{w.Yqkv, nullptr, c.nqkv, 0, 1.f, c.let ? w.B_qkv : nullptr, nullptr, c.nqkv, 0.f};
    OMQ_TRY(gemm_launch_qb(st, c.T, c.nqkv, c.d, a, b, ep,
                           qkv_operand(w.sq_qkv, cfg, c.d, c.let ? th->s1 : nullptr, c.let ? w.r_qkv : nullptr), status));
  } else {
    OMQ_TRY(gemm_kk(st, c.T, c.nqkv, c.d, w.a_h, c.d, w.Wqkv_h, c.d, w.Yqkv, nullptr, c.nqkv,
                    c.let ? w.B_qkv : nullptr, nullptr, status));
  }
  QkvArgs qa{};
  qa.T = (int)c.T; qa.H = (int)c.H; qa.Hkv = (int)c.Hkv; qa.hd = (int)c.hd; qa.Y = w.Yqkv; qa.ldy = c.nqkv; qa.cs = w.cs;
  qa.sa_exp = c.let ? sa_e : nullptr; qa.sa = c.let ? th->sa : nullptr;
  qa.Qh = w.Qh; qa.Kh = w.Kh; qa.Vh = w.Vh;
  qa.h = w.sqkv.h; qa.z = w.sqkv.z; qa.imax = w.sqkv.imax; qa.imin = w.sqkv.imin; qa.abits = cfg.abits; qa.eps = cfg.h_eps;
  OMQ_TRY(qkv_fwd_launch(st, qa));
  FlashArgs fa{};
  fa.T = (int)c.T; fa.H = (int)c.H; fa.Hkv = (int)c.Hkv; fa.hd = (int)c.hd;
  fa.Q = w.Qh; fa.K = w.Kh; fa.V = w.Vh; fa.ldq = c.dq; fa.ldkv = c.dkv;
  fa.O = w.O; fa.ldo = c.dq; fa.lse = w.lse; fa.status = status;
  fa.pbits = cfg.pbits; fa.eps = cfg.h_eps; fa.pqr = w.pqr; fa.ldl = (int)((c.T + 3) / 4 * 4);
  OMQ_TRY(flash_fwd_launch(st, fa));
  ActFwdArgs ao{};
  ao.producer = AP_PLAIN; ao.X = w.O; ao.ldx = c.dq; ao.T = c.T; ao.C = c.dq; ao.Xq = w.O_h; ao.ldq = c.dq;
  ao.h = w.so.h; ao.z = w.so.z; ao.imax = w.so.imax; ao.imin = w.so.imin; ao.abits = cfg.abits; ao.eps = cfg.h_eps;
  ao.status = status;
  OMQ_TRY(act_fwd_launch(st, ao));
  OMQ_REQUIRE(cudaStreamWaitEvent(st, ev[1], 0) == cudaSuccess, OMQ_ERR_CUDA);      // W_hat of o_proj
  OMQ_TRY(gemm_kk(st, c.T, c.d, c.dq, w.O_h, c.dq, w.Wo_h, c.dq, w.h1, nullptr, c.d, c.let ? w.B_o : nullptr, x, status));

  // ---- FFN half ---------------------------------------------------------------------------------
  ActFwdArgs ab = af;
  ab.X = w.h1; ab.s = c.let ? th->s2 : nullptr; ab.delta = c.let ? th->d2 : nullptr; ab.rstd = w.rstd2; ab.Xq = w.b_h;
  ab.h = w.sb.h; ab.z = w.sb.z; ab.imax = w.sb.imax; ab.imin = w.sb.imin;
  OMQ_TRY(act_fwd_launch(st, ab));
  OMQ_REQUIRE(cudaStreamWaitEvent(st, ev[2], 0) == cudaSuccess, OMQ_ERR_CUDA);      // W_hat of gate|up
  OMQ_TRY(gemm_kk(st, c.T, 2 * c.f, c.d, w.b_h, c.d, w.Wgu_h, c.d, w.Ygu, nullptr, 2 * c.f, c.let ? w.B_gu : nullptr,
                  nullptr, status));
  ActFwdArgs am{};
  am.producer = AP_SWIGLU; am.X = w.Ygu; am.ldx = 2 * c.f; am.U = w.Ygu + c.f; am.ldu = 2 * c.f; am.T = c.T; am.C = c.f;
  am.Xq = w.m_h; am.ldq = c.f; am.h = w.sm.h; am.z = w.sm.z; am.imax = w.sm.imax; am.imin = w.sm.imin;
  am.abits = cfg.abits; am.eps = cfg.h_eps; am.status = status;
  OMQ_TRY(act_fwd_launch(st, am));
  OMQ_REQUIRE(cudaStreamWaitEvent(st, ev[3], 0) == cudaSuccess, OMQ_ERR_CUDA);      // W_hat of down (joins)
  OMQ_TRY(gemm_kk(st, c.T, c.d, c.f, w.m_h, c.f, w.Wd_h, c.f, y, nullptr, c.d, nullptr, w.h1, status));
  return OMQ_OK;
}

omq_status block_bwd(Ctx& c, const float* x, const float* y, const float* y_fp, float* loss, const omq_block_params* g) {
  cudaStream_t st = c.st;
  BlockWS& w = c.ws;
  const omq_qcfg& cfg = c.cfg;
  const omq_block_params* th = c.th;
  // s_o, delta_o, s_a per query channel (broadcast over the query heads of a kv head)
  const float* so_e = c.rep > 1 ? c.ws.so_exp : th->so;
  const float* sa_e = c.rep > 1 ? c.ws.sa_exp : th->sa;
  int32_t* status = cfg.dev_status;
  const bf16* Wqkv = (const bf16*)c.w->wqkv;
  const bf16* Wo = (const bf16*)c.w->wo;
  const bf16* Wgu = (const bf16*)c.w->wgu;
  const bf16* Wd = (const bf16*)c.w->wd;
  const int acc = cfg.accumulate;

  // The weight-gradient products with their LWC backward run on the auxiliary stream (scratch
  // part_aux, fallback dW), each started once its inputs exist; the caller's stream waits for
  // them only where their outputs are accumulated further, and for all of them at the end.
  cudaStream_t ax = c.aux->s;
  cudaEvent_t* ev = c.aux->ev;

  // ---- loss (Eq. 1) ------------------------------------------------------------------------------
  OMQ_TRY(loss_launch(st, c.T * c.d, y, y_fp, loss, w.dy, w.dy_b, w.loss_part));

  // ---- down_proj ----------------------------------------------------------------------------------
  OMQ_TRY(join(st, ax, ev[4]));
  OMQ_TRY(lwc_bwd_dw(ax, c.T, w.dy_b, w.m_h, Wd, c.d, c.f, cfg, nullptr, nullptr, th->gamma_d, th->beta_d, w.sq_d,
                     g->gamma_d, g->beta_d, nullptr, nullptr, nullptr, nullptr, 0, w.part_aux, w.dW, status));
  OMQ_TRY(gemm_dx(st, c.T, c.d, c.f, w.dy_b, w.Wd_h, w.dm, status));
  ActBwdArgs bm{};
  bm.producer = AP_SWIGLU; bm.X = w.Ygu; bm.ldx = 2 * c.f; bm.U = w.Ygu + c.f; bm.ldu = 2 * c.f; bm.T = c.T; bm.C = c.f;
  bm.h = w.sm.h; bm.z = w.sm.z; bm.imax = w.sm.imax; bm.imin = w.sm.imin; bm.dXq = w.dm; bm.lddq = c.f;
  bm.dX = nullptr; bm.lddx = 2 * c.f; bm.dXb = w.dYgu_b; bm.lddxb = 2 * c.f; bm.dU = nullptr; bm.dUb = w.dYgu_b + c.f;
  bm.rows_per_cta = kRowsSwiglu; bm.abits = cfg.abits; bm.eps = cfg.h_eps;
  OMQ_TRY(act_bwd_launch(st, bm));

  // ---- gate / up ----------------------------------------------------------------------------------
  // LET bias gradient dB~ = sum_t dY: the column sums of the bf16 gradient, the operand every product of
  // this backward takes (R13); only the LWC backward of the weight-gradient product reads it, so it is
  // formed on the auxiliary stream just before that product
  OMQ_TRY(join(st, ax, ev[5]));
  if (c.let) OMQ_TRY(colsum_rows_bf16(ax, w.dYgu_b, c.T, 2 * c.f, 2 * c.f, w.part_aux, w.dB_gu, 1.f, 0));
  OMQ_TRY(lwc_bwd_dw(ax, c.T, w.dYgu_b, w.b_h, Wgu, 2 * c.f, c.d, cfg, c.let ? th->s2 : nullptr, nullptr,
                     th->gamma_gu, th->beta_gu, w.sq_gu, g->gamma_gu, g->beta_gu, nullptr,
                     c.let ? w.dB_gu : nullptr, c.let ? g->s2 : nullptr, c.let ? g->d2 : nullptr, acc, w.part_aux,
                     w.dW, status));
  OMQ_TRY(gemm_dx(st, c.T, 2 * c.f, c.d, w.dYgu_b, w.Wgu_h, w.db, status));
  ActBwdArgs bb{};
  bb.producer = AP_RMS_LET; bb.X = w.h1; bb.ldx = c.d; bb.s = c.let ? th->s2 : nullptr; bb.delta = c.let ? th->d2 : nullptr;
  bb.rstd = w.rstd2; bb.T = c.T; bb.C = c.d; bb.h = w.sb.h; bb.z = w.sb.z; bb.imax = w.sb.imax; bb.imin = w.sb.imin;
  bb.dXq = w.db; bb.lddq = c.d; bb.dX = nullptr; bb.lddx = c.d; bb.dXb = w.dh1_b; bb.lddxb = c.d; bb.resid = w.dy;
  bb.part_s = c.let ? w.part2 : nullptr; bb.part_d = c.let ? w.part2 + rms_parts(c.T) * c.d : nullptr;
  bb.rows_per_cta = kRowsRms; bb.abits = cfg.abits; bb.eps = cfg.h_eps;
  OMQ_TRY(act_bwd_launch(st, bb));

  // ---- o_proj -------------------------------------------------------------------------------------
  OMQ_TRY(join(st, ax, ev[7]));
  if (c.let) {
    // ds2, dd2: the RMSNorm backward's part added after the LWC part (earlier on this stream), then dB~_o
    OMQ_TRY(omq_colsum_partials2(ax, ColsumJob{bb.part_s, rms_parts(c.T), c.d, g->s2, 1.f, 1},
                                 ColsumJob{bb.part_d, rms_parts(c.T), c.d, g->d2, 1.f, 1}));
    OMQ_TRY(colsum_rows_bf16(ax, w.dh1_b, c.T, c.d, c.d, w.part_aux, w.dB_o, 1.f, 0));
  }
  // ds_o, ddelta_o per query channel; with one query head per kv head straight into the gradients
  const bool fold_o = c.rep > 1;
  OMQ_TRY(lwc_bwd_dw(ax, c.T, w.dh1_b, w.O_h, Wo, c.d, c.dq, cfg, c.let ? so_e : nullptr, nullptr, th->gamma_o,
                     th->beta_o, w.sq_o, g->gamma_o, g->beta_o, nullptr, c.let ? w.dB_o : nullptr,
                     c.let ? (fold_o ? w.vtmp0 : g->so) : nullptr, c.let ? (fold_o ? w.vtmp1 : g->do_) : nullptr,
                     fold_o ? 0 : acc, w.part_aux, w.dW, status));
  OMQ_REQUIRE(cudaEventRecord(ev[8], ax) == cudaSuccess, OMQ_ERR_CUDA);
  OMQ_TRY(gemm_dx(st, c.T, c.d, c.dq, w.dh1_b, w.Wo_h, w.dOh, status));
  ActBwdArgs bo{};
  bo.producer = AP_PLAIN; bo.X = w.O; bo.ldx = c.dq; bo.T = c.T; bo.C = c.dq; bo.h = w.so.h; bo.z = w.so.z;
  bo.imax = w.so.imax; bo.imin = w.so.imin; bo.dXq = w.dOh; bo.lddq = c.dq; bo.dX = nullptr; bo.lddx = c.dq;
  bo.dXb = w.dO_b; bo.lddxb = c.dq; bo.rows_per_cta = kRowsPlain; bo.abits = cfg.abits; bo.eps = cfg.h_eps;
  const bool d_fused = !flash_pq_on(cfg.pbits);   // rowsum(dO * O) of the attention backward, formed here
  if (d_fused) { bo.rowdot = w.Drow; bo.ldrow = (c.T + 3) / 4 * 4; }
  OMQ_TRY(act_bwd_launch(st, bo));

  // ---- attention: dQ, dK, dV from the saved log-sum-exp (scores recomputed, never stored) --------
  FlashArgs fa{};
  fa.T = (int)c.T; fa.H = (int)c.H; fa.Hkv = (int)c.Hkv; fa.hd = (int)c.hd;
  fa.Q = w.Qh; fa.K = w.Kh; fa.V = w.Vh; fa.ldq = c.dq; fa.ldkv = c.dkv;
  fa.O = w.O; fa.ldo = c.dq; fa.lse = w.lse; fa.dO = w.dO_b; fa.lddo = c.dq; fa.D = w.Drow; fa.d_ready = d_fused;
  fa.dQ = w.dQKV; fa.ldg = c.nqkv; fa.dK = w.dQKV + c.dq; fa.dV = w.dQKV + c.dq + c.dkv; fa.ldgkv = c.nqkv;
  fa.status = status;
  fa.pbits = cfg.pbits; fa.eps = cfg.h_eps; fa.pqr = w.pqr; fa.pqb = w.pqb; fa.ldl = (int)((c.T + 3) / 4 * 4);
  OMQ_TRY(flash_bwd_launch(st, fa));
  QkvArgs qa{};
  qa.T = (int)c.T; qa.H = (int)c.H; qa.Hkv = (int)c.Hkv; qa.hd = (int)c.hd; qa.Y = w.Yqkv; qa.ldy = c.nqkv; qa.cs = w.cs;
  qa.sa_exp = c.let ? sa_e : nullptr; qa.sa = c.let ? th->sa : nullptr;
  qa.h = w.sqkv.h; qa.z = w.sqkv.z; qa.imax = w.sqkv.imax; qa.imin = w.sqkv.imin; qa.abits = cfg.abits; qa.eps = cfg.h_eps;
  qa.dQKV = w.dQKV; qa.ldd = c.nqkv; qa.dY = nullptr; qa.dYb = w.dYqkv_b;
  const int64_t nsq = qkv_bwd_nslab((int)c.T);
  qa.part_q = c.let ? w.part : nullptr;
  qa.part_k = c.let ? w.part + nsq * c.dq : nullptr;
  OMQ_TRY(qkv_bwd_launch(st, qa, nullptr));
  if (c.let) {
    if (c.rep == 1) {       // q and k partials are one contiguous [2 nslab, d_kv] array over the same channels
      OMQ_TRY(omq_colsum_partials(st, qa.part_q, 2 * nsq, c.dq, g->sa, 1.f, acc));
    } else {
      OMQ_TRY(omq_colsum_partials2(st, ColsumJob{qa.part_q, nsq, c.dq, w.vtmp2, 1.f, 0},
                                   ColsumJob{qa.part_k, nsq, c.dkv, g->sa, 1.f, acc}));
      OMQ_TRY(gqa_fold(st, w.vtmp2, g->sa, (int)c.Hkv, (int)c.rep, (int)c.hd, 1));
    }
    // [v, out] pair: o_proj column-scale part (folded over the query heads), then v rows
    OMQ_REQUIRE(cudaStreamWaitEvent(st, ev[8], 0) == cudaSuccess, OMQ_ERR_CUDA);   // o_proj LWC backward
    if (fold_o) {
      OMQ_TRY(gqa_fold(st, w.vtmp0, g->so, (int)c.Hkv, (int)c.rep, (int)c.hd, acc));
      OMQ_TRY(gqa_fold(st, w.vtmp1, g->do_, (int)c.Hkv, (int)c.rep, (int)c.hd, acc));
    }
  }

  // ---- q / k / v projections ---------------------------------------------------------------------------
  OMQ_TRY(join(st, ax, ev[9]));
  if (c.let) OMQ_TRY(colsum_rows_bf16(ax, w.dYqkv_b, c.T, c.nqkv, c.nqkv, w.part_aux, w.dB_qkv, 1.f, 0));
  OMQ_TRY(lwc_bwd_dw(ax, c.T, w.dYqkv_b, w.a_h, Wqkv, c.nqkv, c.d, cfg, c.let ? th->s1 : nullptr,
                     c.let ? w.r_qkv : nullptr, th->gamma_qkv, th->beta_qkv, w.sq_qkv, g->gamma_qkv, g->beta_qkv,
                     c.let ? w.dr_qkv : nullptr, c.let ? w.dB_qkv : nullptr, c.let ? g->s1 : nullptr,
                     c.let ? g->d1 : nullptr, acc, w.part_aux, w.dW, status));
  OMQ_REQUIRE(cudaEventRecord(ev[10], ax) == cudaSuccess, OMQ_ERR_CUDA);
  if (c.let) {
    const int64_t off = c.dq + c.dkv;
    OMQ_TRY(qkv_dx(c, status));
    OMQ_REQUIRE(cudaStreamWaitEvent(st, ev[10], 0) == cudaSuccess, OMQ_ERR_CUDA);  // dr of the v rows, ds1, dd1
    OMQ_TRY(let_vo_finalize(st, (int)c.dkv, th->so, w.dr_qkv + off, w.dB_qkv + off, w.B_qkv + off, g->so, g->do_, 1));
    ActBwdArgs ba{};
    ba.producer = AP_RMS_LET; ba.X = x; ba.ldx = c.d; ba.s = th->s1; ba.delta = th->d1; ba.rstd = w.rstd1; ba.T = c.T;
    ba.C = c.d; ba.h = w.sa.h; ba.z = w.sa.z; ba.imax = w.sa.imax; ba.imin = w.sa.imin; ba.dXq = w.da; ba.lddq = c.d;
    ba.dX = nullptr; ba.dXb = nullptr; ba.part_s = w.part; ba.part_d = w.part + rms_parts(c.T) * c.d;
    ba.rows_per_cta = kRowsRms; ba.abits = cfg.abits; ba.eps = cfg.h_eps;
    OMQ_TRY(act_bwd_launch(st, ba));
    OMQ_TRY(omq_colsum_partials2(st, ColsumJob{ba.part_s, rms_parts(c.T), c.d, g->s1, 1.f, 1},
                                 ColsumJob{ba.part_d, rms_parts(c.T), c.d, g->d1, 1.f, 1}));
  }
  OMQ_REQUIRE(cudaStreamWaitEvent(st, ev[10], 0) == cudaSuccess, OMQ_ERR_CUDA);    // every auxiliary launch
  return OMQ_OK;
}

omq_status make_ctx(Ctx& c, omq_stream_t stream, const omq_block_shape* shape, const omq_block_weights* w,
                    const omq_block_params* theta, void* workspace, size_t ws_bytes, const omq_qcfg* cfg, bool bwd) {
  OMQ_TRY(check_block(shape, cfg));
  OMQ_REQUIRE(w && w->wqkv && w->wo && w->wgu && w->wd && theta, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(omq_aligned16(w->wqkv) && omq_aligned16(w->wo) && omq_aligned16(w->wgu) && omq_aligned16(w->wd),
              OMQ_ERR_ALIGN);
  if (cfg->wbits < 16)
    OMQ_REQUIRE(theta->gamma_qkv && theta->beta_qkv && theta->gamma_o && theta->beta_o && theta->gamma_gu &&
                    theta->beta_gu && theta->gamma_d && theta->beta_d,
                OMQ_ERR_INVALID_ARG);
  if (cfg->let)
    OMQ_REQUIRE(theta->s1 && theta->d1 && theta->so && theta->do_ && theta->sa && theta->s2 && theta->d2,
                OMQ_ERR_INVALID_ARG);
  Carve dry{nullptr, 0};
  BlockWS tmp;
  carve_block(dry, *shape, *cfg, tmp, bwd);
  OMQ_REQUIRE(workspace && ws_bytes >= dry.off, OMQ_ERR_WORKSPACE);
  OMQ_REQUIRE(omq_aligned16(workspace), OMQ_ERR_ALIGN);
  c.st = (cudaStream_t)stream;
  OMQ_TRY(aux_get(&c.aux));
  c.s = *shape;
  c.cfg = *cfg;
  c.w = w;
  c.th = theta;
  Carve real{(uint8_t*)workspace, 0};
  carve_block(real, *shape, *cfg, c.ws, bwd);
  c.T = shape->T; c.d = shape->d; c.hd = shape->head_dim; c.H = shape->n_heads; c.Hkv = shape->n_kv;
  c.rep = c.H / c.Hkv; c.f = shape->ffn; c.dq = c.H * c.hd; c.dkv = c.Hkv * c.hd; c.nqkv = c.dq + 2 * c.dkv;
  c.let = cfg->let != 0; c.wq = cfg->wbits < 16; c.aq = cfg->abits < 16; c.wprep = c.wq && cfg->wprep == 1;
  return OMQ_OK;
}

}  // namespace

extern "C" {

size_t omq_block_workspace_size(const omq_block_shape* shape, const omq_qcfg* cfg) {
  if (check_block(shape, cfg) != OMQ_OK) return 0;
  Carve dry{nullptr, 0};
  BlockWS tmp;
  carve_block(dry, *shape, *cfg, tmp, true);
  return dry.off + 256;
}

omq_status omq_block_saved_layout(const omq_block_shape* shape, const omq_qcfg* cfg, omq_block_saved* out) {
  OMQ_TRY(check_block(shape, cfg));
  OMQ_REQUIRE(out, OMQ_ERR_INVALID_ARG);
  // carve against a stand-in base address (never dereferenced) and report offsets from it
  uint8_t* const base = reinterpret_cast<uint8_t*>(uintptr_t(1) << 20);
  Carve c{base, 0};
  BlockWS w;
  carve_block(c, *shape, *cfg, w, true);
  auto off = [&](const void* p) -> int64_t { return p ? (int64_t)((const uint8_t*)p - base) : -1; };
  out->a_hat = off(w.a_h); out->a_h = off(w.sa.h); out->a_z = off(w.sa.z);
  out->y_qkv = off(w.Yqkv); out->qkv_h = off(w.sqkv.h); out->qkv_z = off(w.sqkv.z);
  out->q_hat = off(w.Qh); out->k_hat = off(w.Kh); out->v_hat = off(w.Vh);
  out->o = off(w.O); out->o_hat = off(w.O_h); out->o_h = off(w.so.h); out->o_z = off(w.so.z);
  out->h1 = off(w.h1); out->b_hat = off(w.b_h); out->b_h = off(w.sb.h); out->b_z = off(w.sb.z);
  out->y_gu = off(w.Ygu); out->m_hat = off(w.m_h); out->m_h = off(w.sm.h); out->m_z = off(w.sm.z);
  const bf16* wh[4] = {w.Wqkv_h, w.Wo_h, w.Wgu_h, w.Wd_h};
  const QState4* sq[4] = {&w.sq_qkv, &w.sq_o, &w.sq_gu, &w.sq_d};
  for (int i = 0; i < 4; ++i) {
    out->w_hat[i] = off(wh[i]); out->w_h[i] = off(sq[i]->h); out->w_z[i] = off(sq[i]->z);
  }
  out->dy = off(w.dy); out->dy_gu = off(w.dYgu_b); out->dh1 = off(w.dh1_b); out->do_bf16 = off(w.dO_b);
  out->dy_qkv = off(w.dYqkv_b);
  return OMQ_OK;
}

omq_status omq_block_forward(omq_stream_t stream, const omq_block_shape* shape, const omq_block_weights* w,
                             const omq_block_params* theta, const float* x, float* y, void* workspace, size_t ws_bytes,
                             const omq_qcfg* cfg) {
  Ctx c;
  OMQ_TRY(make_ctx(c, stream, shape, w, theta, workspace, ws_bytes, cfg, false));
  OMQ_REQUIRE(x && y && omq_aligned16(x) && omq_aligned16(y), x && y ? OMQ_ERR_ALIGN : OMQ_ERR_INVALID_ARG);
  return block_fwd(c, x, y);
}

omq_status omq_block_step(omq_stream_t stream, const omq_block_shape* shape, const omq_block_weights* w,
                          const omq_block_params* theta, const float* x, const float* y_fp, float* y, float* loss,
                          const omq_block_params* grads, void* workspace, size_t ws_bytes, const omq_qcfg* cfg) {
  Ctx c;
  OMQ_TRY(make_ctx(c, stream, shape, w, theta, workspace, ws_bytes, cfg, true));
  OMQ_REQUIRE(x && y_fp && loss && grads, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(cfg->wbits < 16, OMQ_ERR_UNSUPPORTED);   // the step learns the clipping of Eq. 2
  if (cfg->wbits < 16)
    OMQ_REQUIRE(grads->gamma_qkv && grads->beta_qkv && grads->gamma_o && grads->beta_o && grads->gamma_gu &&
                    grads->beta_gu && grads->gamma_d && grads->beta_d,
                OMQ_ERR_INVALID_ARG);
  if (cfg->let)
    OMQ_REQUIRE(grads->s1 && grads->d1 && grads->so && grads->do_ && grads->sa && grads->s2 && grads->d2,
                OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(omq_aligned16(x) && omq_aligned16(y_fp) && (!y || omq_aligned16(y)), OMQ_ERR_ALIGN);
  float* yy = y ? y : c.ws.y;
  OMQ_TRY(block_fwd(c, x, yy));
  return block_bwd(c, x, yy, y_fp, loss, grads);
}

// ---------------------------------------------------------------------------------------------------
// single quantized linear
// ---------------------------------------------------------------------------------------------------
__global__ void add_vec_kernel(float* y, const float* x, int64_t n) {
  int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) y[i] += x[i];
}

__global__ void f32_to_bf16_kernel(const float* x, __nv_bfloat16* y, int64_t n) {
  int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) y[i] = __float2bfloat16_rn(x[i]);
}

omq_status omq_qlinear_fwd(omq_stream_t stream, int64_t T, int64_t Cin, int64_t Cout, const float* X, const void* W,
                           const float* B, const float* s, const float* delta, const float* gamma_logit,
                           const float* beta_logit, float* Y, const omq_qlinear_saved* sv, const omq_qcfg* cfg) {
  OMQ_TRY(omq_check_cfg(cfg));
  OMQ_REQUIRE(T > 0 && Cin > 0 && Cout > 0, OMQ_ERR_SHAPE);
  OMQ_REQUIRE(X && W && Y && sv && sv->w_hat && sv->x_hat && sv->b_tilde, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(!cfg->let || (s && delta), OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(Cin % 8 == 0 && Cout % 8 == 0, OMQ_ERR_ALIGN);
  cudaStream_t st = (cudaStream_t)stream;
  const int g = cfg->group == 0 ? (int)Cin : cfg->group;
  OMQ_REQUIRE(Cin % g == 0, OMQ_ERR_SHAPE);
  QState4 qw{sv->h_w, sv->z_w, sv->imax_w, sv->imin_w, nullptr, nullptr, nullptr, nullptr};
  const bool let = cfg->let != 0;
  OMQ_TRY(lwc_fwd_launch(st, lwc_args((const bf16*)W, Cout, Cin, *cfg, let ? s : nullptr, nullptr, gamma_logit,
                                      beta_logit, (bf16*)sv->w_hat, qw, let ? delta : nullptr, nullptr,
                                      let ? sv->b_tilde : nullptr)));
  const float* bias = nullptr;
  if (let) {
    if (B) { add_vec_kernel<<<(unsigned)((Cout + 255) / 256), 256, 0, st>>>(sv->b_tilde, B, Cout); OMQ_LAUNCH_CHECK(); }
    bias = sv->b_tilde;
  } else if (B) {
    OMQ_TRY(vec_copy(st, sv->b_tilde, B, Cout));
    bias = sv->b_tilde;
  }
  ActFwdArgs a{};
  a.producer = let ? AP_LET : AP_PLAIN; a.X = X; a.ldx = Cin; a.s = let ? s : nullptr; a.delta = let ? delta : nullptr;
  a.T = T; a.C = Cin; a.Xq = (bf16*)sv->x_hat; a.ldq = Cin; a.h = sv->h_a; a.z = sv->z_a; a.imax = sv->imax_a;
  a.imin = sv->imin_a; a.abits = cfg->abits; a.eps = cfg->h_eps; a.status = cfg->dev_status;
  OMQ_TRY(act_fwd_launch(st, a));
  return gemm_kk(st, T, Cout, Cin, (const bf16*)sv->x_hat, Cin, (const bf16*)sv->w_hat, Cin, Y, nullptr, Cout, bias,
                 nullptr, cfg->dev_status);
}

omq_status omq_qlinear_saved_sizes(int64_t T, int64_t Cin, int64_t Cout, const omq_qcfg* cfg, int64_t* sizes) {
  OMQ_TRY(omq_check_cfg(cfg));
  OMQ_REQUIRE(sizes, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(T > 0 && Cin > 0 && Cout > 0, OMQ_ERR_SHAPE);
  const int64_t g = cfg->group == 0 ? Cin : cfg->group;
  OMQ_REQUIRE(Cin % g == 0, OMQ_ERR_SHAPE);
  const int64_t ng = Cout * (Cin / g);
  const int64_t n[11] = {Cout * Cin, ng, ng, ng, ng, T * Cin, T, T, T, T, Cout};
  for (int i = 0; i < 11; ++i) sizes[i] = n[i];
  return OMQ_OK;
}

size_t omq_qlinear_workspace_size(int64_t T, int64_t Cin, int64_t Cout, const omq_qcfg* cfg) {
  (void)cfg;
  Carve c{nullptr, 0};
  c.take<bf16>(T * Cout);                       // dY in bf16
  c.take<float>(Cout * Cin);                    // dW_hat
  c.take<float>(T * Cin);                       // dX_hat
  c.take<float>(Cout);                          // dB~
  int64_t pe = imax64((int64_t)lwc_bwd_scratch_bytes(Cout, Cin) / 4 + 64, 2 * ((T + 3) / 4) * Cin);
  pe = imax64(pe, colsum_rows_parts(T) * Cout);
  c.take<float>(pe);
  return c.off + 256;
}

omq_status omq_qlinear_bwd(omq_stream_t stream, int64_t T, int64_t Cin, int64_t Cout, const float* X, const void* W,
                           const float* s, const float* delta, const float* gamma_logit, const float* beta_logit,
                           const omq_qlinear_saved* sv, const float* dY, float* dX, float* dgamma, float* dbeta,
                           float* ds, float* ddelta, void* workspace, size_t ws_bytes, const omq_qcfg* cfg) {
  OMQ_TRY(omq_check_cfg(cfg));
  OMQ_REQUIRE(T > 0 && Cin > 0 && Cout > 0, OMQ_ERR_SHAPE);
  OMQ_REQUIRE(cfg->wbits < 16, OMQ_ERR_UNSUPPORTED);
  OMQ_REQUIRE(X && W && sv && dY && dgamma && dbeta, OMQ_ERR_INVALID_ARG);
  const bool let = cfg->let != 0;
  OMQ_REQUIRE(!let || (s && delta && ds && ddelta), OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(workspace && ws_bytes >= omq_qlinear_workspace_size(T, Cin, Cout, cfg), OMQ_ERR_WORKSPACE);
  OMQ_REQUIRE(omq_aligned16(workspace) && omq_aligned16(dY), OMQ_ERR_ALIGN);
  cudaStream_t st = (cudaStream_t)stream;
  Carve c{(uint8_t*)workspace, 0};
  bf16* dYb = c.take<bf16>(T * Cout);
  float* dWh = c.take<float>(Cout * Cin);
  float* dXh = c.take<float>(T * Cin);
  float* dB = c.take<float>(Cout);
  int64_t pe = imax64((int64_t)lwc_bwd_scratch_bytes(Cout, Cin) / 4 + 64, 2 * ((T + 3) / 4) * Cin);
  pe = imax64(pe, colsum_rows_parts(T) * Cout);
  float* part = c.take<float>(pe);
  f32_to_bf16_kernel<<<(unsigned)((T * Cout + 255) / 256), 256, 0, st>>>(dY, dYb, T * Cout);
  OMQ_LAUNCH_CHECK();
  OMQ_TRY(gemm_dw(st, T, Cout, Cin, dYb, (const bf16*)sv->x_hat, dWh, cfg->dev_status));
  if (let) OMQ_TRY(colsum_rows(st, dY, T, Cout, Cout, part, dB, 1.f, 0));
  QState4 qw{sv->h_w, sv->z_w, sv->imax_w, sv->imin_w, nullptr, nullptr, nullptr, nullptr};
  omq_qcfg cf = *cfg;
  OMQ_TRY(lwc_bwd_full(st, (const bf16*)W, Cout, Cin, cf, let ? s : nullptr, nullptr, gamma_logit, beta_logit, qw, dWh,
                       dgamma, dbeta, nullptr, let ? dB : nullptr, let ? ds : nullptr, let ? ddelta : nullptr,
                       cfg->accumulate, part));
  if (dX || let) {
    OMQ_TRY(gemm_dx(st, T, Cout, Cin, dYb, (const bf16*)sv->w_hat, dXh, cfg->dev_status));
    ActBwdArgs a{};
    a.producer = let ? AP_LET : AP_PLAIN; a.X = X; a.ldx = Cin; a.s = let ? s : nullptr; a.delta = let ? delta : nullptr;
    a.T = T; a.C = Cin; a.h = sv->h_a; a.z = sv->z_a; a.imax = sv->imax_a; a.imin = sv->imin_a; a.dXq = dXh; a.lddq = Cin;
    a.dX = dX; a.lddx = Cin; a.rows_per_cta = 4; a.abits = cfg->abits; a.eps = cfg->h_eps;
    a.part_s = let ? part : nullptr;
    a.part_d = let ? part + ((T + 3) / 4) * Cin : nullptr;
    OMQ_TRY(act_bwd_launch(st, a));
    if (let) {
      OMQ_TRY(omq_colsum_partials2(st, ColsumJob{a.part_s, (T + 3) / 4, Cin, ds, 1.f, 1},
                                   ColsumJob{a.part_d, (T + 3) / 4, Cin, ddelta, 1.f, 1}));
    }
  }
  return OMQ_OK;
}

}  // extern "C"

// ---------------------------------------------------------------------------------------------
// LET initialisation: statistics of the full-precision block, then the initial parameters
// ---------------------------------------------------------------------------------------------
extern "C" omq_status omq_let_stats_accumulate(omq_stream_t stream, const omq_block_shape* shape,
                                               const omq_block_weights* w, const float* x,
                                               const omq_let_stats* stats, int32_t first, void* workspace,
                                               size_t ws_bytes, int32_t* dev_status) {
  OMQ_REQUIRE(x && stats && stats->a_absmax && stats->a_sum && stats->q_absmax && stats->k_absmax &&
                  stats->o_absmax && stats->o_sum && stats->b_absmax && stats->b_sum,
              OMQ_ERR_INVALID_ARG);
  omq_qcfg fp{};
  fp.wbits = 16; fp.abits = 16; fp.group = 0; fp.let = 0; fp.h_eps = 1e-5f; fp.accumulate = 0;
  fp.dev_status = dev_status;
  omq_block_params none{};
  Ctx c;
  OMQ_TRY(make_ctx(c, stream, shape, w, &none, workspace, ws_bytes, &fp, false));
  BlockWS& ws = c.ws;
  OMQ_TRY(block_fwd(c, x, ws.y));
  const int f = first ? 1 : 0;
  OMQ_TRY(let_colstats(c.st, x, c.T, c.d, c.d, ws.rstd1, stats->a_absmax, stats->a_sum, f));
  OMQ_TRY(let_colstats_bf16(c.st, ws.Qh, c.T, c.dq, c.dq, stats->q_absmax, f));
  OMQ_TRY(let_colstats_bf16(c.st, ws.Kh, c.T, c.dkv, c.dkv, stats->k_absmax, f));
  OMQ_TRY(let_colstats(c.st, ws.O, c.T, c.dq, c.dq, nullptr, stats->o_absmax, stats->o_sum, f));
  OMQ_TRY(let_colstats(c.st, ws.h1, c.T, c.d, c.d, ws.rstd2, stats->b_absmax, stats->b_sum, f));
  return OMQ_OK;
}

extern "C" size_t omq_let_init_workspace_size(const omq_block_shape* shape) {
  if (!shape) return 0;
  const int64_t d = shape->d, dq = (int64_t)shape->n_heads * shape->head_dim;
  return (size_t)(2 * d + dq) * sizeof(float) + 1024;
}

extern "C" omq_status omq_let_init(omq_stream_t stream, const omq_block_shape* shape, const omq_block_weights* w,
                                   const omq_let_stats* stats, int64_t ntok, float alpha,
                                   const omq_block_params* theta, void* workspace, size_t ws_bytes) {
  OMQ_REQUIRE(shape && w && stats && theta && ntok > 0, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(alpha >= 0.f && alpha <= 1.f, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(theta->s1 && theta->d1 && theta->so && theta->do_ && theta->sa && theta->s2 && theta->d2,
              OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(w->wqkv && w->wo && w->wgu, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(shape->n_heads > 0 && shape->n_kv > 0 && shape->n_heads % shape->n_kv == 0 && shape->head_dim > 0,
              OMQ_ERR_SHAPE);
  OMQ_REQUIRE(workspace && ws_bytes >= omq_let_init_workspace_size(shape), OMQ_ERR_WORKSPACE);
  cudaStream_t st = (cudaStream_t)stream;
  const int64_t d = shape->d, hd = shape->head_dim, dq = shape->n_heads * hd, dkv = shape->n_kv * hd;
  const int64_t f = shape->ffn, nqkv = dq + 2 * dkv;
  float* wm_qkv = (float*)workspace;
  float* wm_gu = wm_qkv + d;
  float* wm_o = wm_gu + d;
  const float floor = 1e-5f;
  OMQ_TRY(let_weight_colmax(st, (const __nv_bfloat16*)w->wqkv, nqkv, d, wm_qkv, 1));
  OMQ_TRY(let_weight_colmax(st, (const __nv_bfloat16*)w->wgu, 2 * f, d, wm_gu, 1));
  OMQ_TRY(let_weight_colmax(st, (const __nv_bfloat16*)w->wo, d, dq, wm_o, 1));
  OMQ_TRY(let_smooth_pair(st, d, stats->a_absmax, stats->a_sum, wm_qkv, (double)ntok, alpha, floor, theta->s1,
                          theta->d1));
  OMQ_TRY(let_smooth_pair(st, d, stats->b_absmax, stats->b_sum, wm_gu, (double)ntok, alpha, floor, theta->s2,
                          theta->d2));
  OMQ_TRY(let_kv_pairs(st, shape->n_kv, shape->n_heads / shape->n_kv, (int)hd, stats->o_absmax, stats->o_sum, wm_o,
                       stats->q_absmax, stats->k_absmax, (double)ntok, alpha, floor, theta->so, theta->do_, theta->sa));
  (void)dkv;
  return OMQ_OK;
}

// ---------------------------------------------------------------------------------------------
// fold & pack
// ---------------------------------------------------------------------------------------------
namespace {
struct PackWS {
  uint8_t* codes; float* r_qkv; float* shift_qkv; float* so_exp; float* do_exp; int32_t* imax; int32_t* imin;
};
PackWS carve_pack(Carve& c, const omq_block_shape& s) {
  const int64_t d = s.d, hd = s.head_dim, dq = (int64_t)s.n_heads * hd, dkv = (int64_t)s.n_kv * hd, f = s.ffn;
  const int64_t nqkv = dq + 2 * dkv;
  const int64_t big = imax64(imax64(nqkv * d, d * dq), imax64(2 * f * d, d * f));
  PackWS p;
  p.codes = c.take<uint8_t>(big);
  p.r_qkv = c.take<float>(nqkv);
  p.shift_qkv = c.take<float>(nqkv);
  p.so_exp = c.take<float>(dq);
  p.do_exp = c.take<float>(dq);
  p.imax = c.take<int32_t>(big / 8 + 64);          // one entry per group, groups of >= 8 columns
  p.imin = c.take<int32_t>(big / 8 + 64);
  return p;
}
}  // namespace

extern "C" size_t omq_block_pack_workspace_size(const omq_block_shape* shape, const omq_qcfg* cfg) {
  if (check_block(shape, cfg) != OMQ_OK) return 0;
  Carve dry{nullptr, 0};
  carve_pack(dry, *shape);
  return dry.off + 256;
}

extern "C" omq_status omq_block_fold_pack(omq_stream_t stream, const omq_block_shape* shape, const omq_block_weights* w,
                                          const omq_block_params* theta, const omq_qcfg* cfg,
                                          const omq_block_packed* out, void* workspace, size_t ws_bytes) {
  OMQ_TRY(check_block(shape, cfg));
  OMQ_REQUIRE(cfg->wbits < 16 && cfg->wbits >= 2 && cfg->wbits <= 8, OMQ_ERR_UNSUPPORTED);
  OMQ_REQUIRE(w && theta && out && w->wqkv && w->wo && w->wgu && w->wd, OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(theta->gamma_qkv && theta->beta_qkv && theta->gamma_o && theta->beta_o && theta->gamma_gu &&
                  theta->beta_gu && theta->gamma_d && theta->beta_d,
              OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(out->codes_qkv && out->codes_o && out->codes_gu && out->codes_d && out->h_qkv && out->z_qkv &&
                  out->h_o && out->z_o && out->h_gu && out->z_gu && out->h_d && out->z_d,
              OMQ_ERR_INVALID_ARG);
  const bool let = cfg->let != 0;
  if (let)
    OMQ_REQUIRE(theta->s1 && theta->d1 && theta->so && theta->do_ && theta->sa && theta->s2 && theta->d2 &&
                    out->b_qkv && out->b_o && out->b_gu && out->ln1_gain && out->ln1_bias && out->ln2_gain &&
                    out->ln2_bias && out->sa,
                OMQ_ERR_INVALID_ARG);
  OMQ_REQUIRE(workspace && ws_bytes >= omq_block_pack_workspace_size(shape, cfg) && omq_aligned16(workspace),
              OMQ_ERR_WORKSPACE);
  cudaStream_t st = (cudaStream_t)stream;
  Carve cv{(uint8_t*)workspace, 0};
  PackWS p = carve_pack(cv, *shape);
  const int64_t d = shape->d, hd = shape->head_dim, H = shape->n_heads, Hkv = shape->n_kv;
  const int64_t dq = H * hd, dkv = Hkv * hd, f = shape->ffn, nqkv = dq + 2 * dkv, rep = H / Hkv;
  if (let) {
    OMQ_TRY(qkv_row_vectors(st, (int)dq, (int)dkv, theta->so, theta->do_, p.r_qkv, p.shift_qkv));
    OMQ_TRY(gqa_expand(st, theta->so, p.so_exp, (int)Hkv, (int)rep, (int)hd, 0));
    OMQ_TRY(gqa_expand(st, theta->do_, p.do_exp, (int)Hkv, (int)rep, (int)hd, 0));
  }
  struct One {
    const void* W; int64_t Cout, Cin; const float *s, *r, *gl, *bl, *delta, *shift; float* Bt;
    uint8_t* codes; float* h; int32_t* z;
  } lin[4] = {
      {w->wqkv, nqkv, d, let ? theta->s1 : nullptr, let ? p.r_qkv : nullptr, theta->gamma_qkv, theta->beta_qkv,
       let ? theta->d1 : nullptr, let ? p.shift_qkv : nullptr, let ? out->b_qkv : nullptr, out->codes_qkv,
       out->h_qkv, out->z_qkv},
      {w->wo, d, dq, let ? p.so_exp : nullptr, nullptr, theta->gamma_o, theta->beta_o, let ? p.do_exp : nullptr,
       nullptr, let ? out->b_o : nullptr, out->codes_o, out->h_o, out->z_o},
      {w->wgu, 2 * f, d, let ? theta->s2 : nullptr, nullptr, theta->gamma_gu, theta->beta_gu,
       let ? theta->d2 : nullptr, nullptr, let ? out->b_gu : nullptr, out->codes_gu, out->h_gu, out->z_gu},
      {w->wd, d, f, nullptr, nullptr, theta->gamma_d, theta->beta_d, nullptr, nullptr, nullptr, out->codes_d,
       out->h_d, out->z_d},
  };
  for (const One& l : lin) {
    LwcFwdArgs a{};
    a.W = (const bf16*)l.W; a.Cout = l.Cout; a.Cin = l.Cin; a.group = cfg->group == 0 ? (int)l.Cin : cfg->group;
    a.s = l.s; a.r = l.r; a.gl = l.gl; a.bl = l.bl; a.lwc = 1; a.Wq = nullptr; a.codes = p.codes;
    a.h = l.h; a.z = l.z; a.imax = p.imax; a.imin = p.imin;
    a.bias_delta = l.delta; a.bias_shift = l.shift; a.Bt = l.Bt;
    a.wbits = cfg->wbits; a.eps = cfg->h_eps; a.status = cfg->dev_status;
    OMQ_TRY(lwc_fwd_launch(st, a));
    OMQ_TRY(pack_codes_launch(st, p.codes, l.Cout, l.Cin, cfg->wbits, l.codes));
  }
  if (let) {
    OMQ_TRY(norm_fold_launch(st, d, theta->s1, theta->d1, out->ln1_gain, out->ln1_bias));
    OMQ_TRY(norm_fold_launch(st, d, theta->s2, theta->d2, out->ln2_gain, out->ln2_bias));
    OMQ_REQUIRE(cudaMemcpyAsync(out->sa, theta->sa, (size_t)dkv * sizeof(float), cudaMemcpyDeviceToDevice, st) ==
                    cudaSuccess,
                OMQ_ERR_CUDA);
  }
  return OMQ_OK;
}
