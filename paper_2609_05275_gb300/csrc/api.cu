// C ABI of the library (include/ld.h): handle, schedule, workspace layout
// and the per-layer launch sequence of the forward and backward passes.
//
// Forward of layer l (kept rows only, compact order, M = kept_cnt[l] * S):
//   xh  = RMSNorm_1(x[kept])                         (gather; copy of x saved)
//   qkv = xh W_qkv^T ; RoPE on the q and k heads
//   o   = causal GQA attention(q, k, v)
//   x[kept] += r * (o W_o^T)                         (= Z^l, saved compact)
//   zh  = RMSNorm_2(Z^l[kept]) ; gu = zh W_gu^T ; h = silu(g) * u
//   x[kept] += r * (h W_d^T)                         (= X^{l+1})
// with r = alpha / (1 - p^{l,t}) (Eq. transformer_layer_dropout_train and the
// Dropout Scale paragraph).  Rows of dropped sequences are never touched.
// The backward walks the layers in reverse and mirrors this; the gradient
// of a dropped row passes through unchanged (it is the identity there).
// Per-token kept lists run the same sequence with row unit 1 (see Rows): the
// compact rows are kept tokens, attention works on per-sequence segments.
// The backward's weight-gradient products run on a side stream (see
// backward_impl).
#include <cmath>
#include <cstdio>
#include <cstring>
#include <new>
#include <vector>

#include "ld_internal.cuh"

using namespace ldk;

namespace {

size_t align_up(size_t v) { return (v + 255) & ~size_t(255); }

struct Layout {
  size_t status, mask, kidx, kcnt, kseg, rcos, rsin, alibi;
  size_t layer0, per_layer;
  size_t xin, xh, qkv, o, lse, z, zh, gu, h, rstd1, rstd2;  // offsets inside a layer block
  size_t dy, dh, dgu, dzh, dz, dO, dqkv, dxh, Dvec, dqacc, part;
  size_t xres, dres;  // float32 residual stream and its gradient (bf16 path)
  size_t total;
};

struct Handle {
  ld_config cfg;
  bool have_sched = false;
  ld_schedule sched;
  std::vector<float> p_expl;
  Layout lay;
  size_t esz = 2;
  int max_rows = 0, nqkv = 0, nf = 0, part_blocks = 0;  // nf: columns of the gate/up projection
  void* last_ws = nullptr;
  cudaStream_t last_stream = nullptr;
  bool have_masks = false;
  bool fwd_valid = false;
  void* fwd_ws = nullptr;
  std::vector<float> fwd_scale;
  size_t eval_xres = 0, eval_total = 0;  // evaluation layout: residual stream offset, total bytes
  // device-time accounting (ld_set_timing): event pairs around launches
  bool timing = false;
  std::vector<cudaEvent_t> ev[LD_KCLASS_COUNT];
  size_t ev_used[LD_KCLASS_COUNT] = {};
  // backward: the four weight-gradient products of a layer run on a side
  // stream forked from (and joined back to) the caller's stream; wg_in[k]
  // orders product k after its inputs, wg_out[k] the next write of those
  // inputs after product k
  cudaStream_t side = nullptr;
  cudaEvent_t wg_in[4] = {}, wg_out[4] = {};
  ~Handle() {
    for (auto& v : ev)
      for (cudaEvent_t e : v) cudaEventDestroy(e);
    for (int k = 0; k < 4; ++k) {
      if (wg_in[k]) cudaEventDestroy(wg_in[k]);
      if (wg_out[k]) cudaEventDestroy(wg_out[k]);
    }
    if (side) cudaStreamDestroy(side);
  }
};

// Create the side stream and its events (once per handle, at the first
// backward).
cudaError_t ensure_side(Handle* h) {
  if (h->side) return cudaSuccess;
  cudaError_t e = cudaStreamCreateWithFlags(&h->side, cudaStreamNonBlocking);
  for (int k = 0; k < 4 && e == cudaSuccess; ++k) {
    e = cudaEventCreateWithFlags(&h->wg_in[k], cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->wg_out[k], cudaEventDisableTiming);
  }
  return e;
}

// Records an event pair around the launches of its scope when timing is on.
struct Timed {
  Handle* h;
  int cls;
  cudaStream_t st;
  Timed(Handle* h_, int cls_, cudaStream_t st_) : h(h_), cls(cls_), st(st_) { mark(); }
  ~Timed() { mark(); }
  void mark() {
    if (!h->timing) return;
    auto& v = h->ev[cls];
    size_t& u = h->ev_used[cls];
    if (u == v.size()) {
      cudaEvent_t e;
      if (cudaEventCreate(&e) != cudaSuccess) return;
      v.push_back(e);
    }
    cudaEventRecord(v[u++], st);
  }
};

Handle* H(void* h) { return static_cast<Handle*>(h); }

bool finite(float v) { return std::isfinite(v); }

// ------------------------------------------------------------------ schedule
// p^l_dist (Dropout Distribution section), widened from float exactly.
double dist_rate(const Handle* h, int l) {
  const int L = h->cfg.L;
  const double pm = (double)h->sched.p_max;
  switch (h->sched.dist) {
    case LD_DIST_UNIFORM: return pm;
    case LD_DIST_ILD: return L == 1 ? 0.0 : (pm * (double)l) / (double)(L - 1);
    case LD_DIST_ALD: return (l % 2 == 1) ? pm : 0.0;
    default: return (double)h->p_expl[l];
  }
}

// time factor (Dropout Schedule section; RAMP is a warm-up ramp).
double time_factor(const Handle* h, long long t) {
  const ld_schedule& s = h->sched;
  switch (s.time) {
    case LD_TIME_ITS: return (double)t / (double)(s.T - 1);
    case LD_TIME_DTS: return 1.0 - (double)t / (double)(s.T - 1);
    case LD_TIME_RAMP: {
      double f = (double)(t - s.ramp_t0) / (double)(s.ramp_t1 - s.ramp_t0);
      f = f < 0.0 ? 0.0 : (f > 1.0 ? 1.0 : f);
      const double s0 = (double)s.ramp_s0, s1 = (double)s.ramp_s1;
      return s0 + (s1 - s0) * f;
    }
    default: return 1.0;
  }
}

void step_rates(const Handle* h, long long t, double* p, unsigned long long* thr, float* scale) {
  for (int l = 0; l < h->cfg.L; ++l) {
    double v = dist_rate(h, l) * time_factor(h, t);
    v = v < 0.0 ? 0.0 : (v > 1.0 ? 1.0 : v);
    if (p) p[l] = v;
    if (thr) thr[l] = (unsigned long long)std::floor(v * 4294967296.0);
    if (scale) scale[l] = v >= 1.0 ? 0.0f : (float)((double)h->cfg.alpha / (1.0 - v));
  }
}

// ------------------------------------------------------------------ layout
void make_layout(Handle* h) {
  const ld_config& c = h->cfg;
  const size_t R = (size_t)c.B * c.S, e = h->esz;
  Layout& y = h->lay;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off = align_up(off + bytes);
    return at;
  };
  y.status = take(64);
  const size_t nm = c.sublayer ? 2 : 1;  // attention and FFN tables with sub-layer granularity
  const size_t per = c.granularity == LD_PER_TOKEN ? R : (size_t)c.B;  // mask entries per (table, layer)
  y.mask = take(nm * c.L * per);
  y.kidx = take(nm * c.L * per * 4);
  y.kcnt = take(nm * c.L * 4);
  y.kseg = take(nm * c.L * (c.B + 1) * 4);
  y.rcos = take((size_t)c.S * (c.Dh / 2) * 4);
  y.rsin = take((size_t)c.S * (c.Dh / 2) * 4);
  y.alibi = take((size_t)c.H * 4);
  // per-layer saved activations
  size_t lo = 0;
  auto ltake = [&](size_t bytes) {
    const size_t at = lo;
    lo = align_up(lo + bytes);
    return at;
  };
  y.xin = ltake(R * c.d * 4);  // float32 copies of X and Z (RMSNorm backward)
  y.xh = ltake(R * c.d * e);
  y.qkv = ltake(R * h->nqkv * e);
  y.o = ltake(R * c.H * c.Dh * e);
  y.lse = ltake((size_t)c.H * R * 4);
  y.z = ltake(R * c.d * 4);
  y.zh = ltake(R * c.d * e);
  y.gu = ltake(R * h->nf * e);  // g || u (SwiGLU) or u (squared ReLU)
  y.h = ltake(R * c.F * e);
  y.rstd1 = ltake(R * 4);
  y.rstd2 = ltake(R * 4);
  y.per_layer = lo;
  y.layer0 = off;
  // evaluation layout (ld_forward_eval): the same header, one block of
  // activations reused by every layer, then the float32 residual stream
  const size_t eo = align_up(off + lo);
  h->eval_xres = c.fp32_debug ? 0 : eo;
  h->eval_total = c.fp32_debug ? eo : align_up(eo + R * c.d * 4);
  off = align_up(off + (size_t)c.L * lo);
  // backward scratch (shared by all layers)
  y.dy = take(R * c.d * e);
  y.dh = take(R * c.F * e);
  y.dgu = take(R * h->nf * e);
  y.dzh = take(R * c.d * 4);  // float32: inputs of the RMSNorm backward
  y.dz = take(R * c.d * e);
  y.dO = take(R * c.H * c.Dh * e);
  y.dqkv = take(R * h->nqkv * e);
  y.dxh = take(R * c.d * 4);
  y.Dvec = take((size_t)c.H * R * 4);
  y.dqacc = take(R * c.H * c.Dh * 4);
  y.part = take((size_t)h->part_blocks * c.d * 4);
  y.xres = c.fp32_debug ? 0 : take(R * c.d * 4);
  y.dres = c.fp32_debug ? 0 : take(R * c.d * 4);
  y.total = off;
}

template <typename T>
T* at(void* ws, size_t off) {
  return reinterpret_cast<T*>(static_cast<char*>(ws) + off);
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15) == 0; }

// The CUDA error behind the last LD_ERR_CUDA this thread returned.
thread_local cudaError_t g_last_cuda = cudaSuccess;

#define LD_CHECK(...)                        \
  do {                                       \
    const cudaError_t e_ = (__VA_ARGS__);    \
    if (e_ != cudaSuccess) {                 \
      g_last_cuda = e_;                      \
      return LD_ERR_CUDA;                    \
    }                                        \
  } while (0)

ld_status check_device() {
  // once per process (initialisation of a function-local static is thread-safe)
  static const ld_status verdict = [] {
    int dev = 0, major = 0, minor = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return LD_ERR_CUDA;
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    return (major == 10 && minor == 3) ? LD_OK : LD_ERR_UNSUPPORTED;
  }();
  return verdict;
}

ld_status check_weights(const Handle* h, const ld_layer_w* W) {
  if (!W) return LD_ERR_ARG;
  for (int l = 0; l < h->cfg.L; ++l) {
    const void* ps[6] = {W[l].w_qkv, W[l].w_o, W[l].w_gu, W[l].w_d, W[l].g1, W[l].g2};
    for (const void* p : ps)
      if (!p || !aligned16(p)) return LD_ERR_ARG;
  }
  return LD_OK;
}

GemmArgs gemm_base() {
  GemmArgs a;
  std::memset(&a, 0, sizeof(a));
  a.alpha = 1.0f;
  return a;
}

// The rows a block runs on.  Whole kept sequences: *cnt of them, `unit` =
// S compact rows each, compact row m from sequence idx[m / S].  Per token:
// *cnt compact rows (the kept-token count rounded up to 64), unit = 1, idx
// the kept tokens' rows b S + s (-1 on the padding rows) and seg the
// per-sequence segments (seg[B] = the kept-token count).
struct Rows {
  const int* cnt;
  const int* idx;
  const int* seg;
  int unit;
  const int* tok() const { return seg ? idx : nullptr; }
};

// Kept rows of table w (0: attention or layer mask, 1: FFN mask with
// sub-layer granularity) of layer l.
Rows rows_of(const Handle* h, void* ws, int w, int l) {
  const ld_config& c = h->cfg;
  const Layout& y = h->lay;
  const bool tokg = c.granularity == LD_PER_TOKEN;
  const size_t wl = (size_t)w * c.L + l;
  Rows r;
  r.cnt = at<int>(ws, y.kcnt) + wl;
  r.idx = at<int>(ws, y.kidx) + wl * (tokg ? (size_t)c.B * c.S : (size_t)c.B);
  r.seg = tokg ? at<int>(ws, y.kseg) + wl * (c.B + 1) : nullptr;
  r.unit = tokg ? 1 : c.S;
  return r;
}

// Per token: zero rows [kept tokens, kept tokens + 128) of a buffer the
// attention reads (the tiles of the last sequence run past its kept tokens)
// or a weight-gradient product contracts over (the padding rows).
template <typename T>
cudaError_t zero_tail(const Handle* h, const Rows& r, T* buf, int ld, int ncols, int planes, cudaStream_t st) {
  if (!r.seg) return cudaSuccess;
  return launch_zero_rows<T>(buf, ld, ncols, planes, (long long)h->max_rows, r.seg + h->cfg.B, 128, h->max_rows, st);
}

// Forward/data-gradient product on the kept rows:
// D[M x N] = alpha * A[M x K] B(n, k), M = *cnt * unit (device-side).
GemmArgs rows_gemm(const Handle* h, const Rows& r, int N, int K, const void* A, int lda, const void* B, int ldb,
                   int b_mn) {
  GemmArgs a = gemm_base();
  a.M_cnt = r.cnt;
  a.M_mul = r.unit;
  a.M_cap = h->max_rows;
  a.N = N;
  a.K = K;
  a.A = A;
  a.lda = lda;
  a.a_mn = 0;
  a.B = B;
  a.ldb = ldb;
  a.b_mn = b_mn;
  return a;
}

// Weight-gradient product: dW[M x N] = sum over the kept rows m of
// X1[m, i] X2[m, j]; the contraction extent is *cnt * unit (device-side; per
// token the padding rows hold zeros in X1 or X2).
GemmArgs wgrad_gemm(const Handle* h, const Rows& r, int M, int N, const void* X1, int ld1, const void* X2, int ld2,
                    float* out) {
  GemmArgs a = gemm_base();
  a.M = M;
  a.N = N;
  a.K_cnt = r.cnt;
  a.K_mul = r.unit;
  a.K_cap = h->max_rows;
  a.A = X1;
  a.lda = ld1;
  a.a_mn = 1;
  a.B = X2;
  a.ldb = ld2;
  a.b_mn = 1;
  a.epi = EPI_STORE_F32;
  a.D = out;
  a.ldd = N;
  return a;
}

template <typename T>
cudaError_t gemm(const GemmArgs& a, cudaStream_t st);
template <>
cudaError_t gemm<bf16>(const GemmArgs& a, cudaStream_t st) {
  return gemm_tc(a, st);
}
template <>
cudaError_t gemm<float>(const GemmArgs& a, cudaStream_t st) {
  return gemm_simt(a, st);
}

// The ALiBi slope table in the workspace, or null without ALiBi.
const float* alibi_table(const Handle* h, void* ws) { return h->cfg.alibi ? at<float>(ws, h->lay.alibi) : nullptr; }

// Attention: tensor-core flash attention on the bf16 path, SIMT float32 on
// the debug path.
template <typename T>
cudaError_t attn_fwd(const Handle* h, void* ws, const T* qkv, T* o, float* lse, const Rows& r, cudaStream_t st);
template <>
cudaError_t attn_fwd<float>(const Handle* h, void* ws, const float* qkv, float* o, float* lse, const Rows& r,
                            cudaStream_t st) {
  const ld_config& c = h->cfg;
  return launch_attn_fwd_simt<float>(qkv, h->nqkv, o, c.H * c.Dh, lse, r.cnt, c.S, c.H, c.Hkv, c.Dh, h->max_rows,
                                     alibi_table(h, ws), r.seg, r.tok(), st);
}
template <>
cudaError_t attn_fwd<bf16>(const Handle* h, void* ws, const bf16* qkv, bf16* o, float* lse, const Rows& r,
                           cudaStream_t st) {
  const ld_config& c = h->cfg;
  if (attn_tc_supported(c.S, c.Dh))
    return launch_attn_fwd_tc(qkv, h->nqkv, o, c.H * c.Dh, lse, r.cnt, c.S, c.H, c.Hkv, c.Dh, c.B, alibi_table(h, ws),
                              r.seg, at<int>(ws, h->lay.status), st);
  // per-token granularity is refused at ld_create on this path
  return launch_attn_fwd_mma(qkv, h->nqkv, o, c.H * c.Dh, lse, r.cnt, c.S, c.H, c.Hkv, c.Dh, c.B, alibi_table(h, ws),
                             st);
}

// Attention backward: dq, dk, dv into dqkv with the inverse RoPE applied to
// dq and dk (in the tcgen05 kernels' epilogues and dq_finish on the bf16
// tcgen05 path, dq_finish and a rotation of the k heads on the mma.sync path,
// a separate rotation on the debug path).
template <typename T>
cudaError_t attn_bwd(const Handle* h, void* ws, const T* qkv, const T* o, const T* dO, const float* lse, float* Dvec,
                     T* dqkv, const Rows& r, cudaStream_t st) {
  const ld_config& c = h->cfg;
  const bool rope = c.rope_theta != 0.0f;
  const float* rcos = rope ? at<float>(ws, h->lay.rcos) : nullptr;
  const float* rsin = rope ? at<float>(ws, h->lay.rsin) : nullptr;
  cudaError_t e = launch_attn_rowdot<T>(dO, o, c.H * c.Dh, c.H, c.Dh, r.cnt, r.unit, h->max_rows, Dvec, st);
  if (e == cudaSuccess) e = zero_tail<float>(h, r, Dvec, 1, 1, c.H, st);
  if (e != cudaSuccess) return e;
  if (sizeof(T) == 4) {
    e = launch_attn_bwd_simt<T>(qkv, h->nqkv, dO, c.H * c.Dh, lse, Dvec, dqkv, r.cnt, c.S, c.H, c.Hkv, c.Dh,
                                h->max_rows, alibi_table(h, ws), r.seg, r.tok(), st);
    if (e != cudaSuccess || !rope) return e;
    return launch_rope_apply<T>(dqkv, h->nqkv, c.H + c.Hkv, c.Dh, rcos, rsin, r.cnt, c.S, h->max_rows, 1, r.tok(),
                                st);
  }
  float* dq_acc = at<float>(ws, h->lay.dqacc);
  const bf16* q16 = reinterpret_cast<const bf16*>(qkv);
  bf16* d16 = reinterpret_cast<bf16*>(dqkv);
  if (attn_bwd_tc_supported(c.S, c.Dh))  // dQ finished inside
    return launch_attn_bwd_tc(q16, h->nqkv, reinterpret_cast<const bf16*>(dO), c.H * c.Dh, lse, Dvec, dq_acc, d16,
                              r.cnt, c.S, c.H, c.Hkv, c.Dh, c.B, rcos, rsin, alibi_table(h, ws), r.seg, r.tok(),
                              at<int>(ws, h->lay.status), st);
  {  // whole sequences only (per-token granularity is refused at ld_create on this path)
    e = launch_attn_bwd_mma(q16, h->nqkv, reinterpret_cast<const bf16*>(o), reinterpret_cast<const bf16*>(dO),
                            c.H * c.Dh, lse, Dvec, dq_acc, d16, r.cnt, c.S, c.H, c.Hkv, c.Dh, c.B, alibi_table(h, ws),
                            st);
    if (e == cudaSuccess && rope)  // the k heads of dqkv
      e = launch_rope_apply<bf16>(d16 + (size_t)c.H * c.Dh, h->nqkv, c.Hkv, c.Dh, rcos, rsin, r.cnt, c.S, h->max_rows,
                                  1, nullptr, st);
  }
  if (e != cudaSuccess) return e;
  return launch_dq_finish(dq_acc, d16, h->nqkv, c.H, c.Dh, rcos, rsin, r.cnt, c.S, h->max_rows, r.tok(), st);
}

// One layer of the forward on the rows of its kept lists: the attention
// block on ra, the FFN block on rf, branch scale s.  `lb` is the layer's
// block of saved activations; x the float32 (or debug-path) residual
// stream, updated in place.
template <typename T>
ld_status forward_layer(Handle* h, void* ws, char* lb, const ld_layer_w& Wl, float* x, const Rows& ra, const Rows& rf,
                        float s, cudaStream_t st) {
  const ld_config& c = h->cfg;
  const Layout& y = h->lay;
  const bool f32 = sizeof(T) == 4;
  const bool fused_rope = !f32 && c.rope_theta != 0.0f && c.Dh >= 64;
  const bool same_rows = ra.cnt == rf.cnt;  // both blocks keep the same rows
  const int HD = c.H * c.Dh;
  float* rcos = at<float>(ws, y.rcos);
  float* rsin = at<float>(ws, y.rsin);
  float* xin = reinterpret_cast<float*>(lb + y.xin);
  T* xh = reinterpret_cast<T*>(lb + y.xh);
  T* qkv = reinterpret_cast<T*>(lb + y.qkv);
  T* o = reinterpret_cast<T*>(lb + y.o);
  float* lse = reinterpret_cast<float*>(lb + y.lse);
  float* z = reinterpret_cast<float*>(lb + y.z);
  T* zh = reinterpret_cast<T*>(lb + y.zh);
  T* gu = reinterpret_cast<T*>(lb + y.gu);
  T* hh = reinterpret_cast<T*>(lb + y.h);
  float* rstd1 = reinterpret_cast<float*>(lb + y.rstd1);
  float* rstd2 = reinterpret_cast<float*>(lb + y.rstd2);
  const T* g1 = static_cast<const T*>(Wl.g1);
  const T* g2 = static_cast<const T*>(Wl.g2);

  { Timed tm_(h, LD_KCLASS_ROWWISE, st); LD_CHECK(launch_rmsnorm_fwd<float, T>(x, 1, ra.idx, ra.cnt, ra.unit, c.d, h->max_rows, g1, c.eps, xin, xh, rstd1, st)); }
  GemmArgs a = rows_gemm(h, ra, h->nqkv, c.d, xh, c.d, Wl.w_qkv, c.d, 0);
  a.epi = EPI_STORE;
  a.D = qkv;
  a.ldd = h->nqkv;
  if (fused_rope) {  // RoPE on the q / k heads in the projection's epilogue
    a.epi = EPI_ROPE;
    a.rope_cos = rcos;
    a.rope_sin = rsin;
    a.Dh = c.Dh;
    a.S = c.S;
    a.pos_tok = ra.tok();
    a.rope_cols = (c.H + c.Hkv) * c.Dh;
  }
  { Timed tm_(h, LD_KCLASS_GEMM, st); LD_CHECK(gemm<T>(a, st)); }
  if (c.rope_theta != 0.0f && !fused_rope)
    { Timed tm_(h, LD_KCLASS_ROWWISE, st); LD_CHECK(launch_rope_apply<T>(qkv, h->nqkv, c.H + c.Hkv, c.Dh, rcos, rsin, ra.cnt, c.S, h->max_rows, 0, ra.tok(), st)); }
  if (ra.seg) { Timed tm_(h, LD_KCLASS_ROWWISE, st); LD_CHECK(zero_tail<T>(h, ra, qkv, h->nqkv, h->nqkv, 1, st)); }
  { Timed tm_(h, LD_KCLASS_ATTN, st); LD_CHECK(attn_fwd<T>(h, ws, qkv, o, lse, ra, st)); }
  if (ra.seg) {
    Timed tm_(h, LD_KCLASS_ROWWISE, st);
    LD_CHECK(zero_tail<T>(h, ra, o, HD, HD, 1, st));
    LD_CHECK(zero_tail<float>(h, ra, lse, 1, 1, c.H, st));
  }
  a = rows_gemm(h, ra, c.d, HD, o, HD, Wl.w_o, HD, 0);
  a.epi = EPI_RESID;
  a.alpha = s;
  a.x = x;
  a.ldx = c.d;
  a.kept_idx = ra.idx;
  a.S = ra.unit;
  a.save = same_rows ? z : nullptr;  // same rows feed the FFN block: keep a compact copy of Z
  a.ld_save = c.d;
  // with the same rows in both blocks nothing reads x between here and the
  // down projection, which adds into Z's compact copy and writes x itself
  a.x_skip = same_rows ? 1 : 0;
  { Timed tm_(h, LD_KCLASS_GEMM, st); LD_CHECK(gemm<T>(a, st)); }
  if (!same_rows) {  // the FFN block gathers its own rows of Z from the residual stream
    Timed tm_(h, LD_KCLASS_ROWWISE, st);
    LD_CHECK(launch_rmsnorm_fwd<float, T>(x, 1, rf.idx, rf.cnt, rf.unit, c.d, h->max_rows, g2, c.eps, z, zh, rstd2, st));
  } else {
    Timed tm_(h, LD_KCLASS_ROWWISE, st);
    LD_CHECK(launch_rmsnorm_fwd<float, T>(z, 0, ra.idx, ra.cnt, ra.unit, c.d, h->max_rows, g2, c.eps, (float*)nullptr, zh, rstd2, st));
  }
  a = rows_gemm(h, rf, h->nf, c.d, zh, c.d, Wl.w_gu, c.d, 0);
  a.epi = EPI_STORE;
  a.D = gu;
  a.ldd = h->nf;
  if (!f32) {  // h = silu(g) u or max(u, 0)^2 in the projection's epilogue
    a.epi = c.act ? EPI_RELU2 : EPI_SWIGLU;
    a.h_out = hh;
    a.F = c.F;
  }
  { Timed tm_(h, LD_KCLASS_GEMM, st); LD_CHECK(gemm<T>(a, st)); }
  if (f32) {
    Timed tm_(h, LD_KCLASS_ROWWISE, st);
    if (c.act) LD_CHECK(launch_relu2<T>(gu, (const T*)nullptr, hh, rf.cnt, rf.unit, c.F, h->max_rows, st));
    else LD_CHECK(launch_swiglu_fwd<T>(gu, hh, rf.cnt, rf.unit, c.F, h->max_rows, st));
  }
  a = rows_gemm(h, rf, c.d, c.F, hh, c.F, Wl.w_d, c.F, 0);
  a.epi = EPI_RESID;
  a.alpha = s;
  a.x = x;
  a.ldx = c.d;
  a.kept_idx = rf.idx;
  a.S = rf.unit;
  a.save = nullptr;
  if (same_rows) {  // x = Z + s FFN on the kept rows (the O projection left x as it was)
    a.resid_src = z;
    a.ld_src = c.d;
  }
  { Timed tm_(h, LD_KCLASS_GEMM, st); LD_CHECK(gemm<T>(a, st)); }
  return LD_OK;
}

// Work shared by the training and evaluation forwards before the layers:
// clear the status word, widen x into the float32 residual stream (bf16
// path), draw the masks (P) and build the RoPE / ALiBi tables.
template <typename T>
ld_status forward_prologue(Handle* h, const MaskParams& P, void* xv, float* x, void* ws, cudaStream_t st) {
  const ld_config& c = h->cfg;
  const Layout& y = h->lay;
  Timed tm_(h, LD_KCLASS_ROWWISE, st);
  LD_CHECK(cudaMemsetAsync(at<int>(ws, y.status), 0, sizeof(int), st));
  if (sizeof(T) == 2) LD_CHECK(launch_convert(xv, 0, x, 1, (long long)h->max_rows * c.d, st));
  LD_CHECK(launch_mask_compact(P, at<unsigned char>(ws, y.mask), at<int>(ws, y.kidx), at<int>(ws, y.kcnt),
                               at<int>(ws, y.kseg), st));
  if (c.rope_theta != 0.0f)
    LD_CHECK(launch_rope_table(at<float>(ws, y.rcos), at<float>(ws, y.rsin), c.S, c.Dh, (double)c.rope_theta, st));
  if (c.alibi) LD_CHECK(launch_alibi_table(at<float>(ws, y.alibi), c.H, st));
  return LD_OK;
}

MaskParams mask_params(const Handle* h, long long step) {
  MaskParams P;  // 2 KB kernel parameter, filled on the host
  P.seed = h->sched.seed;
  P.step = step;
  P.L = h->cfg.L;
  P.B = h->cfg.B;
  P.S = h->cfg.S;
  P.granularity = h->cfg.granularity;
  P.b_offset = h->cfg.b_offset;
  P.nmask = h->cfg.sublayer ? 2 : 1;
  return P;
}

template <typename T>
ld_status forward_impl(Handle* h, long long step, const ld_layer_w* W, void* xv, void* ws, cudaStream_t st) {
  const ld_config& c = h->cfg;
  const Layout& y = h->lay;
  // The residual stream is carried in float32 through the layers (bf16 in
  // and out at the boundary): 2*L in-place bf16 roundings of X would
  // otherwise accumulate to several per cent of |X| at 32 layers.
  const bool f32 = sizeof(T) == 4;
  float* x = f32 ? static_cast<float*>(xv) : at<float>(ws, y.xres);
  MaskParams P = mask_params(h, step);
  std::vector<float> scale(c.L);
  step_rates(h, step, nullptr, P.thr, scale.data());
  ld_status r = forward_prologue<T>(h, P, xv, x, ws, st);
  if (r != LD_OK) return r;
  for (int l = 0; l < c.L; ++l) {
    // kept rows of the attention block and of the FFN block; the same list
    // unless the masks are drawn per sub-layer
    const Rows ra = rows_of(h, ws, 0, l);
    const Rows rf = c.sublayer ? rows_of(h, ws, 1, l) : ra;
    r = forward_layer<T>(h, ws, at<char>(ws, y.layer0 + (size_t)l * y.per_layer), W[l], x, ra, rf, scale[l], st);
    if (r != LD_OK) return r;
  }
  if (!f32) {
    Timed tm_(h, LD_KCLASS_ROWWISE, st);
    LD_CHECK(launch_convert(x, 1, xv, 0, (long long)h->max_rows * c.d, st));
  }
  h->fwd_scale = scale;
  return LD_OK;
}

// Evaluation forward, Eq. (transformer_layer_dropout_eval): every sequence
// runs every executed layer with the branch scale r_eval[l]; skipped layers
// are not launched.  One block of activations (reused layer after layer)
// and the float32 residual stream at the offsets of the evaluation layout.
template <typename T>
ld_status forward_eval_impl(Handle* h, const unsigned char* execute, const float* r_eval, const ld_layer_w* W,
                            void* xv, void* ws, cudaStream_t st) {
  const ld_config& c = h->cfg;
  const Layout& y = h->lay;
  const bool f32 = sizeof(T) == 4;
  float* x = f32 ? static_cast<float*>(xv) : at<float>(ws, h->eval_xres);
  int* kidx = at<int>(ws, y.kidx);
  int* kcnt = at<int>(ws, y.kcnt);
  MaskParams P = mask_params(h, 0);
  P.nmask = 1;
  P.granularity = LD_PER_SEQUENCE;  // every sequence runs every executed layer whole
  for (int l = 0; l < c.L; ++l) P.thr[l] = 0;  // p = 0: every sequence kept, lists 0 .. B-1
  ld_status r = forward_prologue<T>(h, P, xv, x, ws, st);
  if (r != LD_OK) return r;
  for (int l = 0; l < c.L; ++l) {
    if (!execute[l]) continue;
    Rows ra;
    ra.cnt = kcnt + l;
    ra.idx = kidx + (size_t)l * c.B;
    ra.seg = nullptr;
    ra.unit = c.S;
    r = forward_layer<T>(h, ws, at<char>(ws, y.layer0), W[l], x, ra, ra, r_eval ? r_eval[l] : 1.0f, st);
    if (r != LD_OK) return r;
  }
  if (!f32) {
    Timed tm_(h, LD_KCLASS_ROWWISE, st);
    LD_CHECK(launch_convert(x, 1, xv, 0, (long long)h->max_rows * c.d, st));
  }
  return LD_OK;
}

template <typename T>
ld_status backward_impl(Handle* h, const ld_layer_w* W, void* dxv, ld_layer_g* G, void* ws, cudaStream_t st) {
  const ld_config& c = h->cfg;
  const Layout& y = h->lay;
  const bool f32 = sizeof(T) == 4;
  float* dx = f32 ? static_cast<float*>(dxv) : at<float>(ws, y.dres);  // float32 residual gradient
  float* rcos = at<float>(ws, y.rcos);
  float* rsin = at<float>(ws, y.rsin);
  T* dy = at<T>(ws, y.dy);
  T* dh = at<T>(ws, y.dh);
  T* dgu = at<T>(ws, y.dgu);
  float* dzh = at<float>(ws, y.dzh);
  T* dz = at<T>(ws, y.dz);
  T* dO = at<T>(ws, y.dO);
  T* dqkv = at<T>(ws, y.dqkv);
  float* dxh = at<float>(ws, y.dxh);
  float* Dvec = at<float>(ws, y.Dvec);
  float* part = at<float>(ws, y.part);
  const int HD = c.H * c.Dh;
  if (!f32) {
    Timed tm_(h, LD_KCLASS_ROWWISE, st);
    LD_CHECK(launch_convert(dxv, 0, dx, 1, (long long)h->max_rows * c.d, st));
  }
  // The weight gradients of a layer (dW_d, dW_gu, dW_o, dW_qkv: products
  // 0..3) need nothing from each other or from the data-gradient chain after
  // them, so they run on the side stream, where they fill the last partial
  // wave of the persistent GEMMs on the caller's stream.  Product k waits
  // for its inputs (wg_in[k]); the caller's stream waits for product k
  // (wg_out[k]) before the next layer rewrites its scratch input.
  // With device-time accounting on (ld_set_timing) everything stays on the
  // caller's stream, so that each launch's events time it alone.
  const bool overlap = !h->timing;
  if (overlap) {
    LD_CHECK(ensure_side(h));
    // start every wait of this call from a record on the caller's stream (so
    // that a stream capture never waits on an event recorded outside it)
    for (int k = 0; k < 4; ++k) LD_CHECK(cudaEventRecord(h->wg_out[k], st));
  }
  auto wgrad = [&](int k, const GemmArgs& a) -> cudaError_t {
    if (!overlap) {
      Timed tm_(h, LD_KCLASS_GEMM, st);
      return gemm<T>(a, st);
    }
    cudaError_t e = cudaEventRecord(h->wg_in[k], st);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(h->side, h->wg_in[k], 0);
    if (e != cudaSuccess) return e;
    {
      Timed tm_(h, LD_KCLASS_GEMM, h->side);
      e = gemm<T>(a, h->side);
    }
    if (e == cudaSuccess) e = cudaEventRecord(h->wg_out[k], h->side);
    return e;
  };
  auto before_rewrite = [&](int k) { return overlap ? cudaStreamWaitEvent(st, h->wg_out[k], 0) : cudaSuccess; };

  for (int l = c.L - 1; l >= 0; --l) {
    const Rows ra = rows_of(h, ws, 0, l);  // attention block's kept rows; FFN block's below
    const Rows rf = c.sublayer ? rows_of(h, ws, 1, l) : ra;
    char* lb = at<char>(ws, y.layer0 + (size_t)l * y.per_layer);
    float* xin = reinterpret_cast<float*>(lb + y.xin);
    T* xh = reinterpret_cast<T*>(lb + y.xh);
    T* qkv = reinterpret_cast<T*>(lb + y.qkv);
    T* o = reinterpret_cast<T*>(lb + y.o);
    float* lse = reinterpret_cast<float*>(lb + y.lse);
    float* z = reinterpret_cast<float*>(lb + y.z);
    T* zh = reinterpret_cast<T*>(lb + y.zh);
    T* gu = reinterpret_cast<T*>(lb + y.gu);
    T* hh = reinterpret_cast<T*>(lb + y.h);
    float* rstd1 = reinterpret_cast<float*>(lb + y.rstd1);
    float* rstd2 = reinterpret_cast<float*>(lb + y.rstd2);
    const T* g1 = static_cast<const T*>(W[l].g1);
    const T* g2 = static_cast<const T*>(W[l].g2);
    const float s = h->fwd_scale[l];

    // FFN branch: dy = r * dX^{l+1} on the kept rows.
    LD_CHECK(before_rewrite(0));  // dW_d of the layer above has read dy
    { Timed tm_(h, LD_KCLASS_ROWWISE, st); LD_CHECK(launch_gather_scale<T>(dx, rf.idx, rf.cnt, rf.unit, c.d, h->max_rows, s, dy, st)); }
    LD_CHECK(before_rewrite(1));  // dW_gu of the layer above has read dgu
    GemmArgs a = rows_gemm(h, rf, c.F, c.d, dy, c.d, W[l].w_d, c.F, 1);  // dh = dy W_d
    a.epi = EPI_STORE;
    a.D = dh;
    a.ldd = c.F;
    if (!f32) {  // activation backward in the epilogue: dg, du (or du) straight from dh
      a.epi = c.act ? EPI_RELU2_BWD : EPI_SWIGLU_BWD;
      a.D = dgu;
      a.gu = gu;
      a.F = c.F;
    }
    { Timed tm_(h, LD_KCLASS_GEMM, st); LD_CHECK(gemm<T>(a, st)); }
    if (f32) {
      Timed tm_(h, LD_KCLASS_ROWWISE, st);
      if (c.act) LD_CHECK(launch_relu2<T>(gu, dh, dgu, rf.cnt, rf.unit, c.F, h->max_rows, st));
      else LD_CHECK(launch_swiglu_bwd<T>(dh, gu, dgu, rf.cnt, rf.unit, c.F, h->max_rows, st));
    }
    LD_CHECK(wgrad(0, wgrad_gemm(h, rf, c.d, c.F, dy, c.d, hh, c.F, G[l].w_d)));  // dW_d = dy^T h
    a = rows_gemm(h, rf, c.d, h->nf, dgu, h->nf, W[l].w_gu, c.d, 1);  // dzh = dgu W_gu
    a.epi = EPI_STORE_F32;
    a.D = dzh;
    a.ldd = c.d;
    { Timed tm_(h, LD_KCLASS_GEMM, st); LD_CHECK(gemm<T>(a, st)); }
    LD_CHECK(wgrad(1, wgrad_gemm(h, rf, h->nf, c.d, dgu, h->nf, zh, c.d, G[l].w_gu)));  // dW_gu = dgu^T zh
    // dZ = dX^{l+1} + RMSNorm_2 backward; dz = r * dZ for the attention branch
    // (written by the same kernel when both blocks keep the same rows)
    LD_CHECK(before_rewrite(2));  // dW_o of the layer above has read dz
    {
      Timed tm_(h, LD_KCLASS_ROWWISE, st);
      LD_CHECK(launch_rmsnorm_bwd<T>(dzh, z, rstd2, g2, dx, rf.idx, rf.cnt, rf.unit, c.d, h->max_rows, s,
                                     c.sublayer ? (T*)nullptr : dz, part, h->part_blocks, st));
    }
    { Timed tm_(h, LD_KCLASS_ROWWISE, st); LD_CHECK(launch_colsum(part, h->part_blocks, c.d, G[l].g2, st)); }
    if (c.sublayer) { Timed tm_(h, LD_KCLASS_ROWWISE, st); LD_CHECK(launch_gather_scale<T>(dx, ra.idx, ra.cnt, ra.unit, c.d, h->max_rows, s, dz, st)); }
    // attention branch
    a = rows_gemm(h, ra, HD, c.d, dz, c.d, W[l].w_o, HD, 1);  // dO = dz W_o
    a.epi = EPI_STORE;
    a.D = dO;
    a.ldd = HD;
    { Timed tm_(h, LD_KCLASS_GEMM, st); LD_CHECK(gemm<T>(a, st)); }
    if (ra.seg) { Timed tm_(h, LD_KCLASS_ROWWISE, st); LD_CHECK(zero_tail<T>(h, ra, dO, HD, HD, 1, st)); }
    LD_CHECK(wgrad(2, wgrad_gemm(h, ra, c.d, HD, dz, c.d, o, HD, G[l].w_o)));  // dW_o = dz^T o
    LD_CHECK(before_rewrite(3));  // dW_qkv of the layer above has read dqkv
    { Timed tm_(h, LD_KCLASS_ATTN, st); LD_CHECK(attn_bwd<T>(h, ws, qkv, o, dO, lse, Dvec, dqkv, ra, st)); }
    if (ra.seg) { Timed tm_(h, LD_KCLASS_ROWWISE, st); LD_CHECK(zero_tail<T>(h, ra, dqkv, h->nqkv, h->nqkv, 1, st)); }
    a = rows_gemm(h, ra, c.d, h->nqkv, dqkv, h->nqkv, W[l].w_qkv, c.d, 1);  // dxh = dqkv W_qkv
    a.epi = EPI_STORE_F32;
    a.D = dxh;
    a.ldd = c.d;
    { Timed tm_(h, LD_KCLASS_GEMM, st); LD_CHECK(gemm<T>(a, st)); }
    LD_CHECK(wgrad(3, wgrad_gemm(h, ra, h->nqkv, c.d, dqkv, h->nqkv, xh, c.d, G[l].w_qkv)));  // dW_qkv = dqkv^T xh
    // dX^l = dZ + RMSNorm_1 backward
    {
      Timed tm_(h, LD_KCLASS_ROWWISE, st);
      LD_CHECK(launch_rmsnorm_bwd<T>(dxh, xin, rstd1, g1, dx, ra.idx, ra.cnt, ra.unit, c.d, h->max_rows, 1.0f,
                                     (T*)nullptr, part, h->part_blocks, st));
    }
    { Timed tm_(h, LD_KCLASS_ROWWISE, st); LD_CHECK(launch_colsum(part, h->part_blocks, c.d, G[l].g1, st)); }
  }
  if (!f32) {
    Timed tm_(h, LD_KCLASS_ROWWISE, st);
    LD_CHECK(launch_convert(dx, 1, dxv, 0, (long long)h->max_rows * c.d, st));
  }
  for (int k = 0; k < 4; ++k) LD_CHECK(before_rewrite(k));  // join: every weight gradient is done
  return LD_OK;
}

}  // namespace

extern "C" {

const char* ld_last_cuda_error(void) {
  return g_last_cuda == cudaSuccess ? "no CUDA error recorded" : cudaGetErrorString(g_last_cuda);
}

const char* ld_status_str(ld_status s) {
  switch (s) {
    case LD_OK: return "ok";
    case LD_ERR_ARG: return "invalid argument";
    case LD_ERR_SHAPE: return "unsupported shape";
    case LD_ERR_STATE: return "call out of order";
    case LD_ERR_CUDA: return "CUDA error";
    case LD_ERR_TIMEOUT: return "device-side wait timed out";
    case LD_ERR_OOM: return "out of host memory";
    case LD_ERR_UNSUPPORTED: return "unsupported device or build";
  }
  return "unknown status";
}

ld_status ld_create(const ld_config* cfg, void** handle) {
  if (!cfg || !handle) return LD_ERR_ARG;
  *handle = nullptr;
  const ld_config& c = *cfg;
  if (!finite(c.eps) || !finite(c.alpha) || !finite(c.rope_theta) || c.eps < 0.0f || c.rope_theta < 0.0f)
    return LD_ERR_ARG;
  if (c.L < 1 || c.L > LD_MAX_L || c.B < 1 || c.B > LD_MAX_B || c.S < 64 || c.S > 16384 || c.S % 64) return LD_ERR_SHAPE;
  if (c.d < 64 || c.d % 64 || c.F < 64 || c.F % 64 || c.d > 16384) return LD_ERR_SHAPE;
  if (c.Dh != 32 && c.Dh != 64 && c.Dh != 128) return LD_ERR_SHAPE;
  if (c.H < 1 || c.Hkv < 1 || c.H % c.Hkv || (c.H * c.Dh) % 64) return LD_ERR_SHAPE;
  if (c.granularity != LD_PER_SEQUENCE && c.granularity != LD_PER_BATCH && c.granularity != LD_PER_SHARD &&
      c.granularity != LD_PER_TOKEN)
    return LD_ERR_ARG;
  if (c.sublayer != 0 && c.sublayer != 1) return LD_ERR_ARG;
  if (c.alibi != 0 && c.alibi != 1) return LD_ERR_ARG;
  if (c.alibi && c.rope_theta != 0.0f) return LD_ERR_ARG;  // one position scheme
  if (c.granularity == LD_PER_TOKEN) {
    // the ALiBi distance would need the kept tokens' original positions in
    // the attention kernels; the bf16 path runs its per-token attention on
    // the tcgen05 kernels only (head size 64 or 128, S % 128 == 0)
    if (c.alibi) return LD_ERR_ARG;
    if (!c.fp32_debug && (c.Dh < 64 || c.S % 128)) return LD_ERR_SHAPE;
  }
  if (c.act != LD_ACT_SWIGLU && c.act != LD_ACT_RELU2) return LD_ERR_ARG;
  if (c.b_offset < 0 || (long long)c.b_offset + c.B > 0x7fffffffll) return LD_ERR_ARG;
  if ((long long)c.B * c.S > (1ll << 30)) return LD_ERR_SHAPE;
  Handle* h = new (std::nothrow) Handle();
  if (!h) return LD_ERR_OOM;
  h->cfg = c;
  h->esz = c.fp32_debug ? 4 : 2;
  h->max_rows = c.B * c.S;
  h->nqkv = (c.H + 2 * c.Hkv) * c.Dh;
  h->nf = c.act == LD_ACT_RELU2 ? c.F : 2 * c.F;
  // number of blocks (and partial-sum rows of the gain gradient) of the
  // RMSNorm backward inside ld_backward: the two blocks per SM of a 152-SM
  // GPU that its register use lets stay resident, each looping over rows
  // (a launch constant; no CUDA call here)
  h->part_blocks = (h->max_rows + 7) / 8;
  if (h->part_blocks > 2 * 152) h->part_blocks = 2 * 152;
  make_layout(h);
  *handle = h;
  return LD_OK;
}

ld_status ld_workspace_size(void* handle, size_t* bytes) {
  if (!handle || !bytes) return LD_ERR_ARG;
  *bytes = H(handle)->lay.total;
  return LD_OK;
}

ld_status ld_set_schedule(void* handle, const ld_schedule* s) {
  if (!handle || !s) return LD_ERR_ARG;
  Handle* h = H(handle);
  if (s->dist < LD_DIST_UNIFORM || s->dist > LD_DIST_EXPLICIT) return LD_ERR_ARG;
  if (s->time < LD_TIME_CONST || s->time > LD_TIME_RAMP) return LD_ERR_ARG;
  if (!(s->p_max >= 0.0f && s->p_max <= 1.0f)) return LD_ERR_ARG;
  if ((s->time == LD_TIME_ITS || s->time == LD_TIME_DTS) && s->T < 2) return LD_ERR_ARG;
  if (s->time == LD_TIME_RAMP && (s->ramp_t1 <= s->ramp_t0 || !finite(s->ramp_s0) || !finite(s->ramp_s1)))
    return LD_ERR_ARG;
  std::vector<float> pe;
  if (s->dist == LD_DIST_EXPLICIT) {
    if (!s->p_explicit) return LD_ERR_ARG;
    pe.assign(s->p_explicit, s->p_explicit + h->cfg.L);
    for (float v : pe)
      if (!(v >= 0.0f && v <= 1.0f)) return LD_ERR_ARG;
  }
  h->sched = *s;
  h->sched.p_explicit = nullptr;
  h->p_expl.swap(pe);
  h->have_sched = true;
  return LD_OK;
}

ld_status ld_get_rates(void* handle, long long step, double* p, unsigned long long* thr, float* scale) {
  if (!handle) return LD_ERR_ARG;
  Handle* h = H(handle);
  if (!h->have_sched) return LD_ERR_STATE;
  step_rates(h, step, p, thr, scale);
  return LD_OK;
}

ld_status ld_draw_masks(void* handle, long long step, void* ws, void* stream) {
  if (!handle || !ws || !aligned16(ws)) return LD_ERR_ARG;
  Handle* h = H(handle);
  if (!h->have_sched) return LD_ERR_STATE;
  const Layout& y = h->lay;
  MaskParams P = mask_params(h, step);
  step_rates(h, step, nullptr, P.thr, nullptr);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  LD_CHECK(cudaMemsetAsync(at<int>(ws, y.status), 0, sizeof(int), st));
  LD_CHECK(launch_mask_compact(P, at<unsigned char>(ws, y.mask), at<int>(ws, y.kidx), at<int>(ws, y.kcnt),
                               at<int>(ws, y.kseg), st));
  h->last_ws = ws;
  h->last_stream = st;
  h->have_masks = true;
  return LD_OK;
}

ld_status ld_forward(void* handle, long long step, const ld_layer_w* W, void* x, void* ws, void* stream) {
  if (!handle || !x || !ws || !aligned16(x) || !aligned16(ws)) return LD_ERR_ARG;
  Handle* h = H(handle);
  if (!h->have_sched) return LD_ERR_STATE;
  ld_status r = check_weights(h, W);
  if (r != LD_OK) return r;
  if (!h->cfg.fp32_debug && (r = check_device()) != LD_OK) return r;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  h->fwd_valid = false;
  r = h->cfg.fp32_debug ? forward_impl<float>(h, step, W, x, ws, st) : forward_impl<bf16>(h, step, W, x, ws, st);
  h->last_ws = ws;
  h->last_stream = st;
  h->have_masks = true;
  if (r == LD_OK) {
    h->fwd_valid = true;
    h->fwd_ws = ws;
  }
  return r;
}

ld_status ld_eval_workspace_size(void* handle, size_t* bytes) {
  if (!handle || !bytes) return LD_ERR_ARG;
  *bytes = H(handle)->eval_total;
  return LD_OK;
}

ld_status ld_forward_eval(void* handle, const unsigned char* execute, const float* r_eval, const ld_layer_w* W,
                          void* x, void* ws, void* stream) {
  if (!handle || !execute || !W || !x || !ws || !aligned16(x) || !aligned16(ws)) return LD_ERR_ARG;
  Handle* h = H(handle);
  for (int l = 0; l < h->cfg.L; ++l) {
    if (execute[l] > 1) return LD_ERR_ARG;
    if (r_eval && !finite(r_eval[l])) return LD_ERR_ARG;
    if (!execute[l]) continue;  // the weights of skipped layers are never read
    const void* ps[6] = {W[l].w_qkv, W[l].w_o, W[l].w_gu, W[l].w_d, W[l].g1, W[l].g2};
    for (const void* p : ps)
      if (!p || !aligned16(p)) return LD_ERR_ARG;
  }
  ld_status r = LD_OK;
  if (!h->cfg.fp32_debug && (r = check_device()) != LD_OK) return r;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  r = h->cfg.fp32_debug ? forward_eval_impl<float>(h, execute, r_eval, W, x, ws, st)
                        : forward_eval_impl<bf16>(h, execute, r_eval, W, x, ws, st);
  h->last_ws = ws;
  h->last_stream = st;
  h->have_masks = false;  // the workspace holds no training masks now
  h->fwd_valid = false;   // nor a forward a backward could follow
  return r;
}

ld_status ld_backward(void* handle, const ld_layer_w* W, void* dx, ld_layer_g* G, void* ws, void* stream) {
  if (!handle || !dx || !ws || !G || !aligned16(dx)) return LD_ERR_ARG;
  Handle* h = H(handle);
  ld_status r = check_weights(h, W);
  if (r != LD_OK) return r;
  for (int l = 0; l < h->cfg.L; ++l) {
    float* ps[6] = {G[l].w_qkv, G[l].w_o, G[l].w_gu, G[l].w_d, G[l].g1, G[l].g2};
    for (float* p : ps)
      if (!p || !aligned16(p)) return LD_ERR_ARG;
  }
  if (!h->fwd_valid || h->fwd_ws != ws) return LD_ERR_STATE;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  r = h->cfg.fp32_debug ? backward_impl<float>(h, W, dx, G, ws, st) : backward_impl<bf16>(h, W, dx, G, ws, st);
  h->last_ws = ws;
  h->last_stream = st;
  return r;
}

ld_status ld_get_masks(void* handle, unsigned char* mask, int* kept_idx, int* kept_cnt) {
  if (!handle) return LD_ERR_ARG;
  Handle* h = H(handle);
  if (!h->have_masks) return LD_ERR_STATE;
  const Layout& y = h->lay;
  const ld_config& c = h->cfg;
  const bool tokg = c.granularity == LD_PER_TOKEN;
  const size_t nm = c.sublayer ? 2 : 1;
  const size_t LB = nm * c.L * (tokg ? (size_t)c.B * c.S : (size_t)c.B);
  LD_CHECK(cudaStreamSynchronize(h->last_stream));
  if (mask) LD_CHECK(cudaMemcpy(mask, at<unsigned char>(h->last_ws, y.mask), LB, cudaMemcpyDeviceToHost));
  if (kept_idx) LD_CHECK(cudaMemcpy(kept_idx, at<int>(h->last_ws, y.kidx), LB * 4, cudaMemcpyDeviceToHost));
  if (kept_cnt && !tokg)
    LD_CHECK(cudaMemcpy(kept_cnt, at<int>(h->last_ws, y.kcnt), nm * c.L * 4, cudaMemcpyDeviceToHost));
  if (kept_cnt && tokg) {  // the kept-token counts: the last segment offset of each table
    std::vector<int> seg(nm * c.L * (c.B + 1));
    LD_CHECK(cudaMemcpy(seg.data(), at<int>(h->last_ws, y.kseg), seg.size() * 4, cudaMemcpyDeviceToHost));
    for (size_t i = 0; i < nm * c.L; ++i) kept_cnt[i] = seg[i * (c.B + 1) + c.B];
  }
  return LD_OK;
}

ld_status ld_sync(void* handle) {
  if (!handle) return LD_ERR_ARG;
  Handle* h = H(handle);
  if (!h->last_ws) return LD_OK;
  LD_CHECK(cudaStreamSynchronize(h->last_stream));
  LD_CHECK(cudaGetLastError());
  int st = 0;
  int* sw = at<int>(h->last_ws, h->lay.status);
  LD_CHECK(cudaMemcpy(&st, sw, sizeof(int), cudaMemcpyDeviceToHost));
  if (st) LD_CHECK(cudaMemset(sw, 0, sizeof(int)));
  return st ? (ld_status)st : LD_OK;
}

ld_status ld_destroy(void* handle) {
  if (!handle) return LD_ERR_ARG;
  delete H(handle);
  return LD_OK;
}

ld_status ld_set_timing(void* handle, int enable) {
  if (!handle) return LD_ERR_ARG;
  Handle* h = H(handle);
  h->timing = enable != 0;
  for (auto& u : h->ev_used) u = 0;
  return LD_OK;
}

ld_status ld_get_timing(void* handle, int kclass, double* ms, long long* launches) {
  if (!handle || kclass < 0 || kclass >= LD_KCLASS_COUNT) return LD_ERR_ARG;
  Handle* h = H(handle);
  const size_t pairs = h->ev_used[kclass] / 2;
  double tot = 0.0;
  for (size_t i = 0; i < pairs; ++i) {
    float t = 0.f;
    LD_CHECK(cudaEventSynchronize(h->ev[kclass][2 * i + 1]));
    LD_CHECK(cudaEventElapsedTime(&t, h->ev[kclass][2 * i], h->ev[kclass][2 * i + 1]));
    tot += t;
  }
  if (ms) *ms = tot;
  if (launches) *launches = (long long)pairs;
  return LD_OK;
}

ld_status ld_rmsnorm_backward(int B, int S, int d, const float* dyn, const void* xs, const float* rstd,
                              const void* gamma, const int* kept_idx, const int* kept_cnt, float* dx, void* next,
                              float scale, float* dgamma, float* scratch, size_t scratch_bytes, void* stream) {
  if (B < 1 || S < 1 || d < 8 || d % 8 || d > 16384 || (long long)B * S > (1ll << 30)) return LD_ERR_SHAPE;
  const void* ps[] = {dyn, xs, rstd, gamma, dx, dgamma, scratch};
  for (const void* p : ps)
    if (!p || !aligned16(p)) return LD_ERR_ARG;
  if (!kept_idx || !kept_cnt || (next && !aligned16(next))) return LD_ERR_ARG;
  long long nb = ((long long)B * S + 7) / 8;
  if (nb > 320) nb = 320;
  if (scratch_bytes < (size_t)nb * d * sizeof(float)) return LD_ERR_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  LD_CHECK(launch_rmsnorm_bwd<bf16>(dyn, static_cast<const float*>(xs), rstd, static_cast<const bf16*>(gamma), dx,
                                    kept_idx, kept_cnt, S, d, B * S, scale, static_cast<bf16*>(next), scratch,
                                    (int)nb, st));
  LD_CHECK(launch_colsum(scratch, (int)nb, d, dgamma, st));
  return LD_OK;
}

ld_status ld_gemm_bf16(int M, int N, int K, const void* A, int lda, int a_mn, const void* B, int ldb, int b_mn, void* D,
                       int ldd, int d_f32, float alpha, int* status_ws, void* stream) {
  if (!A || !B || !D || !aligned16(A) || !aligned16(B) || !aligned16(D)) return LD_ERR_ARG;
  if (M < 64 || N < 64 || K < 0 || M % 64 || N % 64 || K % 64) return LD_ERR_SHAPE;
  if (lda % 8 || ldb % 8 || ldd % 8) return LD_ERR_SHAPE;
  if (lda < (a_mn ? M : K) || ldb < (b_mn ? N : K) || ldd < N) return LD_ERR_SHAPE;
  ld_status r = check_device();
  if (r != LD_OK) return r;
  GemmArgs a = gemm_base();
  a.M = M;
  a.N = N;
  a.K = K;
  a.A = A;
  a.lda = lda;
  a.a_mn = a_mn ? 1 : 0;
  a.B = B;
  a.ldb = ldb;
  a.b_mn = b_mn ? 1 : 0;
  a.epi = d_f32 ? EPI_STORE_F32 : EPI_STORE;
  a.D = D;
  a.ldd = ldd;
  a.alpha = alpha;
  a.status = status_ws;
  LD_CHECK(gemm_tc(a, static_cast<cudaStream_t>(stream)));
  return LD_OK;
}

ld_status ld_check_wait_timeout(int* status_ws, void* stream) {
  if (!status_ws) return LD_ERR_ARG;
  ld_status r = check_device();
  if (r != LD_OK) return r;
  LD_CHECK(launch_wait_timeout(status_ws, static_cast<cudaStream_t>(stream)));
  return LD_OK;
}

}  // extern "C"
