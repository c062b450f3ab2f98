// C ABI of the library (include/proxyformer.h): argument validation,
// workspace / saved-buffer planning and the launch sequence of one layer.
#include <stdarg.h>
#include <stdio.h>

#include <algorithm>
#include <string>
#include <array>
#include <vector>

#include "kernels.h"
#include "proxyformer.h"

using namespace pf;

namespace {

thread_local std::string g_msg;

pf_status fail(pf_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_msg = buf;
  return s;
}

#define PF_CUDA(call)                                                                 \
  do {                                                                                \
    cudaError_t e_ = (call);                                                          \
    if (e_ != cudaSuccess) return fail(PF_ERR_CUDA, "%s: %s", #call, cudaGetErrorString(e_)); \
  } while (0)

// Sub-allocator over a caller buffer: 256-byte aligned slices.
struct Carve {
  char* base;
  size_t off = 0;
  explicit Carve(void* p) : base(static_cast<char*>(p)) {}
  template <class T>
  T* take(size_t n) {
    off = (off + 255) & ~size_t(255);
    T* p = base ? reinterpret_cast<T*>(base + off) : nullptr;
    off += n * sizeof(T);
    return p;
  }
};

// Derived sizes of a validated 1D / 2D layer.
struct Dims {
  long B, L, d, df, nh, P, k1, k2, m, R, rows1, N1, Lp;  // d: proxy width, df: token width
  long T, ldq;  // tokens B*L; width of the token-query matrix [Q | gate | 0] (cross)
  bool causal, ragged, cross;
  int f;      // proxy interaction: PF_F_ATTENTION / PF_F_IDENTITY / PF_F_MLP
  bool rope;  // RoPE on the proxies' queries and keys
};

Dims dims_of(const pf_layer_desc& s) {
  Dims g;
  g.B = s.batch;
  g.L = s.L;
  g.d = s.d;
  g.df = s.d_fine > 0 ? s.d_fine : s.d;
  g.nh = s.n_heads;
  g.P = s.P;
  g.k1 = s.levels == 2 ? s.k1 : s.P;
  g.k2 = s.levels == 2 ? s.k2 : 1;
  g.m = (g.L + g.P - 1) / g.P;
  g.R = g.B * g.m;
  g.rows1 = g.R * g.k2;
  g.N1 = g.k1 * g.df;
  g.Lp = g.m * g.P;
  g.causal = s.mode == PF_CAUSAL_1D;
  g.ragged = g.Lp != g.L;
  g.cross = s.inject == PF_INJ_CROSS;
  g.f = s.interact;
  g.rope = s.rope != 0;
  g.T = g.B * g.L;
  g.ldq = g.d + 64;  // the gate's n_heads <= 64 rows, zero-padded to 64
  return g;
}

// Largest split-K scratch needed by the layer's linear GEMMs (forward or
// backward); the GEMM shapes below mirror the launch sequence.
size_t splitk_need(const pf_layer_desc& s, const Dims& g, bool bwd) {
  const int d = (int)g.d, R = (int)g.R, r1 = (int)g.rows1, N1 = (int)g.N1, n2 = (int)(g.k2 * d);
  struct S3 {
    int M, N, K;
  };
  std::vector<S3> v;
  if (s.mode == PF_BIDIR_2D) {
    if (!bwd) v = {{R, d, N1}, {R, 3 * d, d}, {R, d, d}};
    else v = {{2 * N1, d, R}, {R, d, 2 * N1}, {d, d, R}, {R, d, d}, {3 * d, d, R}, {R, d, 3 * d},
              {d, N1, R}};
  } else if (!bwd) {
    v = {{R, 3 * d, d}, {R, d, d}};
    if (s.levels == 1) v.push_back({R, d, N1});
    else v.insert(v.end(), {{r1, d, N1}, {R, d, n2}, {R, n2, d}});
  } else {
    v = {{N1, d, r1}, {r1, d, N1}, {d, d, R}, {R, d, d}, {3 * d, d, R}, {R, d, 3 * d}, {d, N1, r1}};
    if (s.levels == 2) v.insert(v.end(), {{n2, d, R}, {R, d, n2}, {d, n2, R}, {R, n2, d}});
  }
  if (g.f == PF_F_MLP) {  // the single-proxy MLP and its backward
    if (!bwd) v.insert(v.end(), {{R, 4 * d, d}, {R, d, 4 * d}});
    else v.insert(v.end(), {{d, 4 * d, R}, {R, 4 * d, d}, {4 * d, d, R}, {R, d, 4 * d}});
  }
  if (g.cross) {  // token queries + gate, proxy keys / values, output projection
    const int T = (int)g.T, q = (int)g.ldq, nh = (int)g.nh;
    if (!bwd) v.insert(v.end(), {{T, q, d}, {R, 2 * d, d}, {T, d, d}});
    else v.insert(v.end(), {{d, d, T}, {T, d, d}, {d + nh, d, T}, {2 * d, d, R}, {R, d, 2 * d},
                            {T, d, q}});
  }
  size_t m = 0;
  for (const S3& x : v) m = std::max(m, splitk_scratch_bytes(x.M, x.N, x.K));
  return m;
}

EpiLinearArgs with_sk(EpiLinearArgs e, float* sk, size_t skb) {
  e.splitk_scratch = sk;
  e.splitk_bytes = skb;
  return e;
}

// W_qa [d + nh, d] copied into a [ldq, d] buffer whose extra rows are zero,
// so the token-query GEMM writes whole 64-column groups and its transpose
// reads only zeros past the gate rows.
cudaError_t pad_qa(const void* W_qa, bf16* dst, const Dims& g, cudaStream_t cs) {
  const size_t live = (size_t)(g.d + g.nh) * g.d;
  cudaError_t e = cudaMemcpyAsync(dst, W_qa, live * sizeof(bf16), cudaMemcpyDeviceToDevice, cs);
  if (e != cudaSuccess) return e;
  return cudaMemsetAsync(dst + live, 0, ((size_t)g.ldq * g.d - live) * sizeof(bf16), cs);
}

// Buffers the forward saves for the backward pass (order fixes the layout).
struct Saved {
  bf16 *Hb, *QKV, *Aatt, *Hbar, *Y, *Z, *D;
  float* LSE;
  // cross injection: [Q | gate] of the tokens, proxy K | V, attention output
  // ungated and gated, its LSE
  bf16 *QA, *KVx, *Ax, *Ag;
  float* LSEx;
  bf16 *U, *Am;  // single-proxy MLP: pre-activation and SiLU of its hidden layer
};

Saved carve_saved(Carve& c, const pf_layer_desc& s, const Dims& g) {
  Saved v{};
  v.Hb = c.take<bf16>(g.R * g.d);
  if (g.f == PF_F_ATTENTION) {
    v.QKV = c.take<bf16>(g.R * 3 * g.d);
    v.Aatt = c.take<bf16>(g.R * g.d);
  }
  v.Hbar = c.take<bf16>(g.R * g.d);
  if (g.f == PF_F_ATTENTION) v.LSE = c.take<float>(g.B * g.nh * g.m);
  if (g.f == PF_F_MLP) {
    v.U = c.take<bf16>(g.R * 4 * g.d);
    v.Am = c.take<bf16>(g.R * 4 * g.d);
  }
  if (s.levels == 2) v.Y = c.take<bf16>(g.rows1 * g.d);
  if (g.cross) {
    v.QA = c.take<bf16>(g.T * g.ldq);
    v.KVx = c.take<bf16>(g.R * 2 * g.d);
    v.Ax = c.take<bf16>(g.T * g.d);
    v.Ag = c.take<bf16>(g.T * g.d);
    v.LSEx = c.take<float>(g.B * g.nh * g.L);
    return v;
  }
  if (s.levels == 2) v.Z = c.take<bf16>(g.R * g.k2 * g.d);
  v.D = c.take<bf16>(g.rows1 * g.N1);
  return v;
}

// The bf16 forward's workspace: padded copy of a ragged X, split-K partials,
// and the saved activations (in `saved` when given, else here).
struct FwdWs {
  bf16* Xpad;
  float* sk;
  size_t skb;
  bf16* Wqa;     // cross: W_qa zero-padded to [d + 64, d]
  float2* rtab;  // RoPE: (cos, sin) per proxy position and pair [m, 32]
  Saved sv;
};

FwdWs carve_fwd(Carve& wc, const pf_layer_desc& s, const Dims& g, void* saved) {
  FwdWs f{};
  f.Xpad = g.ragged ? wc.take<bf16>(g.B * g.Lp * g.df) : nullptr;
  f.skb = splitk_need(s, g, false);
  f.sk = wc.take<float>(f.skb / sizeof(float));
  if (g.cross) f.Wqa = wc.take<bf16>(g.ldq * g.d);
  if (g.rope) f.rtab = wc.take<float2>(g.m * 32);
  Carve sc(saved);
  f.sv = saved ? carve_saved(sc, s, g) : carve_saved(wc, s, g);
  return f;
}

struct BwdWs {
  bf16 *Xpad, *dXpad, *dD, *dZ, *dHbar, *dA, *dQKV, *dHb, *dY;
  float *Di, *dHf, *part, *sk;
  long part_elems;
  size_t skb;
  // cross injection: padded W_qa, dL/d(alpha A), dL/dA, [dQ | d gate | 0],
  // proxy dK | dV, gate pre-activation gradient (fp32), Di of the tokens
  bf16 *Wqa, *dAg, *dOx, *dQA, *dKVx;
  float *ga, *gsum, *Dix;  // ga: [T, ldga], columns past n_heads zero
  int ldga;
  bf16* dU;      // single-proxy MLP: gradient of the hidden pre-activation
  float2* rtab;  // RoPE angle table [m, 32]
};

BwdWs carve_bwd(Carve& c, const pf_layer_desc& s, const Dims& g) {
  BwdWs w{};
  w.Xpad = g.ragged ? c.take<bf16>(g.B * g.Lp * g.df) : nullptr;
  w.dXpad = g.ragged ? c.take<bf16>(g.B * g.Lp * g.df) : nullptr;
  if (g.cross) {
    w.Wqa = c.take<bf16>(g.ldq * g.d);
    w.dAg = c.take<bf16>(g.T * g.d);
    w.dOx = c.take<bf16>(g.T * g.d);
    w.dQA = c.take<bf16>(g.T * g.ldq);
    w.dKVx = c.take<bf16>(g.R * 2 * g.d);
    w.ldga = (int)((g.nh + 7) & ~7L);  // whole 8-column groups for the column sum
    w.ga = c.take<float>(g.T * w.ldga);
    w.gsum = c.take<float>(w.ldga);
    w.Dix = c.take<float>(g.B * g.nh * g.L);
  } else {
    w.dD = c.take<bf16>(g.rows1 * g.N1);
    if (s.levels == 2) w.dZ = c.take<bf16>(g.R * g.k2 * g.d);
  }
  w.dHbar = c.take<bf16>(g.R * g.d);
  if (g.f == PF_F_ATTENTION) {
    w.dA = c.take<bf16>(g.R * g.d);
    w.dQKV = c.take<bf16>(g.R * 3 * g.d);
  }
  if (g.f == PF_F_MLP) w.dU = c.take<bf16>(g.R * 4 * g.d);
  if (g.rope) w.rtab = c.take<float2>(g.m * 32);
  w.dHb = c.take<bf16>(g.R * g.d);
  if (s.levels == 2) w.dY = c.take<bf16>(g.rows1 * g.d);
  w.Di = c.take<float>(g.B * g.nh * g.m);
  w.dHf = c.take<float>(g.R * g.d);
  long pe = (long)inj_bwd_chunks(g.rows1, (int)g.N1) * 4 * g.N1;
  pe = std::max(pe, colsum_part_elems(g.R, (int)(g.k2 * g.d)));
  pe = std::max(pe, colsum_part_elems(g.R, (int)g.d));
  pe = std::max(pe, colsum_part_elems(g.rows1, (int)g.d));
  if (g.cross) pe = std::max(pe, colsum_part_elems(g.T, (int)((g.nh + 7) & ~7L)));
  if (g.f == PF_F_MLP) pe = std::max(pe, colsum_part_elems(g.R, (int)(4 * g.d)));
  w.part_elems = pe;
  w.part = c.take<float>(pe);
  w.skb = splitk_need(s, g, true);
  w.sk = c.take<float>(w.skb / sizeof(float));
  return w;
}

// Saved buffer of the 2D layer (order fixes the layout).
struct Saved2D {
  bf16 *Xp, *S, *Hb, *QKV, *Aatt, *Hbar;
  float *stats, *nH, *rstdH, *LSE, *e, *a1, *u, *gb;
};

Saved2D carve_saved_2d(Carve& c, const Dims& g) {
  Saved2D v{};
  const long T = g.B * g.L;
  v.Xp = c.take<bf16>(g.R * g.N1);
  v.stats = c.take<float>(2 * T);
  v.S = c.take<bf16>(g.R * g.N1);
  v.nH = c.take<float>(g.R * g.d);
  v.rstdH = c.take<float>(g.R);
  v.Hb = c.take<bf16>(g.R * g.d);
  v.QKV = c.take<bf16>(g.R * 3 * g.d);
  v.Aatt = c.take<bf16>(g.R * g.d);
  v.Hbar = c.take<bf16>(g.R * g.d);
  v.LSE = c.take<float>(g.B * g.nh * g.m);
  v.e = c.take<float>(g.B * 256);
  v.a1 = c.take<float>(g.B * g.d);
  v.u = c.take<float>(g.B * g.d);
  v.gb = c.take<float>(g.B * 2 * g.d);
  return v;
}

struct Bwd2DWs {
  bf16 *dD, *dXd, *dHbar, *dA, *dQKV, *dHb;
  float *Di, *dHq, *dHf, *part, *dgb, *da1, *sk;
  size_t skb;
};

Bwd2DWs carve_bwd_2d(Carve& c, const pf_layer_desc& s, const Dims& g) {
  Bwd2DWs w{};
  w.dD = c.take<bf16>(g.R * 2 * g.N1);
  w.dXd = c.take<bf16>(g.R * g.N1);
  w.dHbar = c.take<bf16>(g.R * g.d);
  w.dA = c.take<bf16>(g.R * g.d);
  w.dQKV = c.take<bf16>(g.R * 3 * g.d);
  w.dHb = c.take<bf16>(g.R * g.d);
  w.Di = c.take<float>(g.B * g.nh * g.m);
  w.dHq = c.take<float>(g.R * g.d);
  w.dHf = c.take<float>(g.R * g.d);
  long pe = inj_bwd_2d_part_elems(g.R, (int)g.d, s.patch);
  pe = std::max(pe, colsum_part_elems(g.R, (int)g.d));
  pe = std::max(pe, (long)g.B * adaln_param_chunks((int)g.m) * 2 * g.d);
  w.part = c.take<float>(pe);
  w.dgb = c.take<float>(g.B * 2 * g.d);
  w.da1 = c.take<float>(g.B * g.d);
  w.skb = splitk_need(s, g, true);
  w.sk = c.take<float>(w.skb / sizeof(float));
  return w;
}

// Workspace of the fp32 forward (all fp32).
struct F32Ws {
  float *Xpad, *Y, *H, *QKV, *A, *Hbar, *Z, *D, *sk;
  size_t skb;
};

size_t splitk_f32_need(const pf_layer_desc& s, const Dims& g) {
  const int d = (int)g.d, R = (int)g.R, r1 = (int)g.rows1, N1 = (int)g.N1, n2 = (int)(g.k2 * d);
  const int shapes[][3] = {{s.levels == 1 ? R : r1, d, N1}, {R, d, n2},   {R, 3 * d, d},
                           {R, d, d},                        {R, n2, d},   {r1, N1, d}};
  size_t m = 0;
  for (const auto& x : shapes)
    m = std::max(m, (size_t)splitk_f32_factor(x[0], x[1], x[2]) * x[0] * x[1] * sizeof(float));
  return m;
}

F32Ws carve_f32(Carve& c, const pf_layer_desc& s, const Dims& g) {
  F32Ws w{};
  w.Xpad = g.ragged ? c.take<float>(g.B * g.Lp * g.d) : nullptr;
  if (s.levels == 2) w.Y = c.take<float>(g.rows1 * g.d);
  w.H = c.take<float>(g.R * g.d);
  w.QKV = c.take<float>(g.R * 3 * g.d);
  w.A = c.take<float>(g.R * g.d);
  w.Hbar = c.take<float>(g.R * g.d);
  if (s.levels == 2) w.Z = c.take<float>(g.R * g.k2 * g.d);
  w.D = c.take<float>(g.rows1 * g.N1);
  w.skb = splitk_f32_need(s, g);
  w.sk = c.take<float>(w.skb / sizeof(float));
  return w;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

bool params_aligned(const pf_layer_params& p) {
  const void* ptrs[] = {p.W_c1, p.b_c1, p.W_c2,  p.b_c2, p.W_qkv, p.W_o,  p.W_d2,  p.b_d2,
                        p.W_d1, p.b_d1, p.w_x,   p.w_dlt, p.b_g,  p.W_t1, p.b_t1, p.W_t2,
                        p.b_t2, p.W_qa, p.b_a,   p.W_kvx, p.W_ox, p.W_m1, p.b_m1, p.W_m2,
                        p.b_m2};
  for (const void* q : ptrs)
    if (!aligned16(q)) return false;
  return true;
}

pf_status check_desc(const pf_layer_desc* s) {
  if (s == nullptr) return fail(PF_ERR_INVALID_ARG, "descriptor is NULL");
  if (s->batch < 1 || s->L < 1) return fail(PF_ERR_INVALID_ARG, "batch and L must be >= 1");
  if (s->d < 64 || s->d % 64 != 0) return fail(PF_ERR_INVALID_ARG, "d must be a positive multiple of 64");
  if (s->n_heads < 1 || s->d % s->n_heads != 0)
    return fail(PF_ERR_INVALID_ARG, "n_heads must divide d");
  if (s->d / s->n_heads != 64) return fail(PF_ERR_UNSUPPORTED, "head width d/n_heads must be 64");
  if (s->P < 1) return fail(PF_ERR_INVALID_ARG, "P must be >= 1");
  if (s->levels != 1 && s->levels != 2) return fail(PF_ERR_INVALID_ARG, "levels must be 1 or 2");
  if (s->levels == 2 && (s->k1 < 1 || s->k2 < 1 || (long)s->k1 * s->k2 != s->P))
    return fail(PF_ERR_INVALID_ARG, "levels == 2 needs k1 * k2 == P");
  if (s->mode < PF_CAUSAL_1D || s->mode > PF_BIDIR_2D) return fail(PF_ERR_INVALID_ARG, "bad mode");
  if (s->interact < PF_F_ATTENTION || s->interact > PF_F_MLP || s->rope < 0 || s->rope > 1)
    return fail(PF_ERR_INVALID_ARG, "bad interact or rope");
  if ((s->interact != PF_F_ATTENTION || s->rope) &&
      (s->mode == PF_BIDIR_2D || s->dtype != PF_BF16))
    return fail(PF_ERR_UNSUPPORTED, "identity / MLP interaction and RoPE are built for 1D bf16");
  if (s->rope && s->interact != PF_F_ATTENTION)
    return fail(PF_ERR_INVALID_ARG, "RoPE needs the attention interaction");
  if (s->d_fine < 0 || s->d_fine % 64 != 0)
    return fail(PF_ERR_INVALID_ARG, "d_fine must be 0 (= d) or a positive multiple of 64");
  if (s->d_fine > 0 && s->d_fine != s->d &&
      (s->mode == PF_BIDIR_2D || s->dtype != PF_BF16 || s->inject == PF_INJ_CROSS))
    return fail(PF_ERR_UNSUPPORTED,
                "d_fine != d is built for 1D bf16 layers with add or gated injection");
  if (s->inject < PF_INJ_ADD || s->inject > PF_INJ_CROSS)
    return fail(PF_ERR_INVALID_ARG, "bad inject");
  if (s->dtype != PF_F32 && s->dtype != PF_BF16) return fail(PF_ERR_INVALID_ARG, "bad dtype");
  if (s->mode == PF_BIDIR_2D) {
    if (s->patch < 1 || s->patch * s->patch != s->P || s->grid_h < 1 || s->grid_w < 1 ||
        (long)s->grid_h * s->grid_w != s->L || s->grid_h % s->patch || s->grid_w % s->patch)
      return fail(PF_ERR_INVALID_ARG, "2D layer needs L = grid_h*grid_w, P = patch^2, patch | grid");
    if (s->inject != PF_INJ_AFFINE || s->levels != 1 || s->dtype != PF_BF16 || s->d % 128 != 0 ||
        s->d > 512)
      return fail(PF_ERR_UNSUPPORTED, "the 2D layer is built for affine injection, one level, "
                                      "bf16, d % 128 == 0, d <= 512");
    return PF_OK;
  }
  if (s->inject == PF_INJ_AFFINE) return fail(PF_ERR_UNSUPPORTED, "affine injection is 2D only");
  if (s->inject == PF_INJ_CROSS && (s->dtype != PF_BF16 || s->n_heads > 64))
    return fail(PF_ERR_UNSUPPORTED, "cross-attention injection is built for bf16, <= 64 heads");
  if (s->inject == PF_INJ_CROSS && (long)s->batch * s->L > (1L << 30))
    return fail(PF_ERR_UNSUPPORTED, "problem too large for 32-bit GEMM extents");

  const long m = (s->L + (long)s->P - 1) / s->P;
  const long k1 = s->levels == 2 ? s->k1 : s->P, k2 = s->levels == 2 ? s->k2 : 1;
  if ((long)s->batch * m * k2 > (1L << 30) || k1 * s->d > (1L << 30))
    return fail(PF_ERR_UNSUPPORTED, "problem too large for 32-bit GEMM extents");
  return PF_OK;
}

// fp32 forward (Alg. 1) on CUDA cores; same steps as the bf16 path.
pf_status layer_fwd_f32(const pf_layer_desc& s, const Dims& g, const pf_layer_params& p,
                        const void* Xv, const float* H_in, void* X_out, float* H_out, void* ws,
                        size_t ws_bytes, cudaStream_t cs) {
  Carve wc(ws);
  const F32Ws w = carve_f32(wc, s, g);
  if (ws == nullptr || wc.off > ws_bytes)
    return fail(PF_ERR_WORKSPACE, "workspace too small: need %zu bytes, got %zu", wc.off, ws_bytes);
  const float* X = static_cast<const float*>(Xv);
  const int d = (int)g.d, N1 = (int)g.N1;
  const float* Xsrc = X;
  if (g.ragged) {
    PF_CUDA(pad_f32(X, w.Xpad, (int)g.B, g.L, g.Lp, d, cs));
    Xsrc = w.Xpad;
  }
  const float* W_c1 = static_cast<const float*>(p.W_c1);
  float* H = H_out ? H_out : w.H;
  if (s.levels == 1) {
    PF_CUDA(gemm_f32((int)g.R, d, N1, Xsrc, N1, W_c1, N1, H, d, p.b_c1, H_in, d, "compress_c1", cs, w.sk, w.skb));
  } else {
    PF_CUDA(gemm_f32((int)g.rows1, d, N1, Xsrc, N1, W_c1, N1, w.Y, d, p.b_c1, nullptr, 0,
                     "compress_c1", cs, w.sk, w.skb));
    const int n2 = (int)(g.k2 * d);
    PF_CUDA(gemm_f32((int)g.R, d, n2, w.Y, n2, static_cast<const float*>(p.W_c2), n2, H, d, p.b_c2,
                     H_in, d, "compress_c2", cs, w.sk, w.skb));
  }
  PF_CUDA(gemm_f32((int)g.R, 3 * d, d, H, d, static_cast<const float*>(p.W_qkv), d, w.QKV, 3 * d,
                   nullptr, nullptr, 0, "proxy_qkv", cs, w.sk, w.skb));
  PF_CUDA(attn_f32(w.QKV, w.A, (int)g.B, (int)g.m, d, (int)g.nh, g.causal, cs));
  PF_CUDA(gemm_f32((int)g.R, d, d, w.A, d, static_cast<const float*>(p.W_o), d, w.Hbar, d, nullptr,
                   nullptr, 0, "proxy_o", cs, w.sk, w.skb));
  const float* Zsrc = w.Hbar;
  if (s.levels == 2) {
    const int n2 = (int)(g.k2 * d);
    PF_CUDA(gemm_f32((int)g.R, n2, d, w.Hbar, d, static_cast<const float*>(p.W_d2), d, w.Z, n2,
                     p.b_d2, nullptr, 0, "decompress_d2", cs, w.sk, w.skb));
    Zsrc = w.Z;
  }
  PF_CUDA(gemm_f32_inject((int)g.rows1, N1, d, Zsrc, d, static_cast<const float*>(p.W_d1), d,
                          p.b_d1, X, static_cast<float*>(X_out), p.w_x, p.w_dlt, p.b_g, (int)g.B,
                          g.L, d, (int)g.P, (int)g.k1, (int)g.k2, (int)g.m, g.causal ? 1 : 0,
                          s.inject == PF_INJ_GATED ? 1 : 0, cs));
  return PF_OK;
}

// 2D bidirectional layer (Sec. 3.9): patch compression, timestep adaLN on
// the proxies, bidirectional proxy attention, decompression with affine
// injection (Eq. inj-affine).
pf_status layer_fwd_2d(const pf_layer_desc& s, const Dims& g, const pf_layer_params& p,
                       const void* Xv, const float* H_in, const float* t, void* X_out,
                       float* H_out, void* saved, void* ws, size_t ws_bytes, cudaStream_t cs) {
  if (!t) return fail(PF_ERR_INVALID_ARG, "the 2D layer needs t");
  if (!p.W_c1 || !p.b_c1 || !p.W_qkv || !p.W_o || !p.W_d1 || !p.b_d1 || !p.W_t1 || !p.b_t1 ||
      !p.W_t2 || !p.b_t2)
    return fail(PF_ERR_INVALID_ARG, "a parameter of the 2D layer is NULL");
  Carve wc(ws);
  float* Hws = wc.take<float>(g.R * g.d);
  const size_t skb = splitk_need(s, g, false);
  float* sk = wc.take<float>(skb / sizeof(float));
  Carve sc(saved);
  const Saved2D sv = saved ? carve_saved_2d(sc, g) : carve_saved_2d(wc, g);
  if (ws == nullptr || wc.off > ws_bytes)
    return fail(PF_ERR_WORKSPACE, "workspace too small: need %zu bytes, got %zu", wc.off, ws_bytes);
  const bf16* X = static_cast<const bf16*>(Xv);
  const int d = (int)g.d, N1 = (int)g.N1;
  const int patch = s.patch, gh = s.grid_h, gw = s.grid_w;
  float* Hf = H_out ? H_out : Hws;
  PF_CUDA(patch_gather_stats(X, sv.Xp, sv.stats, (int)g.B, d, patch, gh, gw, cs));
  // the patch matrix (Eq. partition): X itself through the patch view, else the gathered copy

  {
    EpiLinearArgs e;
    e.bias = p.b_c1;
    e.addend = H_in;
    e.ld_add = d;
    e.out_f32 = Hf;
    e.ld_f32 = d;
    set_gemm_tag("compress_c1", (double)g.R * d * 8.0);
    PF_CUDA(gemm_linear((int)g.R, d, N1, {sv.Xp, N1, 0}, {static_cast<const bf16*>(p.W_c1), N1, 0}, with_sk(e, sk, skb), cs));
  }
  PF_CUDA(temb_fwd(t, (int)g.B, d, static_cast<const bf16*>(p.W_t1), p.b_t1,
                   static_cast<const bf16*>(p.W_t2), p.b_t2, sv.e, sv.a1, sv.u, sv.gb, cs));
  PF_CUDA(adaln_fwd(Hf, sv.gb, sv.nH, sv.rstdH, sv.Hb, g.R, d, (int)g.m, cs));
  {
    EpiLinearArgs e;
    e.out_bf16 = sv.QKV;
    e.ld_bf16 = 3 * d;
    set_gemm_tag("proxy_qkv", (double)g.R * 3 * d * 2.0);
    PF_CUDA(gemm_linear((int)g.R, 3 * d, d, {sv.Hb, d, 0},
                        {static_cast<const bf16*>(p.W_qkv), d, 0}, with_sk(e, sk, skb), cs));
    PF_CUDA(attn_fwd(sv.QKV, sv.Aatt, sv.LSE, (int)g.B, (int)g.m, d, (int)g.nh, false, cs));
    EpiLinearArgs eo;
    eo.out_bf16 = sv.Hbar;
    eo.ld_bf16 = d;
    set_gemm_tag("proxy_o", (double)g.R * d * 2.0);
    PF_CUDA(gemm_linear((int)g.R, d, d, {sv.Aatt, d, 0}, {static_cast<const bf16*>(p.W_o), d, 0}, with_sk(eo, sk, skb), cs));
  }
  {
    EpiAffine2DArgs e{p.b_d1, sv.S, static_cast<bf16*>(X_out), sv.stats, sv.Xp, d, patch, gh, gw,
                      (int)g.m};
    set_gemm_tag("decompress_affine", (double)g.R * N1 * 8.0);
    PF_CUDA(gemm_affine2d((int)g.R, 2 * N1, d, {sv.Hbar, d, 0},
                          {static_cast<const bf16*>(p.W_d1), d, 0}, e, cs));
  }
  return PF_OK;
}

pf_status layer_bwd_2d(const pf_layer_desc& s, const Dims& g, const pf_layer_params& p,
                       const void* Xv, const void* saved, const void* dX_out, const float* dH_out,
                       void* dXv, float* dH_in, const pf_layer_grads& gr, void* ws,
                       size_t ws_bytes, cudaStream_t cs) {
  Carve wc(ws);
  const Bwd2DWs w = carve_bwd_2d(wc, s, g);
  if (ws == nullptr || wc.off > ws_bytes)
    return fail(PF_ERR_WORKSPACE, "workspace too small: need %zu bytes, got %zu", wc.off, ws_bytes);
  Carve sc(const_cast<void*>(saved));
  const Saved2D sv = carve_saved_2d(sc, g);
  const bf16* X = static_cast<const bf16*>(Xv);
  const bf16* G = static_cast<const bf16*>(dX_out);
  bf16* dX = static_cast<bf16*>(dXv);
  const int d = (int)g.d, N1 = (int)g.N1, N2 = 2 * N1;
  const int patch = s.patch, gh = s.grid_h, gw = s.grid_w;
  const bf16* W_qkv = static_cast<const bf16*>(p.W_qkv);
  const bf16* W_o = static_cast<const bf16*>(p.W_o);
  const bf16* W_d1 = static_cast<const bf16*>(p.W_d1);
  const bf16* W_c1 = static_cast<const bf16*>(p.W_c1);
  // affine injection backward (Eq. inj-affine)
  PF_CUDA(inj_bwd_2d(G, X, sv.stats, sv.S, w.dD, w.dXd, gr.b_d1, w.part, g.R, d, patch, gh, gw,
                     cs));
  if (gr.W_d1) {
    EpiLinearArgs e;
    e.out_f32 = gr.W_d1;
    e.ld_f32 = d;
    set_gemm_tag("bwd_dW_d1", (double)N2 * d * 4.0);
    PF_CUDA(gemm_linear(N2, d, (int)g.R, {w.dD, N2, 1}, {sv.Hbar, d, 1}, with_sk(e, w.sk, w.skb), cs));
  }
  {
    EpiLinearArgs e;
    e.out_bf16 = w.dHbar;
    e.ld_bf16 = d;
    set_gemm_tag("bwd_dHbar", (double)g.R * d * 2.0);
    PF_CUDA(gemm_linear((int)g.R, d, N2, {w.dD, N2, 0}, {W_d1, d, 1}, with_sk(e, w.sk, w.skb), cs));
  }
  if (gr.W_o) {
    EpiLinearArgs e;
    e.out_f32 = gr.W_o;
    e.ld_f32 = d;
    set_gemm_tag("bwd_dW_o", (double)d * d * 4.0);
    PF_CUDA(gemm_linear(d, d, (int)g.R, {w.dHbar, d, 1}, {sv.Aatt, d, 1}, with_sk(e, w.sk, w.skb), cs));
  }
  {
    EpiLinearArgs e;
    e.out_bf16 = w.dA;
    e.ld_bf16 = d;
    set_gemm_tag("bwd_dA", (double)g.R * d * 2.0);
    PF_CUDA(gemm_linear((int)g.R, d, d, {w.dHbar, d, 0}, {W_o, d, 1}, with_sk(e, w.sk, w.skb), cs));
  }
  PF_CUDA(attn_bwd(sv.QKV, sv.Aatt, w.dA, sv.LSE, w.Di, w.dQKV, (int)g.B, (int)g.m, d, (int)g.nh,
                   false, cs));
  if (gr.W_qkv) {
    EpiLinearArgs e;
    e.out_f32 = gr.W_qkv;
    e.ld_f32 = d;
    set_gemm_tag("bwd_dW_qkv", (double)3 * d * d * 4.0);
    PF_CUDA(gemm_linear(3 * d, d, (int)g.R, {w.dQKV, 3 * d, 1}, {sv.Hb, d, 1}, with_sk(e, w.sk, w.skb), cs));
  }
  {
    EpiLinearArgs e;
    e.out_f32 = w.dHq;
    e.ld_f32 = d;
    set_gemm_tag("bwd_dHq", (double)g.R * d * 4.0);
    PF_CUDA(gemm_linear((int)g.R, d, 3 * d, {w.dQKV, 3 * d, 0}, {W_qkv, d, 1}, with_sk(e, w.sk, w.skb), cs));
  }
  // adaLN and timestep-MLP backward
  float* dHf = dH_in ? dH_in : w.dHf;
  PF_CUDA(adaln_bwd(w.dHq, sv.nH, sv.rstdH, sv.gb, dH_out, dHf, w.dHb, g.R, d, (int)g.m, cs));
  PF_CUDA(adaln_param_grads(w.dHq, sv.nH, w.part, w.dgb, (int)g.B, d, (int)g.m, cs));
  PF_CUDA(temb_bwd(w.dgb, static_cast<const bf16*>(p.W_t2), sv.a1, sv.u, sv.e, w.da1,
                   TembGrads{gr.W_t2, gr.b_t2, gr.W_t1, gr.b_t1}, (int)g.B, d, cs));
  // compression backward (H = H_in + C, so dC = dH)
  if (gr.b_c1) PF_CUDA(colsum_f32(dHf, g.R, d, gr.b_c1, w.part, cs));
  if (gr.W_c1) {
    EpiLinearArgs e;
    e.out_f32 = gr.W_c1;
    e.ld_f32 = N1;
    set_gemm_tag("bwd_dW_c1", (double)d * N1 * 4.0);
    PF_CUDA(gemm_linear(d, N1, (int)g.R, {w.dHb, d, 1}, {sv.Xp, N1, 1}, with_sk(e, w.sk, w.skb), cs));
  }
  {
    EpiDX2DArgs e{w.dXd, dX, d, patch, gh, gw, (int)g.m};
    set_gemm_tag("bwd_dX", (double)g.R * N1 * 4.0);
    PF_CUDA(gemm_dx2d((int)g.R, N1, d, {w.dHb, d, 0}, {W_c1, N1, 1}, e, cs));
  }
  return PF_OK;
}

}  // namespace

// Sets the thread-local message returned by pf_last_error (for other files of
// the library) and returns `s`.
__attribute__((visibility("hidden"))) pf_status pf_set_error(pf_status s, const char* msg) {
  g_msg = msg;
  return s;
}

extern "C" {

const char* pf_last_error(void) { return g_msg.c_str(); }

pf_status proxy_layer_check(const pf_layer_desc* desc) { return check_desc(desc); }

size_t proxy_layer_saved_size(const pf_layer_desc* desc) {
  if (check_desc(desc) != PF_OK) return 0;
  if (desc->dtype == PF_F32) return 0;  // the fp32 layer is forward-only
  const Dims g = dims_of(*desc);
  Carve c(nullptr);
  if (desc->mode == PF_BIDIR_2D)
    carve_saved_2d(c, g);
  else
    carve_saved(c, *desc, g);
  return (c.off + 255) & ~size_t(255);
}

size_t proxy_layer_workspace_size(const pf_layer_desc* desc, int for_backward) {
  if (check_desc(desc) != PF_OK) return 0;
  const Dims g = dims_of(*desc);
  Carve c(nullptr);
  if (desc->dtype == PF_F32) {
    if (for_backward) return 0;
    carve_f32(c, *desc, g);
  } else if (desc->mode == PF_BIDIR_2D) {
    if (for_backward) {
      carve_bwd_2d(c, *desc, g);
    } else {
      c.take<float>(g.R * g.d);  // H when H_out is NULL
      c.take<float>(splitk_need(*desc, g, false) / sizeof(float));
      carve_saved_2d(c, g);
    }
  } else if (for_backward) {
    carve_bwd(c, *desc, g);
  } else {
    carve_fwd(c, *desc, g, nullptr);  // saved activations here when saved == NULL
  }
  return ((c.off + 255) & ~size_t(255)) + 256;
}

pf_status proxy_layer_fwd(const pf_layer_desc* desc, const pf_layer_params* prm, const void* X,
                          const float* H_in, const float* t, void* X_out, float* H_out, void* saved,
                          void* ws, size_t ws_bytes, void* stream) {
  pf_status st = check_desc(desc);
  if (st != PF_OK) return st;
  (void)t;
  const pf_layer_desc& s = *desc;
  const Dims g = dims_of(s);
  if (prm == nullptr || X == nullptr || X_out == nullptr || X == X_out)
    return fail(PF_ERR_INVALID_ARG, "params, X and X_out are required and must not alias");
  const bool cross = s.inject == PF_INJ_CROSS;
  const bool attn = s.interact == PF_F_ATTENTION, mlp = s.interact == PF_F_MLP;
  if (!prm->W_c1 || !prm->b_c1 || (attn && (!prm->W_qkv || !prm->W_o)) ||
      (mlp && (!prm->W_m1 || !prm->b_m1 || !prm->W_m2 || !prm->b_m2)) ||
      (!cross && (!prm->W_d1 || !prm->b_d1)) || (s.levels == 2 && (!prm->W_c2 || !prm->b_c2)) ||
      (s.levels == 2 && !cross && (!prm->W_d2 || !prm->b_d2)) ||
      (s.inject == PF_INJ_GATED && (!prm->w_x || !prm->w_dlt || !prm->b_g)) ||
      (cross && (!prm->W_qa || !prm->b_a || !prm->W_kvx || !prm->W_ox)))
    return fail(PF_ERR_INVALID_ARG, "a parameter this layer uses is NULL");
  if (!aligned16(X) || !aligned16(X_out) || !aligned16(saved) || !aligned16(ws) ||
      !aligned16(H_in) || !aligned16(H_out) || !params_aligned(*prm))
    return fail(PF_ERR_INVALID_ARG, "buffers must be 16-byte aligned");
  if (s.dtype == PF_F32) return layer_fwd_f32(s, g, *prm, X, H_in, X_out, H_out, ws, ws_bytes,
                                             static_cast<cudaStream_t>(stream));
  if (s.mode == PF_BIDIR_2D)
    return layer_fwd_2d(s, g, *prm, X, H_in, t, X_out, H_out, saved, ws, ws_bytes,
                        static_cast<cudaStream_t>(stream));
  Carve wc(ws);
  const FwdWs fw = carve_fwd(wc, s, g, saved);
  bf16* Xpad = fw.Xpad;
  const size_t skb = fw.skb;
  float* sk = fw.sk;
  const Saved sv = fw.sv;
  if (wc.off > ws_bytes)
    return fail(PF_ERR_WORKSPACE, "workspace too small: need %zu bytes, got %zu", wc.off, ws_bytes);
  if (ws == nullptr && wc.off > 0) return fail(PF_ERR_WORKSPACE, "workspace is NULL");
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  const bf16* Xb = static_cast<const bf16*>(X);
  bf16* Xo = static_cast<bf16*>(X_out);
  const int d = (int)g.d, df = (int)g.df;  // proxy and token widths

  // a1: partition (a zero-copy view; the ragged tail goes through a padded copy)
  const bf16* Xsrc = Xb;
  if (g.ragged) {
    PF_CUDA(pad_rows(Xb, Xpad, (int)g.B, g.L, g.Lp, df, cs));
    Xsrc = Xpad;
  }
  // a2 + a3: compression (Eq. compress-linear / factor-cascade), H = H_in + C
  {
    EpiLinearArgs e;
    if (s.levels == 1) {
      e.bias = prm->b_c1;
      e.addend = H_in;
      e.ld_add = d;
      e.out_f32 = H_out;
      e.ld_f32 = d;
      e.out_bf16 = sv.Hb;
      e.ld_bf16 = d;
      set_gemm_tag("compress_c1", (double)g.R * d * 6.0);
      PF_CUDA(gemm_linear((int)g.R, d, (int)g.N1, {Xsrc, g.N1, 0},
                          {static_cast<const bf16*>(prm->W_c1), g.N1, 0}, with_sk(e, sk, skb), cs));
    } else {
      e.bias = prm->b_c1;
      e.out_bf16 = sv.Y;
      e.ld_bf16 = d;
      set_gemm_tag("compress_c1", (double)g.rows1 * d * 2.0);
      PF_CUDA(gemm_linear((int)g.rows1, d, (int)g.N1, {Xsrc, g.N1, 0},
                          {static_cast<const bf16*>(prm->W_c1), g.N1, 0}, with_sk(e, sk, skb), cs));
      EpiLinearArgs e2;
      e2.bias = prm->b_c2;
      e2.addend = H_in;
      e2.ld_add = d;
      e2.out_f32 = H_out;
      e2.ld_f32 = d;
      e2.out_bf16 = sv.Hb;
      e2.ld_bf16 = d;
      set_gemm_tag("compress_c2", (double)g.R * d * 10.0);
      PF_CUDA(gemm_linear((int)g.R, d, (int)(g.k2 * d), {sv.Y, g.k2 * d, 0},
                          {static_cast<const bf16*>(prm->W_c2), g.k2 * d, 0}, with_sk(e2, sk, skb), cs));
    }
  }
  // a4: proxy interaction F (Sec. 3.4)
  if (g.f == PF_F_IDENTITY) {
    PF_CUDA(cudaMemcpyAsync(sv.Hbar, sv.Hb, g.R * d * sizeof(bf16), cudaMemcpyDeviceToDevice, cs));
  } else if (g.f == PF_F_MLP) {  // Hbar = W_m2 SiLU(W_m1 H + b_m1) + b_m2, one proxy at a time
    EpiLinearArgs e;
    e.bias = prm->b_m1;
    e.pre_bf16 = sv.U;
    e.ld_pre = 4 * d;
    e.act_silu = 1;
    e.out_bf16 = sv.Am;
    e.ld_bf16 = 4 * d;
    set_gemm_tag("proxy_mlp1", (double)g.R * 9 * d * 2.0);
    PF_CUDA(gemm_linear((int)g.R, 4 * d, d, {sv.Hb, d, 0},
                        {static_cast<const bf16*>(prm->W_m1), d, 0}, e, cs));
    EpiLinearArgs e2;
    e2.bias = prm->b_m2;
    e2.out_bf16 = sv.Hbar;
    e2.ld_bf16 = d;
    set_gemm_tag("proxy_mlp2", (double)g.R * 5 * d * 2.0);
    PF_CUDA(gemm_linear((int)g.R, d, 4 * d, {sv.Am, 4 * d, 0},
                        {static_cast<const bf16*>(prm->W_m2), 4 * d, 0}, with_sk(e2, sk, skb), cs));
  } else {  // attention (Eq. proxy-attn), queries and keys rotated first with RoPE
    EpiLinearArgs e;
    e.out_bf16 = sv.QKV;
    e.ld_bf16 = 3 * d;
    set_gemm_tag("proxy_qkv", (double)g.R * 3 * d * 2.0);
    PF_CUDA(gemm_linear((int)g.R, 3 * d, d, {sv.Hb, d, 0},
                        {static_cast<const bf16*>(prm->W_qkv), d, 0}, with_sk(e, sk, skb), cs));
    if (g.rope) PF_CUDA(rope_qk(sv.QKV, 3 * d, (int)g.B, (int)g.m, d, fw.rtab, false, cs));
    PF_CUDA(attn_fwd(sv.QKV, sv.Aatt, sv.LSE, (int)g.B, (int)g.m, d, (int)g.nh, g.causal, cs));
    EpiLinearArgs eo;
    eo.out_bf16 = sv.Hbar;
    eo.ld_bf16 = d;
    set_gemm_tag("proxy_o", (double)g.R * d * 2.0);
    PF_CUDA(gemm_linear((int)g.R, d, d, {sv.Aatt, d, 0}, {static_cast<const bf16*>(prm->W_o), d, 0}, with_sk(eo, sk, skb), cs));
  }
  if (g.cross) {
    // a5 + a6 as gated cross-attention (Eq. inj-cross with the gate of Eq.
    // llm-gate): [Q | gate] of the tokens, the proxies' keys and values, the
    // attention with its per-head gate, and the output projection plus X
    PF_CUDA(pad_qa(prm->W_qa, fw.Wqa, g, cs));
    {
      EpiLinearArgs e;
      e.out_bf16 = sv.QA;
      e.ld_bf16 = g.ldq;
      set_gemm_tag("cross_qa", (double)g.T * (d + g.ldq) * 2.0);
      PF_CUDA(gemm_linear((int)g.T, (int)g.ldq, d, {Xb, d, 0}, {fw.Wqa, d, 0}, with_sk(e, sk, skb), cs));
    }
    {
      EpiLinearArgs e;
      e.out_bf16 = sv.KVx;
      e.ld_bf16 = 2 * d;
      set_gemm_tag("cross_kv", (double)g.R * 3 * d * 2.0);
      PF_CUDA(gemm_linear((int)g.R, 2 * d, d, {sv.Hbar, d, 0},
                          {static_cast<const bf16*>(prm->W_kvx), d, 0}, with_sk(e, sk, skb), cs));
    }
    PF_CUDA(attn_cross_fwd(sv.QA, g.ldq, sv.KVx, prm->b_a, saved ? sv.Ax : nullptr, sv.Ag,
                           sv.LSEx, (int)g.B, (int)g.L, (int)g.m, d, (int)g.nh, (int)g.P,
                           g.causal, cs));
    EpiLinearArgs e;
    e.add_bf16 = Xb;
    e.ld_add_bf16 = d;
    e.out_bf16 = Xo;
    e.ld_bf16 = d;
    set_gemm_tag("cross_out", (double)g.T * d * 6.0);
    PF_CUDA(gemm_linear((int)g.T, d, d, {sv.Ag, d, 0}, {static_cast<const bf16*>(prm->W_ox), d, 0},
                        with_sk(e, sk, skb), cs));
    return PF_OK;
  }
  // a5 + a6: decompression (Eq. decompress-linear / factor-dec), routing and
  // injection (Eq. inj-gate / inj-add), fused into the last level's GEMM
  const bf16* Zsrc = sv.Hbar;
  if (s.levels == 2) {
    EpiLinearArgs e;
    e.bias = prm->b_d2;
    e.out_bf16 = sv.Z;
    e.ld_bf16 = g.k2 * d;
    set_gemm_tag("decompress_d2", (double)g.R * g.k2 * d * 2.0);
    PF_CUDA(gemm_linear((int)g.R, (int)(g.k2 * d), d, {sv.Hbar, d, 0},
                        {static_cast<const bf16*>(prm->W_d2), d, 0}, with_sk(e, sk, skb), cs));
    Zsrc = sv.Z;
  }
  {
    EpiInjectArgs e{prm->b_d1, sv.D, Xsrc, Xo,
                    prm->w_x, prm->w_dlt, prm->b_g,
                    df, (int)g.k1, (int)g.k2, (int)g.m, (int)g.L, g.causal ? 1 : 0,
                    s.inject == PF_INJ_GATED ? 1 : 0};
    set_gemm_tag("decompress_d1_inject", (double)g.rows1 * g.N1 * 8.0);
    PF_CUDA(gemm_inject1d((int)g.rows1, (int)g.N1, d, {Zsrc, d, 0},
                          {static_cast<const bf16*>(prm->W_d1), d, 0}, e, cs));
  }
  if (g.causal) PF_CUDA(copy_block0(Xb, g.L, Xo, g.L, (int)g.B, df, (int)std::min(g.P, g.L), cs));
  return PF_OK;
}

pf_status proxy_layer_bwd(const pf_layer_desc* desc, const pf_layer_params* prm, const void* X,
                          const float* H_in, const float* t, const void* saved, const void* dX_out,
                          const float* dH_out, void* dX, float* dH_in, const pf_layer_grads* grads,
                          void* ws, size_t ws_bytes, void* stream) {
  pf_status st = check_desc(desc);
  if (st != PF_OK) return st;
  (void)H_in;
  (void)t;
  const pf_layer_desc& s = *desc;
  const Dims g = dims_of(s);
  if (!prm || !X || !saved || !dX_out || !dX || !grads)
    return fail(PF_ERR_INVALID_ARG, "params, X, saved, dX_out, dX and grads are required");
  if (!aligned16(X) || !aligned16(saved) || !aligned16(dX_out) || !aligned16(dX) ||
      !aligned16(ws) || !aligned16(dH_out) || !aligned16(dH_in) || !params_aligned(*prm))
    return fail(PF_ERR_INVALID_ARG, "buffers must be 16-byte aligned");
  if (s.dtype == PF_F32) return fail(PF_ERR_UNSUPPORTED, "the fp32 layer is forward-only");
  if (s.mode == PF_BIDIR_2D)
    return layer_bwd_2d(s, g, *prm, X, saved, dX_out, dH_out, dX, dH_in, *grads, ws, ws_bytes,
                        static_cast<cudaStream_t>(stream));
  const bool gated = s.inject == PF_INJ_GATED;
  if (g.cross ? (!prm->W_qa || !prm->b_a || !prm->W_kvx || !prm->W_ox)
              : (!grads->b_d1 || (gated && (!grads->w_x || !grads->w_dlt || !grads->b_g))))
    return fail(PF_ERR_INVALID_ARG, g.cross ? "a cross-injection parameter is NULL"
                                            : "grads->b_d1 (and the gate gradients) must be given");
  Carve wc(ws);
  BwdWs w = carve_bwd(wc, s, g);
  if (ws == nullptr || wc.off > ws_bytes)
    return fail(PF_ERR_WORKSPACE, "workspace too small: need %zu bytes, got %zu", wc.off, ws_bytes);
  Carve sc(const_cast<void*>(saved));
  const Saved sv = carve_saved(sc, s, g);
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  const bf16* Xb = static_cast<const bf16*>(X);
  const bf16* G = static_cast<const bf16*>(dX_out);
  bf16* dXb = static_cast<bf16*>(dX);
  const int d = (int)g.d, N1 = (int)g.N1, df = (int)g.df;  // proxy and token widths
  const bf16* W_c1 = static_cast<const bf16*>(prm->W_c1);
  const bf16* W_c2 = static_cast<const bf16*>(prm->W_c2);
  const bf16* W_qkv = static_cast<const bf16*>(prm->W_qkv);
  const bf16* W_o = static_cast<const bf16*>(prm->W_o);
  const bf16* W_d2 = static_cast<const bf16*>(prm->W_d2);
  const bf16* W_d1 = static_cast<const bf16*>(prm->W_d1);

  const bf16* Xsrc = Xb;
  if (g.ragged) {
    PF_CUDA(pad_rows(Xb, w.Xpad, (int)g.B, g.L, g.Lp, df, cs));
    Xsrc = w.Xpad;
  }
  // direct injection gradient: written into dX, or into a block-padded buffer
  // when L % P != 0 so the dX GEMM epilogue can prefetch it as whole tiles
  bf16* dXd = g.ragged ? w.dXpad : dXb;
  if (g.cross) {
    // the gated cross injection backward: output projection, gate, the
    // cross-attention (dQ of the tokens, dK / dV of the proxies), then the
    // direct dX = dX_out + [dQ | d gate] W_qa and dHbar = [dK | dV] W_kvx
    const bf16* W_ox = static_cast<const bf16*>(prm->W_ox);
    const bf16* W_kvx = static_cast<const bf16*>(prm->W_kvx);
    const int T = (int)g.T, q = (int)g.ldq;
    PF_CUDA(pad_qa(prm->W_qa, w.Wqa, g, cs));
    if (grads->W_ox) {
      EpiLinearArgs e;
      e.out_f32 = grads->W_ox;
      e.ld_f32 = d;
      set_gemm_tag("bwd_dW_ox", (double)d * d * 4.0);
      PF_CUDA(gemm_linear(d, d, T, {G, d, 1}, {sv.Ag, d, 1}, with_sk(e, w.sk, w.skb), cs));
    }
    {
      EpiLinearArgs e;
      e.out_bf16 = w.dAg;
      e.ld_bf16 = d;
      set_gemm_tag("bwd_dAg", (double)T * d * 4.0);
      PF_CUDA(gemm_linear(T, d, d, {G, d, 0}, {W_ox, d, 1}, with_sk(e, w.sk, w.skb), cs));
    }
    PF_CUDA(cross_gate_bwd(w.dAg, sv.Ax, sv.QA, g.ldq, prm->b_a, w.dOx, w.Dix, w.dQA, w.ga,
                           w.ldga, (int)g.B, (int)g.L, d, (int)g.nh, cs));
    if (grads->b_a) {
      PF_CUDA(colsum_f32(w.ga, g.T, w.ldga, w.gsum, w.part, cs));
      PF_CUDA(cudaMemcpyAsync(grads->b_a, w.gsum, g.nh * sizeof(float), cudaMemcpyDeviceToDevice,
                              cs));
    }
    PF_CUDA(attn_cross_bwd(sv.QA, g.ldq, sv.KVx, w.dOx, sv.LSEx, w.Dix, w.dQA, w.dKVx, (int)g.B,
                           (int)g.L, (int)g.m, d, (int)g.nh, (int)g.P, g.causal, cs));
    if (grads->W_qa) {
      EpiLinearArgs e;
      e.out_f32 = grads->W_qa;
      e.ld_f32 = d;
      set_gemm_tag("bwd_dW_qa", (double)(d + g.nh) * d * 4.0);
      PF_CUDA(gemm_linear(d + (int)g.nh, d, T, {w.dQA, g.ldq, 1}, {Xb, d, 1},
                          with_sk(e, w.sk, w.skb), cs));
    }
    if (grads->W_kvx) {
      EpiLinearArgs e;
      e.out_f32 = grads->W_kvx;
      e.ld_f32 = d;
      set_gemm_tag("bwd_dW_kvx", (double)2 * d * d * 4.0);
      PF_CUDA(gemm_linear(2 * d, d, (int)g.R, {w.dKVx, 2 * d, 1}, {sv.Hbar, d, 1},
                          with_sk(e, w.sk, w.skb), cs));
    }
    {
      EpiLinearArgs e;
      e.out_bf16 = w.dHbar;
      e.ld_bf16 = d;
      set_gemm_tag("bwd_dHbar", (double)g.R * 3 * d * 2.0);
      PF_CUDA(gemm_linear((int)g.R, d, 2 * d, {w.dKVx, 2 * d, 0}, {W_kvx, d, 1},
                          with_sk(e, w.sk, w.skb), cs));
    }
    // direct dX, in the block-padded layout when L % P != 0 (per sequence
    // then, as the rows of different sequences are spaced differently)
    const bool per_seq = g.ragged && g.B > 1;
    for (long b = 0; b < (per_seq ? g.B : 1); ++b) {
      EpiLinearArgs e;
      e.add_bf16 = G + b * g.L * d;
      e.ld_add_bf16 = d;
      e.out_bf16 = dXd + b * (g.ragged ? g.Lp : g.L) * d;
      e.ld_bf16 = d;
      const int rows = per_seq ? (int)g.L : T;
      set_gemm_tag("bwd_dX_direct", (double)rows * (q + 2 * d) * 2.0);
      PF_CUDA(gemm_linear(rows, d, q, {w.dQA + b * g.L * q, q, 0}, {w.Wqa, d, 1},
                          with_sk(e, w.sk, w.skb), cs));
    }
  } else {
    // injection backward: dD (proxy order), direct dX, gate and b_d1 gradients
    {
      const int nch = inj_bwd_chunks(g.rows1, N1);
      InjBwdArgs a{G, Xb, sv.D, w.dD, dXd, g.ragged ? g.Lp : g.L, prm->w_x, prm->w_dlt, prm->b_g,
                   df, (int)g.k1, (int)g.k2, (int)g.m, (int)g.L, (int)g.B, g.causal ? 1 : 0,
                   gated ? 1 : 0};
      PF_CUDA(inj_bwd_1d(a, w.part, nch, cs));
      if (g.causal)
        PF_CUDA(copy_block0(G, g.L, dXd, g.ragged ? g.Lp : g.L, (int)g.B, df,
                            (int)std::min(g.P, g.L), cs));
      PF_CUDA(inj_bwd_finalize(w.part, nch, N1, df, grads->b_d1, gated ? grads->w_x : nullptr,
                               gated ? grads->w_dlt : nullptr, gated ? grads->b_g : nullptr, cs));
    }
    // decompression level 1 (or single level)
    const bf16* Zsrc = s.levels == 2 ? sv.Z : sv.Hbar;
    if (grads->W_d1) {
      EpiLinearArgs e;
      e.out_f32 = grads->W_d1;
      e.ld_f32 = d;
      set_gemm_tag("bwd_dW_d1", (double)N1 * d * 4.0);
      PF_CUDA(gemm_linear(N1, d, (int)g.rows1, {w.dD, N1, 1}, {Zsrc, d, 1}, with_sk(e, w.sk, w.skb), cs));
    }
    {
      EpiLinearArgs e;
      e.out_bf16 = s.levels == 2 ? w.dZ : w.dHbar;
      e.ld_bf16 = d;
      set_gemm_tag("bwd_dZ", (double)g.rows1 * d * 2.0);
      PF_CUDA(gemm_linear((int)g.rows1, d, N1, {w.dD, N1, 0}, {W_d1, d, 1}, with_sk(e, w.sk, w.skb), cs));
    }
    if (s.levels == 2) {
      const int n2 = (int)(g.k2 * d);
      if (grads->b_d2) PF_CUDA(colsum_bf16(w.dZ, g.R, n2, grads->b_d2, w.part, cs));
      if (grads->W_d2) {
        EpiLinearArgs e;
        e.out_f32 = grads->W_d2;
        e.ld_f32 = d;
        set_gemm_tag("bwd_dW_d2", (double)n2 * d * 4.0);
        PF_CUDA(gemm_linear(n2, d, (int)g.R, {w.dZ, n2, 1}, {sv.Hbar, d, 1}, with_sk(e, w.sk, w.skb), cs));
      }
      EpiLinearArgs e;
      e.out_bf16 = w.dHbar;
      e.ld_bf16 = d;
      set_gemm_tag("bwd_dHbar", (double)g.R * d * 2.0);
      PF_CUDA(gemm_linear((int)g.R, d, n2, {w.dZ, n2, 0}, {W_d2, d, 1}, with_sk(e, w.sk, w.skb), cs));
    }
  }
  // proxy interaction F: identity, single-proxy MLP, or attention
  float* dHf = dH_in ? dH_in : w.dHf;
  if (g.f == PF_F_IDENTITY) {
    PF_CUDA(add_f32_bf16(w.dHbar, dH_out, dHf, w.dHb, g.R * d, cs));
  } else if (g.f == PF_F_MLP) {
    const bf16* W_m1 = static_cast<const bf16*>(prm->W_m1);
    const bf16* W_m2 = static_cast<const bf16*>(prm->W_m2);
    if (grads->W_m2) {
      EpiLinearArgs e;
      e.out_f32 = grads->W_m2;
      e.ld_f32 = 4 * d;
      set_gemm_tag("bwd_dW_m2", (double)4 * d * d * 4.0);
      PF_CUDA(gemm_linear(d, 4 * d, (int)g.R, {w.dHbar, d, 1}, {sv.Am, 4 * d, 1},
                          with_sk(e, w.sk, w.skb), cs));
    }
    if (grads->b_m2) PF_CUDA(colsum_bf16(w.dHbar, g.R, d, grads->b_m2, w.part, cs));
    {
      EpiLinearArgs e;  // dU = (dHbar W_m2) * SiLU'(U)
      e.dsilu_of = sv.U;
      e.ld_dsilu = 4 * d;
      e.out_bf16 = w.dU;
      e.ld_bf16 = 4 * d;
      set_gemm_tag("bwd_dU", (double)g.R * 9 * d * 2.0);
      PF_CUDA(gemm_linear((int)g.R, 4 * d, d, {w.dHbar, d, 0}, {W_m2, 4 * d, 1}, e, cs));
    }
    if (grads->W_m1) {
      EpiLinearArgs e;
      e.out_f32 = grads->W_m1;
      e.ld_f32 = d;
      set_gemm_tag("bwd_dW_m1", (double)4 * d * d * 4.0);
      PF_CUDA(gemm_linear(4 * d, d, (int)g.R, {w.dU, 4 * d, 1}, {sv.Hb, d, 1},
                          with_sk(e, w.sk, w.skb), cs));
    }
    if (grads->b_m1) PF_CUDA(colsum_bf16(w.dU, g.R, 4 * d, grads->b_m1, w.part, cs));
    EpiLinearArgs e;
    e.addend = dH_out;
    e.ld_add = d;
    e.out_f32 = dHf;
    e.ld_f32 = d;
    e.out_bf16 = w.dHb;
    e.ld_bf16 = d;
    set_gemm_tag("bwd_dH", (double)g.R * d * 14.0);
    PF_CUDA(gemm_linear((int)g.R, d, 4 * d, {w.dU, 4 * d, 0}, {W_m1, d, 1},
                        with_sk(e, w.sk, w.skb), cs));
  } else {
    if (grads->W_o) {
      EpiLinearArgs e;
      e.out_f32 = grads->W_o;
      e.ld_f32 = d;
      set_gemm_tag("bwd_dW_o", (double)d * d * 4.0);
      PF_CUDA(gemm_linear(d, d, (int)g.R, {w.dHbar, d, 1}, {sv.Aatt, d, 1}, with_sk(e, w.sk, w.skb), cs));
    }
    {
      EpiLinearArgs e;
      e.out_bf16 = w.dA;
      e.ld_bf16 = d;
      set_gemm_tag("bwd_dA", (double)g.R * d * 2.0);
      PF_CUDA(gemm_linear((int)g.R, d, d, {w.dHbar, d, 0}, {W_o, d, 1}, with_sk(e, w.sk, w.skb), cs));
    }
    PF_CUDA(attn_bwd(sv.QKV, sv.Aatt, w.dA, sv.LSE, w.Di, w.dQKV, (int)g.B, (int)g.m, d, (int)g.nh,
                     g.causal, cs));
    if (g.rope) PF_CUDA(rope_qk(w.dQKV, 3 * d, (int)g.B, (int)g.m, d, w.rtab, true, cs));  // back
    if (grads->W_qkv) {
      EpiLinearArgs e;
      e.out_f32 = grads->W_qkv;
      e.ld_f32 = d;
      set_gemm_tag("bwd_dW_qkv", (double)3 * d * d * 4.0);
      PF_CUDA(gemm_linear(3 * d, d, (int)g.R, {w.dQKV, 3 * d, 1}, {sv.Hb, d, 1}, with_sk(e, w.sk, w.skb), cs));
    }
    {
      EpiLinearArgs e;
      e.addend = dH_out;
      e.ld_add = d;
      e.out_f32 = dHf;
      e.ld_f32 = d;
      e.out_bf16 = w.dHb;
      e.ld_bf16 = d;
      set_gemm_tag("bwd_dH", (double)g.R * d * 10.0);
      PF_CUDA(gemm_linear((int)g.R, d, 3 * d, {w.dQKV, 3 * d, 0}, {W_qkv, d, 1}, with_sk(e, w.sk, w.skb), cs));
    }
  }
  // compression (H = H_in + C, so dC = dH)
  const bf16* dYsrc = w.dHb;
  if (s.levels == 2) {
    const int n2 = (int)(g.k2 * d);
    if (grads->b_c2) PF_CUDA(colsum_f32(dHf, g.R, d, grads->b_c2, w.part, cs));
    if (grads->W_c2) {
      EpiLinearArgs e;
      e.out_f32 = grads->W_c2;
      e.ld_f32 = n2;
      set_gemm_tag("bwd_dW_c2", (double)d * n2 * 4.0);
      PF_CUDA(gemm_linear(d, n2, (int)g.R, {w.dHb, d, 1}, {sv.Y, n2, 1}, with_sk(e, w.sk, w.skb), cs));
    }
    EpiLinearArgs e;
    e.out_bf16 = w.dY;
    e.ld_bf16 = n2;
    set_gemm_tag("bwd_dY", (double)g.R * n2 * 2.0);
    PF_CUDA(gemm_linear((int)g.R, n2, d, {w.dHb, d, 0}, {W_c2, n2, 1}, with_sk(e, w.sk, w.skb), cs));
    if (grads->b_c1) PF_CUDA(colsum_bf16(w.dY, g.rows1, d, grads->b_c1, w.part, cs));
    dYsrc = w.dY;
  } else if (grads->b_c1) {
    PF_CUDA(colsum_f32(dHf, g.R, d, grads->b_c1, w.part, cs));
  }
  if (grads->W_c1) {
    EpiLinearArgs e;
    e.out_f32 = grads->W_c1;
    e.ld_f32 = N1;
    set_gemm_tag("bwd_dW_c1", (double)d * N1 * 4.0);
    PF_CUDA(gemm_linear(d, N1, (int)g.rows1, {dYsrc, d, 1}, {Xsrc, N1, 1}, with_sk(e, w.sk, w.skb), cs));
  }
  {
    EpiDXArgs e{dXd, dXb, df, (int)g.k1, (int)g.k2, (int)g.m, (int)g.L};
    set_gemm_tag("bwd_dX", (double)g.rows1 * N1 * 4.0);
    PF_CUDA(gemm_dx1d((int)g.rows1, N1, d, {dYsrc, d, 0}, {W_c1, N1, 1}, e, cs));
  }
  return PF_OK;
}

}  // extern "C"

namespace {

pf_status check_decode_desc(const pf_decode_desc* s) {
  if (s == nullptr) return fail(PF_ERR_INVALID_ARG, "decode descriptor is NULL");
  if (s->batch < 1) return fail(PF_ERR_INVALID_ARG, "batch must be >= 1");
  if (s->d < 64 || s->d % 64 != 0 || s->d > 4096)
    return fail(PF_ERR_INVALID_ARG, "d must be a multiple of 64 in [64, 4096]");
  if (s->n_heads < 1 || s->d % s->n_heads != 0)
    return fail(PF_ERR_INVALID_ARG, "n_heads must divide d");
  const int dh = s->d / s->n_heads;
  if (dh != 64 && dh != 128) return fail(PF_ERR_UNSUPPORTED, "head width must be 64 or 128");
  if (s->P < 1 || s->P > PF_DECODE_MAX_P)
    return fail(PF_ERR_UNSUPPORTED, "P must be in [1, %d]", PF_DECODE_MAX_P);
  if (s->levels != 1 && s->levels != 2) return fail(PF_ERR_INVALID_ARG, "levels must be 1 or 2");
  if (s->levels == 2 && (s->k1 < 1 || s->k2 < 1 || (long)s->k1 * s->k2 != s->P))
    return fail(PF_ERR_INVALID_ARG, "levels == 2 needs k1 * k2 == P");
  if (s->capacity < 1) return fail(PF_ERR_INVALID_ARG, "capacity must be >= 1");
  return PF_OK;
}

bool cache_ok(const pf_kv_cache* c) {
  return c && c->K_proxy && c->V_proxy && c->X_open && c->K_open && c->V_open && c->n_proxy &&
         c->n_open && aligned16(c->K_proxy) && aligned16(c->V_proxy) && aligned16(c->X_open) &&
         aligned16(c->K_open) && aligned16(c->V_open) && aligned16(c->n_proxy) &&
         aligned16(c->n_open);
}

struct AppendWs {
  bf16* Y;
  float* Hf;
  bf16* Hb;
  float* sk;  // split-K partials of the compression GEMMs (M = batch rows only)
  size_t skb;
};

AppendWs carve_append(Carve& c, const pf_decode_desc& s) {
  AppendWs w{};
  const long k1 = s.levels == 2 ? s.k1 : s.P, k2 = s.levels == 2 ? s.k2 : 1;
  if (s.levels == 2) w.Y = c.take<bf16>((size_t)s.batch * k2 * s.d);
  w.Hf = c.take<float>((size_t)s.batch * s.d);
  w.Hb = c.take<bf16>((size_t)s.batch * s.d);
  w.skb = splitk_scratch_bytes((int)(s.batch * k2), s.d, (int)(k1 * s.d));
  if (s.levels == 2)
    w.skb = std::max(w.skb, splitk_scratch_bytes(s.batch, s.d, (int)(k2 * s.d)));
  w.sk = c.take<float>(w.skb / sizeof(float));
  return w;
}

}  // namespace

extern "C" {

size_t proxy_decode_workspace_size(const pf_decode_desc* desc) {
  if (check_decode_desc(desc) != PF_OK) return 0;
  const int splits = decode_splits(desc->batch, desc->n_heads, desc->capacity);
  return decode_workspace_bytes(desc->batch, desc->d, desc->n_heads, splits);
}

size_t proxy_append_workspace_size(const pf_decode_desc* desc) {
  if (check_decode_desc(desc) != PF_OK) return 0;
  Carve c(nullptr);
  carve_append(c, *desc);
  return ((c.off + 255) & ~size_t(255)) + 256;
}

pf_status proxy_decode_step(const pf_decode_desc* desc, const pf_decode_params* prm,
                            const void* x, pf_kv_cache* cache, void* y, void* ws, size_t ws_bytes,
                            void* stream) {
  pf_status st = check_decode_desc(desc);
  if (st != PF_OK) return st;
  if (!prm || !prm->W_qkv || !prm->W_o || !prm->rms_w || !prm->W_a1 || !prm->b_a1 || !prm->W_a2 ||
      !prm->b_a2)
    return fail(PF_ERR_INVALID_ARG, "a decode parameter is NULL");
  if (!x || !y || !cache_ok(cache) || !aligned16(x) || !aligned16(y) || !aligned16(ws) ||
      !aligned16(prm->W_qkv) || !aligned16(prm->W_o) || !aligned16(prm->rms_w) ||
      !aligned16(prm->W_a1) || !aligned16(prm->b_a1) || !aligned16(prm->W_a2) ||
      !aligned16(prm->b_a2))
    return fail(PF_ERR_INVALID_ARG, "x, y and every cache buffer are required, 16-byte aligned");
  const size_t need = proxy_decode_workspace_size(desc);
  if (ws == nullptr || ws_bytes < need)
    return fail(PF_ERR_WORKSPACE, "workspace too small: need %zu bytes, got %zu", need, ws_bytes);
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  DecodeLaunch L{};
  L.B = desc->batch;
  L.d = desc->d;
  L.nh = desc->n_heads;
  L.P = desc->P;
  L.cap = desc->capacity;
  L.splits = decode_splits(desc->batch, desc->n_heads, desc->capacity);
  L.x = static_cast<const bf16*>(x);
  L.y = static_cast<bf16*>(y);
  L.W_qkv = static_cast<const bf16*>(prm->W_qkv);
  L.W_o = static_cast<const bf16*>(prm->W_o);
  L.W_a1 = static_cast<const bf16*>(prm->W_a1);
  L.W_a2 = static_cast<const bf16*>(prm->W_a2);
  L.rms_w = prm->rms_w;
  L.b_a1 = prm->b_a1;
  L.b_a2 = prm->b_a2;
  L.K_proxy = static_cast<const bf16*>(cache->K_proxy);
  L.V_proxy = static_cast<const bf16*>(cache->V_proxy);
  L.X_open = static_cast<bf16*>(cache->X_open);
  L.K_open = static_cast<bf16*>(cache->K_open);
  L.V_open = static_cast<bf16*>(cache->V_open);
  L.n_proxy = cache->n_proxy;
  L.n_open = cache->n_open;
  L.ws = static_cast<float*>(ws);
  PF_CUDA(decode_step_launch(L, cs));
  return PF_OK;
}

pf_status proxy_kv_append(const pf_decode_desc* desc, const pf_append_params* prm,
                          const float* H_in, pf_kv_cache* cache, void* ws, size_t ws_bytes,
                          void* stream) {
  pf_status st = check_decode_desc(desc);
  if (st != PF_OK) return st;
  const pf_decode_desc& s = *desc;
  if (!prm || !prm->W_c1 || !prm->b_c1 || !prm->W_kvh ||
      (s.levels == 2 && (!prm->W_c2 || !prm->b_c2)))
    return fail(PF_ERR_INVALID_ARG, "an append parameter is NULL");
  if (!cache_ok(cache) || !aligned16(H_in) || !aligned16(ws) || !aligned16(prm->W_c1) ||
      !aligned16(prm->b_c1) || !aligned16(prm->W_c2) || !aligned16(prm->b_c2) ||
      !aligned16(prm->W_kvh))
    return fail(PF_ERR_INVALID_ARG, "every cache buffer is required; buffers 16-byte aligned");
  Carve wc(ws);
  const AppendWs w = carve_append(wc, s);
  if (ws == nullptr || wc.off > ws_bytes)
    return fail(PF_ERR_WORKSPACE, "workspace too small: need %zu bytes, got %zu", wc.off, ws_bytes);
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  const int B = s.batch, d = s.d, P = s.P;
  const long k1 = s.levels == 2 ? s.k1 : s.P, k2 = s.levels == 2 ? s.k2 : 1;
  const bf16* Xo = static_cast<const bf16*>(cache->X_open);
  // compression of the open block (Eq. compress-linear / factor-cascade),
  // H = H_in + C (Eq. proxy-res)
  if (s.levels == 1) {
    EpiLinearArgs e;
    e.bias = prm->b_c1;
    e.addend = H_in;
    e.ld_add = d;
    e.out_f32 = w.Hf;
    e.ld_f32 = d;
    e.out_bf16 = w.Hb;
    e.ld_bf16 = d;
    set_gemm_tag("append_compress_c1", (double)B * d * 10.0);
    PF_CUDA(gemm_linear(B, d, (int)(k1 * d), {Xo, k1 * d, 0},
                        {static_cast<const bf16*>(prm->W_c1), k1 * d, 0}, with_sk(e, w.sk, w.skb),
                        cs));
  } else {
    EpiLinearArgs e;
    e.bias = prm->b_c1;
    e.out_bf16 = w.Y;
    e.ld_bf16 = d;
    set_gemm_tag("append_compress_c1", (double)B * k2 * d * 2.0);
    PF_CUDA(gemm_linear((int)(B * k2), d, (int)(k1 * d), {Xo, k1 * d, 0},
                        {static_cast<const bf16*>(prm->W_c1), k1 * d, 0}, with_sk(e, w.sk, w.skb),
                        cs));
    EpiLinearArgs e2;
    e2.bias = prm->b_c2;
    e2.addend = H_in;
    e2.ld_add = d;
    e2.out_f32 = w.Hf;
    e2.ld_f32 = d;
    e2.out_bf16 = w.Hb;
    e2.ld_bf16 = d;
    set_gemm_tag("append_compress_c2", (double)B * d * 10.0);
    PF_CUDA(gemm_linear(B, d, (int)(k2 * d), {w.Y, k2 * d, 0},
                        {static_cast<const bf16*>(prm->W_c2), k2 * d, 0}, with_sk(e2, w.sk, w.skb),
                        cs));
  }
  // the proxy's key and value rows into cache row n_proxy[b]
  {
    EpiAppendArgs e{static_cast<bf16*>(cache->K_proxy), static_cast<bf16*>(cache->V_proxy),
                    cache->n_open, cache->n_proxy, d, P, s.capacity};
    set_gemm_tag("append_kv", (double)B * 2 * d * 2.0);
    PF_CUDA(gemm_append_kv(B, 2 * d, d, {w.Hb, d, 0}, {static_cast<const bf16*>(prm->W_kvh), d, 0},
                           e, cs));
  }
  PF_CUDA(append_finish(cache->n_open, cache->n_proxy, B, P, s.capacity, cs));
  return PF_OK;
}

// ---------------------------------------------------------------- prefill
namespace {

struct PrefillWs {
  bf16 *Xc, *Y, *Hb;  // gathered blocks [B m P, d] (remainder and B > 1), level-1 rows
                      // [B m k2, d] (two levels), proxies [B m, d]
};

PrefillWs carve_prefill(Carve& c, const pf_decode_desc& s, long L_hist) {
  PrefillWs w{};
  const long m = L_hist / s.P, r = L_hist - m * s.P, B = s.batch;
  const long k2 = s.levels == 2 ? s.k2 : 1;
  if (r > 0 && B > 1) w.Xc = c.take<bf16>((size_t)B * m * s.P * s.d);
  if (s.levels == 2) w.Y = c.take<bf16>((size_t)B * m * k2 * s.d);
  w.Hb = c.take<bf16>((size_t)B * m * s.d);
  return w;
}

// The tail of a prefill: each sequence's last r = L_hist mod P tokens become
// its open block (features, W_k x, W_v x with the decode W_qkv), and the
// counters are set to m = floor(L_hist / P) proxies and r open tokens.
pf_status prefill_open(const pf_decode_desc& s, const pf_decode_params* dp, const bf16* X,
                       long L_hist, pf_kv_cache* cache, cudaStream_t cs) {
  const long P = s.P, d = s.d, B = s.batch;
  const long m = L_hist / P, r = L_hist - m * P;
  for (long b = 0; b < B && r > 0; ++b) {
    const bf16* Xr = X + (b * L_hist + m * P) * d;
    bf16* Xo = static_cast<bf16*>(cache->X_open) + b * P * d;
    PF_CUDA(cudaMemcpyAsync(Xo, Xr, (size_t)r * d * sizeof(bf16), cudaMemcpyDeviceToDevice, cs));
    const bf16* Wqkv = static_cast<const bf16*>(dp->W_qkv);
    for (int kv = 0; kv < 2; ++kv) {
      EpiLinearArgs e;
      e.out_bf16 = static_cast<bf16*>(kv ? cache->V_open : cache->K_open) + b * P * d;
      e.ld_bf16 = d;
      set_gemm_tag("prefill_open_kv", (double)r * d * 2.0);
      PF_CUDA(gemm_linear((int)r, (int)d, (int)d, {Xr, d, 0}, {Wqkv + (1 + kv) * d * d, d, 0}, e,
                          cs));
    }
  }
  PF_CUDA(prefill_counts(cache->n_open, cache->n_proxy, (int)B, (int)m, (int)r, cs));
  return PF_OK;
}

}  // namespace

size_t proxy_prefill_workspace_size(const pf_decode_desc* desc, int32_t L_hist) {
  if (check_decode_desc(desc) != PF_OK || L_hist < 0) return 0;
  Carve c(nullptr);
  carve_prefill(c, *desc, L_hist);
  return ((c.off + 255) & ~size_t(255)) + 256;
}

pf_status proxy_kv_prefill(const pf_decode_desc* desc, const pf_append_params* ap,
                           const pf_decode_params* dp, const void* X_hist, int32_t L_hist,
                           const float* H_in, pf_kv_cache* cache, void* ws, size_t ws_bytes,
                           void* stream) {
  pf_status st = check_decode_desc(desc);
  if (st != PF_OK) return st;
  const pf_decode_desc& s = *desc;
  if (L_hist < 0) return fail(PF_ERR_INVALID_ARG, "L_hist must be >= 0");
  const long P = s.P, d = s.d, B = s.batch;
  const long m = L_hist / P, r = L_hist - m * P;
  if (m > s.capacity)
    return fail(PF_ERR_CAPACITY, "history of %d tokens needs %ld proxies; capacity %d", L_hist, m,
                s.capacity);
  if (!ap || !ap->W_c1 || !ap->b_c1 || !ap->W_kvh || (s.levels == 2 && (!ap->W_c2 || !ap->b_c2)))
    return fail(PF_ERR_INVALID_ARG, "an append parameter is NULL");
  if (r > 0 && (!dp || !dp->W_qkv))
    return fail(PF_ERR_INVALID_ARG, "the decode W_qkv is required for an open remainder");
  if ((L_hist > 0 && X_hist == nullptr) || !cache_ok(cache) || !aligned16(X_hist) ||
      !aligned16(H_in) || !aligned16(ws) || !aligned16(ap->W_c1) || !aligned16(ap->b_c1) ||
      !aligned16(ap->W_c2) || !aligned16(ap->b_c2) || !aligned16(ap->W_kvh) ||
      (dp && !aligned16(dp->W_qkv)))
    return fail(PF_ERR_INVALID_ARG, "every cache buffer is required; buffers 16-byte aligned");
  Carve wc(ws);
  const PrefillWs w = carve_prefill(wc, s, L_hist);
  if ((m > 0 && ws == nullptr) || wc.off > ws_bytes)
    return fail(PF_ERR_WORKSPACE, "workspace too small: need %zu bytes, got %zu", wc.off, ws_bytes);
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  const long k1 = s.levels == 2 ? s.k1 : P, k2 = s.levels == 2 ? s.k2 : 1;
  const bf16* X = static_cast<const bf16*>(X_hist);
  const bf16* Wkv = static_cast<const bf16*>(ap->W_kvh);
  if (m > 0) {
    // all sequences' complete blocks as one matrix of rows of k1 tokens:
    // in place when they are contiguous, else gathered
    const bf16* Xb = X;
    if (r > 0 && B > 1) {
      PF_CUDA(cudaMemcpy2DAsync(w.Xc, (size_t)m * P * d * sizeof(bf16), X,
                                (size_t)L_hist * d * sizeof(bf16), (size_t)m * P * d * sizeof(bf16),
                                (size_t)B, cudaMemcpyDeviceToDevice, cs));
      Xb = w.Xc;
    }
    // the proxies H = H_in + C(block) (Eq. proxy-res, Eq. compress-linear /
    // factor-cascade), rows (b, i) in sequence order.  H_in has ceil(L_hist/P)
    // rows per sequence: with a partial block and several sequences its rows
    // are not those of the output, and the last GEMM runs per sequence.
    const long mh = m + (r > 0 ? 1 : 0);
    const bool per_seq = H_in != nullptr && mh != m && B > 1;
    const bf16* Wc1 = static_cast<const bf16*>(ap->W_c1);
    if (s.levels == 2) {
      EpiLinearArgs e;
      e.bias = ap->b_c1;
      e.out_bf16 = w.Y;
      e.ld_bf16 = d;
      set_gemm_tag("prefill_compress_c1", (double)B * m * k2 * d * 2.0);
      PF_CUDA(gemm_linear((int)(B * m * k2), (int)d, (int)(k1 * d), {Xb, k1 * d, 0},
                          {Wc1, k1 * d, 0}, e, cs));
    }
    // the last level: W_c1 over the blocks (one level) or W_c2 over the
    // level-1 rows (two levels), plus b and H_in
    const bf16* A = s.levels == 2 ? w.Y : Xb;
    const long lda = s.levels == 2 ? k2 * d : k1 * d;
    const bf16* Wl = s.levels == 2 ? static_cast<const bf16*>(ap->W_c2) : Wc1;
    const float* bl = s.levels == 2 ? ap->b_c2 : ap->b_c1;
    for (long b = 0; b < (per_seq ? B : 1); ++b) {
      EpiLinearArgs e;
      e.bias = bl;
      e.addend = H_in ? H_in + b * mh * d : nullptr;
      e.ld_add = d;
      e.out_bf16 = w.Hb + b * m * d;
      e.ld_bf16 = d;
      const long rows = per_seq ? m : B * m;
      set_gemm_tag(s.levels == 2 ? "prefill_compress_c2" : "prefill_compress_c1",
                   (double)rows * d * 2.0);
      PF_CUDA(gemm_linear((int)rows, (int)d, (int)lda, {A + b * m * lda, lda, 0}, {Wl, lda, 0},
                          e, cs));
    }
    // their key and value rows into cache rows 0..m-1 of each sequence (one
    // GEMM over all sequences when the cache rows are contiguous, m = capacity)
    const bool whole = m == s.capacity;
    for (long b = 0; b < (whole ? 1 : B); ++b)
      for (int kv = 0; kv < 2; ++kv) {
        EpiLinearArgs e;
        e.out_bf16 =
            static_cast<bf16*>(kv ? cache->V_proxy : cache->K_proxy) + b * (long)s.capacity * d;
        e.ld_bf16 = d;
        const long rows = whole ? B * m : m;
        set_gemm_tag("prefill_kv", (double)rows * d * 2.0);
        PF_CUDA(gemm_linear((int)rows, (int)d, (int)d, {w.Hb + b * m * d, d, 0},
                            {Wkv + kv * d * d, d, 0}, e, cs));
      }
  }
  return prefill_open(s, dp, X, L_hist, cache, cs);
}

pf_status proxy_layer_prefill(const pf_layer_desc* desc, const pf_layer_params* prm,
                              const pf_decode_desc* cdesc, const pf_decode_params* dp,
                              const void* X, const float* H_in, void* X_out, float* H_out,
                              pf_kv_cache* cache, void* ws, size_t ws_bytes, void* stream) {
  pf_status st = check_desc(desc);
  if (st != PF_OK) return st;
  st = check_decode_desc(cdesc);
  if (st != PF_OK) return st;
  const pf_layer_desc& s = *desc;
  const pf_decode_desc& c = *cdesc;
  if (s.mode != PF_CAUSAL_1D || s.dtype != PF_BF16 || (s.d_fine > 0 && s.d_fine != s.d) ||
      s.interact != PF_F_ATTENTION || s.rope)
    return fail(PF_ERR_UNSUPPORTED,
                "prefill needs a causal 1D bf16 attention layer with d_fine == d, no RoPE");
  if (c.batch != s.batch || c.d != s.d || c.n_heads != s.n_heads || c.P != s.P ||
      c.levels != s.levels || (s.levels == 2 && (c.k1 != s.k1 || c.k2 != s.k2)))
    return fail(PF_ERR_INVALID_ARG, "the cache descriptor does not match the layer");
  const Dims g = dims_of(s);
  const long m = s.L / s.P, r = s.L - m * s.P, d = s.d, B = s.batch;
  if (m > c.capacity)
    return fail(PF_ERR_CAPACITY, "history of %ld tokens needs %ld proxies; capacity %d", (long)s.L,
                m, c.capacity);
  if (r > 0 && (!dp || !dp->W_qkv || !aligned16(dp->W_qkv)))
    return fail(PF_ERR_INVALID_ARG, "the decode W_qkv is required for an open remainder");
  if (!cache_ok(cache)) return fail(PF_ERR_INVALID_ARG, "every cache buffer is required, 16-byte aligned");
  // the layer's inference forward; its proxy attention projects K and V of
  // the proxies H = H_in + C(block) into the saved-activation area of ws
  st = proxy_layer_fwd(desc, prm, X, H_in, nullptr, X_out, H_out, nullptr, ws, ws_bytes, stream);
  if (st != PF_OK) return st;
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  Carve wc(ws);
  const bf16* QKV = carve_fwd(wc, s, g, nullptr).sv.QKV;  // [B, ceil(L/P), 3d]
  // complete blocks' key and value columns into cache rows 0..m-1
  const bool whole = m == g.m && m == c.capacity;  // source and cache rows both contiguous
  for (long b = 0; b < (whole ? 1 : B) && m > 0; ++b)
    for (int kv = 0; kv < 2; ++kv) {
      bf16* dst = static_cast<bf16*>(kv ? cache->V_proxy : cache->K_proxy) + b * c.capacity * d;
      const bf16* src = QKV + b * g.m * 3 * d + (1 + kv) * d;
      PF_CUDA(cudaMemcpy2DAsync(dst, d * sizeof(bf16), src, 3 * d * sizeof(bf16),
                                d * sizeof(bf16), whole ? B * m : m, cudaMemcpyDeviceToDevice, cs));
    }
  return prefill_open(c, dp, static_cast<const bf16*>(X), s.L, cache, cs);
}

// ------------------------------------------- temporal-distance ratios (Sec. 3.6)
namespace {

struct Seg {
  long L, P, k1, k2, m, off, g0, rows1, N1;
  bool ragged;
};
struct SegPlan {
  long d, nh, M;
  int levels;
  bool gated;
  std::vector<Seg> s;
};

pf_status seg_plan(const pf_layer_desc* desc, int32_t n, const pf_segment* segs, SegPlan& p) {
  pf_status st = check_desc(desc);
  if (st != PF_OK) return st;
  const pf_layer_desc& q = *desc;
  if (q.batch != 1 || q.mode != PF_CAUSAL_1D || q.dtype != PF_BF16 ||
      (q.inject != PF_INJ_GATED && q.inject != PF_INJ_ADD) || q.interact != PF_F_ATTENTION ||
      q.rope || (q.d_fine > 0 && q.d_fine != q.d))
    return fail(PF_ERR_UNSUPPORTED,
                "segments need batch 1, causal 1D, bf16, gated or add injection, attention");
  if (n < 1 || segs == nullptr) return fail(PF_ERR_INVALID_ARG, "no segments");
  p.d = q.d;
  p.nh = q.n_heads;
  p.levels = q.levels;
  p.gated = q.inject == PF_INJ_GATED;
  p.s.clear();
  long off = 0, g0 = 0;
  for (int i = 0; i < n; ++i) {
    const pf_segment& a = segs[i];
    if (a.L < 1 || a.P < 1) return fail(PF_ERR_INVALID_ARG, "segment %d: L and P must be >= 1", i);
    if (q.levels == 2 && (a.k1 < 1 || a.k2 < 1 || (long)a.k1 * a.k2 != a.P))
      return fail(PF_ERR_INVALID_ARG, "segment %d: levels == 2 needs k1 * k2 == P", i);
    if (i + 1 < n && a.L % a.P != 0)
      return fail(PF_ERR_INVALID_ARG, "segment %d: only the last segment may end mid-block", i);
    Seg g;
    g.L = a.L;
    g.P = a.P;
    g.k1 = q.levels == 2 ? a.k1 : a.P;
    g.k2 = q.levels == 2 ? a.k2 : 1;
    g.m = (a.L + a.P - 1) / a.P;
    g.off = off;
    g.g0 = g0;
    g.rows1 = g.m * g.k2;
    g.N1 = g.k1 * q.d;
    g.ragged = g.m * g.P != g.L;
    if (g.N1 > (1L << 30)) return fail(PF_ERR_UNSUPPORTED, "segment %d too large", i);
    p.s.push_back(g);
    off += a.L;
    g0 += g.m;
  }
  if (off != q.L) return fail(PF_ERR_INVALID_ARG, "segment lengths sum to %ld, desc L is %d", off, q.L);
  p.M = g0;
  return PF_OK;
}

struct SegSaved {
  bf16 *Hb, *QKV, *Aatt, *Hbar;
  float* LSE;
  std::vector<bf16*> Y, Z, D;
};

SegSaved carve_seg_saved(Carve& c, const SegPlan& p) {
  SegSaved v;
  v.Hb = c.take<bf16>(p.M * p.d);
  v.QKV = c.take<bf16>(p.M * 3 * p.d);
  v.Aatt = c.take<bf16>(p.M * p.d);
  v.Hbar = c.take<bf16>(p.M * p.d);
  v.LSE = c.take<float>(p.nh * p.M);
  for (const Seg& g : p.s) {
    v.Y.push_back(p.levels == 2 ? c.take<bf16>(g.rows1 * p.d) : nullptr);
    v.Z.push_back(p.levels == 2 ? c.take<bf16>(g.m * g.k2 * p.d) : nullptr);
    v.D.push_back(c.take<bf16>(g.rows1 * g.N1));
  }
  return v;
}

size_t seg_splitk(const SegPlan& p, bool bwd) {
  const int d = (int)p.d, M = (int)p.M;
  std::vector<std::array<int, 3>> v;
  if (!bwd) v = {{M, 3 * d, d}, {M, d, d}};
  else v = {{d, d, M}, {M, d, d}, {3 * d, d, M}, {M, d, 3 * d}};
  for (const Seg& g : p.s) {
    const int m = (int)g.m, r1 = (int)g.rows1, N1 = (int)g.N1, n2 = (int)(g.k2 * d);
    if (!bwd) {
      v.push_back({r1, d, N1});
      if (p.levels == 2) v.insert(v.end(), {{m, d, n2}, {m, n2, d}});
    } else {
      v.insert(v.end(), {{N1, d, r1}, {r1, d, N1}, {d, N1, r1}});
      if (p.levels == 2) v.insert(v.end(), {{n2, d, m}, {m, d, n2}, {d, n2, m}, {m, n2, d}});
    }
  }
  size_t b = 0;
  for (const auto& x : v) b = std::max(b, splitk_scratch_bytes(x[0], x[1], x[2]));
  return b;
}

struct SegFwdWs {
  bf16* Xpad;  // the last segment, zero-padded to whole blocks (if ragged)
  float* sk;
  size_t skb;
  SegSaved sv;
};

SegFwdWs carve_seg_fwd(Carve& wc, const SegPlan& p, void* saved) {
  SegFwdWs f;
  const Seg& z = p.s.back();
  f.Xpad = z.ragged ? wc.take<bf16>(z.m * z.P * p.d) : nullptr;
  f.skb = seg_splitk(p, false);
  f.sk = wc.take<float>(f.skb / sizeof(float));
  Carve sc(saved);
  f.sv = saved ? carve_seg_saved(sc, p) : carve_seg_saved(wc, p);
  return f;
}

struct SegBwdWs {
  bf16 *Xpad, *dXpad, *dD, *dZ, *dHbar, *dA, *dQKV, *dHb, *dY;
  float *Di, *dHf, *part, *sk, *gtmp, *gsum;
  size_t skb;
};

SegBwdWs carve_seg_bwd(Carve& c, const SegPlan& p) {
  SegBwdWs w{};
  const Seg& z = p.s.back();
  long dD = 0, dZ = 0, dY = 0, pe = 0;
  for (const Seg& g : p.s) {
    dD = std::max(dD, g.rows1 * g.N1);
    dZ = std::max(dZ, g.m * g.k2 * p.d);
    dY = std::max(dY, g.rows1 * p.d);
    pe = std::max(pe, (long)inj_bwd_chunks(g.rows1, (int)g.N1) * 4 * g.N1);
    pe = std::max(pe, colsum_part_elems(g.m, (int)(g.k2 * p.d)));
    pe = std::max(pe, colsum_part_elems(g.m, (int)p.d));
    pe = std::max(pe, colsum_part_elems(g.rows1, (int)p.d));
  }
  pe = std::max(pe, colsum_part_elems((long)p.s.size(), (int)(3 * p.d)));
  w.Xpad = z.ragged ? c.take<bf16>(z.m * z.P * p.d) : nullptr;
  w.dXpad = z.ragged ? c.take<bf16>(z.m * z.P * p.d) : nullptr;
  w.dD = c.take<bf16>(dD);
  if (p.levels == 2) w.dZ = c.take<bf16>(dZ);
  w.dHbar = c.take<bf16>(p.M * p.d);
  w.dA = c.take<bf16>(p.M * p.d);
  w.dQKV = c.take<bf16>(p.M * 3 * p.d);
  w.dHb = c.take<bf16>(p.M * p.d);
  if (p.levels == 2) w.dY = c.take<bf16>(dY);
  w.Di = c.take<float>(p.nh * p.M);
  w.dHf = c.take<float>(p.M * p.d);
  w.part = c.take<float>(pe);
  w.skb = seg_splitk(p, true);
  w.sk = c.take<float>(w.skb / sizeof(float));
  w.gtmp = c.take<float>((long)p.s.size() * 3 * p.d);
  w.gsum = c.take<float>(3 * p.d);
  return w;
}

bool seg_params_ok(const SegPlan& p, const pf_segment_params* sp) {
  if (!sp) return false;
  for (size_t i = 0; i < p.s.size(); ++i) {
    const pf_segment_params& a = sp[i];
    if (!a.W_c1 || !a.b_c1 || !a.W_d1 || !a.b_d1 ||
        (p.levels == 2 && (!a.W_c2 || !a.b_c2 || !a.W_d2 || !a.b_d2)))
      return false;
    const void* ptrs[] = {a.W_c1, a.b_c1, a.W_c2, a.b_c2, a.W_d1, a.b_d1, a.W_d2, a.b_d2};
    for (const void* q : ptrs)
      if (!aligned16(q)) return false;
  }
  return true;
}

// the source rows of segment i's decompression: proxy g0 - 1 onwards, or for
// the first segment proxy 0 onwards with the usual one-block routing shift
const bf16* seg_src(const SegSaved& sv, const SegPlan& p, size_t i) {
  return i == 0 ? sv.Hbar : sv.Hbar + (p.s[i].g0 - 1) * p.d;
}

}  // namespace

size_t proxy_segments_saved_size(const pf_layer_desc* desc, int32_t n_seg, const pf_segment* segs) {
  SegPlan p;
  if (seg_plan(desc, n_seg, segs, p) != PF_OK) return 0;
  Carve c(nullptr);
  carve_seg_saved(c, p);
  return (c.off + 255) & ~size_t(255);
}

size_t proxy_segments_workspace_size(const pf_layer_desc* desc, int32_t n_seg,
                                     const pf_segment* segs, int for_backward) {
  SegPlan p;
  if (seg_plan(desc, n_seg, segs, p) != PF_OK) return 0;
  Carve c(nullptr);
  if (for_backward)
    carve_seg_bwd(c, p);
  else
    carve_seg_fwd(c, p, nullptr);
  return ((c.off + 255) & ~size_t(255)) + 256;
}

pf_status proxy_segments_fwd(const pf_layer_desc* desc, int32_t n_seg, const pf_segment* segs,
                             const pf_layer_params* prm, const pf_segment_params* sp,
                             const void* X, void* X_out, void* saved, void* ws, size_t ws_bytes,
                             void* stream) {
  SegPlan p;
  pf_status st = seg_plan(desc, n_seg, segs, p);
  if (st != PF_OK) return st;
  if (!prm || !prm->W_qkv || !prm->W_o || (p.gated && (!prm->w_x || !prm->w_dlt || !prm->b_g)) ||
      !seg_params_ok(p, sp) || !X || !X_out || X == X_out || !params_aligned(*prm) ||
      !aligned16(X) || !aligned16(X_out) || !aligned16(saved) || !aligned16(ws))
    return fail(PF_ERR_INVALID_ARG, "a parameter or buffer is NULL, aliased or misaligned");
  Carve wc(ws);
  const SegFwdWs f = carve_seg_fwd(wc, p, saved);
  if (ws == nullptr || wc.off > ws_bytes)
    return fail(PF_ERR_WORKSPACE, "workspace too small: need %zu bytes, got %zu", wc.off, ws_bytes);
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  const SegSaved& sv = f.sv;
  const int d = (int)p.d;
  const bf16* Xb = static_cast<const bf16*>(X);
  bf16* Xo = static_cast<bf16*>(X_out);
  // compression, segment by segment, into the proxies' rows g0 .. g0 + m - 1
  std::vector<const bf16*> xs(p.s.size());
  for (size_t i = 0; i < p.s.size(); ++i) {
    const Seg& g = p.s[i];
    const bf16* Xs = Xb + g.off * d;
    if (g.ragged) {
      PF_CUDA(pad_rows(Xs, f.Xpad, 1, g.L, g.m * g.P, d, cs));
      Xs = f.Xpad;
    }
    xs[i] = Xs;
    const bf16* W_c1 = static_cast<const bf16*>(sp[i].W_c1);
    EpiLinearArgs e;
    e.bias = sp[i].b_c1;
    e.ld_bf16 = d;
    if (p.levels == 1) {
      e.out_bf16 = sv.Hb + g.g0 * d;
      set_gemm_tag("seg_compress_c1", (double)g.m * d * 2.0);
      PF_CUDA(gemm_linear((int)g.m, d, (int)g.N1, {Xs, g.N1, 0}, {W_c1, g.N1, 0},
                          with_sk(e, f.sk, f.skb), cs));
    } else {
      const int n2 = (int)(g.k2 * d);
      e.out_bf16 = sv.Y[i];
      set_gemm_tag("seg_compress_c1", (double)g.rows1 * d * 2.0);
      PF_CUDA(gemm_linear((int)g.rows1, d, (int)g.N1, {Xs, g.N1, 0}, {W_c1, g.N1, 0},
                          with_sk(e, f.sk, f.skb), cs));
      EpiLinearArgs e2;
      e2.bias = sp[i].b_c2;
      e2.out_bf16 = sv.Hb + g.g0 * d;
      e2.ld_bf16 = d;
      set_gemm_tag("seg_compress_c2", (double)g.m * d * 2.0);
      PF_CUDA(gemm_linear((int)g.m, d, n2, {sv.Y[i], n2, 0},
                          {static_cast<const bf16*>(sp[i].W_c2), n2, 0}, with_sk(e2, f.sk, f.skb),
                          cs));
    }
  }
  // one causal attention over all proxies in time order (Eq. proxy-attn)
  {
    EpiLinearArgs e;
    e.out_bf16 = sv.QKV;
    e.ld_bf16 = 3 * d;
    set_gemm_tag("proxy_qkv", (double)p.M * 3 * d * 2.0);
    PF_CUDA(gemm_linear((int)p.M, 3 * d, d, {sv.Hb, d, 0},
                        {static_cast<const bf16*>(prm->W_qkv), d, 0}, with_sk(e, f.sk, f.skb), cs));
    PF_CUDA(attn_fwd(sv.QKV, sv.Aatt, sv.LSE, 1, (int)p.M, d, (int)p.nh, true, cs));
    EpiLinearArgs eo;
    eo.out_bf16 = sv.Hbar;
    eo.ld_bf16 = d;
    set_gemm_tag("proxy_o", (double)p.M * d * 2.0);
    PF_CUDA(gemm_linear((int)p.M, d, d, {sv.Aatt, d, 0}, {static_cast<const bf16*>(prm->W_o), d, 0},
                        with_sk(eo, f.sk, f.skb), cs));
  }
  // decompression and injection, each block through its own segment's weights
  for (size_t i = 0; i < p.s.size(); ++i) {
    const Seg& g = p.s[i];
    const bf16* src = seg_src(sv, p, i);
    const bf16* Zsrc = src;
    if (p.levels == 2) {
      const int n2 = (int)(g.k2 * d);
      EpiLinearArgs e;
      e.bias = sp[i].b_d2;
      e.out_bf16 = sv.Z[i];
      e.ld_bf16 = n2;
      set_gemm_tag("seg_decompress_d2", (double)g.m * n2 * 2.0);
      PF_CUDA(gemm_linear((int)g.m, n2, d, {src, d, 0}, {static_cast<const bf16*>(sp[i].W_d2), d, 0},
                          with_sk(e, f.sk, f.skb), cs));
      Zsrc = sv.Z[i];
    }
    EpiInjectArgs e{sp[i].b_d1, sv.D[i], xs[i], Xo + g.off * d, prm->w_x, prm->w_dlt, prm->b_g,
                    d, (int)g.k1, (int)g.k2, (int)g.m, (int)g.L, i == 0 ? 1 : 0, p.gated ? 1 : 0};
    set_gemm_tag("seg_decompress_d1_inject", (double)g.rows1 * g.N1 * 8.0);
    PF_CUDA(gemm_inject1d((int)g.rows1, (int)g.N1, d, {Zsrc, d, 0},
                          {static_cast<const bf16*>(sp[i].W_d1), d, 0}, e, cs));
  }
  const Seg& g0 = p.s.front();
  PF_CUDA(copy_block0(Xb, g0.L, Xo, g0.L, 1, d, (int)std::min(g0.P, g0.L), cs));
  return PF_OK;
}

pf_status proxy_segments_bwd(const pf_layer_desc* desc, int32_t n_seg, const pf_segment* segs,
                             const pf_layer_params* prm, const pf_segment_params* sp,
                             const void* X, const void* saved, const void* dX_out, void* dX,
                             const pf_layer_grads* grads, const pf_segment_grads* sg, void* ws,
                             size_t ws_bytes, void* stream) {
  SegPlan p;
  pf_status st = seg_plan(desc, n_seg, segs, p);
  if (st != PF_OK) return st;
  if (!prm || !prm->W_qkv || !prm->W_o || (p.gated && (!prm->w_x || !prm->w_dlt || !prm->b_g)) ||
      !seg_params_ok(p, sp) || !X || !saved || !dX_out || !dX || !grads || !sg ||
      !params_aligned(*prm) || !aligned16(X) || !aligned16(saved) || !aligned16(dX_out) ||
      !aligned16(dX) || !aligned16(ws))
    return fail(PF_ERR_INVALID_ARG, "a parameter or buffer is NULL or misaligned");
  for (size_t i = 0; i < p.s.size(); ++i)
    if (!sg[i].b_d1) return fail(PF_ERR_INVALID_ARG, "seg_grads[%zu].b_d1 must be given", i);
  Carve wc(ws);
  const SegBwdWs w = carve_seg_bwd(wc, p);
  if (ws == nullptr || wc.off > ws_bytes)
    return fail(PF_ERR_WORKSPACE, "workspace too small: need %zu bytes, got %zu", wc.off, ws_bytes);
  Carve sc(const_cast<void*>(saved));
  const SegSaved sv = carve_seg_saved(sc, p);
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  const int d = (int)p.d;
  const bf16* Xb = static_cast<const bf16*>(X);
  const bf16* G = static_cast<const bf16*>(dX_out);
  bf16* dXb = static_cast<bf16*>(dX);
  const bf16* W_qkv = static_cast<const bf16*>(prm->W_qkv);
  const bf16* W_o = static_cast<const bf16*>(prm->W_o);
  // the last proxy feeds no block
  PF_CUDA(cudaMemsetAsync(w.dHbar + (p.M - 1) * d, 0, d * sizeof(bf16), cs));
  if (p.gated) PF_CUDA(cudaMemsetAsync(w.gtmp, 0, p.s.size() * 3 * d * sizeof(float), cs));
  std::vector<const bf16*> xs(p.s.size());
  std::vector<bf16*> dxd(p.s.size());
  // injection and decompression backward, segment by segment (segment 0 first:
  // its last proxy row, which feeds no block of its own, is overwritten by
  // segment 1's first source row)
  for (size_t i = 0; i < p.s.size(); ++i) {
    const Seg& g = p.s[i];
    const bf16* Xs = Xb + g.off * d;
    xs[i] = Xs;
    dxd[i] = dXb + g.off * d;
    if (g.ragged) {
      PF_CUDA(pad_rows(Xs, w.Xpad, 1, g.L, g.m * g.P, d, cs));
      xs[i] = w.Xpad;
      dxd[i] = w.dXpad;
    }
    const int N1 = (int)g.N1, r1 = (int)g.rows1;
    const int nch = inj_bwd_chunks(g.rows1, N1);
    InjBwdArgs a{G + g.off * d, Xs, sv.D[i], w.dD, dxd[i], g.ragged ? g.m * g.P : g.L, prm->w_x,
                 prm->w_dlt, prm->b_g, d, (int)g.k1, (int)g.k2, (int)g.m, (int)g.L, 1,
                 i == 0 ? 1 : 0, p.gated ? 1 : 0};
    PF_CUDA(inj_bwd_1d(a, w.part, nch, cs));
    if (i == 0)
      PF_CUDA(copy_block0(G, g.L, dxd[0], g.ragged ? g.m * g.P : g.L, 1, d,
                          (int)std::min(g.P, g.L), cs));
    float* gt = w.gtmp + i * 3 * d;
    PF_CUDA(inj_bwd_finalize(w.part, nch, N1, d, sg[i].b_d1, p.gated ? gt : nullptr,
                             p.gated ? gt + d : nullptr, p.gated ? gt + 2 * d : nullptr, cs));
    const bf16* src = seg_src(sv, p, i);
    bf16* dsrc = w.dHbar + (i == 0 ? 0 : (g.g0 - 1)) * d;
    const bf16* Zsrc = p.levels == 2 ? sv.Z[i] : src;
    if (sg[i].W_d1) {
      EpiLinearArgs e;
      e.out_f32 = sg[i].W_d1;
      e.ld_f32 = d;
      set_gemm_tag("seg_bwd_dW_d1", (double)N1 * d * 4.0);
      PF_CUDA(gemm_linear(N1, d, r1, {w.dD, N1, 1}, {Zsrc, d, 1}, with_sk(e, w.sk, w.skb), cs));
    }
    EpiLinearArgs e;
    e.out_bf16 = p.levels == 2 ? w.dZ : dsrc;
    e.ld_bf16 = d;
    set_gemm_tag("seg_bwd_dZ", (double)r1 * d * 2.0);
    PF_CUDA(gemm_linear(r1, d, N1, {w.dD, N1, 0}, {static_cast<const bf16*>(sp[i].W_d1), d, 1},
                        with_sk(e, w.sk, w.skb), cs));
    if (p.levels == 2) {
      const int n2 = (int)(g.k2 * d), m = (int)g.m;
      if (sg[i].b_d2) PF_CUDA(colsum_bf16(w.dZ, g.m, n2, sg[i].b_d2, w.part, cs));
      if (sg[i].W_d2) {
        EpiLinearArgs e2;
        e2.out_f32 = sg[i].W_d2;
        e2.ld_f32 = d;
        set_gemm_tag("seg_bwd_dW_d2", (double)n2 * d * 4.0);
        PF_CUDA(gemm_linear(n2, d, m, {w.dZ, n2, 1}, {src, d, 1}, with_sk(e2, w.sk, w.skb), cs));
      }
      EpiLinearArgs e3;
      e3.out_bf16 = dsrc;
      e3.ld_bf16 = d;
      set_gemm_tag("seg_bwd_dHbar", (double)m * d * 2.0);
      PF_CUDA(gemm_linear(m, d, n2, {w.dZ, n2, 0}, {static_cast<const bf16*>(sp[i].W_d2), d, 1},
                          with_sk(e3, w.sk, w.skb), cs));
    }
  }
  if (p.gated) {  // the gate vectors are shared: sum the segments' contributions
    PF_CUDA(colsum_f32(w.gtmp, (long)p.s.size(), 3 * d, w.gsum, w.part, cs));
    float* dst[3] = {grads->w_x, grads->w_dlt, grads->b_g};
    for (int k = 0; k < 3; ++k)
      if (dst[k])
        PF_CUDA(cudaMemcpyAsync(dst[k], w.gsum + k * d, d * sizeof(float),
                                cudaMemcpyDeviceToDevice, cs));
  }
  // the shared attention
  if (grads->W_o) {
    EpiLinearArgs e;
    e.out_f32 = grads->W_o;
    e.ld_f32 = d;
    set_gemm_tag("bwd_dW_o", (double)d * d * 4.0);
    PF_CUDA(gemm_linear(d, d, (int)p.M, {w.dHbar, d, 1}, {sv.Aatt, d, 1}, with_sk(e, w.sk, w.skb), cs));
  }
  {
    EpiLinearArgs e;
    e.out_bf16 = w.dA;
    e.ld_bf16 = d;
    set_gemm_tag("bwd_dA", (double)p.M * d * 2.0);
    PF_CUDA(gemm_linear((int)p.M, d, d, {w.dHbar, d, 0}, {W_o, d, 1}, with_sk(e, w.sk, w.skb), cs));
  }
  PF_CUDA(attn_bwd(sv.QKV, sv.Aatt, w.dA, sv.LSE, w.Di, w.dQKV, 1, (int)p.M, d, (int)p.nh, true,
                   cs));
  if (grads->W_qkv) {
    EpiLinearArgs e;
    e.out_f32 = grads->W_qkv;
    e.ld_f32 = d;
    set_gemm_tag("bwd_dW_qkv", (double)3 * d * d * 4.0);
    PF_CUDA(gemm_linear(3 * d, d, (int)p.M, {w.dQKV, 3 * d, 1}, {sv.Hb, d, 1},
                        with_sk(e, w.sk, w.skb), cs));
  }
  {
    EpiLinearArgs e;
    e.out_f32 = w.dHf;
    e.ld_f32 = d;
    e.out_bf16 = w.dHb;
    e.ld_bf16 = d;
    set_gemm_tag("bwd_dH", (double)p.M * d * 10.0);
    PF_CUDA(gemm_linear((int)p.M, d, 3 * d, {w.dQKV, 3 * d, 0}, {W_qkv, d, 1},
                        with_sk(e, w.sk, w.skb), cs));
  }
  // compression backward and dX, segment by segment
  for (size_t i = 0; i < p.s.size(); ++i) {
    const Seg& g = p.s[i];
    const int N1 = (int)g.N1, r1 = (int)g.rows1, m = (int)g.m;
    const bf16* dHb = w.dHb + g.g0 * d;
    const float* dHf = w.dHf + g.g0 * d;
    const bf16* dYsrc = dHb;
    if (p.levels == 2) {
      const int n2 = (int)(g.k2 * d);
      if (sg[i].b_c2) PF_CUDA(colsum_f32(dHf, g.m, d, sg[i].b_c2, w.part, cs));
      if (sg[i].W_c2) {
        EpiLinearArgs e;
        e.out_f32 = sg[i].W_c2;
        e.ld_f32 = n2;
        set_gemm_tag("seg_bwd_dW_c2", (double)d * n2 * 4.0);
        PF_CUDA(gemm_linear(d, n2, m, {dHb, d, 1}, {sv.Y[i], n2, 1}, with_sk(e, w.sk, w.skb), cs));
      }
      EpiLinearArgs e;
      e.out_bf16 = w.dY;
      e.ld_bf16 = n2;
      set_gemm_tag("seg_bwd_dY", (double)m * n2 * 2.0);
      PF_CUDA(gemm_linear(m, n2, d, {dHb, d, 0}, {static_cast<const bf16*>(sp[i].W_c2), n2, 1},
                          with_sk(e, w.sk, w.skb), cs));
      if (sg[i].b_c1) PF_CUDA(colsum_bf16(w.dY, g.rows1, d, sg[i].b_c1, w.part, cs));
      dYsrc = w.dY;
    } else if (sg[i].b_c1) {
      PF_CUDA(colsum_f32(dHf, g.m, d, sg[i].b_c1, w.part, cs));
    }
    if (sg[i].W_c1) {
      EpiLinearArgs e;
      e.out_f32 = sg[i].W_c1;
      e.ld_f32 = N1;
      set_gemm_tag("seg_bwd_dW_c1", (double)d * N1 * 4.0);
      PF_CUDA(gemm_linear(d, N1, r1, {dYsrc, d, 1}, {xs[i], N1, 1}, with_sk(e, w.sk, w.skb), cs));
    }
    EpiDXArgs e{dxd[i], dXb + g.off * d, d, (int)g.k1, (int)g.k2, (int)g.m, (int)g.L};
    set_gemm_tag("seg_bwd_dX", (double)r1 * N1 * 4.0);
    PF_CUDA(gemm_dx1d(r1, N1, d, {dYsrc, d, 0}, {static_cast<const bf16*>(sp[i].W_c1), N1, 1}, e,
                      cs));
  }
  return PF_OK;
}

pf_status pf_sync_check(void* stream) {
  PF_CUDA(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)));
  PF_CUDA(cudaGetLastError());
  int e = 0;
  for (int v : {take_dev_error_gemm(), take_dev_error_attention(), take_dev_error_attention_tc(),
                take_dev_error_attention_bwd_tc(),
                take_dev_error_elementwise(), take_dev_error_decode(), take_dev_error_fp32(),
                take_dev_error_layer2d()})
    if (v != 0 && e == 0) e = v;
  if (e < 0) return fail(PF_ERR_CUDA, "reading the device error flag failed");
  if (e == DEVERR_TIMEOUT) return fail(PF_ERR_TIMEOUT, "a kernel's bounded wait ran out");
  if (e == DEVERR_CAPACITY) return fail(PF_ERR_CAPACITY, "cache bookkeeping violated in a kernel");
  return PF_OK;
}

pf_status pf_debug_set_wait_limit_ns(unsigned long long ns) {
  if (ns == 0) ns = kWaitLimitNs;
  int bad = 0;
  for (int r : {set_wait_limit_gemm(ns), set_wait_limit_attention(ns),
                set_wait_limit_attention_tc(ns), set_wait_limit_attention_bwd_tc(ns),
                set_wait_limit_elementwise(ns), set_wait_limit_decode(ns), set_wait_limit_fp32(ns),
                set_wait_limit_layer2d(ns)})
    bad |= r;
  if (bad) return fail(PF_ERR_CUDA, "pf_debug_set_wait_limit_ns: writing the limit failed");
  return PF_OK;
}

pf_status pf_debug_gemm_skip_loads(int on) {
  if (set_debug_skip_loads_gemm(on ? 1 : 0))
    return fail(PF_ERR_CUDA, "pf_debug_gemm_skip_loads: writing the flag failed");
  return PF_OK;
}

pf_status pf_gemm_bf16(int M, int N, int K, const void* A, int a_mn, const void* B, int b_mn,
                       float* D, int ldd, void* stream) {
  if (M < 1 || N < 1 || K < 1 || N % 32 != 0 || !A || !B || !D || ldd < N || ldd % 4 != 0)
    return fail(PF_ERR_INVALID_ARG, "pf_gemm_bf16: bad sizes or pointers (N must be a multiple of 32)");
  const long lda = a_mn ? M : K, ldb = b_mn ? N : K;
  if ((lda * 2) % 16 || (ldb * 2) % 16)
    return fail(PF_ERR_INVALID_ARG, "pf_gemm_bf16: rows must be multiples of 16 bytes");
  EpiLinearArgs e;
  e.out_f32 = D;
  e.ld_f32 = ldd;
  set_gemm_tag("pf_gemm_bf16", (double)M * N * 4.0);
  PF_CUDA(gemm_linear(M, N, K, {static_cast<const bf16*>(A), lda, a_mn ? 1 : 0},
                      {static_cast<const bf16*>(B), ldb, b_mn ? 1 : 0}, e,
                      static_cast<cudaStream_t>(stream)));
  return PF_OK;
}

}  // extern "C"
