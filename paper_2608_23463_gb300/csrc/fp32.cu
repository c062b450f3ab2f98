// fp32 forward of the 1D layer (Alg. 1) on CUDA cores: a tiled SIMT GEMM for
// the compression / Q,K,V / output / decompression projections, an
// online-softmax proxy attention with one warp per query, and the routing +
// injection pass.  Used when the descriptor's dtype is PF_F32 (the tensor
// cores have no fp32 path that meets fp32 accuracy).
#include <algorithm>

#include "kernels.h"

namespace pf {

int take_dev_error_fp32() { return take_dev_error_tu(); }
int set_wait_limit_fp32(unsigned long long ns) { return set_wait_limit_tu(ns); }

namespace {

constexpr int FT = 64;   // output tile (FT x FT)
constexpr int FK = 32;   // K slab
constexpr int FTHREADS = 256;

// Routing + injection (Eq. inj-gate / inj-add) applied to the last
// decompression's output instead of storing it: output (row r, column c) of
// that GEMM is D for token (i + shift) * P + a * k1 + c / d, channel c % d of
// sequence b, with r = (b * m + i) * k2 + a.
struct InjF32 {
  const float* X;    // [B, L, d]
  float* Xo;         // null: a plain GEMM epilogue
  const float *w_x, *w_dlt, *b_g;
  long L;
  int d, P, k1, k2, m, shift, gated;
};

// C[M, N] = A[M, K] B[N, K]^T (+ bias[n]) (+ addend[m, n]), all row-major fp32
// with leading dimensions lda, ldb, ldc.  Each thread computes 4 x 4 outputs.
// The next K slab is fetched into registers while the current one is used
// (two shared-memory buffers, one barrier per slab); with `vec` the fetch
// uses 16-byte loads (lda, ldb, the K range and the pointers 4-aligned).
// With gridDim.z = S > 1 each z-slice reduces K range [z*Kc, (z+1)*Kc) and
// writes raw partials to C + z*M*ldc (bias / addend are then applied by
// splitk_f32_reduce).  With inj.Xo the epilogue injects instead of storing C.
__global__ void __launch_bounds__(FTHREADS) gemm_f32_kernel(const float* __restrict__ A, long lda,
                                                           const float* __restrict__ Bm, long ldb,
                                                           float* __restrict__ C, long ldc, int M,
                                                           int N, int K, int Kc,
                                                           const float* __restrict__ bias,
                                                           const float* __restrict__ addend,
                                                           long ld_add, int vec, InjF32 inj) {
  __shared__ __align__(16) float As[2][FK][FT + 4], Bs[2][FK][FT + 4];
  const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
  const int m0 = blockIdx.y * FT, n0 = blockIdx.x * FT;
  const int kbeg = blockIdx.z * Kc, kend = min(K, kbeg + Kc);
  C += (long)blockIdx.z * M * ldc;
  // thread t loads rows r = t / 8 + 32 i (i = 0, 1) and k = (t % 8) * 4 .. + 4
  const int lr = threadIdx.x >> 3, lk = (threadIdx.x & 7) * 4;
  float ra[2][4], rb[2][4];
  auto fetch = [&](int k0) {
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const int gm = m0 + lr + 32 * i, gn = n0 + lr + 32 * i;
      const int gk = k0 + lk;
      if (vec) {
        const float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
        const float4 va = (gm < M && gk < kend) ? *reinterpret_cast<const float4*>(A + (long)gm * lda + gk) : z;
        const float4 vb = (gn < N && gk < kend) ? *reinterpret_cast<const float4*>(Bm + (long)gn * ldb + gk) : z;
        ra[i][0] = va.x; ra[i][1] = va.y; ra[i][2] = va.z; ra[i][3] = va.w;
        rb[i][0] = vb.x; rb[i][1] = vb.y; rb[i][2] = vb.z; rb[i][3] = vb.w;
      } else {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          ra[i][e] = (gm < M && gk + e < kend) ? A[(long)gm * lda + gk + e] : 0.f;
          rb[i][e] = (gn < N && gk + e < kend) ? Bm[(long)gn * ldb + gk + e] : 0.f;
        }
      }
    }
  };
  auto stash = [&](int buf) {
#pragma unroll
    for (int i = 0; i < 2; ++i)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        As[buf][lk + e][lr + 32 * i] = ra[i][e];
        Bs[buf][lk + e][lr + 32 * i] = rb[i][e];
      }
  };
  float acc[4][4] = {};
  int buf = 0;
  if (kbeg < kend) {
    fetch(kbeg);
    stash(0);
  }
  __syncthreads();
  for (int k0 = kbeg; k0 < kend; k0 += FK) {
    const bool more = k0 + FK < kend;
    if (more) fetch(k0 + FK);  // in flight during the FMAs below
#pragma unroll
    for (int kk = 0; kk < FK; ++kk) {
      const float4 a4 = *reinterpret_cast<const float4*>(&As[buf][kk][ty * 4]);
      const float4 b4 = *reinterpret_cast<const float4*>(&Bs[buf][kk][tx * 4]);
      const float a[4] = {a4.x, a4.y, a4.z, a4.w}, b[4] = {b4.x, b4.y, b4.z, b4.w};
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    if (more) stash(buf ^ 1);
    __syncthreads();
    buf ^= 1;
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int gm = m0 + ty * 4 + i;
    if (gm >= M) continue;
    if (inj.Xo) {
      // row gm = (b * m + iprox) * k2 + a: the target block and first token
      const int a = gm % inj.k2, prox = gm / inj.k2;
      const int b = prox / inj.m, ip = prox % inj.m + inj.shift;
      const long tok0 = (long)ip * inj.P + (long)a * inj.k1;
      if (ip >= inj.m) continue;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int gn = n0 + tx * 4 + j;
        if (gn >= N) continue;
        const long t = tok0 + gn / inj.d;
        if (t >= inj.L) continue;
        const int ch = gn % inj.d;
        const float v = acc[i][j] + (bias ? bias[gn] : 0.f);
        const long o = ((long)b * inj.L + t) * inj.d + ch;
        const float x = inj.X[o];
        inj.Xo[o] = inj.gated
                        ? x + v / (1.f + expf(-(inj.w_x[ch] * x + inj.w_dlt[ch] * v + inj.b_g[ch])))
                        : x + v;
      }
      continue;
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int gn = n0 + tx * 4 + j;
      if (gn >= N) continue;
      float v = acc[i][j];
      if (bias) v += bias[gn];
      if (addend) v += addend[(long)gm * ld_add + gn];
      C[(long)gm * ldc + gn] = v;
    }
  }
}

// The same product with a CP_STAGES-deep ring of cp.async copies (16-byte,
// zero-filled past M, N and the K range), for 16-byte aligned operands with
// K, lda, ldb multiples of 4.  A and B tiles stay row-major in shared memory
// (rows 36 floats apart), and each thread reads four K values of a row with
// one 16-byte load, so a 4-deep K group costs eight shared loads for 64 FMAs.
// A thread owns rows 4 ty .. 4 ty + 3 and columns tx + 16 j: the B rows that
// eight consecutive lanes read are 36 floats apart, so their 16-byte loads
// fall in distinct banks (contiguous column quartets, 144 floats apart, would
// collide eight ways).
constexpr int CP_STAGES = 4;
constexpr int CP_LD = FK + 4;  // floats per row of a shared tile
constexpr int CP_SMEM = CP_STAGES * 2 * FT * CP_LD * 4;

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, bool valid) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src),
               "r"(valid ? 16 : 0)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

__global__ void __launch_bounds__(FTHREADS, 2) gemm_f32_cp_kernel(
    const float* __restrict__ A, long lda, const float* __restrict__ Bm, long ldb,
    float* __restrict__ C, long ldc, int M, int N, int K, int Kc, const float* __restrict__ bias,
    const float* __restrict__ addend, long ld_add, InjF32 inj) {
  extern __shared__ __align__(16) float cps[];
  float* As = cps;                              // [stage][FT][CP_LD]
  float* Bs = cps + CP_STAGES * FT * CP_LD;     // [stage][FT][CP_LD]
  const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
  const int m0 = blockIdx.y * FT, n0 = blockIdx.x * FT;
  const int kbeg = blockIdx.z * Kc, kend = min(K, kbeg + Kc);
  const int nslab = kend > kbeg ? (kend - kbeg + FK - 1) / FK : 0;
  C += (long)blockIdx.z * M * ldc;
  // thread t copies rows t / 8 and t / 8 + 32, K offset (t % 8) * 4, of A and B
  const int lr = threadIdx.x >> 3, lk = (threadIdx.x & 7) * 4;
  const uint32_t as0 = static_cast<uint32_t>(__cvta_generic_to_shared(As));
  const uint32_t bs0 = static_cast<uint32_t>(__cvta_generic_to_shared(Bs));
  auto load = [&](int buf, int slab) {
    const int gk = kbeg + slab * FK + lk;
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const int r = lr + 32 * i, gm = m0 + r, gn = n0 + r;
      const bool ka = gk < kend;
      const uint32_t off = (uint32_t)(((buf * FT + r) * CP_LD + lk) * 4);
      cp_async16(as0 + off, A + (long)(gm < M ? gm : 0) * lda + (ka ? gk : 0), ka && gm < M);
      cp_async16(bs0 + off, Bm + (long)(gn < N ? gn : 0) * ldb + (ka ? gk : 0), ka && gn < N);
    }
  };
#pragma unroll
  for (int st = 0; st < CP_STAGES - 1; ++st) {
    if (st < nslab) load(st, st);
    cp_async_commit();
  }
  float acc[4][4] = {};
  for (int sl = 0; sl < nslab; ++sl) {
    cp_async_wait<CP_STAGES - 2>();
    __syncthreads();  // slab sl landed for all threads; buffer (sl - 1) % S is free
    if (sl + CP_STAGES - 1 < nslab) load((sl + CP_STAGES - 1) % CP_STAGES, sl + CP_STAGES - 1);
    cp_async_commit();
    const float* a_t = As + (sl % CP_STAGES) * FT * CP_LD + (ty * 4) * CP_LD;
    const float* b_t = Bs + (sl % CP_STAGES) * FT * CP_LD + tx * CP_LD;
#pragma unroll
    for (int kk = 0; kk < FK; kk += 4) {
      float4 a4[4], b4[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        a4[i] = *reinterpret_cast<const float4*>(a_t + i * CP_LD + kk);
        b4[i] = *reinterpret_cast<const float4*>(b_t + i * 16 * CP_LD + kk);
      }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          acc[i][j] = fmaf(a4[i].x, b4[j].x, acc[i][j]);
          acc[i][j] = fmaf(a4[i].y, b4[j].y, acc[i][j]);
          acc[i][j] = fmaf(a4[i].z, b4[j].z, acc[i][j]);
          acc[i][j] = fmaf(a4[i].w, b4[j].w, acc[i][j]);
        }
    }
  }
  cp_async_wait<0>();
  if (inj.Xo) {
    // per-column parameters once, then all X loads before any X_out store (X
    // and X_out are distinct tensors, but the compiler cannot know it)
    float pb[4], pwx[4], pwd[4], pbg[4];
    int chs[4], tko[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int gn = min(n0 + tx + 16 * j, N - 1);
      chs[j] = gn % inj.d;
      tko[j] = gn / inj.d;
      pb[j] = bias ? bias[gn] : 0.f;
      pwx[j] = inj.gated ? inj.w_x[chs[j]] : 0.f;
      pwd[j] = inj.gated ? inj.w_dlt[chs[j]] : 0.f;
      pbg[j] = inj.gated ? inj.b_g[chs[j]] : 0.f;
    }
    const float* __restrict__ Xr = inj.X;
    float* __restrict__ Xw = inj.Xo;
#pragma unroll
    for (int i = 0; i < 4; ++i) {  // a row: its four X loads, then its stores
      const int gm = m0 + ty * 4 + i;
      if (gm >= M) continue;
      // row gm = (b * m + iprox) * k2 + a: the target block and first token
      const int a = gm % inj.k2, prox = gm / inj.k2;
      const int b = prox / inj.m, ip = prox % inj.m + inj.shift;
      if (ip >= inj.m) continue;
      const long tok0 = (long)ip * inj.P + (long)a * inj.k1, seq0 = (long)b * inj.L;
      float xv[4];
      bool ok[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const long t = tok0 + tko[j];
        ok[j] = n0 + tx + 16 * j < N && t < inj.L;
        xv[j] = ok[j] ? Xr[(seq0 + t) * inj.d + chs[j]] : 0.f;
      }
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        if (!ok[j]) continue;
        const float v = acc[i][j] + pb[j], x = xv[j];
        Xw[(seq0 + tok0 + tko[j]) * inj.d + chs[j]] =
            inj.gated ? x + v / (1.f + expf(-(pwx[j] * x + pwd[j] * v + pbg[j]))) : x + v;
      }
    }
    return;
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int gm = m0 + ty * 4 + i;
    if (gm >= M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int gn = n0 + tx + 16 * j;
      if (gn >= N) continue;
      float v = acc[i][j];
      if (bias) v += bias[gn];
      if (addend) v += addend[(long)gm * ld_add + gn];
      C[(long)gm * ldc + gn] = v;
    }
  }
}

// Eq. proxy-attn in fp32, head width 64.  CTA = (sequence, head, block of
// ATT_Q queries), 8 warps of ATT_Q / 8 queries each.  Keys and values are
// staged in shared memory 64 at a time (K transposed, so lane j reads key j's
// dimensions without bank conflicts); each warp keeps an online softmax per
// query: lane j scores keys j and j + 32 of the chunk and accumulates output
// dimensions j and j + 32.
constexpr int ATT_Q = 8;  // one query per warp: 4x the CTAs of 32, a quarter of the serial chains
__global__ void __launch_bounds__(256) attn_f32_kernel(const float* __restrict__ qkv,
                                                       float* __restrict__ out, int m, int d,
                                                       int causal, float scale) {
  __shared__ float Kt[64][65];                  // [dim][key]
  __shared__ __align__(16) float Vs[64][64];    // [key][dim]
  __shared__ __align__(16) float Qs[ATT_Q][64];
  __shared__ float Ps[8][64];    // per warp: the chunk's probabilities
  const int b = blockIdx.z, h = blockIdx.y, q0 = blockIdx.x * ATT_Q;
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  const long ld = 3L * d, rb = (long)b * m;
  for (int i = tid; i < ATT_Q * 16; i += 256) {
    const int r = i >> 4, c = (i & 15) * 4;
    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
    if (q0 + r < m) v = *reinterpret_cast<const float4*>(qkv + (rb + q0 + r) * ld + h * 64 + c);
    *reinterpret_cast<float4*>(&Qs[r][c]) = make_float4(v.x * scale, v.y * scale, v.z * scale,
                                                        v.w * scale);
  }
  constexpr int QW = ATT_Q / 8;
  float mx[QW], l[QW], o0[QW], o1[QW];
#pragma unroll
  for (int t = 0; t < QW; ++t) {
    mx[t] = -INFINITY;
    l[t] = 0.f;
    o0[t] = o1[t] = 0.f;
  }
  const int kend = causal ? min(m, q0 + ATT_Q) : m;
  for (int k0 = 0; k0 < kend; k0 += 64) {
    __syncthreads();  // previous chunk fully used (and Qs written)
    for (int i = tid; i < 64 * 16; i += 256) {
      const int r = i >> 4, c = (i & 15) * 4;
      float4 kv = make_float4(0.f, 0.f, 0.f, 0.f), vv = kv;
      if (k0 + r < m) {
        const float* row = qkv + (rb + k0 + r) * ld + h * 64 + c;
        kv = *reinterpret_cast<const float4*>(row + d);
        vv = *reinterpret_cast<const float4*>(row + 2 * d);
      }
      Kt[c][r] = kv.x;
      Kt[c + 1][r] = kv.y;
      Kt[c + 2][r] = kv.z;
      Kt[c + 3][r] = kv.w;
      *reinterpret_cast<float4*>(&Vs[r][c]) = vv;
    }
    __syncthreads();
#pragma unroll
    for (int t = 0; t < QW; ++t) {
      const int ql = w * QW + t, q = q0 + ql;
      float s0 = 0.f, s1 = 0.f;
#pragma unroll 16
      for (int e = 0; e < 64; ++e) {
        const float qe = Qs[ql][e];
        s0 = fmaf(qe, Kt[e][lane], s0);
        s1 = fmaf(qe, Kt[e][lane + 32], s1);
      }
      const int j0 = k0 + lane, j1 = k0 + lane + 32;
      if (j0 >= m || (causal && j0 > q)) s0 = -INFINITY;
      if (j1 >= m || (causal && j1 > q)) s1 = -INFINITY;
      float cm = fmaxf(s0, s1);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) cm = fmaxf(cm, __shfl_xor_sync(0xffffffffu, cm, o));
      const float mn = fmaxf(mx[t], cm);
      const float mref = (mn == -INFINITY) ? 0.f : mn;
      const float corr = expf(mx[t] - mref);
      const float p0 = expf(s0 - mref), p1 = expf(s1 - mref);
      float ps = p0 + p1;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) ps += __shfl_xor_sync(0xffffffffu, ps, o);
      l[t] = l[t] * corr + ps;
      mx[t] = mn;
      Ps[w][lane] = p0;
      Ps[w][lane + 32] = p1;
      __syncwarp();
      float a0 = o0[t] * corr, a1 = o1[t] * corr;
#pragma unroll 16
      for (int j = 0; j < 64; ++j) {
        const float pj = Ps[w][j];
        a0 = fmaf(pj, Vs[j][lane], a0);
        a1 = fmaf(pj, Vs[j][lane + 32], a1);
      }
      o0[t] = a0;
      o1[t] = a1;
      __syncwarp();
    }
  }
#pragma unroll
  for (int t = 0; t < QW; ++t) {
    const int q = q0 + w * QW + t;
    if (q >= m) continue;
    float* op = out + (rb + q) * d + h * 64;
    op[lane] = o0[t] / l[t];
    op[lane + 32] = o1[t] / l[t];
  }
}

// Routing + injection (Eq. inj-gate / inj-add) in fp32, four channels per
// thread.  D is [B*m*k2, k1*d] in proxy order; token t of block i reads the
// row of proxy i - shift.
__global__ void inject_f32_kernel(const float* __restrict__ X, const float* __restrict__ D,
                                  float* __restrict__ Xo, const float* __restrict__ w_x,
                                  const float* __restrict__ w_dlt, const float* __restrict__ b_g,
                                  long L, int d, int P, int k1, int k2, int m, int shift, int gated,
                                  long total4) {
  const long e4 = (long)blockIdx.x * blockDim.x + threadIdx.x;
  if (e4 >= total4) return;
  const int d4 = d >> 2;
  const long tokg = e4 / d4;  // global token (b * L + t)
  const int ch = (int)(e4 - tokg * d4) * 4;
  const long b = tokg / L, t = tokg - b * L;
  const long i = t / P, p = t - i * P;
  const float4 x = *reinterpret_cast<const float4*>(X + e4 * 4);
  if (i < shift) {
    *reinterpret_cast<float4*>(Xo + e4 * 4) = x;
    return;
  }
  const long prox = b * m + (i - shift);
  const long row = prox * k2 + p / k1;
  const float4 dv = *reinterpret_cast<const float4*>(D + row * ((long)k1 * d) + (p % k1) * d + ch);
  float4 o;
  if (gated) {
    const float4 wx = *reinterpret_cast<const float4*>(w_x + ch);
    const float4 wd = *reinterpret_cast<const float4*>(w_dlt + ch);
    const float4 bg = *reinterpret_cast<const float4*>(b_g + ch);
    o.x = x.x + dv.x / (1.f + expf(-(wx.x * x.x + wd.x * dv.x + bg.x)));
    o.y = x.y + dv.y / (1.f + expf(-(wx.y * x.y + wd.y * dv.y + bg.y)));
    o.z = x.z + dv.z / (1.f + expf(-(wx.z * x.z + wd.z * dv.z + bg.z)));
    o.w = x.w + dv.w / (1.f + expf(-(wx.w * x.w + wd.w * dv.w + bg.w)));
  } else {
    o = make_float4(x.x + dv.x, x.y + dv.y, x.z + dv.z, x.w + dv.w);
  }
  *reinterpret_cast<float4*>(Xo + e4 * 4) = o;
}

__global__ void pad_f32_kernel(const float* __restrict__ src, float* __restrict__ dst, long L,
                               long Lp, int d, long total) {
  const long e = (long)blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= total) return;
  const long b = e / (Lp * d), r = e % (Lp * d);
  dst[e] = (r < L * d) ? src[b * L * d + r] : 0.f;
}


// Deterministic split-K reduction: C = sum_s part[s] (+ bias) (+ addend).  A
// CTA takes 32 four-column groups of one row segment and 8 split groups; split
// group g sums splits g, g + 8, ... in that order, and the 8 group sums are
// added in order 0..7, so the result does not depend on scheduling.
constexpr int RED_G = 8;
__global__ void __launch_bounds__(256) splitk_f32_reduce(const float* __restrict__ part, int S, int M,
                                                         int N, float* __restrict__ C, long ldc,
                                                         const float* __restrict__ bias,
                                                         const float* __restrict__ addend,
                                                         long ld_add) {
  __shared__ float4 sums[RED_G][32];
  const int g = threadIdx.x >> 5, l = threadIdx.x & 31;
  const long n4 = (long)(N + 3) / 4;
  const long q = (long)blockIdx.x * 32 + l;  // four-column group over [M, N / 4]
  const bool in = q < (long)M * n4;
  const long r = in ? q / n4 : 0;
  const int c = in ? (int)(q % n4) * 4 : 0;
  const bool vec4 = (N % 4) == 0;
  float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
  if (in) {
    for (int s = g; s < S; s += RED_G) {
      const float* p = part + ((long)s * M + r) * N + c;
      if (vec4) {
        const float4 x = *reinterpret_cast<const float4*>(p);
        v.x += x.x; v.y += x.y; v.z += x.z; v.w += x.w;
      } else {
        v.x += p[0];
        if (c + 1 < N) v.y += p[1];
        if (c + 2 < N) v.z += p[2];
        if (c + 3 < N) v.w += p[3];
      }
    }
  }
  sums[g][l] = v;
  __syncthreads();
  if (g != 0 || !in) return;
  float4 t = sums[0][l];
#pragma unroll
  for (int k = 1; k < RED_G; ++k) {
    const float4 u = sums[k][l];
    t.x += u.x; t.y += u.y; t.z += u.z; t.w += u.w;
  }
  const float tv[4] = {t.x, t.y, t.z, t.w};
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    if (c + j >= N) break;
    float o = tv[j];
    if (bias) o += bias[c + j];
    if (addend) o += addend[r * ld_add + c + j];
    C[r * ldc + c + j] = o;
  }
}

}  // namespace

int splitk_f32_factor(int M, int N, int K) {
  // about one wave of a 152-SM part; slices of at least two 32-wide K slabs
  const long tiles = (long)((M + FT - 1) / FT) * ((N + FT - 1) / FT);
  if (tiles >= 152) return 1;
  int S = (int)((152 + tiles - 1) / tiles);
  S = std::min(S, std::max(1, K / 64));
  return std::min(S, 64);
}

namespace {
int vec_ok(const float* A, long lda, const float* B, long ldb, int K) {
  return ((reinterpret_cast<uintptr_t>(A) | reinterpret_cast<uintptr_t>(B)) & 15) == 0 &&
         lda % 4 == 0 && ldb % 4 == 0 && K % 4 == 0;
}
}  // namespace

namespace {
// launch the product (cp.async ring when the operands allow it)
cudaError_t launch_f32(dim3 grid, int vec, const float* A, long lda, const float* B, long ldb,
                       float* C, long ldc, int M, int N, int K, int Kc, const float* bias,
                       const float* addend, long ld_add, const InjF32& inj, cudaStream_t st) {
  if (vec) {
    static const cudaError_t attr = cudaFuncSetAttribute(
        gemm_f32_cp_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, CP_SMEM);
    if (attr != cudaSuccess) return attr;
    gemm_f32_cp_kernel<<<grid, FTHREADS, CP_SMEM, st>>>(A, lda, B, ldb, C, ldc, M, N, K, Kc, bias,
                                                        addend, ld_add, inj);
  } else {
    gemm_f32_kernel<<<grid, FTHREADS, 0, st>>>(A, lda, B, ldb, C, ldc, M, N, K, Kc, bias, addend,
                                               ld_add, 0, inj);
  }
  return cudaGetLastError();
}
}  // namespace

cudaError_t gemm_f32(int M, int N, int K, const float* A, long lda, const float* B, long ldb,
                     float* C, long ldc, const float* bias, const float* addend, long ld_add,
                     const char* label, cudaStream_t st, float* scratch, size_t scratch_bytes) {
  const int S = splitk_f32_factor(M, N, K);
  const int vec = vec_ok(A, lda, B, ldb, K);
  LaunchTimer lt(label, st, 2.0 * M * N * (double)K, 4.0 * ((double)M * K + (double)N * K + (double)M * N));
  if (S > 1 && scratch && (size_t)S * M * N * sizeof(float) <= scratch_bytes) {
    const int Kc = ((K + S - 1) / S + FK - 1) / FK * FK;
    dim3 grid((N + FT - 1) / FT, (M + FT - 1) / FT, S);
    cudaError_t e = launch_f32(grid, vec, A, lda, B, ldb, scratch, N, M, N, K, Kc, nullptr, nullptr,
                               0, InjF32{}, st);
    if (e != cudaSuccess) return e;
    const long groups = (long)M * ((N + 3) / 4);
    splitk_f32_reduce<<<(unsigned)((groups + 31) / 32), 256, 0, st>>>(scratch, S, M, N, C, ldc, bias,
                                                                     addend, ld_add);
    return cudaGetLastError();
  }
  dim3 grid((N + FT - 1) / FT, (M + FT - 1) / FT, 1);
  return launch_f32(grid, vec, A, lda, B, ldb, C, ldc, M, N, K, K, bias, addend, ld_add, InjF32{},
                    st);
}

cudaError_t gemm_f32_inject(int M, int N, int K, const float* A, long lda, const float* B, long ldb,
                            const float* bias, const float* X, float* Xo, const float* w_x,
                            const float* w_dlt, const float* b_g, int Bsz, long L, int d, int P,
                            int k1, int k2, int m, int shift, int gated, cudaStream_t st) {
  const int vec = vec_ok(A, lda, B, ldb, K);
  {
    LaunchTimer lt("decompress_d1_inject", st, 2.0 * M * N * (double)K,
                   4.0 * ((double)M * K + (double)N * K) + 12.0 * Bsz * L * (double)d);
    dim3 grid((N + FT - 1) / FT, (M + FT - 1) / FT, 1);
    const cudaError_t e = launch_f32(grid, vec, A, lda, B, ldb, nullptr, 0, M, N, K, K, bias,
                                     nullptr, 0, InjF32{X, Xo, w_x, w_dlt, b_g, L, d, P, k1, k2, m,
                                                        shift, gated},
                                     st);
    if (e != cudaSuccess) return e;
  }
  if (shift > 0) {  // the first block of every sequence receives nothing: X_out = X
    const long rows = std::min<long>((long)shift * P, L);
    cudaError_t e = cudaMemcpy2DAsync(Xo, (size_t)L * d * sizeof(float), X,
                                      (size_t)L * d * sizeof(float),
                                      (size_t)rows * d * sizeof(float), (size_t)Bsz,
                                      cudaMemcpyDeviceToDevice, st);
    if (e != cudaSuccess) return e;
  }
  return cudaGetLastError();
}

cudaError_t attn_f32(const float* qkv, float* out, int B, int m, int d, int nh, bool causal,
                     cudaStream_t st) {
  const double pairs = (double)B * nh * (causal ? 0.5 * m * (m + 1.0) : (double)m * m);
  LaunchTimer lt("attn_f32", st, 4.0 * 64 * pairs, 4.0 * B * m * 4.0 * d);
  dim3 grid((m + ATT_Q - 1) / ATT_Q, nh, B);
  attn_f32_kernel<<<grid, 256, 0, st>>>(qkv, out, m, d, causal ? 1 : 0, 1.0f / sqrtf(64.0f));
  return cudaGetLastError();
}

cudaError_t inject_f32(const float* X, const float* D, float* Xo, const float* w_x,
                       const float* w_dlt, const float* b_g, int B, long L, int d, int P, int k1,
                       int k2, int m, int shift, int gated, cudaStream_t st) {
  const long total4 = (long)B * L * d / 4;
  LaunchTimer lt("inject_f32", st, 0.0, 48.0 * total4);
  inject_f32_kernel<<<(unsigned)((total4 + 255) / 256), 256, 0, st>>>(
      X, D, Xo, w_x, w_dlt, b_g, L, d, P, k1, k2, m, shift, gated, total4);
  return cudaGetLastError();
}

cudaError_t pad_f32(const float* src, float* dst, int B, long L, long Lp, int d, cudaStream_t st) {
  const long total = (long)B * Lp * d;
  LaunchTimer lt("pad_rows", st, 0.0, 4.0 * B * (L + Lp) * d);
  pad_f32_kernel<<<(unsigned)((total + 255) / 256), 256, 0, st>>>(src, dst, L, Lp, d, total);
  return cudaGetLastError();
}

}  // namespace pf
