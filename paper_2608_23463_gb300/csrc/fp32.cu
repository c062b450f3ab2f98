// fp32 forward of the 1D layer (Alg. 1) on CUDA cores: a tiled SIMT GEMM for
// the compression / Q,K,V / output / decompression projections, an
// online-softmax proxy attention with one warp per query, and the routing +
// injection pass.  Used when the descriptor's dtype is PF_F32 (the tensor
// cores have no fp32 path that meets fp32 accuracy).
#include <algorithm>

#include "kernels.h"

namespace pf {

int take_dev_error_fp32() { return take_dev_error_tu(); }

namespace {

constexpr int FT = 64;   // output tile (FT x FT)
constexpr int FK = 16;   // K slab
constexpr int FTHREADS = 256;

// C[M, N] = A[M, K] B[N, K]^T (+ bias[n]) (+ addend[m, n]), all row-major fp32
// with leading dimensions lda, ldb, ldc.  Each thread computes 4 x 4 outputs.
// With gridDim.z = S > 1 each z-slice reduces K range [z*Kc, (z+1)*Kc) and
// writes raw partials to C + z*M*ldc (bias / addend are then applied by
// splitk_f32_reduce).
__global__ void __launch_bounds__(FTHREADS) gemm_f32_kernel(const float* __restrict__ A, long lda,
                                                           const float* __restrict__ Bm, long ldb,
                                                           float* __restrict__ C, long ldc, int M,
                                                           int N, int K, int Kc,
                                                           const float* __restrict__ bias,
                                                           const float* __restrict__ addend,
                                                           long ld_add) {
  __shared__ float As[FK][FT + 4], Bs[FK][FT + 4];
  const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
  const int m0 = blockIdx.y * FT, n0 = blockIdx.x * FT;
  const int kbeg = blockIdx.z * Kc, kend = min(K, kbeg + Kc);
  C += (long)blockIdx.z * M * ldc;
  float acc[4][4] = {};
  for (int k0 = kbeg; k0 < kend; k0 += FK) {
    for (int i = threadIdx.x; i < FT * FK; i += FTHREADS) {
      const int r = i / FK, kk = i % FK;
      const int gm = m0 + r, gn = n0 + r, gk = k0 + kk;
      As[kk][r] = (gm < M && gk < kend) ? A[(long)gm * lda + gk] : 0.f;
      Bs[kk][r] = (gn < N && gk < kend) ? Bm[(long)gn * ldb + gk] : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < FK; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        a[i] = As[kk][ty * 4 + i];
        b[i] = Bs[kk][tx * 4 + i];
      }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int gm = m0 + ty * 4 + i;
    if (gm >= M) continue;
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

// Eq. proxy-attn in fp32: one warp per (query, head, sequence), online
// softmax over the visible keys (j <= i when causal).  Head width 64: two
// dimensions per lane.
__global__ void attn_f32_kernel(const float* __restrict__ qkv, float* __restrict__ out, int B,
                                int m, int d, int nh, int causal, float scale) {
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (warp >= B * nh * m) return;  // whole warps only
  const int i = warp % m, h = (warp / m) % nh, b = warp / (m * nh);
  const long ld = 3L * d, rb = (long)b * m;
  const float* qrow = qkv + (rb + i) * ld + h * 64;
  const float q0 = qrow[lane] * scale, q1 = qrow[lane + 32] * scale;
  float mx = -INFINITY, l = 0.f, a0 = 0.f, a1 = 0.f;
  const int nk = causal ? i + 1 : m;
  for (int j = 0; j < nk; ++j) {
    const float* krow = qkv + (rb + j) * ld + d + h * 64;
    float s = q0 * krow[lane] + q1 * krow[lane + 32];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    const float mn = fmaxf(mx, s);
    const float c = expf(mx - mn), p = expf(s - mn);
    const float* vrow = qkv + (rb + j) * ld + 2 * d + h * 64;
    l = l * c + p;
    a0 = a0 * c + p * vrow[lane];
    a1 = a1 * c + p * vrow[lane + 32];
    mx = mn;
  }
  float* o = out + (rb + i) * d + h * 64;
  o[lane] = a0 / l;
  o[lane + 32] = a1 / l;
}

// Routing + injection (Eq. inj-gate / inj-add) in fp32, one thread per output
// element of X_out.  D is [B*m*k2, k1*d] in proxy order; token t of block i
// reads the row of proxy i - shift.
__global__ void inject_f32_kernel(const float* __restrict__ X, const float* __restrict__ D,
                                  float* __restrict__ Xo, const float* __restrict__ w_x,
                                  const float* __restrict__ w_dlt, const float* __restrict__ b_g,
                                  long L, int d, int P, int k1, int k2, int m, int shift, int gated,
                                  long total) {
  const long e = (long)blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= total) return;
  const long t = (e / d) % L, b = e / ((long)L * d);
  const int ch = (int)(e % d);
  const long i = t / P, p = t % P;
  const float x = X[e];
  if (i < shift) {
    Xo[e] = x;
    return;
  }
  const long prox = b * m + (i - shift);
  const long row = prox * k2 + p / k1;
  const float dv = D[row * ((long)k1 * d) + (p % k1) * d + ch];
  if (gated) {
    const float g = w_x[ch] * x + w_dlt[ch] * dv + b_g[ch];
    Xo[e] = x + dv / (1.f + expf(-g));
  } else {
    Xo[e] = x + dv;
  }
}

__global__ void pad_f32_kernel(const float* __restrict__ src, float* __restrict__ dst, long L,
                               long Lp, int d, long total) {
  const long e = (long)blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= total) return;
  const long b = e / (Lp * d), r = e % (Lp * d);
  dst[e] = (r < L * d) ? src[b * L * d + r] : 0.f;
}


__global__ void splitk_f32_reduce(const float* __restrict__ part, int S, int M, int N,
                                  float* __restrict__ C, long ldc, const float* __restrict__ bias,
                                  const float* __restrict__ addend, long ld_add) {
  const long i = (long)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (long)M * N) return;
  const long r = i / N;
  const int c = (int)(i % N);
  float v = 0.f;
  for (int s = 0; s < S; ++s) v += part[((long)s * M + r) * N + c];
  if (bias) v += bias[c];
  if (addend) v += addend[r * ld_add + c];
  C[r * ldc + c] = v;
}

}  // namespace

int splitk_f32_factor(int M, int N, int K) {
  const long tiles = (long)((M + FT - 1) / FT) * ((N + FT - 1) / FT);
  if (tiles >= 304) return 1;
  int S = (int)((304 + tiles - 1) / tiles);
  S = std::min(S, std::max(1, K / 512));
  return std::min(S, 64);
}

cudaError_t gemm_f32(int M, int N, int K, const float* A, long lda, const float* B, long ldb,
                     float* C, long ldc, const float* bias, const float* addend, long ld_add,
                     const char* label, cudaStream_t st, float* scratch, size_t scratch_bytes) {
  const int S = splitk_f32_factor(M, N, K);
  LaunchTimer lt(label, st, 2.0 * M * N * (double)K, 4.0 * ((double)M * K + (double)N * K + (double)M * N));
  if (S > 1 && scratch && (size_t)S * M * N * sizeof(float) <= scratch_bytes) {
    const int Kc = ((K + S - 1) / S + FK - 1) / FK * FK;
    dim3 grid((N + FT - 1) / FT, (M + FT - 1) / FT, S);
    gemm_f32_kernel<<<grid, FTHREADS, 0, st>>>(A, lda, B, ldb, scratch, N, M, N, K, Kc, nullptr,
                                               nullptr, 0);
    const long total = (long)M * N;
    splitk_f32_reduce<<<(unsigned)((total + 255) / 256), 256, 0, st>>>(scratch, S, M, N, C, ldc, bias,
                                                                      addend, ld_add);
    return cudaGetLastError();
  }
  dim3 grid((N + FT - 1) / FT, (M + FT - 1) / FT, 1);
  gemm_f32_kernel<<<grid, FTHREADS, 0, st>>>(A, lda, B, ldb, C, ldc, M, N, K, K, bias, addend,
                                             ld_add);
  return cudaGetLastError();
}


cudaError_t attn_f32(const float* qkv, float* out, int B, int m, int d, int nh, bool causal,
                     cudaStream_t st) {
  const long warps = (long)B * nh * m;
  const double pairs = (double)B * nh * (causal ? 0.5 * m * (m + 1.0) : (double)m * m);
  LaunchTimer lt("attn_f32", st, 4.0 * 64 * pairs, 4.0 * B * m * 4.0 * d);
  attn_f32_kernel<<<(unsigned)((warps * 32 + 255) / 256), 256, 0, st>>>(
      qkv, out, B, m, d, nh, causal ? 1 : 0, 1.0f / sqrtf(64.0f));
  return cudaGetLastError();
}

cudaError_t inject_f32(const float* X, const float* D, float* Xo, const float* w_x,
                       const float* w_dlt, const float* b_g, int B, long L, int d, int P, int k1,
                       int k2, int m, int shift, int gated, cudaStream_t st) {
  const long total = (long)B * L * d;
  LaunchTimer lt("inject_f32", st, 0.0, 12.0 * total);
  inject_f32_kernel<<<(unsigned)((total + 255) / 256), 256, 0, st>>>(
      X, D, Xo, w_x, w_dlt, b_g, L, d, P, k1, k2, m, shift, gated, total);
  return cudaGetLastError();
}

cudaError_t pad_f32(const float* src, float* dst, int B, long L, long Lp, int d, cudaStream_t st) {
  const long total = (long)B * Lp * d;
  LaunchTimer lt("pad_rows", st, 0.0, 4.0 * B * (L + Lp) * d);
  pad_f32_kernel<<<(unsigned)((total + 255) / 256), 256, 0, st>>>(src, dst, L, Lp, d, total);
  return cudaGetLastError();
}

}  // namespace pf
