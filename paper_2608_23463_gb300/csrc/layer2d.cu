// Kernels specific to the 2D bidirectional layer (Sec. 3.9): patch gather,
// per-token LayerNorm statistics, timestep conditioning of the proxies
// (sinusoidal embedding -> SiLU MLP -> adaLN scale/shift) and the backward of
// the affine injection, adaLN and the timestep MLP.  The contractions use the
// tcgen05 GEMM (gemm_tc.cuh).
#include "kernels.h"

namespace pf {

int take_dev_error_layer2d() { return take_dev_error_tu(); }
int set_wait_limit_layer2d(unsigned long long ns) { return set_wait_limit_tu(ns); }

namespace {

__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
  for (int s = 16; s > 0; s >>= 1) v += __shfl_xor_sync(0xffffffffu, v, s);
  return v;
}

// One pass over the tokens of the 2D layer, one warp per token t = (b, y, x):
// the patch copy Xp[r, (py*p + px)*d + ch] = X[t, ch] for patch r = (b, by, bx)
// (Eq. partition, the compression GEMM's operand) and the token's LayerNorm
// statistics stats[t] = (mean, 1/sqrt(var + 1e-6)) (Eq. inj-affine), from
// registers (two passes over the row held by the warp).  d <= 512.
__global__ void __launch_bounds__(256) patch_gather_stats_kernel(
    const bf16* __restrict__ X, bf16* __restrict__ Xp, float* __restrict__ stats, long T, int d,
    int patch, int gh, int gw) {
  const long t = ((long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (t >= T) return;
  const long HW = (long)gh * gw;
  const int b = (int)(t / HW), yx = (int)(t % HW), y = yx / gw, x = yx % gw;
  const int npw = gw / patch, m = (gh / patch) * npw;
  const long row = (long)b * m + (y / patch) * npw + x / patch;
  const int p = (y % patch) * patch + (x % patch);
  const bf16* src = X + t * d;
  bf16* dst = Xp + row * ((long)patch * patch * d) + (long)p * d;
  uint4 u[2];
  float s = 0.f;
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int c = lane * 8 + 256 * i;
    if (c >= d) break;
    u[i] = __ldcs(reinterpret_cast<const uint4*>(src + c));
    *reinterpret_cast<uint4*>(dst + c) = u[i];
    const uint32_t w[4] = {u[i].x, u[i].y, u[i].z, u[i].w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float2 f = unpack_bf16(w[j]);
      s += f.x + f.y;
    }
  }
  const float mu = warp_sum_f(s) / d;
  float q = 0.f;
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int c = lane * 8 + 256 * i;
    if (c >= d) break;
    const uint32_t w[4] = {u[i].x, u[i].y, u[i].z, u[i].w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float2 f = unpack_bf16(w[j]);
      q += (f.x - mu) * (f.x - mu) + (f.y - mu) * (f.y - mu);
    }
  }
  const float var = warp_sum_f(q) / d;
  if (lane == 0) {
    stats[2 * t] = mu;
    stats[2 * t + 1] = rsqrtf(var + 1e-6f);
  }
}

// Timestep conditioning of one image: e = [cos(1000 t w_k), sin(1000 t w_k)],
// w_k = 10000^(-k/128); a1 = W_t1 e + b_t1; u = SiLU(a1); gb = W_t2 u + b_t2
// = [gamma | beta].  One CTA per image, one warp per output.
__global__ void __launch_bounds__(256) temb_fwd_kernel(const float* __restrict__ t, int d,
                                                       const bf16* __restrict__ W_t1,
                                                       const float* __restrict__ b_t1,
                                                       const bf16* __restrict__ W_t2,
                                                       const float* __restrict__ b_t2,
                                                       float* __restrict__ e_out,
                                                       float* __restrict__ a1_out,
                                                       float* __restrict__ u_out,
                                                       float* __restrict__ gb_out) {
  extern __shared__ float sm[];  // e [256], u [d]
  float* e = sm;
  float* u = sm + 256;
  const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const float tb = 1000.f * t[b];
  if (tid < 128) {
    const float w = expf(-(float)tid * (9.210340371976184f / 128.f));  // ln(10000)/128
    const float a = tb * w;
    e[tid] = cosf(a);
    e[tid + 128] = sinf(a);
  }
  __syncthreads();
  if (tid < 256) e_out[b * 256 + tid] = e[tid];
  for (int o = warp; o < d; o += 8) {
    float acc = 0.f;
    for (int k = lane; k < 256; k += 32) acc = fmaf(__bfloat162float(W_t1[(long)o * 256 + k]), e[k], acc);
    acc = warp_sum_f(acc);
    if (lane == 0) {
      const float a = acc + b_t1[o];
      a1_out[(long)b * d + o] = a;
      const float uu = a * sigmoidf_(a);
      u[o] = uu;
      u_out[(long)b * d + o] = uu;
    }
  }
  __syncthreads();
  for (int o = warp; o < 2 * d; o += 8) {
    float acc = 0.f;
    for (int k = lane; k < d; k += 32) acc = fmaf(__bfloat162float(W_t2[(long)o * d + k]), u[k], acc);
    acc = warp_sum_f(acc);
    if (lane == 0) gb_out[(long)b * 2 * d + o] = acc + b_t2[o];
  }
}

// adaLN of the proxies (one warp per proxy row r of image b = r / m):
// n = LayerNorm(H_r); Hq = (1 + gamma_b) n + beta_b -> bf16.  Saves n and 1/std.
__global__ void adaln_fwd_kernel(const float* __restrict__ H, const float* __restrict__ gb,
                                 float* __restrict__ n_out, float* __restrict__ rstd_out,
                                 bf16* __restrict__ Hq, long R, int d, int m) {
  const long r = ((long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (r >= R) return;
  const float* h = H + r * d;
  const float* gam = gb + (r / m) * 2 * d;
  const float* bet = gam + d;
  float s = 0.f;
  for (int c = lane; c < d; c += 32) s += h[c];
  const float mu = warp_sum_f(s) / d;
  float q = 0.f;
  for (int c = lane; c < d; c += 32) q += (h[c] - mu) * (h[c] - mu);
  const float rs = rsqrtf(warp_sum_f(q) / d + 1e-6f);
  for (int c = lane; c < d; c += 32) {
    const float n = (h[c] - mu) * rs;
    n_out[r * d + c] = n;
    Hq[r * d + c] = __float2bfloat16(fmaf(1.f + gam[c], n, bet[c]));
  }
  if (lane == 0) rstd_out[r] = rs;
}

// Backward of X_out = (1 + s) n + t, n = LayerNorm(X), one warp per token:
// ds = G n, dt = G, dn = G (1 + s), dX = rstd (dn - mean(dn) - n mean(dn n)).
// dD [B*m, 2*P*d] (patch order: token p of a patch at columns [2pd, 2pd+d) for
// ds and [2pd+d, 2(p+1)d) for dt) and dXd [B*m, P*d] (patch order).  A block
// takes the tokens at one position p of their patch for IB2_CP consecutive
// patches and also sums its ds and dt over them: part[chunk][2pd + c], the
// first pass of the deterministic bias gradient (no second read of dD).
// d <= 512.
constexpr int IB2_CP = 256;   // patches per block
constexpr int IB2_MAXI = 2;   // channel groups of 256 per lane: d <= 512
__global__ void __launch_bounds__(256) inj_bwd_2d_kernel(
    const bf16* __restrict__ G, const bf16* __restrict__ X, const float* __restrict__ stats,
    const bf16* __restrict__ S, bf16* __restrict__ dD, bf16* __restrict__ dXd,
    float* __restrict__ part, long R, int d, int patch, int gh, int gw) {
  __shared__ float red[8][2 * 256 * IB2_MAXI];
  const int p = blockIdx.y, chunk = blockIdx.x;
  const int py = p / patch, px = p % patch;
  const int npw = gw / patch, m = (gh / patch) * npw, P = patch * patch;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float cs[IB2_MAXI][8], ct[IB2_MAXI][8];
#pragma unroll
  for (int i = 0; i < IB2_MAXI; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) cs[i][j] = ct[i][j] = 0.f;
  const long r1 = min(R, (long)(chunk + 1) * IB2_CP);
  for (long row = (long)chunk * IB2_CP + warp; row < r1; row += 8) {
    const int b = (int)(row / m), pr = (int)(row % m), by = pr / npw, bx = pr % npw;
    const long t = ((long)b * gh + by * patch + py) * gw + bx * patch + px;
    const float mu = stats[2 * t], rs = stats[2 * t + 1];
    const bf16* g = G + t * d;
    const bf16* xr = X + t * d;
    const bf16* sr = S + row * ((long)P * d) + (long)p * d;
    bf16* dds = dD + row * (2L * P * d) + (long)p * 2 * d;
    bf16* ddt = dds + d;
    bf16* dxo = dXd + row * ((long)P * d) + (long)p * d;
    float s1 = 0.f, s2 = 0.f;
#pragma unroll
    for (int i = 0; i < IB2_MAXI; ++i) {
      const int c = lane * 8 + 256 * i;
      if (c >= d) break;
      float gv[8], xv[8], sv[8], o[8];
      load8_bf16(g + c, gv);
      load8_bf16(xr + c, xv);
      load8_bf16(sr + c, sv);
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const float n = (xv[j] - mu) * rs, dn = gv[j] * (1.f + sv[j]);
        o[j] = gv[j] * n;
        s1 += dn;
        s2 += dn * n;
        cs[i][j] += o[j];
        ct[i][j] += gv[j];
      }
      store8_bf16(dds + c, o);
      *reinterpret_cast<uint4*>(ddt + c) = *reinterpret_cast<const uint4*>(g + c);
    }
    const float m1 = warp_sum_f(s1) / d, m2 = warp_sum_f(s2) / d;
#pragma unroll
    for (int i = 0; i < IB2_MAXI; ++i) {
      const int c = lane * 8 + 256 * i;
      if (c >= d) break;
      float gv[8], xv[8], sv[8], o[8];
      load8_bf16(g + c, gv);
      load8_bf16(xr + c, xv);
      load8_bf16(sr + c, sv);
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const float n = (xv[j] - mu) * rs, dn = gv[j] * (1.f + sv[j]);
        o[j] = rs * (dn - m1 - n * m2);
      }
      store8_bf16(dxo + c, o);
    }
  }
  // the block's sums over its patches, in a fixed order (deterministic)
#pragma unroll
  for (int i = 0; i < IB2_MAXI; ++i) {
    const int c = lane * 8 + 256 * i;
    if (c >= d) break;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      red[warp][c + j] = cs[i][j];
      red[warp][d + c + j] = ct[i][j];
    }
  }
  __syncthreads();
  float* dst = part + (long)chunk * (2L * P * d) + (long)p * 2 * d;
  for (int c = threadIdx.x; c < 2 * d; c += 256) {
    float v = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) v += red[w][c];
    dst[c] = v;
  }
}

// out[c] = sum over chunks of part[chunk][c] (the bias gradient), one thread
// per column, chunks in order.
__global__ void colsum_chunks_kernel(const float* __restrict__ part, int n_chunks, long C,
                                     float* __restrict__ out) {
  const long c = (long)blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= C) return;
  float v = 0.f;
  for (int k = 0; k < n_chunks; ++k) v += part[(long)k * C + c];
  out[c] = v;
}

// Backward of Hq = (1 + gamma) n + beta, n = LayerNorm(H), one warp per row:
// dn = dHq (1 + gamma); dH = rstd (dn - mean(dn) - n mean(dn n)) + dH_out.
__global__ void adaln_bwd_kernel(const float* __restrict__ dHq, const float* __restrict__ nH,
                                 const float* __restrict__ rstd, const float* __restrict__ gb,
                                 const float* __restrict__ dH_out, float* __restrict__ dHf,
                                 bf16* __restrict__ dHb, long R, int d, int m) {
  const long r = ((long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (r >= R) return;
  const float* gam = gb + (r / m) * 2 * d;
  const float rs = rstd[r];
  float s1 = 0.f, s2 = 0.f;
  for (int c = lane; c < d; c += 32) {
    const float dn = dHq[r * d + c] * (1.f + gam[c]);
    s1 += dn;
    s2 += dn * nH[r * d + c];
  }
  const float m1 = warp_sum_f(s1) / d, m2 = warp_sum_f(s2) / d;
  for (int c = lane; c < d; c += 32) {
    const float dn = dHq[r * d + c] * (1.f + gam[c]);
    float v = rs * (dn - m1 - nH[r * d + c] * m2);
    if (dH_out) v += dH_out[r * d + c];
    dHf[r * d + c] = v;
    dHb[r * d + c] = __float2bfloat16(v);
  }
}

// Per-image partial sums of dgamma = sum_r dHq_r n_r and dbeta = sum_r dHq_r
// over a chunk of rows: part[b][chunk][0..d) and [d..2d).
__global__ void adaln_param_part_kernel(const float* __restrict__ dHq, const float* __restrict__ nH,
                                        float* __restrict__ part, int d, int m, int chunks) {
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  const int ck = blockIdx.y, b = blockIdx.z;
  if (c >= d) return;
  const int rows = (m + chunks - 1) / chunks;
  const long r0 = (long)b * m + (long)ck * rows, r1 = (long)b * m + min(m, (ck + 1) * rows);
  float g = 0.f, be = 0.f;
  for (long r = r0; r < r1; ++r) {
    const float v = dHq[r * d + c];
    g = fmaf(v, nH[r * d + c], g);
    be += v;
  }
  float* o = part + ((long)b * chunks + ck) * 2 * d;
  o[c] = g;
  o[d + c] = be;
}

__global__ void adaln_param_final_kernel(const float* __restrict__ part, float* __restrict__ dgb,
                                         int d, int chunks, int B) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= B * 2 * d) return;
  const int b = i / (2 * d), j = i % (2 * d);
  float s = 0.f;
  for (int ck = 0; ck < chunks; ++ck) s += part[((long)b * chunks + ck) * 2 * d + j];
  dgb[i] = s;
}

// du = W_t2^T dgb, da1 = du * SiLU'(a1), per image (thread per column i).
__global__ void temb_bwd_du_kernel(const float* __restrict__ dgb, const bf16* __restrict__ W_t2,
                                   const float* __restrict__ a1, float* __restrict__ da1, int d) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x, b = blockIdx.y;
  if (i >= d) return;
  float du = 0.f;
  for (int o = 0; o < 2 * d; ++o) du = fmaf(__bfloat162float(W_t2[(long)o * d + i]), dgb[(long)b * 2 * d + o], du);
  const float z = a1[(long)b * d + i], sg = sigmoidf_(z);
  da1[(long)b * d + i] = du * sg * (1.f + z * (1.f - sg));
}

// Weight gradients of the timestep MLP (sums over the B images):
// dW_t2[o, i] = sum_b dgb[b, o] u[b, i], db_t2 = sum_b dgb,
// dW_t1[o, k] = sum_b da1[b, o] e[b, k], db_t1 = sum_b da1.
__global__ void temb_wgrad_kernel(const float* __restrict__ dgb, const float* __restrict__ u,
                                  const float* __restrict__ da1, const float* __restrict__ e,
                                  float* gW_t2, float* gb_t2, float* gW_t1, float* gb_t1, int d,
                                  int B) {
  const long i = (long)blockIdx.x * blockDim.x + threadIdx.x;
  const long n_w2 = 2L * d * d, n_b2 = 2L * d, n_w1 = (long)d * 256, n_b1 = d;
  float s = 0.f;
  if (i < n_w2) {
    const long o = i / d, k = i % d;
    for (int b = 0; b < B; ++b) s = fmaf(dgb[(long)b * 2 * d + o], u[(long)b * d + k], s);
    if (gW_t2) gW_t2[i] = s;
  } else if (i < n_w2 + n_b2) {
    const long o = i - n_w2;
    for (int b = 0; b < B; ++b) s += dgb[(long)b * 2 * d + o];
    if (gb_t2) gb_t2[o] = s;
  } else if (i < n_w2 + n_b2 + n_w1) {
    const long j = i - n_w2 - n_b2, o = j / 256, k = j % 256;
    for (int b = 0; b < B; ++b) s = fmaf(da1[(long)b * d + o], e[(long)b * 256 + k], s);
    if (gW_t1) gW_t1[j] = s;
  } else if (i < n_w2 + n_b2 + n_w1 + n_b1) {
    const long o = i - n_w2 - n_b2 - n_w1;
    for (int b = 0; b < B; ++b) s += da1[(long)b * d + o];
    if (gb_t1) gb_t1[o] = s;
  }
}

}  // namespace

cudaError_t patch_gather_stats(const bf16* X, bf16* Xp, float* stats, int B, int d, int patch,
                               int gh, int gw, cudaStream_t st) {
  if (d > 512 || d % 8 != 0) return cudaErrorInvalidValue;
  const long T = (long)B * gh * gw;
  LaunchTimer lt("patch_gather_stats", st, 0.0, 4.0 * T * d + 8.0 * T);
  patch_gather_stats_kernel<<<(unsigned)((T * 32 + 255) / 256), 256, 0, st>>>(X, Xp, stats, T, d,
                                                                             patch, gh, gw);
  return cudaGetLastError();
}

cudaError_t temb_fwd(const float* t, int B, int d, const bf16* W_t1, const float* b_t1,
                     const bf16* W_t2, const float* b_t2, float* e, float* a1, float* u, float* gb,
                     cudaStream_t st) {
  LaunchTimer lt("temb_fwd", st, 2.0 * B * (256.0 * d + 2.0 * d * d), 2.0 * (256.0 * d + 2.0 * d * d));
  temb_fwd_kernel<<<B, 256, (256 + d) * sizeof(float), st>>>(t, d, W_t1, b_t1, W_t2, b_t2, e, a1,
                                                             u, gb);
  return cudaGetLastError();
}

cudaError_t adaln_fwd(const float* H, const float* gb, float* nH, float* rstd, bf16* Hq, long R,
                      int d, int m, cudaStream_t st) {
  LaunchTimer lt("adaln_fwd", st, 0.0, 10.0 * R * d);
  adaln_fwd_kernel<<<(unsigned)((R * 32 + 255) / 256), 256, 0, st>>>(H, gb, nH, rstd, Hq, R, d, m);
  return cudaGetLastError();
}

long inj_bwd_2d_part_elems(long R, int d, int patch) {
  return (R + IB2_CP - 1) / IB2_CP * 2L * patch * patch * d;
}

cudaError_t inj_bwd_2d(const bf16* G, const bf16* X, const float* stats, const bf16* S, bf16* dD,
                       bf16* dXd, float* db_d1, float* part, long R, int d, int patch, int gh,
                       int gw, cudaStream_t st) {
  if (d > 256 * IB2_MAXI || d % 8 != 0) return cudaErrorInvalidValue;
  const int P = patch * patch;
  const int n_chunks = (int)((R + IB2_CP - 1) / IB2_CP);
  {
    LaunchTimer lt("inj_bwd_2d", st, 0.0, 12.0 * R * P * (double)d);
    dim3 grid(n_chunks, P);
    inj_bwd_2d_kernel<<<grid, 256, 0, st>>>(G, X, stats, S, dD, dXd, part, R, d, patch, gh, gw);
  }
  if (db_d1) {
    const long C = 2L * P * d;
    LaunchTimer lt("colsum_final", st, (double)n_chunks * C, 4.0 * n_chunks * C);
    colsum_chunks_kernel<<<(unsigned)((C + 255) / 256), 256, 0, st>>>(part, n_chunks, C, db_d1);
  }
  return cudaGetLastError();
}

cudaError_t adaln_bwd(const float* dHq, const float* nH, const float* rstd, const float* gb,
                      const float* dH_out, float* dHf, bf16* dHb, long R, int d, int m,
                      cudaStream_t st) {
  LaunchTimer lt("adaln_bwd", st, 0.0, 18.0 * R * d);
  adaln_bwd_kernel<<<(unsigned)((R * 32 + 255) / 256), 256, 0, st>>>(dHq, nH, rstd, gb, dH_out, dHf,
                                                                    dHb, R, d, m);
  return cudaGetLastError();
}

int adaln_param_chunks(int m) { return m < 64 ? 1 : (m < 4096 ? m / 64 : 64); }

cudaError_t adaln_param_grads(const float* dHq, const float* nH, float* part, float* dgb, int B,
                              int d, int m, cudaStream_t st) {
  const int chunks = adaln_param_chunks(m);
  {
    LaunchTimer lt("adaln_param", st, 0.0, 8.0 * B * m * (double)d);
    dim3 grid((d + 255) / 256, chunks, B);
    adaln_param_part_kernel<<<grid, 256, 0, st>>>(dHq, nH, part, d, m, chunks);
  }
  adaln_param_final_kernel<<<(B * 2 * d + 255) / 256, 256, 0, st>>>(part, dgb, d, chunks, B);
  return cudaGetLastError();
}

cudaError_t temb_bwd(const float* dgb, const bf16* W_t2, const float* a1, const float* u,
                     const float* e, float* da1, const TembGrads& g, int B, int d,
                     cudaStream_t st) {
  LaunchTimer lt("temb_bwd", st, 0.0, 8.0 * d * d);
  dim3 g1((d + 255) / 256, B);
  temb_bwd_du_kernel<<<g1, 256, 0, st>>>(dgb, W_t2, a1, da1, d);
  const long total = 2L * d * d + 2L * d + (long)d * 256 + d;
  temb_wgrad_kernel<<<(unsigned)((total + 255) / 256), 256, 0, st>>>(dgb, u, da1, e, g.W_t2, g.b_t2,
                                                                    g.W_t1, g.b_t1, d, B);
  return cudaGetLastError();
}

}  // namespace pf
