// Proxy-only KV-cache decode step and block-triggered append (Sec. 3.7 and
// 3.8, Eq. llm-cross, Eq. llm-gate, Eq. proxy-cache), bf16 storage with fp32
// arithmetic.
//
// Decode step, per sequence b (all on the caller's stream):
//   1. gemv_kernel<QKV>   q,k,v = W_qkv x; k, v go to the open slot n_o as
//                          bf16, q stays fp32 in the workspace
//   2. alpha_kernel       x -> X_open[n_o]; alpha = sigmoid(W_a2 SiLU(W_a1
//                          RMSNorm(x) + b_a1) + b_a2), one value per head
//   3. split_kernel       flash-decoding over the cached proxies: each CTA
//                          streams one slice of K_proxy/V_proxy rows of one
//                          (b, head) with 16-byte loads and leaves (max, sum,
//                          acc[dh]) partials
//   4. combine_kernel     merges the partials into A_h, computes A_x over the
//                          open slots 0..n_o, A = A_x + alpha_h A_h
//   5. gemv_kernel<OUT>   y = x + W_o A
//   6. finish_kernel      n_open += 1
// A sequence whose open block is already full is flagged (DEVERR_CAPACITY)
// and left untouched, y included.
#include <algorithm>

#include "kernels.h"
#include "proxyformer.h"

namespace pf {

int take_dev_error_decode() { return take_dev_error_tu(); }

namespace {

constexpr int GEMV_WARPS = 8;
constexpr int GEMV_ROWS = 4;     // output rows per warp
constexpr int GEMV_MAXB = 8;     // batch rows handled per launch
constexpr int SPLIT_THREADS = 128;

enum { EPI_QKV = 0, EPI_OUT = 1, EPI_F32 = 2 };

__device__ __forceinline__ void load8f(const float* p, float* v) {
  const float4 a = *reinterpret_cast<const float4*>(p), b = *reinterpret_cast<const float4*>(p + 4);
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}

struct GemvArgs {
  const bf16* W;   // [N, K]
  const void* x;   // [B, K], bf16 (x_f32 = 0) or fp32
  int x_f32;
  int B, N, K;
  // EPI_QKV: q (fp32 [B, d]) and the open-slot K/V rows
  float* q;
  bf16 *K_open, *V_open;
  const int* n_open;
  int d, P;
  // EPI_OUT: y = resid + acc (bf16); EPI_F32: out = acc (fp32 [B, N])
  const bf16* resid;
  bf16* y;
  float* out;
};

// y[b, n] = sum_k W[n, k] x[b, k] for b < B <= 8.  Each warp owns GEMV_ROWS
// rows of W; lane l reads 16-byte chunks l, l+32, ... of those rows, so each
// W element is loaded once and reused for every batch row (x is staged in
// shared memory as fp32).
template <int EPI>
__global__ void __launch_bounds__(GEMV_WARPS * 32) gemv_kernel(GemvArgs a) {
  extern __shared__ float xs[];  // [B][K]
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int i = tid * 8; i < a.B * a.K; i += blockDim.x * 8) {
    float v[8];
    if (a.x_f32)
      load8f(reinterpret_cast<const float*>(a.x) + i, v);
    else
      load8_bf16(reinterpret_cast<const bf16*>(a.x) + i, v);
#pragma unroll
    for (int j = 0; j < 8; ++j) xs[i + j] = v[j];
  }
  __syncthreads();
  const int n0 = (blockIdx.x * GEMV_WARPS + warp) * GEMV_ROWS;
  if (n0 >= a.N) return;
  float acc[GEMV_ROWS][GEMV_MAXB] = {};
  for (int k = lane * 8; k < a.K; k += 256) {
    float w[GEMV_ROWS][8];
#pragma unroll
    for (int r = 0; r < GEMV_ROWS; ++r) {
      if (n0 + r < a.N)
        load8_bf16(a.W + (long)(n0 + r) * a.K + k, w[r]);
      else
#pragma unroll
        for (int j = 0; j < 8; ++j) w[r][j] = 0.f;
    }
#pragma unroll
    for (int b = 0; b < GEMV_MAXB; ++b) {
      if (b >= a.B) break;
      float xv[8];
      load8f(xs + b * a.K + k, xv);
#pragma unroll
      for (int r = 0; r < GEMV_ROWS; ++r)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[r][b] = fmaf(w[r][j], xv[j], acc[r][b]);
    }
  }
#pragma unroll
  for (int r = 0; r < GEMV_ROWS; ++r)
#pragma unroll
    for (int b = 0; b < GEMV_MAXB; ++b)
#pragma unroll
      for (int s = 16; s > 0; s >>= 1) acc[r][b] += __shfl_xor_sync(0xffffffffu, acc[r][b], s);
  // lane (r * 8 + b) writes output (n0 + r, b)
#pragma unroll
  for (int r = 0; r < GEMV_ROWS; ++r) {
#pragma unroll
    for (int b = 0; b < GEMV_MAXB; ++b) {
      if (lane != r * GEMV_MAXB + b) continue;
      const int n = n0 + r;
      if (n >= a.N || b >= a.B) continue;
      const float v = acc[r][b];
      if (EPI == EPI_QKV) {
        const int slot = a.n_open[b];
        if (slot < 0 || slot >= a.P) continue;  // flagged by alpha_kernel
        if (n < a.d) {
          a.q[(long)b * a.d + n] = v;
        } else if (n < 2 * a.d) {
          a.K_open[((long)b * a.P + slot) * a.d + (n - a.d)] = __float2bfloat16(v);
        } else {
          a.V_open[((long)b * a.P + slot) * a.d + (n - 2 * a.d)] = __float2bfloat16(v);
        }
      } else if (EPI == EPI_OUT) {
        const int slot = a.n_open[b];
        if (slot < 0 || slot >= a.P) continue;  // flagged: y left untouched
        a.y[(long)b * a.N + n] = __float2bfloat16(__bfloat162float(a.resid[(long)b * a.N + n]) + v);
      } else {
        a.out[(long)b * a.N + n] = v;
      }
    }
  }
}

__device__ __forceinline__ float block_sum(float v, float* red) {
#pragma unroll
  for (int s = 16; s > 0; s >>= 1) v += __shfl_xor_sync(0xffffffffu, v, s);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  float t = 0.f;
  for (int i = 0; i < nw; ++i) t += red[i];
  return t;
}

// One CTA per sequence: copies x into the open slot (after checking it), and
// computes the per-head gate alpha (Eq. llm-gate).
__global__ void __launch_bounds__(256) alpha_kernel(const bf16* __restrict__ x, int d, int nh,
                                                    int P, const int* __restrict__ n_open,
                                                    bf16* __restrict__ X_open,
                                                    const float* __restrict__ rms_w,
                                                    const bf16* __restrict__ W_a1,
                                                    const float* __restrict__ b_a1,
                                                    const bf16* __restrict__ W_a2,
                                                    const float* __restrict__ b_a2,
                                                    float* __restrict__ alpha) {
  extern __shared__ float sm[];  // r [d], u [d/8], red [32]
  float* r = sm;
  float* u = sm + d;
  float* red = u + d / 8;
  const int b = blockIdx.x, tid = threadIdx.x;
  const int slot = n_open[b];
  const bool ok = slot >= 0 && slot < P;
  if (!ok && tid == 0) set_dev_error(DEVERR_CAPACITY);
  float ss = 0.f;
  for (int i = tid; i < d; i += blockDim.x) {
    const bf16 xv = x[(long)b * d + i];
    if (ok) X_open[((long)b * P + slot) * d + i] = xv;
    const float f = __bfloat162float(xv);
    r[i] = f;
    ss += f * f;
  }
  const float inv = rsqrtf(block_sum(ss, red) / d + 1e-6f);
  for (int i = tid; i < d; i += blockDim.x) r[i] = r[i] * inv * rms_w[i];
  __syncthreads();
  const int H = d / 8, lane = tid & 31, warp = tid >> 5, nw = blockDim.x >> 5;
  for (int o = warp; o < H; o += nw) {  // u = SiLU(W_a1 r + b_a1)
    float acc = 0.f;
    for (int k = lane * 8; k < d; k += 256) {
      float w[8];
      load8_bf16(W_a1 + (long)o * d + k, w);
#pragma unroll
      for (int j = 0; j < 8; ++j) acc = fmaf(w[j], r[k + j], acc);
    }
#pragma unroll
    for (int s = 16; s > 0; s >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, s);
    if (lane == 0) {
      const float z = acc + b_a1[o];
      u[o] = z * sigmoidf_(z);
    }
  }
  __syncthreads();
  for (int h = warp; h < nh; h += nw) {  // alpha = sigmoid(W_a2 u + b_a2)
    float acc = 0.f;
    for (int k = lane; k < H; k += 32) acc = fmaf(__bfloat162float(W_a2[(long)h * H + k]), u[k], acc);
#pragma unroll
    for (int s = 16; s > 0; s >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, s);
    if (lane == 0) alpha[b * nh + h] = sigmoidf_(acc + b_a2[h]);
  }
}

// Flash-decoding over the cached proxies.  Grid (splits, heads, batch); each
// CTA handles proxies [s*chunk, (s+1)*chunk) of its (b, h).  A key row of one
// head is DH bf16 = DH/8 lanes x 16 bytes, so a warp holds 256/DH keys at once;
// each such lane group keeps its own online-softmax state (max, sum, acc), and
// the groups are merged through shared memory at the end.
template <int DH>
__global__ void __launch_bounds__(SPLIT_THREADS) split_kernel(
    const float* __restrict__ q, const bf16* __restrict__ Kc, const bf16* __restrict__ Vc,
    const int* __restrict__ n_proxy, int cap, int d, int nh, int splits, float sl2,
    float* __restrict__ part) {
  constexpr int LPK = DH / 8;               // lanes per key
  constexpr int GROUPS = SPLIT_THREADS / LPK;
  constexpr int U = 4;                      // keys in flight per group
  __shared__ float s_m[GROUPS], s_l[GROUPS];
  __shared__ float s_acc[GROUPS][DH];
  const int s = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, grp = tid / LPK, gl = tid % LPK;
  const int np = min(max(n_proxy[b], 0), cap);
  const int chunk = (np + splits - 1) / splits;
  const int j0 = s * chunk, j1 = min(np, j0 + chunk);
  float qv[8];
  load8f(q + (long)b * d + h * DH + gl * 8, qv);
#pragma unroll
  for (int j = 0; j < 8; ++j) qv[j] *= sl2;
  float m = -INFINITY, l = 0.f, acc[8] = {};
  const long base = ((long)b * cap) * d + h * DH + gl * 8;
  // uniform trip count across the CTA (the shuffles below span whole warps)
  for (int jb = j0; jb < j1; jb += GROUPS * U) {
    float kv[U][8], vv[U][8];
    bool val[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int jj = jb + grp + u * GROUPS;
      val[u] = jj < j1;
      if (val[u]) {
        load8_bf16(Kc + base + (long)jj * d, kv[u]);
        load8_bf16(Vc + base + (long)jj * d, vv[u]);
      } else {  // keep p * v finite for the padded slots (p = 0 there)
#pragma unroll
        for (int e = 0; e < 8; ++e) kv[u][e] = vv[u][e] = 0.f;
      }
    }
    float sc[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      float t = 0.f;
#pragma unroll
      for (int e = 0; e < 8; ++e) t = fmaf(qv[e], kv[u][e], t);
#pragma unroll
      for (int o = LPK / 2; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
      sc[u] = val[u] ? t : -INFINITY;
    }
    float mx = m;
#pragma unroll
    for (int u = 0; u < U; ++u) mx = fmaxf(mx, sc[u]);
    const float corr = (mx == -INFINITY) ? 1.f : exp2f(m - mx);  // 0 on the first keys
    l *= corr;
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[e] *= corr;
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const float p = val[u] ? exp2f(sc[u] - mx) : 0.f;
      l += p;
#pragma unroll
      for (int e = 0; e < 8; ++e) acc[e] = fmaf(p, vv[u][e], acc[e]);
    }
    m = mx;
  }
  if (gl == 0) {
    s_m[grp] = m;
    s_l[grp] = l;
  }
#pragma unroll
  for (int e = 0; e < 8; ++e) s_acc[grp][gl * 8 + e] = acc[e];
  __syncthreads();
  if (tid < DH) {
    float M = -INFINITY;
    for (int g = 0; g < GROUPS; ++g) M = fmaxf(M, s_m[g]);
    float L = 0.f, A = 0.f;
    if (M != -INFINITY) {
      for (int g = 0; g < GROUPS; ++g) {
        const float w = exp2f(s_m[g] - M);
        L += s_l[g] * w;
        A += s_acc[g][tid] * w;
      }
    }
    float* o = part + (((long)b * nh + h) * splits + s) * (DH + 2);
    o[2 + tid] = A;
    if (tid == 0) {
      o[0] = M;
      o[1] = L;
    }
  }
}

// Per (b, h): A_h from the split partials, A_x over the open slots 0..n_o,
// A = A_x + alpha_h A_h (fp32 [B, d]).  One thread per head dimension.
template <int DH>
__global__ void __launch_bounds__(DH) combine_kernel(
    const float* __restrict__ part, int splits, const float* __restrict__ q,
    const bf16* __restrict__ K_open, const bf16* __restrict__ V_open,
    const int* __restrict__ n_open, int P, int d, int nh, float sl2,
    const float* __restrict__ alpha, float* __restrict__ A) {
  __shared__ float s_p[PF_DECODE_MAX_P];
  __shared__ float s_red[DH / 32];
  const int h = blockIdx.x, b = blockIdx.y, t = threadIdx.x;
  const int slot = n_open[b];
  if (slot < 0 || slot >= P) return;  // flagged in alpha_kernel
  // A_h
  const float* pb = part + ((long)b * nh + h) * splits * (DH + 2);
  float M = -INFINITY;
  for (int s = 0; s < splits; ++s) M = fmaxf(M, pb[s * (DH + 2)]);
  float Ah = 0.f;
  if (M != -INFINITY) {
    float L = 0.f, acc = 0.f;
    for (int s = 0; s < splits; ++s) {
      const float w = exp2f(pb[s * (DH + 2)] - M);
      L += pb[s * (DH + 2) + 1] * w;
      acc += pb[s * (DH + 2) + 2 + t] * w;
    }
    Ah = acc / L;
  }
  // A_x: softmax over open slots 0..slot of q.k / sqrt(dh)
  const float qt = q[(long)b * d + h * DH + t] * sl2;
  const int n = slot + 1;
  for (int j = 0; j < n; ++j) {
    float v = qt * __bfloat162float(K_open[((long)b * P + j) * d + h * DH + t]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    __syncthreads();
    if ((t & 31) == 0) s_red[t >> 5] = v;
    __syncthreads();
    if (t == 0) {
      float sum = 0.f;
      for (int w = 0; w < DH / 32; ++w) sum += s_red[w];
      s_p[j] = sum;
    }
  }
  __syncthreads();
  float mx = -INFINITY;
  for (int j = 0; j < n; ++j) mx = fmaxf(mx, s_p[j]);
  float L = 0.f, Ax = 0.f;
  for (int j = 0; j < n; ++j) {
    const float p = exp2f(s_p[j] - mx);
    L += p;
    Ax = fmaf(p, __bfloat162float(V_open[((long)b * P + j) * d + h * DH + t]), Ax);
  }
  A[(long)b * d + h * DH + t] = Ax / L + alpha[b * nh + h] * Ah;
}

__global__ void decode_finish_kernel(int* n_open, int B, int P) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b < B && n_open[b] >= 0 && n_open[b] < P) n_open[b] += 1;
}

// Append bookkeeping: a sequence is appended iff its block is full and its
// cache has room; others are flagged.  Runs after the cache rows are written.
__global__ void append_finish_kernel(int* n_open, int* n_proxy, int B, int P, int cap) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  if (n_open[b] == P && n_proxy[b] >= 0 && n_proxy[b] < cap) {
    n_proxy[b] += 1;
    n_open[b] = 0;
  } else {
    set_dev_error(DEVERR_CAPACITY);
  }
}

template <int EPI>
cudaError_t launch_gemv(const GemvArgs& a, cudaStream_t st, const char* label) {
  const int rows_per_cta = GEMV_WARPS * GEMV_ROWS;
  const size_t smem = (size_t)a.B * a.K * sizeof(float);
  auto k = gemv_kernel<EPI>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  LaunchTimer lt(label, st, 2.0 * a.B * a.N * a.K, 2.0 * a.N * a.K + 6.0 * a.B * a.K);
  k<<<(a.N + rows_per_cta - 1) / rows_per_cta, GEMV_WARPS * 32, smem, st>>>(a);
  return cudaGetLastError();
}

}  // namespace

namespace {
size_t round64(size_t n) { return (n + 63) & ~size_t(63); }
}  // namespace

size_t decode_workspace_bytes(int B, int d, int nh, int splits) {
  const int dh = d / nh;
  const size_t n = round64((size_t)B * d) + round64((size_t)B * nh) + round64((size_t)B * d) +
                   round64((size_t)B * nh * splits * (dh + 2));
  return n * sizeof(float) + 256;
}

int decode_splits(int B, int nh, int cap) {
  // about 1216 CTAs in total (8 per SM of a 152-SM part), at most one split
  // per 128 cache rows; independent of the device so sizes are fixed
  int s = (1216 + B * nh - 1) / (B * nh);
  s = std::max(1, std::min(s, std::max(1, cap / 128)));
  return std::min(s, 64);
}

cudaError_t decode_step_launch(const DecodeLaunch& L, cudaStream_t st) {
  const int d = L.d, nh = L.nh, dh = d / nh, B = L.B;
  float* q = L.ws;
  float* alpha = q + round64((size_t)B * d);
  float* A = alpha + round64((size_t)B * nh);
  float* part = A + round64((size_t)B * d);
  const float sl2 = 1.4426950408889634f / sqrtf((float)dh);
  cudaError_t e;
  {
    LaunchTimer lt("decode_alpha", st, 2.0 * B * (d * (d / 8) + (d / 8) * nh),
                   2.0 * d * (d / 8) + 4.0 * B * d);
    const size_t smem = (size_t)(d + d / 8 + 32) * sizeof(float);
    alpha_kernel<<<B, 256, smem, st>>>(L.x, d, nh, L.P, L.n_open, L.X_open, L.rms_w, L.W_a1, L.b_a1,
                                       L.W_a2, L.b_a2, alpha);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  for (int b0 = 0; b0 < B; b0 += GEMV_MAXB) {  // the GEMV handles 8 sequences per launch
    GemvArgs g{};
    g.W = L.W_qkv;
    g.x = L.x + (size_t)b0 * d;
    g.x_f32 = 0;
    g.B = std::min(GEMV_MAXB, B - b0);
    g.N = 3 * d;
    g.K = d;
    g.q = q + (size_t)b0 * d;
    g.K_open = L.K_open + (size_t)b0 * L.P * d;
    g.V_open = L.V_open + (size_t)b0 * L.P * d;
    g.n_open = L.n_open + b0;
    g.d = d;
    g.P = L.P;
    if ((e = launch_gemv<EPI_QKV>(g, st, "decode_qkv")) != cudaSuccess) return e;
  }
  {
    dim3 grid(L.splits, nh, B);
    LaunchTimer lt("decode_split", st, 4.0 * B * (double)L.cap * d,
                   4.0 * B * (double)L.cap * d);  // bytes: upper bound (full cache)
    if (dh == 128)
      split_kernel<128><<<grid, SPLIT_THREADS, 0, st>>>(q, L.K_proxy, L.V_proxy, L.n_proxy, L.cap, d,
                                                        nh, L.splits, sl2, part);
    else
      split_kernel<64><<<grid, SPLIT_THREADS, 0, st>>>(q, L.K_proxy, L.V_proxy, L.n_proxy, L.cap, d,
                                                       nh, L.splits, sl2, part);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  {
    dim3 grid(nh, B);
    LaunchTimer lt("decode_combine", st, 4.0 * B * d * L.P, 4.0 * B * d * L.P);
    if (dh == 128)
      combine_kernel<128><<<grid, 128, 0, st>>>(part, L.splits, q, L.K_open, L.V_open, L.n_open,
                                                L.P, d, nh, sl2, alpha, A);
    else
      combine_kernel<64><<<grid, 64, 0, st>>>(part, L.splits, q, L.K_open, L.V_open, L.n_open,
                                              L.P, d, nh, sl2, alpha, A);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  for (int b0 = 0; b0 < B; b0 += GEMV_MAXB) {
    GemvArgs o{};
    o.W = L.W_o;
    o.x = A + (size_t)b0 * d;
    o.x_f32 = 1;
    o.B = std::min(GEMV_MAXB, B - b0);
    o.N = d;
    o.K = d;
    o.resid = L.x + (size_t)b0 * d;
    o.y = L.y + (size_t)b0 * d;
    o.n_open = L.n_open + b0;
    o.P = L.P;
    if ((e = launch_gemv<EPI_OUT>(o, st, "decode_out")) != cudaSuccess) return e;
  }
  {
    LaunchTimer lt("decode_finish", st, 0.0, 8.0 * B);
    decode_finish_kernel<<<1, 32 * ((B + 31) / 32), 0, st>>>(L.n_open, B, L.P);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  return cudaSuccess;
}

cudaError_t append_finish(int* n_open, int* n_proxy, int B, int P, int cap, cudaStream_t st) {
  LaunchTimer lt("append_finish", st, 0.0, 16.0 * B);
  append_finish_kernel<<<1, 32 * ((B + 31) / 32), 0, st>>>(n_open, n_proxy, B, P, cap);
  return cudaGetLastError();
}

}  // namespace pf
