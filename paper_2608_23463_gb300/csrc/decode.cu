// Proxy-only KV-cache decode step and block-triggered append (Sec. 3.7 and
// 3.8, Eq. llm-cross, Eq. llm-gate, Eq. proxy-cache), bf16 storage with fp32
// arithmetic.
//
// Decode step, per sequence b (all on the caller's stream, four launches):
//   1. gemv_kernel<QKV>  one launch over two weight matrices.  Row tiles of
//                         W_qkv: q,k,v = W_qkv x; k, v go to the open slot n_o
//                         as bf16, q stays fp32 in the workspace; CTA b also
//                         copies x into X_open[n_o].  Row tiles of W_a1: the
//                         hidden layer of the alpha gate u = SiLU(W_a1
//                         RMSNorm(x) + b_a1) with the norm folded in (x * rms_w
//                         is fed to the MMA and the product scaled by
//                         1/rms(x) afterwards).
//   2. split_kernel      flash-decoding over the cached proxies: each CTA
//                         streams one slice of whole K_proxy/V_proxy rows (all
//                         heads) of one sequence and leaves (max, sum, acc[dh])
//                         partials per head.  CTA (0, b) also records whether
//                         the step is valid for b and advances n_open[b].
//   3. combine_kernel    alpha_h = sigmoid(W_a2[h] u + b_a2[h]); merges the
//                         partials into A_h, computes A_x over the open slots
//                         0..n_o, A = A_x + alpha_h A_h
//   4. gemv_kernel<OUT>  y = x + W_o A
// A sequence whose open block is already full (or whose n_open is out of
// range) is flagged (DEVERR_CAPACITY) and left untouched, y included.
#include <algorithm>

#include "kernels.h"
#include "proxyformer.h"

namespace pf {

int take_dev_error_decode() { return take_dev_error_tu(); }
int set_wait_limit_decode(unsigned long long ns) { return set_wait_limit_tu(ns); }

namespace {

constexpr int GEMV_WARPS = 8;     // K slices per CTA
constexpr int GEMV_MAXB = 8;      // batch rows handled per launch (the MMA's N)
constexpr int SPLIT_STAGES = 3;  // depth of the split kernel's copy ring
constexpr int SPLIT_STAGE_BYTES = 32768;  // K + V rows of one stage
constexpr int MAX_SPLITS = 1024;

enum { EPI_QKV = 0, EPI_OUT = 1 };

__device__ __forceinline__ void load8f(const float* p, float* v) {
  const float4 a = *reinterpret_cast<const float4*>(p), b = *reinterpret_cast<const float4*>(p + 4);
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}

struct GemvArgs {
  const bf16* W;  // [N, K]
  const bf16* x;  // [B, K]
  int B, N, K;    // B <= 8, K % 32 == 0
  // EPI_QKV: q (fp32 [B, d]), the open-slot X/K/V rows, and the alpha tiles
  float* q;
  bf16 *X_open, *K_open, *V_open;
  const int* n_open;
  int d, P;
  const bf16* W2;      // W_a1 [N2, K]: row tiles after the first ceil(N / 16)
  int N2;
  const float* rms_w;  // [K]
  const float* bias2;  // b_a1 [N2]
  bf16* out2;          // u [B, N2]
  // EPI_OUT: y = resid + acc (bf16), skipped where valid[b] == 0
  const bf16* resid;
  bf16* y;
  const int* valid;
};

// y[b, n] = sum_k W[n, k] x[b, k] for b < B <= 8 on the tensor cores: one
// m16n8k16 tile has 16 rows of W as M and the (up to) 8 sequences as N.  A CTA
// owns 16 rows; warp w takes the 32-wide K chunks w, w+8, ...  Within a chunk
// thread (g, t) loads 16 bytes at k = 8t of rows g and g+8 of W and of x row g
// and feeds them to two MMAs; the sum over k is order-free, so this
// permutation of k (the same for W and x) is exact.  The 8 warps' partial
// tiles are added in shared memory.
template <int EPI>
__global__ void __launch_bounds__(GEMV_WARPS * 32) gemv_kernel(GemvArgs a) {
  constexpr int U = 4;  // K chunks in flight per warp
  __shared__ float red[GEMV_WARPS][16][GEMV_MAXB];
  __shared__ float s_inv[GEMV_MAXB];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int g = lane >> 2, t = lane & 3;
  const int nt1 = (a.N + 15) / 16;
  // EPI_QKV launches also cover the alpha gate's W_a1 in tiles nt1, nt1+1, ...
  const bool second = EPI == EPI_QKV && (int)blockIdx.x >= nt1;
  const bf16* W = second ? a.W2 : a.W;
  const int N = second ? a.N2 : a.N;
  const int n0 = (second ? blockIdx.x - nt1 : blockIdx.x) * 16;
  const bool ra = n0 + g < N, rb = n0 + g + 8 < N, xb = g < a.B;
  const bf16* wa = W + (long)(ra ? n0 + g : 0) * a.K + 8 * t;
  const bf16* wb = W + (long)(rb ? n0 + g + 8 : 0) * a.K + 8 * t;
  const bf16* xr = a.x + (long)(xb ? g : 0) * a.K + 8 * t;
  if (EPI == EPI_QKV && !second && (int)blockIdx.x < a.B) {
    // CTA b: x -> X_open[b, n_o] (or flag a full / invalid open block)
    const int b = blockIdx.x, slot = a.n_open[b];
    if (slot >= 0 && slot < a.P) {
      for (int i = tid * 8; i < a.K; i += blockDim.x * 8)
        *reinterpret_cast<uint4*>(a.X_open + ((long)b * a.P + slot) * a.d + i) =
            *reinterpret_cast<const uint4*>(a.x + (long)b * a.K + i);
    } else if (tid == 0) {
      set_dev_error(DEVERR_CAPACITY);
    }
  }
  if (second) {
    // 1 / rms(x_b) for b = warp (Eq. llm-gate's RMSNorm)
    float ss = 0.f;
    if (warp < a.B)
      for (int i = lane * 8; i < a.K; i += 256) {
        float v[8];
        load8_bf16(a.x + (long)warp * a.K + i, v);
#pragma unroll
        for (int j = 0; j < 8; ++j) ss = fmaf(v[j], v[j], ss);
      }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    if (lane == 0) s_inv[warp] = rsqrtf(ss / a.K + 1e-6f);
  }
  float c[4] = {};
  for (int k0 = warp * 32; k0 < a.K; k0 += U * GEMV_WARPS * 32) {
    uint4 va[U], vb[U], vx[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int k = k0 + u * GEMV_WARPS * 32;
      const bool in = k < a.K;
      va[u] = (in && ra) ? *reinterpret_cast<const uint4*>(wa + k) : make_uint4(0, 0, 0, 0);
      vb[u] = (in && rb) ? *reinterpret_cast<const uint4*>(wb + k) : make_uint4(0, 0, 0, 0);
      vx[u] = (in && xb) ? *reinterpret_cast<const uint4*>(xr + k) : make_uint4(0, 0, 0, 0);
      if (second && in && xb) {  // x * rms_w, rounded to bf16 for the MMA
        const float* rw = a.rms_w + k + 8 * t;
        uint32_t* px = &vx[u].x;
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float2 f = unpack_bf16(px[e]);
          px[e] = pack_bf16(f.x * rw[2 * e], f.y * rw[2 * e + 1]);
        }
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const uint32_t a0[4] = {va[u].x, vb[u].x, va[u].y, vb[u].y};
      mma16816(c, a0, vx[u].x, vx[u].y);
      const uint32_t a1[4] = {va[u].z, vb[u].z, va[u].w, vb[u].w};
      mma16816(c, a1, vx[u].z, vx[u].w);
    }
  }
  red[warp][g][2 * t] = c[0];
  red[warp][g][2 * t + 1] = c[1];
  red[warp][g + 8][2 * t] = c[2];
  red[warp][g + 8][2 * t + 1] = c[3];
  __syncthreads();
  if (tid >= 16 * GEMV_MAXB) return;
  const int r = tid / GEMV_MAXB, b = tid % GEMV_MAXB, n = n0 + r;
  if (n >= N || b >= a.B) return;
  float v = 0.f;
#pragma unroll
  for (int w = 0; w < GEMV_WARPS; ++w) v += red[w][r][b];
  if (EPI == EPI_QKV) {
    const int slot = a.n_open[b];
    if (slot < 0 || slot >= a.P) return;  // flagged above
    if (second) {
      const float z = v * s_inv[b] + a.bias2[n];
      a.out2[(long)b * N + n] = __float2bfloat16(z * sigmoidf_(z));
    } else if (n < a.d) {
      a.q[(long)b * a.d + n] = v;
    } else if (n < 2 * a.d) {
      a.K_open[((long)b * a.P + slot) * a.d + (n - a.d)] = __float2bfloat16(v);
    } else {
      a.V_open[((long)b * a.P + slot) * a.d + (n - 2 * a.d)] = __float2bfloat16(v);
    }
  } else {
    if (!a.valid[b]) return;  // flagged: y left untouched
    a.y[(long)b * a.N + n] = __float2bfloat16(__bfloat162float(a.resid[(long)b * a.N + n]) + v);
  }
}

// Flash-decoding over the cached proxies.  Grid (splits, batch); CTA (s, b)
// owns proxies [j0, j1) = [s*chunk, (s+1)*chunk) of sequence b, for all heads.
// Those rows are contiguous in K_proxy / V_proxy, so thread 0 streams them in
// chunks of R rows with cp.async.bulk into a SPLIT_STAGES-deep shared-memory
// ring (one mbarrier per stage); the bytes in flight do not depend on the
// register count.  Thread t handles dimensions [8t, 8t+8) of every row (one
// 16-byte shared load of K and of V), so the DH/8 threads of a head form one
// online-softmax lane group.  The CTA is rounded up to whole warps; threads
// past d/8 hold zeros and write nothing.
// Partials: part[((b * splits + s) * nh + h) * (DH + 2)] = (max, sum, acc[DH]).
template <int DH>
__global__ void __launch_bounds__(512) split_kernel(
    const float* __restrict__ q, const bf16* __restrict__ Kc, const bf16* __restrict__ Vc,
    const int* __restrict__ n_proxy, int cap, int d, int nh, int splits, int R, float sl2,
    float* __restrict__ part, int* __restrict__ n_open, int P, int* __restrict__ valid) {
  constexpr int LPK = DH / 8;  // threads per head
  constexpr int U = 4;
  extern __shared__ __align__(128) unsigned char ring[];  // [stage][K rows | V rows]
  __shared__ __align__(8) uint64_t full[SPLIT_STAGES];
  const int s = blockIdx.x, b = blockIdx.y, tid = threadIdx.x;
  const int h = tid / LPK, gl = tid % LPK;
  const bool active = tid * 8 < d;
  const int np = min(max(n_proxy[b], 0), cap);
  const int chunk = (np + splits - 1) / splits;
  const int j0 = min(np, s * chunk), j1 = min(np, j0 + chunk);
  const int nchunks = (j1 - j0 + R - 1) / R;
  const uint32_t row_bytes = (uint32_t)d * 2u;
  const uint32_t half = (uint32_t)R * row_bytes;  // K (or V) bytes of one stage
  const uint32_t ring0 = smem_u32(ring), bar0 = smem_u32(full);
  if (tid == 0) {
    for (int i = 0; i < SPLIT_STAGES; ++i) mbar_init(bar0 + 8 * i, 1);
    fence_barrier_init();
    if (s == 0) {  // step bookkeeping: nothing else reads n_open during this kernel
      const int slot = n_open[b];
      const int ok = slot >= 0 && slot < P;
      valid[b] = ok;
      if (ok) n_open[b] = slot + 1;
    }
  }
  __syncthreads();
  int issued = 0;
  auto issue = [&](int c) {
    const int st = c % SPLIT_STAGES, r0 = j0 + c * R;
    const uint32_t bytes = (uint32_t)min(R, j1 - r0) * row_bytes;
    const long g = ((long)b * cap + r0) * d;
    mbar_arrive_expect_tx(bar0 + 8 * st, 2 * bytes);
    bulk_load(ring0 + st * 2 * half, Kc + g, bytes, bar0 + 8 * st);
    bulk_load(ring0 + st * 2 * half + half, Vc + g, bytes, bar0 + 8 * st);
  };
  if (tid == 0)
    for (; issued < min(SPLIT_STAGES, nchunks); ++issued) issue(issued);

  float qv[8] = {};
  if (active) load8f(q + (long)b * d + tid * 8, qv);
#pragma unroll
  for (int j = 0; j < 8; ++j) qv[j] *= sl2;
  float m = -INFINITY, l = 0.f, acc[8] = {};
  int c = 0;
  bool failed = false;
  for (; c < nchunks; ++c) {
    const int st = c % SPLIT_STAGES;
    const bool ok = mbar_wait(bar0 + 8 * st, (c / SPLIT_STAGES) & 1);
    const int nr = min(R, j1 - (j0 + c * R));  // uniform across the CTA
    const unsigned char* ks = ring + st * 2 * half + tid * 16;
    const unsigned char* vs = ks + half;
    for (int r = 0; ok && r < nr; r += U) {
      uint4 kr[U], vr[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        if (active && r + u < nr) {
          kr[u] = *reinterpret_cast<const uint4*>(ks + (r + u) * row_bytes);
          vr[u] = *reinterpret_cast<const uint4*>(vs + (r + u) * row_bytes);
        } else {
          kr[u] = make_uint4(0, 0, 0, 0);
          vr[u] = make_uint4(0, 0, 0, 0);
        }
      }
      float sc[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const uint32_t* pk = &kr[u].x;
        float t = 0.f;
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float2 f = unpack_bf16(pk[e]);
          t = fmaf(qv[2 * e], f.x, fmaf(qv[2 * e + 1], f.y, t));
        }
#pragma unroll
        for (int o = LPK / 2; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
        sc[u] = (r + u < nr) ? t : -INFINITY;
      }
      float mx = m;
#pragma unroll
      for (int u = 0; u < U; ++u) mx = fmaxf(mx, sc[u]);
      const float corr = exp2f(m - mx);  // m = -inf only before the first row: corr = 0
      l *= corr;
#pragma unroll
      for (int e = 0; e < 8; ++e) acc[e] *= corr;
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const float p = exp2f(sc[u] - mx);  // padded rows: exp2(-inf) = 0
        l += p;
        const uint32_t* pv = &vr[u].x;
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float2 f = unpack_bf16(pv[e]);
          acc[2 * e] = fmaf(p, f.x, acc[2 * e]);
          acc[2 * e + 1] = fmaf(p, f.y, acc[2 * e + 1]);
        }
      }
      m = mx;
    }
    // every thread is done with stage st: refill it (or leave together)
    if (__syncthreads_or(!ok)) {
      failed = true;
      break;
    }
    if (tid == 0 && issued < nchunks) issue(issued++);
  }
  if (failed) {  // a wait ran out: let this CTA's own copies land, then leave
    if (tid == 0)
      for (int it = c; it < issued; ++it)
        mbar_wait_drain(bar0 + 8 * (it % SPLIT_STAGES), (it / SPLIT_STAGES) & 1);
    __syncthreads();
    return;
  }
  if (!active) return;
  float* o = part + (((long)b * splits + s) * nh + h) * (DH + 2);
#pragma unroll
  for (int e = 0; e < 8; ++e) o[2 + gl * 8 + e] = acc[e];
  if (gl == 0) {
    o[0] = m;
    o[1] = l;
  }
}

// Per (b, h): A_h from the split partials, A_x over the open slots 0..n_o,
// alpha_h = sigmoid(W_a2[h] u_b + b_a2[h]), A = A_x + alpha_h A_h (fp32
// [B, d]).  COMBINE_G groups of DH threads: thread (g, t) owns head dim t and
// sums splits s = g, g+G, ... and open keys j = g, g+G, ...; the groups are
// added in shared memory.  Open-key scores take one thread per key.
constexpr int COMBINE_G = 4;
template <int DH>
__global__ void __launch_bounds__(COMBINE_G * DH) combine_kernel(
    const float* __restrict__ part, int splits, const float* __restrict__ q,
    const bf16* __restrict__ K_open, const bf16* __restrict__ V_open,
    const int* __restrict__ n_open, const int* __restrict__ valid, int P, int d, int nh, float sl2,
    const bf16* __restrict__ u, const bf16* __restrict__ W_a2, const float* __restrict__ b_a2,
    bf16* __restrict__ A) {
  __shared__ float s_p[PF_DECODE_MAX_P];
  __shared__ float s_m[MAX_SPLITS], s_l[MAX_SPLITS];
  __shared__ __align__(16) float s_q[DH];
  __shared__ float s_red[2][COMBINE_G - 1][DH];
  __shared__ float s_alpha;
  const int h = blockIdx.x, b = blockIdx.y, tid = threadIdx.x, lane = tid & 31;
  const int g = tid / DH, t = tid % DH;
  if (!valid[b]) return;  // flagged earlier; sequence untouched
  const int n = n_open[b];  // already advanced: open slots 0..n-1 incl. the new token
  if (tid < DH) s_q[tid] = q[(long)b * d + h * DH + tid] * sl2;
  const float* pb = part + ((long)b * splits * nh + h) * (DH + 2);
  const long pstride = (long)nh * (DH + 2);  // between splits
  for (int s = tid; s < splits; s += blockDim.x) {
    s_m[s] = pb[s * pstride];
    s_l[s] = pb[s * pstride + 1];
  }
  // alpha (Eq. llm-gate): the last warp
  if (tid >= blockDim.x - 32) {
    const int H = d / 8;
    float acc = 0.f;
    for (int k = lane; k < H; k += 32)
      acc = fmaf(__bfloat162float(W_a2[(long)h * H + k]), __bfloat162float(u[(long)b * H + k]),
                 acc);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (lane == 0) s_alpha = sigmoidf_(acc + b_a2[h]);
  }
  __syncthreads();
  // open-key scores: thread j < n computes key j's dot product (16-byte loads)
  if (tid < n) {
    const bf16* kr = K_open + ((long)b * P + tid) * d + h * DH;
    float v = 0.f;
#pragma unroll
    for (int e = 0; e < DH; e += 8) {
      float kv[8];
      load8_bf16(kr + e, kv);
#pragma unroll
      for (int i = 0; i < 8; ++i) v = fmaf(s_q[e + i], kv[i], v);
    }
    s_p[tid] = v;
  }
  __syncthreads();
  float M = -INFINITY;
  for (int s = 0; s < splits; ++s) M = fmaxf(M, s_m[s]);
  float mx = -INFINITY;
  for (int j = 0; j < n; ++j) mx = fmaxf(mx, s_p[j]);
  float ah = 0.f, ax = 0.f;
  if (M != -INFINITY) {
#pragma unroll 8
    for (int s = g; s < splits; s += COMBINE_G)
      ah = fmaf(pb[s * pstride + 2 + t], exp2f(s_m[s] - M), ah);
  }
#pragma unroll 8
  for (int j = g; j < n; j += COMBINE_G)
    ax = fmaf(exp2f(s_p[j] - mx), __bfloat162float(V_open[((long)b * P + j) * d + h * DH + t]),
              ax);
  if (g > 0) {
    s_red[0][g - 1][t] = ah;
    s_red[1][g - 1][t] = ax;
  }
  __syncthreads();
  if (g > 0) return;
  float Lh = 0.f, Lx = 0.f;
  if (M != -INFINITY)
    for (int s = 0; s < splits; ++s) Lh = fmaf(s_l[s], exp2f(s_m[s] - M), Lh);
  for (int j = 0; j < n; ++j) Lx += exp2f(s_p[j] - mx);
#pragma unroll
  for (int i = 0; i < COMBINE_G - 1; ++i) {
    ah += s_red[0][i][t];
    ax += s_red[1][i][t];
  }
  const float Ah = (M != -INFINITY) ? ah / Lh : 0.f;
  A[(long)b * d + h * DH + t] = __float2bfloat16(ax / Lx + s_alpha * Ah);
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

}  // namespace

namespace {
size_t round64(size_t n) { return (n + 63) & ~size_t(63); }
// cache rows per stage of the split kernel's ring (K and V of R rows fill
// SPLIT_STAGE_BYTES)
int split_rows(int d) { return std::max(1, SPLIT_STAGE_BYTES / (4 * d)); }
}  // namespace

size_t decode_workspace_bytes(int B, int d, int nh, int splits) {
  const int dh = d / nh;
  // q, u, A, valid, partials (fp32-sized slots, each a multiple of 256 bytes)
  const size_t n = round64((size_t)B * d) + round64((size_t)B * d / 8) + round64((size_t)B * d) +
                   round64((size_t)B) + round64((size_t)B * nh * splits * (dh + 2));
  return n * sizeof(float) + 256;
}

int decode_splits(int B, int nh, int cap) {
  (void)nh;
  // about 304 CTAs in total (2 per SM of a 152-SM part: each holds a 96 KB
  // copy ring), at least 16 cache rows per split; independent of the device
  // so sizes are fixed
  int s = (304 + B - 1) / B;
  s = std::max(1, std::min(s, std::max(1, cap / 16)));
  return std::min(s, MAX_SPLITS);
}

cudaError_t decode_step_launch(const DecodeLaunch& L, cudaStream_t st) {
  const int d = L.d, nh = L.nh, dh = d / nh, B = L.B, H = d / 8;
  float* q = L.ws;
  bf16* u = reinterpret_cast<bf16*>(q + round64((size_t)B * d));  // bf16 arrays in fp32-sized slots
  bf16* A = u + 2 * round64((size_t)B * H);
  int* valid = reinterpret_cast<int*>(A + 2 * round64((size_t)B * d));
  float* part = reinterpret_cast<float*>(valid + round64((size_t)B));
  const float sl2 = 1.4426950408889634f / sqrtf((float)dh);
  cudaError_t e;
  for (int b0 = 0; b0 < B; b0 += GEMV_MAXB) {  // the GEMV handles 8 sequences per launch
    const int nb = std::min(GEMV_MAXB, B - b0);
    GemvArgs g{};
    g.W = L.W_qkv;
    g.x = L.x + (size_t)b0 * d;
    g.B = nb;
    g.N = 3 * d;
    g.K = d;
    g.q = q + (size_t)b0 * d;
    g.X_open = L.X_open + (size_t)b0 * L.P * d;
    g.K_open = L.K_open + (size_t)b0 * L.P * d;
    g.V_open = L.V_open + (size_t)b0 * L.P * d;
    g.n_open = L.n_open + b0;
    g.d = d;
    g.P = L.P;
    g.W2 = L.W_a1;
    g.N2 = H;
    g.rms_w = L.rms_w;
    g.bias2 = L.b_a1;
    g.out2 = u + (size_t)b0 * H;
    LaunchTimer lt("decode_qkv_alpha", st, 2.0 * nb * (3.0 * d + H) * d,
                   2.0 * (3.0 * d + H) * d + 6.0 * nb * d);
    const int tiles = (3 * d + 15) / 16 + (H + 15) / 16;
    gemv_kernel<EPI_QKV><<<tiles, GEMV_WARPS * 32, 0, st>>>(g);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  {
    dim3 grid(L.splits, B);
    const int nthr = (d / 8 + 31) / 32 * 32;
    const int R = split_rows(d);
    const size_t smem = (size_t)SPLIT_STAGES * 2 * R * d * sizeof(bf16);
    auto k = dh == 128 ? split_kernel<128> : split_kernel<64>;
    if ((e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) !=
        cudaSuccess)
      return e;
    LaunchTimer lt("decode_split", st, 4.0 * B * (double)L.cap * d,
                   4.0 * B * (double)L.cap * d);  // bytes: upper bound (full cache)
    k<<<grid, nthr, smem, st>>>(q, L.K_proxy, L.V_proxy, L.n_proxy, L.cap, d, nh, L.splits, R,
                                sl2, part, L.n_open, L.P, valid);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  {
    dim3 grid(nh, B);
    LaunchTimer lt("decode_combine", st, 4.0 * B * d * L.P, 4.0 * B * d * L.P);
    if (dh == 128)
      combine_kernel<128><<<grid, COMBINE_G * 128, 0, st>>>(part, L.splits, q, L.K_open, L.V_open,
                                                            L.n_open, valid, L.P, d, nh, sl2, u,
                                                            L.W_a2, L.b_a2, A);
    else
      combine_kernel<64><<<grid, COMBINE_G * 64, 0, st>>>(part, L.splits, q, L.K_open, L.V_open,
                                                          L.n_open, valid, L.P, d, nh, sl2, u,
                                                          L.W_a2, L.b_a2, A);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  for (int b0 = 0; b0 < B; b0 += GEMV_MAXB) {
    GemvArgs o{};
    o.W = L.W_o;
    o.x = A + (size_t)b0 * d;
    o.B = std::min(GEMV_MAXB, B - b0);
    o.N = d;
    o.K = d;
    o.resid = L.x + (size_t)b0 * d;
    o.y = L.y + (size_t)b0 * d;
    o.valid = valid + b0;
    LaunchTimer lt("decode_out", st, 2.0 * o.B * d * (double)d, 2.0 * d * (double)d + 6.0 * o.B * d);
    gemv_kernel<EPI_OUT><<<(d + 15) / 16, GEMV_WARPS * 32, 0, st>>>(o);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  return cudaSuccess;
}

// Prefill: every sequence's cache holds m proxies and r open tokens.
__global__ void prefill_counts_kernel(int* n_open, int* n_proxy, int B, int m, int r) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b < B) {
    n_proxy[b] = m;
    n_open[b] = r;
  }
}

cudaError_t prefill_counts(int* n_open, int* n_proxy, int B, int m, int r, cudaStream_t st) {
  LaunchTimer lt("prefill_counts", st, 0.0, 8.0 * B);
  prefill_counts_kernel<<<(B + 127) / 128, 128, 0, st>>>(n_open, n_proxy, B, m, r);
  return cudaGetLastError();
}

cudaError_t append_finish(int* n_open, int* n_proxy, int B, int P, int cap, cudaStream_t st) {
  LaunchTimer lt("append_finish", st, 0.0, 16.0 * B);
  append_finish_kernel<<<1, 32 * ((B + 31) / 32), 0, st>>>(n_open, n_proxy, B, P, cap);
  return cudaGetLastError();
}

}  // namespace pf
