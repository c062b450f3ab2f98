// Proxy-space multi-head attention (Eq. proxy-attn), forward and backward,
// head width 64, bf16 operands with fp32 softmax statistics.
//
// Q, K, V live in one [B*m, 3d] bf16 matrix (columns [Q | K | V], head h at
// h*64 inside each third); the attention output A is [B*m, d].  The forward
// (attention_tc.cu) saves LSE (log2 units) per (b, h, query).  The backward
// here recomputes the probabilities from LSE: one kernel accumulates dK, dV
// per key tile over the query tiles, a second accumulates dQ per query tile
// over the key tiles, so no atomics are needed and results are deterministic.
#include "kernels.h"

namespace pf {

namespace {

constexpr int AT = 64;  // tile rows (queries or keys) and head width

__device__ __forceinline__ void ldsm4(uint32_t* r, uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
__device__ __forceinline__ void ldsm4t(uint32_t* r, uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, bool valid) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src),
               "r"(valid ? 16 : 0)
               : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// 64 x 64 bf16 tile, 128-byte rows, 16-byte chunk c of row r stored at chunk
// c ^ (r & 7) (conflict-free ldmatrix).
__device__ __forceinline__ uint32_t tile_off(int r, int c) {
  return (uint32_t)(r * 128 + ((c ^ (r & 7)) << 4));
}

// Load rows [r0, r0+64) x 64 columns starting at `col` of a row-major matrix
// with `ld` elements per row; rows >= nrows are zero-filled.
__device__ __forceinline__ void load_tile(uint32_t s, const bf16* g, long row_base, int r0,
                                          int nrows, long ld, int col) {
#pragma unroll
  for (int it = 0; it < 4; ++it) {
    const int idx = threadIdx.x + it * 128;  // 512 chunks
    const int r = idx >> 3, c = idx & 7;
    const bool ok = (r0 + r) < nrows;
    const bf16* src = ok ? g + (row_base + r0 + r) * ld + col + c * 8 : g;
    cp_async16(s + tile_off(r, c), src, ok);
  }
}

// A-operand fragments (16 rows x 64) of rows [w*16, w*16+16) of a tile.
__device__ __forceinline__ void load_afrag(uint32_t (*f)[4], uint32_t s, int w) {
  const int lane = threadIdx.x & 31, mi = lane >> 3;
#pragma unroll
  for (int kc = 0; kc < 4; ++kc) {
    const int r = w * 16 + (mi & 1) * 8 + (lane & 7);
    ldsm4(f[kc], s + tile_off(r, kc * 2 + (mi >> 1)));
  }
}

// acc[8][4] (16 x 64) += A(16 x 64, fragments) * T^T where T is a 64x64 smem
// tile indexed [n][k] (B operand "col" layout straight from row-major rows).
__device__ __forceinline__ void mma_abt(float (*acc)[4], uint32_t (*a)[4], uint32_t s) {
  const int lane = threadIdx.x & 31, mi = lane >> 3;
#pragma unroll
  for (int kc = 0; kc < 4; ++kc) {
#pragma unroll
    for (int np = 0; np < 4; ++np) {
      uint32_t b[4];
      ldsm4(b, s + tile_off(np * 16 + (mi >> 1) * 8 + (lane & 7), kc * 2 + (mi & 1)));
      mma16816(acc[2 * np], a[kc], b[0], b[1]);
      mma16816(acc[2 * np + 1], a[kc], b[2], b[3]);
    }
  }
}

// acc[8][4] (16 x 64) += P(16 x 64, C-layout fp32 in p[8][4]) * T where T is
// a 64x64 smem tile indexed [k][n].
__device__ __forceinline__ void mma_pt(float (*acc)[4], const float (*p)[4], uint32_t s) {
  const int lane = threadIdx.x & 31, mi = lane >> 3;
#pragma unroll
  for (int kc = 0; kc < 4; ++kc) {
    uint32_t a[4];
    a[0] = pack_bf16(p[2 * kc][0], p[2 * kc][1]);
    a[1] = pack_bf16(p[2 * kc][2], p[2 * kc][3]);
    a[2] = pack_bf16(p[2 * kc + 1][0], p[2 * kc + 1][1]);
    a[3] = pack_bf16(p[2 * kc + 1][2], p[2 * kc + 1][3]);
#pragma unroll
    for (int dp = 0; dp < 4; ++dp) {
      uint32_t b[4];
      ldsm4t(b, s + tile_off(kc * 16 + (mi & 1) * 8 + (lane & 7), dp * 2 + (mi >> 1)));
      mma16816(acc[2 * dp], a, b[0], b[1]);
      mma16816(acc[2 * dp + 1], a, b[2], b[3]);
    }
  }
}

// Di = rowsum(dO * O) per (b, h, query): one warp per (row, head).
__global__ void attn_bwd_dot_kernel(const bf16* __restrict__ dO, const bf16* __restrict__ O,
                                    float* __restrict__ Dout, int rows, int m, int d, int nh) {
  const long wid = ((long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (wid >= (long)rows * nh) return;
  const long row = wid / nh;
  const int h = (int)(wid % nh);
  const long off = row * d + h * AT + lane * 2;
  const float2 a = unpack_bf16(*reinterpret_cast<const uint32_t*>(dO + off));
  const float2 c = unpack_bf16(*reinterpret_cast<const uint32_t*>(O + off));
  float v = a.x * c.x + a.y * c.y;
#pragma unroll
  for (int s = 16; s > 0; s >>= 1) v += __shfl_xor_sync(0xffffffffu, v, s);
  if (lane == 0) {
    const long b = row / m, i = row % m;
    Dout[(b * nh + h) * m + i] = v;
  }
}

// dK, dV for one 64-key tile, looping over query tiles.  Warp w owns keys
// k0 + 16w .. k0 + 16w + 15.
template <bool CAUSAL>
__global__ void __launch_bounds__(128) attn_bwd_dkdv_kernel(
    const bf16* __restrict__ qkv, const bf16* __restrict__ dO, const float* __restrict__ lse,
    const float* __restrict__ Di, bf16* __restrict__ dqkv, int m, int d, int nh, float sl2,
    float scale) {
  extern __shared__ __align__(128) uint8_t sm[];  // 6 tiles of 8 KB
  __shared__ float sL[2][AT], sD[2][AT];
  const uint32_t sK = smem_u32(sm), sV = sK + 8192, sQ0 = sK + 2 * 8192, sO0 = sK + 4 * 8192;
  const int b = blockIdx.z, h = blockIdx.y, k0 = blockIdx.x * AT;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
  const long ld = 3L * d, rb = (long)b * m;
  const int qc = h * AT, kc_ = d + h * AT, vc = 2 * d + h * AT;
  const float* lse_bh = lse + ((long)b * nh + h) * m;
  const float* D_bh = Di + ((long)b * nh + h) * m;
  const int qt0 = CAUSAL ? k0 / AT : 0, n_qt = (m + AT - 1) / AT;

  load_tile(sK, qkv, rb, k0, m, ld, kc_);
  load_tile(sV, qkv, rb, k0, m, ld, vc);
  cp_commit();
  auto load_q = [&](int qt, int buf) {
    load_tile(sQ0 + buf * 8192, qkv, rb, qt * AT, m, ld, qc);
    load_tile(sO0 + buf * 8192, dO, rb, qt * AT, m, (long)d, h * AT);
    if (threadIdx.x < AT) {
      const int q = qt * AT + threadIdx.x;
      sL[buf][threadIdx.x] = q < m ? lse_bh[q] : 0.f;
      sD[buf][threadIdx.x] = q < m ? D_bh[q] : 0.f;
    }
  };
  load_q(qt0, 0);
  cp_commit();

  uint32_t kf[4][4], vf[4][4];
  float dk[8][4] = {}, dv[8][4] = {};
  const int key0 = k0 + w * 16 + g;

  for (int qt = qt0; qt < n_qt; ++qt) {
    const int buf = (qt - qt0) & 1;
    if (qt + 1 < n_qt) {
      load_q(qt + 1, buf ^ 1);
      cp_commit();
      cp_wait<1>();
    } else {
      cp_wait<0>();
    }
    __syncthreads();
    if (qt == qt0) {
      load_afrag(kf, sK, w);
      load_afrag(vf, sV, w);
    }
    const uint32_t sQ = sQ0 + buf * 8192, sO = sO0 + buf * 8192;
    float p[8][4] = {};
    mma_abt(p, kf, sQ);  // S^T = K Q^T (16 keys x 64 queries)
#pragma unroll
    for (int nt = 0; nt < 8; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int ql = nt * 8 + 2 * t + (e & 1);
        const int q = qt * AT + ql;
        const int key = key0 + (e >> 1) * 8;
        const bool ok = q < m && key < m && (!CAUSAL || q >= key);
        p[nt][e] = ok ? exp2f(p[nt][e] * sl2 - sL[buf][ql]) : 0.f;
      }
    mma_pt(dv, p, sO);   // dV += P^T dO
    float dp[8][4] = {};
    mma_abt(dp, vf, sO);  // dP^T = V dO^T
#pragma unroll
    for (int nt = 0; nt < 8; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int ql = nt * 8 + 2 * t + (e & 1);
        dp[nt][e] = p[nt][e] * (dp[nt][e] - sD[buf][ql]);
      }
    mma_pt(dk, dp, sQ);  // dK += dS^T Q
    __syncthreads();
  }
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const int key = key0 + r * 8;
    if (key >= m) continue;
    bf16* kp = dqkv + (rb + key) * ld + kc_ + 2 * t;
    bf16* vp = dqkv + (rb + key) * ld + vc + 2 * t;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      *reinterpret_cast<uint32_t*>(kp + nt * 8) =
          pack_bf16(dk[nt][2 * r] * scale, dk[nt][2 * r + 1] * scale);
      *reinterpret_cast<uint32_t*>(vp + nt * 8) = pack_bf16(dv[nt][2 * r], dv[nt][2 * r + 1]);
    }
  }
}

// dQ for one 64-query tile, looping over key tiles.
template <bool CAUSAL>
__global__ void __launch_bounds__(128) attn_bwd_dq_kernel(
    const bf16* __restrict__ qkv, const bf16* __restrict__ dO, const float* __restrict__ lse,
    const float* __restrict__ Di, bf16* __restrict__ dqkv, int m, int d, int nh, float sl2,
    float scale) {
  extern __shared__ __align__(128) uint8_t sm[];  // 6 tiles of 8 KB
  const uint32_t sQ = smem_u32(sm), sO = sQ + 8192, sK0 = sQ + 2 * 8192, sV0 = sQ + 4 * 8192;
  const int b = blockIdx.z, h = blockIdx.y, q0 = blockIdx.x * AT;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
  const long ld = 3L * d, rb = (long)b * m;
  const int qc = h * AT, kc_ = d + h * AT, vc = 2 * d + h * AT;
  const int n_kt = CAUSAL ? (min(q0 + AT, m) + AT - 1) / AT : (m + AT - 1) / AT;
  const float* lse_bh = lse + ((long)b * nh + h) * m;
  const float* D_bh = Di + ((long)b * nh + h) * m;

  load_tile(sQ, qkv, rb, q0, m, ld, qc);
  load_tile(sO, dO, rb, q0, m, (long)d, h * AT);
  cp_commit();
  load_tile(sK0, qkv, rb, 0, m, ld, kc_);
  load_tile(sV0, qkv, rb, 0, m, ld, vc);
  cp_commit();

  const int qrow0 = q0 + w * 16 + g;
  float lrow[2], drow[2];
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const int q = qrow0 + r * 8;
    lrow[r] = q < m ? lse_bh[q] : 0.f;
    drow[r] = q < m ? D_bh[q] : 0.f;
  }
  uint32_t qf[4][4], of[4][4];
  float dq[8][4] = {};
  for (int kt = 0; kt < n_kt; ++kt) {
    const int buf = kt & 1;
    if (kt + 1 < n_kt) {
      load_tile(sK0 + (buf ^ 1) * 8192, qkv, rb, (kt + 1) * AT, m, ld, kc_);
      load_tile(sV0 + (buf ^ 1) * 8192, qkv, rb, (kt + 1) * AT, m, ld, vc);
      cp_commit();
      cp_wait<1>();
    } else {
      cp_wait<0>();
    }
    __syncthreads();
    if (kt == 0) {
      load_afrag(qf, sQ, w);
      load_afrag(of, sO, w);
    }
    float p[8][4] = {};
    mma_abt(p, qf, sK0 + buf * 8192);
#pragma unroll
    for (int nt = 0; nt < 8; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = kt * AT + nt * 8 + 2 * t + (e & 1);
        const int q = qrow0 + (e >> 1) * 8;
        const bool ok = q < m && key < m && (!CAUSAL || key <= q);
        p[nt][e] = ok ? exp2f(p[nt][e] * sl2 - lrow[e >> 1]) : 0.f;
      }
    float dp[8][4] = {};
    mma_abt(dp, of, sV0 + buf * 8192);  // dP = dO V^T
#pragma unroll
    for (int nt = 0; nt < 8; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) dp[nt][e] = p[nt][e] * (dp[nt][e] - drow[e >> 1]);
    mma_pt(dq, dp, sK0 + buf * 8192);  // dQ += dS K
    __syncthreads();
  }
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const int q = qrow0 + r * 8;
    if (q >= m) continue;
    bf16* qp = dqkv + (rb + q) * ld + qc + 2 * t;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt)
      *reinterpret_cast<uint32_t*>(qp + nt * 8) =
          pack_bf16(dq[nt][2 * r] * scale, dq[nt][2 * r + 1] * scale);
  }
}

}  // namespace

int take_dev_error_attention() { return take_dev_error_tu(); }

cudaError_t attn_bwd(const bf16* qkv, const bf16* O, const bf16* dO, const float* lse, float* Di,
                     bf16* dqkv, int B, int m, int d, int nh, bool causal, cudaStream_t st) {
  const float scale = 1.0f / sqrtf((float)AT);
  const float sl2 = scale * 1.4426950408889634f;
  const long warps = (long)B * m * nh;
  const double pairs = (double)B * nh * (causal ? 0.5 * m * (m + 1.0) : (double)m * m);
  {
    LaunchTimer lt("attn_bwd_dot", st, 2.0 * B * m * d, 4.0 * B * m * d + 4.0 * B * nh * m);
    attn_bwd_dot_kernel<<<(unsigned)((warps * 32 + 255) / 256), 256, 0, st>>>(dO, O, Di, B * m, m,
                                                                              d, nh);
  }
  constexpr int SMEM = 6 * AT * AT * 2;
  dim3 grid((m + AT - 1) / AT, nh, B);
  auto k1 = causal ? attn_bwd_dkdv_kernel<true> : attn_bwd_dkdv_kernel<false>;
  auto k2 = causal ? attn_bwd_dq_kernel<true> : attn_bwd_dq_kernel<false>;
  cudaFuncSetAttribute(k1, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM);
  cudaFuncSetAttribute(k2, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM);
  {
    LaunchTimer lt("attn_bwd_dkdv", st, 4.0 * AT * pairs, 2.0 * B * m * (5.0 * d));
    k1<<<grid, 128, SMEM, st>>>(qkv, dO, lse, Di, dqkv, m, d, nh, sl2, scale);
  }
  {
    LaunchTimer lt("attn_bwd_dq", st, 4.0 * AT * pairs, 2.0 * B * m * (5.0 * d));
    k2<<<grid, 128, SMEM, st>>>(qkv, dO, lse, Di, dqkv, m, d, nh, sl2, scale);
  }
  return cudaGetLastError();
}

}  // namespace pf
