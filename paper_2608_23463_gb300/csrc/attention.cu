// Proxy-space multi-head attention (Eq. proxy-attn): host entry of the
// backward and the Di = rowsum(dO * O) kernel it starts with.
//
// Q, K, V live in one [B*m, 3d] bf16 matrix (columns [Q | K | V], head h at
// h*64 inside each third); the attention output A is [B*m, d].  The forward
// (attention_tc.cu) saves LSE (log2 units) per (b, h, query); the backward
// (attention_bwd_tc.cu) recomputes the probabilities from LSE and Di in two
// deterministic tcgen05 kernels, one for dK / dV and one for dQ.
#include "kernels.h"

namespace pf {

namespace {

constexpr int AT = 64;  // head width

// Di = rowsum(dO * O) per (b, h, query): eight lanes per (row, head), each
// eight of the head's 64 columns with 16-byte loads.
__global__ void attn_bwd_dot_kernel(const bf16* __restrict__ dO, const bf16* __restrict__ O,
                                    float* __restrict__ Dout, int rows, int m, int d, int nh) {
  const long gid = ((long)blockIdx.x * blockDim.x + threadIdx.x) >> 3;
  const int sub = threadIdx.x & 7;
  const long items = (long)rows * nh;
  const bool live = gid < items;
  const long wid = live ? gid : items - 1;
  const long row = wid / nh;
  const int h = (int)(wid % nh);
  const long off = row * d + h * AT + sub * 8;
  const uint4 gu = *reinterpret_cast<const uint4*>(dO + off);
  const uint4 ou = *reinterpret_cast<const uint4*>(O + off);
  const uint32_t gw[4] = {gu.x, gu.y, gu.z, gu.w}, ow[4] = {ou.x, ou.y, ou.z, ou.w};
  float v = 0.f;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const float2 a = unpack_bf16(gw[k]), c = unpack_bf16(ow[k]);
    v = fmaf(a.x, c.x, v);
    v = fmaf(a.y, c.y, v);
  }
#pragma unroll
  for (int s = 4; s > 0; s >>= 1) v += __shfl_xor_sync(0xffffffffu, v, s);
  if (live && sub == 0) {
    const long b = row / m, i = row % m;
    Dout[(b * nh + h) * m + i] = v;
  }
}

// Gate of the cross injection, backward: eight lanes per (token row, head),
// each lane eight of the head's 64 columns with 16-byte loads and stores, so
// a warp covers four items per instruction (one item per warp, with 4-byte
// loads, left too few bytes in flight to stream at HBM speed).
__global__ void cross_gate_bwd_kernel(const bf16* __restrict__ dAg, const bf16* __restrict__ A,
                                      const bf16* __restrict__ qa, long ldq,
                                      const float* __restrict__ b_a, bf16* __restrict__ dO,
                                      float* __restrict__ Di, bf16* __restrict__ dqa,
                                      float* __restrict__ ga, int ldga, long rows, int L, int d,
                                      int nh) {
  const long gid = ((long)blockIdx.x * blockDim.x + threadIdx.x) >> 3;  // item
  const int sub = threadIdx.x & 7;                                      // lane in the item
  const long items = rows * nh;
  const bool live = gid < items;
  const long wid = live ? gid : items - 1;
  const long row = wid / nh;
  const int h = (int)(wid % nh);
  const long off = row * d + h * AT + sub * 8;
  const uint4 gu = *reinterpret_cast<const uint4*>(dAg + off);
  const uint4 au = *reinterpret_cast<const uint4*>(A + off);
  const float x = __bfloat162float(qa[row * ldq + d + h]) + b_a[h];
  const uint32_t gw[4] = {gu.x, gu.y, gu.z, gu.w}, aw[4] = {au.x, au.y, au.z, au.w};
  float sum = 0.f;
  float2 g2[4];
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    g2[k] = unpack_bf16(gw[k]);
    const float2 a2 = unpack_bf16(aw[k]);
    sum = fmaf(g2[k].x, a2.x, sum);
    sum = fmaf(g2[k].y, a2.y, sum);
  }
#pragma unroll
  for (int s = 4; s > 0; s >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, s);
  if (!live) return;
  const float al = 1.f / (1.f + __expf(-x));
  *reinterpret_cast<uint4*>(dO + off) =
      make_uint4(pack_bf16(al * g2[0].x, al * g2[0].y), pack_bf16(al * g2[1].x, al * g2[1].y),
                 pack_bf16(al * g2[2].x, al * g2[2].y), pack_bf16(al * g2[3].x, al * g2[3].y));
  if (sub == 0) {
    const long b = row / L, t = row % L;
    Di[(b * nh + h) * L + t] = al * sum;
    const float gp = sum * al * (1.f - al);
    dqa[row * ldq + d + h] = __float2bfloat16(gp);
    ga[row * ldga + h] = gp;
  }
  if (h == 0) {  // the padding columns past the gate rows stay zero
    for (long c = d + nh + sub; c < ldq; c += 8) dqa[row * ldq + c] = __float2bfloat16(0.f);
    for (int c = nh + sub; c < ldga; c += 8) ga[row * ldga + c] = 0.f;
  }
}

}  // namespace

cudaError_t cross_gate_bwd(const bf16* dAg, const bf16* A, const bf16* qa, long ldq,
                           const float* b_a, bf16* dO, float* Di, bf16* dqa, float* ga, int ldga,
                           int B, int L, int d, int nh, cudaStream_t st) {
  if (d != nh * AT || ldq < d + nh || ldga < nh) return cudaErrorInvalidValue;
  const long rows = (long)B * L, warps = rows * nh;
  LaunchTimer lt("cross_gate_bwd", st, 4.0 * rows * d,
                 6.0 * rows * d + 2.0 * rows * ldq / 8.0 + 8.0 * rows * nh);
  if (((uintptr_t)dAg | (uintptr_t)A | (uintptr_t)dO) & 15) return cudaErrorInvalidValue;
  cross_gate_bwd_kernel<<<(unsigned)((warps * 8 + 255) / 256), 256, 0, st>>>(
      dAg, A, qa, ldq, b_a, dO, Di, dqa, ga, ldga, rows, L, d, nh);
  return cudaGetLastError();
}

int take_dev_error_attention() { return take_dev_error_tu(); }
int set_wait_limit_attention(unsigned long long ns) { return set_wait_limit_tu(ns); }

cudaError_t attn_bwd(const bf16* qkv, const bf16* O, const bf16* dO, const float* lse, float* Di,
                     bf16* dqkv, int B, int m, int d, int nh, bool causal, cudaStream_t st) {
  const long warps = (long)B * m * nh;
  {
    LaunchTimer lt("attn_bwd_dot", st, 2.0 * B * m * d, 4.0 * B * m * d + 4.0 * B * nh * m);
    if (((uintptr_t)dO | (uintptr_t)O) & 15) return cudaErrorInvalidValue;
    attn_bwd_dot_kernel<<<(unsigned)((warps * 8 + 255) / 256), 256, 0, st>>>(dO, O, Di, B * m, m,
                                                                             d, nh);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  return attn_bwd_tc(qkv, dO, lse, Di, dqkv, B, m, d, nh, causal, st);
}

}  // namespace pf
