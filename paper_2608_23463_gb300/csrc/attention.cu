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

}  // namespace

int take_dev_error_attention() { return take_dev_error_tu(); }

cudaError_t attn_bwd(const bf16* qkv, const bf16* O, const bf16* dO, const float* lse, float* Di,
                     bf16* dqkv, int B, int m, int d, int nh, bool causal, cudaStream_t st) {
  const long warps = (long)B * m * nh;
  {
    LaunchTimer lt("attn_bwd_dot", st, 2.0 * B * m * d, 4.0 * B * m * d + 4.0 * B * nh * m);
    attn_bwd_dot_kernel<<<(unsigned)((warps * 32 + 255) / 256), 256, 0, st>>>(dO, O, Di, B * m, m,
                                                                              d, nh);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  return attn_bwd_tc(qkv, dO, lse, Di, dqkv, B, m, d, nh, causal, st);
}

}  // namespace pf
