// tcgen05 / TMEM / TMA GEMM for sm_103a with fused epilogues.
//
//   D[M, N] = sum_k A[m, k] * B[n, k]     (bf16 operands, fp32 accumulation)
//
// A is K-major (stored [M, K]) or MN-major (stored [K, M]); likewise B ([N, K]
// or [K, N]).  Every contraction of the layer (compression, proxy Q/K/V/O,
// decompression, and all of their weight / input gradients) is one of these.
//
// One CTA computes one 128 x BN output tile:
//   warp 0   : TMA producer (one elected thread), STAGES-deep smem ring of
//              128B-swizzled 64-wide K slices of A and B
//   warp 1   : TMEM allocator + MMA issuer (one thread issues tcgen05.mma
//              M=128, N=BN, K=16; tcgen05.commit frees smem stages)
//   warps 2-5: epilogue: tcgen05.ld 32 columns at a time from the TMEM
//              accumulator (warp w reads TMEM lanes 32*(w%4)..), applies the
//              fused epilogue functor and writes global memory.
// Every mbarrier wait is bounded (common.cuh); on a timeout the kernel flags
// the error, drains its own copies and MMAs (bounded), frees TMEM and returns.
#pragma once

#include "common.cuh"

namespace pf {

constexpr int GEMM_BM = 128;
constexpr int GEMM_BK = 64;
constexpr int GEMM_THREADS = 192;

template <int BN>
struct GemmCfg {
  static constexpr int STAGES = (BN == 256) ? 4 : 6;
  static constexpr uint32_t A_BYTES = GEMM_BM * GEMM_BK * 2;  // 16 KB
  static constexpr uint32_t B_BYTES = BN * GEMM_BK * 2;       // 16/32 KB
  static constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr uint32_t SMEM_BYTES = STAGES * STAGE_BYTES + 1024 /*align*/ + 256 /*bars*/;
};

// Optional remap of the B tile's rows (K-major B only): B tile `n_tile` is
// loaded as BN/128 boxes of 128 rows; box j starts at row brow(n_tile, j).
struct BRowsLinear {
  __device__ __forceinline__ int operator()(int n_tile, int j, int BN) const {
    return n_tile * BN + j * 128;
  }
};

template <int BN, bool A_MN, bool B_MN, class Epi, class BRows = BRowsLinear>
__global__ void __launch_bounds__(GEMM_THREADS, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   int M, int N, int K, Epi epi, BRows brows) {
  using Cfg = GemmCfg<BN>;
  constexpr int STAGES = Cfg::STAGES;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * Cfg::STAGE_BYTES);
  // bars[0..S): full, bars[S..2S): empty, bars[2S]: done
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * STAGES + 1);
  __shared__ int s_consumed;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_tile = blockIdx.x, m_tile = blockIdx.y;
  const int m0 = m_tile * GEMM_BM, n0 = n_tile * BN;
  const int num_k = (K + GEMM_BK - 1) / GEMM_BK;
  const uint32_t full0 = smem_u32(bars), empty0 = smem_u32(bars + STAGES),
                 done = smem_u32(bars + 2 * STAGES);

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    mbar_init(done, 1);
    fence_barrier_init();
    s_consumed = 0;
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), BN);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  int issued = 0;

  if (warp == 0 && lane == 0) {
    // ---------------------------------------------------------- producer
    prefetch_tmap(&tmA);
    prefetch_tmap(&tmB);
    for (int kt = 0; kt < num_k; ++kt) {
      const int s = kt % STAGES;
      const uint32_t ph = (kt / STAGES) & 1;
      if (!mbar_wait(empty0 + 8 * s, ph ^ 1)) break;
      const uint32_t fb = full0 + 8 * s;
      mbar_arrive_expect_tx(fb, Cfg::STAGE_BYTES);
      const uint32_t a_dst = smem_u32(smem + s * Cfg::STAGE_BYTES);
      const uint32_t b_dst = a_dst + Cfg::A_BYTES;
      const int k0 = kt * GEMM_BK;
      if (!A_MN) {
        tma_load_2d(a_dst, &tmA, fb, k0, m0);
      } else {
        tma_load_2d(a_dst, &tmA, fb, m0, k0);
        tma_load_2d(a_dst + 8192, &tmA, fb, m0 + 64, k0);
      }
      if (!B_MN) {
#pragma unroll
        for (int j = 0; j < BN / 128; ++j) tma_load_2d(b_dst + j * 16384, &tmB, fb, k0, brows(n_tile, j, BN));
      } else {
#pragma unroll
        for (int j = 0; j < BN / 64; ++j) tma_load_2d(b_dst + j * 8192, &tmB, fb, n0 + 64 * j, k0);
      }
      issued = kt + 1;
    }
  } else if (warp == 1 && lane == 0) {
    // ---------------------------------------------------------- MMA issuer
    constexpr uint32_t idesc = idesc_bf16_f32(GEMM_BM, BN, A_MN ? 1 : 0, B_MN ? 1 : 0);
    int kt = 0;
    for (; kt < num_k; ++kt) {
      const int s = kt % STAGES;
      const uint32_t ph = (kt / STAGES) & 1;
      if (!mbar_wait(full0 + 8 * s, ph)) break;
      tc_fence_after();
      const uint32_t a_base = smem_u32(smem + s * Cfg::STAGE_BYTES);
      const uint32_t b_base = a_base + Cfg::A_BYTES;
#pragma unroll
      for (int kk = 0; kk < GEMM_BK / 16; ++kk) {
        // K-major: 16 K-elements = 32 bytes along the swizzled 128-byte row,
        //          8-row groups 1024 bytes apart (SBO).
        // MN-major: 16 K-rows = 2048 bytes; 64-wide MN slabs 8192 bytes apart
        //          (LBO), 8-row K groups 1024 bytes apart (SBO).
        const uint64_t ad = A_MN ? smem_desc_sw128(a_base + kk * 2048, 8192, 1024)
                                 : smem_desc_sw128(a_base + kk * 32, 16, 1024);
        const uint64_t bd = B_MN ? smem_desc_sw128(b_base + kk * 2048, 8192, 1024)
                                 : smem_desc_sw128(b_base + kk * 32, 16, 1024);
        tc_mma_f16(tmem, ad, bd, idesc, (kt | kk) != 0 ? 1u : 0u);
      }
      tc_commit(empty0 + 8 * s);
    }
    s_consumed = kt;
    tc_commit(done);
  } else if (warp >= 2) {
    // ---------------------------------------------------------- epilogue
    mbar_wait(done, 0);
    tc_fence_after();
    const int q = warp & 3;
    const int row = m0 + q * 32 + lane;
#pragma unroll 1
    for (int c = 0; c < BN; c += 32) {
      float v[32];
      tmem_ld32(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)c, v);
      if (num_k == 0) {
#pragma unroll
        for (int i = 0; i < 32; ++i) v[i] = 0.f;
      }
      epi.apply(row, n0 + c, v);
    }
  }
  tc_fence_before();
  if (__syncthreads_or(*(volatile int*)&g_dev_error != 0)) {
    // error path: let in-flight TMA copies and MMAs land before TMEM/smem go.
    if (warp == 0 && lane == 0) {
      for (int kt = s_consumed; kt < issued; ++kt)
        mbar_wait(full0 + 8 * (kt % STAGES), (kt / STAGES) & 1);
    }
    if (warp == 1 && lane == 0) mbar_wait(done, 0);
    __syncthreads();
  }
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, BN);
  }
}

// ------------------------------------------------------------------ epilogues
// Each epilogue's apply(row, col, v) receives 32 consecutive accumulator
// columns [col, col+32) of output row `row` (N is a multiple of 32).

// v = acc (+ bias[col]) (+ addend[row, col]); stored as fp32 and/or bf16.
struct EpiLinear {
  int M, N;
  const float* bias;
  const float* addend;
  long ld_add;
  float* out_f32;
  long ld_f32;
  bf16* out_bf16;
  long ld_bf16;
  __device__ __forceinline__ void apply(int row, int col, float* v) const {
    if (row >= M || col >= N) return;
    if (bias) {
#pragma unroll
      for (int i = 0; i < 32; i += 4) {
        float4 b = *reinterpret_cast<const float4*>(bias + col + i);
        v[i] += b.x; v[i + 1] += b.y; v[i + 2] += b.z; v[i + 3] += b.w;
      }
    }
    if (addend) {
      const float* a = addend + (long)row * ld_add + col;
#pragma unroll
      for (int i = 0; i < 32; i += 4) {
        float4 b = *reinterpret_cast<const float4*>(a + i);
        v[i] += b.x; v[i + 1] += b.y; v[i + 2] += b.z; v[i + 3] += b.w;
      }
    }
    if (out_f32) {
      float* o = out_f32 + (long)row * ld_f32 + col;
#pragma unroll
      for (int i = 0; i < 32; i += 4)
        *reinterpret_cast<float4*>(o + i) = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
    }
    if (out_bf16) {
      bf16* o = out_bf16 + (long)row * ld_bf16 + col;
#pragma unroll
      for (int i = 0; i < 32; i += 8) store8_bf16(o + i, v + i);
    }
  }
};

// Last decompression level of a 1D layer fused with routing and injection.
// GEMM rows are proxy-order rows r = (b*m + i)*k2 + a (proxy i of sequence b,
// level-1 row a); columns c in [0, k1*d) are (token c/d of the k1-group,
// channel c%d).  D = acc + b_d1 is saved in that layout; it is injected into
// block i + shift (shift = 1: causal routing, 0: bidirectional) at token
// (i+shift)*P + a*k1 + c/d:
//   gated: X_out = X + sigmoid(w_x X + w_dlt D + b_g) D    (Eq. inj-gate)
//   add:   X_out = X + D                                    (Eq. inj-add)
struct EpiInject1D {
  int M, N;
  const float* bias;
  bf16* D_save;
  const bf16* X;
  bf16* X_out;
  const float *w_x, *w_dlt, *b_g;
  int d, k1, k2, m, L, shift, gated;
  __device__ __forceinline__ void apply(int row, int col, float* v) const {
    if (row >= M || col >= N) return;
#pragma unroll
    for (int i = 0; i < 32; i += 4) {
      float4 b = *reinterpret_cast<const float4*>(bias + col + i);
      v[i] += b.x; v[i + 1] += b.y; v[i + 2] += b.z; v[i + 3] += b.w;
    }
    if (D_save) {
      bf16* o = D_save + (long)row * N + col;
#pragma unroll
      for (int i = 0; i < 32; i += 8) store8_bf16(o + i, v + i);
    }
    const int a = row % k2, prox = row / k2;
    const int b = prox / m, i = prox % m;
    const int it = i + shift;
    if (it >= m) return;
    const long tok = (long)it * (k1 * k2) + (long)a * k1 + col / d;
    if (tok >= L) return;
    const int ch = col % d;
    const long off = ((long)b * L + tok) * d + ch;
#pragma unroll
    for (int i8 = 0; i8 < 32; i8 += 8) {
      float x[8], o[8];
      load8_bf16(X + off + i8, x);
      if (gated) {
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const int c = ch + i8 + j;
          const float g = w_x[c] * x[j] + w_dlt[c] * v[i8 + j] + b_g[c];
          o[j] = x[j] + sigmoidf_(g) * v[i8 + j];
        }
      } else {
#pragma unroll
        for (int j = 0; j < 8; ++j) o[j] = x[j] + v[i8 + j];
      }
      store8_bf16(X_out + off + i8, o);
    }
  }
};

// First compression level's input gradient, accumulated onto the direct
// injection gradient already held in dX: rows r = (b*m + i)*k2 + a, columns
// (token c/d of the group, channel c%d) -> token i*P + a*k1 + c/d of sequence b.
struct EpiDX1D {
  int M, N;
  bf16* dX;
  int d, k1, k2, m, L;
  __device__ __forceinline__ void apply(int row, int col, float* v) const {
    if (row >= M || col >= N) return;
    const int per_seq = m * k2;
    const int b = row / per_seq, rr = row % per_seq;
    const long tok = (long)rr * k1 + col / d;
    if (tok >= L) return;
    const long off = ((long)b * L + tok) * d + (col % d);
#pragma unroll
    for (int i8 = 0; i8 < 32; i8 += 8) {
      float x[8];
      load8_bf16(dX + off + i8, x);
#pragma unroll
      for (int j = 0; j < 8; ++j) x[j] += v[i8 + j];
      store8_bf16(dX + off + i8, x);
    }
  }
};

}  // namespace pf
