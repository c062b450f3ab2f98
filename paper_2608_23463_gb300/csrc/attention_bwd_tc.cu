// Backward of the proxy-space attention (Eq. proxy-attn) on the tcgen05
// tensor cores, head width 64.  With P = softmax(Q K^T / 8) recomputed from
// the saved LSE and Di = rowsum(dO * O):
//   dP = dO V^T,   dS = P * (dP - Di),   dV = P^T dO,   dK = dS^T Q / 8,
//   dQ = dS K / 8.
// Two kernels share one skeleton (no atomics, deterministic):
//   DKDV: item = (128-key tile, head, sequence); stationary X1 = K, X2 = V;
//         streamed 64-query tiles Y1 = Q_j, Y2 = dO_j.
//           T1 = X1 Y1^T = S^T,  T2 = X2 Y2^T = dP^T     (TMEM, M=128 N=64)
//           E1 = P^T, E2 = dS^T  (bf16, written to TMEM by the row warps)
//           dV += E1 Y2,  dK += E2 Y1    (A from TMEM; TMEM accumulators)
//   DQ:   item = (128-query tile, head, sequence); stationary X1 = Q, X2 = dO;
//         streamed 64-key tiles Y1 = K_j, Y2 = V_j.
//           T1 = S,  T2 = dP,  E2 = dS,  dQ += E2 Y1
// Roles: warp 0 TMA producer (DKDV: it also stages each step's (LSE, Di)
// pairs of the streamed queries in shared memory), warp 1 MMA issuer, warps
// 2-9 the row warps: two per TMEM lane quarter, each thread one row (TMEM
// lane) and one half of the 64 streamed columns.  T1/T2 and E are double-buffered so the MMAs of step
// j+1 overlap the row work of step j.  E stays in TMEM as the A operand of the
// accumulating MMAs, so those read only their B tile from shared memory
// (shared-memory bandwidth, not the tensor pipe, bounds M=128 N=64 MMAs whose
// operands both come from shared memory).  Every wait is bounded.
//
// The cross-attention of the injection (Eq. inj-cross) runs on the same
// kernels: queries are tokens, keys / values proxies (separate matrices, Lq
// and Lk rows per sequence), and token q sees proxies j < q / P (causal) or
// all.  Stationary tiles that no pair reaches are not work items; the host
// zero-fills their output rows.
#include <algorithm>
#include <type_traits>

#include "kernels.h"

namespace pf {

namespace {

constexpr int BW_M = 128;  // stationary rows (TMEM lanes)
constexpr int BW_N = 64;   // streamed rows per step
constexpr int BW_D = 64;   // head width
constexpr int BW_STAGES = 4;
constexpr int BW_ROW_THREADS = 256;  // warps 2-9
constexpr int BW_THREADS = 64 + BW_ROW_THREADS;
constexpr uint32_t BW_X_BYTES = BW_M * BW_D * 2;  // 16 KB per stationary tile
constexpr uint32_t BW_Y_BYTES = BW_N * BW_D * 2;  // 8 KB per streamed tile
constexpr uint32_t BW_OFF_Y = 2 * 2 * BW_X_BYTES;                       // X: [2 bufs][X1, X2]
constexpr uint32_t BW_OFF_LD = BW_OFF_Y + BW_STAGES * 2 * BW_Y_BYTES;  // Y: [stage][Y1, Y2]
constexpr uint32_t BW_OFF_BAR = BW_OFF_LD + BW_STAGES * BW_N * 8;      // (lse, Di) [stage][64]
constexpr uint32_t BW_SMEM = BW_OFF_BAR + 256 + 1024;
// TMEM columns: T1 at 0 / 64, T2 at 128 / 192 (fp32, per buffer), accumulators
// at 256 (dV or dQ) and 320 (dK), E at 384 / 448 (per buffer: E1 at +0, E2 at
// +32, bf16 pairs: streamed column c in 32-bit column c / 2)
constexpr uint32_t BW_TMEM_COLS = 512;
constexpr uint32_t BW_TM_E = 384;

struct BwArgs {
  // outputs, head h of stationary row (b, r) at out + (b*Lx + r)*ld + col + 64h:
  // DKDV u = dV, w = dK; DQ u = dQ
  bf16 *out_u, *out_w;
  long ld_u, ld_w;
  int col_u, col_w;
  const float* lse;   // [B, nh, Lq], log2 units
  const float* Di;    // [B, nh, Lq]
  int B, Lq, Lk, d, nh, causal, P;  // P > 0: cross-attention with block size P
  int Lx, Ly;         // stationary / streamed rows per sequence
  int n_tiles, n_steps_total, n_items;
  float sl2, scale;
};

// Keys visible to query q (all, causal prefix, or the proxies of earlier
// blocks), and the first query that sees key k.
__host__ __device__ __forceinline__ int bw_vis(const BwArgs& a, int q) {
  const int v = !a.causal ? a.Lk : a.P ? q / a.P : q + 1;
  return v < a.Lk ? v : a.Lk;
}
__host__ __device__ __forceinline__ int bw_first_q(const BwArgs& a, int k) {
  return !a.causal ? 0 : a.P ? (k + 1) * a.P : k;
}

__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Snake order over the CTAs of items ranked heaviest first.
__device__ __forceinline__ int bw_rank(int c, int round) {
  return round * (int)gridDim.x + ((round & 1) ? (int)gridDim.x - 1 - c : c);
}

// Item k -> stationary tile t (128 rows), head, sequence, first streamed tile
// j0 and step count n.  DKDV: the keys of tile t are seen by the queries from
// bw_first_q on, so the heaviest items have the smallest t; DQ: the largest t.
// The host sizes n_items so that every item has n >= 1.
template <bool DKDV>
__device__ __forceinline__ void bw_item(const BwArgs& a, int k, int& t, int& h, int& b, int& j0,
                                        int& n) {
  const int per = a.nh * a.B;
  const int rnk = k / per, r = k % per;
  h = r % a.nh;
  b = r / a.nh;
  if (DKDV) {
    t = rnk;
    j0 = bw_first_q(a, t * BW_M) / BW_N;
    n = a.n_steps_total - j0;
  } else {
    t = a.n_tiles - 1 - rnk;
    j0 = 0;
    n = min((bw_vis(a, min(t * BW_M + BW_M - 1, a.Lq - 1)) + BW_N - 1) / BW_N, a.n_steps_total);
  }
}

template <bool DKDV>
__global__ void __launch_bounds__(BW_THREADS, 1)
    attn_bwd_tc_kernel(const __grid_constant__ CUtensorMap tmX1, const __grid_constant__ CUtensorMap tmX2,
                       const __grid_constant__ CUtensorMap tmY1, const __grid_constant__ CUtensorMap tmY2,
                       int x1c, int x2c, int y1c, int y2c, BwArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  const uint32_t b0 = smem_u32(smem + BW_OFF_BAR);
  // x_full[2] x_empty[2] y_full[S] y_empty[S] t_full[2] t_free[2] e_full[2] e_free[2]
  // acc_full acc_free done
  const uint32_t x_full = b0, x_empty = b0 + 16, y_full = b0 + 32,
                 y_empty = y_full + 8 * BW_STAGES, t_full = y_empty + 8 * BW_STAGES,
                 t_free = t_full + 16, e_full = t_free + 16, e_free = e_full + 16,
                 acc_full = e_free + 16, acc_free = acc_full + 8, done = acc_free + 8;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + BW_OFF_BAR + 240);
  const uint32_t sbase = smem_u32(smem);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(x_full + 8 * i, 1);
      mbar_init(x_empty + 8 * i, 1);
      mbar_init(t_full + 8 * i, 1);
      mbar_init(t_free + 8 * i, BW_ROW_THREADS / 32);  // one arrival per row warp
      mbar_init(e_full + 8 * i, BW_ROW_THREADS / 32);
      mbar_init(e_free + 8 * i, 1);
    }
    for (int i = 0; i < BW_STAGES; ++i) {
      mbar_init(y_full + 8 * i, 1);
      mbar_init(y_empty + 8 * i, 1);
    }
    mbar_init(acc_full, 1);
    mbar_init(acc_free, BW_ROW_THREADS / 32);
    mbar_init(done, 1);
    fence_barrier_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), BW_TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  uint32_t y_issued = 0, x_issued = 0;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    // Lane 0 issues the copies.  DKDV: the whole warp also stages the (lse,
    // Di) pairs of each step's 64 streamed queries in the stage's slot before
    // lane 0 arms the stage's full barrier, so that the row warps read them
    // after that barrier (the values for the next step are loaded one step
    // ahead, two queries per lane).
    if (lane == 0) {
      prefetch_tmap(&tmX1);
      prefetch_tmap(&tmX2);
      prefetch_tmap(&tmY1);
      prefetch_tmap(&tmY2);
    }
    float2* ld_ring = reinterpret_cast<float2*>(smem + BW_OFF_LD);
    auto fetch_ld = [&](int b, int h, int q0, int c) -> float2 {
      const int qq = q0 + c;
      if (qq >= a.Lq) return make_float2(0.f, 0.f);
      const long o = ((long)b * a.nh + h) * a.Lq + qq;
      return make_float2(a.lse[o], a.Di[o]);
    };
    float2 ld0 = make_float2(0.f, 0.f), ld1 = ld0;  // next step's pairs of queries lane, lane + 32
    int k = bw_rank(blockIdx.x, 0);
    if (DKDV && k < a.n_items) {
      int t, h, b, j0, n;
      bw_item<DKDV>(a, k, t, h, b, j0, n);
      ld0 = fetch_ld(b, h, j0 * BW_N, lane);
      ld1 = fetch_ld(b, h, j0 * BW_N, lane + 32);
    }
    bool ok = true;
    uint32_t it = 0;
    for (int rd = 0; k < a.n_items && ok; k = bw_rank(blockIdx.x, ++rd), ++it) {
      int t, h, b, j0, n;
      bw_item<DKDV>(a, k, t, h, b, j0, n);
      const int row0 = b * a.Lx;
      const uint32_t xb = it & 1;
      if (!mbar_wait_warp(x_empty + 8 * xb, ((it >> 1) & 1) ^ 1)) break;
      if (lane == 0) {
        const uint32_t xdst = sbase + xb * 2 * BW_X_BYTES;
        mbar_arrive_expect_tx(x_full + 8 * xb, 2 * BW_X_BYTES);
        tma_load_2d(xdst, &tmX1, x_full + 8 * xb, x1c + h * BW_D, row0 + t * BW_M);
        tma_load_2d(xdst + BW_X_BYTES, &tmX2, x_full + 8 * xb, x2c + h * BW_D, row0 + t * BW_M);
      }
      x_issued = it + 1;
      for (int j = 0; j < n; ++j) {
        const uint32_t G = y_issued, st = G % BW_STAGES;
        if (!mbar_wait_warp(y_empty + 8 * st, ((G / BW_STAGES) & 1) ^ 1)) {
          ok = false;
          break;
        }
        if (DKDV) {
          ld_ring[st * BW_N + lane] = ld0;
          ld_ring[st * BW_N + 32 + lane] = ld1;
          __syncwarp();
        }
        if (lane == 0) {
          const uint32_t ydst = sbase + BW_OFF_Y + st * 2 * BW_Y_BYTES;
          const int yrow = b * a.Ly + (j0 + j) * BW_N;
          mbar_arrive_expect_tx(y_full + 8 * st, 2 * BW_Y_BYTES);
          tma_load_2d(ydst, &tmY1, y_full + 8 * st, y1c + h * BW_D, yrow);
          tma_load_2d(ydst + BW_Y_BYTES, &tmY2, y_full + 8 * st, y2c + h * BW_D, yrow);
        }
        y_issued = G + 1;
        if (DKDV) {  // the pairs of the next step (this item's or the next item's first)
          if (j + 1 < n) {
            ld0 = fetch_ld(b, h, (j0 + j + 1) * BW_N, lane);
            ld1 = fetch_ld(b, h, (j0 + j + 1) * BW_N, lane + 32);
          } else {
            const int k2 = bw_rank(blockIdx.x, rd + 1);
            if (k2 < a.n_items) {
              int t2, h2, b2, j02, n2;
              bw_item<DKDV>(a, k2, t2, h2, b2, j02, n2);
              ld0 = fetch_ld(b2, h2, j02 * BW_N, lane);
              ld1 = fetch_ld(b2, h2, j02 * BW_N, lane + 32);
            }
          }
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    // The whole warp runs the loop; one elected lane issues and commits.
    constexpr uint32_t idesc_t = idesc_bf16_f32(BW_M, BW_N, 0, 0);
    constexpr uint32_t idesc_a = idesc_bf16_f32(BW_M, BW_D, 0, 1);
    bool ok = true;
    uint32_t it = 0, G = 0;
    // accumulate step G (local step j of its item): E_G times the step's Y tiles
    auto acc_step = [&](uint32_t G_, int j, uint32_t it_) -> bool {
      const uint32_t eb = G_ & 1, st = G_ % BW_STAGES;
      if (!mbar_wait_warp(e_full + 8 * eb, (G_ >> 1) & 1)) return false;
      if (j == 0 && !mbar_wait_warp(acc_free, (it_ & 1) ^ 1)) return false;
      tc_fence_after();
      const uint32_t e1 = tmem + BW_TM_E + eb * 64, e2 = e1 + 32;
      const uint32_t y1 = sbase + BW_OFF_Y + st * 2 * BW_Y_BYTES, y2 = y1 + BW_Y_BYTES;
      if (elect_one()) {
#pragma unroll
        for (int kk = 0; kk < BW_N / 16; ++kk) {
          const uint32_t acc = (j > 0 || kk > 0) ? 1u : 0u;
          const uint64_t bd1 = smem_desc_sw128(y1 + kk * 2048, 8192, 1024);
          if (DKDV) {
            const uint64_t bd2 = smem_desc_sw128(y2 + kk * 2048, 8192, 1024);
            tc_mma_f16_ts(tmem + 256, e1 + kk * 8, bd2, idesc_a, acc);  // dV += P^T dO
            tc_mma_f16_ts(tmem + 320, e2 + kk * 8, bd1, idesc_a, acc);  // dK += dS^T Q
          } else {
            tc_mma_f16_ts(tmem + 256, e2 + kk * 8, bd1, idesc_a, acc);  // dQ += dS K
          }
        }
        tc_commit(e_free + 8 * eb);
        tc_commit(y_empty + 8 * st);
      }
      __syncwarp();
      return true;
    };
    for (int rd = 0, k = bw_rank(blockIdx.x, 0); k < a.n_items && ok;
         k = bw_rank(blockIdx.x, ++rd), ++it) {
      int t, h, b, j0, n;
      bw_item<DKDV>(a, k, t, h, b, j0, n);
      const uint32_t xb = it & 1;
      if (!mbar_wait_warp(x_full + 8 * xb, (it >> 1) & 1)) break;
      tc_fence_after();
      const uint32_t x1 = sbase + xb * 2 * BW_X_BYTES, x2 = x1 + BW_X_BYTES;
      for (int j = 0; j < n; ++j) {
        const uint32_t Gj = G + j, st = Gj % BW_STAGES, tb = Gj & 1;
        if (!mbar_wait_warp(y_full + 8 * st, (Gj / BW_STAGES) & 1) ||
            !mbar_wait_warp(t_free + 8 * tb, ((Gj >> 1) & 1) ^ 1)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t y1 = sbase + BW_OFF_Y + st * 2 * BW_Y_BYTES, y2 = y1 + BW_Y_BYTES;
        if (elect_one()) {
#pragma unroll
          for (int kk = 0; kk < BW_D / 16; ++kk) {
            tc_mma_f16(tmem + tb * BW_N, smem_desc_sw128(x1 + kk * 32, 16, 1024),
                       smem_desc_sw128(y1 + kk * 32, 16, 1024), idesc_t, kk ? 1u : 0u);
            tc_mma_f16(tmem + 128 + tb * BW_N, smem_desc_sw128(x2 + kk * 32, 16, 1024),
                       smem_desc_sw128(y2 + kk * 32, 16, 1024), idesc_t, kk ? 1u : 0u);
          }
          tc_commit(t_full + 8 * tb);
          if (j == n - 1) tc_commit(x_empty + 8 * xb);
        }
        __syncwarp();
        if (j > 0 && !acc_step(Gj - 1, j - 1, it)) {
          ok = false;
          break;
        }
      }
      if (!ok || !acc_step(G + n - 1, n - 1, it)) break;
      if (elect_one()) tc_commit(acc_full);
      __syncwarp();
      G += n;
    }
    if (elect_one()) tc_commit(done);
    __syncwarp();
  } else if (warp >= 2) {
    // ------------------------------------------------------------ row warps
    const int q4 = warp & 3;
    const int r = q4 * 32 + lane;  // stationary row in the tile = TMEM lane
    const int ch = (warp - 2) >> 2;   // half of the streamed columns: [32 ch, 32 ch + 32)
    const uint32_t tl = tmem + ((uint32_t)(q4 * 32) << 16);
    const float2* ld_ring = reinterpret_cast<const float2*>(smem + BW_OFF_LD);  // [stage][64]
    bool ok = true;
    uint32_t G = 0, it = 0;
    for (int rd = 0, k = bw_rank(blockIdx.x, 0); k < a.n_items && ok;
         k = bw_rank(blockIdx.x, ++rd), ++it) {
      int t, h, b, j0, n;
      bw_item<DKDV>(a, k, t, h, b, j0, n);
      const int row = t * BW_M + r;  // key (DKDV) or query (DQ) index in the sequence
      float lse_r = 0.f, di_r = 0.f;
      if (!DKDV && row < a.Lq) {
        const long o = ((long)b * a.nh + h) * a.Lq + row;
        lse_r = a.lse[o];
        di_r = a.Di[o];
      }
      for (int j = 0; j < n; ++j) {
        const uint32_t Gj = G + j, tb = Gj & 1;
        const int c0 = (j0 + j) * BW_N;  // first streamed index of this step
        // DKDV: the step's (lse, Di) pairs, staged by the producer before the
        // stage's full barrier (already complete: the step's scores used it;
        // the slot is refilled only after this step's E has been consumed)
        if (DKDV && !mbar_wait(y_full + 8 * (Gj % BW_STAGES), (Gj / BW_STAGES) & 1)) {
          ok = false;
          break;
        }
        if (!mbar_wait(t_full + 8 * tb, (Gj >> 1) & 1)) {
          ok = false;
          break;
        }
        tc_fence_after();
        uint32_t s1[32], p1[32];
        tmem_ld32_async(tl + tb * BW_N + 32 * ch, s1);
        tmem_ld32_async(tl + 128 + tb * BW_N + 32 * ch, p1);
        tmem_wait_ld(s1);
        tmem_wait_ld(p1);
        tc_fence_before();
        mbar_arrive_warp(t_free + 8 * tb);
        // valid streamed columns: [lo, hi)
        int lo = 0, hi = min(BW_N, a.Ly - c0);
        if (DKDV)
          lo = max(0, bw_first_q(a, row) - c0);  // the queries that see this key
        else
          hi = min(hi, bw_vis(a, row) - c0);  // the keys this query sees
        if (!mbar_wait(e_free + 8 * tb, ((Gj >> 1) & 1) ^ 1)) {
          ok = false;
          break;
        }
        const float2* lds = ld_ring + (Gj % BW_STAGES) * BW_N;
        uint32_t pk[16], dk[16];  // this thread's 32 columns of E1 and E2, bf16 pairs
        // P and dS of this thread's 32 columns; columns outside [lo, hi) are
        // masked (only the diagonal and tail steps have any)
        auto emit = [&](auto masked) {
#pragma unroll
          for (int g = 0; g < 4; ++g) {
            const int kg = 4 * ch + g;  // 8-column group in the 64-wide row
            const uint32_t* sv = s1 + g * 8;
            const uint32_t* dv = p1 + g * 8;
            float pe[8], de[8];
            // DKDV: the group's (lse, Di) with 128-bit shared loads, two columns
            // each (the compiler cannot prove the alignment of the float2 array)
            float l8[8], d8[8];
            if (DKDV) {
              const float4* l4 = reinterpret_cast<const float4*>(lds) + kg * 4;
#pragma unroll
              for (int e2 = 0; e2 < 4; ++e2) {
                const float4 v = l4[e2];
                l8[2 * e2] = v.x;
                d8[2 * e2] = v.y;
                l8[2 * e2 + 1] = v.z;
                d8[2 * e2 + 1] = v.w;
              }
            }
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              const int c = kg * 8 + e;
              const float l2 = DKDV ? l8[e] : lse_r, dd = DKDV ? d8[e] : di_r;
              float p = ex2_approx(fmaf(__uint_as_float(sv[e]), a.sl2, -l2));
              if (decltype(masked)::value && (c < lo || c >= hi)) p = 0.f;
              pe[e] = p;
              de[e] = p * (__uint_as_float(dv[e]) - dd);
            }
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              pk[4 * g + e] = pack_bf16(pe[2 * e], pe[2 * e + 1]);
              dk[4 * g + e] = pack_bf16(de[2 * e], de[2 * e + 1]);
            }
          }
        };
        if (lo <= 32 * ch && hi >= 32 * ch + 32)
          emit(std::false_type{});
        else
          emit(std::true_type{});
        const uint32_t te = tl + BW_TM_E + tb * 64 + 16 * ch;
        if (DKDV) tmem_st16(te, pk);
        tmem_st16(te + 32, dk);
        tmem_wait_st();
        tc_fence_before();
        mbar_arrive_warp(e_full + 8 * tb);
      }
      if (!ok) break;
      G += n;
      // accumulators -> dK, dV (DKDV) or dQ (DQ) rows
      if (!mbar_wait(acc_full, it & 1)) break;
      tc_fence_after();
      uint32_t u0[32], w0[32];  // this thread's 32 columns of dV / dQ and of dK
      tmem_ld32_async(tl + 256 + 32 * ch, u0);
      if (DKDV) tmem_ld32_async(tl + 320 + 32 * ch, w0);
      tmem_wait_ld(u0);
      if (DKDV) tmem_wait_ld(w0);
      tc_fence_before();
      mbar_arrive_warp(acc_free);
      if (row < a.Lx) {
        const long srow = (long)b * a.Lx + row;
        bf16* pu = a.out_u + srow * a.ld_u + a.col_u + h * BW_D + 32 * ch;
        const float su = DKDV ? 1.f : a.scale;
#pragma unroll
        for (int i = 0; i < 32; i += 8)
          *reinterpret_cast<uint4*>(pu + i) = make_uint4(
              pack_bf16(__uint_as_float(u0[i]) * su, __uint_as_float(u0[i + 1]) * su),
              pack_bf16(__uint_as_float(u0[i + 2]) * su, __uint_as_float(u0[i + 3]) * su),
              pack_bf16(__uint_as_float(u0[i + 4]) * su, __uint_as_float(u0[i + 5]) * su),
              pack_bf16(__uint_as_float(u0[i + 6]) * su, __uint_as_float(u0[i + 7]) * su));
        if (DKDV) {
          bf16* pw = a.out_w + srow * a.ld_w + a.col_w + h * BW_D + 32 * ch;
#pragma unroll
          for (int i = 0; i < 32; i += 8)
            *reinterpret_cast<uint4*>(pw + i) = make_uint4(
                pack_bf16(__uint_as_float(w0[i]) * a.scale, __uint_as_float(w0[i + 1]) * a.scale),
                pack_bf16(__uint_as_float(w0[i + 2]) * a.scale, __uint_as_float(w0[i + 3]) * a.scale),
                pack_bf16(__uint_as_float(w0[i + 4]) * a.scale, __uint_as_float(w0[i + 5]) * a.scale),
                pack_bf16(__uint_as_float(w0[i + 6]) * a.scale, __uint_as_float(w0[i + 7]) * a.scale));
        }
      }
    }
  }
  tc_fence_before();
  if (__syncthreads_or(*(volatile int*)&g_dev_error != 0)) {
    // error path: let this CTA's copies and MMAs land before smem / TMEM go
    if (warp == 0 && lane == 0) {
      for (uint32_t Gd = y_issued > BW_STAGES ? y_issued - BW_STAGES : 0; Gd < y_issued; ++Gd)
        mbar_wait_drain(y_full + 8 * (Gd % BW_STAGES), (Gd / BW_STAGES) & 1);
      for (uint32_t t = x_issued > 2 ? x_issued - 2 : 0; t < x_issued; ++t)
        mbar_wait_drain(x_full + 8 * (t & 1), (t >> 1) & 1);
    }
    if (warp == 1 && lane == 0) mbar_wait_drain(done, 0);
  } else if (warp == 1 && lane == 0) {
    mbar_wait(done, 0);
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, BW_TMEM_COLS);
  }
}

}  // namespace

int take_dev_error_attention_bwd_tc() { return take_dev_error_tu(); }
int set_wait_limit_attention_bwd_tc(unsigned long long ns) { return set_wait_limit_tu(ns); }

namespace {

// zero rows [r0, r1) of every sequence in a [B*Lx, ld] matrix, columns [col, col + d)
cudaError_t zero_rows(bf16* o, long ld, int col, int d, int B, int Lx, int r0, int r1,
                      cudaStream_t st) {
  if (r1 <= r0) return cudaSuccess;
  for (int b = 0; b < B; ++b) {
    const cudaError_t e = cudaMemset2DAsync(o + ((long)b * Lx + r0) * ld + col, ld * sizeof(bf16),
                                            0, (size_t)d * sizeof(bf16), (size_t)(r1 - r0), st);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

template <bool DKDV>
cudaError_t bw_launch(const CUtensorMap& x1, const CUtensorMap& x2, const CUtensorMap& y1,
                      const CUtensorMap& y2, int x1c, int x2c, int y1c, int y2c, BwArgs a,
                      const char* label, double flops, double bytes, cudaStream_t st) {
  a.Lx = DKDV ? a.Lk : a.Lq;
  a.Ly = DKDV ? a.Lq : a.Lk;
  a.n_tiles = (a.Lx + BW_M - 1) / BW_M;
  a.n_steps_total = (a.Ly + BW_N - 1) / BW_N;
  a.scale = 1.0f / sqrtf((float)BW_D);
  a.sl2 = a.scale * 1.4426950408889634f;
  // stationary tiles with work: DKDV [0, hi), DQ [lo, n_tiles)
  int lo = 0, hi = a.n_tiles;
  if (DKDV)
    while (hi > 0 && bw_first_q(a, (hi - 1) * BW_M) >= a.Lq) --hi;
  else
    while (lo < a.n_tiles && bw_vis(a, std::min(lo * BW_M + BW_M - 1, a.Lq - 1)) == 0) ++lo;
  a.n_items = (hi - lo) * a.nh * a.B;
  auto kern = attn_bwd_tc_kernel<DKDV>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, BW_SMEM);
  if (e != cudaSuccess) return e;
  LaunchTimer lt(label, st, flops, bytes);
  const int r0 = DKDV ? std::min(hi * BW_M, a.Lx) : 0, r1 = DKDV ? a.Lx : std::min(lo * BW_M, a.Lx);
  if ((e = zero_rows(a.out_u, a.ld_u, a.col_u, a.d, a.B, a.Lx, r0, r1, st)) != cudaSuccess) return e;
  if (DKDV && (e = zero_rows(a.out_w, a.ld_w, a.col_w, a.d, a.B, a.Lx, r0, r1, st)) != cudaSuccess)
    return e;
  if (a.n_items == 0) return cudaSuccess;
  const int grid = std::min(a.n_items, num_sms());
  kern<<<grid, BW_THREADS, BW_SMEM, st>>>(x1, x2, y1, y2, x1c, x2c, y1c, y2c, a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t attn_bwd_tc(const bf16* qkv, const bf16* dO, const float* lse, const float* Di,
                        bf16* dqkv, int B, int m, int d, int nh, bool causal, cudaStream_t st) {
  if (d != nh * BW_D || ((uintptr_t)qkv & 15) || ((uintptr_t)dO & 15) || ((uintptr_t)dqkv & 15))
    return cudaErrorInvalidValue;
  const uint64_t rows = (uint64_t)B * m;
  CUtensorMap qkv128, qkv64, do128, do64;
  if (!tmap_bf16_2d(&qkv128, qkv, 3ull * d, rows, 3ull * d, 64, BW_M) ||
      !tmap_bf16_2d(&qkv64, qkv, 3ull * d, rows, 3ull * d, 64, BW_N) ||
      !tmap_bf16_2d(&do128, dO, (uint64_t)d, rows, (uint64_t)d, 64, BW_M) ||
      !tmap_bf16_2d(&do64, dO, (uint64_t)d, rows, (uint64_t)d, 64, BW_N))
    return cudaErrorInvalidValue;
  BwArgs a{};
  a.lse = lse;
  a.Di = Di;
  a.B = B;
  a.Lq = a.Lk = m;
  a.d = d;
  a.nh = nh;
  a.causal = causal ? 1 : 0;
  a.P = 0;
  a.out_u = a.out_w = dqkv;
  a.ld_u = a.ld_w = 3L * d;
  const double pairs = (double)B * nh * (causal ? 0.5 * m * (m + 1.0) : (double)m * m);
  cudaError_t e;
  // DKDV: X1 = K, X2 = V (128 rows); Y1 = Q, Y2 = dO (64 rows); u = dV, w = dK
  a.col_u = 2 * d;
  a.col_w = d;
  if ((e = bw_launch<true>(qkv128, qkv128, qkv64, do64, d, 2 * d, 0, 0, a, "attn_bwd_dkdv",
                           8.0 * BW_D * pairs, 2.0 * B * m * (5.0 * d), st)) != cudaSuccess)
    return e;
  // DQ: X1 = Q, X2 = dO (128 rows); Y1 = K, Y2 = V (64 rows); u = dQ
  a.col_u = 0;
  return bw_launch<false>(qkv128, do128, qkv64, qkv64, 0, 0, d, 2 * d, a, "attn_bwd_dq",
                          6.0 * BW_D * pairs, 2.0 * B * m * (4.0 * d), st);
}

cudaError_t attn_cross_bwd(const bf16* qa, long ldq, const bf16* kv, const bf16* dO,
                           const float* lse, const float* Di, bf16* dqa, bf16* dkv, int B, int Lq,
                           int Lk, int d, int nh, int P, bool causal, cudaStream_t st) {
  if (d != nh * BW_D || P < 1 || ldq < d || ((uintptr_t)qa & 15) || ((uintptr_t)kv & 15) ||
      ((uintptr_t)dO & 15) || ((uintptr_t)dqa & 15) || ((uintptr_t)dkv & 15) || (ldq * 2) % 16)
    return cudaErrorInvalidValue;
  const uint64_t rq = (uint64_t)B * Lq, rk = (uint64_t)B * Lk;
  CUtensorMap qa128, qa64, kv128, kv64, do128, do64;
  if (!tmap_bf16_2d(&qa128, qa, (uint64_t)ldq, rq, (uint64_t)ldq, 64, BW_M) ||
      !tmap_bf16_2d(&qa64, qa, (uint64_t)ldq, rq, (uint64_t)ldq, 64, BW_N) ||
      !tmap_bf16_2d(&kv128, kv, 2ull * d, rk, 2ull * d, 64, BW_M) ||
      !tmap_bf16_2d(&kv64, kv, 2ull * d, rk, 2ull * d, 64, BW_N) ||
      !tmap_bf16_2d(&do128, dO, (uint64_t)d, rq, (uint64_t)d, 64, BW_M) ||
      !tmap_bf16_2d(&do64, dO, (uint64_t)d, rq, (uint64_t)d, 64, BW_N))
    return cudaErrorInvalidValue;
  BwArgs a{};
  a.lse = lse;
  a.Di = Di;
  a.B = B;
  a.Lq = Lq;
  a.Lk = Lk;
  a.d = d;
  a.nh = nh;
  a.causal = causal ? 1 : 0;
  a.P = P;
  double pairs = 0.0;  // visible (token, proxy) pairs per head and sequence
  if (!causal) {
    pairs = (double)Lq * Lk;
  } else {
    for (int i = 0; (long)i * P < Lq; ++i) pairs += (double)std::min(P, Lq - i * P) * std::min(i, Lk);
  }
  pairs *= (double)B * nh;
  cudaError_t e;
  // DKDV: X1 = K, X2 = V (proxies, 128 rows); Y1 = Q, Y2 = dO (tokens, 64 rows);
  // u = dV (dkv columns [d, 2d)), w = dK (columns [0, d))
  a.out_u = a.out_w = dkv;
  a.ld_u = a.ld_w = 2L * d;
  a.col_u = d;
  a.col_w = 0;
  if ((e = bw_launch<true>(kv128, kv128, qa64, do64, 0, d, 0, 0, a, "attn_cross_bwd_dkdv",
                           8.0 * BW_D * pairs, 2.0 * B * (Lk * 4.0 * d + Lq * 2.0 * d), st)) !=
      cudaSuccess)
    return e;
  // DQ: X1 = Q, X2 = dO (tokens, 128 rows); Y1 = K, Y2 = V (proxies, 64 rows);
  // u = dQ (dqa columns [0, d))
  a.out_u = dqa;
  a.ld_u = ldq;
  a.col_u = 0;
  return bw_launch<false>(qa128, do128, kv64, kv64, 0, 0, 0, d, a, "attn_cross_bwd_dq",
                          6.0 * BW_D * pairs, 2.0 * B * (Lq * 3.0 * d + Lk * 2.0 * d), st);
}

}  // namespace pf
