// Proxy-space attention forward (Eq. proxy-attn) on the 5th-generation tensor
// cores: tcgen05.mma with TMEM accumulators, TMA tiles, head width 64.
//
// Work item = (128-query tile, head, sequence); one persistent CTA per SM
// walks the items heaviest first (causal rows with the most key tiles).
//   warp 0    TMA producer: the item's Q tile (double-buffered across items)
//             and a FA_STAGES-deep ring of (K, V) 128-key tiles
//   warp 1    MMA issuer: S_j = Q K_j^T (M=128, N=128, K=64) into one of two
//             TMEM S buffers, and O_j = P_j V_j (M=128, N=64, K=128) into one
//             of two TMEM O buffers; S_{j+1} is issued before O_j so that the
//             softmax always has the next scores ready
//   warps 2-5 softmax, one query row per thread (TMEM lane): online max /
//             sum in log2 units, P_j written as bf16 into shared memory in the
//             128B-swizzled K-major layout the MMA reads, then O_j read back
//             from TMEM and folded into a register accumulator with the
//             running-max correction
// Saved per (b, h, query): LSE = max + log2(sum) (log2 units), the input of
// the backward.  Every mbarrier wait is bounded.
//
// The same kernel serves the cross-attention injection (Eq. inj-cross): the
// queries are tokens and the keys / values proxies, from separate matrices,
// and token q sees the proxies of earlier blocks, j < q / P (causal) or all
// of them.  Query tiles that see no proxy are not work items (the host
// zero-fills their rows); a row that sees none writes zeros and LSE 0.  An
// optional second output applies the per-head gate sigmoid(a + b_a) (the
// ungated output is optional too, for inference).
#include <algorithm>

#include "kernels.h"

namespace pf {

namespace {

constexpr int FA_M = 128;  // query rows per tile (TMEM lanes)
constexpr int FA_N = 128;  // keys per tile
constexpr int FA_D = 64;   // head width
constexpr int FA_STAGES = 3;
constexpr int FA_THREADS = 192;
constexpr uint32_t FA_Q_BYTES = FA_M * FA_D * 2;   // 16 KB
constexpr uint32_t FA_KV_BYTES = FA_N * FA_D * 2;  // 16 KB each of K and V
constexpr uint32_t FA_P_BYTES = FA_M * FA_N * 2;   // 32 KB
constexpr uint32_t FA_OFF_KV = 2 * FA_Q_BYTES;
constexpr uint32_t FA_OFF_P = FA_OFF_KV + FA_STAGES * 2 * FA_KV_BYTES;
constexpr uint32_t FA_OFF_BAR = FA_OFF_P + 2 * FA_P_BYTES;
constexpr uint32_t FA_SMEM = FA_OFF_BAR + 256 + 1024;
// TMEM columns: S buffers at 0 and 128, O buffers at 256 and 320
constexpr uint32_t FA_TMEM_COLS = 512;

struct FaArgs {
  bf16* out;          // [B*Lq, ldo], head h at column h*64
  bf16* out_g;        // gated copy sigmoid(gate + b_a[h]) * out, or null
  const bf16* gpre;   // gate pre-activations: row b*Lq + q, column gcol + h
  const float* b_a;   // [nh]
  float* lse;         // [B, nh, Lq]
  long ldo, ldg;
  int gcol, qcol, kcol, vcol;  // column offsets of gate, Q, K, V in their matrices
  int B, Lq, Lk, d, nh, causal, P;  // P > 0: cross-attention with block size P
  int n_qt, qt_min, n_kt, n_items;
  float sl2;  // log2(e) / sqrt(64)
};

// Keys visible to query q: all, the causal prefix j <= q, or (cross) the
// proxies of the blocks before q's.
__host__ __device__ __forceinline__ int fa_vis(const FaArgs& a, int q) {
  const int v = !a.causal ? a.Lk : a.P ? q / a.P : q + 1;
  return v < a.Lk ? v : a.Lk;
}

// Items are ranked heaviest first (causal: the query tiles with the most key
// tiles); CTA c takes rank c of round 0, rank G-1-c of round 1, and so on
// (snake order over the G CTAs), which evens out the per-CTA work.
__device__ __forceinline__ int fa_rank(int c, int round) {
  return round * (int)gridDim.x + ((round & 1) ? (int)gridDim.x - 1 - c : c);
}

__device__ __forceinline__ void fa_item(const FaArgs& a, int k, int& qt, int& h, int& b, int& n) {
  const int per = a.nh * a.B;
  qt = a.n_qt - 1 - k / per;
  const int r = k % per;
  h = r % a.nh;
  b = r / a.nh;
  n = (fa_vis(a, min(qt * FA_M + FA_M - 1, a.Lq - 1)) + FA_N - 1) / FA_N;
}

// 2^x on the SFU (ex2.approx, flush-to-zero): relative error about 2^-22,
// far below the bf16 rounding of P
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__global__ void __launch_bounds__(FA_THREADS, 1)
    attn_fwd_tc_kernel(const __grid_constant__ CUtensorMap tmQ,
                       const __grid_constant__ CUtensorMap tmKV, FaArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + FA_OFF_BAR);
  // q_full[2] q_empty[2] kv_full[S] kv_empty[S] s_full[2] p_full[2] o_full[2] o_free[2] done
  const uint32_t b0 = smem_u32(bars);
  const uint32_t q_full = b0, q_empty = b0 + 16, kv_full = b0 + 32,
                 kv_empty = kv_full + 8 * FA_STAGES, s_full = kv_empty + 8 * FA_STAGES,
                 p_full = s_full + 16, o_full = p_full + 16, o_free = o_full + 16,
                 done = o_free + 16;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + FA_OFF_BAR + 240);
  const uint32_t sbase = smem_u32(smem);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(q_full + 8 * i, 1);
      mbar_init(q_empty + 8 * i, 1);
      mbar_init(s_full + 8 * i, 1);
      mbar_init(p_full + 8 * i, 128);
      mbar_init(o_full + 8 * i, 1);
      mbar_init(o_free + 8 * i, 128);
    }
    for (int i = 0; i < FA_STAGES; ++i) {
      mbar_init(kv_full + 8 * i, 1);
      mbar_init(kv_empty + 8 * i, 1);
    }
    mbar_init(done, 1);
    fence_barrier_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), FA_TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  uint32_t kv_issued = 0, q_issued = 0;

  if (warp == 0 && lane == 0) {
    // ------------------------------------------------------------ producer
    prefetch_tmap(&tmQ);
    prefetch_tmap(&tmKV);
    bool ok = true;
    uint32_t it = 0;
    for (int rd = 0, k = fa_rank(blockIdx.x, 0); k < a.n_items && ok;
         k = fa_rank(blockIdx.x, ++rd), ++it) {
      int qt, h, b, n;
      fa_item(a, k, qt, h, b, n);
      const int krow0 = b * a.Lk;
      const uint32_t qb = it & 1;
      if (!mbar_wait(q_empty + 8 * qb, ((it >> 1) & 1) ^ 1)) break;
      mbar_arrive_expect_tx(q_full + 8 * qb, FA_Q_BYTES);
      tma_load_2d(sbase + qb * FA_Q_BYTES, &tmQ, q_full + 8 * qb, a.qcol + h * FA_D,
                  b * a.Lq + qt * FA_M);
      q_issued = it + 1;
      for (int j = 0; j < n; ++j) {
        const uint32_t g = kv_issued, st = g % FA_STAGES;
        if (!mbar_wait(kv_empty + 8 * st, ((g / FA_STAGES) & 1) ^ 1)) {
          ok = false;
          break;
        }
        const uint32_t kdst = sbase + FA_OFF_KV + st * 2 * FA_KV_BYTES;
        mbar_arrive_expect_tx(kv_full + 8 * st, 2 * FA_KV_BYTES);
        tma_load_2d(kdst, &tmKV, kv_full + 8 * st, a.kcol + h * FA_D, krow0 + j * FA_N);
        tma_load_2d(kdst + FA_KV_BYTES, &tmKV, kv_full + 8 * st, a.vcol + h * FA_D,
                    krow0 + j * FA_N);
        kv_issued = g + 1;
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    // The whole warp runs the loop; one elected lane issues and commits.
    constexpr uint32_t idesc_s = idesc_bf16_f32(FA_M, FA_N, 0, 0);
    constexpr uint32_t idesc_o = idesc_bf16_f32(FA_M, FA_D, 0, 1);
    bool ok = true;
    auto issue_o = [&](uint32_t G) -> bool {
      const uint32_t ob = G & 1, st = G % FA_STAGES;
      if (!mbar_wait_warp(p_full + 8 * ob, (G >> 1) & 1)) return false;
      if (!mbar_wait_warp(o_free + 8 * ob, ((G >> 1) & 1) ^ 1)) return false;
      tc_fence_after();
      const uint32_t pb = sbase + FA_OFF_P + ob * FA_P_BYTES;
      const uint32_t vb = sbase + FA_OFF_KV + st * 2 * FA_KV_BYTES + FA_KV_BYTES;
      if (elect_one()) {
#pragma unroll
        for (int kk = 0; kk < FA_N / 16; ++kk) {
          const uint64_t ad =
              smem_desc_sw128(pb + (kk >> 2) * (FA_M * 128) + (kk & 3) * 32, 16, 1024);
          const uint64_t bd = smem_desc_sw128(vb + kk * 2048, 8192, 1024);
          tc_mma_f16(tmem + 256 + ob * FA_D, ad, bd, idesc_o, kk ? 1u : 0u);
        }
        tc_commit(o_full + 8 * ob);
        tc_commit(kv_empty + 8 * st);
      }
      __syncwarp();
      return true;
    };
    uint32_t g = 0, it = 0;
    for (int rd = 0, k = fa_rank(blockIdx.x, 0); k < a.n_items && ok;
         k = fa_rank(blockIdx.x, ++rd), ++it) {
      int qt, h, b, n;
      fa_item(a, k, qt, h, b, n);
      const uint32_t qb = it & 1;
      if (!mbar_wait_warp(q_full + 8 * qb, (it >> 1) & 1)) break;
      tc_fence_after();
      const uint32_t qs = sbase + qb * FA_Q_BYTES;
      for (int j = 0; j < n; ++j) {
        const uint32_t G = g + j, st = G % FA_STAGES, sb = G & 1;
        if (!mbar_wait_warp(kv_full + 8 * st, (G / FA_STAGES) & 1)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t ks = sbase + FA_OFF_KV + st * 2 * FA_KV_BYTES;
        if (elect_one()) {
#pragma unroll
          for (int kk = 0; kk < FA_D / 16; ++kk)
            tc_mma_f16(tmem + sb * FA_N, smem_desc_sw128(qs + kk * 32, 16, 1024),
                       smem_desc_sw128(ks + kk * 32, 16, 1024), idesc_s, kk ? 1u : 0u);
          tc_commit(s_full + 8 * sb);
          if (j == n - 1) tc_commit(q_empty + 8 * qb);
        }
        __syncwarp();
        if (j > 0 && !issue_o(G - 1)) {
          ok = false;
          break;
        }
      }
      if (!ok || !issue_o(g + n - 1)) break;
      g += n;
    }
    if (elect_one()) tc_commit(done);
    __syncwarp();
  } else if (warp >= 2) {
    // ------------------------------------------------------------ softmax
    const int q4 = warp & 3;
    const int r = q4 * 32 + lane;  // query row in the tile = TMEM lane
    const uint32_t tl = tmem + ((uint32_t)(q4 * 32) << 16);
    bool ok = true;
    uint32_t g = 0;
    for (int rd = 0, k = fa_rank(blockIdx.x, 0); k < a.n_items && ok;
         k = fa_rank(blockIdx.x, ++rd)) {
      int qt, h, b, n;
      fa_item(a, k, qt, h, b, n);
      const int q = qt * FA_M + r;  // query index in the sequence
      const int vis = fa_vis(a, q);
      float mrun = -INFINITY, l = 0.f, corr_prev = 1.f;
      float o[FA_D];
#pragma unroll
      for (int i = 0; i < FA_D; ++i) o[i] = 0.f;
      auto consume_o = [&](uint32_t G, float c) -> bool {
        const uint32_t ob = G & 1;
        if (!mbar_wait(o_full + 8 * ob, (G >> 1) & 1)) return false;
        tc_fence_after();
        uint32_t x0[32], x1[32];
        tmem_ld32_async(tl + 256 + ob * FA_D, x0);
        tmem_ld32_async(tl + 256 + ob * FA_D + 32, x1);
        tmem_wait_ld(x0);
        tmem_wait_ld(x1);
        tc_fence_before();
        mbar_arrive(o_free + 8 * ob);
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          o[i] = fmaf(o[i], c, __uint_as_float(x0[i]));
          o[32 + i] = fmaf(o[32 + i], c, __uint_as_float(x1[i]));
        }
        return true;
      };
      for (int j = 0; j < n; ++j) {
        const uint32_t G = g + j, sb = G & 1;
        if (!mbar_wait(s_full + 8 * sb, (G >> 1) & 1)) {
          ok = false;
          break;
        }
        tc_fence_after();
        // two passes over the 128 scores, 64 TMEM columns at a time: the row
        // maximum, then the probabilities (keeps the live registers low).
        // Keys c >= lim of this tile are masked (causal diagonal or block
        // boundary, sequence end); lim <= 0 masks the whole tile.
        const int key0 = j * FA_N;
        const int lim = min(FA_N, min(a.Lk, vis) - key0);
        const uint32_t ts = tl + sb * FA_N;
        uint32_t ra[32], rb[32];
        float m8[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) m8[i] = -INFINITY;
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          tmem_ld32_async(ts + hh * 64, ra);
          tmem_ld32_async(ts + hh * 64 + 32, rb);
          tmem_wait_ld(ra);
          tmem_wait_ld(rb);
          if (lim >= FA_N) {
#pragma unroll
            for (int c = 0; c < 32; ++c)
              m8[c & 7] = fmaxf(m8[c & 7], fmaxf(__uint_as_float(ra[c]), __uint_as_float(rb[c])));
          } else {
#pragma unroll
            for (int c = 0; c < 32; ++c) {
              const float va = hh * 64 + c < lim ? __uint_as_float(ra[c]) : -INFINITY;
              const float vb = hh * 64 + 32 + c < lim ? __uint_as_float(rb[c]) : -INFINITY;
              m8[c & 7] = fmaxf(m8[c & 7], fmaxf(va, vb));
            }
          }
        }
        const float mx = fmaxf(mrun, fmaxf(fmaxf(fmaxf(m8[0], m8[1]), fmaxf(m8[2], m8[3])),
                                           fmaxf(fmaxf(m8[4], m8[5]), fmaxf(m8[6], m8[7]))) *
                                         a.sl2);
        const float mref = (mx == -INFINITY) ? 0.f : mx;
        const float corr = ex2_approx(mrun - mref);
        float ps[4] = {0.f, 0.f, 0.f, 0.f};
        // P_j (bf16) into shared memory: row r, 8-key group kg at 16-byte
        // slot (kg & 7) ^ (r & 7) of the row's 128-byte line in half kg >> 3
        uint8_t* prow = smem + FA_OFF_P + sb * FA_P_BYTES + r * 128;
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          tmem_ld32_async(ts + hh * 64, ra);
          tmem_ld32_async(ts + hh * 64 + 32, rb);
          tmem_wait_ld(ra);
          tmem_wait_ld(rb);
#pragma unroll
          for (int kg = 0; kg < 8; ++kg) {
            const uint32_t* src = kg < 4 ? ra + kg * 8 : rb + (kg - 4) * 8;
            float p[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              p[e] = ex2_approx(fmaf(__uint_as_float(src[e]), a.sl2, -mref));
              if (lim < FA_N && hh * 64 + kg * 8 + e >= lim) p[e] = 0.f;
              ps[e & 3] += p[e];
            }
            const uint4 v = make_uint4(pack_bf16(p[0], p[1]), pack_bf16(p[2], p[3]),
                                       pack_bf16(p[4], p[5]), pack_bf16(p[6], p[7]));
            *reinterpret_cast<uint4*>(prow + hh * (FA_M * 128) + ((kg ^ (r & 7)) << 4)) = v;
          }
        }
        const float psum = (ps[0] + ps[1]) + (ps[2] + ps[3]);
        l = fmaf(l, corr, psum);
        mrun = mx;
        fence_proxy_async_smem();
        tc_fence_before();
        mbar_arrive(p_full + 8 * sb);
        if (j > 0 && !consume_o(G - 1, corr_prev)) {
          ok = false;
          break;
        }
        corr_prev = corr;
      }
      if (!ok || !consume_o(g + n - 1, corr_prev)) break;
      g += n;
      if (q < a.Lq) {
        const float inv = l > 0.f ? 1.f / l : 0.f;  // a row that sees no key: 0
        const long row = (long)b * a.Lq + q;
        if (a.out) {
          bf16* op = a.out + row * a.ldo + h * FA_D;
#pragma unroll
          for (int i = 0; i < FA_D; i += 8) {
            const uint4 v = make_uint4(pack_bf16(o[i] * inv, o[i + 1] * inv),
                                       pack_bf16(o[i + 2] * inv, o[i + 3] * inv),
                                       pack_bf16(o[i + 4] * inv, o[i + 5] * inv),
                                       pack_bf16(o[i + 6] * inv, o[i + 7] * inv));
            *reinterpret_cast<uint4*>(op + i) = v;
          }
        }
        if (a.out_g) {
          const float x = __bfloat162float(a.gpre[row * a.ldg + a.gcol + h]) + a.b_a[h];
          const float gi = inv / (1.f + __expf(-x));
          bf16* gp = a.out_g + row * a.ldo + h * FA_D;
#pragma unroll
          for (int i = 0; i < FA_D; i += 8)
            *reinterpret_cast<uint4*>(gp + i) =
                make_uint4(pack_bf16(o[i] * gi, o[i + 1] * gi), pack_bf16(o[i + 2] * gi, o[i + 3] * gi),
                           pack_bf16(o[i + 4] * gi, o[i + 5] * gi), pack_bf16(o[i + 6] * gi, o[i + 7] * gi));
        }
        a.lse[((long)b * a.nh + h) * a.Lq + q] = l > 0.f ? mrun + log2f(l) : 0.f;  // log2 units
      }
    }
  }
  tc_fence_before();
  if (__syncthreads_or(*(volatile int*)&g_dev_error != 0)) {
    // error path: let this CTA's copies and MMAs land before smem / TMEM go
    if (warp == 0 && lane == 0) {
      for (uint32_t G = kv_issued > FA_STAGES ? kv_issued - FA_STAGES : 0; G < kv_issued; ++G)
        mbar_wait_drain(kv_full + 8 * (G % FA_STAGES), (G / FA_STAGES) & 1);
      for (uint32_t t = q_issued > 2 ? q_issued - 2 : 0; t < q_issued; ++t)
        mbar_wait_drain(q_full + 8 * (t & 1), (t >> 1) & 1);
    }
    if (warp == 1 && lane == 0) mbar_wait_drain(done, 0);
  } else if (warp == 1 && lane == 0) {
    mbar_wait(done, 0);
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, FA_TMEM_COLS);
  }
}

}  // namespace

int take_dev_error_attention_tc() { return take_dev_error_tu(); }
int set_wait_limit_attention_tc(unsigned long long ns) { return set_wait_limit_tu(ns); }

namespace {

cudaError_t fa_launch(const CUtensorMap& tq, const CUtensorMap& tkv, FaArgs& a, const char* label,
                      double pairs, double bytes, cudaStream_t st) {
  a.n_qt = (a.Lq + FA_M - 1) / FA_M;
  a.n_kt = (a.Lk + FA_N - 1) / FA_N;
  a.qt_min = 0;
  while (a.qt_min < a.n_qt && fa_vis(a, std::min(a.qt_min * FA_M + FA_M - 1, a.Lq - 1)) == 0)
    ++a.qt_min;
  a.n_items = (a.n_qt - a.qt_min) * a.nh * a.B;
  a.sl2 = 1.4426950408889634f / sqrtf((float)FA_D);
  auto kern = attn_fwd_tc_kernel;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, FA_SMEM);
  if (e != cudaSuccess) return e;
  LaunchTimer lt(label, st, 4.0 * FA_D * pairs, bytes);
  if (a.qt_min > 0) {  // query tiles that see no key: zero rows, LSE 0
    const size_t rows = (size_t)std::min(a.qt_min * FA_M, a.Lq);
    for (int b = 0; b < a.B; ++b) {
      bf16* dsts[2] = {a.out, a.out_g};
      for (bf16* o : dsts)
        if (o && (e = cudaMemset2DAsync(o + (long)b * a.Lq * a.ldo, a.ldo * sizeof(bf16), 0,
                                        (size_t)a.d * sizeof(bf16), rows, st)) != cudaSuccess)
          return e;
    }
    if ((e = cudaMemset2DAsync(a.lse, (size_t)a.Lq * sizeof(float), 0, rows * sizeof(float),
                               (size_t)a.B * a.nh, st)) != cudaSuccess)
      return e;
  }
  if (a.n_items == 0) return cudaSuccess;
  const int grid = std::min(a.n_items, num_sms());
  kern<<<grid, FA_THREADS, FA_SMEM, st>>>(tq, tkv, a);
  return cudaGetLastError();
}

double cross_pairs(int Lq, int Lk, int P, bool causal) {
  if (!causal) return (double)Lq * Lk;
  double s = 0.0;
  for (int i = 0; (long)i * P < Lq; ++i)  // block i's tokens see min(i, Lk) proxies
    s += (double)std::min(P, Lq - i * P) * std::min(i, Lk);
  return s;
}

}  // namespace

cudaError_t attn_fwd(const bf16* qkv, bf16* out, float* lse, int B, int m, int d, int nh,
                        bool causal, cudaStream_t st) {
  if (d != nh * FA_D || ((uintptr_t)qkv & 15) || ((uintptr_t)out & 15))
    return cudaErrorInvalidValue;
  CUtensorMap tm;
  if (!tmap_bf16_2d(&tm, qkv, (uint64_t)3 * d, (uint64_t)B * m, (uint64_t)3 * d, 64, 128))
    return cudaErrorInvalidValue;
  FaArgs a{};
  a.out = out;
  a.lse = lse;
  a.ldo = d;
  a.qcol = 0;
  a.kcol = d;
  a.vcol = 2 * d;
  a.B = B;
  a.Lq = a.Lk = m;
  a.d = d;
  a.nh = nh;
  a.causal = causal ? 1 : 0;
  a.P = 0;
  const double pairs = (double)B * nh * (causal ? 0.5 * m * (m + 1.0) : (double)m * m);
  return fa_launch(tm, tm, a, "attn_fwd", pairs, 2.0 * B * m * (4.0 * d) + 4.0 * B * nh * m, st);
}

cudaError_t attn_cross_fwd(const bf16* qa, long ldq, const bf16* kv, const float* b_a, bf16* out,
                           bf16* out_g, float* lse, int B, int Lq, int Lk, int d, int nh, int P,
                           bool causal, cudaStream_t st) {
  if (d != nh * FA_D || P < 1 || ldq < d + nh || ((uintptr_t)qa & 15) || ((uintptr_t)kv & 15) ||
      ((uintptr_t)out & 15) || ((uintptr_t)out_g & 15) || (ldq * 2) % 16 || !b_a)
    return cudaErrorInvalidValue;
  CUtensorMap tq, tkv;
  if (!tmap_bf16_2d(&tq, qa, (uint64_t)ldq, (uint64_t)B * Lq, (uint64_t)ldq, 64, 128) ||
      !tmap_bf16_2d(&tkv, kv, (uint64_t)2 * d, (uint64_t)B * Lk, (uint64_t)2 * d, 64, 128))
    return cudaErrorInvalidValue;
  FaArgs a{};
  a.out = out;
  a.out_g = out_g;
  a.gpre = qa;
  a.b_a = b_a;
  a.lse = lse;
  a.ldo = d;
  a.ldg = ldq;
  a.gcol = d;
  a.qcol = 0;
  a.kcol = 0;
  a.vcol = d;
  a.B = B;
  a.Lq = Lq;
  a.Lk = Lk;
  a.d = d;
  a.nh = nh;
  a.causal = causal ? 1 : 0;
  a.P = P;
  const double pairs = (double)B * nh * cross_pairs(Lq, Lk, P, causal);
  const double bytes = 2.0 * B * ((double)Lq * (d + nh) + 2.0 * Lk * d +
                                  (out_g ? 2.0 : 1.0) * Lq * d) + 4.0 * B * nh * Lq;
  return fa_launch(tq, tkv, a, "attn_cross_fwd", pairs, bytes, st);
}

}  // namespace pf
