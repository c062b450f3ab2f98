// Proxy-space attention forward (Eq. proxy-attn) on the 5th-generation tensor
// cores: tcgen05.mma with TMEM accumulators, TMA tiles, head width 64.
//
// Work item = (two consecutive 128-query tiles A and B, head, sequence); one
// persistent CTA per SM walks the items heaviest first.  Two softmax warp
// groups, one per query tile, take turns on the SM's exponential unit (SFU):
// while one evaluates the exponentials of its tile, the other loads its next
// scores, finds their maximum and stores its probabilities, so the SFU -- the
// bound of a 64-wide head, 16384 exponentials per 128 x 128 tile against 512
// cycles of MMAs -- stays busy.
//   warp 0    TMA producer: the item's two Q tiles (double-buffered across
//             items) and a FA_STAGES-deep ring of (K, V) 128-key tiles, shared
//             by both query tiles
//   warp 1    MMA issuer: S_w = Q_w K_j^T (M=128, N=128, K=64) into tile w's
//             TMEM score buffer, and O_w += P_w V_j (M=128, N=64, K=128) with
//             P_w read from TMEM (only V comes from shared memory)
//   warps 2-5 softmax group A, warps 6-9 group B: one query row per thread
//             (TMEM lane); the 128 scores are loaded once into registers,
//             P_j = 2^(s - m) goes back to TMEM as bf16 pairs
// O accumulates in TMEM across the key tiles.  A row's probabilities are
// taken against a reference m: the maximum of its first key tile, raised only
// when a later tile's maximum exceeds it by more than FA_RESCALE (log2
// units); then the row's O and running sum are scaled by 2^(m_old - m_new).
// Every P stays at most 2^FA_RESCALE (as exact in bf16 as any other value,
// harmless in the fp32 sums).  Saved per (b, h, query): LSE = m + log2(sum)
// (log2 units), the input of the backward.  Every mbarrier wait is bounded.
//
// The same kernel serves the cross-attention injection (Eq. inj-cross): the
// queries are tokens and the keys / values proxies, from separate matrices,
// and token q sees the proxies of earlier blocks, j < q / P (causal) or all
// of them.  Query tiles that see no proxy are not computed (the host
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
constexpr int FA_STAGES = 4;
constexpr int FA_THREADS = 320;  // producer, MMA, two softmax groups of four warps
constexpr float FA_RESCALE = 8.f;
constexpr uint32_t FA_Q_BYTES = FA_M * FA_D * 2;   // 16 KB
constexpr uint32_t FA_KV_BYTES = FA_N * FA_D * 2;  // 16 KB each of K and V
constexpr uint32_t FA_OFF_KV = 4 * FA_Q_BYTES;     // Q: [2 items][tiles A, B]
constexpr uint32_t FA_OFF_BAR = FA_OFF_KV + FA_STAGES * 2 * FA_KV_BYTES;
constexpr uint32_t FA_SMEM = FA_OFF_BAR + 256 + 1024;
// TMEM columns of group w: scores S at 128 w (fp32), O at 256 + 64 w (fp32),
// P at 384 + 64 w (bf16 pairs: key 2c in the low half of column c)
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
  int n_qt, n_st, st_min, n_items;  // query tiles, tile pairs, first pair with work
  float sl2;  // log2(e) / sqrt(64)
};

// Keys visible to query q: all, the causal prefix j <= q, or (cross) the
// proxies of the blocks before q's.
__host__ __device__ __forceinline__ int fa_vis(const FaArgs& a, int q) {
  const int v = !a.causal ? a.Lk : a.P ? q / a.P : q + 1;
  return v < a.Lk ? v : a.Lk;
}

// Key tiles query tile t reads (0 past the last tile or when it sees none).
__host__ __device__ __forceinline__ int fa_ntiles(const FaArgs& a, int t) {
  if (t >= a.n_qt) return 0;
  const int last = t * FA_M + FA_M - 1 < a.Lq - 1 ? t * FA_M + FA_M - 1 : a.Lq - 1;
  return (fa_vis(a, last) + FA_N - 1) / FA_N;
}

// Items are ranked heaviest first (causal: the tile pairs with the most key
// tiles); CTA c takes rank c of round 0, rank G-1-c of round 1, and so on
// (snake order over the G CTAs), which evens out the per-CTA work.
__device__ __forceinline__ int fa_rank(int c, int round) {
  return round * (int)gridDim.x + ((round & 1) ? (int)gridDim.x - 1 - c : c);
}

__device__ __forceinline__ void fa_item(const FaArgs& a, int k, int& u, int& h, int& b, int* n) {
  const int per = a.nh * a.B;
  u = a.n_st - 1 - k / per;
  const int r = k % per;
  h = r % a.nh;
  b = r / a.nh;
  n[0] = fa_ntiles(a, 2 * u);
  n[1] = fa_ntiles(a, 2 * u + 1);
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
  // q_full[2] q_empty[2] kv_full[S] kv_empty[S], per group w: s_full s_free
  // p_full p_free o_full o_free, done
  const uint32_t b0 = smem_u32(bars);
  const uint32_t q_full = b0, q_empty = b0 + 16, kv_full = b0 + 32,
                 kv_empty = kv_full + 8 * FA_STAGES, grp0 = kv_empty + 8 * FA_STAGES,
                 done = grp0 + 2 * 48;
  auto s_full = [&](int w) { return grp0 + 48 * w; };
  auto s_free = [&](int w) { return grp0 + 48 * w + 8; };
  auto p_full = [&](int w) { return grp0 + 48 * w + 16; };
  auto p_free = [&](int w) { return grp0 + 48 * w + 24; };
  auto o_full = [&](int w) { return grp0 + 48 * w + 32; };
  auto o_free = [&](int w) { return grp0 + 48 * w + 40; };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + FA_OFF_BAR + 240);
  const uint32_t sbase = smem_u32(smem);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(q_full + 8 * i, 1);
      mbar_init(q_empty + 8 * i, 1);
      mbar_init(s_full(i), 1);
      mbar_init(s_free(i), 4);  // one arrival per softmax warp of the group
      mbar_init(p_full(i), 4);
      mbar_init(p_free(i), 1);
      mbar_init(o_full(i), 1);
      mbar_init(o_free(i), 4);
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
      int u, h, b, n2[2];
      fa_item(a, k, u, h, b, n2);
      const int n = max(n2[0], n2[1]);
      const int krow0 = b * a.Lk;
      const uint32_t qb = it & 1;
      if (!mbar_wait(q_empty + 8 * qb, ((it >> 1) & 1) ^ 1)) break;
      mbar_arrive_expect_tx(q_full + 8 * qb, (n2[0] > 0 ? FA_Q_BYTES : 0u) +
                                                 (n2[1] > 0 ? FA_Q_BYTES : 0u));
      for (int w = 0; w < 2; ++w)
        if (n2[w] > 0)
          tma_load_2d(sbase + (2 * qb + w) * FA_Q_BYTES, &tmQ, q_full + 8 * qb,
                      a.qcol + h * FA_D, b * a.Lq + (2 * u + w) * FA_M);
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
    uint32_t G = 0, it = 0;
    uint32_t gs[2] = {0, 0};  // score / probability tiles of each group so far
    uint32_t io[2] = {0, 0};  // items of each group so far
    // O_w (+)= P_w V for key tile jj of the current item (G: its first stage)
    auto issue_pv = [&](const int* n2, int jj) -> bool {
      const uint32_t st = (G + jj) % FA_STAGES;
      const uint32_t vb = sbase + FA_OFF_KV + st * 2 * FA_KV_BYTES + FA_KV_BYTES;
      for (int w = 0; w < 2; ++w) {
        if (jj >= n2[w]) continue;
        const uint32_t g = gs[w] + jj;
        if (!mbar_wait_warp(p_full(w), g & 1)) return false;
        if (jj == 0 && io[w] > 0 && !mbar_wait_warp(o_free(w), (io[w] - 1) & 1)) return false;
        tc_fence_after();
        const uint32_t pt = tmem + 384 + 64 * w, ot = tmem + 256 + 64 * w;
        if (elect_one()) {
#pragma unroll
          for (int kk = 0; kk < FA_N / 16; ++kk)
            tc_mma_f16_ts(ot, pt + kk * 8, smem_desc_sw128(vb + kk * 2048, 8192, 1024), idesc_o,
                          (jj > 0 || kk > 0) ? 1u : 0u);
          tc_commit(p_free(w));
          if (jj == n2[w] - 1) tc_commit(o_full(w));
        }
        __syncwarp();
      }
      if (elect_one()) tc_commit(kv_empty + 8 * st);
      __syncwarp();
      return true;
    };
    for (int rd = 0, k = fa_rank(blockIdx.x, 0); k < a.n_items && ok;
         k = fa_rank(blockIdx.x, ++rd), ++it) {
      int u, h, b, n2[2];
      fa_item(a, k, u, h, b, n2);
      const int n = max(n2[0], n2[1]);
      const uint32_t qb = it & 1;
      if (!mbar_wait_warp(q_full + 8 * qb, (it >> 1) & 1)) break;
      tc_fence_after();
      for (int j = 0; j < n && ok; ++j) {
        const uint32_t st = (G + j) % FA_STAGES;
        if (!mbar_wait_warp(kv_full + 8 * st, ((G + j) / FA_STAGES) & 1)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t ks = sbase + FA_OFF_KV + st * 2 * FA_KV_BYTES;
        for (int w = 0; w < 2; ++w) {
          if (j >= n2[w]) continue;
          const uint32_t g = gs[w] + j;
          if (g > 0 && !mbar_wait_warp(s_free(w), (g - 1) & 1)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t qs = sbase + (2 * qb + w) * FA_Q_BYTES;
          if (elect_one()) {
#pragma unroll
            for (int kk = 0; kk < FA_D / 16; ++kk)
              tc_mma_f16(tmem + 128 * w, smem_desc_sw128(qs + kk * 32, 16, 1024),
                         smem_desc_sw128(ks + kk * 32, 16, 1024), idesc_s, kk ? 1u : 0u);
            tc_commit(s_full(w));
          }
          __syncwarp();
        }
        if (!ok) break;
        if (j == n - 1) {
          if (elect_one()) tc_commit(q_empty + 8 * qb);
          __syncwarp();
        }
        if (j > 0 && !issue_pv(n2, j - 1)) ok = false;
      }
      if (!ok || !issue_pv(n2, n - 1)) break;
      for (int w = 0; w < 2; ++w)
        if (n2[w] > 0) {
          gs[w] += n2[w];
          ++io[w];
        }
      G += n;
    }
    if (elect_one()) tc_commit(done);
    __syncwarp();
  } else if (warp >= 2) {
    // ------------------------------------------------------------ softmax
    const int w = (warp - 2) >> 2;  // group: query tile A (0) or B (1)
    const int q4 = warp & 3;         // TMEM lane quarter
    const int r = q4 * 32 + lane;    // query row in the tile = TMEM lane
    const uint32_t tl = tmem + ((uint32_t)(q4 * 32) << 16);
    const uint32_t ts = tl + 128 * w, to = tl + 256 + 64 * w, tp = tl + 384 + 64 * w;
    bool ok = true;
    uint32_t g = 0, io = 0;
    for (int rd = 0, k = fa_rank(blockIdx.x, 0); k < a.n_items && ok;
         k = fa_rank(blockIdx.x, ++rd)) {
      int u, h, b, n2[2];
      fa_item(a, k, u, h, b, n2);
      const int nw = n2[w];
      if (nw == 0) continue;
      const int q = (2 * u + w) * FA_M + r;  // query index in the sequence
      const int vis = fa_vis(a, q);
      float mref = 0.f, l = 0.f;
      for (int j = 0; j < nw; ++j, ++g) {
        if (!mbar_wait_warp(s_full(w), g & 1)) {
          ok = false;
          break;
        }
        tc_fence_after();
        // keys c >= lim of this tile are masked (causal diagonal or block
        // boundary, sequence end); lim <= 0 masks the whole tile
        const int lim = min(FA_N, vis - j * FA_N);
        // the tile's row maximum (log2 units): 64 TMEM columns at a time,
        // three-input maxima
        float mt;
        {
          float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll 1
          for (int hh = 0; hh < 2; ++hh) {
            uint32_t ra[32], rb[32];
            tmem_ld32_async(ts + 64 * hh, ra);
            tmem_ld32_async(ts + 64 * hh + 32, rb);
            tmem_wait_ld(ra);
            tmem_wait_ld(rb);
            if (lim >= FA_N) {
#pragma unroll
              for (int c = 0; c < 32; c += 2) {
                mx0 = max3f(mx0, __uint_as_float(ra[c]), __uint_as_float(ra[c + 1]));
                mx1 = max3f(mx1, __uint_as_float(rb[c]), __uint_as_float(rb[c + 1]));
              }
            } else {
#pragma unroll
              for (int c = 0; c < 32; ++c) {
                const float va = 64 * hh + c < lim ? __uint_as_float(ra[c]) : -INFINITY;
                const float vb = 64 * hh + 32 + c < lim ? __uint_as_float(rb[c]) : -INFINITY;
                mx0 = max3f(mx0, va, vb);
              }
            }
          }
          mt = fmaxf(mx0, mx1) * a.sl2;
        }
        // the first tile sets the reference m; later tiles raise it only by
        // more than FA_RESCALE, scaling O and the running sum
        float corr = 1.f, mnew = mref;
        if (j == 0) {
          mnew = mt == -INFINITY ? 0.f : mt;
        } else if (mt > mref + FA_RESCALE) {
          mnew = mt;
          corr = ex2_approx(mref - mnew);
        }
        // P_w of the previous tile has been consumed (and O_w updated) by
        // the time this wait returns; a new item waited on o_full instead
        if (j > 0 && !mbar_wait_warp(p_free(w), (g - 1) & 1)) {
          ok = false;
          break;
        }
        tc_fence_after();
        // P = 2^(s * sl2 - m) into TMEM as bf16 pairs (key 2c, 2c + 1 in
        // column c) and the row sum, with packed fp32x2 arithmetic
        float2 ps = make_float2(0.f, 0.f);
        {
          const float2 sl = make_float2(a.sl2, a.sl2), nm = make_float2(-mnew, -mnew);
#pragma unroll 1
          for (int hh = 0; hh < 2; ++hh) {
            uint32_t ra[32], rb[32], pk[32];
            tmem_ld32_async(ts + 64 * hh, ra);
            tmem_ld32_async(ts + 64 * hh + 32, rb);
            tmem_wait_ld(ra);
            tmem_wait_ld(rb);
#pragma unroll
            for (int c = 0; c < 64; c += 2) {
              const uint32_t* src = c < 32 ? ra + c : rb + (c - 32);
              const float2 z = __ffma2_rn(
                  make_float2(__uint_as_float(src[0]), __uint_as_float(src[1])), sl, nm);
              float2 pp = make_float2(ex2_approx(z.x), ex2_approx(z.y));
              if (lim < FA_N) {
                if (64 * hh + c >= lim) pp.x = 0.f;
                if (64 * hh + c + 1 >= lim) pp.y = 0.f;
              }
              ps = __fadd2_rn(ps, pp);
              pk[c >> 1] = pack_bf16(pp.x, pp.y);
            }
            tmem_st32(tp + 32 * hh, pk);
          }
        }
        const float psum = ps.x + ps.y;
        if (__any_sync(0xffffffffu, corr != 1.f)) {  // rescale this warp's rows of O
#pragma unroll 1
          for (int c = 0; c < 64; c += 16) {
            uint32_t ov[16];
            tmem_ld16(to + c, ov);
#pragma unroll
            for (int i = 0; i < 16; ++i) ov[i] = __float_as_uint(__uint_as_float(ov[i]) * corr);
            tmem_st16(to + c, ov);
          }
        }
        tc_fence_before();
        mbar_arrive_warp(s_free(w));  // this group's scores are no longer read
        l = fmaf(l, corr, psum);
        mref = mnew;
        tmem_wait_st();
        tc_fence_before();
        mbar_arrive_warp(p_full(w));
      }
      if (!ok) break;
      // the item's O: after its last P.V
      if (!mbar_wait_warp(o_full(w), io & 1)) break;
      ++io;
      tc_fence_after();
      uint32_t ov[64];
      tmem_ld32_async(to, ov);
      tmem_ld32_async(to + 32, ov + 32);
      tmem_wait_ld(ov);
      tmem_wait_ld(ov + 32);
      tc_fence_before();
      mbar_arrive_warp(o_free(w));
      if (q < a.Lq) {
        const float inv = l > 0.f ? 1.f / l : 0.f;  // a row that sees no key: 0
        const long row = (long)b * a.Lq + q;
        if (a.out) {
          bf16* op = a.out + row * a.ldo + h * FA_D;
#pragma unroll
          for (int i = 0; i < FA_D; i += 8) {
            const float* o = reinterpret_cast<const float*>(ov + i);
            *reinterpret_cast<uint4*>(op + i) =
                make_uint4(pack_bf16(o[0] * inv, o[1] * inv), pack_bf16(o[2] * inv, o[3] * inv),
                           pack_bf16(o[4] * inv, o[5] * inv), pack_bf16(o[6] * inv, o[7] * inv));
          }
        }
        if (a.out_g) {
          const float x = __bfloat162float(a.gpre[row * a.ldg + a.gcol + h]) + a.b_a[h];
          const float gi = inv / (1.f + __expf(-x));
          bf16* gp = a.out_g + row * a.ldo + h * FA_D;
#pragma unroll
          for (int i = 0; i < FA_D; i += 8) {
            const float* o = reinterpret_cast<const float*>(ov + i);
            *reinterpret_cast<uint4*>(gp + i) =
                make_uint4(pack_bf16(o[0] * gi, o[1] * gi), pack_bf16(o[2] * gi, o[3] * gi),
                           pack_bf16(o[4] * gi, o[5] * gi), pack_bf16(o[6] * gi, o[7] * gi));
          }
        }
        a.lse[((long)b * a.nh + h) * a.Lq + q] = l > 0.f ? mref + log2f(l) : 0.f;  // log2 units
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
  a.n_st = (a.n_qt + 1) / 2;
  int qt_min = 0;  // query tiles before qt_min see no key
  while (qt_min < a.n_qt && fa_ntiles(a, qt_min) == 0) ++qt_min;
  a.st_min = qt_min / 2;
  a.n_items = qt_min >= a.n_qt ? 0 : (a.n_st - a.st_min) * a.nh * a.B;
  a.sl2 = 1.4426950408889634f / sqrtf((float)FA_D);
  auto kern = attn_fwd_tc_kernel;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, FA_SMEM);
  if (e != cudaSuccess) return e;
  LaunchTimer lt(label, st, 4.0 * FA_D * pairs, bytes);
  if (qt_min > 0) {  // query tiles that see no key: zero rows, LSE 0
    const size_t rows = (size_t)std::min(qt_min * FA_M, a.Lq);
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
