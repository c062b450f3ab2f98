// tcgen05 / TMEM / TMA GEMM for sm_103a with fused epilogues.
//
//   D[M, N] = sum_k A[m, k] * B[n, k]     (bf16 operands, fp32 accumulation)
//
// A is K-major (stored [M, K]) or MN-major (stored [K, M]); likewise B ([N, K]
// or [K, N]).  Every contraction of the layer (compression, proxy Q/K/V/O,
// decompression, and all of their weight / input gradients) is one of these.
//
// Persistent: one CTA per SM walks the 128 x BN output tiles tile = blockIdx.x
// + k * gridDim.x (N fastest, so co-running CTAs share A panels and all of B
// in L2; M fastest when A has at most 16 row tiles and B is wider than the
// grid, so co-running CTAs share B tiles).  With BN = 256 and enough tiles the
// kernel runs on CTA pairs (clusters of two): a pair owns a 256 x 256 tile,
// rank 0 issues tcgen05.mma.cta_group::2 (M = 256) and each CTA stages its 128
// rows of A and half of B, so a stage is 32 KB instead of 48 and 7 (4-5 with an
// X tile) fit where 4 (3) did: the deeper ring hides the HBM latency of the
// streamed operand (a mainloop measured at ~680 cycles per 64-deep K block
// with 4 stages runs at ~525 with 6, the MMAs' own time being 512).  Roles:
//   warp 0   : TMA producer (one thread): STAGES-deep ring of 128B-swizzled
//              64-wide K slices of A and B, continuing across tiles
//   warp 1   : TMEM allocator + MMA issuer (one elected lane): tcgen05.mma
//              M=128 (a pair: 256), N=BN, K=16 into one of two TMEM
//              accumulators (2*BN columns), tcgen05.commit frees smem stages
//              and hands a finished accumulator to the epilogue (a pair: to
//              both CTAs; both CTAs' stage loads complete on rank 0's full
//              barriers, and rank 1's MMA warp has nothing to issue)
//   warps 2-9: epilogue: tcgen05.ld 32 columns at a time (warp w reads TMEM
//              lanes 32*(w%4).. and half of the tile's columns), fused
//              epilogue functor, global stores.  While they drain
//              accumulator i, the MMA warp fills the other.
// Epilogues that read a bf16 tile shaped like the output (the local stream X
// for injection, the direct gradient for dX) have it prefetched by TMA into
// shared memory (128 x BN, 128B-swizzled, 64-column boxes).  Unpaired ones get
//   warp 10  : X loader: refills each box for the next tile as soon as the
//              four epilogue warps of its column half are done with it, so
//              the load overlaps the rest of the tile instead of waiting for
//              the whole tile to drain (the single buffer has no room for a
//              second one next to the operand stages);
// paired ones (2D affine) load the whole tile at the start of its epilogue.
// Every mbarrier wait is bounded (common.cuh); on a timeout the kernel flags
// the error, drains its own copies and MMAs (bounded), frees TMEM and returns.
#pragma once

#include "common.cuh"

namespace pf {

constexpr int GEMM_BM = 128;
constexpr int GEMM_BK = 64;
constexpr int GEMM_EPI_WARPS = 8;  // two per TMEM lane quarter, each owning half the columns
constexpr int GEMM_THREADS = 64 + 32 * GEMM_EPI_WARPS;

// Unpaired X-tile epilogues run an X-loader warp after the epilogue warps.
template <class Epi>
struct GemmRoles {
  static constexpr bool kXLoader = Epi::kXTile && !Epi::kPaired;
  static constexpr int kThreads = GEMM_THREADS + (kXLoader ? 32 : 0);
};

// XCOLS: columns of the bf16 tile an epilogue prefetches (0: none).
// PAR: the epilogue stages one float4 of per-column parameters per output
// column in shared memory (two tiles' worth, filled one tile ahead).
// PAIR: the tile is shared by a CTA pair, each CTA staging half of B.
constexpr uint32_t GEMM_SMEM_MAX = 232448;  // dynamic shared memory per CTA (227 KB)
// SB: bytes of shared memory the epilogue stages its output in (0: none).
template <int BN, int XCOLS, bool PAR = false, bool PAIR = false, uint32_t SB = 0>
struct GemmCfg {
  static constexpr int B_ROWS = PAIR ? BN / 2 : BN;            // B rows staged by one CTA
  static constexpr uint32_t A_BYTES = GEMM_BM * GEMM_BK * 2;  // 16 KB
  static constexpr uint32_t B_BYTES = B_ROWS * GEMM_BK * 2;   // 16/32 KB
  static constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr uint32_t X_BYTES = GEMM_BM * XCOLS * 2;
  static constexpr uint32_t PAR_BYTES = PAR ? 2 * BN * 16 : 0;
  static constexpr uint32_t FIXED_BYTES =
      X_BYTES + 1024 /*align*/ + 256 /*barriers*/ + PAR_BYTES + SB;
  static constexpr int PAIR_STAGES = (int)((GEMM_SMEM_MAX - FIXED_BYTES) / STAGE_BYTES);
  static constexpr int TABLE_STAGES =
      PAIR ? 7
           : (XCOLS ? (BN == 256 && (XCOLS == 256 || PAR) ? 3 : (BN == 256 ? 4 : 5))
                    : (BN == 256 ? 4 : 6));
  static constexpr int STAGES = PAIR_STAGES < TABLE_STAGES ? PAIR_STAGES : TABLE_STAGES;
  static constexpr uint32_t SMEM_BYTES = STAGES * STAGE_BYTES + FIXED_BYTES;
  static_assert(SMEM_BYTES <= GEMM_SMEM_MAX, "shared memory");
  static_assert(2 * STAGES + 14 <= 31, "barrier region");
};

// Barrier of the epilogue threads (named barrier 1) that also ANDs a predicate
// across them, so that every epilogue thread takes the same branch.
__device__ __forceinline__ bool epi_bar_and(bool p) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred pi, po;\n\t"
      "setp.ne.u32 pi, %1, 0;\n\t"
      "bar.red.and.pred po, 1, %2, pi;\n\t"
      "selp.u32 %0, 1, 0, po;\n\t}"
      : "=r"(r)
      : "r"((uint32_t)p), "n"(32 * GEMM_EPI_WARPS)
      : "memory");
  return r != 0;
}

// 8 bf16 of row r, columns [c, c+8) of a 128 x BN tile stored as BN/64 boxes
// of 128 rows x 64 columns with 128-byte swizzle (TMA SWIZZLE_128B layout).
__device__ __forceinline__ void xtile_load8(const uint8_t* xt, int r, int c, float* v) {
  const uint8_t* p = xt + (c >> 6) * 16384 + r * 128 + ((((c & 63) >> 3) ^ (r & 7)) << 4);
  uint4 u = *reinterpret_cast<const uint4*>(p);
  float2 a = unpack_bf16(u.x), b = unpack_bf16(u.y), e = unpack_bf16(u.z), f = unpack_bf16(u.w);
  v[0] = a.x; v[1] = a.y; v[2] = b.x; v[3] = b.y; v[4] = e.x; v[5] = e.y; v[6] = f.x; v[7] = f.y;
}

// Address of 8 bf16 at row r, columns [c, c+8) of the swizzled tile above.
__device__ __forceinline__ uint8_t* xtile_ptr(uint8_t* xt, int r, int c) {
  return xt + (c >> 6) * 16384 + r * 128 + ((((c & 63) >> 3) ^ (r & 7)) << 4);
}

// Coalesced store of a warp's 32 rows x 32 columns (tile rows 32q.., tile
// columns cl..) that its threads have staged, one row each, in the swizzled
// tile: every store instruction writes 8 rows x 64 contiguous bytes.  dst(rr,
// p) returns the global address of row rr's 16-byte piece p (or null to skip);
// it is called by all lanes in step (it may shuffle).
template <class F>
__device__ __forceinline__ void warp_store_rows(uint8_t* xt, int q, int cl, F dst) {
  const int lane = threadIdx.x & 31, p = lane & 3;
#pragma unroll
  for (int it = 0; it < 4; ++it) {
    const int rr = it * 8 + (lane >> 2);
    bf16* g = dst(rr, p);
    const uint4 val = *reinterpret_cast<const uint4*>(xtile_ptr(xt, q * 32 + rr, cl + p * 8));
    if (g) *reinterpret_cast<uint4*>(g) = val;
  }
}

// Destinations of warp_store_rows' four store instructions for whole-row
// segments: this lane stores (in instruction it) for row 8 it + lane / 4 of
// the warp's 32 rows, whose element offset and valid column count are
// gathered here once per tile (not shuffled again for every chunk).
struct SegRows {
  long long off[4];
  int lim[4];
  __device__ __forceinline__ void gather(long long my_off, int my_lim) {
    const int src = (threadIdx.x & 31) >> 2;
#pragma unroll
    for (int it = 0; it < 4; ++it) {
      off[it] = __shfl_sync(0xffffffffu, my_off, it * 8 + src);
      lim[it] = __shfl_sync(0xffffffffu, my_lim, it * 8 + src);
    }
  }
};

__device__ __forceinline__ void xtile_put8(uint8_t* xt, int r, int c, const float* v) {
  *reinterpret_cast<uint4*>(xtile_ptr(xt, r, c)) =
      make_uint4(pack_bf16(v[0], v[1]), pack_bf16(v[2], v[3]), pack_bf16(v[4], v[5]),
                 pack_bf16(v[6], v[7]));
}

template <int BN, bool A_MN, bool B_MN, class Epi, bool PAIR = false>
__global__ void __launch_bounds__(GemmRoles<Epi>::kThreads, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmX, int M, int N, int K, int splits,
                   Epi epi) {
  static_assert(!PAIR || BN == 256, "CTA pairs use 256-wide tiles");
  constexpr int XCOLS = Epi::kXTile ? (Epi::kPaired ? BN / 2 : BN) : 0;
  using Cfg = GemmCfg<BN, XCOLS, Epi::kColPar, PAIR, Epi::kStageBytes>;
  constexpr int STAGES = Cfg::STAGES;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* xtile = smem + STAGES * Cfg::STAGE_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(xtile + Cfg::X_BYTES);
  // bars: full[S], empty[S], tfull[2], tempty[2], xfull, done, xbox_full[4],
  // xbox_empty[4]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * STAGES + 14);
  constexpr bool XL = GemmRoles<Epi>::kXLoader;
  constexpr int XBOXES = XCOLS / 64;       // 64-column boxes of the X tile
  constexpr int XB_HALF = XBOXES / 2;      // boxes per epilogue column half (XL)
  // column parameters (kColPar), [2 tiles][BN/4 groups][4 params] float4: the
  // float4 at (c / 4) * 4 + k holds parameter k of columns c & ~3 .. (c & ~3) + 3
  float4* cpar = reinterpret_cast<float4*>(xtile + Cfg::X_BYTES + 256);
  auto cpar_put = [&](int b, int col, float4 p) {
    float* f = reinterpret_cast<float*>(cpar + b * BN) + (col >> 2) * 16 + (col & 3);
    f[0] = p.x;
    f[4] = p.y;
    f[8] = p.z;
    f[12] = p.w;
  };
  __shared__ uint32_t s_consumed;
  // output staging of the epilogue warps (kStageBytes epilogues), after the
  // column parameters; other epilogues get the X tile
  uint8_t* const epi_smem =
      Epi::kStageBytes ? xtile + Cfg::X_BYTES + 256 + Cfg::PAR_BYTES : xtile;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // a pair (cluster of two CTAs) works on one tile of 2 x 128 rows: `unit` is
  // the pair (or the lone CTA), `rank` this CTA's half of the rows
  const uint32_t rank = PAIR ? cluster_ctarank() : 0u;
  const int unit = PAIR ? (int)(blockIdx.x >> 1) : (int)blockIdx.x;
  const int n_units = PAIR ? (int)(gridDim.x >> 1) : (int)gridDim.x;
  constexpr int TILE_M = PAIR ? 2 * GEMM_BM : GEMM_BM;
  const int num_n = (N + BN - 1) / BN, num_m = (M + TILE_M - 1) / TILE_M;
  const int mn_tiles = num_m * num_n;
  // N fastest keeps the co-running CTAs on one A panel with all of B in L2;
  // when A is a few row tiles and B is wider than the grid, M fastest instead
  // lets the co-running CTAs share each B tile (B is then read once)
  const bool m_fast = num_m <= 16 && num_n > n_units;
  const int tiles = mn_tiles * splits;
  const int num_k = (K + GEMM_BK - 1) / GEMM_BK;
  const int kps = (num_k + splits - 1) / splits;  // K tiles per split
  // tile t -> split t / mn_tiles (slowest), then M, then N (fastest); m0 is
  // this CTA's first row
#define PF_TILE_DECODE(t)                                                        \
  const int sp = (t) / mn_tiles, rem = (t) % mn_tiles;                           \
  const int m0 = (m_fast ? rem % num_m : rem / num_n) * TILE_M + (int)rank * GEMM_BM; \
  const int n0 = (m_fast ? rem / num_m : rem % num_n) * BN;                      \
  const int kb = sp * kps, ke = min(num_k, kb + kps);
  const uint32_t full0 = smem_u32(bars), empty0 = smem_u32(bars + STAGES);
  const uint32_t tfull0 = smem_u32(bars + 2 * STAGES), tempty0 = tfull0 + 16;
  const uint32_t xfull = tfull0 + 32, done = tfull0 + 40;
  const uint32_t xbf0 = tfull0 + 48, xbe0 = xbf0 + 32;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(tfull0 + 8 * b, 1);
      // one arrival per epilogue warp (of both CTAs of a pair, on rank 0)
      mbar_init(tempty0 + 8 * b, PAIR ? 2 * GEMM_EPI_WARPS : GEMM_EPI_WARPS);
    }
    mbar_init(xfull, 1);
    mbar_init(done, 1);
    for (int j = 0; j < 4; ++j) {
      mbar_init(xbf0 + 8 * j, 1);
      mbar_init(xbe0 + 8 * j, 4);  // the four epilogue warps of the box's column half
    }
    fence_barrier_init();
    s_consumed = 0;
  }
  if (warp == 1) {
    if (PAIR) {
      tmem_alloc_pair(smem_u32(tmem_slot), 2 * BN);
      tmem_relinquish_pair();
    } else {
      tmem_alloc(smem_u32(tmem_slot), 2 * BN);
      tmem_relinquish();
    }
  }
  tc_fence_before();
  __syncthreads();
  if (PAIR) cluster_sync_all();  // both CTAs' barriers exist before any remote arrival
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  uint32_t issued = 0;
  bool x_pending = false;
  uint32_t x_parity = 0;
  uint32_t xb_issued[4] = {0, 0, 0, 0};  // X loader: loads issued per box

  if (warp == 0 && lane == 0) {
    // ---------------------------------------------------------- producer
    prefetch_tmap(&tmA);
    prefetch_tmap(&tmB);
    // test hook: arm no stage and issue no load, so that nothing is ever in
    // flight and the MMA warp's first wait runs out
    const bool skip_loads = *(volatile int*)&g_debug_skip_loads != 0;
    uint32_t it = 0;
    bool ok = true;
    for (int tile = unit; tile < tiles && ok; tile += n_units) {
      PF_TILE_DECODE(tile)
      (void)sp;
      for (int kt = kb; kt < ke; ++kt, ++it) {
        const int s = it % STAGES;
        const uint32_t ph = (it / STAGES) & 1;
        if (!mbar_wait(empty0 + 8 * s, ph ^ 1)) {
          ok = false;
          break;
        }
        if (skip_loads) continue;
        // a pair: both CTAs' loads complete on rank 0's full barrier, which
        // rank 0 arms for the two CTAs' bytes
        const uint32_t fb = PAIR ? smem_map_rank(full0 + 8 * s, 0) : full0 + 8 * s;
        if (!PAIR || rank == 0)
          mbar_arrive_expect_tx(full0 + 8 * s, (PAIR ? 2u : 1u) * Cfg::STAGE_BYTES);
        auto ld = [&](uint32_t dst, const CUtensorMap* map, int c0, int c1) {
          if (PAIR)
            tma_load_2d_pair(dst, map, fb, c0, c1);
          else
            tma_load_2d(dst, map, fb, c0, c1);
        };
        const uint32_t a_dst = smem_u32(smem + s * Cfg::STAGE_BYTES);
        const uint32_t b_dst = a_dst + Cfg::A_BYTES;
        const int k0 = kt * GEMM_BK;
        if (!A_MN) {
          ld(a_dst, &tmA, k0, m0);
        } else {
          ld(a_dst, &tmA, m0, k0);
          ld(a_dst + 8192, &tmA, m0 + 64, k0);
        }
        // this CTA's B rows: all of them, or (a pair) its half of the columns
        if (!B_MN) {
          constexpr int JB = Cfg::B_ROWS / 128;
#pragma unroll
          for (int j = 0; j < JB; ++j)
            ld(b_dst + j * 16384, &tmB, k0, epi.b_row(n0, j + (int)rank * JB));
        } else {
          constexpr int JB = Cfg::B_ROWS / 64;
#pragma unroll
          for (int j = 0; j < JB; ++j)
            ld(b_dst + j * 8192, &tmB, n0 + 64 * (j + (int)rank * JB), k0);
        }
        issued = it + 1;
      }
    }
  } else if (warp == 1 && PAIR && rank == 1) {
    // rank 1 of a pair: rank 0 issues the MMAs for both CTAs
  } else if (warp == 1) {
    // ---------------------------------------------------------- MMA issuer
    // The whole warp runs the loop; one elected lane issues and commits.
    constexpr uint32_t idesc = idesc_bf16_f32(TILE_M, BN, A_MN ? 1 : 0, B_MN ? 1 : 0);
    uint32_t it = 0, lt = 0;
    bool ok = true;
    for (int tile = unit; tile < tiles && ok; tile += n_units, ++lt) {
      const uint32_t buf = lt & 1, use = lt >> 1;
      if (!mbar_wait_warp(tempty0 + 8 * buf, (use & 1) ^ 1)) break;
      tc_fence_after();
      const uint32_t d_tmem = tmem + buf * BN;
      PF_TILE_DECODE(tile)
      (void)sp;
      (void)m0;
      (void)n0;
      for (int kt = kb; kt < ke; ++kt, ++it) {
        const int s = it % STAGES;
        const uint32_t ph = (it / STAGES) & 1;
        if (!mbar_wait_warp(full0 + 8 * s, ph)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t a_base = smem_u32(smem + s * Cfg::STAGE_BYTES);
        const uint32_t b_base = a_base + Cfg::A_BYTES;
        if (elect_one()) {
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
            if (PAIR)
              tc_mma_f16_pair(d_tmem, ad, bd, idesc, (kt != kb || kk != 0) ? 1u : 0u);
            else
              tc_mma_f16(d_tmem, ad, bd, idesc, (kt != kb || kk != 0) ? 1u : 0u);
          }
          if (PAIR)
            tc_commit_pair(empty0 + 8 * s);
          else
            tc_commit(empty0 + 8 * s);
        }
        __syncwarp();
      }
      if (elect_one()) {
        if (PAIR)
          tc_commit_pair(tfull0 + 8 * buf);
        else
          tc_commit(tfull0 + 8 * buf);
      }
      __syncwarp();
    }
    if (lane == 0) s_consumed = it;
    if (elect_one()) {
      if (PAIR)
        tc_commit_pair(done);
      else
        tc_commit(done);
    }
    __syncwarp();
  } else if (XL && warp == 2 + GEMM_EPI_WARPS) {
    // ---------------------------------------------------------- X loader
    if (lane == 0) {
      prefetch_tmap(&tmX);
      uint32_t lt = 0;
      bool ok = true;
      for (int tile = unit; tile < tiles && ok; tile += n_units, ++lt) {
        PF_TILE_DECODE(tile)
        (void)sp;
        (void)kb;
        (void)ke;
        const int xr = epi.x_row(m0);
        // in the order the halves free them: box i of each half, then box i+1
        for (int i = 0; i < XB_HALF && ok; ++i) {
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const int j = h * XB_HALF + i;
            if (!mbar_wait(xbe0 + 8 * j, (lt & 1) ^ 1)) {
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(xbf0 + 8 * j, 16384);
            tma_load_2d(smem_u32(xtile) + j * 16384, &tmX, xbf0 + 8 * j, epi.x_col(n0, j), xr);
            xb_issued[j] = lt + 1;
          }
        }
      }
    }
  } else if (warp >= 2) {
    // ---------------------------------------------------------- epilogue
    const int et = threadIdx.x - 64;
    const int q = warp & 3;                               // TMEM lane quarter
    const int c_begin = ((warp - 2) >> 2) * (BN / 2);     // this warp's column half
    auto tile_n0 = [&](int t) {
      const int r = t % mn_tiles;
      return (m_fast ? r / num_m : r % num_n) * BN;
    };
    if constexpr (Epi::kColPar) {  // parameters of the first tile
      if (unit < tiles && et < BN) cpar_put(0, et, epi.col_param(tile_n0(unit), et));
      epi_bar_and(true);
    }
    uint32_t lt = 0;
    for (int tile = unit; tile < tiles; tile += n_units, ++lt) {
      PF_TILE_DECODE(tile)
      const bool no_k = ke <= kb;
      const uint32_t buf = lt & 1, use = lt >> 1;
      if (Epi::kXTile && !XL && et == 0) {
        mbar_arrive_expect_tx(xfull, Cfg::X_BYTES);
        const int xr = epi.x_row(m0);
#pragma unroll
        for (int j = 0; j < XCOLS / 64; ++j)
          tma_load_2d(smem_u32(xtile) + j * 16384, &tmX, xfull, epi.x_col(n0, j), xr);
        x_pending = true;
        x_parity = lt & 1;
      }
      // next tile's column parameters: loaded now, stored after this tile
      const int ntile = tile + n_units;
      float4 npar = make_float4(0.f, 0.f, 0.f, 0.f);
      if constexpr (Epi::kColPar)
        if (ntile < tiles && et < BN) npar = epi.col_param(tile_n0(ntile), et);
      const float4* cp = cpar + (lt & 1) * BN;
      bool ok = mbar_wait(tfull0 + 8 * buf, use & 1);
      tc_fence_after();
      if (Epi::kXTile && !XL) {
        mbar_wait(xfull, lt & 1);
        x_pending = false;
      }
      const int rl = q * 32 + lane;
      // split-K partial epilogues address row (split * M + row); -1 = out of range
      const int erow = Epi::kSplitRows ? (m0 + rl < M ? sp * M + m0 + rl : -1) : m0 + rl;
      const typename Epi::Row ri = epi.row_info(erow, n0);
      const uint32_t trow = tmem + buf * BN + ((uint32_t)(q * 32) << 16);
      if constexpr (Epi::kPaired) {
        // columns c and c + BN/2 belong together (e.g. s and t of one channel)
#pragma unroll 1
        for (int c = c_begin / 2; c < c_begin / 2 + BN / 4; c += 32) {
          float v[32], w[32];
          tmem_ld32(trow + (uint32_t)c, v);
          tmem_ld32(trow + (uint32_t)(c + BN / 2), w);
          if (no_k) {
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = w[i] = 0.f;
          }
          epi.apply_pair(ri, erow, n0, c, v, w, xtile, rl, cp);
        }
      } else {
        // 32-column chunks, the TMEM load of chunk i+1 in flight while chunk i
        // is processed
        constexpr int NCH = BN / 64;
        auto run = [&](uint32_t* r, int c) {
          if (no_k) {  // uniform: a split with no K blocks
#pragma unroll
            for (int i = 0; i < 32; ++i) r[i] = 0u;
          }
          float v[32];
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
          epi.apply(ri, erow, n0 + c, v, epi_smem, rl, c, cp);
        };
        uint32_t ra[32], rb[32];
        tmem_ld32_async(trow + (uint32_t)c_begin, ra);
        tmem_wait_ld(ra);
#pragma unroll 1
        for (int ci = 0; ci < NCH; ci += 2) {
          const int c = c_begin + ci * 32;
          const int xb = c >> 6;  // the X box of this chunk pair (XL)
          if (XL) ok = mbar_wait(xbf0 + 8 * xb, lt & 1) && ok;
          tmem_ld32_async(trow + (uint32_t)(c + 32), rb);
          run(ra, c);
          tmem_wait_ld(rb);
          if (ci + 2 < NCH) tmem_ld32_async(trow + (uint32_t)(c + 64), ra);
          run(rb, c + 32);
          if (XL) {  // this warp is done with the box: staging writes before the refill
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(xbe0 + 8 * xb);
          }
          if (ci + 2 < NCH) tmem_wait_ld(ra);
        }
      }
      if constexpr (Epi::kColPar)
        if (ntile < tiles && et < BN) cpar_put((lt + 1) & 1, et, npar);
      // staging writes into the X tile are ordered before the next tile's
      // TMA load of it
      if (Epi::kXTile && !XL) fence_proxy_async_smem();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (PAIR && rank == 1)
          mbar_arrive_remote(smem_map_rank(tempty0 + 8 * buf, 0));
        else
          mbar_arrive(tempty0 + 8 * buf);
      }
      // all epilogue threads are done with the X tile (free for the next
      // prefetch); leave together if any of them saw a wait run out
      if (!epi_bar_and(ok)) break;
    }
  }
  tc_fence_before();
  if (__syncthreads_or(*(volatile int*)&g_dev_error != 0)) {
    // error path: let in-flight TMA copies and MMAs land before TMEM/smem go.
    if (warp == 0 && lane == 0) {
      if (PAIR && rank == 1) {
        // its loads complete on rank 0's barriers: give them a bounded time
        // (far above a load's latency) to land before the CTA goes
        const unsigned long long t0 = globaltimer();
        while (globaltimer() - t0 < 50000ull) {
        }
      } else {
        for (uint32_t it = s_consumed; it < issued; ++it)
          mbar_wait_drain(full0 + 8 * (it % STAGES), (it / STAGES) & 1);
      }
    }
    if (warp == 2 && lane == 0 && x_pending) mbar_wait_drain(xfull, x_parity);
    if (XL && warp == 2 + GEMM_EPI_WARPS && lane == 0) {
      for (int j = 0; j < XBOXES; ++j)
        if (xb_issued[j]) mbar_wait_drain(xbf0 + 8 * j, (xb_issued[j] - 1) & 1);
    }
    if (warp == 1 && lane == 0) mbar_wait_drain(done, 0);
    __syncthreads();
  } else if (warp == 1 && lane == 0) {
    mbar_wait(done, 0);
  }
  __syncthreads();
  // a pair: neither CTA leaves (or frees TMEM) while the other may still use
  // its shared memory or TMEM
  if (PAIR) cluster_sync_all();
  if (warp == 1) {
    tc_fence_after();
    if (PAIR)
      tmem_dealloc_pair(tmem, 2 * BN);
    else
      tmem_dealloc(tmem, 2 * BN);
  }
}

// ------------------------------------------------------------------ epilogues
// row_info(row, n0) is evaluated once per tile and output row; apply(ri, row,
// col, v, xt, rl, cl) then receives 32 consecutive accumulator columns [col,
// col+32) of that row, with rl / cl the row and column inside the tile and xt
// the prefetched bf16 tile (kXTile epilogues: x_row(m0) / x_col(n0, j) give the
// coordinates of the tile's 64-column boxes in the X tensor map).  kPaired
// epilogues receive columns c and c + BN/2 together through apply_pair, and
// prefetch BN/2 columns.  b_row(n0, j) is the first row of B (K-major) loaded
// for 128-row box j of the tile starting at output column n0.  N is a
// multiple of 32.
struct EpiBase {
  static constexpr bool kXTile = false;
  static constexpr bool kPaired = false;
  static constexpr bool kSplitRows = false;
  static constexpr bool kColPar = false;
  // may run on CTA pairs (256-wide tiles with enough of them); an epilogue
  // slower than its mainloop does better on single CTAs, whose tiles do not
  // wait for the other CTA's epilogue
  static constexpr bool kPairs = true;
  // shared memory for staging the output (0: the epilogue stores from registers)
  static constexpr uint32_t kStageBytes = 0;
  __device__ __forceinline__ float4 col_param(int, int) const { return make_float4(0, 0, 0, 0); }
  __device__ __forceinline__ int x_row(int m0) const { return m0; }
  __device__ __forceinline__ int x_col(int n0, int j) const { return n0 + 64 * j; }
  __device__ __forceinline__ int b_row(int n0, int j) const { return n0 + 128 * j; }
  template <class R>
  __device__ __forceinline__ void apply_pair(const R&, int, int, int, float*, float*, uint8_t*,
                                             int, const float4*) const {}
};

// v = acc (+ bias[col]) (+ addend[row, col]); stored as fp32 and/or bf16.
struct EpiLinear : EpiBase {
  struct Row {
    bool ok;
  };
  int M, N;
  const float* bias;
  const float* addend;
  long ld_add;
  float* out_f32;
  long ld_f32;
  bf16* out_bf16;
  long ld_bf16;
  const bf16* add_bf16;
  long ld_add_bf16;
  int act_silu;
  bf16* pre_bf16;
  long ld_pre;
  const bf16* dsilu_of;
  long ld_dsilu;
  __device__ __forceinline__ Row row_info(int row, int) const { return Row{row < M}; }
  __device__ __forceinline__ void apply(const Row& ri, int row, int col, float* v, const uint8_t*,
                                        int, int, const float4*) const {
    if (!ri.ok || col >= N) return;
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
    if (add_bf16) {
      const bf16* a = add_bf16 + (long)row * ld_add_bf16 + col;
#pragma unroll
      for (int i = 0; i < 32; i += 8) {
        const uint4 u = *reinterpret_cast<const uint4*>(a + i);
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const float2 f = unpack_bf16(w[j]);
          v[i + 2 * j] += f.x;
          v[i + 2 * j + 1] += f.y;
        }
      }
    }
    if (pre_bf16) {
      bf16* o = pre_bf16 + (long)row * ld_pre + col;
#pragma unroll
      for (int i = 0; i < 32; i += 8) store8_bf16(o + i, v + i);
    }
    if (act_silu) {
#pragma unroll
      for (int i = 0; i < 32; ++i) v[i] = v[i] / (1.f + __expf(-v[i]));
    }
    if (dsilu_of) {
      const bf16* u = dsilu_of + (long)row * ld_dsilu + col;
#pragma unroll
      for (int i = 0; i < 32; i += 8) {
        const uint4 q = *reinterpret_cast<const uint4*>(u + i);
        const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const float2 f = unpack_bf16(w[j]);
          const float s0 = 1.f / (1.f + __expf(-f.x)), s1 = 1.f / (1.f + __expf(-f.y));
          v[i + 2 * j] *= s0 * (1.f + f.x * (1.f - s0));
          v[i + 2 * j + 1] *= s1 * (1.f + f.y * (1.f - s1));
        }
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

// A linear epilogue (v = acc + bias, fp32 and / or bf16 out) that stores
// whole rows: each warp stages its 32 x 32 chunk in shared memory (rows 36
// floats apart, so neither the row-per-lane writes nor the row reads conflict)
// and writes it back row by row, 128 contiguous bytes of fp32 per row.
// Used where the output is large next to the contraction (short K), so that
// the stores from one row per lane would bound the epilogue.
struct EpiLinearStaged : EpiBase {
  static constexpr int kRowF = 36;  // floats per staged row
  static constexpr uint32_t kStageBytes = GEMM_EPI_WARPS * 32 * kRowF * 4;
  struct Row {
    bool ok;
  };
  int M, N;
  const float* bias;
  float* out_f32;
  long ld_f32;
  bf16* out_bf16;
  long ld_bf16;
  __device__ __forceinline__ Row row_info(int row, int) const { return Row{row < M}; }
  __device__ __forceinline__ void apply(const Row&, int row, int col, float* v, uint8_t* stg,
                                        int rl, int, const float4*) const {
    if (col >= N) return;  // uniform across the warp
    const int lane = threadIdx.x & 31, ew = (threadIdx.x >> 5) - 2;
    float* s = reinterpret_cast<float*>(stg) + ew * (32 * kRowF);
    if (bias) {
#pragma unroll
      for (int i = 0; i < 32; i += 4) {
        const float4 b = *reinterpret_cast<const float4*>(bias + col + i);
        v[i] += b.x; v[i + 1] += b.y; v[i + 2] += b.z; v[i + 3] += b.w;
      }
    }
#pragma unroll
    for (int i = 0; i < 32; i += 4)
      *reinterpret_cast<float4*>(s + lane * kRowF + i) = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
    __syncwarp();
    const int rfirst = row - (rl & 31);
    if (out_f32) {  // 8 lanes per row, 4 rows per instruction
#pragma unroll
      for (int it = 0; it < 8; ++it) {
        const int rr = it * 4 + (lane >> 3), pc = (lane & 7) * 4;
        const float4 val = *reinterpret_cast<const float4*>(s + rr * kRowF + pc);
        if (rfirst + rr < M)
          *reinterpret_cast<float4*>(out_f32 + (long)(rfirst + rr) * ld_f32 + col + pc) = val;
      }
    }
    if (out_bf16) {  // 4 lanes per row (8 values each), 8 rows per instruction
#pragma unroll
      for (int it = 0; it < 4; ++it) {
        const int rr = it * 8 + (lane >> 2), pc = (lane & 3) * 8;
        const float4 a = *reinterpret_cast<const float4*>(s + rr * kRowF + pc);
        const float4 b = *reinterpret_cast<const float4*>(s + rr * kRowF + pc + 4);
        if (rfirst + rr < M)
          *reinterpret_cast<uint4*>(out_bf16 + (long)(rfirst + rr) * ld_bf16 + col + pc) =
              make_uint4(pack_bf16(a.x, a.y), pack_bf16(a.z, a.w), pack_bf16(b.x, b.y),
                         pack_bf16(b.z, b.w));
      }
    }
    __syncwarp();  // the staging is reused by the next chunk
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
// X is read from the prefetched tile: rows r + shift*k2 of the view
// [B*m*k2, k1*d] of X (zero-padded to whole blocks when L % P != 0).
struct EpiInject1D : EpiBase {
  static constexpr bool kXTile = true;
  static constexpr bool kPairs = false;  // epilogue-bound (measured slower on pairs)
  struct Row {
    bool ok;    // row < M
    long off0;  // element offset of the group's first token in X_out
    int lim;    // columns < lim belong to tokens < L of a target block
    SegRows seg;
  };
  int M, N;
  const float* bias;
  bf16* D_save;
  bf16* X_out;
  const float *w_x, *w_dlt, *b_g;
  int d, k1, k2, m, L, shift, gated;
  __device__ __forceinline__ int x_row(int m0) const { return m0 + shift * k2; }
  __device__ __forceinline__ Row row_info(int row, int) const {
    Row r{row < M, 0, 0};
    const int a = row % k2, prox = row / k2;
    const int b = prox / m, i = prox % m;
    const int it = i + shift;
    const long tok0 = (long)it * (k1 * k2) + (long)a * k1;
    if (r.ok && it < m && tok0 < L) {
      r.off0 = ((long)b * L + tok0) * d;
      const long lim = (L - tok0) * d;
      r.lim = lim < N ? (int)lim : N;
    }
    r.seg.gather(r.off0, r.ok ? r.lim : 0);
    return r;
  }
  // staged per column: (bias, w_x, w_dlt, b_g)
  static constexpr bool kColPar = true;
  __device__ __forceinline__ float4 col_param(int n0, int cl) const {
    const int col = n0 + cl;
    if (col >= N) return make_float4(0.f, 0.f, 0.f, 0.f);
    const float b = bias[col];
    if (!gated) return make_float4(b, 0.f, 0.f, 0.f);
    const int ch = col % d;
    return make_float4(b, w_x[ch], w_dlt[ch], b_g[ch]);
  }
  // The warp's 32 x 32 chunk of X_out and then of D is staged in the X tile
  // cells it has just read and stored with whole-row segments.  cp: the
  // staged parameters, one float4 per (4-column group, parameter).  The gate
  // arithmetic runs on column pairs with packed fp32x2 FMAs (each lane an
  // IEEE fp32 FMA, as the scalar form), and the cell addresses are formed
  // once per chunk.
  __device__ __forceinline__ void apply(const Row& ri, int row, int col, float* v, uint8_t* xt,
                                        int rl, int cl, const float4* cp) const {
    if (col >= N) return;  // uniform across the warp
    const int lane = threadIdx.x & 31, q = rl >> 5;
    const float4* cg = cp + (cl >> 2) * 4;
    // this row's four 16-byte cells of the chunk (128-byte swizzle)
    const int c8 = (cl & 63) >> 3, sw = rl & 7;
    uint8_t* const rowp = xt + (cl >> 6) * 16384 + rl * 128;
    uint4* cell[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) cell[j] = reinterpret_cast<uint4*>(rowp + (((c8 | j) ^ sw) << 4));
    uint32_t dpk[16];  // D = acc + bias, bf16 pairs
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const uint4 xu = *cell[j];
      const uint32_t xw[4] = {xu.x, xu.y, xu.z, xu.w};
      uint32_t ow[4];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int g4 = 2 * j + h;  // 4-column group of the chunk
        const float4 b = cg[g4 * 4];
        const float bb[4] = {b.x, b.y, b.z, b.w};
        float wx[4], wd[4], bg[4];
        if (gated) {
          const float4 a = cg[g4 * 4 + 1], dd = cg[g4 * 4 + 2], e = cg[g4 * 4 + 3];
          wx[0] = a.x; wx[1] = a.y; wx[2] = a.z; wx[3] = a.w;
          wd[0] = dd.x; wd[1] = dd.y; wd[2] = dd.z; wd[3] = dd.w;
          bg[0] = e.x; bg[1] = e.y; bg[2] = e.z; bg[3] = e.w;
        }
#pragma unroll
        for (int pr = 0; pr < 2; ++pr) {
          const int e0 = 8 * j + 4 * h + 2 * pr, k = 2 * pr;
          const float2 x2 = unpack_bf16(xw[2 * h + pr]);
          const float2 d2 = __fadd2_rn(make_float2(v[e0], v[e0 + 1]), make_float2(bb[k], bb[k + 1]));
          float2 o2;
          if (gated) {
            const float2 g2 = __ffma2_rn(make_float2(wx[k], wx[k + 1]), x2,
                                         __ffma2_rn(make_float2(wd[k], wd[k + 1]), d2,
                                                    make_float2(bg[k], bg[k + 1])));
            const float2 hg = __fmul2_rn(g2, make_float2(0.5f, 0.5f));
            const float2 t2 = make_float2(tanh_approx(hg.x), tanh_approx(hg.y));
            const float2 s2 = __ffma2_rn(make_float2(0.5f, 0.5f), t2, make_float2(0.5f, 0.5f));
            o2 = __ffma2_rn(s2, d2, x2);
          } else {
            o2 = __fadd2_rn(x2, d2);
          }
          ow[2 * h + pr] = pack_bf16(o2.x, o2.y);
          dpk[(e0 >> 1)] = pack_bf16(d2.x, d2.y);
        }
      }
      *cell[j] = make_uint4(ow[0], ow[1], ow[2], ow[3]);
    }
    __syncwarp();
    // whole-row stores: instruction it writes rows 8 it + lane / 4 of the warp,
    // 16-byte piece p = lane % 4; the swizzle phase of those rows is lane / 4
    const int p = lane & 3, rq = lane >> 2;
    const uint8_t* srow = xt + (cl >> 6) * 16384 + (q * 32 + rq) * 128 + (((c8 | p) ^ rq) << 4);
#pragma unroll
    for (int it = 0; it < 4; ++it) {
      const uint4 val = *reinterpret_cast<const uint4*>(srow + it * 8 * 128);
      if (col + p * 8 < ri.seg.lim[it])
        *reinterpret_cast<uint4*>(X_out + ri.seg.off[it] + col + p * 8) = val;
    }
    __syncwarp();
    if (D_save) {
#pragma unroll
      for (int j = 0; j < 4; ++j)
        *cell[j] = make_uint4(dpk[4 * j], dpk[4 * j + 1], dpk[4 * j + 2], dpk[4 * j + 3]);
      __syncwarp();
      const int rfirst = row - (rl & 31);
      bf16* dbase = D_save + (long)(rfirst + rq) * N + col + p * 8;
#pragma unroll
      for (int it = 0; it < 4; ++it) {
        const uint4 val = *reinterpret_cast<const uint4*>(srow + it * 8 * 128);
        if (rfirst + rq + 8 * it < M) *reinterpret_cast<uint4*>(dbase + (long)it * 8 * N) = val;
      }
      __syncwarp();
    }
  }
};

// First compression level's input gradient added to the direct injection
// gradient: rows r = (b*m + i)*k2 + a, columns (token c/d of the group, channel
// c%d) -> token i*P + a*k1 + c/d of sequence b.  The direct gradient is read
// from the prefetched tile of dXd, the view [B*m*k2, k1*d] of a buffer padded
// to whole blocks (dX itself when L % P == 0); the sum is written to dX.
struct EpiDX1D : EpiBase {
  static constexpr bool kXTile = true;
  struct Row {
    bool ok;
    long off0;
    int lim;
    SegRows seg;
  };
  int M, N;
  bf16* dX;
  int d, k1, k2, m, L;
  __device__ __forceinline__ Row row_info(int row, int) const {
    Row r{row < M, 0, 0};
    const int per_seq = m * k2;
    const int b = row / per_seq, rr = row % per_seq;
    const long tok0 = (long)rr * k1;
    if (r.ok && tok0 < L) {
      r.off0 = ((long)b * L + tok0) * d;
      const long lim = (L - tok0) * d;
      r.lim = lim < N ? (int)lim : N;
    }
    r.seg.gather(r.off0, r.ok ? r.lim : 0);
    return r;
  }
  // staged in the tile cells just read, stored with whole-row segments
  __device__ __forceinline__ void apply(const Row& ri, int, int col, float* v, uint8_t* xt,
                                        int rl, int cl, const float4*) const {
    if (col >= N) return;  // uniform across the warp
#pragma unroll
    for (int i8 = 0; i8 < 32; i8 += 8) {
      float x[8];
      xtile_load8(xt, rl, cl + i8, x);
#pragma unroll
      for (int j = 0; j < 8; ++j) x[j] += v[i8 + j];
      xtile_put8(xt, rl, cl + i8, x);
    }
    __syncwarp();
    warp_store_rows(xt, rl >> 5, cl, [&](int rr, int p) -> bf16* {
      const int it = rr >> 3;
      return col + p * 8 < ri.seg.lim[it] ? dX + ri.seg.off[it] + col + p * 8 : nullptr;
    });
    __syncwarp();
  }
};

// KV append (Sec. 3.8): rows are sequences b, columns [0, 2d) the proxy's key
// and value rows W_kh H and W_vh H, written as bf16 at cache row n_proxy[b] of
// the sequences whose open block is full and whose cache has room.
struct EpiAppendKV : EpiBase {
  struct Row {
    bool ok;
    long off;
  };
  int M, N;
  bf16 *K, *V;
  const int *n_open, *n_proxy;
  int d, P, cap;
  __device__ __forceinline__ Row row_info(int row, int) const {
    Row r{false, 0};
    if (row < M) {
      const int np = n_proxy[row];
      r.ok = n_open[row] == P && np >= 0 && np < cap;
      r.off = ((long)row * cap + (r.ok ? np : 0)) * d;
    }
    return r;
  }
  __device__ __forceinline__ void apply(const Row& ri, int, int col, float* v, const uint8_t*, int,
                                        int, const float4*) const {
    if (!ri.ok || col >= N) return;
    bf16* o = col < d ? K + ri.off + col : V + ri.off + (col - d);
#pragma unroll
    for (int i = 0; i < 32; i += 8) store8_bf16(o + i, v + i);
  }
};

// Decompression of the 2D layer fused with affine injection (Eq. inj-affine):
// X_out = (1 + s) * LayerNorm(X) + t.  GEMM rows are patches r = (b, by, bx);
// W_d1 [2*P*d, d] holds s for token p of a patch at rows [2pd, 2pd+d) and t at
// [2pd+d, 2(p+1)d).  Output tile n0 = 256*nt covers token p = nt / (d/128) and
// channels [cb, cb+128), cb = 128 * (nt % (d/128)): its B rows are loaded as
// s (columns 0..127) then t (128..255), so each thread holds matching s and t.
// X comes from the prefetched tile of the patch-ordered copy Xp [B*m, P*d];
// LayerNorm statistics per token from `stats` (mean, 1/std).  s is saved in
// patch order [B*m, P*d] for the backward.
struct EpiAffine2D : EpiBase {
  static constexpr bool kXTile = true;
  static constexpr bool kPaired = true;
  struct Row {
    bool ok;
    long xoff;  // element offset of (token, channel cb) in X_out
    float mu, rs;
    SegRows seg;  // X_out offsets of the rows this lane stores (lim 1: row exists)
  };
  int M;
  const float* bias;
  bf16* S_save;
  bf16* X_out;
  const float* stats;
  int d, patch, gh, gw, m;
  __device__ __forceinline__ int ptok(int n0) const { return n0 / (2 * d); }
  __device__ __forceinline__ int cbase(int n0) const { return ((n0 >> 8) % (d >> 7)) << 7; }
  __device__ __forceinline__ int b_row(int n0, int j) const {
    return ptok(n0) * 2 * d + j * d + cbase(n0);
  }
  __device__ __forceinline__ int x_col(int n0, int j) const {
    return ptok(n0) * d + cbase(n0) + 64 * j;
  }
  __device__ __forceinline__ Row row_info(int row, int n0) const {
    Row r{row < M, 0, 0.f, 0.f};
    if (r.ok) {
      const int npw = gw / patch;
      const int b = row / m, pr = row % m, by = pr / npw, bx = pr % npw;
      const int p = ptok(n0), py = p / patch, px = p % patch;
      const long tok = (long)b * gh * gw + (long)(by * patch + py) * gw + bx * patch + px;
      r.xoff = tok * d + cbase(n0);
      r.mu = stats[2 * tok];
      r.rs = stats[2 * tok + 1];
    }
    r.seg.gather(r.xoff, r.ok ? 1 : 0);
    return r;
  }
  // staged per column c of the s half: (bias of s, bias of t)
  static constexpr bool kColPar = true;
  __device__ __forceinline__ float4 col_param(int n0, int cl) const {
    if (cl >= 128) return make_float4(0.f, 0.f, 0.f, 0.f);
    const float* bs = bias + (long)ptok(n0) * 2 * d + cbase(n0) + cl;
    return make_float4(bs[0], bs[d], 0.f, 0.f);
  }
  // The warp's 32 x 32 chunk of X_out and then of S is staged in the X tile
  // cells it has just read and stored with whole-row segments.
  __device__ __forceinline__ void apply_pair(const Row& ri, int row, int n0, int c, float* vs,
                                             float* vt, uint8_t* xt, int rl,
                                             const float4* cp) const {
    const int q = rl >> 5, p = ptok(n0), ch0 = cbase(n0) + c;
    const float4* cg = cp + (c >> 2) * 4;
#pragma unroll
    for (int i8 = 0; i8 < 32; i8 += 8) {
      float x[8], o[8];
      xtile_load8(xt, rl, c + i8, x);
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int g4 = (i8 >> 2) + h;
        const float4 bs = cg[g4 * 4], bt = cg[g4 * 4 + 1];
        const float bsa[4] = {bs.x, bs.y, bs.z, bs.w}, bta[4] = {bt.x, bt.y, bt.z, bt.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const int e = h * 4 + j;
          const float sv = vs[i8 + e] + bsa[j];
          vs[i8 + e] = sv;
          o[e] = fmaf(1.f + sv, (x[e] - ri.mu) * ri.rs, vt[i8 + e] + bta[j]);
        }
      }
      xtile_put8(xt, rl, c + i8, o);
    }
    __syncwarp();
    warp_store_rows(xt, q, c, [&](int rr, int pc) -> bf16* {
      const int it = rr >> 3;
      return ri.seg.lim[it] ? X_out + ri.seg.off[it] + c + pc * 8 : nullptr;
    });
    __syncwarp();
#pragma unroll
    for (int i8 = 0; i8 < 32; i8 += 8) xtile_put8(xt, rl, c + i8, vs + i8);
    __syncwarp();
    const int rfirst = row - (rl & 31);
    const long pd = (long)patch * patch * d;
    warp_store_rows(xt, q, c, [&](int rr, int pc) -> bf16* {
      const int r2 = rfirst + rr;
      return r2 < M ? S_save + (long)r2 * pd + (long)p * d + ch0 + pc * 8 : nullptr;
    });
    __syncwarp();
  }
};

// Compression input gradient of the 2D layer: rows are patches, columns
// (token p = c / d of the patch, channel c % d); the direct gradient comes from
// the prefetched tile of dXd (same patch order) and the sum is written to dX
// at the token's raster position.
struct EpiDX2D : EpiBase {
  static constexpr bool kXTile = true;
  struct Row {
    bool ok;
    long base;  // offset of the patch's top-left token in dX
    SegRows seg;
  };
  int M, N;
  bf16* dX;
  int d, patch, gh, gw, m;
  __device__ __forceinline__ Row row_info(int row, int) const {
    Row r{row < M, 0};
    if (r.ok) {
      const int npw = gw / patch;
      const int b = row / m, pr = row % m, by = pr / npw, bx = pr % npw;
      r.base = ((long)b * gh * gw + (long)by * patch * gw + bx * patch) * d;
    }
    r.seg.gather(r.base, r.ok ? N : 0);
    return r;
  }
  // staged in the tile cells just read, stored with whole-row segments: a
  // 32-column chunk is 32 channels of one token of the patch (d is a multiple
  // of 32), 64 contiguous bytes of dX per row
  __device__ __forceinline__ void apply(const Row& ri, int, int col, float* v, uint8_t* xt,
                                        int rl, int cl, const float4*) const {
    if (col >= N) return;  // uniform across the warp
#pragma unroll
    for (int i8 = 0; i8 < 32; i8 += 8) {
      float x[8];
      xtile_load8(xt, rl, cl + i8, x);
#pragma unroll
      for (int j = 0; j < 8; ++j) x[j] += v[i8 + j];
      xtile_put8(xt, rl, cl + i8, x);
    }
    __syncwarp();
    const int p = col / d, ch = col - p * d, py = p / patch, px = p - py * patch;
    const long colofs = ((long)py * gw + px) * d + ch;
    warp_store_rows(xt, rl >> 5, cl, [&](int rr, int q) -> bf16* {
      const int it = rr >> 3;
      return col + q * 8 < ri.seg.lim[it] ? dX + ri.seg.off[it] + colofs + q * 8 : nullptr;
    });
    __syncwarp();
  }
};

// Split-K partial: raw fp32 accumulator of split s written to
// part[(s * M + row) * N + col]; a reduce kernel applies the linear epilogue.
struct EpiPartial : EpiBase {
  static constexpr bool kSplitRows = true;
  struct Row {
    long off;
  };
  int N;
  float* part;
  __device__ __forceinline__ Row row_info(int erow, int) const {
    return Row{erow < 0 ? -1L : (long)erow * N};
  }
  __device__ __forceinline__ void apply(const Row& ri, int, int col, float* v, const uint8_t*, int,
                                        int, const float4*) const {
    if (ri.off < 0 || col >= N) return;
    float* o = part + ri.off + col;
#pragma unroll
    for (int i = 0; i < 32; i += 4)
      *reinterpret_cast<float4*>(o + i) = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
  }
};

}  // namespace pf
