// Bandwidth-bound kernels of the layer: injection backward with its column
// reductions, deterministic column sums (bias gradients), block-0 copies and
// zero padding.  All accesses are 16-byte vectors over contiguous rows.
#include <algorithm>

#include "kernels.h"

namespace pf {

namespace {

constexpr int EW_THREADS = 256;

__global__ void copy_block0_kernel(const bf16* __restrict__ src, long Ls, bf16* __restrict__ dst,
                                   long Ld, int d, long per_seq_vec) {
  const long i = (long)blockIdx.x * blockDim.x + threadIdx.x;
  const int b = blockIdx.y;
  if (i >= per_seq_vec) return;
  *reinterpret_cast<uint4*>(dst + (long)b * Ld * d + i * 8) =
      *reinterpret_cast<const uint4*>(src + (long)b * Ls * d + i * 8);
}

__global__ void pad_rows_kernel(const bf16* __restrict__ src, bf16* __restrict__ dst, long L,
                                long Lp, int d) {
  const long i = (long)blockIdx.x * blockDim.x + threadIdx.x;  // vector index in [Lp*d/8]
  const int b = blockIdx.y;
  if (i >= Lp * d / 8) return;
  const long tok = i * 8 / d;
  uint4 v = make_uint4(0, 0, 0, 0);
  if (tok < L) v = *reinterpret_cast<const uint4*>(src + (long)b * L * d + i * 8);
  *reinterpret_cast<uint4*>(dst + (long)b * Lp * d + i * 8) = v;
}

// Each thread owns 8 consecutive columns (16-byte vectors) and walks a
// contiguous chunk of rows, INJ_U rows at a time with their loads issued
// together (kept packed until used); the row -> (sequence, proxy, group)
// indices advance incrementally, without divisions.
constexpr int INJ_COLS = 8;
constexpr int INJ_U = 2;

struct RowIdx {  // row r = (b*m + i)*k2 + grp
  int b, i, grp;
  __device__ __forceinline__ void next(int k2, int m) {
    if (++grp == k2) {
      grp = 0;
      if (++i == m) {
        i = 0;
        ++b;
      }
    }
  }
};

__global__ void __launch_bounds__(EW_THREADS, 2) inj_bwd_kernel(InjBwdArgs a, float* __restrict__ part,
                                                                long M, int N, long rows_per_chunk) {
  const int col = (blockIdx.x * EW_THREADS + threadIdx.x) * INJ_COLS;
  if (col >= N) return;
  const bf16* __restrict__ G = a.G;
  const bf16* __restrict__ X = a.X;
  const bf16* __restrict__ D = a.D;
  bf16* __restrict__ dD = a.dD;
  bf16* __restrict__ dX = a.dX;
  const long r0 = (long)blockIdx.y * rows_per_chunk;
  const long r1 = min(M, r0 + rows_per_chunk);
  const int P = a.k1 * a.k2;
  const int ch = col % a.d, tq = col / a.d;
  float wx[8], wd[8], bg[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    wx[j] = a.gated ? a.w_x[ch + j] : 0.f;
    wd[j] = a.gated ? a.w_dlt[ch + j] : 0.f;
    bg[j] = a.gated ? a.b_g[ch + j] : 0.f;
  }
  RowIdx ix;
  {
    const long prox = r0 / a.k2;
    ix.grp = (int)(r0 % a.k2);
    ix.b = (int)(prox / a.m);
    ix.i = (int)(prox % a.m);
  }
  float acc[4][8] = {};
  for (long rb = r0; rb < r1; rb += INJ_U) {
    uint4 gv[INJ_U], xv[INJ_U], dv[INJ_U];
    long offx[INJ_U];
    bool valid[INJ_U];
#pragma unroll
    for (int u = 0; u < INJ_U; ++u) {
      const long r = rb + u;
      const int it = ix.i + a.shift;
      const long tok = (long)it * P + (long)ix.grp * a.k1 + tq;
      valid[u] = r < r1 && it < a.m && tok < a.L;
      offx[u] = ((long)ix.b * a.Ldx + tok) * a.d + ch;
      if (valid[u]) {
        const long off = ((long)ix.b * a.L + tok) * a.d + ch;
        gv[u] = *reinterpret_cast<const uint4*>(G + off);
        xv[u] = *reinterpret_cast<const uint4*>(X + off);
        dv[u] = *reinterpret_cast<const uint4*>(D + r * N + col);
      }
      ix.next(a.k2, a.m);
    }
#pragma unroll
    for (int u = 0; u < INJ_U; ++u) {
      const long r = rb + u;
      if (r >= r1) break;
      float dd[8];
      if (valid[u]) {
        float g[8], x[8], Dv[8], dx[8];
        const uint32_t* pg = &gv[u].x;
        const uint32_t* px = &xv[u].x;
        const uint32_t* pd = &dv[u].x;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float2 a2 = unpack_bf16(pg[q]), b2 = unpack_bf16(px[q]), c2 = unpack_bf16(pd[q]);
          g[2 * q] = a2.x; g[2 * q + 1] = a2.y;
          x[2 * q] = b2.x; x[2 * q + 1] = b2.y;
          Dv[2 * q] = c2.x; Dv[2 * q + 1] = c2.y;
        }
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          if (a.gated) {
            const float sg = sigmoidf_(fmaf(wx[j], x[j], fmaf(wd[j], Dv[j], bg[j])));
            const float ds = g[j] * Dv[j] * sg * (1.f - sg);
            dx[j] = fmaf(ds, wx[j], g[j]);
            dd[j] = fmaf(g[j], sg, ds * wd[j]);
            acc[1][j] = fmaf(ds, x[j], acc[1][j]);
            acc[2][j] = fmaf(ds, Dv[j], acc[2][j]);
            acc[3][j] += ds;
          } else {
            dx[j] = g[j];
            dd[j] = g[j];
          }
        }
        store8_bf16(dX + offx[u], dx);
      } else {
#pragma unroll
        for (int j = 0; j < 8; ++j) dd[j] = 0.f;
      }
      // round dD once; the column sum uses the same rounded values the
      // downstream GEMMs see.
      uint4 o;
      o.x = pack_bf16(dd[0], dd[1]);
      o.y = pack_bf16(dd[2], dd[3]);
      o.z = pack_bf16(dd[4], dd[5]);
      o.w = pack_bf16(dd[6], dd[7]);
      *reinterpret_cast<uint4*>(dD + r * N + col) = o;
      const uint32_t* po = &o.x;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float2 f = unpack_bf16(po[q]);
        acc[0][2 * q] += f.x;
        acc[0][2 * q + 1] += f.y;
      }
    }
  }
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    float* p = part + ((long)blockIdx.y * 4 + q) * N + col;
    *reinterpret_cast<float4*>(p) = make_float4(acc[q][0], acc[q][1], acc[q][2], acc[q][3]);
    *reinterpret_cast<float4*>(p + 4) = make_float4(acc[q][4], acc[q][5], acc[q][6], acc[q][7]);
  }
}

// Streaming form for slices of IB_W columns (N a multiple of IB_W): two
// 256-thread CTAs per SM, each owning one column slice and a contiguous range
// of rows;
// thread 0 pulls each row's slices of D, G and X (contiguous, 4 KB each) with
// cp.async.bulk into an IB_STAGES-deep ring of IB_R-row stages, so the bytes
// in flight per SM do not depend on registers.  Thread t handles columns
// [8t, 8t+8) of the slice; the arithmetic and the partial sums are those of
// inj_bwd_kernel.
constexpr int IB_W = 2048;
constexpr int IB_R = 2;
constexpr int IB_STAGES = 4;
constexpr uint32_t IB_ROW_BYTES = IB_W * 2;
constexpr uint32_t IB_STAGE_BYTES = 3 * IB_R * IB_ROW_BYTES;  // [D | G | X] x IB_R rows
constexpr uint32_t IB_SMEM = IB_STAGES * IB_STAGE_BYTES + 128;

struct IbRow {
  bool valid;   // the row has target tokens
  int lim;      // valid columns of the row (tokens < L), 0 if none
  long gx_off;  // element offset of the row's tokens in G / X
  long dx_off;  // element offset in dX
};

__device__ __forceinline__ IbRow ib_row(const InjBwdArgs& a, const RowIdx& ix, int N) {
  IbRow r{false, 0, 0, 0};
  const int it = ix.i + a.shift;
  const long tok0 = (long)it * (a.k1 * a.k2) + (long)ix.grp * a.k1;
  if (it < a.m && tok0 < a.L) {
    r.valid = true;
    const long lim = (a.L - tok0) * a.d;
    r.lim = lim < N ? (int)lim : N;
    r.gx_off = ((long)ix.b * a.L + tok0) * a.d;
    r.dx_off = ((long)ix.b * a.Ldx + tok0) * a.d;
  }
  return r;
}

__global__ void __launch_bounds__(256, 2) inj_bwd_stream_kernel(InjBwdArgs a,
                                                               float* __restrict__ part, long M,
                                                               int N, long rows_per_chunk) {
  extern __shared__ __align__(128) uint8_t ib_smem[];
  __shared__ __align__(8) uint64_t full[IB_STAGES];
  const int tid = threadIdx.x;
  const int col0 = blockIdx.x * IB_W, col = col0 + tid * 8;
  const long r0 = (long)blockIdx.y * rows_per_chunk;
  const long r1 = min(M, r0 + rows_per_chunk);
  const int nst = (int)((max(r1 - r0, 0L) + IB_R - 1) / IB_R);
  const uint32_t sm0 = smem_u32(ib_smem), bar0 = smem_u32(full);
  RowIdx ix0;
  {
    const long prox = r0 / a.k2;
    ix0.grp = (int)(r0 % a.k2);
    ix0.b = (int)(prox / a.m);
    ix0.i = (int)(prox % a.m);
  }
  if (tid == 0) {
    for (int i = 0; i < IB_STAGES; ++i) mbar_init(bar0 + 8 * i, 1);
    fence_barrier_init();
  }
  __syncthreads();
  // producer state (thread 0): next stage to issue and the row index there
  int issued = 0;
  RowIdx pix = ix0;
  auto issue = [&]() {
    const int st = issued % IB_STAGES;
    const uint32_t base = sm0 + st * IB_STAGE_BYTES, bar = bar0 + 8 * st;
    const long rs = r0 + (long)issued * IB_R;
    uint32_t bytes = 0;
    uint32_t dbytes[IB_R], gbytes[IB_R];
    long goff[IB_R];
    for (int u = 0; u < IB_R; ++u) {
      dbytes[u] = gbytes[u] = 0;
      goff[u] = 0;
      if (rs + u < r1) {
        dbytes[u] = IB_ROW_BYTES;
        const IbRow rr = ib_row(a, pix, N);
        if (rr.valid && rr.lim > col0) {
          gbytes[u] = (uint32_t)(min(rr.lim - col0, IB_W)) * 2u;
          goff[u] = rr.gx_off + col0;
        }
        pix.next(a.k2, a.m);
      }
      bytes += dbytes[u] + 2 * gbytes[u];
    }
    mbar_arrive_expect_tx(bar, bytes);
    for (int u = 0; u < IB_R; ++u) {
      if (dbytes[u])
        bulk_load(base + u * IB_ROW_BYTES, a.D + (rs + u) * N + col0, dbytes[u], bar);
      if (gbytes[u]) {
        bulk_load(base + (IB_R + u) * IB_ROW_BYTES, a.G + goff[u], gbytes[u], bar);
        bulk_load(base + (2 * IB_R + u) * IB_ROW_BYTES, a.X + goff[u], gbytes[u], bar);
      }
    }
    ++issued;
  };
  if (tid == 0)
    while (issued < min(IB_STAGES, nst)) issue();

  const int ch = col % a.d;
  float wx[8], wd[8], bg[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    wx[j] = a.gated ? a.w_x[ch + j] : 0.f;
    wd[j] = a.gated ? a.w_dlt[ch + j] : 0.f;
    bg[j] = a.gated ? a.b_g[ch + j] : 0.f;
  }
  float acc[4][8] = {};
  RowIdx ix = ix0;
  bool failed = false;
  int s = 0;
  for (; s < nst; ++s) {
    const int st = s % IB_STAGES;
    const bool ok = mbar_wait(bar0 + 8 * st, (s / IB_STAGES) & 1);
    const uint8_t* base = ib_smem + st * IB_STAGE_BYTES + tid * 16;
    const long rs = r0 + (long)s * IB_R;
#pragma unroll
    for (int u = 0; u < IB_R; ++u) {
      const long r = rs + u;
      if (r >= r1) break;
      const IbRow rr = ib_row(a, ix, N);
      ix.next(a.k2, a.m);
      if (!ok) continue;
      const bool v = rr.valid && col < rr.lim;
      float dd[8];
      if (v) {
        const uint4 gv = *reinterpret_cast<const uint4*>(base + (IB_R + u) * IB_ROW_BYTES);
        const uint4 xv = *reinterpret_cast<const uint4*>(base + (2 * IB_R + u) * IB_ROW_BYTES);
        const uint4 dv = *reinterpret_cast<const uint4*>(base + u * IB_ROW_BYTES);
        float g[8], x[8], Dv[8], dx[8];
        const uint32_t *pg = &gv.x, *px = &xv.x, *pd = &dv.x;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float2 a2 = unpack_bf16(pg[q]), b2 = unpack_bf16(px[q]), c2 = unpack_bf16(pd[q]);
          g[2 * q] = a2.x; g[2 * q + 1] = a2.y;
          x[2 * q] = b2.x; x[2 * q + 1] = b2.y;
          Dv[2 * q] = c2.x; Dv[2 * q + 1] = c2.y;
        }
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          if (a.gated) {
            const float sg = sigmoidf_(fmaf(wx[j], x[j], fmaf(wd[j], Dv[j], bg[j])));
            const float ds = g[j] * Dv[j] * sg * (1.f - sg);
            dx[j] = fmaf(ds, wx[j], g[j]);
            dd[j] = fmaf(g[j], sg, ds * wd[j]);
            acc[1][j] = fmaf(ds, x[j], acc[1][j]);
            acc[2][j] = fmaf(ds, Dv[j], acc[2][j]);
            acc[3][j] += ds;
          } else {
            dx[j] = g[j];
            dd[j] = g[j];
          }
        }
        store8_bf16(a.dX + rr.dx_off + col, dx);
      } else {
#pragma unroll
        for (int j = 0; j < 8; ++j) dd[j] = 0.f;
      }
      uint4 o;
      o.x = pack_bf16(dd[0], dd[1]);
      o.y = pack_bf16(dd[2], dd[3]);
      o.z = pack_bf16(dd[4], dd[5]);
      o.w = pack_bf16(dd[6], dd[7]);
      *reinterpret_cast<uint4*>(a.dD + r * N + col) = o;
      const uint32_t* po = &o.x;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float2 f = unpack_bf16(po[q]);
        acc[0][2 * q] += f.x;
        acc[0][2 * q + 1] += f.y;
      }
    }
    // every thread is done with stage st: refill it (or leave together)
    if (__syncthreads_or(!ok)) {
      failed = true;
      break;
    }
    if (tid == 0 && issued < nst) issue();
  }
  if (failed) {  // a wait ran out: let this CTA's own copies land, then leave
    if (tid == 0)
      for (int it = s; it < issued; ++it)
        mbar_wait_drain(bar0 + 8 * (it % IB_STAGES), (it / IB_STAGES) & 1);
    __syncthreads();
    return;
  }
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    float* p = part + ((long)blockIdx.y * 4 + q) * N + col;
    *reinterpret_cast<float4*>(p) = make_float4(acc[q][0], acc[q][1], acc[q][2], acc[q][3]);
    *reinterpret_cast<float4*>(p + 4) = make_float4(acc[q][4], acc[q][5], acc[q][6], acc[q][7]);
  }
}

// Deterministic warp sum: lane j adds summands j, j+32, ... in order, then a
// fixed xor-shuffle tree.
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int s = 16; s > 0; s >>= 1) v += __shfl_xor_sync(0xffffffffu, v, s);
  return v;
}

// Column totals of the partials, one thread per (quantity q, column), chunks
// added in order (coalesced across threads): q = 0 gives db_d1; the totals of
// q = 1..3 are left in chunk 0's slots of part for the gate reduction below.
__global__ void inj_bwd_colsum_kernel(float* __restrict__ part, int n_chunks, int N,
                                      float* __restrict__ db_d1, int gates) {
  const long i = (long)blockIdx.x * blockDim.x + threadIdx.x;
  const int nq = gates ? 4 : 1;
  if (i >= (long)nq * N) return;
  const int q = (int)(i / N), col = (int)(i % N);
  float s = 0.f;
#pragma unroll 8
  for (int c = 0; c < n_chunks; ++c) s += part[((long)c * 4 + q) * N + col];
  if (q == 0)
    db_d1[col] = s;
  else
    part[(long)q * N + col] = s;
}

// Gate gradients: g_q[ch] = sum over the k1 token positions t of the column
// totals of quantity q (q = 1: w_x, 2: w_dlt, 3: b_g).
__global__ void inj_bwd_gates_kernel(const float* __restrict__ part, int N, int d, float* gw_x,
                                     float* gw_dlt, float* gb_g) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= 3 * d) return;
  const int q = 1 + i / d, ch = i % d, T = N / d;
  float s = 0.f;
  for (int t = 0; t < T; ++t) s += part[(long)q * N + (long)t * d + ch];
  (q == 1 ? gw_x : (q == 2 ? gw_dlt : gb_g))[ch] = s;
}

template <typename T>
__device__ __forceinline__ void load8(const T* p, float* v);
template <>
__device__ __forceinline__ void load8<bf16>(const bf16* p, float* v) {
  load8_bf16(p, v);
}
template <>
__device__ __forceinline__ void load8<float>(const float* p, float* v) {
  const float4 a = *reinterpret_cast<const float4*>(p), b = *reinterpret_cast<const float4*>(p + 4);
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}

// Column sums of an [R, C] matrix (C a multiple of 8), pass 1: CTA (x, y)
// adds rows chunk y of the CG * 8 columns from x * CG * 8 on.  Thread t reads
// 8 columns (16 or 32 bytes) of every 256 / CG-th row from row (t / CG), so
// a warp reads whole row segments; the 256 / CG row lanes are then added in
// lane order through shared memory.  CG: the smallest power of two of
// 8-column groups covering C, at most 32.
template <typename T>
__global__ void __launch_bounds__(EW_THREADS) colsum_part_kernel(const T* __restrict__ X, long R,
                                                                 int C, int CG, long rows_per_chunk,
                                                                 float* __restrict__ part) {
  __shared__ float s_acc[EW_THREADS * 8];
  const int RL = EW_THREADS / CG, cg = threadIdx.x % CG, rl = threadIdx.x / CG;
  const int col = (blockIdx.x * CG + cg) * 8;
  const long r0 = (long)blockIdx.y * rows_per_chunk, r1 = min(R, r0 + rows_per_chunk);
  float acc[8] = {};
  if (col < C) {
    long r = r0 + rl;
#pragma unroll 1
    for (; r + 3 * RL < r1; r += 4 * RL) {  // four rows' loads in flight
      float v[4][8];
#pragma unroll
      for (int u = 0; u < 4; ++u) load8<T>(X + (r + u * RL) * C + col, v[u]);
#pragma unroll
      for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[j] += v[u][j];
    }
    for (; r < r1; r += RL) {
      float v[8];
      load8<T>(X + r * C + col, v);
#pragma unroll
      for (int j = 0; j < 8; ++j) acc[j] += v[j];
    }
  }
#pragma unroll
  for (int j = 0; j < 8; ++j) s_acc[rl * CG * 8 + cg * 8 + j] = acc[j];
  __syncthreads();
  const int c = threadIdx.x;  // one column of the CTA's CG * 8 per thread
  const int gcol = blockIdx.x * CG * 8 + c;
  if (c < CG * 8 && gcol < C) {
    float t = 0.f;
    for (int l = 0; l < RL; ++l) t += s_acc[l * CG * 8 + c];
    part[(long)blockIdx.y * C + gcol] = t;
  }
}

// Pass 2: block = 32 consecutive columns x CS_WARPS warps; warp w adds chunks
// w, w + CS_WARPS, ... of its lane's column (a chunk row is one 128-byte
// segment per warp), then the warp totals are added in warp order.
constexpr int CS_WARPS = 16;
__global__ void __launch_bounds__(32 * CS_WARPS)
    colsum_final_kernel(const float* __restrict__ part, int n_chunks, int C,
                        float* __restrict__ out) {
  __shared__ float s_w[CS_WARPS][32];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int col = blockIdx.x * 32 + lane;
  float a = 0.f;
  if (col < C)
    for (int c = w; c < n_chunks; c += CS_WARPS) a += part[(long)c * C + col];
  s_w[w][lane] = a;
  __syncthreads();
  if (w == 0 && col < C) {
    float t = 0.f;
#pragma unroll
    for (int k = 0; k < CS_WARPS; ++k) t += s_w[k][lane];
    out[col] = t;
  }
}

// Row chunks of a column reduction: about 1024 CTAs in total, independent of
// the device so that results (summation order) and workspace sizes are fixed.
int chunks_for(long R, int C) {
  const int gx = (C / 8 + EW_THREADS - 1) / EW_THREADS;
  long want = (1024 + gx - 1) / gx;
  if (want > R) want = R;
  if (want < 1) want = 1;
  return (int)want;
}

// 8-column groups per column-sum CTA (a power of two, at most 32).
int colsum_groups(int C) {
  int cg = 1;
  while (cg < 32 && cg * 8 < C) cg *= 2;
  return cg;
}

// Row chunks of a column sum: about 1216 CTAs in all (eight per SM of a
// 152-SM part) with at least 64 rows each, independent of the device so that
// the summation order and the workspace size are fixed.
int colsum_chunks(long R, int C) {
  const int gx = (C + colsum_groups(C) * 8 - 1) / (colsum_groups(C) * 8);
  long want = (1216 + gx - 1) / gx;
  want = std::min(want, (R + 63) / 64);
  return (int)std::max(want, 1L);
}

template <typename T>
cudaError_t colsum_impl(const T* X, long R, int C, float* out, float* part, cudaStream_t st) {
  if (C % 8 != 0) return cudaErrorInvalidValue;
  if (R < 1) return cudaMemsetAsync(out, 0, (size_t)C * sizeof(float), st);  // an empty sum
  const int cg = colsum_groups(C), nc = colsum_chunks(R, C);
  const long rpc = (R + nc - 1) / nc;
  dim3 grid((C + cg * 8 - 1) / (cg * 8), nc);
  {
    LaunchTimer lt("colsum", st, (double)R * C, (double)R * C * sizeof(T));
    colsum_part_kernel<T><<<grid, EW_THREADS, 0, st>>>(X, R, C, cg, rpc, part);
  }
  {
    LaunchTimer lt("colsum_final", st, (double)nc * C, 4.0 * nc * C);
    colsum_final_kernel<<<(C + 31) / 32, 32 * CS_WARPS, 0, st>>>(part, nc, C, out);
  }
  return cudaGetLastError();
}

}  // namespace

cudaError_t copy_block0(const bf16* src, long Ls, bf16* dst, long Ld, int B, int d, int rows,
                        cudaStream_t st) {
  const long nvec = (long)rows * d / 8;
  dim3 grid((unsigned)((nvec + 255) / 256), B);
  LaunchTimer lt("copy_block0", st, 0.0, 32.0 * nvec * B);
  copy_block0_kernel<<<grid, 256, 0, st>>>(src, Ls, dst, Ld, d, nvec);
  return cudaGetLastError();
}

cudaError_t pad_rows(const bf16* src, bf16* dst, int B, long L, long Lp, int d, cudaStream_t st) {
  const long nvec = Lp * d / 8;
  dim3 grid((unsigned)((nvec + 255) / 256), B);
  LaunchTimer lt("pad_rows", st, 0.0, 2.0 * B * (L + Lp) * d);
  pad_rows_kernel<<<grid, 256, 0, st>>>(src, dst, L, Lp, d);
  return cudaGetLastError();
}

// The streaming form needs whole IB_W slices and enough rows per CTA to fill
// its ring (about two CTAs per SM of a 152-SM part, at least 128 rows each).
long ib_stream_chunks(long M, int N) {
  if (N % IB_W != 0) return 0;
  const long c = (304 + N / IB_W - 1) / (N / IB_W);
  return M / c >= 128 ? c : 0;
}

int inj_bwd_chunks(long M, int N) {
  const long c = ib_stream_chunks(M, N);
  return c ? (int)c : chunks_for(M, N);
}

int take_dev_error_elementwise() { return take_dev_error_tu(); }
int set_wait_limit_elementwise(unsigned long long ns) { return set_wait_limit_tu(ns); }

cudaError_t inj_bwd_1d(const InjBwdArgs& a, float* part, int n_chunks, cudaStream_t st) {
  const long M = (long)a.B * a.m * a.k2;
  const int N = a.k1 * a.d;
  const long rpc = (M + n_chunks - 1) / n_chunks;
  LaunchTimer lt("inj_bwd", st, 0.0, 10.0 * M * N + 16.0 * n_chunks * N);
  if (ib_stream_chunks(M, N) == n_chunks) {
    cudaError_t e = cudaFuncSetAttribute(inj_bwd_stream_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, IB_SMEM);
    if (e != cudaSuccess) return e;
    dim3 grid(N / IB_W, n_chunks);
    inj_bwd_stream_kernel<<<grid, 256, IB_SMEM, st>>>(a, part, M, N, rpc);
    return cudaGetLastError();
  }
  dim3 grid((N / INJ_COLS + EW_THREADS - 1) / EW_THREADS, n_chunks);
  inj_bwd_kernel<<<grid, EW_THREADS, 0, st>>>(a, part, M, N, rpc);
  return cudaGetLastError();
}

cudaError_t inj_bwd_finalize(const float* part, int n_chunks, int N, int d, float* db_d1,
                             float* gw_x, float* gw_dlt, float* gb_g, cudaStream_t st) {
  LaunchTimer lt("inj_bwd_finalize", st, 0.0, 16.0 * n_chunks * N);
  const int gates = gw_x != nullptr ? 1 : 0;
  const long n = (long)(gates ? 4 : 1) * N;
  float* pw = const_cast<float*>(part);  // the column totals reuse chunk 0's slots
  inj_bwd_colsum_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(pw, n_chunks, N, db_d1, gates);
  if (gates)
    inj_bwd_gates_kernel<<<(3 * d + 255) / 256, 256, 0, st>>>(part, N, d, gw_x, gw_dlt, gb_g);
  return cudaGetLastError();
}

namespace {

// RoPE angles, one thread per (position i < m, pair j < 32): i * 10000^(-2j/64)
// formed and reduced modulo 2 pi in double precision, (cos, sin) stored in
// single precision.  Shared by every sequence, head and by Q and K.
__global__ void rope_table_kernel(float2* __restrict__ tab, int m) {
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= m * 32) return;
  const int i = t >> 5, j = t & 31;
  const double theta = exp2(-(double)(2 * j) / 64.0 * 13.287712379549449);  // log2(10000)
  double a = (double)i * theta;
  a -= 6.283185307179586 * rint(a / 6.283185307179586);
  float sn, cs;
  sincosf((float)a, &sn, &cs);
  tab[t] = make_float2(cs, sn);
}

// RoPE on Q | K in place, one thread per rotated pair, angles from the table.
__global__ void rope_qk_kernel(bf16* __restrict__ qk, long ld, long rows, int m, int d,
                               const float2* __restrict__ tab, float sgn) {
  const long t = (long)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= rows * d) return;  // d pairs per row: d / 2 in Q, d / 2 in K
  const long row = t / d;
  const int col = 2 * (int)(t % d);
  const float2 cs = tab[(row % m) * 32 + ((col & 63) >> 1)];  // pair within the 64-wide head
  const float sn = sgn * cs.y;
  uint32_t* q = reinterpret_cast<uint32_t*>(qk + row * ld + col);
  const float2 v = unpack_bf16(*q);
  *q = pack_bf16(v.x * cs.x - v.y * sn, v.x * sn + v.y * cs.x);
}

__global__ void add_f32_bf16_kernel(const bf16* __restrict__ a, const float* __restrict__ b,
                                    float* __restrict__ of, bf16* __restrict__ ob, long n4) {
  const long t = (long)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= n4) return;
  const uint2 u = reinterpret_cast<const uint2*>(a)[t];
  const float2 x = unpack_bf16(u.x), y = unpack_bf16(u.y);
  float4 v = make_float4(x.x, x.y, y.x, y.y);
  if (b) {
    const float4 c = reinterpret_cast<const float4*>(b)[t];
    v.x += c.x; v.y += c.y; v.z += c.z; v.w += c.w;
  }
  reinterpret_cast<float4*>(of)[t] = v;
  reinterpret_cast<uint2*>(ob)[t] = make_uint2(pack_bf16(v.x, v.y), pack_bf16(v.z, v.w));
}

}  // namespace

cudaError_t rope_qk(bf16* qk, long ld, int B, int m, int d, float2* tab, bool inverse,
                    cudaStream_t st) {
  if (d % 64 || ld < 2 * d || !tab) return cudaErrorInvalidValue;
  const long rows = (long)B * m, n = rows * d;
  {
    LaunchTimer lt("rope_table", st, 0.0, 8.0 * m * 32);
    rope_table_kernel<<<(m * 32 + 255) / 256, 256, 0, st>>>(tab, m);
  }
  LaunchTimer lt("rope_qk", st, 6.0 * n, 8.0 * n);
  rope_qk_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(qk, ld, rows, m, d, tab,
                                                              inverse ? -1.f : 1.f);
  return cudaGetLastError();
}

cudaError_t add_f32_bf16(const bf16* a, const float* b, float* out_f, bf16* out_b, long n,
                         cudaStream_t st) {
  if (n % 4) return cudaErrorInvalidValue;
  const long n4 = n / 4;
  LaunchTimer lt("add_f32_bf16", st, (double)n, 2.0 * n + (b ? 4.0 : 0.0) * n + 6.0 * n);
  add_f32_bf16_kernel<<<(unsigned)((n4 + 255) / 256), 256, 0, st>>>(a, b, out_f, out_b, n4);
  return cudaGetLastError();
}

long colsum_part_elems(long R, int C) { return (long)colsum_chunks(R, C) * C; }

cudaError_t colsum_bf16(const bf16* X, long R, int C, float* out, float* part, cudaStream_t st) {
  return colsum_impl<bf16>(X, R, C, out, part, st);
}
cudaError_t colsum_f32(const float* X, long R, int C, float* out, float* part, cudaStream_t st) {
  return colsum_impl<float>(X, R, C, out, part, st);
}

}  // namespace pf
