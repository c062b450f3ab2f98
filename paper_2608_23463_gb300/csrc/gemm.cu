// Host side of the tcgen05 GEMM: TMA tensor maps, tile-width choice and the
// instantiations used by the layer (see gemm_tc.cuh for the kernel).
#include <cudaTypedefs.h>

#include <algorithm>

#include "gemm_tc.cuh"
#include "kernels.h"

namespace pf {

int take_dev_error_gemm() { return take_dev_error_tu(); }
int set_wait_limit_gemm(unsigned long long ns) { return set_wait_limit_tu(ns); }
int set_debug_skip_loads_gemm(int on) {
  return cudaMemcpyToSymbol(g_debug_skip_loads, &on, sizeof(on)) == cudaSuccess ? 0 : -1;
}

int num_sms() {
  static int n = 0;
  if (n == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 148;
  }
  return n;
}

namespace {

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (fn == nullptr) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// 2D bf16 map over a row-major [outer, inner] matrix with `ld` elements per
// row, 128-byte swizzle, zero fill outside the matrix.
bool make_map(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer, uint64_t ld,
              uint32_t box_inner, uint32_t box_outer) {
  auto fn = encode_fn();
  if (fn == nullptr) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {ld * 2};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t es[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// rows = M (for A) or N (for B).
bool make_operand_map(CUtensorMap* m, const Operand& op, int rows, int K) {
  if (op.mn) return make_map(m, op.ptr, (uint64_t)rows, (uint64_t)K, (uint64_t)op.ld, 64, 64);
  return make_map(m, op.ptr, (uint64_t)K, (uint64_t)rows, (uint64_t)op.ld, 64, 128);
}

// Co-resident CTA pairs of the pair kernel (at most half the SMs).
template <class Kern>
int max_pairs(Kern kern, int threads, int smem) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * (num_sms() / 2));
  cfg.blockDim = dim3(threads);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = 2;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess || n <= 0) {
    cudaGetLastError();
    return 0;
  }
  return std::min(n, num_sms() / 2);
}

template <int BN, bool AMN, bool BMN, class Epi>
cudaError_t launch(int M, int N, int K, const CUtensorMap& ta, const CUtensorMap& tb,
                   const CUtensorMap& tx, const Epi& epi, cudaStream_t st, int splits) {
  constexpr int XCOLS = Epi::kXTile ? (Epi::kPaired ? BN / 2 : BN) : 0;
  if constexpr (BN == 256 && Epi::kPairs) {
    // CTA pairs (256 x 256 tiles, half of B per CTA, a deeper stage ring)
    // when every co-resident pair gets a tile
    auto kern2 = gemm_tc_kernel<BN, AMN, BMN, Epi, true>;
    constexpr int smem2 = GemmCfg<BN, XCOLS, Epi::kColPar, true, Epi::kStageBytes>::SMEM_BYTES;
    constexpr int threads = GemmRoles<Epi>::kThreads;
    cudaError_t e = cudaFuncSetAttribute(kern2, cudaFuncAttributeMaxDynamicSharedMemorySize, smem2);
    if (e != cudaSuccess) return e;
    static const int pairs = max_pairs(kern2, threads, smem2);
    const long pair_tiles =
        (long)((N + BN - 1) / BN) * ((M + 2 * GEMM_BM - 1) / (2 * GEMM_BM)) * splits;
    if (pairs > 0 && pair_tiles >= pairs) {
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3(2 * (unsigned)std::min<long>(pair_tiles, pairs));
      cfg.blockDim = dim3(threads);
      cfg.dynamicSmemBytes = smem2;
      cfg.stream = st;
      cudaLaunchAttribute at[1];
      at[0].id = cudaLaunchAttributeClusterDimension;
      at[0].val.clusterDim.x = 2;
      at[0].val.clusterDim.y = 1;
      at[0].val.clusterDim.z = 1;
      cfg.attrs = at;
      cfg.numAttrs = 1;
      e = cudaLaunchKernelEx(&cfg, kern2, ta, tb, tx, M, N, K, splits, epi);
      if (e != cudaSuccess) return e;
      return cudaGetLastError();
    }
  }
  auto kern = gemm_tc_kernel<BN, AMN, BMN, Epi>;
  constexpr int smem = GemmCfg<BN, XCOLS, Epi::kColPar, false, Epi::kStageBytes>::SMEM_BYTES;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  const long tiles = (long)((N + BN - 1) / BN) * ((M + GEMM_BM - 1) / GEMM_BM) * splits;
  const int grid = (int)std::min<long>(tiles, num_sms());
  kern<<<grid, GemmRoles<Epi>::kThreads, smem, st>>>(ta, tb, tx, M, N, K, splits, epi);
  return cudaGetLastError();
}

template <int BN, class Epi>
cudaError_t launch_majors(int M, int N, int K, const Operand& A, const Operand& B,
                          const CUtensorMap& ta, const CUtensorMap& tb, const CUtensorMap& tx,
                          const Epi& epi, cudaStream_t st, int splits = 1) {
  if (!A.mn && !B.mn) return launch<BN, false, false>(M, N, K, ta, tb, tx, epi, st, splits);
  if (!A.mn && B.mn) return launch<BN, false, true>(M, N, K, ta, tb, tx, epi, st, splits);
  if (A.mn && B.mn) return launch<BN, true, true>(M, N, K, ta, tb, tx, epi, st, splits);
  return launch<BN, true, false>(M, N, K, ta, tb, tx, epi, st, splits);
}

bool operand_ok(const Operand& op) {
  return op.ptr != nullptr && (reinterpret_cast<uintptr_t>(op.ptr) & 15) == 0 && op.ld > 0 &&
         (op.ld * 2) % 16 == 0;
}

// X tile source (kXTile epilogues): the [rows, N] bf16 view the epilogue
// prefetches by TMA; for other epilogues `xsrc` is ignored.
template <class Epi>
cudaError_t gemm_dispatch(int M, int N, int K, Operand A, Operand B, const Epi& epi,
                          const bf16* xsrc, long x_rows, cudaStream_t st, long x_cols = -1) {
  if (x_cols < 0) x_cols = N;
  if (M <= 0 || N <= 0 || N % 32 != 0 || K < 0 || !operand_ok(A) || !operand_ok(B))
    return cudaErrorInvalidValue;
  CUtensorMap ta, tb, tx;
  if (!make_operand_map(&ta, A, M, K) || !make_operand_map(&tb, B, N, K))
    return cudaErrorInvalidValue;
  if (Epi::kXTile) {
    if (xsrc == nullptr || (reinterpret_cast<uintptr_t>(xsrc) & 15) != 0 ||
        !make_map(&tx, xsrc, (uint64_t)x_cols, (uint64_t)x_rows, (uint64_t)x_cols, 64, 128))
      return cudaErrorInvalidValue;
  } else {
    tx = ta;
  }
  const long tiles256 = (long)((N + 255) / 256) * ((M + GEMM_BM - 1) / GEMM_BM);
  LaunchTimer lt(gemm_tag_label(), st, 2.0 * M * N * (double)K,
                 2.0 * ((double)M * K + (double)N * K) + gemm_tag_bytes());
  // 128 x 256 tiles move about 2/3 of the shared-memory bytes per FLOP of
  // 128 x 128 tiles (the mainloop's bound); take them unless they need more
  // than 1.5x the waves
  const long tiles128 = (long)((N + 127) / 128) * ((M + GEMM_BM - 1) / GEMM_BM);
  const long sms = num_sms(), w256 = (tiles256 + sms - 1) / sms, w128 = (tiles128 + sms - 1) / sms;
  if (Epi::kPaired || (N >= 256 && 3 * w256 <= 2 * w128))
    return launch_majors<256>(M, N, K, A, B, ta, tb, tx, epi, st);
  return launch_majors<128>(M, N, K, A, B, ta, tb, tx, epi, st);
}

// out = sum_s part[s] (+ bias) (+ addend) -> fp32 and/or bf16, 4 columns per thread.
__global__ void splitk_reduce_kernel(const float* __restrict__ part, int S, int M, int N,
                                     EpiLinearArgs e) {
  const long i = ((long)blockIdx.x * blockDim.x + threadIdx.x) * 4;
  if (i >= (long)M * N) return;
  const long row = i / N;
  const int col = (int)(i % N);
  float4 v = *reinterpret_cast<const float4*>(part + i);
  for (int s = 1; s < S; ++s) {
    const float4 w = *reinterpret_cast<const float4*>(part + (long)s * M * N + i);
    v.x += w.x; v.y += w.y; v.z += w.z; v.w += w.w;
  }
  if (e.bias) {
    const float4 b = *reinterpret_cast<const float4*>(e.bias + col);
    v.x += b.x; v.y += b.y; v.z += b.z; v.w += b.w;
  }
  if (e.addend) {
    const float4 a = *reinterpret_cast<const float4*>(e.addend + row * e.ld_add + col);
    v.x += a.x; v.y += a.y; v.z += a.z; v.w += a.w;
  }
  if (e.add_bf16) {
    const uint2 u = *reinterpret_cast<const uint2*>(e.add_bf16 + row * e.ld_add_bf16 + col);
    const float2 a0 = unpack_bf16(u.x), a1 = unpack_bf16(u.y);
    v.x += a0.x; v.y += a0.y; v.z += a1.x; v.w += a1.y;
  }
  if (e.out_f32) *reinterpret_cast<float4*>(e.out_f32 + row * e.ld_f32 + col) = v;
  if (e.out_bf16)
    *reinterpret_cast<uint2*>(e.out_bf16 + row * e.ld_bf16 + col) =
        make_uint2(pack_bf16(v.x, v.y), pack_bf16(v.z, v.w));
}

}  // namespace

bool tmap_bf16_2d(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer, uint64_t ld,
                  uint32_t box_inner, uint32_t box_outer) {
  return make_map(m, base, inner, outer, ld, box_inner, box_outer);
}

int splitk_factor(int M, int N, int K) {
  constexpr int kSms = 152;  // planning target (GB300); fixed so sizes are device-independent
  const long tiles = (long)((N + 127) / 128) * ((M + GEMM_BM - 1) / GEMM_BM);
  const int num_k = (K + GEMM_BK - 1) / GEMM_BK;
  if (tiles >= kSms || num_k < 32) return 1;
  int best = 1;
  double best_eff = (double)tiles / kSms;
  for (int S = 2; S <= 16 && num_k / S >= 16; ++S) {
    const long t = tiles * S;
    const double eff = (double)t / (((t + kSms - 1) / kSms) * kSms);
    if (eff > best_eff + 1e-9) {
      best = S;
      best_eff = eff;
    }
  }
  return best;
}

size_t splitk_scratch_bytes(int M, int N, int K) {
  const int S = splitk_factor(M, N, K);
  return S > 1 ? (size_t)S * M * N * sizeof(float) : 0;
}

cudaError_t gemm_linear(int M, int N, int K, Operand A, Operand B, const EpiLinearArgs& e,
                        cudaStream_t st) {
  const int S = splitk_factor(M, N, K);
  if (S > 1 && e.splitk_scratch && (size_t)S * M * N * sizeof(float) <= e.splitk_bytes &&
      N % 4 == 0 && !e.act_silu && !e.pre_bf16 && !e.dsilu_of) {
    // deterministic split-K: raw partials, then one reduce applying the epilogue
    if (M <= 0 || N % 32 != 0 || !operand_ok(A) || !operand_ok(B)) return cudaErrorInvalidValue;
    CUtensorMap ta, tb;
    if (!make_operand_map(&ta, A, M, K) || !make_operand_map(&tb, B, N, K))
      return cudaErrorInvalidValue;
    EpiPartial epi{{}, N, e.splitk_scratch};
    {
      LaunchTimer lt(gemm_tag_label(), st, 2.0 * M * N * (double)K,
                     2.0 * ((double)M * K + (double)N * K) + 4.0 * S * M * N);
      cudaError_t err = launch_majors<128>(M, N, K, A, B, ta, tb, ta, epi, st, S);
      if (err != cudaSuccess) return err;
    }
    LaunchTimer lt("splitk_reduce", st, (double)S * M * N, 4.0 * (S + 1.0) * M * N);
    const long quads = (long)M * N / 4;
    splitk_reduce_kernel<<<(unsigned)((quads + 255) / 256), 256, 0, st>>>(e.splitk_scratch, S, M,
                                                                          N, e);
    return cudaGetLastError();
  }
  if ((e.add_bf16 && ((uintptr_t)e.add_bf16 & 15)) || (e.add_bf16 && e.ld_add_bf16 % 8))
    return cudaErrorInvalidValue;
  if ((e.pre_bf16 && ((uintptr_t)e.pre_bf16 & 15 || e.ld_pre % 8)) ||
      (e.dsilu_of && ((uintptr_t)e.dsilu_of & 15 || e.ld_dsilu % 8)))
    return cudaErrorInvalidValue;
  // a short contraction with a plain (bias) epilogue stores whole rows from a
  // shared-memory stage: its output, not its mainloop, would bound it
  if (K <= 2048 && !e.addend && !e.add_bf16 && !e.act_silu && !e.pre_bf16 && !e.dsilu_of &&
      (e.out_f32 == nullptr || e.ld_f32 % 4 == 0) && (e.out_bf16 == nullptr || e.ld_bf16 % 8 == 0)) {
    EpiLinearStaged epi{{}, M, N, e.bias, e.out_f32, e.ld_f32, e.out_bf16, e.ld_bf16};
    return gemm_dispatch(M, N, K, A, B, epi, nullptr, 0, st);
  }
  EpiLinear epi{{},         M,          N,          e.bias,      e.addend,  e.ld_add,
                e.out_f32,  e.ld_f32,   e.out_bf16, e.ld_bf16,   e.add_bf16, e.ld_add_bf16,
                e.act_silu, e.pre_bf16, e.ld_pre,   e.dsilu_of,  e.ld_dsilu};
  return gemm_dispatch(M, N, K, A, B, epi, nullptr, 0, st);
}

cudaError_t gemm_inject1d(int M, int N, int K, Operand A, Operand B, const EpiInjectArgs& e,
                          cudaStream_t st) {
  EpiInject1D epi{{}, M, N, e.bias, e.D_save, e.X_out, e.w_x, e.w_dlt, e.b_g,
                  e.d, e.k1, e.k2, e.m, e.L, e.shift, e.gated};
  if (A.mn || B.mn) return cudaErrorInvalidValue;
  return gemm_dispatch(M, N, K, A, B, epi, e.Xsrc, M, st);
}

cudaError_t gemm_dx1d(int M, int N, int K, Operand A, Operand B, const EpiDXArgs& e,
                      cudaStream_t st) {
  EpiDX1D epi{{}, M, N, e.dX, e.d, e.k1, e.k2, e.m, e.L};
  if (A.mn || !B.mn) return cudaErrorInvalidValue;
  return gemm_dispatch(M, N, K, A, B, epi, e.dXd, M, st);
}

cudaError_t gemm_append_kv(int M, int N, int K, Operand A, Operand B, const EpiAppendArgs& e,
                           cudaStream_t st) {
  EpiAppendKV epi{{}, M, N, e.K, e.V, e.n_open, e.n_proxy, e.d, e.P, e.cap};
  if (A.mn || B.mn) return cudaErrorInvalidValue;
  return gemm_dispatch(M, N, K, A, B, epi, nullptr, 0, st);
}

cudaError_t gemm_affine2d(int M, int N, int K, Operand A, Operand B, const EpiAffine2DArgs& e,
                          cudaStream_t st) {
  EpiAffine2D epi{{}, M, e.bias, e.S_save, e.X_out, e.stats, e.d, e.patch, e.gh, e.gw, e.m};
  if (A.mn || B.mn || e.d % 128 != 0) return cudaErrorInvalidValue;
  return gemm_dispatch(M, N, K, A, B, epi, e.Xp, M, st, (long)e.patch * e.patch * e.d);
}

cudaError_t gemm_dx2d(int M, int N, int K, Operand A, Operand B, const EpiDX2DArgs& e,
                      cudaStream_t st) {
  EpiDX2D epi{{}, M, N, e.dX, e.d, e.patch, e.gh, e.gw, e.m};
  if (A.mn || !B.mn || e.d % 32 != 0) return cudaErrorInvalidValue;
  return gemm_dispatch(M, N, K, A, B, epi, e.dXd, M, st);
}

}  // namespace pf
