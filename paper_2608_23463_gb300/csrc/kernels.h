// Internal launch interface between the C ABI (api.cu) and the kernels.
#pragma once

#include "common.cuh"

namespace pf {

// ------------------------------------------------------------------ GEMM
// Operand of D[M,N] = sum_k A[m,k] B[n,k]: `mn` = 0 for K-major storage
// ([rows=M or N, K], leading dimension ld >= K), 1 for MN-major storage
// ([K, M or N], ld >= M or N).  bf16, 16-byte aligned, ld*2 % 16 == 0.
struct Operand {
  const bf16* ptr;
  long ld;
  int mn;
};

struct EpiLinearArgs {
  const float* bias = nullptr;    // [N]
  const float* addend = nullptr;  // [M, ld_add] fp32
  long ld_add = 0;
  const bf16* add_bf16 = nullptr;  // [M, ld_add_bf16] bf16, added like addend
  long ld_add_bf16 = 0;
  // SiLU: the value after bias / addends is stored to pre_bf16 (if given),
  // then out = SiLU(value); dsilu_of: out = value * SiLU'(u), u read from a
  // bf16 matrix [M, ld_dsilu].  Either one disables split-K.
  int act_silu = 0;
  bf16* pre_bf16 = nullptr;
  long ld_pre = 0;
  const bf16* dsilu_of = nullptr;
  long ld_dsilu = 0;
  float* out_f32 = nullptr;
  long ld_f32 = 0;
  bf16* out_bf16 = nullptr;
  long ld_bf16 = 0;
  // optional scratch for deterministic split-K (used when the output tiles
  // alone cannot fill the GPU and splitk_scratch_bytes() bytes are given)
  float* splitk_scratch = nullptr;
  size_t splitk_bytes = 0;
};
// Split-K factor chosen for an M x N x K linear GEMM (1: none) and the fp32
// scratch it needs; independent of the device.
int splitk_factor(int M, int N, int K);
size_t splitk_scratch_bytes(int M, int N, int K);

struct EpiInjectArgs {
  const float* bias;  // b_d1 [k1*d]
  bf16* D_save;       // [M, k1*d] or null
  const bf16* Xsrc;   // X as [B*m*k2, k1*d] (zero-padded to whole blocks if L % P != 0)
  bf16* X_out;
  const float *w_x, *w_dlt, *b_g;  // gate vectors (gated) or null (add)
  int d, k1, k2, m, L, shift, gated;
};

struct EpiDXArgs {
  const bf16* dXd;  // direct gradient as [B*m*k2, k1*d] (padded like Xsrc)
  bf16* dX;
  int d, k1, k2, m, L;
};

cudaError_t gemm_linear(int M, int N, int K, Operand A, Operand B, const EpiLinearArgs& e,
                        cudaStream_t st);
cudaError_t gemm_inject1d(int M, int N, int K, Operand A, Operand B, const EpiInjectArgs& e,
                          cudaStream_t st);
cudaError_t gemm_dx1d(int M, int N, int K, Operand A, Operand B, const EpiDXArgs& e,
                      cudaStream_t st);

// 2D layer: decompression + affine injection, and the compression dX.
struct EpiAffine2DArgs {
  const float* bias;   // b_d1 [2*P*d]
  bf16* S_save;        // s in patch order [B*m, P*d]
  bf16* X_out;         // [B, gh*gw, d]
  const float* stats;  // [B*gh*gw, 2] mean, 1/std of X per token
  const bf16* Xp;      // X in patch order [B*m, P*d]
  int d, patch, gh, gw, m;
};
cudaError_t gemm_affine2d(int M, int N, int K, Operand A, Operand B, const EpiAffine2DArgs& e,
                          cudaStream_t st);
struct EpiDX2DArgs {
  const bf16* dXd;  // direct gradient in patch order [B*m, P*d]
  bf16* dX;         // [B, gh*gw, d]
  int d, patch, gh, gw, m;
};
cudaError_t gemm_dx2d(int M, int N, int K, Operand A, Operand B, const EpiDX2DArgs& e,
                      cudaStream_t st);

// KV append: rows b = sequences, columns [0, d) -> K_proxy[b, n_proxy[b]],
// [d, 2d) -> V_proxy[b, n_proxy[b]] (bf16), only for sequences whose open
// block is full (n_open[b] == P) and whose cache has room.
struct EpiAppendArgs {
  bf16 *K, *V;
  const int *n_open, *n_proxy;
  int d, P, cap;
};
cudaError_t gemm_append_kv(int M, int N, int K, Operand A, Operand B, const EpiAppendArgs& e,
                           cudaStream_t st);
int num_sms();

// Per-file device error flags (see common.cuh): value, cleared on read.  The
// per-file wait limits (set_wait_limit_*) and the GEMM producer's load-skip
// hook serve the timeout test (pf_debug_set_wait_limit_ns); 0 = success.
int set_wait_limit_gemm(unsigned long long ns);
int set_wait_limit_decode(unsigned long long ns);
int set_wait_limit_attention(unsigned long long ns);
int set_wait_limit_attention_tc(unsigned long long ns);
int set_wait_limit_attention_bwd_tc(unsigned long long ns);
int set_wait_limit_elementwise(unsigned long long ns);
int set_wait_limit_fp32(unsigned long long ns);
int set_wait_limit_layer2d(unsigned long long ns);
int set_debug_skip_loads_gemm(int on);
int take_dev_error_gemm();
int take_dev_error_decode();
int take_dev_error_attention();
int take_dev_error_attention_tc();
int take_dev_error_attention_bwd_tc();
int take_dev_error_elementwise();

// ------------------------------------------------------------- 2D layer
int take_dev_error_layer2d();
// The patch-order copy Xp [B*m, P*d] of X [B, gh*gw, d] and every token's
// LayerNorm statistics (mean, 1/std), in one pass over X (d <= 512).
cudaError_t patch_gather_stats(const bf16* X, bf16* Xp, float* stats, int B, int d, int patch,
                               int gh, int gw, cudaStream_t st);

cudaError_t temb_fwd(const float* t, int B, int d, const bf16* W_t1, const float* b_t1,
                     const bf16* W_t2, const float* b_t2, float* e, float* a1, float* u, float* gb,
                     cudaStream_t st);
cudaError_t adaln_fwd(const float* H, const float* gb, float* nH, float* rstd, bf16* Hq, long R,
                      int d, int m, cudaStream_t st);
// Backward of the affine injection over R patches (d <= 512): dD, the direct
// dX in patch order, and (db_d1 non-null) the bias gradient of the
// decompression from per-block partial sums in `part`
// (inj_bwd_2d_part_elems floats).
long inj_bwd_2d_part_elems(long R, int d, int patch);
cudaError_t inj_bwd_2d(const bf16* G, const bf16* X, const float* stats, const bf16* S, bf16* dD,
                       bf16* dXd, float* db_d1, float* part, long R, int d, int patch, int gh,
                       int gw, cudaStream_t st);
cudaError_t adaln_bwd(const float* dHq, const float* nH, const float* rstd, const float* gb,
                      const float* dH_out, float* dHf, bf16* dHb, long R, int d, int m,
                      cudaStream_t st);
int adaln_param_chunks(int m);
cudaError_t adaln_param_grads(const float* dHq, const float* nH, float* part, float* dgb, int B,
                              int d, int m, cudaStream_t st);
struct TembGrads {
  float *W_t2, *b_t2, *W_t1, *b_t1;
};
cudaError_t temb_bwd(const float* dgb, const bf16* W_t2, const float* a1, const float* u,
                     const float* e, float* da1, const TembGrads& g, int B, int d,
                     cudaStream_t st);

// ---------------------------------------------------------- fp32 forward
int take_dev_error_fp32();
// fp32 GEMM C = A B^T (+ bias) (+ addend); split-K over `scratch` when the
// output tiles cannot fill the GPU (splitk_f32_factor(M, N, K) * M * N floats).
int splitk_f32_factor(int M, int N, int K);
cudaError_t gemm_f32(int M, int N, int K, const float* A, long lda, const float* B, long ldb,
                     float* C, long ldc, const float* bias, const float* addend, long ld_add,
                     const char* label, cudaStream_t st, float* scratch = nullptr,
                     size_t scratch_bytes = 0);
// The last decompression level fused with routing and injection (Eq. inj-gate
// / inj-add): X_out instead of D; block 0 of every sequence (shift = 1) is
// copied from X.
cudaError_t gemm_f32_inject(int M, int N, int K, const float* A, long lda, const float* B, long ldb,
                            const float* bias, const float* X, float* Xo, const float* w_x,
                            const float* w_dlt, const float* b_g, int Bsz, long L, int d, int P,
                            int k1, int k2, int m, int shift, int gated, cudaStream_t st);
cudaError_t attn_f32(const float* qkv, float* out, int B, int m, int d, int nh, bool causal,
                     cudaStream_t st);
cudaError_t inject_f32(const float* X, const float* D, float* Xo, const float* w_x,
                       const float* w_dlt, const float* b_g, int B, long L, int d, int P, int k1,
                       int k2, int m, int shift, int gated, cudaStream_t st);
cudaError_t pad_f32(const float* src, float* dst, int B, long L, long Lp, int d, cudaStream_t st);

// ---------------------------------------------------------------- decode
#define PF_DECODE_MAX_P 256
struct DecodeLaunch {
  int B, d, nh, P, cap, splits;
  const bf16* x;
  bf16* y;
  const bf16 *W_qkv, *W_o, *W_a1, *W_a2;
  const float *rms_w, *b_a1, *b_a2;
  const bf16 *K_proxy, *V_proxy;
  bf16 *X_open, *K_open, *V_open;
  int *n_proxy, *n_open;
  float* ws;
};
size_t decode_workspace_bytes(int B, int d, int nh, int splits);
int decode_splits(int B, int nh, int cap);
cudaError_t decode_step_launch(const DecodeLaunch& L, cudaStream_t st);
cudaError_t append_finish(int* n_open, int* n_proxy, int B, int P, int cap, cudaStream_t st);
// n_proxy[b] = m, n_open[b] = r for every sequence (bulk prefill)
cudaError_t prefill_counts(int* n_open, int* n_proxy, int B, int m, int r, cudaStream_t st);

// 2D bf16 TMA map over a row-major [outer, inner] matrix (ld elements per
// row), 128-byte swizzle, zero fill outside; box box_inner x box_outer.
bool tmap_bf16_2d(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer, uint64_t ld,
                  uint32_t box_inner, uint32_t box_outer);

// ------------------------------------------------------------- attention
cudaError_t attn_fwd(const bf16* qkv, bf16* out, float* lse, int B, int m, int d, int nh,
                     bool causal, cudaStream_t st);
// Cross-attention of the injection (Eq. inj-cross): queries from qa [B*Lq,
// ldq] (columns [0, d), the gate pre-activations at [d, d + nh)), keys and
// values from kv [B*Lk, 2d]; token q sees proxies j < q / P (causal) or all.
// Writes out (ungated), out_g = sigmoid(gate + b_a) * out per head (if not
// null), both [B*Lq, d], and LSE [B, nh, Lq].
cudaError_t attn_cross_fwd(const bf16* qa, long ldq, const bf16* kv, const float* b_a, bf16* out,
                           bf16* out_g, float* lse, int B, int Lq, int Lk, int d, int nh, int P,
                           bool causal, cudaStream_t st);
// Its backward, given dO (the gradient of the ungated output) and Di =
// rowsum(dO * O): dQ into dqa columns [0, d) (row stride ldq), dK and dV into
// dkv [B*Lk, 2d].
cudaError_t attn_cross_bwd(const bf16* qa, long ldq, const bf16* kv, const bf16* dO,
                           const float* lse, const float* Di, bf16* dqa, bf16* dkv, int B, int Lq,
                           int Lk, int d, int nh, int P, bool causal, cudaStream_t st);
// Gate of the cross injection, backward, one warp per (token row, head):
// s = sum over the head's columns of dAg * A, alpha = sigmoid(qa[row, d + h] +
// b_a[h]); dO = alpha * dAg, Di = alpha * s (= rowsum(dO * A)), and the gate
// pre-activation gradient s alpha (1 - alpha) into dqa[row, d + h] (bf16;
// columns [d + nh, ldq) zeroed) and ga[row, h] (fp32, row stride ldga,
// columns [nh, ldga) zeroed).
cudaError_t cross_gate_bwd(const bf16* dAg, const bf16* A, const bf16* qa, long ldq,
                           const float* b_a, bf16* dO, float* Di, bf16* dqa, float* ga, int ldga,
                           int B, int L, int d, int nh, cudaStream_t st);
// RoPE on the proxies' queries and keys, in place: rows (b, i) of a [B*m, ld]
// matrix, columns [0, 2d) = Q | K, pair (2j, 2j+1) of head h turned by the
// angle i * 10000^(-2j/64) (backwards when inverse).  tab: scratch of m * 32
// float2 for the (cos, sin) table.
cudaError_t rope_qk(bf16* qk, long ld, int B, int m, int d, float2* tab, bool inverse,
                    cudaStream_t st);
// out_f = a + b (b may be null), out_b = bf16(out_f), n elements (n % 4 == 0)
cudaError_t add_f32_bf16(const bf16* a, const float* b, float* out_f, bf16* out_b, long n,
                         cudaStream_t st);
cudaError_t attn_bwd_tc(const bf16* qkv, const bf16* dO, const float* lse, const float* Di,
                        bf16* dqkv, int B, int m, int d, int nh, bool causal, cudaStream_t st);
cudaError_t attn_bwd(const bf16* qkv, const bf16* O, const bf16* dO, const float* lse, float* Di,
                     bf16* dqkv, int B, int m, int d, int nh, bool causal, cudaStream_t st);

// ----------------------------------------------------------- elementwise
// Copy the first `rows` rows (width d) of each sequence of src [B, Ls, d] to
// dst [B, Ld, d] (block 0 of the causal routing: X_out = X, dX = dX_out).
cudaError_t copy_block0(const bf16* src, long Ls, bf16* dst, long Ld, int B, int d, int rows,
                        cudaStream_t st);
// dst [B, Lp, d] = src [B, L, d] padded with zero rows (Lp >= L).
cudaError_t pad_rows(const bf16* src, bf16* dst, int B, long L, long Lp, int d, cudaStream_t st);

// Backward of the 1D injection (Eq. inj-gate / inj-add) in proxy order.
// Rows r of D / dD are [M = B*m*k2, N = k1*d]; row r's values belong to the
// tokens of block i + shift.  Writes dD (zero where no token exists), the
// direct gradient into dX, and fills `part` [n_chunks][4][N] partial column
// sums (dD, ds*X, ds*D, ds with ds = G*D*s*(1-s)).  Returns n_chunks via out.
struct InjBwdArgs {
  const bf16* G;
  const bf16* X;
  const bf16* D;
  bf16* dD;
  bf16* dX;     // direct gradient, [B, Ldx, d]
  long Ldx;     // rows per sequence of dX (L, or m*P when padded)
  const float *w_x, *w_dlt, *b_g;
  int d, k1, k2, m, L, B, shift, gated;
};
int inj_bwd_chunks(long M, int N);
cudaError_t inj_bwd_1d(const InjBwdArgs& a, float* part, int n_chunks, cudaStream_t st);
// Reduce the partials: db_d1[c] = sum part[.][0][c]; gate grads (if non-null)
// summed over chunks and the k1 token positions: g[ch] = sum part[.][j][q*d+ch].
// part is scratch: its chunk-0 slots hold the column totals afterwards.
cudaError_t inj_bwd_finalize(const float* part, int n_chunks, int N, int d, float* db_d1,
                             float* gw_x, float* gw_dlt, float* gb_g, cudaStream_t st);

// out[c] = sum_r X[r, c] for a row-major [R, C] matrix (bf16 or fp32),
// deterministic two-pass reduction using `part` (colsum_part_elems floats).
long colsum_part_elems(long R, int C);
cudaError_t colsum_bf16(const bf16* X, long R, int C, float* out, float* part, cudaStream_t st);
cudaError_t colsum_f32(const float* X, long R, int C, float* out, float* part, cudaStream_t st);

}  // namespace pf

namespace pf {
// ------------------------------------------------------------ launch timing
// When enabled (pf_timing_enable), every kernel launch of the library is
// bracketed by CUDA events recorded on its own stream and tagged with a label
// and its algorithmic work; pf_timing_collect aggregates them after the caller
// has synchronised.  Disabled, a LaunchTimer does nothing.
struct LaunchTimer {
  LaunchTimer(const char* label, cudaStream_t st, double flops, double bytes);
  ~LaunchTimer();
  int idx;
  cudaStream_t st;
};
// Label (and epilogue bytes) of the next GEMM launches, set by the caller.
void set_gemm_tag(const char* label, double epi_bytes);
const char* gemm_tag_label();
double gemm_tag_bytes();
}  // namespace pf
