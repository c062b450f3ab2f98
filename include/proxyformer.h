/*
 * proxyformer.h -- C ABI of the GB300 (sm_103a) ProxyFormer hot path.
 *
 * One ProxyFormer layer (Alg. 1 of "ProxyFormer: A Dual-Stream Proxy
 * Architecture for Ultra-Long Context and High-Resolution Generation"):
 *   Partition (Eq. partition) -> compression c_i = Proj(Flatten(X_i))
 *   (Eq. compress-linear; two-level cascade Eq. factor-cascade) -> proxy state
 *   H = H_in + C (Eq. proxy-res) -> proxy attention (Eq. proxy-attn) ->
 *   decompression (Eq. decompress-linear / Eq. factor-dec) -> injection into
 *   the local stream (Eq. inj-add, Eq. inj-gate, Eq. inj-affine),
 * its backward pass, and the proxy-only KV-cache decode step and block append
 * (Sec. 3.8, Eq. proxy-cache, Eq. llm-cross, Eq. llm-gate).
 *
 * Conventions common to every entry point
 *   - Pointers named "device" are CUDA device pointers owned by the caller;
 *     the library never allocates and never frees them.  Scratch memory comes
 *     from the caller's workspace buffer (size from the *_workspace_size
 *     query).  Buffers must be 16-byte aligned.
 *   - Every call is asynchronous on `stream` (a cudaStream_t cast to void*;
 *     NULL is the legacy default stream).  Argument errors are detected on the
 *     host before anything is launched and reported as a pf_status; the
 *     message is available from pf_last_error() (thread-local).
 *   - Errors raised inside kernels (a bounded wait that ran out) are recorded
 *     in a device flag and reported by pf_sync_check() as PF_ERR_TIMEOUT.
 *   - Weight matrices are row-major [out, in] (y = W x + b).  Matrices and
 *     activations use the descriptor's dtype (bf16 or fp32); bias, gate and
 *     norm vectors, the proxy state H and all parameter gradients are fp32.
 *   - Flattening a block is token-major: element (token p, channel ch) of a
 *     block sits at index p*d + ch of its vector.
 *   - Causal 1D routing: the tokens of block i receive the decompression of
 *     interacted proxy i-1 and block 0 receives zero, so no token ever reads a
 *     later token (the library's reading of Eq. proxy-attn's causal mask for
 *     the local stream).
 */
#ifndef PROXYFORMER_H
#define PROXYFORMER_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  PF_OK = 0,
  PF_ERR_INVALID_ARG = 1, /* a descriptor field, pointer or alignment is wrong  */
  PF_ERR_UNSUPPORTED = 2, /* valid per the paper, not built in this library       */
  PF_ERR_WORKSPACE = 3,   /* workspace (or saved) buffer smaller than required    */
  PF_ERR_CAPACITY = 4,    /* KV cache full / open block full or not full          */
  PF_ERR_CUDA = 5,        /* a CUDA runtime call failed (message has details)     */
  PF_ERR_TIMEOUT = 6      /* a kernel's bounded wait ran out (pf_sync_check)      */
} pf_status;

enum { PF_CAUSAL_1D = 0, PF_BIDIR_1D = 1, PF_BIDIR_2D = 2 };
enum { PF_INJ_ADD = 0, PF_INJ_GATED = 1, PF_INJ_AFFINE = 2, PF_INJ_CROSS = 3 };
enum { PF_F32 = 0, PF_BF16 = 1 };
enum { PF_F_ATTENTION = 0, PF_F_IDENTITY = 1, PF_F_MLP = 2 };

/* One ProxyFormer layer (Alg. 1; m = ceil(L/P), Sec. 3.1).
 *   batch, L   : sequences and tokens per sequence (2D: L = grid_h*grid_w,
 *                tokens in raster order)
 *   grid_h, grid_w, patch : 2D only; P must equal patch*patch
 *   d, n_heads : proxy width d_proxy = d; head width d/n_heads must be 64
 *   d_fine     : token (local stream) width; 0 means d (the paper's
 *                simplification, Sec. 4).  Another positive multiple of 64
 *                gives the asymmetric history stream of the language model
 *                (Sec. 3.3: d_h = 64 against d = 512): X, X_out, dX are
 *                [batch, L, d_fine], W_c1 is [d, k1*d_fine], W_d1 [k1*d_fine,
 *                d], the gate vectors d_fine wide; 1D bf16 layers with add or
 *                gated injection only
 *   interact   : proxy interaction F (Sec. 3.4): PF_F_ATTENTION (Eq.
 *                proxy-attn), PF_F_IDENTITY (Hbar = H) or PF_F_MLP (Hbar =
 *                W_m2 SiLU(W_m1 H + b_m1) + b_m2, hidden width 4d, one proxy
 *                at a time); other than attention: 1D bf16 only
 *   rope       : 1 rotates the proxies' queries and keys by proxy index before
 *                the attention (RoPE, base 10000, pairs (2j, 2j+1) of each
 *                head); attention, 1D bf16 only
 *   P          : block size (compression ratio) of this layer (Sec. 3.6
 *                allows a different P per layer)
 *   levels     : 1 or 2 (Eq. factor with M = 2); levels == 2 needs k1*k2 == P,
 *                level 1 maps k1 tokens to one row, level 2 k2 rows to a proxy
 *   mode       : PF_CAUSAL_1D | PF_BIDIR_1D | PF_BIDIR_2D (Eq. proxy-attn mask)
 *   inject     : PF_INJ_ADD | PF_INJ_GATED (1D) | PF_INJ_AFFINE (2D) |
 *                PF_INJ_CROSS (1D, bf16): gated cross-attention (Eq. inj-cross
 *                in the gated form of Eq. llm-cross / llm-gate): token t of
 *                block i queries, per head, the interacted proxies j < i
 *                (causal) or all proxies (bidirectional); a per-head gate
 *                alpha = sigmoid(W_a x + b_a) scales each head; X_out = X +
 *                W_ox (alpha * A).  No decompression; a token that sees no
 *                proxy is left unchanged
 *   dtype      : PF_BF16 (fp32 accumulation) or PF_F32                         */
typedef struct {
  int32_t batch, L;
  int32_t grid_h, grid_w, patch;
  int32_t d, n_heads;
  int32_t P, levels, k1, k2;
  int32_t mode, inject, dtype;
  int32_t d_fine;
  int32_t interact, rope;
} pf_layer_desc;

/* Layer parameters (device pointers).  "mat" = dtype, "vec" = fp32.
 *   W_c1 [d, k1*df] mat, b_c1 [d] vec      compression level 1 (or single);
 *                                          df = d_fine (d when 0)
 *   W_c2 [d, k2*d] mat, b_c2 [d] vec       compression level 2 (levels == 2)
 *   W_qkv [3d, d] mat                      proxy Q, K, V projections, stacked
 *   W_o  [d, d] mat                        proxy attention output projection
 *   W_d2 [k2*d, d] mat, b_d2 [k2*d] vec    decompression level 2 (levels == 2)
 *   W_d1 [k1*w, d] mat, b_d1 [k1*w] vec    decompression level 1 (or single);
 *                                          w = df, or 2d for PF_INJ_AFFINE where
 *                                          token p's rows are [s | t] at
 *                                          [2pd, 2pd+d) and [2pd+d, 2(p+1)d)
 *   w_x, w_dlt, b_g [df] vec               gate g = w_x*X + w_dlt*D + b_g
 *                                          (PF_INJ_GATED, Eq. inj-gate)
 *   W_t1 [d, 256] mat, b_t1 [d] vec,       timestep conditioning of the 2D
 *   W_t2 [2d, d] mat, b_t2 [2d] vec        proxies: u = SiLU(W_t1 e(t) + b_t1),
 *                                          [gamma|beta] = W_t2 u + b_t2
 *   W_qa [d + n_heads, d] mat              PF_INJ_CROSS: token queries (rows
 *                                          [0, d)) over the gate rows W_a
 *   b_a [n_heads] vec                      PF_INJ_CROSS: gate bias
 *   W_kvx [2d, d] mat                      PF_INJ_CROSS: proxy keys, values
 *   W_ox [d, d] mat                        PF_INJ_CROSS: output projection
 *   W_m1 [4d, d] mat, b_m1 [4d] vec,       PF_F_MLP: the single-proxy MLP
 *   W_m2 [d, 4d] mat, b_m2 [d] vec
 * Unused pointers may be NULL.                                                  */
typedef struct {
  const void *W_c1;  const float *b_c1;
  const void *W_c2;  const float *b_c2;
  const void *W_qkv; const void *W_o;
  const void *W_d2;  const float *b_d2;
  const void *W_d1;  const float *b_d1;
  const float *w_x, *w_dlt, *b_g;
  const void *W_t1;  const float *b_t1;
  const void *W_t2;  const float *b_t2;
  const void *W_qa;  const float *b_a;
  const void *W_kvx; const void *W_ox;
  const void *W_m1;  const float *b_m1;
  const void *W_m2;  const float *b_m2;
} pf_layer_params;

/* Parameter gradients, fp32 device buffers shaped like pf_layer_params.
 * proxy_layer_bwd overwrites every non-NULL pointer that the layer uses.        */
typedef struct {
  float *W_c1, *b_c1, *W_c2, *b_c2, *W_qkv, *W_o, *W_d2, *b_d2, *W_d1, *b_d1;
  float *w_x, *w_dlt, *b_g, *W_t1, *b_t1, *W_t2, *b_t2;
  float *W_qa, *b_a, *W_kvx, *W_ox;
  float *W_m1, *b_m1, *W_m2, *b_m2;
} pf_layer_grads;

/* Validates a descriptor; PF_OK or the reason it is rejected. */
pf_status proxy_layer_check(const pf_layer_desc *desc);

/* Bytes of the `saved` buffer that proxy_layer_fwd fills for the backward
 * pass (intermediate proxy-side tensors and the decompressed update).       */
size_t proxy_layer_saved_size(const pf_layer_desc *desc);

/* Bytes of workspace needed by proxy_layer_fwd (for_backward = 0; when the
 * forward is given saved == NULL it keeps those tensors in the workspace) or
 * by proxy_layer_bwd (for_backward = 1).  0 on an invalid descriptor.       */
size_t proxy_layer_workspace_size(const pf_layer_desc *desc, int for_backward);

/* Forward of one layer (Alg. 1).
 *   X      [batch, L, d] dtype, device, read only
 *   H_in   [batch, m, d] fp32 incoming proxy state, or NULL for H_in = 0
 *          (Eq. proxy-res degenerates to direct compression)
 *   t      [batch] fp32 flow-matching time (PF_BIDIR_2D only, else NULL)
 *   X_out  [batch, L, d] dtype, device, written (must not alias X)
 *   H_out  [batch, m, d] fp32 proxy state H = H_in + C, or NULL
 *   saved  proxy_layer_saved_size() bytes for the backward, or NULL
 *   ws     workspace of proxy_layer_workspace_size(desc, 0) bytes           */
pf_status proxy_layer_fwd(const pf_layer_desc *desc, const pf_layer_params *params,
                          const void *X, const float *H_in, const float *t,
                          void *X_out, float *H_out, void *saved,
                          void *ws, size_t ws_bytes, void *stream);

/* Backward of one layer: the chain rule through proxy_layer_fwd.
 *   X, H_in, t     the forward's inputs; saved  the forward's saved buffer
 *   dX_out [batch, L, d] dtype: gradient of the loss w.r.t. X_out
 *   dH_out [batch, m, d] fp32 gradient w.r.t. H_out, or NULL for zero
 *   dX     [batch, L, d] dtype, written
 *   dH_in  [batch, m, d] fp32, written if non-NULL
 *   grads  fp32 parameter gradients, overwritten (not accumulated)
 *   ws     workspace of proxy_layer_workspace_size(desc, 1) bytes           */
pf_status proxy_layer_bwd(const pf_layer_desc *desc, const pf_layer_params *params,
                          const void *X, const float *H_in, const float *t,
                          const void *saved, const void *dX_out, const float *dH_out,
                          void *dX, float *dH_in, const pf_layer_grads *grads,
                          void *ws, size_t ws_bytes, void *stream);

/* ---------------------------------------------------------------------------
 * Proxy-only KV cache (Sec. 3.8, Eq. proxy-cache) and streaming decode
 * (Eq. llm-cross, Eq. llm-gate), bf16 with fp32 accumulation.
 *   batch, d, n_heads : head width d/n_heads must be 64 or 128
 *   P, levels, k1, k2 : block size and compression cascade of the append
 *   capacity          : proxy rows the cache can hold per sequence          */
typedef struct {
  int32_t batch, d, n_heads, P, levels, k1, k2, capacity;
} pf_decode_desc;

/* Cache state, all device memory owned by the caller.
 *   K_proxy, V_proxy [batch, capacity, d] bf16  frozen history proxies
 *   X_open           [batch, P, d] bf16         open block's token features
 *   K_open, V_open   [batch, P, d] bf16         their self-attention keys/values
 *   n_proxy, n_open  int32 [batch]              rows in use                     */
typedef struct {
  void *K_proxy, *V_proxy;
  void *X_open, *K_open, *V_open;
  int32_t *n_proxy, *n_open;
} pf_kv_cache;

/* Decode-side parameters (bf16 matrices, fp32 vectors):
 *   W_qkv [3d, d], W_o [d, d], rms_w [d], W_a1 [d/8, d], b_a1 [d/8],
 *   W_a2 [n_heads, d/8], b_a2 [n_heads]   (alpha = sigmoid(MLP(RMSNorm x)))  */
typedef struct {
  const void *W_qkv; const void *W_o; const float *rms_w;
  const void *W_a1;  const float *b_a1; const void *W_a2; const float *b_a2;
} pf_decode_params;

/* Append-side parameters: compression cascade W_c1/b_c1 (+W_c2/b_c2) as in
 * pf_layer_params, and W_kvh [2d, d] bf16 projecting the new proxy to its
 * cached key and value rows.                                                   */
typedef struct {
  const void *W_c1; const float *b_c1; const void *W_c2; const float *b_c2;
  const void *W_kvh;
} pf_append_params;

size_t proxy_decode_workspace_size(const pf_decode_desc *desc);

/* One decode step for every sequence b: q,k,v = W_qkv x_b; (x_b,k,v) are
 * written at open slot n_open[b]; A_x = causal attention over the open slots
 * 0..n_open[b]; A_h = attention over the n_proxy[b] cached proxies (zero if
 * none); A = A_x + alpha (.) A_h per head; y_b = x_b + W_o A; n_open[b] += 1.
 *   x [batch, d] bf16 in, y [batch, d] bf16 out (device).
 * Host-side precondition: the caller guarantees n_open[b] < P (append first
 * when a block is full); the kernel also checks and flags PF_ERR_CAPACITY
 * through pf_sync_check if it is violated, leaving that sequence untouched.  */
pf_status proxy_decode_step(const pf_decode_desc *desc, const pf_decode_params *params,
                            const void *x, pf_kv_cache *cache, void *y,
                            void *ws, size_t ws_bytes, void *stream);

size_t proxy_append_workspace_size(const pf_decode_desc *desc);

/* Block-triggered append (Sec. 3.8): compress each sequence's full open block
 * (n_open[b] == P) into a proxy H = H_in + C(X_open) (Eq. proxy-res), write
 * K_proxy[b, n_proxy[b]] = W_kh H, V_proxy[...] = W_vh H, n_proxy[b] += 1,
 * n_open[b] = 0.  H_in [batch, d] fp32 or NULL.  A sequence whose block is
 * not full, or whose cache is at capacity, is left untouched and flagged
 * (PF_ERR_CAPACITY via pf_sync_check).                                        */
pf_status proxy_kv_append(const pf_decode_desc *desc, const pf_append_params *params,
                          const float *H_in, pf_kv_cache *cache,
                          void *ws, size_t ws_bytes, void *stream);

size_t proxy_prefill_workspace_size(const pf_decode_desc *desc, int32_t L_hist);

/* Bulk prefill of the proxy cache from a history (Sec. 3.8: the prefill stage
 * compresses the historical blocks and caches only their proxies' keys and
 * values).  For every sequence b the history X_hist[b] ([L_hist, d] bf16,
 * sequences contiguous) is split into m = floor(L_hist / P) complete blocks
 * and r = L_hist - m P remaining tokens:
 *   H_i = H_in[b, i] + C(block i)               (Eq. proxy-res, Eq. compress-
 *                                                 linear / factor-cascade)
 *   K_proxy[b, i] = W_kh H_i, V_proxy[b, i] = W_vh H_i       (i < m)
 *   X_open[b, j] = x, K_open[b, j] = W_k x, V_open[b, j] = W_v x   (j < r, x the
 *                                                 history's token m P + j)
 *   n_proxy[b] = m, n_open[b] = r.
 * This equals m block appends (proxy_kv_append) followed by the open-slot
 * writes of r decode steps, and replaces the cache's previous contents.
 * H_in fp32 or NULL, laid out as a layer's proxy stream over the history:
 * [batch, ceil(L_hist / P), d], the row of a partial last block (r > 0)
 * unused.  W_k, W_v are rows [d, 3d) of the decode parameters' W_qkv
 * (dparams is only read when r > 0).  Requires
 * m <= capacity (else PF_ERR_CAPACITY, nothing launched).                    */
pf_status proxy_kv_prefill(const pf_decode_desc *desc, const pf_append_params *aparams,
                           const pf_decode_params *dparams, const void *X_hist, int32_t L_hist,
                           const float *H_in, pf_kv_cache *cache, void *ws, size_t ws_bytes,
                           void *stream);

/* Prefill of one causal layer (Sec. 3.8: the prefill stage runs compression
 * and proxy interaction over the history, then keeps only the proxies' keys
 * and values).  Runs the layer's inference forward over the history X
 * ([batch, L, d] bf16, exactly proxy_layer_fwd with saved = NULL, writing
 * X_out and H_out) and fills `cache` from it:
 *   K_proxy[b, i], V_proxy[b, i] = the keys and values the forward's proxy
 *     attention projected for proxy i < m = floor(L / P) (Eq. proxy-attn), so
 *     the cache's W_kh, W_vh are this layer's W_k, W_v (rows [d, 3d) of its
 *     W_qkv) and later appends must use those same rows as W_kvh;
 *   the open block from the last r = L mod P tokens as in proxy_kv_prefill
 *     (dparams->W_qkv, read only when r > 0); n_proxy[b] = m, n_open[b] = r.
 * cdesc must match the layer (batch, d, n_heads, P, levels, k1, k2); the
 * layer must be PF_CAUSAL_1D in PF_BF16 (else PF_ERR_UNSUPPORTED).  ws needs
 * proxy_layer_workspace_size(desc, 0) bytes.  m > capacity gives
 * PF_ERR_CAPACITY with nothing launched.                                      */
pf_status proxy_layer_prefill(const pf_layer_desc *desc, const pf_layer_params *params,
                              const pf_decode_desc *cdesc, const pf_decode_params *dparams,
                              const void *X, const float *H_in, void *X_out, float *H_out,
                              pf_kv_cache *cache, void *ws, size_t ws_bytes, void *stream);

/* ---------------------------------------------------------------------------
 * Temporal-distance ratios (Sec. 3.6): one causal 1D sequence whose blocks
 * grow coarser with temporal distance.  The sequence is split into n_seg
 * segments in time order; segment s has L tokens, block size P (and, with
 * levels == 2, factors k1 * k2 == P) and its own compression / decompression
 * weights.  The proxies of all segments, in time order, share one causal
 * attention (Eq. proxy-attn, W_qkv and W_o of the shared parameters); the
 * block with global proxy index g receives the interacted proxy g - 1
 * through its own segment's decompression, block 0 nothing; gated (or add)
 * injection with the shared gate vectors.  One segment is the ordinary
 * layer.
 * desc: batch 1, PF_CAUSAL_1D, PF_BF16, PF_INJ_GATED or PF_INJ_ADD,
 * attention interaction without RoPE, d_fine 0, L = the segments' total;
 * its P, k1, k2 are not used (give segs[0]'s).  Every segment but the last
 * has L a multiple of P.  The shared parameters are pf_layer_params' W_qkv,
 * W_o, w_x, w_dlt, b_g; the gradients land in the same fields of
 * pf_layer_grads.  Buffers: X, X_out, dX_out, dX [L, d] bf16.                */
typedef struct { int32_t L, P, k1, k2; } pf_segment;
typedef struct {
  const void *W_c1; const float *b_c1; const void *W_c2; const float *b_c2;  /* [d, k1*d] ... */
  const void *W_d1; const float *b_d1; const void *W_d2; const float *b_d2;  /* [k1*d, d] ... */
} pf_segment_params;
typedef struct {
  float *W_c1, *b_c1, *W_c2, *b_c2, *W_d1, *b_d1, *W_d2, *b_d2;
} pf_segment_grads;

size_t proxy_segments_saved_size(const pf_layer_desc *desc, int32_t n_seg,
                                 const pf_segment *segs);
size_t proxy_segments_workspace_size(const pf_layer_desc *desc, int32_t n_seg,
                                     const pf_segment *segs, int for_backward);
pf_status proxy_segments_fwd(const pf_layer_desc *desc, int32_t n_seg, const pf_segment *segs,
                             const pf_layer_params *shared, const pf_segment_params *seg_params,
                             const void *X, void *X_out, void *saved, void *ws, size_t ws_bytes,
                             void *stream);
pf_status proxy_segments_bwd(const pf_layer_desc *desc, int32_t n_seg, const pf_segment *segs,
                             const pf_layer_params *shared, const pf_segment_params *seg_params,
                             const void *X, const void *saved, const void *dX_out, void *dX,
                             const pf_layer_grads *grads, const pf_segment_grads *seg_grads,
                             void *ws, size_t ws_bytes, void *stream);

/* Thread-local message describing the last non-OK status of this thread. */
const char *pf_last_error(void);

/* Synchronises `stream`, then reports asynchronous CUDA errors and errors
 * flagged by kernels (bounded-wait timeouts, capacity violations) since the
 * previous pf_sync_check, clearing the flag.                                 */
pf_status pf_sync_check(void *stream);

/* Plain bf16 GEMM through the same tcgen05 kernel the layer uses, exposed for
 * testing the contraction on its own (not a paper operation):
 *   D[M, N] (fp32, ldd) = sum_k A[m, k] B[n, k], with
 *   A stored row-major [M, K] (a_mn = 0) or [K, M] (a_mn = 1), and
 *   B stored row-major [N, K] (b_mn = 0) or [K, N] (b_mn = 1), bf16, device.  */
pf_status pf_gemm_bf16(int M, int N, int K, const void *A, int a_mn, const void *B,
                       int b_mn, float *D, int ldd, void *stream);

/* Test utilities for the bounded waits (not paper operations).  Every
 * mbarrier wait of the library's kernels gives up after a time limit (4 s by
 * default), records PF_ERR_TIMEOUT for pf_sync_check, lets its own copies and
 * MMAs land (a separately bounded wait), frees its tensor memory and returns.
 *   pf_debug_set_wait_limit_ns(ns): sets that limit for every kernel launched
 *     afterwards; 0 restores the default.  Synchronous (the device is idle
 *     when it returns).  Returns PF_ERR_CUDA if the device write fails.
 *   pf_debug_gemm_skip_loads(on): while on, the GEMM kernel (pf_gemm_bf16 and
 *     every contraction of the layer) issues none of its operand loads, so its
 *     MMA warp waits for data that never comes and the wait runs out.  Nothing
 *     is in flight when the kernel leaves; the outputs hold garbage.  For tests
 *     of the timeout path only; off by default.                              */
pf_status pf_debug_set_wait_limit_ns(unsigned long long ns);
pf_status pf_debug_gemm_skip_loads(int on);

/* ---------------------------------------------------------------------------
 * Allocation-free backward.  The paper has no counterpart; this is a calling
 * convenience of the library.  Some callers cannot provide a workspace: host
 * frameworks whose memory planner owns all device memory and hands plugins no
 * scratch, and latency-critical loops that cannot pay cudaMalloc's implicit
 * device synchronisation.  This
 * entry point computes exactly what proxy_layer_bwd computes, with its scratch
 * taken from a fixed device array of PF_NOALLOC_SCRATCH_BYTES inside the
 * library instead of a caller buffer; it calls no allocator.  The caller still
 * passes every input and output.
 *   - Layers whose backward needs more scratch than PF_NOALLOC_SCRATCH_BYTES
 *     (proxy_layer_workspace_size(desc, 1)) are rejected with
 *     PF_ERR_WORKSPACE before anything is launched.
 *   - The array exists once per GPU that loads the library and stays
 *     allocated until the process exits.
 *   - The first call on a device looks up the array's device address (with
 *     that device current); make that first call before any stream capture.
 *   - All calls share the one array and the backward writes every scratch
 *     byte before reading it (nothing needs to start at zero); calls whose
 *     execution overlaps on the GPU (other streams, concurrent graphs) race
 *     on the array and must be serialised by the caller.                    */
#define PF_NOALLOC_SCRATCH_BYTES (16u << 20)
pf_status proxy_layer_bwd_noalloc(const pf_layer_desc *desc, const pf_layer_params *params,
                                  const void *X, const float *H_in, const float *t,
                                  const void *saved, const void *dX_out, const float *dH_out,
                                  void *dX, float *dH_in, const pf_layer_grads *grads,
                                  void *stream);

/* ---------------------------------------------------------------------------
 * Launch timing (a measurement utility, not a paper operation).  While enabled,
 * every kernel the library launches is bracketed by two CUDA events recorded
 * on the stream it is launched on, tagged with a label naming the step of the
 * layer it runs and with its algorithmic work (FLOPs, bytes).  After the
 * caller has synchronised, pf_timing_collect() aggregates the records by label
 * and returns the number of labels; the accessors read label i's total
 * elapsed milliseconds, launch count and per-launch algorithmic FLOPs and
 * bytes.  pf_timing_enable(0/1) discards previous records.  Not thread safe.  */
void        pf_timing_enable(int on);
/* FP32 FMA peak probe (measurement utility): `blocks` CTAs of 512 threads,
 * each thread 8 independent fmaf chains of `iters` steps, i.e.
 * blocks * 512 * 8 * iters FMAs = twice that many FLOPs; `out` (device,
 * blocks * 512 floats) receives one value per thread.  The caller times it.  */
pf_status   pf_probe_ffma(void *out, int blocks, int iters, void *stream);
int         pf_timing_collect(void);
const char *pf_timing_label(int i);
double      pf_timing_ms(int i);
int         pf_timing_launches(int i);
double      pf_timing_flops(int i);
double      pf_timing_bytes(int i);

#ifdef __cplusplus
}
#endif
#endif /* PROXYFORMER_H */
