/*
 * flglm_kernels.h -- kernel-level C ABI of the FL-GLM server library.
 *
 * These entry points launch one hot-path kernel on caller-owned DEVICE buffers.
 * The server calls in flglm.h are built from them; they are exported so that each
 * kernel can be checked on its own against the oracle.  Every pointer is a device
 * pointer unless its name ends in _host; every call is asynchronous on `stream`
 * (a cudaStream_t, NULL = legacy default stream) unless stated.  Return codes are
 * the FL_* codes of flglm.h; the message is in fl_server_last_error(NULL).
 * `status` (optional, device int) receives a nonzero code if a bounded wait inside
 * the kernel gave up; the kernel then returns without finishing its output.
 * Alignment: a pointer must be aligned to the width its kernel accesses it with: 16 bytes
 * for row tensors and parameter vectors read or written in 16-byte pieces (the operands
 * and outputs of the GEMM, LayerNorm, attention, column-sum, AdamW and embedding-gather
 * calls), 8 bytes for the GEMM's rotary table and AdamW's bf16 copy, 4 bytes for per-row
 * scalars and index arrays; a misaligned pointer returns FL_ERR_INVALID_ARG before any
 * work is enqueued.
 */
#ifndef FLGLM_KERNELS_H
#define FLGLM_KERNELS_H

#include <stddef.h>
#include <stdint.h>

#include "flglm.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Element types of the row kernels' and epilogues' activation operands. */
enum { FL_DT_BF16 = 0, FL_DT_F32 = 1 };

/* GEMM epilogues.  acc = sum_k A(m,k) B(n,k) in fp32 (tcgen05, TMEM accumulator). */
enum {
  FL_EPI_STORE = 0,      /* D = acc (+ bias[n] if bias)                                   bf16 */
  FL_EPI_BIAS_GELU = 1,  /* U = acc + bias[n] -> aux_out;  D = gelu_tanh(U)               bf16 */
  FL_EPI_BIAS_RESID = 2, /* D = acc + bias[n] + alpha * R[m,n]                            bf16/fp32 */
  FL_EPI_BIAS_ROPE = 3,  /* D = acc + bias[n]; columns [0, 2*n_heads*head_dim) (q and k) are
                            then rotated: dims [0, rotary_dim) of each head, pairs
                            (i, i + rotary_dim/2), angle pos[m] * rope_base^(-2i/rotary_dim)
                            taken from rope_tab[pos[m]][i] = (cos, sin)                  bf16 */
  FL_EPI_GELU_BWD = 4,   /* D = acc * gelu_tanh'(aux[m,n])   (aux = pre-activation U)     bf16 */
  FL_EPI_RESID = 5,      /* D = acc + alpha * R[m,n]                                      bf16/fp32 */
  FL_EPI_ACCUM_F32 = 6,  /* D[m,n] += acc                                                 fp32 */
  FL_EPI_STORE_F32 = 7,  /* D[m,n] = acc                                                  fp32 */
  FL_EPI_ADAMW = 8,      /* g = acc is a weight gradient: AdamW update of the fp32 weight
                            D[m,n] and its moments adam_m, adam_v (same layout, ldd), the
                            bf16 copy aux_out (ld_aux_out); g itself is not stored      */
  FL_EPI_COUNT
};

/* Tile shapes of fl_gemm_args.tile. */
#define FL_TILE_AUTO 0
#define FL_TILE_128x128 1      /* one SM per 128 x 128 tile */
#define FL_TILE_128x256 2      /* one SM per 128 x 256 tile (N % 256 == 0) */
#define FL_TILE_256x256_PAIR 3 /* a cluster of two SMs per 256 x 256 tile, tcgen05.mma.cta_group::2
                                  (N % 256 == 0) */

/* D[M,N] = epilogue(A . B^T) with bf16 operands.
 * A(m,k) is A[m*lda + k] when a_mn_major == 0 (row-major [M,K]) and A[k*lda + m] when
 * a_mn_major == 1 (row-major [K,M]); B(n,k) likewise with ldb / b_mn_major.
 * Forward GEMMs are (0,0), data-gradient GEMMs (0,1), weight-gradient GEMMs (1,1).
 * Residual epilogues: R = aux (aux_dtype bf16 or fp32), or, when ln_mean != NULL, the
 * LayerNorm of aux recomputed in fp32: R = (aux[m,n] - ln_mean[m]) ln_rstd[m] ln_gamma[n]
 * + ln_beta[n] (this keeps the alpha-scaled residual stream of a block in fp32).
 * d_dtype selects a bf16 or fp32 D for FL_EPI_STORE, FL_EPI_BIAS_RESID and FL_EPI_RESID.
 * Requirements: N % 128 == 0; K % 8 == 0 when a or b is K-major; lda, ldb, ldd,
 * ld_aux, ld_aux_out multiples of 8 elements; pointers 16-byte aligned.  M and K may
 * be ragged (zero-filled by the tensor-memory-accelerator loads). */
typedef struct {
  int32_t M, N, K;
  const void* A; int64_t lda; int32_t a_mn_major;
  const void* B; int64_t ldb; int32_t b_mn_major;
  void* D; int64_t ldd;
  int32_t epilogue;
  const float* bias;            /* [N] fp32 or NULL */
  const void* aux; int64_t ld_aux;          /* bf16 [M,N] for BIAS_RESID / RESID / GELU_BWD */
  float alpha;
  void* aux_out; int64_t ld_aux_out;        /* bf16 [M,N] for BIAS_GELU */
  const int32_t* pos;                       /* [M] positions for BIAS_ROPE */
  const float* rope_tab;                    /* [max_pos][rotary_dim/2][2] for BIAS_ROPE */
  int32_t n_heads, head_dim, rotary_dim;
  int32_t aux_dtype;                        /* FL_DT_BF16 or FL_DT_F32 (residual epilogues) */
  int32_t d_dtype;                          /* FL_DT_BF16 or FL_DT_F32 (STORE / residual epilogues) */
  const float* ln_mean;                     /* [M] or NULL: residual = LayerNorm of aux */
  const float* ln_rstd;                     /* [M] */
  const float* ln_gamma;                    /* [N] */
  const float* ln_beta;                     /* [N] */
  float* adam_m;                            /* FL_EPI_ADAMW: first and second moments */
  float* adam_v;
  float lr, beta1, beta2, eps, weight_decay;   /* FL_EPI_ADAMW hyperparameters */
  float inv_bc1, inv_bc2;                      /* 1 / (1 - beta1^t), 1 / (1 - beta2^t) */
  const int32_t* pos2;                      /* [M] GLM block positions for BIAS_ROPE, or NULL: dims
                                               [rotary_dim, 2*rotary_dim) of each q/k head then turn
                                               by pos2 (2D rotary; needs rotary_dim = head_dim/2) */
  int32_t tile;                             /* FL_TILE_*: tile shape, FL_TILE_AUTO (0) lets the library
                                               pick (256-column tiles on CTA pairs unless smaller tiles
                                               leave clearly fewer SMs idle in the last wave) */
  float* colsum;                            /* FL_EPI_GELU_BWD only, or NULL: colsum[n] += sum over m of
                                               D[m,n] (fp32, before rounding; fp32 atomics, so the
                                               order of the additions is not fixed); 16-byte aligned */
  /* Batched launch (the replicas of the server-hierarchical strategy, §3.3): `batch`
   * independent problems of the same shape and epilogue in one launch (0 or 1: one problem;
   * at most FL_GEMM_MAX_BATCH).  Problem r reads A + r*a_bstride and B + r*b_bstride and its
   * epilogue uses every pointer above offset by r times its stride, in elements of the
   * pointer's own type: D by d_bstride, aux by aux_bstride, aux_out by aux_out_bstride,
   * bias and colsum by bias_bstride, pos, pos2, ln_mean and ln_rstd by row_bstride,
   * ln_gamma and ln_beta by lnp_bstride, adam_m and adam_v by adam_bstride.  Strides keep
   * every problem's pointers 16-byte aligned.  Each problem's result is bit-identical to
   * its own unbatched launch. */
  int32_t batch;
  int64_t a_bstride, b_bstride, d_bstride, aux_bstride, aux_out_bstride;
  int64_t bias_bstride, row_bstride, lnp_bstride, adam_bstride;
} fl_gemm_args;

#define FL_GEMM_MAX_BATCH 4

int fl_k_gemm(const fl_gemm_args* args, int* status, void* stream);

/* n (1..FL_GEMM_MAX_BATCH) problems of one shape run as one launch, each with its own
 * pointers: problem r's tiles follow problem r-1's in one persistent grid, so the last wave
 * of one problem is filled by the next (e.g. the weight gradients of several matrices of
 * one block, which the backward of §3.1 produces side by side).  Every problem is checked
 * as by fl_k_gemm and must share M, N, K, the operand layouts, the epilogue and its
 * scalars (alpha, AdamW hyper-parameters, RoPE arguments and table), tile, and the output
 * leading dimensions ldd, ld_aux, ld_aux_out; A, B, lda and ldb are free per problem.  An
 * optional operand (aux, aux_out, bias, colsum, pos, pos2, LayerNorm, Adam moments) is
 * given for every problem or for none; pos / pos2 / ln_mean / ln_rstd of one problem lie
 * at one offset from problem 0's, as do ln_gamma / ln_beta, bias / colsum, adam_m /
 * adam_v.  batch must be 0 or 1 in every entry.  Results are bit-identical to launching
 * the problems one by one.  Errors: INVALID_ARG (as fl_k_gemm, or the problems differ),
 * UNSUPPORTED, CUDA. */
int fl_k_gemm_multi(const fl_gemm_args* probs, int32_t n, int* status, void* stream);

/* Row LayerNorm, biased variance, fp32 statistics.  x: [T,H] of x_dtype (bf16 or fp32);
 * y: bf16 [T,H]; mean, rstd: [T].  H a multiple of 256 up to 2048, or a multiple of 512 up
 * to 4096 (other H: UNSUPPORTED); T < 0: INVALID_ARG; T = 0 does nothing. */
int fl_k_layernorm_fwd(int32_t T, int32_t H, const void* x, int32_t x_dtype, const float* gamma,
                       const float* beta, float eps, void* y, float* mean, float* rstd, void* stream);

/* LayerNorm backward.  dy, x and resid are [T,H] of io_dtype (bf16 or fp32), H a multiple
 * of 256 up to 4096 (other H: UNSUPPORTED), T < 0: INVALID_ARG, T = 0 does nothing;
 * dx = rstd (g - mean(g) - xhat mean(g xhat)), g = gamma dy, plus resid_alpha * resid[t,:]
 * when resid != NULL; written to dx_bf16 and/or dx_f32 (either may be NULL, not both).
 * dgamma[H] += sum_t dy xhat and dbeta[H] += sum_t dy (fp32, accumulated).
 * workspace: fp32 scratch of at least fl_k_layernorm_bwd_workspace(T, H) bytes. */
size_t fl_k_layernorm_bwd_workspace(int32_t T, int32_t H);
int fl_k_layernorm_bwd(int32_t T, int32_t H, const void* dy, const void* x, int32_t io_dtype, const float* mean,
                       const float* rstd, const float* gamma, const void* resid, float resid_alpha,
                       void* dx_bf16, float* dx_f32, float* dgamma, float* dbeta, void* workspace, void* stream);

/* Allocation-free variant of fl_k_layernorm_bwd for bf16 tensors only: dy, x, resid and
 * the single dx output are bf16 [T,H] (no io_dtype, no fp32 dx, no workspace); results
 * equal fl_k_layernorm_bwd's bf16 dx up to the summation order of dgamma/dbeta.  The paper has no
 * counterpart: this exists for callers that cannot call cudaMalloc, such as a plug-in
 * inside a host framework that owns all device memory through its own pool, a serving
 * loop that must not pay cudaMalloc's implicit device synchronisation, or a process whose
 * device-memory budget is fully reserved.  Its per-CTA partial sums live in a fixed
 * 8 MiB array inside the library image (held by every GPU that loads the library until
 * the process exits); the call allocates nothing.  Limits: H <= 4096 (larger H returns
 * FL_ERR_CAPACITY), at most 256 CTAs; T < 0 returns FL_ERR_INVALID_ARG.  The first call on
 * each device looks up the array's device address (cudaGetSymbolAddress) with that device
 * current and keeps it for the life of the process; make that first call before any stream
 * capture, and do not call this function after cudaDeviceReset in the same process (the
 * kept address would be stale).  All calls share the array: calls that overlap
 * on the GPU race, so serialise them (one stream, or events).  Nothing in the array
 * needs to start at zero: every CTA overwrites its slice before it is read. */
int fl_k_layernorm_bwd_noalloc(int32_t T, int32_t H, const void* dy, const void* x, const float* mean,
                               const float* rstd, const float* gamma, const void* resid, float resid_alpha,
                               void* dx, float* dgamma, float* dbeta, void* stream);

/* Varlen causal attention over packed segments (App. A scale 1/sqrt(head_dim)).
 * qkv: bf16 [T, 3*H] (q | k | v, head j at column j*head_dim of each part, RoPE already
 * applied); cu_seqlens_host / cu_seqlens: host and device copies of int32 [S+1].
 * o: bf16 [T,H]; lse: fp32 [n_heads, T] (log-sum-exp of the scaled scores).
 * tile_ws: device int32 scratch of at least fl_k_attention_tiles(cu_seqlens_host, S) * 2
 * entries.  This call copies the tile list synchronously.  head_dim in {64, 128}.
 * P-tuning v2 (App. A: K' = [prefix_key : key], V' = [prefix_value : value]): with
 * prefix_len in 1..128, prefix_k / prefix_v are bf16 [prefix_len, H] (head j at column
 * j*head_dim), seen by every query before its causal keys; the prefix keys are not
 * rotated.  prefix_len = 0: no prefix (the pointers are ignored).
 * GLM blank infilling (§4.1.1: each task is a context holding a mask token followed by
 * the generated answer span): context_lens, device int32 [S] or NULL, gives segment s a
 * context of context_lens[s] tokens (clamped to [0, L_s]); query t then sees the keys
 * u <= max(t, context_lens[s] - 1) of its segment (bidirectional context, causal span).
 * NULL or 0: plainly causal. */
int32_t fl_k_attention_tiles(const int32_t* cu_seqlens_host, int32_t S);
int fl_k_attention_fwd(int32_t T, int32_t n_heads, int32_t head_dim, const void* qkv,
                       const int32_t* cu_seqlens_host, const int32_t* cu_seqlens, int32_t S,
                       int32_t* tile_ws, void* o, float* lse, const void* prefix_k, const void* prefix_v,
                       int32_t prefix_len, const int32_t* context_lens, void* stream);

/* Attention backward: dqkv (bf16 [T, 3H]) receives dq | dk | dv.  When rope_tab != NULL
 * the inverse rotation by each token's position inside its segment is applied to dq and
 * dk (rotary_dim must be head_dim / 2), giving the gradient w.r.t. the un-rotated q, k.
 * With a prefix, dprefix_k / dprefix_v (fp32 [prefix_len, H]) receive the ADDED gradients
 * of the prefix summed over every segment (fp32 atomics: the summation order varies).
 * delta_ws: fp32 scratch [n_heads * T].  This call copies the tile list synchronously.
 * context_lens: as in the forward.  positions / block_positions: device int32 [T] or NULL;
 * the inverse rotation of dims [0, head_dim/2) uses positions[t] (NULL: the index inside
 * the segment) and, when block_positions != NULL, dims [head_dim/2, head_dim) turn back by
 * block_positions[t] (GLM 2D rotary).  Every position must be below the rows of rope_tab,
 * and rope_tab 16-byte aligned (INVALID_ARG otherwise). */
int fl_k_attention_bwd(int32_t T, int32_t n_heads, int32_t head_dim, const void* qkv, const void* o,
                       const float* lse, const void* dout, const int32_t* cu_seqlens_host,
                       const int32_t* cu_seqlens, int32_t S, int32_t* tile_ws, float* delta_ws,
                       const float* rope_tab, int32_t rotary_dim, void* dqkv, const void* prefix_k,
                       const void* prefix_v, int32_t prefix_len, float* dprefix_k, float* dprefix_v,
                       const int32_t* context_lens, const int32_t* positions, const int32_t* block_positions,
                       void* stream);

/* Client parts (§3.1).  Embedding gather: out[t, :] = table[tokens[t], :] (bf16 [T, H] from
 * a bf16 [vocab, H] table, H % 8 == 0); an id outside [0, vocab) gives a zero row and sets
 * bit 1 of *status (device int).  Scatter-add backward: dtable[tokens[t], :] += dx[t, :]
 * (fp32 atomics, so the order of equal tokens' additions varies; ids outside are skipped). */
int fl_k_embedding_gather(int32_t T, int32_t H, const int32_t* tokens, const void* table, int32_t vocab,
                          void* out, int* status, void* stream);
int fl_k_embedding_scatter_add(int32_t T, int32_t H, const int32_t* tokens, int32_t vocab, const void* dx,
                               float* dtable, void* stream);

/* Cross-entropy of T rows of fp32 logits (row stride ld >= vocab, ld % 4 == 0, 16-byte
 * aligned): count = #{t : 0 <= labels[t] < vocab}; row_loss[t] = logsumexp(row) -
 * logits[t, labels[t]] (0 without a target); *loss = sum(row_loss) / max(count, 1), summed
 * in a fixed order; dlogits (bf16, same stride) = (softmax(row) - onehot(label)) / count
 * on rows with a target, 0 elsewhere and on the columns [vocab, ld).  A label >= vocab is
 * ignored and sets bit 2 of *status. */
int fl_k_cross_entropy(int32_t T, int32_t vocab, int64_t ld, const float* logits, const int32_t* labels,
                       float* row_loss, void* dlogits, float* loss, int* count, int* status, void* stream);

/* AdamW over n contiguous fp32 elements; bc1 = 1 - beta1^t, bc2 = 1 - beta2^t.
 * w_bf16 (optional) receives the rounded new weights; g is zeroed. */
int fl_k_adamw(int64_t n, float* w, float* g, float* m, float* v, void* w_bf16, float lr, float beta1,
               float beta2, float eps, float weight_decay, float bc1, float bc2, void* stream);

/* Client packing (§3.3 client-batch stacks the clients' tensors into one batch):
 * gather copies client buffer k (bytes[k] bytes, a multiple of 16, 16-byte aligned)
 * to packed + sum(bytes[0..k)); scatter copies the other way.  Bit-exact.
 * clients_host is a host array of K device pointers; K <= 4096. */
int fl_k_pack_clients(int32_t K, void* const* clients_host, const int64_t* bytes_host, void* packed, int32_t scatter,
                      void* stream);

/* out[n] += sum_t x[t, n] for bf16 x [T, N] (bias gradients), fp32 out. */
int fl_k_colsum(int32_t T, int32_t N, const void* x, float* out, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* FLGLM_KERNELS_H */
