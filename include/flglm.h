/*
 * flglm.h -- C ABI of the FL-GLM server block stack on one GB300 (sm_103a).
 *
 * FL-GLM (arXiv 2406.14898) splits a GLM language model in three (§3.1, Model
 * Split): each client keeps the embedding, block 0, block N-1 and the output
 * layer; the server holds blocks 1..N-2.  A client sends its smashed data h_0,
 * the server returns h_{N-2} = Block_(1,N-2)(h_0), later receives the gradient
 * of the client's loss w.r.t. h_{N-2}, back-propagates it and updates its own
 * parameters.  Under the client-batch strategy (§3.3, Parallel Acceleration) the
 * server stacks the tensors of several clients into one batch and runs them in
 * one pass.  This library is that server: one call per protocol step.
 *
 * Block computed per token row (the ChatGLM-6B block; the paper names the model
 * in §4.1.4 but does not print the block, see the design notes):
 *     a = LN1(x);  [q|k|v] = a Wqkv^T + bqkv;  q,k <- RoPE(position in segment)
 *     o = softmax(q k^T / sqrt(head_dim), causal within the segment) v      (App. A)
 *     h = alpha*a + o Wd^T + bd            (alpha*x when residual_from_ln == 0)
 *     m = LN2(h);  y = alpha*m + gelu_tanh(m W1^T + b1) W2^T + b2  (alpha*h when 0)
 *
 * Conventions for every call:
 *   - Return value: FL_OK (0) or a negative FL_ERR_* code; no exceptions cross the
 *     ABI.  The message of the last failure is in fl_server_last_error().
 *   - All work is enqueued on the handle's CUDA stream (the legacy default stream
 *     unless fl_server_set_stream was called) and is asynchronous.  Device results
 *     are valid after the stream has reached the call (fl_server_sync()).
 *   - Client tensors are DEVICE pointers to bf16 [client_batch, seq_lens[k], hidden],
 *     row-major, contiguous, 16-byte aligned, owned by the caller.  With
 *     client_batch == 1 this is byte-for-byte the paper's {seqlength, batch=1,
 *     hidden} tensor.  Each (client, row) is one causal segment, positions 0..L-1.
 *   - The library owns its parameters (fp32 master, bf16 working copy), gradients,
 *     Adam moments and saved activations; it allocates only in fl_server_create.
 */
#ifndef FLGLM_H
#define FLGLM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define FL_OK 0
#define FL_ERR_INVALID_ARG (-1)  /* null pointer, bad size, misaligned buffer, bad id */
#define FL_ERR_CAPACITY (-2)     /* a size exceeds a fixed capacity: total tokens of a call over
                                  * cfg.max_tokens, or a fixed scratch array's limit */
#define FL_ERR_STATE (-3)        /* protocol order violated (e.g. backward without forward) */
#define FL_ERR_OOM (-4)          /* device allocation failed in fl_server_create */
#define FL_ERR_CUDA (-5)         /* a CUDA runtime/driver call failed */
#define FL_ERR_TIMEOUT (-6)      /* a bounded device-side wait gave up (reported by fl_server_sync) */
#define FL_ERR_UNSUPPORTED (-7)  /* shape the kernels do not support (see fl_server_create) */

typedef struct fl_server* fl_server_t; /* opaque; created and freed by the library */

/* Server configuration.  Sizes: hidden = n_heads * head_dim; hidden % 256 == 0;
 * ffn_hidden % 256 == 0; head_dim in {64, 128}; rotary_dim in {head_dim/2} with
 * rotary_dim % 32 == 0 (the paper's ChatGLM-6B rotates half of each head). */
typedef struct {
  int32_t n_blocks;         /* server blocks (26 for the ChatGLM-6B split, §3.1) */
  int32_t hidden;           /* H */
  int32_t n_heads;          /* nh */
  int32_t head_dim;         /* hd */
  int32_t ffn_hidden;       /* F */
  int32_t rotary_dim;       /* rotated dims at the start of each head; 0 -> head_dim/2 */
  float rope_base;          /* 10000 */
  float ln_eps;             /* 1e-5 */
  float residual_alpha;     /* sqrt(2 * layers of the full model) */
  int32_t residual_from_ln; /* 1: residual = alpha * LN output (GLM block); 0: alpha * LN input */
  int32_t client_batch;     /* rows per client tensor, the same for every client */
  int32_t max_tokens;       /* capacity: most tokens (sum of client_batch * seq_lens) per call */
  int32_t max_seq_len;      /* longest segment accepted; sizes the rotary table (0 -> max_tokens) */
  int32_t recompute;        /* 0: every block's activations are kept (about 1.07 GB per block at
                             * T = 8192, H 4096, F 16384); 1: only the fp32 block inputs are
                             * kept and each block's forward (without its FFN down-projection)
                             * runs again right before its backward: one block's activations
                             * instead of n_blocks, for 2/9 more GEMM FLOPs per step (16 of
                             * 72 H^2 per token and block); results are bit-identical */
  float init_std;           /* N(0, init_std) for weights and biases; LN gamma = 1, beta = 0 */
  float adam_beta1, adam_beta2, adam_eps, weight_decay; /* 0.9, 0.999, 1e-8, 0 */
  int32_t prefix_len;       /* P-tuning v2 (App. A): learnable prefix keys/values per block, 0..128 */
  int32_t freeze_base;      /* 1: only the prefixes are trained (needs prefix_len > 0) */
  int32_t fused_step_min_tokens; /* fl_server_backward_step applies AdamW inside the weight-
                             * gradient GEMMs when the pending call has at least this many
                             * tokens, else it runs the backward and then fl_server_step;
                             * 0 -> 4608 (the crossover measured on GB300: with fewer tokens
                             * the weight-gradient main loop is too short to hide the 26 B per
                             * parameter of the fused update); 1 -> always fused */
  int32_t n_replicas;       /* server-hierarchical strategy (§3.3) on one GPU: 0 or 1 = one
                             * server; 2..4 = that many replicas in one handle, each with its
                             * own parameters, gradients and Adam state (arena of replica r at
                             * r * the per-replica size), started from the same seeded values.
                             * A call's K clients are split in order into n_replicas equal groups
                             * of equal token counts, group r trained by replica r: the block GEMMs
                             * of all replicas run as one batched launch each.  No prefix. */
} fl_server_cfg;

/* Fills *cfg with the ChatGLM-6B server defaults (26 blocks, H 4096, 32 x 128, F 16384,
 * alpha sqrt(56), client_batch 1, max_tokens 8192). */
void fl_server_cfg_default(fl_server_cfg* cfg);

/* Validates cfg, allocates every device buffer (parameters, gradients, Adam moments,
 * activations for cfg->max_tokens tokens) and initialises the parameters on the
 * device from the seeded SplitMix64/Box-Muller streams: tensor t of block b uses the
 * stream keyed (seed, purpose 1, b, t); weights, biases and prefixes N(0, init_std)
 * rounded to fp32, LN gamma = 1, beta = 0.  Gradients and moments start at zero, step 0.
 * With prefix_len > 0 every query of block b also attends to the block's prefix keys and
 * values (P-tuning v2, App. A); with freeze_base the backward computes no block-weight
 * gradients and the step updates only the prefixes (the paper's training setting).
 * Errors: INVALID_ARG (null), UNSUPPORTED (shape), OOM, CUDA.  On failure *out is NULL. */
int fl_server_create(const fl_server_cfg* cfg, uint64_t seed, fl_server_t* out);

/* Client-batched forward (§3.1 h_{N-2} = Block_(1,N-2)(h_0); §3.3 client-batch).
 * client_states[k] (k < K) is client k's bf16 [client_batch, seq_lens[k], hidden] device
 * tensor; out_states[k] receives h_{N-2} in the same layout.  The K tensors are packed
 * into one ragged batch of T = client_batch * sum(seq_lens) tokens with no padding;
 * client k row r is one causal segment.  Inputs may be reused once the stream has
 * passed this call.  Starts a pending step: the next call must be fl_server_backward.
 * Errors: INVALID_ARG (null, K < 1, seq_len < 1, seq_len > max_seq_len, misaligned),
 * CAPACITY (T > max_tokens), STATE (a forward is already pending), CUDA. */
int fl_server_forward(fl_server_t h, const void* const client_states[], const int32_t seq_lens[],
                      int32_t K, void* const out_states[]);

/* fl_server_forward with GLM blank-infilling segments (§4.1.1 casts every task as GLM
 * blank infilling: a context holding a mask token [M], then the answer span).  Segment
 * s = k * client_batch + r (client k, row r) has context_lens[s] context tokens and its
 * [M] at mask_pos[s] (HOST int32 arrays of K * client_batch entries; mask_pos NULL = the
 * last context token, the summarisation layout).  Context tokens attend to the whole
 * context, span tokens to the context and causally to the span; positions are GLM's two
 * streams: context token i has (i, 0), span token i has (mask_pos, i - c + 1); the
 * second stream rotates dims [head_dim/2, head_dim) of q and k (needs rotary_dim =
 * head_dim / 2).  context_lens[s] = 0 keeps segment s plainly causal.  The backward uses
 * the same structure.  Errors: as fl_server_forward, plus INVALID_ARG when
 * context_lens[s] > seq_len or mask_pos[s] is outside [0, context_lens[s]). */
int fl_server_forward_glm(fl_server_t h, const void* const client_states[], const int32_t seq_lens[],
                          int32_t K, const int32_t context_lens[], const int32_t mask_pos[],
                          void* const out_states[]);

/* Backward of the pending forward.  grad_out[k] is client k's bf16 gradient of its
 * loss w.r.t. out_states[k] (same layout); grad_in[k] receives the bf16 gradient
 * w.r.t. client_states[k].  Weight gradients are ADDED (fp32) to the gradient arena,
 * so several forward/backward pairs before one step accumulate (the paper's serial
 * strategy, §3.3).  Errors: INVALID_ARG (null), STATE (no pending forward), CUDA. */
int fl_server_backward(fl_server_t h, const void* const grad_out[], void* const grad_in[]);

/* One AdamW step over every parameter (Adam of §4.1.4 with decoupled weight decay and
 * bias correction): t += 1; m = b1 m + (1-b1) g; v = b2 v + (1-b2) g^2;
 * w -= lr (m/(1-b1^t) / (sqrt(v/(1-b2^t)) + eps) + wd w); refreshes the bf16 copy.
 * Afterwards the gradients are zero (fl_server_get_grad returns zeros): the next
 * backward stores its weight gradients instead of adding them, so the step never has to
 * write the gradient arena.  Errors: STATE (a forward is pending), CUDA. */
int fl_server_step(fl_server_t h, float lr);

/* fl_server_backward followed by fl_server_step(h, lr), in one call.  When no gradients
 * are pending (no backward since the last step), the AdamW update of the four weight
 * matrices of every block runs in the epilogue of their weight-gradient GEMMs: the fp32
 * matrix gradients are never written to memory, and the update's traffic overlaps the
 * tensor-core work.  The bias and LayerNorm vectors get one AdamW launch at the end.
 * Otherwise (gradients accumulated by earlier backward calls, or fewer tokens in the
 * pending call than cfg.fused_step_min_tokens) it runs the two calls as they are.
 * Results equal backward + step up to fp32 rounding.  Errors: as fl_server_backward. */
int fl_server_backward_step(fl_server_t h, const void* const grad_out[], void* const grad_in[], float lr);

/* Frees every device buffer of h after synchronising its stream.  NULL is accepted. */
int fl_server_destroy(fl_server_t h);

/* Routes all later work of h to the given cudaStream_t (NULL = legacy default stream). */
int fl_server_set_stream(fl_server_t h, void* cuda_stream);

/* Synchronises the handle's stream and reads the device status word: returns
 * FL_ERR_TIMEOUT if a kernel's bounded wait gave up since the last sync (the word is
 * then cleared), FL_ERR_CUDA on a CUDA error, else FL_OK. */
int fl_server_sync(fl_server_t h);

/* Parameter tensor ids of a block.  12 and 13 exist when cfg.prefix_len > 0. */
enum {
  FL_T_WQKV = 0, /* [3H, H]: rows [0,H) query, [H,2H) key, [2H,3H) value; head j = rows j*hd.. */
  FL_T_BQKV,     /* [3H] */
  FL_T_WDENSE,   /* [H, H] attention output projection */
  FL_T_BDENSE,   /* [H] */
  FL_T_WUP,      /* [F, H] */
  FL_T_BUP,      /* [F] */
  FL_T_WDOWN,    /* [H, F] */
  FL_T_BDOWN,    /* [H] */
  FL_T_LN1_G,    /* [H] */
  FL_T_LN1_B,    /* [H] */
  FL_T_LN2_G,    /* [H] */
  FL_T_LN2_B,    /* [H] */
  FL_T_BLOCK_COUNT,              /* 12 block tensors */
  FL_T_PREFIX_K = FL_T_BLOCK_COUNT, /* [prefix_len, H]: prefix keys (head j at column j*hd), not rotated */
  FL_T_PREFIX_V,                 /* [prefix_len, H]: prefix values */
  FL_T_COUNT
};

/* Number of elements of tensor tensor_id (same for every block), or -1 if invalid. */
int64_t fl_server_tensor_numel(fl_server_t h, int32_t tensor_id);

/* Synchronous copies between a host fp32 buffer of exactly n elements and the fp32
 * master weights / accumulated gradients / Adam moments of (block, tensor_id).
 * set_param also refreshes the bf16 working copy.  With cfg.n_replicas > 1 the getters read
 * replica 0 and set_param writes every replica.  Errors: INVALID_ARG (ids, n, null). */
int fl_server_get_param(fl_server_t h, int32_t block, int32_t tensor_id, float* host_dst, size_t n);
int fl_server_set_param(fl_server_t h, int32_t block, int32_t tensor_id, const float* host_src, size_t n);
int fl_server_get_grad(fl_server_t h, int32_t block, int32_t tensor_id, float* host_dst, size_t n);
int fl_server_get_adam_moments(fl_server_t h, int32_t block, int32_t tensor_id, float* host_m,
                               float* host_v, size_t n);

/* Server-hierarchical strategy (§3.3): one server replica per client, run side by side,
 * the replicas' parameters averaged at the end of each training period.
 * fl_server_average replaces the fp32 master weights of each of the n replicas (same
 * configuration, same device) by their arithmetic mean (summed in replica order) and
 * refreshes their bf16 copies.  Adam moments and step counts stay per replica (local
 * optimizer state).  It waits for every replica's stream, runs on replicas[0]'s stream
 * and returns after the mean is written.  Errors: INVALID_ARG (n outside 1..64, null,
 * duplicate, different shapes), STATE (a replica has a pending forward), CUDA. */
int fl_server_average(fl_server_t const* replicas, int32_t n);

/* Device address and element count of the fp32 master-weight arena, for averaging across
 * processes (one replica per GPU: all-reduce (sum) the arena, then call
 * fl_server_average_finish).  With cfg.n_replicas > 1 it spans every replica's arena.
 * The arena is owned by the library. */
int fl_server_param_arena(fl_server_t h, float** dev_w, int64_t* n);

/* Completes the §3.3 period-end average across processes: the caller has replaced this
 * replica's master arena by the sum over n_replicas replicas (an all-reduce); this call
 * scales it by 1/n_replicas in fp32, as fl_server_average does (so two replicas give the
 * same bits either way), and refreshes the bf16 working copy, on the handle's stream.
 * Errors: INVALID_ARG (null, n_replicas < 1), STATE (a forward is pending), CUDA. */
int fl_server_average_finish(fl_server_t h, int32_t n_replicas);

/* The period-end average of the replicas of one handle (cfg.n_replicas > 1): every
 * replica's fp32 master weights are replaced by their mean over the replicas (summed in
 * replica order, scaled by 1/n as fl_server_average does) and the bf16 copies refreshed;
 * Adam moments and the step count stay per replica.  Errors: INVALID_ARG (null handle),
 * STATE (a forward is pending), CUDA. */
int fl_server_average_replicas(fl_server_t h);

/* fp32 master values of tensor_id of block `block` of replica `replica` (0 <=
 * replica < cfg.n_replicas, or 0 with one replica) into host_dst[n] (n = the tensor's
 * element count), synchronously; fl_server_get_param reads replica 0.  Errors:
 * INVALID_ARG (replica, block or tensor id out of range, n not the element count, null). */
int fl_server_get_replica_param(fl_server_t h, int32_t replica, int32_t block, int32_t tensor_id, float* host_dst,
                                size_t n);

/* Recomputes the bf16 working copy from the fp32 master weights (after they were changed
 * outside the library), on the handle's stream. */
int fl_server_refresh_working_copy(fl_server_t h);

/* Kernel timing by class (GEMM, attention, LayerNorm, AdamW, other) with CUDA events
 * recorded on the handle's stream around each launch.  enable != 0 starts recording
 * (and clears the totals); fl_server_profile_read fills ms[c] and launches[c] for
 * c < n_classes (n_classes <= FL_PROF_CLASSES) after synchronising the stream. */
enum { FL_PROF_GEMM = 0, FL_PROF_ATTN, FL_PROF_LN, FL_PROF_ADAMW, FL_PROF_OTHER, FL_PROF_CLASSES };
int fl_server_profile(fl_server_t h, int enable);
int fl_server_profile_read(fl_server_t h, double* ms, int64_t* launches, int32_t n_classes);

/* Kernel launches the handle has enqueued since creation (all classes). */
int64_t fl_server_launch_count(fl_server_t h);

/* Message of the last failure of a call on h, or of the calling thread's last failure
 * if h is NULL.  The string stays valid until the next failing call on that thread. */
const char* fl_server_last_error(fl_server_t h);

#ifdef __cplusplus
}
#endif
#endif /* FLGLM_H */
