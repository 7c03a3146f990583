/*
 * flglm_client.h -- C ABI of the FL-GLM client parts (§3.1 Model Split).
 *
 * A client holds the two ends of the model: the embedding layer and block 0 (the
 * "bottom": h_0 = Block_0(Embedding(x)), the smashed data sent to the server) and block
 * N-1 with the output layer (the "top": y' = Linear(Block_{N-1}(h_{N-2})) and the
 * cross-entropy loss against the client's own labels, which never leave it).  Reading of
 * the top (the ChatGLM-6B model the paper uses): a final LayerNorm (eps of the block
 * cfg) before a bias-free LM head; the loss is the mean over the tokens that carry a
 * target.  Each client block is the server's block (same shapes, residual reading,
 * GLM segment structure and, with prefix_len, its own P-tuning v2 prefix).
 *
 * One training round of client k with the server (flglm.h):
 *   fl_client_bottom_forward  -> h_0 ............ fl_server_forward (all clients)
 *   fl_client_top_forward_backward(h_{N-2}) -> loss, dL/dh_{N-2} ... fl_server_backward
 *   fl_client_bottom_backward(dL/dh_0); fl_client_step / fl_server_step
 * and at the end of a period fl_client_average over the clients (§3.3: client-side
 * parameters are averaged like the server's).
 *
 * Every tensor argument is a DEVICE pointer owned by the caller unless its name ends in
 * _host; calls are asynchronous on the handle's stream.  Return codes are the FL_* codes
 * of flglm.h; the message is in fl_client_last_error.
 */
#ifndef FLGLM_CLIENT_H
#define FLGLM_CLIENT_H

#include <stddef.h>
#include <stdint.h>

#include "flglm.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef struct fl_client* fl_client_t;

typedef struct {
  fl_server_cfg block; /* block shape, optimizer, prefix_len, freeze_base, client_batch (rows b per
                          call), max_tokens (capacity b * L), max_seq_len; n_blocks is ignored;
                          n_replicas must be 0 or 1 */
  int32_t vocab;       /* embedding and LM head rows (ChatGLM-6B: 130528) */
} fl_client_cfg;

/* Client parameter groups for get/set/grad; tensor ids inside each group:
 * BOTTOM / TOP: the block tensors FL_T_* of flglm.h (prefixes with prefix_len);
 * EMBED: 0 = table [vocab, H]; HEAD: 0 = LM head weight [vocab, H];
 * FINAL_LN: 0 = gamma [H], 1 = beta [H]. */
enum { FL_CP_BOTTOM = 0, FL_CP_TOP = 1, FL_CP_EMBED = 2, FL_CP_HEAD = 3, FL_CP_FINAL_LN = 4, FL_CP_COUNT };

/* ChatGLM-6B client defaults (the server defaults of fl_server_cfg_default, vocab 130528). */
void fl_client_cfg_default(fl_client_cfg* cfg);

/* Validates cfg (as fl_server_create, plus vocab in [1, 2^24)), allocates every device
 * buffer and initialises the parameters on the device from the seeded streams: block 0 and
 * block N-1 tensor t from (seed, purpose 6, block 0 / 1, t), the embedding from
 * (seed, 6, 2, 0), the LM head from (seed, 6, 3, 0), all N(0, init_std); final LayerNorm
 * gamma = 1, beta = 0.  Clients created with the same seed start from the same model.
 * With freeze_base only the two blocks' prefixes are trained (P-tuning v2, App. A): the
 * embedding, the head and the final LayerNorm then carry no gradient or optimizer state.
 * Errors: INVALID_ARG, UNSUPPORTED, OOM, CUDA.  On failure *out is NULL. */
int fl_client_create(const fl_client_cfg* cfg, uint64_t seed, fl_client_t* out);
int fl_client_destroy(fl_client_t c);
int fl_client_set_stream(fl_client_t c, void* cuda_stream);
/* Waits for the handle's stream; reports TIMEOUT from a bounded device wait and
 * INVALID_ARG when a token id or a label was >= vocab (such tokens embed as zeros, such
 * labels are ignored). */
int fl_client_sync(fl_client_t c);

/* Bottom forward: h0 (bf16 [b, seq_len, H]) = Block_0(Embedding(tokens)); tokens is int32
 * [b, seq_len].  context_lens_host / mask_pos_host (int32 [b] each, or NULL) give the rows
 * the GLM blank-infilling structure of fl_server_forward_glm; both client blocks use it.
 * The token ids are copied: the caller may reuse the buffer once the stream passed.
 * Errors: INVALID_ARG (null, seq_len < 1, b * seq_len > max_tokens, bad context),
 * STATE (a round is already open). */
int fl_client_bottom_forward(fl_client_t c, const int32_t* tokens, int32_t seq_len,
                             const int32_t* context_lens_host, const int32_t* mask_pos_host, void* h0);

/* Top forward and backward of the round opened by fl_client_bottom_forward: h (bf16
 * [b, seq_len, H], the server's h_{N-2}) through block N-1, the final LayerNorm and the
 * LM head (logits kept in fp32); loss (device fp32 scalar) = mean over the targets of
 * -log softmax(logits)[label], labels int32 [b, seq_len], negative = no target; grad_h
 * (bf16 [b, seq_len, H]) receives dloss/dh.  Gradients of the top's trained parameters
 * are ADDED to the client's gradients.  Errors: INVALID_ARG, STATE (no open bottom
 * forward, or the top already ran). */
int fl_client_top_forward_backward(fl_client_t c, const void* h, const int32_t* labels, float* loss,
                                   void* grad_h);

/* Bottom backward: grad_h0 (bf16 [b, seq_len, H], the server's input gradient) through
 * block 0 and the embedding (its rows receive the summed gradients of their tokens, fp32
 * atomics).  Closes the round.  Errors: INVALID_ARG, STATE (the top has not run). */
int fl_client_bottom_backward(fl_client_t c, const void* grad_h0);

/* AdamW step (the server's optimizer and hyperparameters) over every trained client
 * parameter; clears the gradients.  Errors: STATE (a round is open). */
int fl_client_step(fl_client_t c, float lr);

/* Element count of a parameter tensor (0 when absent, -1 on bad ids). */
int64_t fl_client_tensor_numel(fl_client_t c, int32_t part, int32_t tensor);
/* Host copies of fp32 master values / gradients (synchronous).  n must equal the numel. */
int fl_client_get_param(fl_client_t c, int32_t part, int32_t tensor, float* host_dst, size_t n);
int fl_client_set_param(fl_client_t c, int32_t part, int32_t tensor, const float* host_src, size_t n);
int fl_client_get_grad(fl_client_t c, int32_t part, int32_t tensor, float* host_dst, size_t n);

/* End of a training period (§3.3): every client's parameters become the fp32 mean over
 * the n clients (summed in list order), bf16 copies refreshed; optimizer moments and step
 * counts stay local.  The clients must have the same cfg and no open round.  Synchronous. */
int fl_client_average(fl_client_t const* clients, int32_t n);

/* Kernels this handle (and its two blocks) has launched so far. */
int64_t fl_client_launch_count(fl_client_t c);
const char* fl_client_last_error(fl_client_t c);

#ifdef __cplusplus
}
#endif

#endif /* FLGLM_CLIENT_H */
