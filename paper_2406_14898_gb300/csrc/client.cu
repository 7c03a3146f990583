// Client parts of the FL-GLM split (§3.1 Model Split): the C ABI of flglm_client.h.
//
// bottom: h_0 = Block_0(Embedding(x));  top: loss = CE(Linear(LN(Block_{N-1}(h_{N-2})))).
// The two blocks are one-block server handles (same kernels, arenas and optimizer as the
// server stack, seeded from the client's own streams).  The client's own parameters
// (embedding [V, H], LM head [Vp, H] with the vocabulary padded to a multiple of 256 by
// zero rows, final LayerNorm gamma/beta) live in one flat arena like the server's, so one
// AdamW launch updates them all.
//
// Kernels here: embedding gather (warp per token, 16-byte rows) and its scatter-add
// backward (fp32 atomics); the target count; the cross-entropy row kernel (one CTA per
// row: online max / sum-exp over the fp32 logits, then the bf16 logit gradient
// (softmax - onehot) / n_targets, zero on the padded columns); the fixed-order loss sum.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdarg>
#include <cstring>
#include <string>
#include <vector>

#include "../../include/flglm.h"
#include "../../include/flglm_client.h"
#include "../../include/flglm_kernels.h"
#include "common.cuh"
#include "kernels.cuh"

int fl_server_create_keyed(const fl_server_cfg* cfg, uint64_t seed, int purpose, int block0, fl_server_t* out);

namespace {

typedef __nv_bfloat16 bf16;
constexpr int CE_THREADS = 512;
constexpr int RED_THREADS = 1024;
constexpr int ST_TOKEN = 1, ST_LABEL = 2;  // client status bits: token / label id >= vocab
constexpr int PURPOSE_CLIENT = 6;
constexpr int BLOCK_BOTTOM = 0, BLOCK_TOP = 1, BLOCK_EMBED = 2, BLOCK_HEAD = 3;

// ---------------------------------------------------------------------------- kernels

__global__ void embed_gather_kernel(int T, int H, const int32_t* __restrict__ tokens, const bf16* __restrict__ table,
                                    int V, bf16* __restrict__ out, int* __restrict__ status) {
  const int64_t w = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (w >= T) return;
  const int tok = tokens[w];
  const bool ok = tok >= 0 && tok < V;
  if (!ok && lane == 0) atomicOr(status, ST_TOKEN);
  const uint4* src = reinterpret_cast<const uint4*>(table + (int64_t)(ok ? tok : 0) * H);
  uint4* dst = reinterpret_cast<uint4*>(out + w * H);
  for (int i = lane; i < H / 8; i += 32) dst[i] = ok ? __ldg(src + i) : make_uint4(0u, 0u, 0u, 0u);
}

__global__ void embed_scatter_kernel(int T, int H, const int32_t* __restrict__ tokens, int V,
                                     const bf16* __restrict__ dX, float* __restrict__ dE) {
  const int64_t w = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (w >= T) return;
  const int tok = tokens[w];
  if (tok < 0 || tok >= V) return;
  const uint32_t* src = reinterpret_cast<const uint32_t*>(dX + w * H);
  float* dst = dE + (int64_t)tok * H;
  for (int i = lane; i < H / 2; i += 32) {
    const float2 v = unpack_bf16x2(src[i]);
    atomicAdd(dst + 2 * i, v.x);
    atomicAdd(dst + 2 * i + 1, v.y);
  }
}

template <typename T>
FL_DEV T block_sum(T v, T* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  T s = 0;
  for (int i = 0; i < nw; ++i) s += red[i];  // fixed order
  return s;
}

__global__ void __launch_bounds__(RED_THREADS) count_kernel(int T, const int32_t* __restrict__ labels, int V,
                                                            int* __restrict__ count, int* __restrict__ status) {
  __shared__ int red[32];
  int c = 0, bad = 0;
  for (int t = threadIdx.x; t < T; t += blockDim.x) {
    const int y = labels[t];
    c += (y >= 0 && y < V);
    bad |= (y >= V);
  }
  c = block_sum(c, red);
  if (threadIdx.x == 0) *count = c;
  if (bad) atomicOr(status, ST_LABEL);
}

// (max, sum of exp(x - max)) pairs: combine two partial softmax denominators
FL_DEV void lse_combine(float& m, float& s, float m2, float s2) {
  const float mn = fmaxf(m, m2);
  if (mn == -INFINITY) return;  // both empty
  s = (m == -INFINITY ? 0.f : s * __expf(m - mn)) + (m2 == -INFINITY ? 0.f : s2 * __expf(m2 - mn));
  m = mn;
}

__global__ void __launch_bounds__(CE_THREADS) ce_kernel(int V, int64_t ld, const float* __restrict__ logits,
                                                        const int32_t* __restrict__ labels,
                                                        const int* __restrict__ count, float* __restrict__ row_loss,
                                                        bf16* __restrict__ dlogits) {
  __shared__ float rm[CE_THREADS / 32], rs[CE_THREADS / 32];
  const int row = blockIdx.x;
  const float* l = logits + (int64_t)row * ld;
  // pass 1: online max and sum of exponentials
  float m = -INFINITY, s = 0.f;
  const int V4 = V / 4;
  for (int j = threadIdx.x; j < V4; j += blockDim.x) {
    const float4 x = __ldg(reinterpret_cast<const float4*>(l) + j);
    const float xs[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) lse_combine(m, s, xs[q], 1.f);
  }
  for (int j = 4 * V4 + threadIdx.x; j < V; j += blockDim.x) lse_combine(m, s, __ldg(l + j), 1.f);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o), s2 = __shfl_xor_sync(0xffffffffu, s, o);
    lse_combine(m, s, m2, s2);
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) {
    rm[warp] = m;
    rs[warp] = s;
  }
  __syncthreads();
  m = -INFINITY;
  s = 0.f;
  for (int i = 0; i < CE_THREADS / 32; ++i) lse_combine(m, s, rm[i], rs[i]);
  const float lse = m + __logf(s);
  const int y = labels[row];
  const bool valid = y >= 0 && y < V;
  const float inv = valid ? 1.f / (float)max(*count, 1) : 0.f;
  if (threadIdx.x == 0) row_loss[row] = valid ? lse - l[y] : 0.f;
  // pass 2: gradient of the mean loss w.r.t. the logits, 4 columns per thread; the
  // padded columns [V, ld) get zeros
  bf16* d = dlogits + (int64_t)row * ld;
  const int ld4 = (int)(ld / 4);
  for (int j4 = threadIdx.x; j4 < ld4; j4 += blockDim.x) {
    float g[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int j = 4 * j4 + q;
      g[q] = j < V ? (__expf(__ldg(l + j) - lse) - (j == y ? 1.f : 0.f)) * inv : 0.f;
    }
    *reinterpret_cast<uint2*>(d + 4 * j4) = make_uint2(pack_bf16x2(g[0], g[1]), pack_bf16x2(g[2], g[3]));
  }
}

__global__ void __launch_bounds__(RED_THREADS) loss_kernel(int T, const float* __restrict__ row_loss,
                                                           const int* __restrict__ count, float* __restrict__ loss) {
  __shared__ float red[32];
  float s = 0.f;
  for (int t = threadIdx.x; t < T; t += blockDim.x) s += row_loss[t];
  s = block_sum(s, red);
  if (threadIdx.x == 0) *loss = s / (float)max(*count, 1);
}

int warps_grid(int64_t rows) { return (int)((rows * 32 + 255) / 256); }

}  // namespace

// ---------------------------------------------------------------------------- kernel-level API

extern "C" int fl_k_embedding_gather(int32_t T, int32_t H, const int32_t* tokens, const void* table, int32_t vocab,
                                     void* out, int* status, void* stream) {
  if (T < 0 || H <= 0 || (H % 8) || vocab < 1 || !tokens || !table || !out || !status)
    return fl_internal_error(FL_ERR_INVALID_ARG, "embedding gather: args");
  if (fl_misaligned(table, 16) || fl_misaligned(out, 16) || fl_misaligned(tokens, 4) || fl_misaligned(status, 4))
    return fl_internal_error(FL_ERR_INVALID_ARG, "embedding gather: table and out must be 16-byte aligned");
  if (T == 0) return FL_OK;
  embed_gather_kernel<<<warps_grid(T), 256, 0, (cudaStream_t)stream>>>(T, H, tokens, (const bf16*)table, vocab,
                                                                       (bf16*)out, status);
  FL_CUDA_TRY(cudaGetLastError());
  return FL_OK;
}

extern "C" int fl_k_embedding_scatter_add(int32_t T, int32_t H, const int32_t* tokens, int32_t vocab, const void* dx,
                                          float* dtable, void* stream) {
  if (T < 0 || H <= 0 || (H % 2) || vocab < 1 || !tokens || !dx || !dtable)
    return fl_internal_error(FL_ERR_INVALID_ARG, "embedding scatter: args");
  if (fl_misaligned(dx, 4) || fl_misaligned(dtable, 4) || fl_misaligned(tokens, 4))
    return fl_internal_error(FL_ERR_INVALID_ARG, "embedding scatter: dx, dtable and tokens must be 4-byte aligned");
  if (T == 0) return FL_OK;
  embed_scatter_kernel<<<warps_grid(T), 256, 0, (cudaStream_t)stream>>>(T, H, tokens, vocab, (const bf16*)dx, dtable);
  FL_CUDA_TRY(cudaGetLastError());
  return FL_OK;
}

extern "C" int fl_k_cross_entropy(int32_t T, int32_t vocab, int64_t ld, const float* logits, const int32_t* labels,
                                  float* row_loss, void* dlogits, float* loss, int* count, int* status, void* stream) {
  if (T < 0 || vocab < 1 || ld < vocab || (ld % 4) || !logits || !labels || !row_loss || !dlogits || !loss ||
      !count || !status)
    return fl_internal_error(FL_ERR_INVALID_ARG, "cross entropy: args");
  if ((reinterpret_cast<uintptr_t>(logits) & 15) || (reinterpret_cast<uintptr_t>(dlogits) & 7))
    return fl_internal_error(FL_ERR_INVALID_ARG, "cross entropy: alignment");
  cudaStream_t st = (cudaStream_t)stream;
  count_kernel<<<1, RED_THREADS, 0, st>>>(T, labels, vocab, count, status);
  if (T > 0) ce_kernel<<<T, CE_THREADS, 0, st>>>(vocab, ld, logits, labels, count, row_loss, (bf16*)dlogits);
  loss_kernel<<<1, RED_THREADS, 0, st>>>(T, row_loss, count, loss);
  FL_CUDA_TRY(cudaGetLastError());
  return FL_OK;
}

// ---------------------------------------------------------------------------- client handle

struct fl_client {
  fl_client_cfg cfg;
  fl_server_t bottom = nullptr, top = nullptr;
  cudaStream_t stream = nullptr;
  std::string err;
  int H = 0, V = 0, Tm = 0;
  int64_t Vp = 0;
  bool train_own = true;
  // own parameter arena: [embedding V*H | head Vp*H | gamma H | beta H], 64-byte aligned parts
  int64_t off_embed = 0, off_head = 0, off_lnf = 0, n_own = 0;
  float *w = nullptr, *g = nullptr, *m = nullptr, *v = nullptr;
  bf16* wb = nullptr;
  float* lnf_scratch = nullptr;  // dgamma / dbeta sink when the LayerNorm is frozen
  int64_t step_t = 0;
  // activations
  int32_t* tokens = nullptr;
  bf16 *x0 = nullptr, *dx0 = nullptr, *y = nullptr, *z = nullptr, *dz = nullptr, *dy = nullptr;
  float *mean = nullptr, *rstd = nullptr, *logits = nullptr, *row_loss = nullptr, *ln_ws = nullptr;
  bf16* dlogits = nullptr;
  int *count = nullptr, *status = nullptr, *gemm_status = nullptr;
  std::vector<void*> allocations;
  // the open round
  int phase = 0;  // 0 idle, 1 bottom forward done, 2 top done
  int b = 0, L = 0, T = 0;
  std::vector<int32_t> ctx, mpos;
  bool glm = false;
  int64_t launches = 0;
};

namespace {

int cl_err(fl_client* c, int rc) {  // copies the message of a failed internal call
  if (rc != FL_OK && c) c->err = fl_server_last_error(nullptr);
  return rc;
}
int cl_set(fl_client* c, int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  fl_internal_error(code, "%s", buf);
  if (c) c->err = buf;
  return code;
}
int srv_err(fl_client* c, fl_server_t s, int rc) {  // message of a failed block call
  if (rc != FL_OK && c) c->err = fl_server_last_error(s);
  return rc;
}

template <typename T>
int calloc_dev(fl_client* c, T** p, size_t count) {
  void* q = nullptr;
  const size_t bytes = count * sizeof(T) + 256;
  if (cudaMalloc(&q, bytes) != cudaSuccess) {
    cudaGetLastError();
    return cl_set(c, FL_ERR_OOM, "client: cudaMalloc of %zu bytes failed", bytes);
  }
  c->allocations.push_back(q);
  *p = reinterpret_cast<T*>(q);
  return FL_OK;
}

int64_t round_up(int64_t x, int64_t a) { return (x + a - 1) / a * a; }

uint64_t mix64_h(uint64_t z) {
  z ^= z >> 30;
  z *= 0xBF58476D1CE4E5B9ull;
  z ^= z >> 27;
  z *= 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}
uint64_t client_key(uint64_t seed, uint64_t block, uint64_t tensor) {
  const uint64_t tag = ((uint64_t)PURPOSE_CLIENT << 56) | (block << 40) | (tensor << 32);
  return mix64_h(mix64_h(seed + 0x9E3779B97F4A7C15ull) ^ tag);
}

int run_gemm(fl_client* c, const fl_gemm_args& a) {
  c->launches += 1;
  return cl_err(c, fl_k_gemm(&a, c->gemm_status, c->stream));
}

fl_gemm_args gemm_base() {
  fl_gemm_args a;
  memset(&a, 0, sizeof a);
  return a;
}

fl_server_t part_server(fl_client* c, int part) {
  return part == FL_CP_BOTTOM ? c->bottom : part == FL_CP_TOP ? c->top : nullptr;
}

// own tensor (part, t) -> (offset, numel), or -1
int64_t own_tensor(const fl_client* c, int part, int t, int64_t* n) {
  const int64_t H = c->H;
  if (part == FL_CP_EMBED && t == 0) {
    *n = (int64_t)c->V * H;
    return c->off_embed;
  }
  if (part == FL_CP_HEAD && t == 0) {
    *n = (int64_t)c->V * H;  // the padded rows are not part of the parameter
    return c->off_head;
  }
  if (part == FL_CP_FINAL_LN && (t == 0 || t == 1)) {
    *n = H;
    return c->off_lnf + t * round_up(H, 16);
  }
  return -1;
}

}  // namespace

extern "C" void fl_client_cfg_default(fl_client_cfg* cfg) {
  if (!cfg) return;
  fl_server_cfg_default(&cfg->block);
  cfg->block.n_blocks = 1;
  cfg->vocab = 130528;
}

extern "C" int fl_client_destroy(fl_client_t c) {
  if (!c) return FL_OK;
  cudaStreamSynchronize(c->stream);
  fl_server_destroy(c->bottom);
  fl_server_destroy(c->top);
  for (void* p : c->allocations) cudaFree(p);
  delete c;
  return FL_OK;
}

extern "C" int fl_client_create(const fl_client_cfg* cfg, uint64_t seed, fl_client_t* out) {
  if (!out) return fl_internal_error(FL_ERR_INVALID_ARG, "client create: out is null");
  *out = nullptr;
  if (!cfg) return fl_internal_error(FL_ERR_INVALID_ARG, "client create: cfg is null");
  if (cfg->vocab < 1 || cfg->vocab >= (1 << 24))
    return fl_internal_error(FL_ERR_INVALID_ARG, "client create: vocab %d outside [1, 2^24)", cfg->vocab);
  if (cfg->block.n_replicas > 1)
    return fl_internal_error(FL_ERR_INVALID_ARG, "client create: block.n_replicas %d (a client has one replica)",
                             cfg->block.n_replicas);
  fl_client* c = new fl_client();
  c->cfg = *cfg;
  c->cfg.block.n_blocks = 1;
  auto fail = [&](int rc) {
    c->err.clear();
    fl_client_destroy(c);
    return rc;
  };
  int rc;
  if ((rc = fl_server_create_keyed(&c->cfg.block, seed, PURPOSE_CLIENT, BLOCK_BOTTOM, &c->bottom)) ||
      (rc = fl_server_create_keyed(&c->cfg.block, seed, PURPOSE_CLIENT, BLOCK_TOP, &c->top)))
    return fail(rc);
  const fl_server_cfg& bc = c->cfg.block;
  c->H = bc.hidden;
  c->V = cfg->vocab;
  c->Vp = round_up(c->V, 256);
  c->Tm = bc.max_tokens;
  c->train_own = bc.freeze_base == 0;
  const int64_t H = c->H, Tm = c->Tm;
  c->off_embed = 0;
  c->off_head = round_up((int64_t)c->V * H, 16);
  c->off_lnf = c->off_head + c->Vp * H;
  c->n_own = c->off_lnf + 2 * round_up(H, 16);
  if ((rc = calloc_dev(c, &c->w, c->n_own)) || (rc = calloc_dev(c, &c->wb, c->n_own))) return fail(rc);
  if (c->train_own) {
    if ((rc = calloc_dev(c, &c->g, c->n_own)) || (rc = calloc_dev(c, &c->m, c->n_own)) ||
        (rc = calloc_dev(c, &c->v, c->n_own)))
      return fail(rc);
  } else if ((rc = calloc_dev(c, &c->lnf_scratch, 2 * H))) {
    return fail(rc);
  }
  if ((rc = calloc_dev(c, &c->tokens, Tm)) || (rc = calloc_dev(c, &c->x0, Tm * H)) ||
      (rc = calloc_dev(c, &c->dx0, Tm * H)) || (rc = calloc_dev(c, &c->y, Tm * H)) ||
      (rc = calloc_dev(c, &c->z, Tm * H)) || (rc = calloc_dev(c, &c->dz, Tm * H)) ||
      (rc = calloc_dev(c, &c->dy, Tm * H)) || (rc = calloc_dev(c, &c->mean, Tm)) ||
      (rc = calloc_dev(c, &c->rstd, Tm)) || (rc = calloc_dev(c, &c->logits, Tm * c->Vp)) ||
      (rc = calloc_dev(c, &c->dlogits, Tm * c->Vp)) || (rc = calloc_dev(c, &c->row_loss, Tm)) ||
      (rc = calloc_dev(c, &c->ln_ws, fl_k_layernorm_bwd_workspace((int32_t)Tm, (int32_t)H) / sizeof(float))) ||
      (rc = calloc_dev(c, &c->count, 1)) || (rc = calloc_dev(c, &c->status, 2)))
    return fail(rc);
  c->gemm_status = c->status + 1;
  // parameters: zero everything (the head's padded rows stay zero), then the seeded draws
  cudaStream_t st = nullptr;
  if (cudaMemset(c->w, 0, c->n_own * sizeof(float)) != cudaSuccess ||
      (c->g && cudaMemset(c->g, 0, c->n_own * sizeof(float)) != cudaSuccess) ||
      (c->m && cudaMemset(c->m, 0, c->n_own * sizeof(float)) != cudaSuccess) ||
      (c->v && cudaMemset(c->v, 0, c->n_own * sizeof(float)) != cudaSuccess) ||
      cudaMemset(c->status, 0, 2 * sizeof(int)) != cudaSuccess)
    return fail(cl_set(c, FL_ERR_CUDA, "client create: memset"));
  const double std_ = (double)bc.init_std;
  if ((rc = fl_launch_normal_init((int64_t)c->V * H, client_key(seed, BLOCK_EMBED, 0), 0.0, std_, c->w + c->off_embed,
                                  st)) ||
      (rc = fl_launch_normal_init((int64_t)c->V * H, client_key(seed, BLOCK_HEAD, 0), 0.0, std_, c->w + c->off_head,
                                  st)) ||
      (rc = fl_launch_fill(H, 1.f, c->w + c->off_lnf, st)) ||
      (rc = fl_launch_f32_to_bf16(c->n_own, c->w, c->wb, st)))
    return fail(rc);
  if (cudaDeviceSynchronize() != cudaSuccess) return fail(cl_set(c, FL_ERR_CUDA, "client create: init"));
  *out = c;
  return FL_OK;
}

extern "C" int fl_client_set_stream(fl_client_t c, void* s) {
  if (!c) return fl_internal_error(FL_ERR_INVALID_ARG, "client set_stream: null handle");
  c->stream = reinterpret_cast<cudaStream_t>(s);
  fl_server_set_stream(c->bottom, s);
  fl_server_set_stream(c->top, s);
  return FL_OK;
}

extern "C" int fl_client_sync(fl_client_t c) {
  if (!c) return fl_internal_error(FL_ERR_INVALID_ARG, "client sync: null handle");
  if (int rc = fl_server_sync(c->bottom)) return srv_err(c, c->bottom, rc);
  if (int rc = fl_server_sync(c->top)) return srv_err(c, c->top, rc);
  cudaError_t e = cudaStreamSynchronize(c->stream);
  int st[2] = {0, 0};
  if (e == cudaSuccess) e = cudaMemcpy(st, c->status, sizeof st, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cl_set(c, FL_ERR_CUDA, "client sync: %s", cudaGetErrorString(e));
  if (st[0] || st[1]) cudaMemset(c->status, 0, sizeof st);
  if (st[1]) return cl_set(c, FL_ERR_TIMEOUT, "client: a bounded device wait gave up (code %d)", st[1]);
  if (st[0] & ST_TOKEN) return cl_set(c, FL_ERR_INVALID_ARG, "client: a token id was outside [0, vocab)");
  if (st[0] & ST_LABEL) return cl_set(c, FL_ERR_INVALID_ARG, "client: a label was >= vocab (ignored)");
  return FL_OK;
}

extern "C" int fl_client_bottom_forward(fl_client_t c, const int32_t* tokens, int32_t seq_len,
                                        const int32_t* context_lens_host, const int32_t* mask_pos_host, void* h0) {
  if (!c) return fl_internal_error(FL_ERR_INVALID_ARG, "bottom_forward: null handle");
  if (c->phase != 0) return cl_set(c, FL_ERR_STATE, "bottom_forward: a round is open (finish it with bottom_backward)");
  if (!tokens || !h0) return cl_set(c, FL_ERR_INVALID_ARG, "bottom_forward: null tokens or h0");
  const int b = c->cfg.block.client_batch;
  if (seq_len < 1 || (int64_t)b * seq_len > c->Tm)
    return cl_set(c, FL_ERR_INVALID_ARG, "bottom_forward: %d x %d tokens outside [1, max_tokens %d]", b, seq_len, c->Tm);
  c->b = b;
  c->L = seq_len;
  c->T = b * seq_len;
  c->glm = context_lens_host != nullptr;
  if (c->glm) {
    c->ctx.assign(context_lens_host, context_lens_host + b);
    if (mask_pos_host) c->mpos.assign(mask_pos_host, mask_pos_host + b);
    else c->mpos.clear();
  }
  cudaError_t e = cudaMemcpyAsync(c->tokens, tokens, (size_t)c->T * sizeof(int32_t), cudaMemcpyDeviceToDevice, c->stream);
  if (e != cudaSuccess) return cl_set(c, FL_ERR_CUDA, "bottom_forward: token copy: %s", cudaGetErrorString(e));
  embed_gather_kernel<<<warps_grid(c->T), 256, 0, c->stream>>>(c->T, c->H, c->tokens, c->wb + c->off_embed, c->V, c->x0,
                                                               c->status);
  c->launches += 1;
  if ((e = cudaGetLastError()) != cudaSuccess) return cl_set(c, FL_ERR_CUDA, "embed gather: %s", cudaGetErrorString(e));
  const void* in[1] = {c->x0};
  void* outp[1] = {h0};
  const int32_t lens[1] = {seq_len};
  int rc = c->glm ? fl_server_forward_glm(c->bottom, in, lens, 1, c->ctx.data(), c->mpos.empty() ? nullptr : c->mpos.data(), outp)
                  : fl_server_forward(c->bottom, in, lens, 1, outp);
  if (rc) return srv_err(c, c->bottom, rc);
  c->phase = 1;
  return FL_OK;
}

extern "C" int fl_client_top_forward_backward(fl_client_t c, const void* h, const int32_t* labels, float* loss,
                                              void* grad_h) {
  if (!c) return fl_internal_error(FL_ERR_INVALID_ARG, "top: null handle");
  if (c->phase != 1) return cl_set(c, FL_ERR_STATE, "top: needs an open round after bottom_forward");
  if (!h || !labels || !loss || !grad_h) return cl_set(c, FL_ERR_INVALID_ARG, "top: null argument");
  const int T = c->T, H = c->H;
  cudaStream_t st = c->stream;
  // block N-1 on the server's h_{N-2}
  const void* in[1] = {h};
  void* outp[1] = {c->y};
  const int32_t lens[1] = {c->L};
  int rc = c->glm ? fl_server_forward_glm(c->top, in, lens, 1, c->ctx.data(), c->mpos.empty() ? nullptr : c->mpos.data(), outp)
                  : fl_server_forward(c->top, in, lens, 1, outp);
  if (rc) return srv_err(c, c->top, rc);
  // z = final LayerNorm(y); logits = z W_head^T (fp32)
  float* gamma = c->w + c->off_lnf;
  float* beta = gamma + round_up(H, 16);
  c->launches += 1;
  if ((rc = fl_k_layernorm_fwd(T, H, c->y, FL_DT_BF16, gamma, beta, c->cfg.block.ln_eps, c->z, c->mean, c->rstd, st)))
    return cl_err(c, rc);
  fl_gemm_args a = gemm_base();
  a.M = T; a.N = (int32_t)c->Vp; a.K = H;
  a.A = c->z; a.lda = H;
  a.B = c->wb + c->off_head; a.ldb = H;
  a.D = c->logits; a.ldd = c->Vp;
  a.epilogue = FL_EPI_STORE_F32;
  if ((rc = run_gemm(c, a))) return rc;
  // loss and dloss/dlogits
  count_kernel<<<1, RED_THREADS, 0, st>>>(T, labels, c->V, c->count, c->status);
  ce_kernel<<<T, CE_THREADS, 0, st>>>(c->V, c->Vp, c->logits, labels, c->count, c->row_loss, c->dlogits);
  loss_kernel<<<1, RED_THREADS, 0, st>>>(T, c->row_loss, c->count, loss);
  c->launches += 3;
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cl_set(c, FL_ERR_CUDA, "cross-entropy: %s", cudaGetErrorString(e));
  // head gradient (accumulated), then dz = dlogits W_head
  if (c->train_own) {
    fl_gemm_args wg = gemm_base();
    wg.M = (int32_t)c->Vp; wg.N = H; wg.K = T;
    wg.A = c->dlogits; wg.lda = c->Vp; wg.a_mn_major = 1;
    wg.B = c->z; wg.ldb = H; wg.b_mn_major = 1;
    wg.D = c->g + c->off_head; wg.ldd = H;
    wg.epilogue = FL_EPI_ACCUM_F32;
    if ((rc = run_gemm(c, wg))) return rc;
  }
  fl_gemm_args dg = gemm_base();
  dg.M = T; dg.N = H; dg.K = (int32_t)c->Vp;
  dg.A = c->dlogits; dg.lda = c->Vp;
  dg.B = c->wb + c->off_head; dg.ldb = H; dg.b_mn_major = 1;
  dg.D = c->dz; dg.ldd = H;
  dg.epilogue = FL_EPI_STORE;
  if ((rc = run_gemm(c, dg))) return rc;
  // final LayerNorm backward (its gamma/beta gradients accumulate, or go to a sink)
  float* dgam = c->train_own ? c->g + c->off_lnf : c->lnf_scratch;
  float* dbet = c->train_own ? dgam + round_up(H, 16) : c->lnf_scratch + H;
  c->launches += 2;
  if ((rc = fl_k_layernorm_bwd(T, H, c->dz, c->y, FL_DT_BF16, c->mean, c->rstd, gamma, nullptr, 0.f, c->dy, nullptr,
                               dgam, dbet, c->ln_ws, st)))
    return cl_err(c, rc);
  // block N-1 backward: dloss/dh_{N-2}
  const void* go[1] = {c->dy};
  void* gi[1] = {grad_h};
  if ((rc = fl_server_backward(c->top, go, gi))) return srv_err(c, c->top, rc);
  c->phase = 2;
  return FL_OK;
}

extern "C" int fl_client_bottom_backward(fl_client_t c, const void* grad_h0) {
  if (!c) return fl_internal_error(FL_ERR_INVALID_ARG, "bottom_backward: null handle");
  if (c->phase != 2) return cl_set(c, FL_ERR_STATE, "bottom_backward: the top has not run in this round");
  if (!grad_h0) return cl_set(c, FL_ERR_INVALID_ARG, "bottom_backward: null grad_h0");
  const void* go[1] = {grad_h0};
  void* gi[1] = {c->dx0};
  if (int rc = fl_server_backward(c->bottom, go, gi)) return srv_err(c, c->bottom, rc);
  if (c->train_own) {
    embed_scatter_kernel<<<warps_grid(c->T), 256, 0, c->stream>>>(c->T, c->H, c->tokens, c->V, c->dx0,
                                                                  c->g + c->off_embed);
    c->launches += 1;
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cl_set(c, FL_ERR_CUDA, "embed scatter: %s", cudaGetErrorString(e));
  }
  c->phase = 0;
  return FL_OK;
}

extern "C" int fl_client_step(fl_client_t c, float lr) {
  if (!c) return fl_internal_error(FL_ERR_INVALID_ARG, "client step: null handle");
  if (c->phase != 0) return cl_set(c, FL_ERR_STATE, "client step: a round is open");
  if (int rc = fl_server_step(c->bottom, lr)) return srv_err(c, c->bottom, rc);
  if (int rc = fl_server_step(c->top, lr)) return srv_err(c, c->top, rc);
  if (!c->train_own) return FL_OK;
  const fl_server_cfg& bc = c->cfg.block;
  c->step_t += 1;
  const double bc1 = 1.0 - std::pow((double)bc.adam_beta1, (double)c->step_t);
  const double bc2 = 1.0 - std::pow((double)bc.adam_beta2, (double)c->step_t);
  c->launches += 1;
  return cl_err(c, fl_launch_adamw(c->n_own, c->w, c->g, c->m, c->v, c->wb, lr, bc.adam_beta1, bc.adam_beta2,
                                   bc.adam_eps, bc.weight_decay, (float)bc1, (float)bc2, 1, c->stream));
}

extern "C" int64_t fl_client_tensor_numel(fl_client_t c, int32_t part, int32_t t) {
  if (!c) return -1;
  if (fl_server_t s = part_server(c, part)) return fl_server_tensor_numel(s, t);
  int64_t n = 0;
  return own_tensor(c, part, t, &n) < 0 ? -1 : n;
}

static int own_copy(fl_client* c, int32_t part, int32_t t, size_t n, int64_t* off) {
  int64_t numel = 0;
  *off = own_tensor(c, part, t, &numel);
  if (*off < 0) return cl_set(c, FL_ERR_INVALID_ARG, "client: bad part %d / tensor %d", part, t);
  if ((int64_t)n != numel) return cl_set(c, FL_ERR_INVALID_ARG, "client: n=%zu but the tensor has %lld", n, (long long)numel);
  if (cudaStreamSynchronize(c->stream) != cudaSuccess) return cl_set(c, FL_ERR_CUDA, "client: sync");
  return FL_OK;
}

extern "C" int fl_client_get_param(fl_client_t c, int32_t part, int32_t t, float* dst, size_t n) {
  if (!c || !dst) return fl_internal_error(FL_ERR_INVALID_ARG, "client get_param: null");
  if (fl_server_t s = part_server(c, part)) return srv_err(c, s, fl_server_get_param(s, 0, t, dst, n));
  int64_t off;
  if (int rc = own_copy(c, part, t, n, &off)) return rc;
  if (cudaMemcpy(dst, c->w + off, n * sizeof(float), cudaMemcpyDeviceToHost) != cudaSuccess)
    return cl_set(c, FL_ERR_CUDA, "client get_param: copy");
  return FL_OK;
}

extern "C" int fl_client_get_grad(fl_client_t c, int32_t part, int32_t t, float* dst, size_t n) {
  if (!c || !dst) return fl_internal_error(FL_ERR_INVALID_ARG, "client get_grad: null");
  if (fl_server_t s = part_server(c, part)) return srv_err(c, s, fl_server_get_grad(s, 0, t, dst, n));
  int64_t off;
  if (int rc = own_copy(c, part, t, n, &off)) return rc;
  if (!c->train_own) {  // frozen: no gradient
    memset(dst, 0, n * sizeof(float));
    return FL_OK;
  }
  if (cudaMemcpy(dst, c->g + off, n * sizeof(float), cudaMemcpyDeviceToHost) != cudaSuccess)
    return cl_set(c, FL_ERR_CUDA, "client get_grad: copy");
  return FL_OK;
}

extern "C" int fl_client_set_param(fl_client_t c, int32_t part, int32_t t, const float* src, size_t n) {
  if (!c || !src) return fl_internal_error(FL_ERR_INVALID_ARG, "client set_param: null");
  if (fl_server_t s = part_server(c, part)) return srv_err(c, s, fl_server_set_param(s, 0, t, src, n));
  int64_t off;
  if (int rc = own_copy(c, part, t, n, &off)) return rc;
  if (cudaMemcpy(c->w + off, src, n * sizeof(float), cudaMemcpyHostToDevice) != cudaSuccess)
    return cl_set(c, FL_ERR_CUDA, "client set_param: copy");
  if (int rc = fl_launch_f32_to_bf16((int64_t)n, c->w + off, c->wb + off, c->stream)) return cl_err(c, rc);
  if (cudaStreamSynchronize(c->stream) != cudaSuccess) return cl_set(c, FL_ERR_CUDA, "client set_param: sync");
  return FL_OK;
}

extern "C" int fl_client_average(fl_client_t const* clients, int32_t n) {
  if (!clients || n < 1 || n > FL_MAX_REPLICAS)
    return fl_internal_error(FL_ERR_INVALID_ARG, "client average: need 1..%d clients", FL_MAX_REPLICAS);
  std::vector<fl_server_t> bot(n), top(n);
  ReplicaTable t;
  memset(&t, 0, sizeof t);
  t.n = n;
  for (int r = 0; r < n; ++r) {
    fl_client* c = clients[r];
    if (!c) return fl_internal_error(FL_ERR_INVALID_ARG, "client average: null client %d", r);
    if (c->n_own != clients[0]->n_own || c->H != clients[0]->H)
      return fl_internal_error(FL_ERR_INVALID_ARG, "client average: client %d has another shape", r);
    if (c->phase != 0) return cl_set(c, FL_ERR_STATE, "client average: client %d has an open round", r);
    for (int q = 0; q < r; ++q)
      if (clients[q] == c) return fl_internal_error(FL_ERR_INVALID_ARG, "client average: client %d listed twice", r);
    bot[r] = c->bottom;
    top[r] = c->top;
    t.w[r] = c->w;
    t.wb[r] = c->wb;
  }
  if (int rc = fl_server_average(bot.data(), n)) return rc;
  if (int rc = fl_server_average(top.data(), n)) return rc;
  fl_client* c0 = clients[0];
  for (int r = 0; r < n; ++r)
    if (cudaStreamSynchronize(clients[r]->stream) != cudaSuccess)
      return cl_set(c0, FL_ERR_CUDA, "client average: sync");
  c0->launches += 1;
  if (int rc = fl_launch_average(t, c0->n_own, c0->stream)) return cl_err(c0, rc);
  if (cudaStreamSynchronize(c0->stream) != cudaSuccess) return cl_set(c0, FL_ERR_CUDA, "client average");
  return FL_OK;
}

extern "C" int64_t fl_client_launch_count(fl_client_t c) {
  if (!c) return -1;
  return c->launches + fl_server_launch_count(c->bottom) + fl_server_launch_count(c->top);
}

extern "C" const char* fl_client_last_error(fl_client_t c) {
  if (c) return c->err.c_str();
  return fl_server_last_error(nullptr);
}
