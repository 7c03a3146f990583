// Server runtime of the FL-GLM block stack: the C ABI of flglm.h.
//
// Protocol (§3.1 Model Split, §3.3 client-batch): forward packs the K clients' smashed
// data into one ragged batch and runs blocks 1..N-2; backward takes the clients'
// output-state gradients back through the stack, accumulating fp32 weight gradients;
// step applies AdamW (the optimizer of §4.1.4) and clears them.
//
// Device memory (allocated once in fl_server_create, nothing allocated later):
//   parameter arenas  fp32 master w, grad g, Adam m, v and the bf16 working copy, one flat
//                     array each with identical offsets, so that one AdamW launch covers
//                     every parameter: first the four weight matrices of every block
//                     (block b at b * mat_stride), then the bias and LayerNorm vectors of
//                     every block in one contiguous region (block b at vec_base +
//                     b * vec_stride); every tensor 64-byte aligned; the FFN up-projection
//                     weight is stored transposed ([H, F]: its weight gradient then has the
//                     down-projection's shape and the two run as one launch; the parameter
//                     access functions transpose on the host); with cfg.n_replicas
//                     = R > 1 each arena holds R such layouts back to back (replica r at
//                     r * n_params), and replica r trains on the r-th of R equal, contiguous
//                     token groups of each call (§3.3 server-hierarchical on one GPU): the
//                     GEMMs of all replicas run as one batched launch, attention over
//                     the whole packed batch (segments are independent), the LayerNorm
//                     and vector kernels once per replica;
//   activations       per block: LN1 out A, rotated QKV, attention O, LSE, residual stream
//                     Hres (fp32), LN2 out M, FFN pre-activation U and GeLU output G, LN
//                     statistics; xs[0..n_blocks]: block inputs / outputs in fp32
//                     (xs[0] = packed client states, widened exactly); with cfg.recompute
//                     only one block's set, refilled before each block's backward by
//                     running that block's forward again from its kept input xs[b];
//   backward scratch  one set of gradient buffers reused by every block; the gradient of
//                     the residual stream is kept in fp32 next to the bf16 copy the GEMMs
//                     read;
//
// Precision: GEMM operands are bf16 (tcgen05 kind::f16), accumulation fp32.  The
// alpha-scaled residual path (block inputs, Hres, the alpha * LN(.) terms, and their
// gradients) stays fp32 end to end: with alpha = sqrt(56) it carries most of each
// block's output, and bf16 roundings on it would add up over 26 blocks.
//   metadata          cu_seqlens, per-token positions, attention tile list, rotary table.
#include <cuda_runtime.h>

#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <set>
#include <string>
#include <tuple>
#include <utility>
#include <vector>

#include "../../include/flglm.h"
#include "../../include/flglm_kernels.h"
#include "common.cuh"
#include "kernels.cuh"

// ------------------------------------------------------------------ errors
static thread_local std::string g_last_error;

int fl_internal_error(int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return code;
}

int fl_internal_cuda_error(cudaError_t e, const char* what, const char* file, int line) {
  return fl_internal_error(FL_ERR_CUDA, "%s failed: %s (%s:%d)", what, cudaGetErrorString(e), file, line);
}

// ------------------------------------------------------------------ launch set-up
int fl_sm_count() {
  constexpr int MAX_DEV = 64;
  static std::atomic<int> cache[MAX_DEV];  // 0: not queried yet
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 148;
  const bool cached = dev >= 0 && dev < MAX_DEV;
  if (cached) {
    const int c = cache[dev].load(std::memory_order_relaxed);
    if (c > 0) return c;
  }
  int c = 0;
  if (cudaDeviceGetAttribute(&c, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || c <= 0) {
    cudaGetLastError();
    c = 148;
  }
  if (cached) cache[dev].store(c, std::memory_order_relaxed);
  return c;
}

cudaError_t fl_func_smem(const void* func, int bytes) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  static std::mutex mu;
  static std::set<std::tuple<const void*, int, int>> done;
  const auto key = std::make_tuple(func, dev, bytes);
  std::lock_guard<std::mutex> lock(mu);
  if (done.count(key)) return cudaSuccess;
  e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess) done.insert(key);
  return e;
}

namespace {

// Tokens from which fl_server_backward_step fuses the AdamW update into the weight-gradient
// GEMMs (measured on GB300 at H 4096, F 16384: fused / separate step 119.1 / 118.3 ms at
// 4096 tokens, 159.9 / 164.2 ms at 6144; the crossover depends on the tokens, the length of
// the weight-gradient main loop, not on the widths).
constexpr int FL_FUSED_STEP_MIN_TOKENS = 4608;

constexpr uint64_t GOLDEN = 0x9E3779B97F4A7C15ull;
uint64_t mix64_host(uint64_t z) {
  z ^= z >> 30;
  z *= 0xBF58476D1CE4E5B9ull;
  z ^= z >> 27;
  z *= 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}
// key(seed, tag) = mix64(mix64(seed + GOLDEN) ^ tag), tag = purpose<<56 | block<<40 | tensor<<32 | client
uint64_t stream_key(uint64_t seed, uint64_t purpose, uint64_t block, uint64_t tensor, uint64_t client) {
  const uint64_t tag = (purpose << 56) | (block << 40) | (tensor << 32) | client;
  return mix64_host(mix64_host(seed + GOLDEN) ^ tag);
}

struct BlockAct {
  __nv_bfloat16 *a, *qkv, *o, *m, *u, *g;
  float* h;  // residual stream after attention, fp32
  float *mean1, *rstd1, *mean2, *rstd2, *lse;
};

struct Prof {
  bool on = false;
  std::vector<cudaEvent_t> pool;
  std::vector<std::pair<int, int>> marks;  // (class, event index of the begin event)
  size_t used = 0;
};

}  // namespace

struct fl_server {
  fl_server_cfg cfg;
  int rdim = 0;
  cudaStream_t stream = nullptr;
  std::string err;

  // parameter arenas
  int64_t tensor_off[FL_T_COUNT] = {};  // inside the block's matrix or vector slice
  int64_t tensor_n[FL_T_COUNT] = {};
  int64_t mat_stride = 0, vec_stride = 0, vec_base = 0, pre_stride = 0, pre_base = 0;
  int64_t n_params = 0;  // padded total of one replica
  int R = 1;             // replicas in the handle (cfg.n_replicas, at least 1)
  int64_t n_all() const { return R * n_params; }  // every replica's arena
  float *w = nullptr, *g = nullptr, *m = nullptr, *v = nullptr;
  __nv_bfloat16* wb = nullptr;
  int64_t step_t = 0;
  // true while every gradient is zero (after create and after each step): the next
  // backward then stores the weight gradients instead of adding to them, and AdamW
  // does not need to clear the 4 B/parameter gradient arena
  bool grads_zero = true;
  // fused backward + step: the weight-gradient GEMMs apply AdamW in their epilogue
  struct {
    bool on = false;
    float lr = 0.f, inv_bc1 = 1.f, inv_bc2 = 1.f;
  } fuse;

  // activations
  std::vector<float*> xs;  // block inputs/outputs, fp32
  std::vector<BlockAct> act;  // one per block, or a single shared set with recompute
  BlockAct& act_of(int b) { return act[cfg.recompute ? 0 : b]; }
  // backward scratch: gradient of a block's output / input as bf16 (GEMM operand) and
  // fp32 (residual chain), ping-pong
  __nv_bfloat16 *dy = nullptr, *dx = nullptr, *du = nullptr, *dh = nullptr, *d_o = nullptr, *dqkv = nullptr;
  float *dyf = nullptr, *dxf = nullptr, *dm = nullptr, *dhf = nullptr, *da = nullptr;
  float *delta = nullptr, *ln_ws = nullptr;
  // metadata
  int32_t *cu = nullptr, *pos = nullptr, *pos2 = nullptr, *ctx = nullptr;
  bool glm = false;  // the pending call has GLM blank-infilling segments
  uint32_t* tiles = nullptr;
  float* rope_tab = nullptr;
  int* status = nullptr;

  std::vector<void*> allocations;

  // pending step
  bool pending = false;
  int T = 0, S = 0, K = 0, n_tiles = 0, n_tiles128 = 0;
  int Tr = 0, Sr = 0;  // tokens and segments of one replica's group (T and S with one replica)
  std::vector<int32_t> seq_lens;

  Prof prof;
  int64_t launches = 0;

  static bool is_matrix(int t) { return t == FL_T_WQKV || t == FL_T_WDENSE || t == FL_T_WUP || t == FL_T_WDOWN; }
  static bool is_prefix(int t) { return t == FL_T_PREFIX_K || t == FL_T_PREFIX_V; }
  int64_t off(int b, int t) const {
    if (is_prefix(t)) return pre_base + b * pre_stride + tensor_off[t];
    return is_matrix(t) ? b * mat_stride + tensor_off[t] : vec_base + b * vec_stride + tensor_off[t];
  }
  AttnPrefix prefix(int b, bool grads) {
    AttnPrefix p;
    if (cfg.prefix_len > 0) {
      p.k = wbt(b, FL_T_PREFIX_K);
      p.v = wbt(b, FL_T_PREFIX_V);
      p.len = cfg.prefix_len;
      if (grads) {
        p.dk = gt(b, FL_T_PREFIX_K);
        p.dv = gt(b, FL_T_PREFIX_V);
      }
    }
    return p;
  }
  AttnGlm glm_args() const {
    AttnGlm a;
    if (glm) {
      a.ctx = ctx;
      a.pos = pos;
      a.pos2 = pos2;
    }
    return a;
  }
  float* wt(int b, int t, int r = 0) { return w + r * n_params + off(b, t); }
  float* gt(int b, int t, int r = 0) { return g + r * n_params + off(b, t); }
  __nv_bfloat16* wbt(int b, int t, int r = 0) { return wb + r * n_params + off(b, t); }
};

namespace {

int set_err(fl_server* h, int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  g_last_error = buf;
  if (h) h->err = buf;
  return code;
}
// Propagates an error from an internal call, copying the thread-local message to h.
int fwd_err(fl_server* h, int rc) {
  if (rc != FL_OK && h) h->err = g_last_error;
  return rc;
}

template <typename T>
int dalloc(fl_server* h, T** p, size_t count) {
  void* q = nullptr;
  const size_t bytes = count * sizeof(T) + 256;
  cudaError_t e = cudaMalloc(&q, bytes);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return set_err(h, FL_ERR_OOM, "cudaMalloc of %zu bytes failed: %s", bytes, cudaGetErrorString(e));
  }
  h->allocations.push_back(q);
  *p = reinterpret_cast<T*>(q);
  return FL_OK;
}

// Marks the start of `nk` kernel launches of class cls on the handle's stream.
void prof_begin(fl_server* h, int cls, int nk = 1) {
  h->launches += nk;
  if (!h->prof.on) return;
  Prof& p = h->prof;
  while (p.pool.size() < p.used + 2) {
    cudaEvent_t e;
    cudaEventCreate(&e);
    p.pool.push_back(e);
  }
  cudaEventRecord(p.pool[p.used], h->stream);
  p.marks.push_back({cls, (int)p.used});
  p.used += 2;
}
void prof_end(fl_server* h) {
  if (!h->prof.on) return;
  cudaEventRecord(h->prof.pool[h->prof.marks.back().second + 1], h->stream);
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

int validate_cfg(const fl_server_cfg& c, int* rdim) {
  if (c.n_blocks < 1 || c.hidden <= 0 || c.n_heads <= 0 || c.head_dim <= 0 || c.ffn_hidden <= 0)
    return fl_internal_error(FL_ERR_INVALID_ARG, "cfg: sizes must be positive");
  if (c.n_heads * c.head_dim != c.hidden)
    return fl_internal_error(FL_ERR_INVALID_ARG, "cfg: hidden != n_heads * head_dim");
  if (c.hidden % 256 || c.hidden > 4096 || (c.hidden & (c.hidden - 1)) != 0)
    return fl_internal_error(FL_ERR_UNSUPPORTED, "cfg: hidden must be a power of two in [256, 4096]");
  if (c.ffn_hidden % 256) return fl_internal_error(FL_ERR_UNSUPPORTED, "cfg: ffn_hidden %% 256 != 0");
  if (!(c.head_dim == 64 || c.head_dim == 128)) return fl_internal_error(FL_ERR_UNSUPPORTED, "cfg: head_dim in {64,128}");
  const int rd = c.rotary_dim ? c.rotary_dim : c.head_dim / 2;
  if (rd != c.head_dim / 2) return fl_internal_error(FL_ERR_UNSUPPORTED, "cfg: rotary_dim must be head_dim/2");
  if (c.max_tokens < 1) return fl_internal_error(FL_ERR_INVALID_ARG, "cfg: max_tokens < 1");
  if (c.client_batch < 1) return fl_internal_error(FL_ERR_INVALID_ARG, "cfg: client_batch < 1");
  if (c.recompute != 0 && c.recompute != 1) return fl_internal_error(FL_ERR_INVALID_ARG, "cfg: recompute must be 0 or 1");
  if (!(c.ln_eps > 0.f) || !(c.rope_base > 1.f)) return fl_internal_error(FL_ERR_INVALID_ARG, "cfg: ln_eps/rope_base");
  if (c.residual_from_ln != 0 && c.residual_from_ln != 1)
    return fl_internal_error(FL_ERR_INVALID_ARG, "cfg: residual_from_ln must be 0 or 1");
  if (c.prefix_len < 0 || c.prefix_len > 128) return fl_internal_error(FL_ERR_UNSUPPORTED, "cfg: prefix_len in 0..128");
  if (c.freeze_base != 0 && c.freeze_base != 1) return fl_internal_error(FL_ERR_INVALID_ARG, "cfg: freeze_base 0 or 1");
  if (c.freeze_base && c.prefix_len == 0)
    return fl_internal_error(FL_ERR_INVALID_ARG, "cfg: freeze_base needs a prefix (prefix_len > 0)");
  if (c.fused_step_min_tokens < 0) return fl_internal_error(FL_ERR_INVALID_ARG, "cfg: fused_step_min_tokens < 0");
  if (c.n_replicas < 0 || c.n_replicas > FL_GEMM_MAX_BATCH)
    return fl_internal_error(FL_ERR_UNSUPPORTED, "cfg: n_replicas in 0..%d", FL_GEMM_MAX_BATCH);
  if (c.n_replicas > 1 && c.prefix_len > 0)
    return fl_internal_error(FL_ERR_UNSUPPORTED, "cfg: n_replicas > 1 with a prefix");
  *rdim = rd;
  return FL_OK;
}

// Launches one block GEMM; with R > 1 replicas one batched launch runs it for every replica:
// problem r reads and writes replica r's Tr token rows and replica r's parameter arena.
// A weight gradient (wgrad) contracts over the tokens: its A and B are token-major, its
// output (gradient, or weight + Adam state + bf16 copy when fused) is a parameter.
int run_gemm(fl_server* h, fl_gemm_args a, bool wgrad = false) {
  if (h->R > 1) {
    const int64_t P = h->n_params, Tr = h->Tr;
    a.batch = h->R;
    a.a_bstride = Tr * a.lda;
    if (wgrad) {
      a.b_bstride = Tr * a.ldb;
      a.d_bstride = P;
      a.adam_bstride = P;
      a.aux_out_bstride = P;
    } else {
      a.b_bstride = P;
      a.d_bstride = Tr * a.ldd;
      a.aux_bstride = Tr * a.ld_aux;
      a.aux_out_bstride = Tr * a.ld_aux_out;
      a.bias_bstride = P;  // the bias, or the column sums of a bias gradient
      a.row_bstride = Tr;  // positions, LayerNorm statistics
      a.lnp_bstride = P;   // LayerNorm gain and shift
    }
  }
  prof_begin(h, FL_PROF_GEMM);
  int rc = fl_k_gemm(&a, h->status, h->stream);
  prof_end(h);
  return rc;
}

// Several weight-gradient problems of one shape (ms[0..n), for replica 0) as one launch
// for every replica (fl_k_gemm_multi) when n x R problems fit one launch, else one
// launch per problem batched over the replicas.  Problem m of replica r reads replica r's
// Tr token rows and updates replica r's arena.
int run_wgrad_group(fl_server* h, const fl_gemm_args* ms, int n) {
  if (n * h->R > FL_GEMM_MAX_BATCH) {
    for (int i = 0; i < n; ++i)
      if (int rc = run_gemm(h, ms[i], true)) return rc;
    return FL_OK;
  }
  fl_gemm_args probs[FL_GEMM_MAX_BATCH];
  const int64_t P = h->n_params, Tr = h->Tr;
  for (int r = 0; r < h->R; ++r)
    for (int i = 0; i < n; ++i) {
      fl_gemm_args a = ms[i];
      a.A = static_cast<const __nv_bfloat16*>(a.A) + r * Tr * a.lda;
      a.B = static_cast<const __nv_bfloat16*>(a.B) + r * Tr * a.ldb;
      a.D = static_cast<float*>(a.D) + r * P;
      if (a.adam_m) {
        a.adam_m += r * P;
        a.adam_v += r * P;
        a.aux_out = static_cast<__nv_bfloat16*>(a.aux_out) + r * P;
      }
      probs[r * n + i] = a;
    }
  prof_begin(h, FL_PROF_GEMM);
  int rc = fl_k_gemm_multi(probs, n * h->R, h->status, h->stream);
  prof_end(h);
  return rc;
}

fl_gemm_args gemm_fwd(int M, int N, int K, const void* A, const void* W, void* D, int epi) {
  fl_gemm_args a;
  memset(&a, 0, sizeof a);
  a.M = M; a.N = N; a.K = K;
  a.A = A; a.lda = K; a.a_mn_major = 0;
  a.B = W; a.ldb = K; a.b_mn_major = 0;
  a.D = D; a.ldd = N;
  a.epilogue = epi;
  return a;
}
// dX[T, Kin] = dY[T, Nout] . W[Nout, Kin]
fl_gemm_args gemm_dgrad(int T, int Kin, int Nout, const void* dY, const void* W, void* dX, int epi) {
  fl_gemm_args a;
  memset(&a, 0, sizeof a);
  a.M = T; a.N = Kin; a.K = Nout;
  a.A = dY; a.lda = Nout; a.a_mn_major = 0;
  a.B = W; a.ldb = Kin; a.b_mn_major = 1;
  a.D = dX; a.ldd = Kin;
  a.epilogue = epi;
  return a;
}
// dW[Nout, Kin] (+)= dY[T, Nout]^T . X[T, Kin]; stores when the gradients are known zero
fl_gemm_args gemm_wgrad_raw(int T, int Nout, int Kin, const void* dY, const void* X, float* dW, bool store) {
  fl_gemm_args a;
  memset(&a, 0, sizeof a);
  a.M = Nout; a.N = Kin; a.K = T;
  a.A = dY; a.lda = Nout; a.a_mn_major = 1;
  a.B = X; a.ldb = Kin; a.b_mn_major = 1;
  a.D = dW; a.ldd = Kin;
  a.epilogue = store ? FL_EPI_STORE_F32 : FL_EPI_ACCUM_F32;
  return a;
}

// Weight gradient of weight matrix t of block b (from element e0 of it on: a block of rows,
// whose gradient dY has row stride ldy): stored / accumulated into the gradient arena, or,
// inside a fused backward + step, applied to the weight by AdamW directly.
fl_gemm_args gemm_wgrad(fl_server* h, int b, int t, int T, int Nout, int Kin, const void* dY, const void* X,
                        int64_t e0 = 0, int64_t ldy = 0) {
  fl_gemm_args a = gemm_wgrad_raw(T, Nout, Kin, dY, X, h->gt(b, t) + e0, h->grads_zero);
  if (ldy) a.lda = ldy;
  if (h->fuse.on) {
    const fl_server_cfg& c = h->cfg;
    a.epilogue = FL_EPI_ADAMW;
    a.D = h->wt(b, t) + e0;
    a.adam_m = h->m + h->off(b, t) + e0;
    a.adam_v = h->v + h->off(b, t) + e0;
    a.aux_out = h->wbt(b, t) + e0;
    a.ld_aux_out = Kin;
    a.lr = h->fuse.lr;
    a.beta1 = c.adam_beta1;
    a.beta2 = c.adam_beta2;
    a.eps = c.adam_eps;
    a.weight_decay = c.weight_decay;
    a.inv_bc1 = h->fuse.inv_bc1;
    a.inv_bc2 = h->fuse.inv_bc2;
  }
  return a;
}

#define TRY(h, expr)                    \
  do {                                  \
    int _rc = (expr);                   \
    if (_rc != FL_OK) return fwd_err(h, _rc); \
  } while (0)

// Forward of block b from xs[b] into its activations and xs[b + 1].  Without `output`
// (recomputing the activations for the backward) the FFN down-projection, whose result
// xs[b + 1] is already kept and which the backward does not read, is skipped.
int block_forward(fl_server* h, int b, bool output = true) {
  const fl_server_cfg& c = h->cfg;
  const int T = h->Tr, H = c.hidden, F = c.ffn_hidden;  // T: the token rows of one replica's GEMM
  BlockAct& A = h->act_of(b);
  const float* x = h->xs[b];
  cudaStream_t st = h->stream;
  // a = LN1(x)
  prof_begin(h, FL_PROF_LN, h->R);
  for (int r = 0; r < h->R; ++r) {
    const int64_t r0 = (int64_t)r * T;
    TRY(h, fl_launch_layernorm_fwd_f32(T, H, x + r0 * H, h->wt(b, FL_T_LN1_G, r), h->wt(b, FL_T_LN1_B, r), c.ln_eps,
                                       (__nv_bfloat16*)A.a + r0 * H, A.mean1 + r0, A.rstd1 + r0, st, h->status));
  }
  prof_end(h);
  // qkv = a Wqkv^T + bqkv, q and k rotated
  fl_gemm_args g1 = gemm_fwd(T, 3 * H, H, A.a, h->wbt(b, FL_T_WQKV), A.qkv, FL_EPI_BIAS_ROPE);
  g1.bias = h->wt(b, FL_T_BQKV);
  g1.pos = h->pos;
  g1.pos2 = h->glm ? h->pos2 : nullptr;
  g1.rope_tab = h->rope_tab;
  g1.n_heads = c.n_heads;
  g1.head_dim = c.head_dim;
  g1.rotary_dim = h->rdim;
  TRY(h, run_gemm(h, g1));
  // o = causal attention within each segment
  prof_begin(h, FL_PROF_ATTN);
  TRY(h, fl_launch_attn_fwd(h->T, c.n_heads, c.head_dim, A.qkv, h->cu, h->tiles, h->n_tiles, h->n_tiles128, A.o,
                            A.lse, h->prefix(b, false), h->glm_args(), st, h->status));
  prof_end(h);
  // h = alpha * (LN1(x) or x) + o Wd^T + bd, fp32; LN1(x) recomputed in fp32 in the epilogue
  fl_gemm_args g2 = gemm_fwd(T, H, H, A.o, h->wbt(b, FL_T_WDENSE), A.h, FL_EPI_BIAS_RESID);
  g2.bias = h->wt(b, FL_T_BDENSE);
  g2.aux = x;
  g2.aux_dtype = FL_DT_F32;
  g2.ld_aux = H;
  g2.d_dtype = FL_DT_F32;
  g2.alpha = c.residual_alpha;
  if (c.residual_from_ln) {
    g2.ln_mean = A.mean1;
    g2.ln_rstd = A.rstd1;
    g2.ln_gamma = h->wt(b, FL_T_LN1_G);
    g2.ln_beta = h->wt(b, FL_T_LN1_B);
  }
  TRY(h, run_gemm(h, g2));
  // m = LN2(h)
  prof_begin(h, FL_PROF_LN, h->R);
  for (int r = 0; r < h->R; ++r) {
    const int64_t r0 = (int64_t)r * T;
    TRY(h, fl_launch_layernorm_fwd_f32(T, H, A.h + r0 * H, h->wt(b, FL_T_LN2_G, r), h->wt(b, FL_T_LN2_B, r), c.ln_eps,
                                       (__nv_bfloat16*)A.m + r0 * H, A.mean2 + r0, A.rstd2 + r0, st, h->status));
  }
  prof_end(h);
  // u = m W1^T + b1, g = gelu(u)
  fl_gemm_args g3 = gemm_fwd(T, F, H, A.m, h->wbt(b, FL_T_WUP), A.g, FL_EPI_BIAS_GELU);
  g3.b_mn_major = 1;  // W1 stored transposed, [H, F]
  g3.ldb = F;
  g3.bias = h->wt(b, FL_T_BUP);
  g3.aux_out = A.u;
  g3.ld_aux_out = F;
  TRY(h, run_gemm(h, g3));
  if (!output) return FL_OK;
  // y = alpha * (LN2(h) or h) + g W2^T + b2, fp32
  fl_gemm_args g4 = gemm_fwd(T, H, F, A.g, h->wbt(b, FL_T_WDOWN), h->xs[b + 1], FL_EPI_BIAS_RESID);
  g4.bias = h->wt(b, FL_T_BDOWN);
  g4.aux = A.h;
  g4.aux_dtype = FL_DT_F32;
  g4.ld_aux = H;
  g4.d_dtype = FL_DT_F32;
  g4.alpha = c.residual_alpha;
  if (c.residual_from_ln) {
    g4.ln_mean = A.mean2;
    g4.ln_rstd = A.rstd2;
    g4.ln_gamma = h->wt(b, FL_T_LN2_G);
    g4.ln_beta = h->wt(b, FL_T_LN2_B);
  }
  TRY(h, run_gemm(h, g4));
  return FL_OK;
}

// dy / dyf hold dL/dy of block b (bf16 and fp32); on return dx / dxf hold dL/dx.
int block_backward(fl_server* h, int b, const __nv_bfloat16* dy, const float* dyf, __nv_bfloat16* dx, float* dxf) {
  const fl_server_cfg& c = h->cfg;
  const int T = h->Tr, H = c.hidden, F = c.ffn_hidden;  // T: the token rows of one replica's GEMM
  const float al = c.residual_alpha;
  const bool glm = c.residual_from_ln != 0;
  BlockAct& A = h->act_of(b);
  cudaStream_t st = h->stream;
  const bool train_base = !c.freeze_base;
  // Bias gradients are column sums of the output gradients, added by the kernels that
  // produce those: db2 (dy) by the LayerNorm-1 backward of block b + 1 (here by a column-sum
  // kernel for the top block, whose dy comes from the clients), db1 (du) by the GeLU'
  // epilogue, dbd (dh) by the LayerNorm-2 backward, dbqkv (dqkv) by the attention backward.
  // Weight gradients run after the data gradients that read the same weights (a fused
  // step updates the weight in the gradient's epilogue), two or four matrices per launch
  // with one replica: [dW2, dW1^T] (both [H, F]) and [dWd, dWq, dWk, dWv] (all [H, H]), so
  // that one matrix's last wave is filled by the next.
  // FFN down: du = (dy W2) * gelu'(u), db1 += colsum(du)
  fl_gemm_args d1 = gemm_dgrad(T, F, H, dy, h->wbt(b, FL_T_WDOWN), h->du, FL_EPI_GELU_BWD);
  d1.aux = A.u;
  d1.ld_aux = F;
  d1.colsum = train_base ? h->gt(b, FL_T_BUP) : nullptr;
  TRY(h, run_gemm(h, d1));
  // FFN up: dm = du W1 (+ alpha dy), fp32 (W1 stored transposed: a K-major operand)
  fl_gemm_args d2 = gemm_dgrad(T, H, F, h->du, h->wbt(b, FL_T_WUP), h->dm, glm ? FL_EPI_RESID : FL_EPI_STORE);
  d2.b_mn_major = 0;
  d2.ldb = F;
  d2.d_dtype = FL_DT_F32;
  if (glm) {
    d2.aux = dyf;
    d2.aux_dtype = FL_DT_F32;
    d2.ld_aux = H;
    d2.alpha = al;
  }
  TRY(h, run_gemm(h, d2));
  if (train_base) {  // weight and bias gradients (skipped when only the prefixes train)
    // dW2 (+)= dy^T g, dW1^T (+)= m^T du
    const fl_gemm_args ffn[2] = {gemm_wgrad(h, b, FL_T_WDOWN, T, H, F, dy, A.g),
                                 gemm_wgrad(h, b, FL_T_WUP, T, H, F, A.m, h->du)};
    TRY(h, run_wgrad_group(h, ffn, 2));
    if (b == c.n_blocks - 1) {
      prof_begin(h, FL_PROF_OTHER, h->R);
      for (int r = 0; r < h->R; ++r) TRY(h, fl_k_colsum(T, H, dy + (int64_t)r * T * H, h->gt(b, FL_T_BDOWN, r), st));
      prof_end(h);
    }
  }
  // LN2 backward: dh = LN2'(dm) (+ alpha dy), bf16 and fp32; dbd += colsum(dh)
  prof_begin(h, FL_PROF_LN, 2 * h->R);
  for (int r = 0; r < h->R; ++r) {
    const int64_t r0 = (int64_t)r * T, e0 = r0 * H;
    TRY(h, fl_launch_layernorm_bwd_f32(T, H, h->dm + e0, A.h + e0, A.mean2 + r0, A.rstd2 + r0,
                                       h->wt(b, FL_T_LN2_G, r), glm ? nullptr : dyf + e0, al, h->dh + e0, h->dhf + e0,
                                       h->gt(b, FL_T_LN2_G, r), h->gt(b, FL_T_LN2_B, r),
                                       train_base ? h->gt(b, FL_T_BDENSE, r) : nullptr, h->ln_ws, st, h->status));
  }
  prof_end(h);
  // dense: do = dh Wd
  TRY(h, run_gemm(h, gemm_dgrad(T, H, H, h->dh, h->wbt(b, FL_T_WDENSE), h->d_o, FL_EPI_STORE)));
  // attention backward -> dqkv (w.r.t. the un-rotated q, k); dbqkv += colsum(dqkv)
  prof_begin(h, FL_PROF_ATTN, 3);
  TRY(h, fl_launch_attn_bwd(h->T, c.n_heads, c.head_dim, A.qkv, A.o, A.lse, h->d_o, h->cu, h->tiles, h->n_tiles,
                            h->n_tiles128, h->delta, h->rope_tab, h->dqkv, h->prefix(b, true), h->glm_args(), st,
                            train_base ? h->gt(b, FL_T_BQKV) : nullptr, h->status, h->R > 1 ? h->Sr : 0,
                            h->n_params));
  prof_end(h);
  // QKV: da = dqkv Wqkv (+ alpha dh), fp32
  fl_gemm_args d3 = gemm_dgrad(T, H, 3 * H, h->dqkv, h->wbt(b, FL_T_WQKV), h->da, glm ? FL_EPI_RESID : FL_EPI_STORE);
  d3.d_dtype = FL_DT_F32;
  if (glm) {
    d3.aux = h->dhf;
    d3.aux_dtype = FL_DT_F32;
    d3.ld_aux = H;
    d3.alpha = al;
  }
  TRY(h, run_gemm(h, d3));
  if (train_base) {  // weight gradients (skipped when only the prefixes train)
    if (h->R == 1) {
      // dWd (+)= dh^T o; rows r H .. of dWqkv (+)= dqkv[:, r H ..]^T a, r = 0, 1, 2
      fl_gemm_args att[4] = {gemm_wgrad(h, b, FL_T_WDENSE, T, H, H, h->dh, A.o)};
      for (int r = 0; r < 3; ++r)
        att[1 + r] = gemm_wgrad(h, b, FL_T_WQKV, T, H, H, h->dqkv + (int64_t)r * H, A.a, (int64_t)r * H * H, 3 * H);
      TRY(h, run_wgrad_group(h, att, 4));
    } else {  // [dWd, dWqkv] batched over the replicas
      TRY(h, run_gemm(h, gemm_wgrad(h, b, FL_T_WDENSE, T, H, H, h->dh, A.o), true));
      TRY(h, run_gemm(h, gemm_wgrad(h, b, FL_T_WQKV, T, 3 * H, H, h->dqkv, A.a), true));
    }
  }
  // LN1 backward: dx = LN1'(da) (+ alpha dh), bf16 and fp32; dx is dy of block b - 1, whose
  // down-projection bias gradient is its column sum
  prof_begin(h, FL_PROF_LN, 2 * h->R);
  for (int r = 0; r < h->R; ++r) {
    const int64_t r0 = (int64_t)r * T, e0 = r0 * H;
    TRY(h, fl_launch_layernorm_bwd_f32(T, H, h->da + e0, h->xs[b] + e0, A.mean1 + r0, A.rstd1 + r0,
                                       h->wt(b, FL_T_LN1_G, r), glm ? nullptr : h->dhf + e0, al, dx + e0, dxf + e0,
                                       h->gt(b, FL_T_LN1_G, r), h->gt(b, FL_T_LN1_B, r),
                                       train_base && b > 0 ? h->gt(b - 1, FL_T_BDOWN, r) : nullptr, h->ln_ws, st,
                                       h->status));
  }
  prof_end(h);
  return FL_OK;
}

// Moves the K client tensors to / from the packed buffers (mode: CopyMode).
int copy_clients(fl_server* h, const void* const* ptrs, int mode, __nv_bfloat16* packed_bf16, float* packed_f32) {
  const int64_t row8 = (int64_t)h->cfg.client_batch * h->cfg.hidden / 8;  // 8-element groups per token
  int64_t off = 0;
  for (int k0 = 0; k0 < h->K; k0 += FL_MAX_COPY) {
    CopyTable tab;
    memset(&tab, 0, sizeof tab);
    tab.mode = mode;
    tab.packed_bf16 = packed_bf16;
    tab.packed_f32 = packed_f32;
    tab.n = (h->K - k0) < FL_MAX_COPY ? (h->K - k0) : FL_MAX_COPY;
    for (int e = 0; e < tab.n; ++e) {
      const int k = k0 + e;
      tab.client[e] = const_cast<void*>(ptrs[k]);
      tab.off8[e] = off;
      tab.n8[e] = row8 * h->seq_lens[k];
      off += tab.n8[e];
    }
    prof_begin(h, FL_PROF_OTHER);
    int rc = fl_launch_copy_clients(tab, h->stream);
    prof_end(h);
    if (rc) return fwd_err(h, rc);
  }
  return FL_OK;
}

int check_ptrs(fl_server* h, const void* const* p, int K, const char* what) {
  if (!p) return set_err(h, FL_ERR_INVALID_ARG, "%s: null array", what);
  for (int k = 0; k < K; ++k) {
    if (!p[k]) return set_err(h, FL_ERR_INVALID_ARG, "%s[%d] is null", what, k);
    if (!aligned16(p[k])) return set_err(h, FL_ERR_INVALID_ARG, "%s[%d] is not 16-byte aligned", what, k);
  }
  return FL_OK;
}

}  // namespace

// ====================================================================== C ABI

extern "C" void fl_server_cfg_default(fl_server_cfg* c) {
  if (!c) return;
  memset(c, 0, sizeof *c);
  c->n_blocks = 26;
  c->hidden = 4096;
  c->n_heads = 32;
  c->head_dim = 128;
  c->ffn_hidden = 16384;
  c->rotary_dim = 64;
  c->rope_base = 10000.f;
  c->ln_eps = 1e-5f;
  c->residual_alpha = sqrtf(56.f);
  c->residual_from_ln = 1;
  c->client_batch = 1;
  c->max_tokens = 8192;
  c->max_seq_len = 0;
  c->recompute = 0;
  c->init_std = 0.02f;
  c->adam_beta1 = 0.9f;
  c->adam_beta2 = 0.999f;
  c->adam_eps = 1e-8f;
  c->weight_decay = 0.f;
}

// Seeded init keys: tensor t of block b from the stream (seed, purpose, block0 + b, t).
// The server uses purpose 1 and block0 = 0; the client's blocks use their own streams.
int fl_server_create_keyed(const fl_server_cfg* cfg, uint64_t seed, int purpose, int block0, fl_server_t* out) {
  if (!out) return fl_internal_error(FL_ERR_INVALID_ARG, "create: out is null");
  *out = nullptr;
  if (!cfg) return fl_internal_error(FL_ERR_INVALID_ARG, "create: cfg is null");
  int rdim = 0;
  if (int rc = validate_cfg(*cfg, &rdim)) return rc;
  fl_server* h = new fl_server();
  h->cfg = *cfg;
  h->rdim = rdim;
  if (h->cfg.max_seq_len <= 0 || h->cfg.max_seq_len > h->cfg.max_tokens) h->cfg.max_seq_len = h->cfg.max_tokens;
  const fl_server_cfg& c = h->cfg;
  const int64_t H = c.hidden, F = c.ffn_hidden, Tm = c.max_tokens;
  auto fail = [&](int rc) {
    fl_server_destroy(h);
    return rc;
  };

  // parameter layout
  const int64_t LpH = (int64_t)c.prefix_len * H;
  const int64_t sizes[FL_T_COUNT] = {3 * H * H, 3 * H, H * H, H, F * H, F, H * F, H, H, H, H, H, LpH, LpH};
  int64_t moff = 0, voff = 0, poff = 0;
  for (int t = 0; t < FL_T_COUNT; ++t) {
    int64_t& o = fl_server::is_prefix(t) ? poff : fl_server::is_matrix(t) ? moff : voff;
    h->tensor_off[t] = o;
    h->tensor_n[t] = sizes[t];
    o += (sizes[t] + 15) / 16 * 16;
  }
  h->mat_stride = moff;
  h->vec_stride = voff;
  h->pre_stride = poff;
  h->vec_base = moff * c.n_blocks;
  h->pre_base = h->vec_base + voff * c.n_blocks;
  h->n_params = h->pre_base + poff * c.n_blocks;
  h->R = c.n_replicas > 1 ? c.n_replicas : 1;
  const int64_t n_all = h->n_all();
  int rc;
  if ((rc = dalloc(h, &h->w, n_all)) || (rc = dalloc(h, &h->g, n_all)) || (rc = dalloc(h, &h->m, n_all)) ||
      (rc = dalloc(h, &h->v, n_all)) || (rc = dalloc(h, &h->wb, n_all)))
    return fail(rc);

  // activations
  h->xs.resize(c.n_blocks + 1);
  for (int b = 0; b <= c.n_blocks; ++b)
    if ((rc = dalloc(h, &h->xs[b], Tm * H))) return fail(rc);  // fp32
  h->act.resize(c.recompute ? 1 : c.n_blocks);
  for (size_t b = 0; b < h->act.size(); ++b) {
    BlockAct& A = h->act[b];
    if ((rc = dalloc(h, &A.a, Tm * H)) || (rc = dalloc(h, &A.qkv, Tm * 3 * H)) || (rc = dalloc(h, &A.o, Tm * H)) ||
        (rc = dalloc(h, &A.h, Tm * H)) || (rc = dalloc(h, &A.m, Tm * H)) || (rc = dalloc(h, &A.u, Tm * F)) ||
        (rc = dalloc(h, &A.g, Tm * F)) || (rc = dalloc(h, &A.mean1, Tm)) || (rc = dalloc(h, &A.rstd1, Tm)) ||
        (rc = dalloc(h, &A.mean2, Tm)) || (rc = dalloc(h, &A.rstd2, Tm)) ||
        (rc = dalloc(h, &A.lse, Tm * c.n_heads)))
      return fail(rc);
  }
  if ((rc = dalloc(h, &h->dy, Tm * H)) || (rc = dalloc(h, &h->dx, Tm * H)) || (rc = dalloc(h, &h->du, Tm * F)) ||
      (rc = dalloc(h, &h->dyf, Tm * H)) || (rc = dalloc(h, &h->dxf, Tm * H)) || (rc = dalloc(h, &h->dhf, Tm * H)) ||
      (rc = dalloc(h, &h->dm, Tm * H)) || (rc = dalloc(h, &h->dh, Tm * H)) || (rc = dalloc(h, &h->d_o, Tm * H)) ||
      (rc = dalloc(h, &h->dqkv, Tm * 3 * H)) || (rc = dalloc(h, &h->da, Tm * H)) ||
      (rc = dalloc(h, &h->delta, Tm * c.n_heads)) ||
      (rc = dalloc(h, &h->ln_ws, fl_launch_layernorm_bwd_workspace((int)Tm, (int)H) / sizeof(float))) ||
      (rc = dalloc(h, &h->cu, FL_MAX_SEGS + 1)) || (rc = dalloc(h, &h->pos, Tm)) || (rc = dalloc(h, &h->pos2, Tm)) ||
      (rc = dalloc(h, &h->ctx, FL_MAX_SEGS)) ||
      (rc = dalloc(h, &h->tiles, 2 * FL_MAX_TILES)) || (rc = dalloc(h, &h->status, 1)))
    return fail(rc);

  // rotary table: [position][pair i] = (cos, sin) of p * base^(-2i/rdim), in double
  const int half = rdim / 2;
  const int64_t npos = c.max_seq_len;
  std::vector<float> tab((size_t)npos * half * 2);
  for (int64_t p = 0; p < npos; ++p)
    for (int i = 0; i < half; ++i) {
      const double ang = (double)p * std::pow((double)c.rope_base, -2.0 * i / (double)rdim);
      tab[(size_t)(p * half + i) * 2] = (float)std::cos(ang);
      tab[(size_t)(p * half + i) * 2 + 1] = (float)std::sin(ang);
    }
  if ((rc = dalloc(h, &h->rope_tab, tab.size()))) return fail(rc);
  cudaStream_t st = nullptr;
  if (cudaMemcpy(h->rope_tab, tab.data(), tab.size() * sizeof(float), cudaMemcpyHostToDevice) != cudaSuccess ||
      cudaMemset(h->g, 0, n_all * sizeof(float)) != cudaSuccess ||
      cudaMemset(h->m, 0, n_all * sizeof(float)) != cudaSuccess ||
      cudaMemset(h->v, 0, n_all * sizeof(float)) != cudaSuccess ||
      cudaMemset(h->w, 0, n_all * sizeof(float)) != cudaSuccess ||
      cudaMemset(h->status, 0, sizeof(int)) != cudaSuccess)
    return fail(fl_internal_cuda_error(cudaGetLastError(), "create: memset/copy", __FILE__, __LINE__));

  // seeded init: tensor t of block b from the stream (seed, purpose 1, b, t)
  for (int b = 0; b < c.n_blocks; ++b)
    for (int t = 0; t < FL_T_COUNT; ++t) {
      if (h->tensor_n[t] == 0) continue;
      float* p = h->wt(b, t);
      if (t == FL_T_LN1_G || t == FL_T_LN2_G) rc = fl_launch_fill(h->tensor_n[t], 1.f, p, st);
      else if (t == FL_T_LN1_B || t == FL_T_LN2_B) rc = fl_launch_fill(h->tensor_n[t], 0.f, p, st);
      else if (t == FL_T_WUP) {
        // drawn in the [F, H] order of its stream into the (zero) gradient arena, then
        // transposed into place and the scratch cleared
        float* tmp = h->gt(b, t);
        rc = fl_launch_normal_init(h->tensor_n[t], stream_key(seed, (uint64_t)purpose, (uint64_t)(block0 + b), t, 0),
                                   0.0, (double)c.init_std, tmp, st);
        if (!rc) rc = fl_launch_transpose_f32(F, H, tmp, p, st);
        if (!rc && cudaMemsetAsync(tmp, 0, h->tensor_n[t] * sizeof(float), st) != cudaSuccess)
          rc = fl_internal_cuda_error(cudaGetLastError(), "create: clear", __FILE__, __LINE__);
      } else
        rc = fl_launch_normal_init(h->tensor_n[t], stream_key(seed, (uint64_t)purpose, (uint64_t)(block0 + b), t, 0), 0.0,
                                   (double)c.init_std, p, st);
      if (rc) return fail(rc);
    }
  // every replica starts from replica 0's values
  for (int r = 1; r < h->R; ++r)
    if (cudaMemcpyAsync(h->w + r * h->n_params, h->w, h->n_params * sizeof(float), cudaMemcpyDeviceToDevice, st) !=
        cudaSuccess)
      return fail(fl_internal_cuda_error(cudaGetLastError(), "create: replica copy", __FILE__, __LINE__));
  if ((rc = fl_launch_f32_to_bf16(n_all, h->w, h->wb, st))) return fail(rc);
  if (cudaDeviceSynchronize() != cudaSuccess)
    return fail(fl_internal_cuda_error(cudaGetLastError(), "create: init", __FILE__, __LINE__));
  *out = h;
  return FL_OK;
}

static int forward_impl(fl_server_t h, const void* const client_states[], const int32_t seq_lens[], int32_t K,
                        const int32_t* context_lens, const int32_t* mask_pos, void* const out_states[]) {
  if (!h) return fl_internal_error(FL_ERR_INVALID_ARG, "forward: null handle");
  const fl_server_cfg& c = h->cfg;
  if (h->pending) return set_err(h, FL_ERR_STATE, "forward: a forward is already pending (call backward first)");
  if (K < 1) return set_err(h, FL_ERR_INVALID_ARG, "forward: K=%d < 1", K);
  if (!seq_lens) return set_err(h, FL_ERR_INVALID_ARG, "forward: seq_lens is null");
  if (int rc = check_ptrs(h, client_states, K, "client_states")) return rc;
  if (int rc = check_ptrs(h, (const void* const*)out_states, K, "out_states")) return rc;
  const int b = c.client_batch;
  int64_t T = 0;
  for (int k = 0; k < K; ++k) {
    if (seq_lens[k] < 1) return set_err(h, FL_ERR_INVALID_ARG, "forward: seq_lens[%d]=%d < 1", k, seq_lens[k]);
    if (seq_lens[k] > c.max_seq_len)
      return set_err(h, FL_ERR_INVALID_ARG, "forward: seq_lens[%d]=%d > max_seq_len %d", k, seq_lens[k], c.max_seq_len);
    T += (int64_t)b * seq_lens[k];
  }
  if (T > c.max_tokens) return set_err(h, FL_ERR_CAPACITY, "forward: %lld tokens > max_tokens %d", (long long)T, c.max_tokens);
  const int64_t S = (int64_t)K * b;
  if (S > FL_MAX_SEGS) return set_err(h, FL_ERR_CAPACITY, "forward: %lld segments > %d", (long long)S, FL_MAX_SEGS);
  // replicas: clients [r K/R, (r+1) K/R) are replica r's group; every group the same tokens
  const int R = h->R;
  if (K % R) return set_err(h, FL_ERR_INVALID_ARG, "forward: K=%d is not a multiple of n_replicas %d", K, R);
  int64_t Tr = T;
  if (R > 1) {
    std::vector<int64_t> group(R, 0);
    for (int k = 0; k < K; ++k) group[k / (K / R)] += (int64_t)b * seq_lens[k];
    for (int r = 1; r < R; ++r)
      if (group[r] != group[0])
        return set_err(h, FL_ERR_INVALID_ARG, "forward: replica %d's clients hold %lld tokens, replica 0's %lld", r,
                       (long long)group[r], (long long)group[0]);
    Tr = group[0];
  }

  // packing metadata: client k row r is segment k*b + r
  static thread_local MetaArgs meta;
  meta.S = (int)S;
  meta.cu[0] = 0;
  for (int k = 0, s = 0; k < K; ++k)
    for (int r = 0; r < b; ++r, ++s) meta.cu[s + 1] = meta.cu[s] + seq_lens[k];
  meta.glm = context_lens != nullptr;
  if (meta.glm) {
    if (2 * h->rdim != c.head_dim)
      return set_err(h, FL_ERR_UNSUPPORTED, "forward: GLM 2D positions need rotary_dim = head_dim / 2");
    for (int s = 0; s < (int)S; ++s) {
      const int L = meta.cu[s + 1] - meta.cu[s];
      const int cl = context_lens[s];
      const int mp = mask_pos ? mask_pos[s] : cl - 1;
      if (cl < 0 || cl > L) return set_err(h, FL_ERR_INVALID_ARG, "forward: context_lens[%d]=%d outside [0, %d]", s, cl, L);
      if (cl > 0 && (mp < 0 || mp >= cl))
        return set_err(h, FL_ERR_INVALID_ARG, "forward: mask_pos[%d]=%d outside [0, %d)", s, mp, cl);
      meta.ctx[s] = cl;
      meta.mpos[s] = cl > 0 ? mp : 0;
    }
  }
  const int nt = fl_build_tiles(meta.cu, (int)S, meta.tiles, FL_MAX_TILES);
  if (nt < 0) return set_err(h, FL_ERR_CAPACITY, "forward: more than %d attention tiles", FL_MAX_TILES);
  const int nt128 = fl_build_tiles(meta.cu, (int)S, meta.tiles + nt, FL_MAX_TILES, 128);  // never more than nt
  meta.n_tiles = nt;
  meta.n_tiles128 = nt128;
  h->T = (int)T;
  h->S = (int)S;
  h->Tr = (int)Tr;
  h->Sr = (int)(S / R);
  h->K = K;
  h->n_tiles = nt;
  h->n_tiles128 = nt128;
  h->seq_lens.assign(seq_lens, seq_lens + K);

  prof_begin(h, FL_PROF_OTHER);
  h->glm = meta.glm;
  int rc = fl_launch_meta(meta, h->cu, h->pos, h->tiles, h->pos2, h->ctx, h->stream);
  prof_end(h);
  if (rc) return fwd_err(h, rc);
  if ((rc = copy_clients(h, client_states, COPY_GATHER_F32, nullptr, h->xs[0]))) return rc;
  for (int blk = 0; blk < c.n_blocks; ++blk)
    if ((rc = block_forward(h, blk))) return rc;
  if ((rc = copy_clients(h, (const void* const*)out_states, COPY_SCATTER_F32, nullptr, h->xs[c.n_blocks]))) return rc;
  h->pending = true;
  return FL_OK;
}

extern "C" int fl_server_create(const fl_server_cfg* cfg, uint64_t seed, fl_server_t* out) {
  return fl_server_create_keyed(cfg, seed, 1, 0, out);
}

extern "C" int fl_server_forward(fl_server_t h, const void* const client_states[], const int32_t seq_lens[], int32_t K,
                                 void* const out_states[]) {
  return forward_impl(h, client_states, seq_lens, K, nullptr, nullptr, out_states);
}

extern "C" int fl_server_forward_glm(fl_server_t h, const void* const client_states[], const int32_t seq_lens[],
                                     int32_t K, const int32_t context_lens[], const int32_t mask_pos[],
                                     void* const out_states[]) {
  if (h && !context_lens) return set_err(h, FL_ERR_INVALID_ARG, "forward_glm: context_lens is null");
  return forward_impl(h, client_states, seq_lens, K, context_lens, mask_pos, out_states);
}

static int backward_impl(fl_server_t h, const void* const grad_out[], void* const grad_in[]) {
  if (!h) return fl_internal_error(FL_ERR_INVALID_ARG, "backward: null handle");
  if (!h->pending) return set_err(h, FL_ERR_STATE, "backward: no pending forward");
  if (int rc = check_ptrs(h, grad_out, h->K, "grad_out")) return rc;
  if (int rc = check_ptrs(h, (const void* const*)grad_in, h->K, "grad_in")) return rc;
  int rc;
  if (h->grads_zero) {
    // bias and LayerNorm gradients accumulate (+=); one memset of their contiguous region
    // (per replica)
    for (int r = 0; r < h->R; ++r) {
      const cudaError_t e = cudaMemsetAsync(h->g + r * h->n_params + h->vec_base, 0,
                                            (h->n_params - h->vec_base) * sizeof(float), h->stream);
      if (e != cudaSuccess) return fwd_err(h, fl_internal_cuda_error(e, "cudaMemsetAsync", __FILE__, __LINE__));
    }
  }
  if ((rc = copy_clients(h, grad_out, COPY_GATHER_F32, h->dy, h->dyf))) return rc;
  __nv_bfloat16* cur = h->dy;
  __nv_bfloat16* nxt = h->dx;
  float* curf = h->dyf;
  float* nxtf = h->dxf;
  for (int blk = h->cfg.n_blocks - 1; blk >= 0; --blk) {
    // with recompute the shared activations hold another block's (or stale) values:
    // refill them from the kept block input; every kernel is deterministic, so they are
    // the same bits the forward computed
    if (h->cfg.recompute && (rc = block_forward(h, blk, false))) return rc;
    if ((rc = block_backward(h, blk, cur, curf, nxt, nxtf))) return rc;
    std::swap(cur, nxt);
    std::swap(curf, nxtf);
  }
  if ((rc = copy_clients(h, (const void* const*)grad_in, COPY_SCATTER_BF16, cur, nullptr))) return rc;
  h->pending = false;
  h->grads_zero = false;
  return FL_OK;
}

extern "C" int fl_server_backward(fl_server_t h, const void* const grad_out[], void* const grad_in[]) {
  return backward_impl(h, grad_out, grad_in);
}

extern "C" int fl_server_backward_step(fl_server_t h, const void* const grad_out[], void* const grad_in[], float lr) {
  if (!h) return fl_internal_error(FL_ERR_INVALID_ARG, "backward_step: null handle");
  if (!h->pending) return set_err(h, FL_ERR_STATE, "backward_step: no pending forward");
  // no fusion while gradients from an earlier backward are pending, nor for calls too
  // short for the weight-gradient main loop to hide the update
  const int min_tokens = h->cfg.fused_step_min_tokens > 0 ? h->cfg.fused_step_min_tokens : FL_FUSED_STEP_MIN_TOKENS;
  if (!h->grads_zero || h->Tr < min_tokens) {
    if (int rc = backward_impl(h, grad_out, grad_in)) return rc;
    return fl_server_step(h, lr);
  }
  const fl_server_cfg& c = h->cfg;
  const int64_t t = h->step_t + 1;
  h->fuse.on = true;
  h->fuse.lr = lr;
  // the same fp32 bias-correction factors fl_server_step passes to the AdamW kernel
  h->fuse.inv_bc1 = 1.f / (float)(1.0 - std::pow((double)c.adam_beta1, (double)t));
  h->fuse.inv_bc2 = 1.f / (float)(1.0 - std::pow((double)c.adam_beta2, (double)t));
  int rc = backward_impl(h, grad_out, grad_in);
  h->fuse.on = false;
  if (rc) return rc;
  h->step_t = t;
  // the bias / LayerNorm vectors and the prefixes (only the prefixes with a frozen base):
  // one AdamW launch over their contiguous region
  // (per replica)
  const int64_t first = c.freeze_base ? h->pre_base : h->vec_base;
  prof_begin(h, FL_PROF_ADAMW, h->R);
  for (int r = 0; r < h->R && rc == FL_OK; ++r) {
    const int64_t o = r * h->n_params + first;
    rc = fl_launch_adamw(h->n_params - first, h->w + o, h->g + o, h->m + o, h->v + o, h->wb + o, lr, c.adam_beta1,
                         c.adam_beta2, c.adam_eps, c.weight_decay,
                         (float)(1.0 - std::pow((double)c.adam_beta1, (double)t)),
                         (float)(1.0 - std::pow((double)c.adam_beta2, (double)t)), 0, h->stream);
  }
  prof_end(h);
  if (rc) return fwd_err(h, rc);
  h->grads_zero = true;  // matrix gradients were never written; vectors are cleared by the next backward
  return FL_OK;
}

extern "C" int fl_server_step(fl_server_t h, float lr) {
  if (!h) return fl_internal_error(FL_ERR_INVALID_ARG, "step: null handle");
  if (h->pending) return set_err(h, FL_ERR_STATE, "step: a forward is pending (call backward first)");
  const fl_server_cfg& c = h->cfg;
  h->step_t += 1;
  const double bc1 = 1.0 - std::pow((double)c.adam_beta1, (double)h->step_t);
  const double bc2 = 1.0 - std::pow((double)c.adam_beta2, (double)h->step_t);
  prof_begin(h, FL_PROF_ADAMW);
  // the gradients are not cleared here: the next backward overwrites them (grads_zero);
  // with a frozen base only the prefix region is updated (there is one replica then); with
  // replicas one launch covers every replica's arena
  const int64_t first = c.freeze_base ? h->pre_base : 0;
  int rc = fl_launch_adamw(h->n_all() - first, h->w + first, h->g + first, h->m + first, h->v + first, h->wb + first,
                           lr, c.adam_beta1, c.adam_beta2, c.adam_eps, c.weight_decay, (float)bc1, (float)bc2, 0,
                           h->stream);
  prof_end(h);
  if (rc == FL_OK) h->grads_zero = true;
  return fwd_err(h, rc);
}

extern "C" int fl_server_destroy(fl_server_t h) {
  if (!h) return FL_OK;
  cudaStreamSynchronize(h->stream);
  for (void* p : h->allocations) cudaFree(p);
  for (cudaEvent_t e : h->prof.pool) cudaEventDestroy(e);
  delete h;
  return FL_OK;
}

extern "C" int fl_server_set_stream(fl_server_t h, void* s) {
  if (!h) return fl_internal_error(FL_ERR_INVALID_ARG, "set_stream: null handle");
  h->stream = reinterpret_cast<cudaStream_t>(s);
  return FL_OK;
}

extern "C" int fl_server_sync(fl_server_t h) {
  if (!h) return fl_internal_error(FL_ERR_INVALID_ARG, "sync: null handle");
  cudaError_t e = cudaStreamSynchronize(h->stream);
  if (e != cudaSuccess) return fwd_err(h, fl_internal_cuda_error(e, "cudaStreamSynchronize", __FILE__, __LINE__));
  int st = 0;
  e = cudaMemcpy(&st, h->status, sizeof(int), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return fwd_err(h, fl_internal_cuda_error(e, "status read", __FILE__, __LINE__));
  if (st != 0) {
    cudaMemset(h->status, 0, sizeof(int));
    return set_err(h, FL_ERR_TIMEOUT, "a bounded device wait gave up (code %d)", st);
  }
  return FL_OK;
}

extern "C" int64_t fl_server_tensor_numel(fl_server_t h, int32_t t) {
  if (!h || t < 0 || t >= FL_T_COUNT) return -1;
  return h->tensor_n[t];  // 0 for the prefix tensors when there is no prefix
}

static int check_tensor(fl_server* h, int32_t b, int32_t t, const void* p, size_t n) {
  if (!h) return fl_internal_error(FL_ERR_INVALID_ARG, "null handle");
  if (b < 0 || b >= h->cfg.n_blocks || t < 0 || t >= FL_T_COUNT || h->tensor_n[t] == 0)
    return set_err(h, FL_ERR_INVALID_ARG, "bad block %d / tensor %d", b, t);
  if (!p) return set_err(h, FL_ERR_INVALID_ARG, "null host buffer");
  if ((int64_t)n != h->tensor_n[t])
    return set_err(h, FL_ERR_INVALID_ARG, "n=%zu but tensor %d has %lld elements", n, t, (long long)h->tensor_n[t]);
  return FL_OK;
}

// dst[c * rows + r] = src[r * cols + c]
static void transpose_host(const float* src, float* dst, int64_t rows, int64_t cols) {
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t c = 0; c < cols; ++c) dst[c * rows + r] = src[r * cols + c];
}

static int d2h(fl_server* h, float* dst, const float* src, size_t n) {
  cudaError_t e = cudaStreamSynchronize(h->stream);
  if (e == cudaSuccess) e = cudaMemcpy(dst, src, n * sizeof(float), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return fwd_err(h, fl_internal_cuda_error(e, "device to host copy", __FILE__, __LINE__));
  return FL_OK;
}

// Copies tensor t's arena values (at src) to dst in the tensor's own [rows, cols] order:
// the FFN up-projection weight, stored [H, F], is transposed back to [F, H].
static int d2h_tensor(fl_server* h, int t, float* dst, const float* src, size_t n) {
  if (t != FL_T_WUP) return d2h(h, dst, src, n);
  std::vector<float> tmp(n);
  if (int rc = d2h(h, tmp.data(), src, n)) return rc;
  transpose_host(tmp.data(), dst, h->cfg.hidden, h->cfg.ffn_hidden);
  return FL_OK;
}

extern "C" int fl_server_get_param(fl_server_t h, int32_t b, int32_t t, float* dst, size_t n) {
  if (int rc = check_tensor(h, b, t, dst, n)) return rc;
  return d2h_tensor(h, t, dst, h->wt(b, t), n);
}
extern "C" int fl_server_get_grad(fl_server_t h, int32_t b, int32_t t, float* dst, size_t n) {
  if (int rc = check_tensor(h, b, t, dst, n)) return rc;
  if (h->grads_zero) {  // after create or a step the gradients are zero by definition
    memset(dst, 0, n * sizeof(float));
    return FL_OK;
  }
  return d2h_tensor(h, t, dst, h->gt(b, t), n);
}
extern "C" int fl_server_get_adam_moments(fl_server_t h, int32_t b, int32_t t, float* hm, float* hv, size_t n) {
  if (int rc = check_tensor(h, b, t, hm, n)) return rc;
  if (!hv) return set_err(h, FL_ERR_INVALID_ARG, "null host buffer");
  const int64_t o = h->off(b, t);
  if (int rc = d2h_tensor(h, t, hm, h->m + o, n)) return rc;
  return d2h_tensor(h, t, hv, h->v + o, n);
}
extern "C" int fl_server_get_replica_param(fl_server_t h, int32_t r, int32_t b, int32_t t, float* dst, size_t n) {
  if (int rc = check_tensor(h, b, t, dst, n)) return rc;
  if (r < 0 || r >= h->R) return set_err(h, FL_ERR_INVALID_ARG, "replica %d outside [0, %d)", r, h->R);
  return d2h_tensor(h, t, dst, h->wt(b, t, r), n);
}
extern "C" int fl_server_set_param(fl_server_t h, int32_t b, int32_t t, const float* src, size_t n) {
  if (int rc = check_tensor(h, b, t, src, n)) return rc;
  std::vector<float> tmp;
  if (t == FL_T_WUP) {  // stored transposed, [H, F]
    tmp.resize(n);
    transpose_host(src, tmp.data(), h->cfg.ffn_hidden, h->cfg.hidden);
    src = tmp.data();
  }
  cudaError_t e = cudaStreamSynchronize(h->stream);
  for (int r = 0; r < h->R && e == cudaSuccess; ++r)  // every replica
    e = cudaMemcpy(h->wt(b, t, r), src, n * sizeof(float), cudaMemcpyHostToDevice);
  if (e != cudaSuccess) return fwd_err(h, fl_internal_cuda_error(e, "host to device copy", __FILE__, __LINE__));
  int rc = FL_OK;
  for (int r = 0; r < h->R && rc == FL_OK; ++r)
    rc = fl_launch_f32_to_bf16((int64_t)n, h->wt(b, t, r), h->wbt(b, t, r), h->stream);
  if (rc) return fwd_err(h, rc);
  e = cudaStreamSynchronize(h->stream);
  if (e != cudaSuccess) return fwd_err(h, fl_internal_cuda_error(e, "set_param", __FILE__, __LINE__));
  return FL_OK;
}

extern "C" int fl_server_average(fl_server_t const* replicas, int32_t n) {
  if (!replicas || n < 1 || n > FL_MAX_REPLICAS)
    return fl_internal_error(FL_ERR_INVALID_ARG, "average: need 1..%d replicas", FL_MAX_REPLICAS);
  fl_server* h0 = replicas[0];
  if (!h0) return fl_internal_error(FL_ERR_INVALID_ARG, "average: null replica");
  ReplicaTable t;
  memset(&t, 0, sizeof t);
  t.n = n;
  for (int r = 0; r < n; ++r) {
    fl_server* h = replicas[r];
    if (!h) return fl_internal_error(FL_ERR_INVALID_ARG, "average: null replica %d", r);
    if (h->n_params != h0->n_params || h->R != h0->R || h->cfg.n_blocks != h0->cfg.n_blocks ||
        h->cfg.hidden != h0->cfg.hidden || h->cfg.ffn_hidden != h0->cfg.ffn_hidden)
      return fl_internal_error(FL_ERR_INVALID_ARG, "average: replica %d has another shape", r);
    if (h->pending) return set_err(h, FL_ERR_STATE, "average: replica %d has a pending forward", r);
    for (int q = 0; q < r; ++q)
      if (replicas[q] == h) return fl_internal_error(FL_ERR_INVALID_ARG, "average: replica %d listed twice", r);
    t.w[r] = h->w;
    t.wb[r] = h->wb;
  }
  // order the averaging after every replica's queued work, on replica 0's stream
  for (int r = 1; r < n; ++r) {
    cudaError_t e = cudaStreamSynchronize(replicas[r]->stream);
    if (e != cudaSuccess) return fwd_err(h0, fl_internal_cuda_error(e, "average: sync", __FILE__, __LINE__));
  }
  prof_begin(h0, FL_PROF_OTHER);
  int rc = fl_launch_average(t, h0->n_all(), h0->stream);
  prof_end(h0);
  if (rc) return fwd_err(h0, rc);
  cudaError_t e = cudaStreamSynchronize(h0->stream);
  if (e != cudaSuccess) return fwd_err(h0, fl_internal_cuda_error(e, "average", __FILE__, __LINE__));
  return FL_OK;
}

extern "C" int fl_server_param_arena(fl_server_t h, float** dev_w, int64_t* n) {
  if (!h || !dev_w || !n) return fl_internal_error(FL_ERR_INVALID_ARG, "param_arena: null");
  *dev_w = h->w;
  *n = h->n_all();
  return FL_OK;
}

extern "C" int fl_server_average_finish(fl_server_t h, int32_t n_replicas) {
  if (!h) return fl_internal_error(FL_ERR_INVALID_ARG, "average finish: null handle");
  if (n_replicas < 1) return set_err(h, FL_ERR_INVALID_ARG, "average finish: n_replicas=%d < 1", n_replicas);
  if (h->pending) return set_err(h, FL_ERR_STATE, "average finish: a forward is pending");
  prof_begin(h, FL_PROF_OTHER);
  int rc = fl_launch_mean_finish(h->n_all(), n_replicas, h->w, h->wb, h->stream);
  prof_end(h);
  return fwd_err(h, rc);
}

extern "C" int fl_server_average_replicas(fl_server_t h) {
  if (!h) return fl_internal_error(FL_ERR_INVALID_ARG, "average replicas: null handle");
  if (h->pending) return set_err(h, FL_ERR_STATE, "average replicas: a forward is pending");
  if (h->R < 2) return FL_OK;
  ReplicaTable t;
  memset(&t, 0, sizeof t);
  t.n = h->R;
  for (int r = 0; r < h->R; ++r) {
    t.w[r] = h->w + r * h->n_params;
    t.wb[r] = h->wb + r * h->n_params;
  }
  prof_begin(h, FL_PROF_OTHER);
  int rc = fl_launch_average(t, h->n_params, h->stream);
  prof_end(h);
  return fwd_err(h, rc);
}

extern "C" int fl_server_refresh_working_copy(fl_server_t h) {
  if (!h) return fl_internal_error(FL_ERR_INVALID_ARG, "refresh: null handle");
  int rc = fl_launch_f32_to_bf16(h->n_all(), h->w, h->wb, h->stream);
  return fwd_err(h, rc);
}

extern "C" int fl_server_profile(fl_server_t h, int enable) {
  if (!h) return fl_internal_error(FL_ERR_INVALID_ARG, "profile: null handle");
  cudaStreamSynchronize(h->stream);
  h->prof.on = enable != 0;
  h->prof.marks.clear();
  h->prof.used = 0;
  return FL_OK;
}

extern "C" int fl_server_profile_read(fl_server_t h, double* ms, int64_t* launches, int32_t n) {
  if (!h || !ms || !launches || n < 0 || n > FL_PROF_CLASSES)
    return fl_internal_error(FL_ERR_INVALID_ARG, "profile_read: args");
  cudaError_t e = cudaStreamSynchronize(h->stream);
  if (e != cudaSuccess) return fwd_err(h, fl_internal_cuda_error(e, "profile sync", __FILE__, __LINE__));
  for (int i = 0; i < n; ++i) {
    ms[i] = 0;
    launches[i] = 0;
  }
  for (auto& mk : h->prof.marks) {
    if (mk.first >= n) continue;
    float t = 0.f;
    cudaEventElapsedTime(&t, h->prof.pool[mk.second], h->prof.pool[mk.second + 1]);
    ms[mk.first] += t;
    launches[mk.first] += 1;
  }
  return FL_OK;
}

extern "C" int64_t fl_server_launch_count(fl_server_t h) { return h ? h->launches : -1; }

extern "C" const char* fl_server_last_error(fl_server_t h) {
  if (h) return h->err.c_str();
  return g_last_error.c_str();
}
