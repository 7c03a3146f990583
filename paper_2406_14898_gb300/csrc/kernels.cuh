// Internal launch interfaces shared by the kernels and the server runtime.
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

constexpr int FL_MAX_COPY = 64;       // client tensors per gather/scatter launch
constexpr int FL_MAX_SEGS = 1024;     // causal segments per call
constexpr int FL_MAX_TILES = 2048;    // 64-row attention tiles per call
constexpr int FL_ATTN_TILE = 64;

// Client <-> packed copies.  Units of 8 elements (16 bytes of bf16, 32 bytes of fp32).
enum CopyMode {
  COPY_GATHER_BF16 = 0,   // client bf16 -> packed bf16 (bit-exact)
  COPY_SCATTER_BF16 = 1,  // packed bf16 -> client bf16 (bit-exact)
  COPY_GATHER_F32 = 2,    // client bf16 -> packed fp32 (exact widening) and, if packed_bf16, a bf16 copy
  COPY_SCATTER_F32 = 3,   // packed fp32 -> client bf16 (round to nearest even)
};
struct CopyTable {
  int n;
  int mode;
  void* packed_bf16;
  float* packed_f32;
  void* client[FL_MAX_COPY];
  int64_t off8[FL_MAX_COPY];  // offset into the packed buffer, 8-element units
  int64_t n8[FL_MAX_COPY];    // length, 8-element units
};

// Packing metadata of one call, passed by value to the metadata kernel.
// tiles[i] = segment << 16 | tile index inside the segment, ordered by decreasing tile
// index (the longest causal rows first).
// With glm = 1 every segment s carries a GLM blank-infilling structure: context length
// ctx[s] (0: plain causal segment) and mask-token position mpos[s] < ctx[s].
struct MetaArgs {
  int S;
  int n_tiles;    // 64-row tiles, then n_tiles128 128-row tiles (the tcgen05 attention kernels)
  int n_tiles128;
  int glm;
  int32_t cu[FL_MAX_SEGS + 1];
  uint32_t tiles[2 * FL_MAX_TILES];
  int32_t ctx[FL_MAX_SEGS];
  int32_t mpos[FL_MAX_SEGS];
};

int fl_launch_copy_clients(const CopyTable& tab, cudaStream_t st);

// Replicas averaged together: fp32 master arenas and bf16 copies, same length.
constexpr int FL_MAX_REPLICAS = 64;
struct ReplicaTable {
  int n;
  float* w[FL_MAX_REPLICAS];
  void* wb[FL_MAX_REPLICAS];
};
int fl_launch_average(const ReplicaTable& t, int64_t n, cudaStream_t st);
// w[i] *= 1/n_replicas (the factor fl_launch_average applies) and wb[i] = bf16(w[i]).
int fl_launch_mean_finish(int64_t n, int n_replicas, float* w, void* wb, cudaStream_t st);
// Writes cu_seqlens, the tile list, per-token positions (and, when pos2 != NULL, the GLM
// block positions and, when ctx != NULL, the per-segment context lengths; both zero
// without glm).
int fl_launch_meta(const MetaArgs& a, int32_t* cu, int32_t* pos, uint32_t* tiles, int32_t* pos2, int32_t* ctx,
                   cudaStream_t st);
int fl_launch_normal_init(int64_t n, uint64_t key, double mean, double std_, float* out, cudaStream_t st);
int fl_launch_fill(int64_t n, float v, float* out, cudaStream_t st);
int fl_launch_adamw(int64_t n, float* w, float* g, float* m, float* v, void* w_bf16, float lr, float beta1,
                    float beta2, float eps, float weight_decay, float bc1, float bc2, int zero_grad, cudaStream_t st);
int fl_launch_f32_to_bf16(int64_t n, const float* src, void* dst, cudaStream_t st);
// dst [cols, rows] = the transpose of src [rows, cols] (fp32; src and dst do not overlap).
int fl_launch_transpose_f32(int64_t rows, int64_t cols, const float* src, float* dst, cudaStream_t st);

// P-tuning v2 prefix of one block's attention: bf16 keys/values [len, H] (head j at
// column j*head_dim) seen by every query, and fp32 gradient accumulators (backward).
struct AttnPrefix {
  const void* k = nullptr;
  const void* v = nullptr;
  int len = 0;
  float* dk = nullptr;
  float* dv = nullptr;
};

// GLM blank-infilling structure of a call (all NULL: plain causal segments, positions =
// index inside the segment, second rotary half not rotated).
struct AttnGlm {
  const int32_t* ctx = nullptr;   // [S] context length per segment (key u visible to query t iff u <= max(t, ctx-1))
  const int32_t* pos = nullptr;   // [T] first position (inverse rotary of dims [0, hd/2))
  const int32_t* pos2 = nullptr;  // [T] block position (inverse rotary of dims [hd/2, hd))
};

// Attention on a device tile list (built by fl_launch_meta): the 64-row list (n_tiles
// entries) followed by the 128-row one (n_tiles128) that the tcgen05 kernels walk.
// head_dim 64 or 128; `status` (device int or null) receives a code if a bounded wait
// inside a kernel gave up.
int fl_launch_attn_fwd(int T, int nh, int hd, const void* qkv, const int32_t* cu, const uint32_t* tiles,
                       int n_tiles, int n_tiles128, void* o, float* lse, const AttnPrefix& pre, const AttnGlm& glm,
                       cudaStream_t st, int* status = nullptr);
// tiles: the 128-row list alone (attention_tc.cu).
int fl_launch_attn_fwd_tc(int T, int nh, int hd, const void* qkv, const int32_t* cu, const uint32_t* tiles,
                          int n_tiles, void* o, float* lse, const AttnPrefix& pre, const AttnGlm& glm, int* status,
                          cudaStream_t st);
// dbias (or null): += the column sums of dqkv [3H] (the QKV bias gradient), per CTA; with
// dbias_segs > 0 the sums of segment s go to dbias + (s / dbias_segs) * dbias_rstride (the
// replicas of one handle, dbias_segs segments each).
// delta: fp32 [nh, T] scratch (rowsum(dO * O), written here).
int fl_launch_attn_bwd(int T, int nh, int hd, const void* qkv, const void* o, const float* lse, const void* dout,
                       const int32_t* cu, const uint32_t* tiles, int n_tiles, int n_tiles128, float* delta,
                       const float* rope_tab,
                       void* dqkv, const AttnPrefix& pre, const AttnGlm& glm, cudaStream_t st,
                       float* dbias = nullptr, int* status = nullptr, int dbias_segs = 0, int64_t dbias_rstride = 0);
// dQ, dK / dV and, with a prefix, the prefix keys' gradients (attention_bwd_tc.cu); tiles:
// the 128-row list alone; delta already computed.
int fl_launch_attn_bwd_tc(int T, int nh, int hd, const void* qkv, const void* dout, const float* lse,
                          const float* delta, const int32_t* cu, const uint32_t* tiles, int n_tiles,
                          const float* rope_tab, void* dqkv, const AttnPrefix& pre, const AttnGlm& glm, float* dbias,
                          int* status, cudaStream_t st, int dbias_segs = 0, int64_t dbias_rstride = 0);

// LayerNorm backward on fp32 dy / x (rowops.cu): fl_k_layernorm_bwd, and, when dcol is not
// null, dcol += the column sums of dx.  workspace: fl_launch_layernorm_bwd_workspace bytes.
size_t fl_launch_layernorm_bwd_workspace(int T, int H);
int fl_launch_layernorm_bwd_f32(int T, int H, const float* dy, const float* x, const float* mean, const float* rstd,
                                const float* gamma, const float* resid, float resid_alpha, __nv_bfloat16* dx_bf16,
                                float* dx_f32, float* dgamma, float* dbeta, float* dcol, float* workspace,
                                cudaStream_t st, int* status = nullptr);
// LayerNorm forward of fp32 rows (fl_k_layernorm_fwd); x 16-byte aligned; `status` (device int
// or null) receives a code if a bounded wait gave up.
int fl_launch_layernorm_fwd_f32(int T, int H, const float* x, const float* gamma, const float* beta, float eps,
                                __nv_bfloat16* y, float* mean, float* rstd, cudaStream_t st, int* status = nullptr);

// Host helper: builds the tile list of a packing, tiles of `rows` query rows (128 for the
// tcgen05 kernels): segments by decreasing length, each segment's tiles consecutive, its
// last tile first (returns the count, -1 if over capacity).  The units of the persistent
// attention kernels are (list entry, head), so the tiles of one segment and head, which
// read the same key / value (or query / output-gradient) tiles, run at about the same
// time and share them in L2.  A device tile list holds the 64-row list followed by the
// 128-row one.
int fl_build_tiles(const int32_t* cu, int S, uint32_t* tiles, int max_tiles, int rows = 64);
