// Varlen causal attention over packed client segments (App. A: softmax(Q K^T / sqrt(d_h)) V),
// each client row attending only to earlier tokens of its own segment (§3.3 stacks
// clients; it does not mix them).  A segment may carry a GLM blank-infilling structure
// (§4.1.1): with context length c, query t sees the keys u <= max(t, c - 1), i.e. the
// context is bidirectional and the answer span causal; c = 0 is the plain causal case.
//
// The tile kernels run on tcgen05 for head_dim 64 and 128 (attention_tc.cu: forward;
// attention_bwd_tc.cu: dQ, dK / dV, and the P-tuning prefix keys' dK / dV).  This file
// holds delta = rowsum(dO * O) of the backward, the tile lists, the dispatch and the
// exported kernel entry points.  dQ and dK leave the backward through the inverse rotary
// rotation (the forward rotation is applied in the QKV GEMM epilogue), so the result is
// the gradient w.r.t. the un-rotated q and k.
#include <algorithm>
#include <cmath>
#include <vector>

#include "../../include/flglm_kernels.h"
#include "common.cuh"
#include "kernels.cuh"
#include "ptx.cuh"

namespace {

typedef __nv_bfloat16 bf16;
constexpr int BT = 64;  // rows of the 64-row tile list (the first part of a tile workspace)

// ---------------------------------------------------------------------------- delta = rowsum(dO * O)
// G = HD/8 lanes per (token, head) pair, one 16-byte load of O and of dO each; pairs
// ordered head-major so that a warp's pairs are consecutive tokens of one head (coalesced
// delta stores).
template <int HD>
__global__ void __launch_bounds__(256) attn_delta_kernel(int T, int H, int nh, const bf16* __restrict__ O,
                                                         const bf16* __restrict__ dO, float* __restrict__ delta) {
  pdl_wait();  // the previous kernel on the stream has completed (see fl_launch)
  pdl_trigger();
  constexpr int G = HD / 8;
  const int64_t gid = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  const int64_t p = gid / G;
  const int sub = threadIdx.x % G;
  const bool ok = p < (int64_t)T * nh;
  float s = 0.f;
  int h = 0, t = 0;
  if (ok) {
    h = int(p / T);
    t = int(p % T);
    const int64_t off = (int64_t)t * H + h * HD + sub * 8;
    const uint4 a = __ldg(reinterpret_cast<const uint4*>(O + off));
    const uint4 b = __ldg(reinterpret_cast<const uint4*>(dO + off));
    const uint32_t aw[4] = {a.x, a.y, a.z, a.w}, bw[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float2 x = unpack_bf16x2(aw[e]), y = unpack_bf16x2(bw[e]);
      s = fmaf(x.x, y.x, fmaf(x.y, y.y, s));
    }
  }
#pragma unroll
  for (int off = G / 2; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
  if (ok && sub == 0) delta[(int64_t)h * T + t] = s;
}

}  // namespace

int fl_build_tiles(const int32_t* cu, int S, uint32_t* tiles, int max_tiles, int rows) {
  // segments by decreasing tile count (stable), each segment's tiles next to each other,
  // its last (longest causal) tile first
  std::vector<int> order(S > 0 ? S : 0);
  for (int s = 0; s < S; ++s) order[s] = s;
  auto ntiles = [&](int s) { return (cu[s + 1] - cu[s] + rows - 1) / rows; };
  std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return ntiles(a) > ntiles(b); });
  int n = 0;
  for (int s : order)
    for (int i = ntiles(s) - 1; i >= 0; --i) {
      if (n >= max_tiles) return -1;
      tiles[n++] = (uint32_t(s) << 16) | uint32_t(i);
    }
  return n;
}

int fl_launch_attn_fwd(int T, int nh, int hd, const void* qkv, const int32_t* cu, const uint32_t* tiles, int n_tiles,
                       int n_tiles128,
                       void* o, float* lse, const AttnPrefix& pre, const AttnGlm& glm, cudaStream_t st, int* status) {
  if (n_tiles <= 0) return FL_OK;
  if (hd != 64 && hd != 128) return fl_internal_error(FL_ERR_UNSUPPORTED, "attention: head_dim %d", hd);
  return fl_launch_attn_fwd_tc(T, nh, hd, qkv, cu, tiles + n_tiles, n_tiles128, o, lse, pre, glm, status, st);
}

int fl_launch_attn_bwd(int T, int nh, int hd, const void* qkv, const void* o, const float* lse, const void* dout,
                       const int32_t* cu, const uint32_t* tiles, int n_tiles, int n_tiles128, float* delta,
                       const float* rope_tab, void* dqkv, const AttnPrefix& pre, const AttnGlm& glm, cudaStream_t st,
                       float* dbias, int* status, int dbias_segs, int64_t dbias_rstride) {
  if (n_tiles <= 0) return FL_OK;
  if (hd != 64 && hd != 128) return fl_internal_error(FL_ERR_UNSUPPORTED, "attention: head_dim %d", hd);
  const int64_t pairs = (int64_t)T * nh;
  const int H = nh * hd;
  if (hd == 128)
    FL_CUDA_TRY(fl_launch(attn_delta_kernel<128>, dim3((unsigned)((pairs * 16 + 255) / 256)), dim3(256), 0, st, T, H,
                          nh, (const bf16*)o, (const bf16*)dout, delta));
  else
    FL_CUDA_TRY(fl_launch(attn_delta_kernel<64>, dim3((unsigned)((pairs * 8 + 255) / 256)), dim3(256), 0, st, T, H,
                          nh, (const bf16*)o, (const bf16*)dout, delta));
  return fl_launch_attn_bwd_tc(T, nh, hd, qkv, dout, lse, delta, cu, tiles + n_tiles, n_tiles128, rope_tab, dqkv, pre,
                               glm, dbias, status, st, dbias_segs, dbias_rstride);
}

// ====================================================================== exported kernel API

extern "C" int32_t fl_k_attention_tiles(const int32_t* cu_host, int32_t S) {
  if (!cu_host || S <= 0) return 0;
  int n = 0;
  for (int s = 0; s < S; ++s) n += (cu_host[s + 1] - cu_host[s] + BT - 1) / BT;
  return n;
}

// The 64-row tile list followed by the 128-row one (at most as long) in tile_ws.
static int upload_tiles(const int32_t* cu_host, int32_t S, int32_t* tile_ws, int* n_out, int* n128_out) {
  const int n = fl_k_attention_tiles(cu_host, S);
  for (int s = 0; s < S; ++s)
    if (cu_host[s + 1] < cu_host[s] || cu_host[s + 1] - cu_host[s] > 65535 * BT)
      return fl_internal_error(FL_ERR_INVALID_ARG, "attention: bad cu_seqlens");
  std::vector<uint32_t> t(2 * (n > 0 ? n : 1));
  const int got = fl_build_tiles(cu_host, S, t.data(), n);
  if (got != n) return fl_internal_error(FL_ERR_INVALID_ARG, "attention: bad cu_seqlens");
  const int n128 = n > 0 ? fl_build_tiles(cu_host, S, t.data() + n, n, 2 * BT) : 0;
  if (n128 < 0) return fl_internal_error(FL_ERR_INVALID_ARG, "attention: bad cu_seqlens");
  if (n > 0) FL_CUDA_TRY(cudaMemcpy(tile_ws, t.data(), (n + n128) * sizeof(uint32_t), cudaMemcpyHostToDevice));
  *n_out = n;
  *n128_out = n128;
  return FL_OK;
}

extern "C" int fl_k_attention_fwd(int32_t T, int32_t n_heads, int32_t head_dim, const void* qkv,
                                  const int32_t* cu_seqlens_host, const int32_t* cu_seqlens, int32_t S,
                                  int32_t* tile_ws, void* o, float* lse, const void* prefix_k, const void* prefix_v,
                                  int32_t prefix_len, const int32_t* context_lens, void* stream) {
  if (!qkv || !cu_seqlens_host || !cu_seqlens || !tile_ws || !o || !lse || S <= 0 || S >= 65536)
    return fl_internal_error(FL_ERR_INVALID_ARG, "attention fwd: args");
  if (cu_seqlens_host[0] != 0 || cu_seqlens_host[S] != T) return fl_internal_error(FL_ERR_INVALID_ARG, "attention fwd: cu_seqlens");
  if (prefix_len < 0 || prefix_len > 128 || (prefix_len > 0 && (!prefix_k || !prefix_v)))
    return fl_internal_error(FL_ERR_INVALID_ARG, "attention fwd: prefix (length 0..128)");
  if (fl_misaligned(qkv, 16) || fl_misaligned(o, 16) || fl_misaligned(lse, 4) || fl_misaligned(cu_seqlens, 4) ||
      fl_misaligned(tile_ws, 4) || fl_misaligned(context_lens, 4))
    return fl_internal_error(FL_ERR_INVALID_ARG, "attention fwd: qkv and o must be 16-byte aligned");
  int n = 0, n128 = 0;
  if (int rc = upload_tiles(cu_seqlens_host, S, tile_ws, &n, &n128)) return rc;
  AttnPrefix pre;
  pre.k = prefix_k;
  pre.v = prefix_v;
  pre.len = prefix_len;
  AttnGlm glm;
  glm.ctx = context_lens;
  return fl_launch_attn_fwd(T, n_heads, head_dim, qkv, cu_seqlens, (const uint32_t*)tile_ws, n, n128, o, lse, pre, glm,
                            (cudaStream_t)stream);
}

extern "C" int fl_k_attention_bwd(int32_t T, int32_t n_heads, int32_t head_dim, const void* qkv, const void* o,
                                  const float* lse, const void* dout, const int32_t* cu_seqlens_host,
                                  const int32_t* cu_seqlens, int32_t S, int32_t* tile_ws, float* delta_ws,
                                  const float* rope_tab, int32_t rotary_dim, void* dqkv, const void* prefix_k,
                                  const void* prefix_v, int32_t prefix_len, float* dprefix_k, float* dprefix_v,
                                  const int32_t* context_lens, const int32_t* positions,
                                  const int32_t* block_positions, void* stream) {
  if (!qkv || !o || !lse || !dout || !cu_seqlens_host || !cu_seqlens || !tile_ws || !delta_ws || !dqkv || S <= 0 ||
      S >= 65536)
    return fl_internal_error(FL_ERR_INVALID_ARG, "attention bwd: args");
  if (cu_seqlens_host[0] != 0 || cu_seqlens_host[S] != T) return fl_internal_error(FL_ERR_INVALID_ARG, "attention bwd: cu_seqlens");
  if (rope_tab && rotary_dim != head_dim / 2)
    return fl_internal_error(FL_ERR_UNSUPPORTED, "attention bwd: rotary_dim must be head_dim / 2");
  if (rope_tab && (reinterpret_cast<uintptr_t>(rope_tab) & 15))  // rows are read as 16-byte vectors
    return fl_internal_error(FL_ERR_INVALID_ARG, "attention bwd: rope_tab is not 16-byte aligned");
  if (prefix_len < 0 || prefix_len > 128 ||
      (prefix_len > 0 && (!prefix_k || !prefix_v || !dprefix_k || !dprefix_v)))
    return fl_internal_error(FL_ERR_INVALID_ARG, "attention bwd: prefix (length 0..128, gradients required)");
  if (fl_misaligned(qkv, 16) || fl_misaligned(o, 16) || fl_misaligned(dout, 16) || fl_misaligned(dqkv, 16) ||
      fl_misaligned(dprefix_k, 16) || fl_misaligned(dprefix_v, 16) || fl_misaligned(lse, 4) ||
      fl_misaligned(delta_ws, 4) || fl_misaligned(cu_seqlens, 4) || fl_misaligned(tile_ws, 4) ||
      fl_misaligned(context_lens, 4) || fl_misaligned(positions, 4) || fl_misaligned(block_positions, 4))
    return fl_internal_error(FL_ERR_INVALID_ARG,
                             "attention bwd: qkv, o, dout, dqkv and the prefix gradients must be 16-byte aligned");
  int n = 0, n128 = 0;
  if (int rc = upload_tiles(cu_seqlens_host, S, tile_ws, &n, &n128)) return rc;
  AttnPrefix pre;
  pre.k = prefix_k;
  pre.v = prefix_v;
  pre.len = prefix_len;
  pre.dk = dprefix_k;
  pre.dv = dprefix_v;
  AttnGlm glm;
  glm.ctx = context_lens;
  glm.pos = positions;
  glm.pos2 = block_positions;
  return fl_launch_attn_bwd(T, n_heads, head_dim, qkv, o, lse, dout, cu_seqlens, (const uint32_t*)tile_ws, n, n128,
                            delta_ws, rope_tab, dqkv, pre, glm, (cudaStream_t)stream);
}
