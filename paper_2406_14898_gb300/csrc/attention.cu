// Varlen causal attention over packed client segments (App. A: softmax(Q K^T / sqrt(d_h)) V),
// each client row attending only to earlier tokens of its own segment (§3.3 stacks
// clients; it does not mix them).  A segment may carry a GLM blank-infilling structure
// (§4.1.1): with context length c, query t sees the keys u <= max(t, c - 1), i.e. the
// context is bidirectional and the answer span causal; c = 0 is the plain causal case.
//
// Forward: one CTA per (64-query tile, head); online softmax over 64-key tiles with bf16
// mma.sync m16n8k16 (fp32 accumulate).  Saves O (bf16) and the row log-sum-exp (fp32).
// One K/V tile buffer and Q fragments re-read from shared memory per key tile: 52 KB of
// shared memory and 128 registers, so four CTAs share an SM and hide each other's copy
// latency (double buffering inside the CTA would cap it at two).
// Backward, deterministic, no atomics:
//   delta = rowsum(dO * O);
//   dQ  kernel: per (query tile, head), loop over key tiles: P, dP = dO V^T, dS, dQ += dS K
//               (one K/V buffer, 70 KB of shared memory: three CTAs per SM);
//   dKV kernel: per (key tile, head), loop over query tiles: dV += P^T dO, dK += dS^T Q;
// dQ and dK leave through the inverse rotary rotation (the forward rotation is applied in
// the QKV GEMM epilogue), so the result is the gradient w.r.t. the un-rotated q and k.
#include <cmath>
#include <vector>

#include "../../include/flglm_kernels.h"
#include "common.cuh"
#include "kernels.cuh"
#include "ptx.cuh"

namespace {

typedef __nv_bfloat16 bf16;
constexpr int BT = 64;  // rows per tile (queries or keys)
constexpr float LOG2E = 1.4426950408889634f;
constexpr float LN2 = 0.6931471805599453f;

template <int HD>
struct AT {
  static constexpr int SROW = HD + 8;                 // padded smem row (elements)
  static constexpr int TILE_ELEMS = BT * SROW;
  static constexpr int TILE_BYTES = TILE_ELEMS * 2;
};

// 64 rows x HD columns from global (row stride ld elements) into padded smem; rows >= valid
// are zero-filled without touching global memory.
template <int HD>
FL_DEV void load_tile(bf16* sdst, const bf16* g, int64_t ld, int valid, int tid) {
  constexpr int CPR = HD / 8;  // 16-byte chunks per row
  for (int c = tid; c < BT * CPR; c += 128) {
    const int r = c / CPR, cc = c % CPR;
    const bool ok = r < valid;
    const bf16* src = ok ? g + (int64_t)r * ld + cc * 8 : g;
    cp_async_16(smem_u32(sdst + r * AT<HD>::SROW + cc * 8), src, ok);
  }
}

// A fragment (16 rows x 16 cols at row0, col0) of a row-major padded smem tile.
template <int HD>
FL_DEV void ld_a(const bf16* s, int row0, int col0, int lane, uint32_t (&a)[4]) {
  const int r = row0 + (lane & 15);
  const int c = col0 + ((lane >> 4) << 3);
  ldmatrix_x4(smem_u32(s + r * AT<HD>::SROW + c), a[0], a[1], a[2], a[3]);
}
// B fragments of two adjacent n-tiles, B(k, n) = S[n][k] (rows of the tile are n):
// n in [n0, n0+16), k in [k0, k0+16).  b[0..1] -> n-tile n0, b[2..3] -> n-tile n0+8.
template <int HD>
FL_DEV void ld_b_rows(const bf16* s, int n0, int k0, int lane, uint32_t (&b)[4]) {
  const int j = lane >> 3;
  const int r = n0 + (lane & 7) + ((j >> 1) << 3);
  const int c = k0 + ((j & 1) << 3);
  ldmatrix_x4(smem_u32(s + r * AT<HD>::SROW + c), b[0], b[1], b[2], b[3]);
}
// B fragments of two adjacent n-tiles, B(k, n) = S[k][n] (rows of the tile are k):
// k in [k0, k0+16), n in [n0, n0+16).
template <int HD>
FL_DEV void ld_b_cols(const bf16* s, int k0, int n0, int lane, uint32_t (&b)[4]) {
  const int j = lane >> 3;
  const int r = k0 + (lane & 7) + ((j & 1) << 3);
  const int c = n0 + ((j >> 1) << 3);
  ldmatrix_x4_trans(smem_u32(s + r * AT<HD>::SROW + c), b[0], b[1], b[2], b[3]);
}

FL_DEV float quad_max(float v) {
  v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 1));
  return fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 2));
}
FL_DEV float quad_sum(float v) {
  v += __shfl_xor_sync(0xffffffffu, v, 1);
  return v + __shfl_xor_sync(0xffffffffu, v, 2);
}

FL_DEV void decode_tile(uint32_t t, int& s, int& idx) {
  s = int(t >> 16);
  idx = int(t & 0xFFFFu);
}

// ---------------------------------------------------------------------------- forward
template <int HD>
__global__ void __launch_bounds__(128, 4) attn_fwd_kernel(int T, int H, const bf16* __restrict__ qkv,
                                                       const int32_t* __restrict__ cu,
                                                       const uint32_t* __restrict__ tiles, bf16* __restrict__ O,
                                                       float* __restrict__ lse, float scale_log2,
                                                       const bf16* __restrict__ pk, const bf16* __restrict__ pv,
                                                       int Lp, const int32_t* __restrict__ ctxs) {
  extern __shared__ __align__(128) uint8_t smem[];
  bf16* sQ = reinterpret_cast<bf16*>(smem);
  bf16* sK = sQ + AT<HD>::TILE_ELEMS;      // one tile
  bf16* sV = sK + AT<HD>::TILE_ELEMS;      // one tile
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  int s, idx;
  decode_tile(tiles[blockIdx.x], s, idx);
  const int h = blockIdx.y;
  const int seg0 = cu[s], L = cu[s + 1] - seg0;
  const int q0 = idx * BT;
  const int64_t ld = 3 * (int64_t)H;
  const bf16* gQ = qkv + (int64_t)(seg0 + q0) * ld + h * HD;
  const bf16* gK = qkv + (int64_t)seg0 * ld + H + h * HD;
  const bf16* gV = qkv + (int64_t)seg0 * ld + 2 * H + h * HD;

  // key tiles: first the prefix tiles (t < npt), then the segment's tiles up to the last
  // key any query of this tile sees (the diagonal, or the end of the GLM context)
  const int npt = (Lp + BT - 1) / BT;
  const int clast = (ctxs ? min(max(ctxs[s], 0), L) : 0) - 1;  // last context key, -1 without a context
  const int n_kv = npt + max(idx, clast >= 0 ? clast / BT : 0) + 1;
  const int qlim0 = max(q0, clast);              // smallest key limit among the tile's queries
  auto load_kv = [&](int t) {
    if (t < npt) {
      const int k0 = t * BT;
      load_tile<HD>(sK, pk + (int64_t)k0 * H + h * HD, H, min(BT, Lp - k0), tid);
      load_tile<HD>(sV, pv + (int64_t)k0 * H + h * HD, H, min(BT, Lp - k0), tid);
    } else {
      const int k0 = (t - npt) * BT;
      load_tile<HD>(sK, gK + (int64_t)k0 * ld, ld, min(BT, L - k0), tid);
      load_tile<HD>(sV, gV + (int64_t)k0 * ld, ld, min(BT, L - k0), tid);
    }
  };
  load_tile<HD>(sQ, gQ, ld, min(BT, L - q0), tid);
  load_kv(0);
  cp_async_commit();

  float o[HD / 8][4];
#pragma unroll
  for (int i = 0; i < HD / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float mrow[2] = {-INFINITY, -INFINITY}, lrow[2] = {0.f, 0.f};

  for (int j = 0; j < n_kv; ++j) {
    cp_async_wait<0>();
    __syncthreads();
    const bf16* K = sK;
    const bf16* V = sV;
    float sc[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i) sc[i][0] = sc[i][1] = sc[i][2] = sc[i][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
      uint32_t qa[4];
      ld_a<HD>(sQ, warp * 16, kk * 16, lane, qa);
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        uint32_t b[4];
        ld_b_rows<HD>(K, np * 16, kk * 16, lane, b);
        mma_bf16_16816(sc[2 * np], qa, b[0], b[1]);
        mma_bf16_16816(sc[2 * np + 1], qa, b[2], b[3]);
      }
    }
    const int kb = (j - npt) * BT;  // first key of a segment tile
    const bool need_mask = j >= npt && kb + BT - 1 > qlim0;
    const int pvalid = j < npt ? min(BT, Lp - j * BT) : BT;  // valid prefix keys of this tile
    float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        float x = sc[nt][e] * scale_log2;
        const int kl = nt * 8 + 2 * (lane & 3) + (e & 1);
        if (need_mask) {
          const int ql = warp * 16 + (lane >> 2) + ((e >> 1) << 3);
          if (kb + kl > max(q0 + ql, clast)) x = -INFINITY;
        }
        if (kl >= pvalid) x = -INFINITY;
        sc[nt][e] = x;
        mx[e >> 1] = fmaxf(mx[e >> 1], x);
      }
    }
    float corr[2];
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const float mn = fmaxf(mrow[r], quad_max(mx[r]));
      corr[r] = exp2f(mrow[r] - mn);
      mrow[r] = mn;
      lrow[r] *= corr[r];
    }
#pragma unroll
    for (int i = 0; i < HD / 8; ++i) {
      o[i][0] *= corr[0]; o[i][1] *= corr[0];
      o[i][2] *= corr[1]; o[i][3] *= corr[1];
    }
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float p = exp2f(sc[nt][e] - mrow[e >> 1]);
        sc[nt][e] = p;
        lrow[e >> 1] += p;
      }
    }
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      uint32_t a[4];
      a[0] = pack_bf16x2(sc[2 * kk][0], sc[2 * kk][1]);
      a[1] = pack_bf16x2(sc[2 * kk][2], sc[2 * kk][3]);
      a[2] = pack_bf16x2(sc[2 * kk + 1][0], sc[2 * kk + 1][1]);
      a[3] = pack_bf16x2(sc[2 * kk + 1][2], sc[2 * kk + 1][3]);
#pragma unroll
      for (int np = 0; np < HD / 16; ++np) {
        uint32_t b[4];
        ld_b_cols<HD>(V, kk * 16, np * 16, lane, b);
        mma_bf16_16816(o[2 * np], a, b[0], b[1]);
        mma_bf16_16816(o[2 * np + 1], a, b[2], b[3]);
      }
    }
    __syncthreads();
    if (j + 1 < n_kv) {  // every warp is done with the tile: load the next one into it
      load_kv(j + 1);
      cp_async_commit();
    }
  }

#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const float lt = quad_sum(lrow[r]);
    const float inv = 1.f / lt;
    const int q = q0 + warp * 16 + (lane >> 2) + 8 * r;
    if (q < L) {
      bf16* orow = O + (int64_t)(seg0 + q) * H + h * HD + 2 * (lane & 3);
#pragma unroll
      for (int nt = 0; nt < HD / 8; ++nt)
        *reinterpret_cast<uint32_t*>(orow + nt * 8) = pack_bf16x2(o[nt][2 * r] * inv, o[nt][2 * r + 1] * inv);
      if ((lane & 3) == 0) lse[(int64_t)h * T + seg0 + q] = (mrow[r] + log2f(lt)) * LN2;
    }
  }
}

// ---------------------------------------------------------------------------- delta = rowsum(dO * O)
// G = HD/8 lanes per (token, head) pair, one 16-byte load of O and of dO each; pairs
// ordered head-major so that a warp's pairs are consecutive tokens of one head (coalesced
// delta stores).
template <int HD>
__global__ void __launch_bounds__(256) attn_delta_kernel(int T, int H, int nh, const bf16* __restrict__ O,
                                                         const bf16* __restrict__ dO, float* __restrict__ delta) {
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

// Inverse rotary rotation of an accumulator fragment: the thread holds, for n-tile nt,
// dims 8 nt + 2 (lane & 3) + {0, 1} of row r (elements 2r, 2r+1).  A rotary region is
// half a head (HD/2 dims starting at n-tile NT0: 0 for the first position, HD/16 for the
// GLM block position), so the partner of region dim i < HD/4 is i + HD/4, which lives in
// n-tile nt + HD/32 of the same thread.
template <int HD, int NT0>
FL_DEV void inverse_rope(float (&acc)[HD / 8][4], int r, int pos, const float2* __restrict__ tab, int lane) {
  constexpr int HALF = HD / 4;
  constexpr int NTP = HALF / 8;
  const float2* tr = tab + (int64_t)pos * HALF;
#pragma unroll
  for (int nt = 0; nt < NTP; ++nt) {
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      const int i = nt * 8 + 2 * (lane & 3) + e;
      const float2 cs = __ldg(tr + i);
      const float x1 = acc[NT0 + nt][2 * r + e], x2 = acc[NT0 + nt + NTP][2 * r + e];
      acc[NT0 + nt][2 * r + e] = x1 * cs.x + x2 * cs.y;
      acc[NT0 + nt + NTP][2 * r + e] = x2 * cs.x - x1 * cs.y;
    }
  }
}

// Both rotary regions of a row at segment index i (global token index t): the first by
// the token's position (i without GLM positions), the second by its block position.
template <int HD>
FL_DEV void inverse_rope_2d(float (&acc)[HD / 8][4], int r, int i, int64_t t, const float2* __restrict__ tab,
                            const int32_t* __restrict__ gpos, const int32_t* __restrict__ gpos2, int lane) {
  inverse_rope<HD, 0>(acc, r, gpos ? __ldg(gpos + t) : i, tab, lane);
  if (gpos2) inverse_rope<HD, HD / 16>(acc, r, __ldg(gpos2 + t), tab, lane);
}

// Adds the column sums of a warp's 16 x HD fragment rows (dq-style accumulator layout:
// thread holds rows lane/4 and lane/4 + 8, columns nt*8 + 2*(lane%4) + {0,1}) of all four
// warps of the CTA to out[0..HD): rows already summed into acc[nt][0..1] by the caller,
// reduced over the warp's 8 row groups with shuffles and over the warps through `red`
// (4 * HD floats of shared memory no thread still reads); one atomic per column.
template <int HD>
FL_DEV void cta_colsum_add(float (&acc)[HD / 8][4], float* red, float* out, int warp, int lane, int tid) {
#pragma unroll
  for (int nt = 0; nt < HD / 8; ++nt)
#pragma unroll
    for (int c = 0; c < 2; ++c) {
      float v = acc[nt][c];
      v += __shfl_xor_sync(0xffffffffu, v, 4);
      v += __shfl_xor_sync(0xffffffffu, v, 8);
      v += __shfl_xor_sync(0xffffffffu, v, 16);
      if (lane < 4) red[warp * HD + nt * 8 + 2 * lane + c] = v;
    }
  __syncthreads();
  if (tid < HD) atomicAdd(out + tid, red[tid] + red[HD + tid] + red[2 * HD + tid] + red[3 * HD + tid]);
  __syncthreads();
}

// ---------------------------------------------------------------------------- dQ
template <int HD>
__global__ void __launch_bounds__(128) attn_bwd_dq_kernel(int T, int H, const bf16* __restrict__ qkv,
                                                          const bf16* __restrict__ dO,
                                                          const float* __restrict__ lse,
                                                          const float* __restrict__ delta,
                                                          const int32_t* __restrict__ cu,
                                                          const uint32_t* __restrict__ tiles,
                                                          const float2* __restrict__ rope_tab, int rotary,
                                                          float scale, bf16* __restrict__ dqkv,
                                                          const bf16* __restrict__ pk, const bf16* __restrict__ pv,
                                                          int Lp, const int32_t* __restrict__ ctxs,
                                                          const int32_t* __restrict__ gpos,
                                                          const int32_t* __restrict__ gpos2,
                                                          float* __restrict__ dbias) {
  extern __shared__ __align__(128) uint8_t smem[];
  bf16* sQ = reinterpret_cast<bf16*>(smem);
  bf16* sdO = sQ + AT<HD>::TILE_ELEMS;
  bf16* sK = sdO + AT<HD>::TILE_ELEMS;  // one tile
  bf16* sV = sK + AT<HD>::TILE_ELEMS;   // one tile
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  int s, idx;
  decode_tile(tiles[blockIdx.x], s, idx);
  const int h = blockIdx.y;
  const int seg0 = cu[s], L = cu[s + 1] - seg0;
  const int q0 = idx * BT;
  const int64_t ld = 3 * (int64_t)H;
  const bf16* gK = qkv + (int64_t)seg0 * ld + H + h * HD;
  const bf16* gV = qkv + (int64_t)seg0 * ld + 2 * H + h * HD;
  const int npt = (Lp + BT - 1) / BT;
  const int clast = (ctxs ? min(max(ctxs[s], 0), L) : 0) - 1;
  const int n_kv = npt + max(idx, clast >= 0 ? clast / BT : 0) + 1;
  const int qlim0 = max(q0, clast);
  auto load_kv = [&](int t) {
    if (t < npt) {
      const int k0 = t * BT;
      load_tile<HD>(sK, pk + (int64_t)k0 * H + h * HD, H, min(BT, Lp - k0), tid);
      load_tile<HD>(sV, pv + (int64_t)k0 * H + h * HD, H, min(BT, Lp - k0), tid);
    } else {
      const int k0 = (t - npt) * BT;
      load_tile<HD>(sK, gK + (int64_t)k0 * ld, ld, min(BT, L - k0), tid);
      load_tile<HD>(sV, gV + (int64_t)k0 * ld, ld, min(BT, L - k0), tid);
    }
  };
  load_tile<HD>(sQ, qkv + (int64_t)(seg0 + q0) * ld + h * HD, ld, min(BT, L - q0), tid);
  load_tile<HD>(sdO, dO + (int64_t)(seg0 + q0) * H + h * HD, H, min(BT, L - q0), tid);
  load_kv(0);
  cp_async_commit();

  const float scale_log2 = scale * LOG2E;
  float lse2[2], dl[2];
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const int q = q0 + warp * 16 + (lane >> 2) + 8 * r;
    lse2[r] = q < L ? lse[(int64_t)h * T + seg0 + q] * LOG2E : 0.f;
    dl[r] = q < L ? delta[(int64_t)h * T + seg0 + q] : 0.f;
  }
  float dq[HD / 8][4];
#pragma unroll
  for (int i = 0; i < HD / 8; ++i) dq[i][0] = dq[i][1] = dq[i][2] = dq[i][3] = 0.f;

  for (int j = 0; j < n_kv; ++j) {
    cp_async_wait<0>();
    __syncthreads();
    const bf16* K = sK;
    const bf16* V = sV;
    float sc[8][4], dp[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
      for (int e = 0; e < 4; ++e) sc[i][e] = dp[i][e] = 0.f;
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
      uint32_t aq[4], ao[4];
      ld_a<HD>(sQ, warp * 16, kk * 16, lane, aq);
      ld_a<HD>(sdO, warp * 16, kk * 16, lane, ao);
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        uint32_t b[4];
        ld_b_rows<HD>(K, np * 16, kk * 16, lane, b);
        mma_bf16_16816(sc[2 * np], aq, b[0], b[1]);
        mma_bf16_16816(sc[2 * np + 1], aq, b[2], b[3]);
        ld_b_rows<HD>(V, np * 16, kk * 16, lane, b);
        mma_bf16_16816(dp[2 * np], ao, b[0], b[1]);
        mma_bf16_16816(dp[2 * np + 1], ao, b[2], b[3]);
      }
    }
    const int kb = (j - npt) * BT;
    const bool need_mask = j >= npt && kb + BT - 1 > qlim0;
    const int pvalid = j < npt ? min(BT, Lp - j * BT) : BT;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int r = e >> 1;
        float p = exp2f(sc[nt][e] * scale_log2 - lse2[r]);
        const int kl = nt * 8 + 2 * (lane & 3) + (e & 1);
        if (need_mask) {
          const int ql = warp * 16 + (lane >> 2) + (r << 3);
          if (kb + kl > max(q0 + ql, clast)) p = 0.f;
        }
        if (kl >= pvalid) p = 0.f;
        sc[nt][e] = p * (dp[nt][e] - dl[r]);  // dS
      }
    }
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      uint32_t a[4];
      a[0] = pack_bf16x2(sc[2 * kk][0], sc[2 * kk][1]);
      a[1] = pack_bf16x2(sc[2 * kk][2], sc[2 * kk][3]);
      a[2] = pack_bf16x2(sc[2 * kk + 1][0], sc[2 * kk + 1][1]);
      a[3] = pack_bf16x2(sc[2 * kk + 1][2], sc[2 * kk + 1][3]);
#pragma unroll
      for (int np = 0; np < HD / 16; ++np) {
        uint32_t b[4];
        ld_b_cols<HD>(K, kk * 16, np * 16, lane, b);
        mma_bf16_16816(dq[2 * np], a, b[0], b[1]);
        mma_bf16_16816(dq[2 * np + 1], a, b[2], b[3]);
      }
    }
    __syncthreads();
    if (j + 1 < n_kv) {  // every warp is done with the tile: load the next one into it
      load_kv(j + 1);
      cp_async_commit();
    }
  }

#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const int q = q0 + warp * 16 + (lane >> 2) + 8 * r;
#pragma unroll
    for (int i = 0; i < HD / 8; ++i) {
      dq[i][2 * r] *= scale;
      dq[i][2 * r + 1] *= scale;
    }
    if (q < L) {
      if (rope_tab) inverse_rope_2d<HD>(dq, r, q, seg0 + q, rope_tab, gpos, gpos2, lane);
      bf16* row = dqkv + (int64_t)(seg0 + q) * ld + h * HD + 2 * (lane & 3);
#pragma unroll
      for (int nt = 0; nt < HD / 8; ++nt)
        *reinterpret_cast<uint32_t*>(row + nt * 8) = pack_bf16x2(dq[nt][2 * r], dq[nt][2 * r + 1]);
    }
  }
  if (dbias) {  // bias gradient of the q columns: sum of the valid rows' (unrotated) dq
    const int qa = q0 + warp * 16 + (lane >> 2);
    const bool va = qa < L, vb = qa + 8 < L;
#pragma unroll
    for (int nt = 0; nt < HD / 8; ++nt) {
      dq[nt][0] = (va ? dq[nt][0] : 0.f) + (vb ? dq[nt][2] : 0.f);
      dq[nt][1] = (va ? dq[nt][1] : 0.f) + (vb ? dq[nt][3] : 0.f);
    }
    cta_colsum_add<HD>(dq, reinterpret_cast<float*>(smem), dbias + h * HD, warp, lane, tid);
  }
}

// ---------------------------------------------------------------------------- dK, dV
// One CTA per (64-key tile, head); a warp owns 16 keys.  The CTA walks the query tiles that
// see its keys: the later tiles of its own segment (causal), or, for a prefix key tile
// (PREFIX), a slice of every query tile of the call (the prefix is shared by all segments;
// the slices' partial sums meet in fp32 with atomics).
struct QTile {
  int row0;   // global token index of the tile's first query
  int valid;  // queries of the tile inside their segment
  int qpos0;  // position of the first query inside its segment
};

template <int HD, bool PREFIX>
__global__ void __launch_bounds__(128) attn_bwd_dkv_kernel(int T, int H, const bf16* __restrict__ qkv,
                                                           const bf16* __restrict__ dO,
                                                           const float* __restrict__ lse,
                                                           const float* __restrict__ delta,
                                                           const int32_t* __restrict__ cu,
                                                           const uint32_t* __restrict__ tiles, int n_tiles,
                                                           const float2* __restrict__ rope_tab, int rotary,
                                                           float scale, bf16* __restrict__ dqkv,
                                                           const bf16* __restrict__ pk, const bf16* __restrict__ pv,
                                                           int Lp, int nsplit, float* __restrict__ dpk,
                                                           float* __restrict__ dpv, const int32_t* __restrict__ ctxs,
                                                           const int32_t* __restrict__ gpos,
                                                           const int32_t* __restrict__ gpos2,
                                                           float* __restrict__ dbias) {
  extern __shared__ __align__(128) uint8_t smem[];
  bf16* sK = reinterpret_cast<bf16*>(smem);
  bf16* sV = sK + AT<HD>::TILE_ELEMS;
  bf16* sQ = sV + AT<HD>::TILE_ELEMS;       // [2]
  bf16* sdO = sQ + 2 * AT<HD>::TILE_ELEMS;  // [2]
  float* sL = reinterpret_cast<float*>(sdO + 2 * AT<HD>::TILE_ELEMS);  // [2][64] lse * log2e
  float* sD = sL + 2 * BT;                                               // [2][64] delta
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int h = blockIdx.y;
  const int64_t ld = 3 * (int64_t)H;
  // this CTA's keys and its range of query tiles
  int seg0 = 0, L = 0, k0, kvalid, it0, it_end, clast = -1;
  if constexpr (PREFIX) {
    const int pt = blockIdx.x / nsplit, z = blockIdx.x % nsplit;
    k0 = pt * BT;
    kvalid = min(BT, Lp - k0);
    const int per = (n_tiles + nsplit - 1) / nsplit;
    it0 = z * per;
    it_end = min(n_tiles, it0 + per);
    load_tile<HD>(sK, pk + (int64_t)k0 * H + h * HD, H, kvalid, tid);
    load_tile<HD>(sV, pv + (int64_t)k0 * H + h * HD, H, kvalid, tid);
  } else {
    int s, idx;
    decode_tile(tiles[blockIdx.x], s, idx);
    seg0 = cu[s];
    L = cu[s + 1] - seg0;
    const int nq = (L + BT - 1) / BT;
    const int kt = nq - 1 - idx;  // key tile: most work first
    k0 = kt * BT;
    kvalid = min(BT, L - k0);
    clast = (ctxs ? min(max(ctxs[s], 0), L) : 0) - 1;
    it0 = k0 <= clast ? 0 : kt;  // a tile holding context keys is seen by every query
    it_end = nq;
    load_tile<HD>(sK, qkv + (int64_t)(seg0 + k0) * ld + H + h * HD, ld, kvalid, tid);
    load_tile<HD>(sV, qkv + (int64_t)(seg0 + k0) * ld + 2 * H + h * HD, ld, kvalid, tid);
  }
  auto qtile = [&](int it) {
    QTile q;
    if constexpr (PREFIX) {
      int s, idx;
      decode_tile(tiles[it], s, idx);
      const int sb = cu[s];
      q.qpos0 = idx * BT;
      q.row0 = sb + q.qpos0;
      q.valid = min(BT, cu[s + 1] - sb - q.qpos0);
    } else {
      q.qpos0 = it * BT;
      q.row0 = seg0 + q.qpos0;
      q.valid = min(BT, L - q.qpos0);
    }
    return q;
  };
  auto load_q = [&](const QTile& q, int buf) {
    load_tile<HD>(sQ + buf * AT<HD>::TILE_ELEMS, qkv + (int64_t)q.row0 * ld + h * HD, ld, q.valid, tid);
    load_tile<HD>(sdO + buf * AT<HD>::TILE_ELEMS, dO + (int64_t)q.row0 * H + h * HD, H, q.valid, tid);
    if (tid < BT) {
      sL[buf * BT + tid] = tid < q.valid ? lse[(int64_t)h * T + q.row0 + tid] * LOG2E : 0.f;
      sD[buf * BT + tid] = tid < q.valid ? delta[(int64_t)h * T + q.row0 + tid] : 0.f;
    }
  };
  QTile cur = qtile(it0 < it_end ? it0 : 0);
  if (it0 < it_end) load_q(cur, 0);
  cp_async_commit();
  const float scale_log2 = scale * LOG2E;
  float dk[HD / 8][4], dv[HD / 8][4];
#pragma unroll
  for (int i = 0; i < HD / 8; ++i)
#pragma unroll
    for (int e = 0; e < 4; ++e) dk[i][e] = dv[i][e] = 0.f;

  for (int it = it0; it < it_end; ++it) {
    const int buf = (it - it0) & 1;
    QTile nxt = cur;
    if (it + 1 < it_end) {
      nxt = qtile(it + 1);
      load_q(nxt, buf ^ 1);
      cp_async_commit();
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    const bf16* Q = sQ + buf * AT<HD>::TILE_ELEMS;
    const bf16* D = sdO + buf * AT<HD>::TILE_ELEMS;
    const float* Lq = sL + buf * BT;
    const float* Dq = sD + buf * BT;
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      const int qb = half * 32;  // query columns [qb, qb + 32) of the tile
      float st[4][4], dpt[4][4];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int e = 0; e < 4; ++e) st[i][e] = dpt[i][e] = 0.f;
#pragma unroll
      for (int kk = 0; kk < HD / 16; ++kk) {
        uint32_t ak[4], av[4];
        ld_a<HD>(sK, warp * 16, kk * 16, lane, ak);
        ld_a<HD>(sV, warp * 16, kk * 16, lane, av);
#pragma unroll
        for (int np = 0; np < 2; ++np) {
          uint32_t b[4];
          ld_b_rows<HD>(Q, qb + np * 16, kk * 16, lane, b);
          mma_bf16_16816(st[2 * np], ak, b[0], b[1]);
          mma_bf16_16816(st[2 * np + 1], ak, b[2], b[3]);
          ld_b_rows<HD>(D, qb + np * 16, kk * 16, lane, b);
          mma_bf16_16816(dpt[2 * np], av, b[0], b[1]);
          mma_bf16_16816(dpt[2 * np + 1], av, b[2], b[3]);
        }
      }
      // P^T and dS^T; rows = keys (warp*16 + lane/4 + 8r), cols = queries
#pragma unroll
      for (int nt = 0; nt < 4; ++nt) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int kl = warp * 16 + (lane >> 2) + ((e >> 1) << 3);
          const int ql = qb + nt * 8 + 2 * (lane & 3) + (e & 1);
          bool ok = ql < cur.valid && kl < kvalid;
          if constexpr (!PREFIX) ok = ok && k0 + kl <= max(cur.qpos0 + ql, clast);  // causal / GLM context
          float p = 0.f;
          if (ok) p = exp2f(st[nt][e] * scale_log2 - Lq[ql]);
          st[nt][e] = p;
          dpt[nt][e] = p * (dpt[nt][e] - Dq[ql]);
        }
      }
#pragma unroll
      for (int kk = 0; kk < 2; ++kk) {
        uint32_t ap[4], as[4];
        ap[0] = pack_bf16x2(st[2 * kk][0], st[2 * kk][1]);
        ap[1] = pack_bf16x2(st[2 * kk][2], st[2 * kk][3]);
        ap[2] = pack_bf16x2(st[2 * kk + 1][0], st[2 * kk + 1][1]);
        ap[3] = pack_bf16x2(st[2 * kk + 1][2], st[2 * kk + 1][3]);
        as[0] = pack_bf16x2(dpt[2 * kk][0], dpt[2 * kk][1]);
        as[1] = pack_bf16x2(dpt[2 * kk][2], dpt[2 * kk][3]);
        as[2] = pack_bf16x2(dpt[2 * kk + 1][0], dpt[2 * kk + 1][1]);
        as[3] = pack_bf16x2(dpt[2 * kk + 1][2], dpt[2 * kk + 1][3]);
#pragma unroll
        for (int np = 0; np < HD / 16; ++np) {
          uint32_t b[4];
          ld_b_cols<HD>(D, qb + kk * 16, np * 16, lane, b);
          mma_bf16_16816(dv[2 * np], ap, b[0], b[1]);
          mma_bf16_16816(dv[2 * np + 1], ap, b[2], b[3]);
          ld_b_cols<HD>(Q, qb + kk * 16, np * 16, lane, b);
          mma_bf16_16816(dk[2 * np], as, b[0], b[1]);
          mma_bf16_16816(dk[2 * np + 1], as, b[2], b[3]);
        }
      }
    }
    __syncthreads();
    cur = nxt;
  }

#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const int kl = warp * 16 + (lane >> 2) + 8 * r;
#pragma unroll
    for (int i = 0; i < HD / 8; ++i) {
      dk[i][2 * r] *= scale;
      dk[i][2 * r + 1] *= scale;
    }
    if (kl < kvalid) {
      if constexpr (PREFIX) {  // the prefix keys enter the scores unrotated
        float* rk = dpk + (int64_t)(k0 + kl) * H + h * HD + 2 * (lane & 3);
        float* rv = dpv + (int64_t)(k0 + kl) * H + h * HD + 2 * (lane & 3);
#pragma unroll
        for (int nt = 0; nt < HD / 8; ++nt) {
          atomicAdd(rk + nt * 8, dk[nt][2 * r]);
          atomicAdd(rk + nt * 8 + 1, dk[nt][2 * r + 1]);
          atomicAdd(rv + nt * 8, dv[nt][2 * r]);
          atomicAdd(rv + nt * 8 + 1, dv[nt][2 * r + 1]);
        }
      } else {
        const int kpos = k0 + kl;
        if (rope_tab) inverse_rope_2d<HD>(dk, r, kpos, seg0 + kpos, rope_tab, gpos, gpos2, lane);
        bf16* rk = dqkv + (int64_t)(seg0 + kpos) * ld + H + h * HD + 2 * (lane & 3);
        bf16* rv = dqkv + (int64_t)(seg0 + kpos) * ld + 2 * H + h * HD + 2 * (lane & 3);
#pragma unroll
        for (int nt = 0; nt < HD / 8; ++nt) {
          *reinterpret_cast<uint32_t*>(rk + nt * 8) = pack_bf16x2(dk[nt][2 * r], dk[nt][2 * r + 1]);
          *reinterpret_cast<uint32_t*>(rv + nt * 8) = pack_bf16x2(dv[nt][2 * r], dv[nt][2 * r + 1]);
        }
      }
    }
  }
  if constexpr (!PREFIX) {
    if (dbias) {  // bias gradients of the k and v columns: sums of the valid keys' dk, dv
      const int ka = warp * 16 + (lane >> 2);
      const bool va = ka < kvalid, vb = ka + 8 < kvalid;
#pragma unroll
      for (int nt = 0; nt < HD / 8; ++nt) {
        dk[nt][0] = (va ? dk[nt][0] : 0.f) + (vb ? dk[nt][2] : 0.f);
        dk[nt][1] = (va ? dk[nt][1] : 0.f) + (vb ? dk[nt][3] : 0.f);
        dv[nt][0] = (va ? dv[nt][0] : 0.f) + (vb ? dv[nt][2] : 0.f);
        dv[nt][1] = (va ? dv[nt][1] : 0.f) + (vb ? dv[nt][3] : 0.f);
      }
      cta_colsum_add<HD>(dk, reinterpret_cast<float*>(smem), dbias + H + h * HD, warp, lane, tid);
      cta_colsum_add<HD>(dv, reinterpret_cast<float*>(smem), dbias + 2 * H + h * HD, warp, lane, tid);
    }
  }
}

template <int HD>
constexpr int fwd_smem() { return 3 * AT<HD>::TILE_BYTES; }
template <int HD>
constexpr int dq_smem() { return 4 * AT<HD>::TILE_BYTES; }
template <int HD>
constexpr int dkv_smem() { return 6 * AT<HD>::TILE_BYTES + 4 * BT * 4; }

template <int HD>
int set_attrs() {
  static bool done = false;
  if (!done) {
    FL_CUDA_TRY(cudaFuncSetAttribute(attn_fwd_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, fwd_smem<HD>()));
    FL_CUDA_TRY(cudaFuncSetAttribute(attn_bwd_dq_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, dq_smem<HD>()));
    FL_CUDA_TRY(cudaFuncSetAttribute(attn_bwd_dkv_kernel<HD, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     dkv_smem<HD>()));
    FL_CUDA_TRY(cudaFuncSetAttribute(attn_bwd_dkv_kernel<HD, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     dkv_smem<HD>()));
    done = true;
  }
  return FL_OK;
}

int sms() {
  static int n = 0;
  if (!n) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 148;
  }
  return n;
}

template <int HD>
int launch_fwd(int T, int nh, const void* qkv, const int32_t* cu, const uint32_t* tiles, int n_tiles, void* o,
               float* lse, const AttnPrefix& pre, const AttnGlm& glm, cudaStream_t st) {
  if (int rc = set_attrs<HD>()) return rc;
  const int H = nh * HD;
  const float scale_log2 = (1.f / sqrtf((float)HD)) * LOG2E;
  attn_fwd_kernel<HD><<<dim3(n_tiles, nh), 128, fwd_smem<HD>(), st>>>(
      T, H, (const bf16*)qkv, cu, tiles, (bf16*)o, lse, scale_log2, (const bf16*)pre.k, (const bf16*)pre.v, pre.len,
      glm.ctx);
  FL_CUDA_TRY(cudaGetLastError());
  return FL_OK;
}

template <int HD>
int launch_bwd(int T, int nh, const void* qkv, const void* o, const float* lse, const void* dout, const int32_t* cu,
               const uint32_t* tiles, int n_tiles, int n_tiles128, float* delta, const float* rope_tab, void* dqkv,
               const AttnPrefix& pre, const AttnGlm& glm, float* dbias, int* status, cudaStream_t st) {
  if (int rc = set_attrs<HD>()) return rc;
  const int H = nh * HD;
  const float scale = 1.f / sqrtf((float)HD);
  const int64_t pairs = (int64_t)T * nh;
  attn_delta_kernel<HD><<<(unsigned)((pairs * (HD / 8) + 255) / 256), 256, 0, st>>>(T, H, nh, (const bf16*)o,
                                                                                    (const bf16*)dout, delta);
  FL_CUDA_TRY(cudaGetLastError());
  const float2* tab = reinterpret_cast<const float2*>(rope_tab);
  const bf16* pk = (const bf16*)pre.k;
  const bf16* pv = (const bf16*)pre.v;
  if (HD == 128) {  // tcgen05 (attention_bwd_tc.cu)
    if (int rc = fl_launch_attn_bwd_dq_tc(T, nh, qkv, dout, lse, delta, cu, tiles + n_tiles, n_tiles128, rope_tab,
                                          dqkv, pre, glm, dbias, status, st))
      return rc;
  } else {
    attn_bwd_dq_kernel<HD><<<dim3(n_tiles, nh), 128, dq_smem<HD>(), st>>>(
        T, H, (const bf16*)qkv, (const bf16*)dout, lse, delta, cu, tiles, tab, HD / 2, scale, (bf16*)dqkv, pk, pv,
        pre.len, glm.ctx, glm.pos, glm.pos2, dbias);
    FL_CUDA_TRY(cudaGetLastError());
  }
  if (HD == 128) {  // the segment's own keys on tcgen05 (attention_bwd_tc.cu)
    if (int rc = fl_launch_attn_bwd_dkv_tc(T, nh, qkv, dout, lse, delta, cu, tiles + n_tiles, n_tiles128, rope_tab,
                                           dqkv, glm, dbias, status, st))
      return rc;
  } else {
    attn_bwd_dkv_kernel<HD, false><<<dim3(n_tiles, nh), 128, dkv_smem<HD>(), st>>>(
        T, H, (const bf16*)qkv, (const bf16*)dout, lse, delta, cu, tiles, n_tiles, tab, HD / 2, scale, (bf16*)dqkv,
        nullptr, nullptr, 0, 1, nullptr, nullptr, glm.ctx, glm.pos, glm.pos2, dbias);
    FL_CUDA_TRY(cudaGetLastError());
  }
  if (pre.len > 0) {
    // prefix key tiles x slices of all query tiles, about two CTAs per SM in total
    const int npt = (pre.len + BT - 1) / BT;
    int nsplit = (2 * sms() + npt * nh - 1) / (npt * nh);
    if (nsplit > n_tiles) nsplit = n_tiles;
    if (nsplit < 1) nsplit = 1;
    attn_bwd_dkv_kernel<HD, true><<<dim3(npt * nsplit, nh), 128, dkv_smem<HD>(), st>>>(
        T, H, (const bf16*)qkv, (const bf16*)dout, lse, delta, cu, tiles, n_tiles, tab, HD / 2, scale, nullptr, pk,
        pv, pre.len, nsplit, pre.dk, pre.dv, nullptr, nullptr, nullptr, nullptr);
    FL_CUDA_TRY(cudaGetLastError());
  }
  return FL_OK;
}

}  // namespace

int fl_build_tiles(const int32_t* cu, int S, uint32_t* tiles, int max_tiles, int rows) {
  int maxq = 0;
  for (int s = 0; s < S; ++s) {
    const int nq = (cu[s + 1] - cu[s] + rows - 1) / rows;
    maxq = nq > maxq ? nq : maxq;
  }
  int n = 0;
  for (int i = maxq - 1; i >= 0; --i)
    for (int s = 0; s < S; ++s) {
      const int nq = (cu[s + 1] - cu[s] + rows - 1) / rows;
      if (i < nq) {
        if (n >= max_tiles) return -1;
        tiles[n++] = (uint32_t(s) << 16) | uint32_t(i);
      }
    }
  return n;
}

int fl_launch_attn_fwd(int T, int nh, int hd, const void* qkv, const int32_t* cu, const uint32_t* tiles, int n_tiles,
                       int n_tiles128,
                       void* o, float* lse, const AttnPrefix& pre, const AttnGlm& glm, cudaStream_t st, int* status) {
  if (n_tiles <= 0) return FL_OK;
  if (hd == 128) return fl_launch_attn_fwd_tc(T, nh, qkv, cu, tiles + n_tiles, n_tiles128, o, lse, pre, glm, status, st);
  if (hd == 64) return launch_fwd<64>(T, nh, qkv, cu, tiles, n_tiles, o, lse, pre, glm, st);
  return fl_internal_error(FL_ERR_UNSUPPORTED, "attention: head_dim %d", hd);
}

int fl_launch_attn_bwd(int T, int nh, int hd, const void* qkv, const void* o, const float* lse, const void* dout,
                       const int32_t* cu, const uint32_t* tiles, int n_tiles, int n_tiles128, float* delta,
                       const float* rope_tab, void* dqkv, const AttnPrefix& pre, const AttnGlm& glm, cudaStream_t st,
                       float* dbias, int* status) {
  if (n_tiles <= 0) return FL_OK;
  if (hd == 128)
    return launch_bwd<128>(T, nh, qkv, o, lse, dout, cu, tiles, n_tiles, n_tiles128, delta, rope_tab, dqkv, pre, glm,
                           dbias, status, st);
  if (hd == 64)
    return launch_bwd<64>(T, nh, qkv, o, lse, dout, cu, tiles, n_tiles, n_tiles128, delta, rope_tab, dqkv, pre, glm,
                          dbias, status, st);
  return fl_internal_error(FL_ERR_UNSUPPORTED, "attention: head_dim %d", hd);
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
  if (prefix_len < 0 || prefix_len > 128 ||
      (prefix_len > 0 && (!prefix_k || !prefix_v || !dprefix_k || !dprefix_v)))
    return fl_internal_error(FL_ERR_INVALID_ARG, "attention bwd: prefix (length 0..128, gradients required)");
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
