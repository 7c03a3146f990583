// Attention forward on the 5th-generation tensor cores (head_dim 128): the same
// computation as attn_fwd_kernel in attention.cu (App. A: softmax(Q K'^T / sqrt(d_h)) V',
// K' / V' = optional P-tuning prefix then the segment's own keys, causal within the
// segment or with a bidirectional GLM context, §3.3 segments never mixed), with the two
// tile contractions on tcgen05 and their accumulators in TMEM.
//
// One CTA (4 warps) per (128-query tile, head).  Thread i owns query row i, which is TMEM
// lane i.  Per 128-key tile j:
//   TMA: K_j, V_j (128 rows x 128 dims, two 128-byte-swizzled boxes each; Q once);
//   S = Q K_j^T   -> TMEM columns [0, 128)       (8 x tcgen05.mma 128x128x16);
//   softmax: two passes over the thread's S row (masked max, then exp2 and the row sum),
//            P (bf16) written into K_j's buffer in the swizzled K-major operand layout,
//            the O row in TMEM rescaled when the running max moved;
//   O += P V_j    -> TMEM columns [128, 256)     (V_j as an MN-major operand).
// Shared memory 96 KB (Q, K/P, V) and 256 TMEM columns: two CTAs per SM overlap each
// other's copies and softmax.  Every mbarrier wait is bounded (2 s): on expiry the CTA
// records a status code and leaves its remaining work undone.
#include <cuda.h>
#include <cuda_runtime.h>

#include <cmath>

#include "../../include/flglm_kernels.h"
#include "common.cuh"
#include "gemm_tc.cuh"
#include "kernels.cuh"
#include "ptx.cuh"

namespace {

typedef __nv_bfloat16 bf16;
constexpr int TBQ = 128;             // queries per tile (UMMA M)
constexpr int TBK = 128;             // keys per tile (UMMA N of S, K of P V)
constexpr int HDT = 128;             // head dim
constexpr int BOX = 64 * 128 * 2;    // one 64-column x 128-row bf16 box: 16 KB
constexpr int TILE = 2 * BOX;        // a 128 x 128 bf16 tile
constexpr int SMEM = 3 * TILE + 1024 /*barriers, holder*/ + 1024 /*alignment*/;
constexpr float LOG2E_T = 1.4426950408889634f;
constexpr float LN2_T = 0.6931471805599453f;

// K-major operand (rows x 128 columns in two swizzled boxes): descriptor of k-step kk.
FL_DEV uint64_t desc_kmajor(uint32_t base, int kk) {
  return smem_desc_sw128(base + (kk >> 2) * BOX + (kk & 3) * 32, 16, 1024);
}
// MN-major operand (K = the tile's 128 rows, N = its 128 columns): descriptor of k-step kk.
FL_DEV uint64_t desc_mnmajor(uint32_t base, int kk) { return smem_desc_sw128(base + kk * 2048, BOX, 1024); }

__global__ void __launch_bounds__(128) attn_fwd_tc_kernel(
    const __grid_constant__ CUtensorMap tm_qkv, const __grid_constant__ CUtensorMap tm_pk,
    const __grid_constant__ CUtensorMap tm_pv, int T, int H, const int32_t* __restrict__ cu,
    const uint32_t* __restrict__ tiles, bf16* __restrict__ O, float* __restrict__ lse, float scale_log2, int Lp,
    const int32_t* __restrict__ ctxs, int* status) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;
  uint8_t* sK = smem + TILE;  // K_j, then P
  uint8_t* sV = smem + 2 * TILE;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + 3 * TILE);
  uint64_t* bar_load = bars;
  uint64_t* bar_s = bars + 1;
  uint64_t* bar_pv = bars + 2;
  uint32_t* holder = reinterpret_cast<uint32_t*>(bars + 4);

  // the 128-row tile list: (segment, query tile)
  const int s = int(tiles[blockIdx.x] >> 16), idx = int(tiles[blockIdx.x] & 0xFFFFu);
  const int h = blockIdx.y;
  const int tid = threadIdx.x, warp = tid >> 5;
  const int seg0 = cu[s], L = cu[s + 1] - seg0;
  const int q0 = idx * TBQ;
  const int npt = Lp > 0 ? 1 : 0;  // at most one prefix tile (Lp <= 128)
  const int clast = (ctxs ? min(max(ctxs[s], 0), L) : 0) - 1;
  const int n_kv = npt + max(idx, clast >= 0 ? clast / TBK : 0) + 1;

  if (tid == 0) {
    mbar_init(bar_load, 1);
    mbar_init(bar_s, 1);
    mbar_init(bar_pv, 1);
    fence_mbar_init();
    tma_prefetch_desc(&tm_qkv);
  }
  if (warp == 0) {
    tmem_alloc(holder, 256);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *holder;
  const uint32_t t_lane = tmem + (uint32_t(warp * 32) << 16);  // this warp's TMEM lanes
  const uint32_t t_s = t_lane, t_o = t_lane + 128;

  auto issue_kv = [&](int j) {  // one elected thread
    if (j < npt) {
      tma_load_2d(sK, &tm_pk, bar_load, h * HDT, 0);
      tma_load_2d(sK + BOX, &tm_pk, bar_load, h * HDT + 64, 0);
      tma_load_2d(sV, &tm_pv, bar_load, h * HDT, 0);
      tma_load_2d(sV + BOX, &tm_pv, bar_load, h * HDT + 64, 0);
    } else {
      const int row = seg0 + (j - npt) * TBK;
      tma_load_2d(sK, &tm_qkv, bar_load, H + h * HDT, row);
      tma_load_2d(sK + BOX, &tm_qkv, bar_load, H + h * HDT + 64, row);
      tma_load_2d(sV, &tm_qkv, bar_load, 2 * H + h * HDT, row);
      tma_load_2d(sV + BOX, &tm_qkv, bar_load, 2 * H + h * HDT + 64, row);
    }
  };
  if (tid == 0) {
    mbar_arrive_expect_tx(bar_load, 3 * TILE);
    tma_load_2d(sQ, &tm_qkv, bar_load, h * HDT, seg0 + q0);
    tma_load_2d(sQ + BOX, &tm_qkv, bar_load, h * HDT + 64, seg0 + q0);
    issue_kv(0);
  }

  constexpr uint32_t IDESC_S = umma_idesc_bf16(TBQ, TBK, false, false);
  constexpr uint32_t IDESC_PV = umma_idesc_bf16(TBQ, HDT, false, true);
  const int q = q0 + tid;  // this thread's query row (inside the segment)
  float m_run = -INFINITY, l_run = 0.f;
  bool ok = true;
  uint32_t ph = 0;
  for (int j = 0; j < n_kv && ok; ++j, ph ^= 1) {
    // every wait's outcome is agreed on by the whole CTA, so that all threads leave together
    if (!__syncthreads_and(mbar_wait(bar_load, ph))) {
      if (tid == 0) report_status(status, FL_DEV_TIMEOUT_FULL);
      ok = false;
      break;
    }
    // ---- S = Q K_j^T
    if (tid == 0) {
      tc_fence_after();
      const uint32_t aq = smem_u32(sQ), bk = smem_u32(sK);
#pragma unroll
      for (int kk = 0; kk < HDT / 16; ++kk) umma_bf16(tmem, desc_kmajor(aq, kk), desc_kmajor(bk, kk), IDESC_S, kk > 0);
      umma_commit(bar_s);
    }
    if (!__syncthreads_and(mbar_wait(bar_s, ph))) {
      if (tid == 0) report_status(status, FL_DEV_TIMEOUT_ACC_FULL);
      ok = false;
      break;
    }
    tc_fence_after();
    // ---- the thread's S row, read once (4 x 32 columns, one wait)
    const bool prefix = j < npt;
    const int kb = prefix ? 0 : (j - npt) * TBK;  // first key of the tile inside its sequence
    const int klim = prefix ? Lp - 1 : min(L - 1, max(q, clast));  // last visible key
    const bool full = kb + TBK - 1 <= klim;      // every key of the tile visible to this row
    uint32_t r[TBK];
    tmem_ld32(t_s, *reinterpret_cast<uint32_t(*)[32]>(r));
    tmem_ld32(t_s + 32, *reinterpret_cast<uint32_t(*)[32]>(r + 32));
    tmem_ld32(t_s + 64, *reinterpret_cast<uint32_t(*)[32]>(r + 64));
    tmem_ld32(t_s + 96, *reinterpret_cast<uint32_t(*)[32]>(r + 96));
    tmem_ld_wait();
    // masked row max; invisible keys become -inf
    float mt = -INFINITY;
#pragma unroll
    for (int e = 0; e < TBK; ++e) {
      float x = __uint_as_float(r[e]) * scale_log2;
      if (!full && kb + e > klim) x = -INFINITY;
      r[e] = __float_as_uint(x);
      mt = fmaxf(mt, x);
    }
    const float m_new = fmaxf(m_run, mt);
    const float mref = m_new == -INFINITY ? 0.f : m_new;
    const float corr = exp2f(m_run - mref);  // 0 on the first tile (m_run = -inf)
    // ---- P = exp2(S - m) into the K buffer: row `tid`, 16-byte chunk c of the 64-key box b
    // at position c ^ (row & 7), the layout of a 128-byte-swizzled TMA box
    float lt = 0.f;
#pragma unroll
    for (int c = 0; c < TBK; c += 8) {
      float p[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        p[e] = exp2f(__uint_as_float(r[c + e]) - mref);
        lt += p[e];
      }
      const int chunk = (c & 63) >> 3;
      *reinterpret_cast<uint4*>(sK + (c >> 6) * BOX + tid * 128 + ((chunk ^ (tid & 7)) << 4)) =
          make_uint4(pack_bf16x2(p[0], p[1]), pack_bf16x2(p[2], p[3]), pack_bf16x2(p[4], p[5]),
                     pack_bf16x2(p[6], p[7]));
    }
    l_run = l_run * corr + lt;
    m_run = m_new;
    // ---- rescale the O rows when a row max moved (not before the first P V); TMEM
    // loads and stores are warp-wide, so the whole warp takes part (factor 1 elsewhere)
    if (j > 0 && __any_sync(0xffffffffu, corr != 1.f)) {
#pragma unroll 1
      for (int c = 0; c < HDT; c += 32) {
        uint32_t r[32];
        tmem_ld32(t_o + c, r);
        tmem_ld_wait();
#pragma unroll
        for (int e = 0; e < 32; ++e) r[e] = __float_as_uint(__uint_as_float(r[e]) * corr);
        tmem_st32(t_o + c, r);
      }
      tmem_st_wait();
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    // ---- O += P V_j
    if (tid == 0) {
      tc_fence_after();
      const uint32_t ap = smem_u32(sK), bv = smem_u32(sV);
#pragma unroll
      for (int kk = 0; kk < TBK / 16; ++kk)
        umma_bf16(tmem + 128, desc_kmajor(ap, kk), desc_mnmajor(bv, kk), IDESC_PV, (j > 0 || kk > 0) ? 1u : 0u);
      umma_commit(bar_pv);
    }
    if (!__syncthreads_and(mbar_wait(bar_pv, ph))) {
      if (tid == 0) report_status(status, FL_DEV_TIMEOUT_ACC_EMPTY);
      ok = false;
      break;
    }
    tc_fence_after();
    // ---- next K / V into the freed buffers
    if (tid == 0 && j + 1 < n_kv) {
      mbar_arrive_expect_tx(bar_load, 2 * TILE);
      issue_kv(j + 1);
    }
  }
  // ---- O / l and the log-sum-exp (every lane reads TMEM; rows past the segment end
  // store nothing)
  if (ok) {
    const bool valid = q < L;
    const float inv = valid ? 1.f / l_run : 0.f;
    bf16* orow = O + (int64_t)(seg0 + (valid ? q : 0)) * H + h * HDT;
#pragma unroll 1
    for (int c = 0; c < HDT; c += 32) {
      uint32_t r[32];
      tmem_ld32(t_o + c, r);
      tmem_ld_wait();
      if (valid) {
#pragma unroll
        for (int u = 0; u < 4; ++u)
          *reinterpret_cast<uint4*>(orow + c + 8 * u) = make_uint4(
              pack_bf16x2(__uint_as_float(r[8 * u]) * inv, __uint_as_float(r[8 * u + 1]) * inv),
              pack_bf16x2(__uint_as_float(r[8 * u + 2]) * inv, __uint_as_float(r[8 * u + 3]) * inv),
              pack_bf16x2(__uint_as_float(r[8 * u + 4]) * inv, __uint_as_float(r[8 * u + 5]) * inv),
              pack_bf16x2(__uint_as_float(r[8 * u + 6]) * inv, __uint_as_float(r[8 * u + 7]) * inv));
      }
    }
    if (valid) lse[(int64_t)h * T + seg0 + q] = (m_run + log2f(l_run)) * LN2_T;
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, 256);
  }
}

}  // namespace

int fl_launch_attn_fwd_tc(int T, int nh, const void* qkv, const int32_t* cu, const uint32_t* tiles, int n_tiles,
                          void* o, float* lse, const AttnPrefix& pre, const AttnGlm& glm, int* status,
                          cudaStream_t st) {
  static bool attr = false;
  if (!attr) {
    FL_CUDA_TRY(cudaFuncSetAttribute(attn_fwd_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM));
    attr = true;
  }
  const int H = nh * HDT;
  CUtensorMap tq, tpk, tpv;
  if (int rc = fl_gemm::make_map(&tq, qkv, (uint64_t)3 * H, (uint64_t)T, 3 * (int64_t)H, 128)) return rc;
  if (pre.len > 0) {
    if (int rc = fl_gemm::make_map(&tpk, pre.k, (uint64_t)H, (uint64_t)pre.len, H, 128)) return rc;
    if (int rc = fl_gemm::make_map(&tpv, pre.v, (uint64_t)H, (uint64_t)pre.len, H, 128)) return rc;
  } else {
    tpk = tq;
    tpv = tq;
  }
  const float scale_log2 = (1.f / sqrtf((float)HDT)) * LOG2E_T;
  attn_fwd_tc_kernel<<<dim3(n_tiles, nh), 128, SMEM, st>>>(tq, tpk, tpv, T, H, cu, tiles, (bf16*)o, lse, scale_log2,
                                                          pre.len, glm.ctx, status);
  FL_CUDA_TRY(cudaGetLastError());
  return FL_OK;
}
