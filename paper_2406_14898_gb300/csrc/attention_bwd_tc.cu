// Attention backward on the 5th-generation tensor cores (head_dim 128): dQ, and dK / dV of
// the segment's own keys, the same computations as attn_bwd_dq_kernel<128> and
// attn_bwd_dkv_kernel<128, false> in attention.cu (the gradient of App. A's
// softmax(Q K^T / sqrt(d_h)) V, causal or with a bidirectional GLM context, with the
// P-tuning prefix keys in dQ; the prefix keys' own gradients stay on the mma.sync kernel).
//
// One CTA (8 warps) per (128-key tile, head).  Warp w reads TMEM lanes 32 (w % 4) .. + 31,
// so thread (w, lane) owns key row r = 32 (w % 4) + lane, and takes query half w / 4 of
// every query tile.  Per 128-query tile i that sees the key tile:
//   TMA: Q_i and dO_i (K and V once), two 128-byte-swizzled 64-column boxes each;
//   S^T  = K Q_i^T  -> TMEM [0, 128)     dP^T = V dO_i^T -> TMEM [128, 256);
//   threads: P^T = exp2(S^T scale log2e - lse_q log2e) where key r is visible to query q,
//            dS^T = P^T (dP^T - delta_q), both bf16 into shared memory as K-major operands
//            (rows = keys, K = queries, the layout of a 128-byte-swizzled TMA box);
//   dV += P^T dO_i  -> TMEM [256, 384)   dK += dS^T Q_i -> TMEM [384, 512)
//            (dO_i and Q_i as MN-major operands).
// Epilogue: dK * scale, the inverse rotary rotation(s), bf16 rows of dqkv, and the k / v
// column sums for the QKV bias gradient.  Shared memory 195 KB and 512 TMEM columns: one
// CTA per SM.  Every mbarrier wait is bounded (2 s): on expiry the CTA records a status
// code and leaves its remaining work undone.
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
constexpr int TB = 128;                 // keys and queries per tile (UMMA M and N)
constexpr int HDT = 128;                // head dim
constexpr int BOX = 64 * 128 * 2;       // one 64-column x 128-row bf16 box: 16 KB
constexpr int TILE = 2 * BOX;           // a 128 x 128 bf16 tile
constexpr int SMEM = 6 * TILE + 2 * TB * 4 + 1024 /*barriers, holder*/ + 1024 /*alignment*/;
constexpr float LOG2E_B = 1.4426950408889634f;

FL_DEV uint64_t desc_k(uint32_t base, int kk) { return smem_desc_sw128(base + (kk >> 2) * BOX + (kk & 3) * 32, 16, 1024); }
FL_DEV uint64_t desc_mn(uint32_t base, int kk) { return smem_desc_sw128(base + kk * 2048, BOX, 1024); }

// Writes 8 values of row r as bf16: 16-byte chunk c of box `b` of a K-major 128 x 128
// operand tile, stored at position c ^ (r & 7) of the row.
FL_DEV void put_chunk8(uint8_t* tile, int b, int r, int c, const float* v) {
  *reinterpret_cast<uint4*>(tile + b * BOX + r * 128 + ((c ^ (r & 7)) << 4)) =
      make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]), pack_bf16x2(v[4], v[5]),
                 pack_bf16x2(v[6], v[7]));
}

// Inverse rotary rotation of one rotary region held by a thread: 64 consecutive dims,
// pairs (i, i + 32), angle (cos, sin) of pair i at tr[i ^ sw] (a row of the rotary table
// staged in shared memory, entries XOR-swizzled by the row).
FL_DEV void inverse_rope_row(float* v, const float2* tr, int sw) {
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    const float2 cs = tr[i ^ sw];
    const float x1 = v[i], x2 = v[i + 32];
    v[i] = x1 * cs.x + x2 * cs.y;
    v[i + 32] = x2 * cs.x - x1 * cs.y;
  }
}

// 2^x by the hardware instruction (PTX ex2.approx.ftz.f32): the probabilities it feeds are
// rounded to bf16 for the tensor cores.
FL_DEV float exp2_hw(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Adds the column sums of a staged 128 x 128 bf16 tile (rows of 256 bytes, 16-byte chunk j
// of row r at j ^ (r & 15)) over its first `rows` rows to out[0..128): thread c < 128 sums
// column c in row order, one atomic per column.
FL_DEV void staged_colsum(const uint8_t* stage, int rows, float* out, int tid) {
  if (tid >= TB) return;
  const int jc = tid >> 3, e = tid & 7;
  float acc = 0.f;
#pragma unroll 8
  for (int row = 0; row < rows; ++row)
    acc += __bfloat162float(*reinterpret_cast<const bf16*>(stage + row * 256 + ((jc ^ (row & 15)) << 4) + 2 * e));
  atomicAdd(out + tid, acc);
}

__global__ void __launch_bounds__(256, 1) attn_bwd_dkv_tc_kernel(
    const __grid_constant__ CUtensorMap tm_qkv, const __grid_constant__ CUtensorMap tm_do, int T, int H,
    const int32_t* __restrict__ cu, const uint32_t* __restrict__ tiles, const float* __restrict__ lse,
    const float* __restrict__ delta, const float2* __restrict__ rope_tab, float scale, float scale_log2,
    bf16* __restrict__ dqkv, const int32_t* __restrict__ ctxs, const int32_t* __restrict__ gpos,
    const int32_t* __restrict__ gpos2, float* __restrict__ dbias, int* status) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sK = smem;
  uint8_t* sV = smem + TILE;
  uint8_t* sQ = smem + 2 * TILE;
  uint8_t* sdO = smem + 3 * TILE;
  uint8_t* sP = smem + 4 * TILE;
  uint8_t* sdS = smem + 5 * TILE;
  float* sL = reinterpret_cast<float*>(smem + 6 * TILE);  // lse * log2e of the query tile
  float* sD = sL + TB;                                    // delta of the query tile
  uint64_t* bars = reinterpret_cast<uint64_t*>(sD + TB);
  uint64_t* bar_load = bars;
  uint64_t* bar_mma1 = bars + 1;
  uint64_t* bar_mma2 = bars + 2;
  uint32_t* holder = reinterpret_cast<uint32_t*>(bars + 4);

  // the 128-row tile list: (segment, tile), tile i standing for key tile nq - 1 - i
  const int s = int(tiles[blockIdx.x] >> 16), idx = int(tiles[blockIdx.x] & 0xFFFFu);
  const int h = blockIdx.y;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int quarter = warp & 3, qh = warp >> 2;
  const int r = quarter * 32 + lane;  // this thread's key row (TMEM lane)
  const int seg0 = cu[s], L = cu[s + 1] - seg0;
  const int nq = (L + TB - 1) / TB;
  const int kt = nq - 1 - idx;  // key tile: most work first
  const int kb = kt * TB;
  const int clast = (ctxs ? min(max(ctxs[s], 0), L) : 0) - 1;
  const int it0 = kb <= clast ? 0 : kt;  // a tile holding context keys is seen by every query
  const int k = kb + r;                  // the key inside its segment
  const bool key_ok = k < L;

  if (tid == 0) {
    mbar_init(bar_load, 1);
    mbar_init(bar_mma1, 1);
    mbar_init(bar_mma2, 1);
    fence_mbar_init();
    tma_prefetch_desc(&tm_qkv);
    tma_prefetch_desc(&tm_do);
  }
  if (warp == 0) {
    tmem_alloc(holder, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *holder;
  const uint32_t t_lane = tmem + (uint32_t(quarter * 32) << 16);

  auto issue_q = [&](int it) {  // one elected thread
    const int row = seg0 + it * TB;
    tma_load_2d(sQ, &tm_qkv, bar_load, h * HDT, row);
    tma_load_2d(sQ + BOX, &tm_qkv, bar_load, h * HDT + 64, row);
    tma_load_2d(sdO, &tm_do, bar_load, h * HDT, row);
    tma_load_2d(sdO + BOX, &tm_do, bar_load, h * HDT + 64, row);
  };
  if (tid == 0) {
    mbar_arrive_expect_tx(bar_load, 4 * TILE);
    tma_load_2d(sK, &tm_qkv, bar_load, H + h * HDT, seg0 + kb);
    tma_load_2d(sK + BOX, &tm_qkv, bar_load, H + h * HDT + 64, seg0 + kb);
    tma_load_2d(sV, &tm_qkv, bar_load, 2 * H + h * HDT, seg0 + kb);
    tma_load_2d(sV + BOX, &tm_qkv, bar_load, 2 * H + h * HDT + 64, seg0 + kb);
    issue_q(it0);
  }

  constexpr uint32_t IDESC_S = umma_idesc_bf16(TB, TB, false, false);
  constexpr uint32_t IDESC_G = umma_idesc_bf16(TB, HDT, false, true);
  bool ok = true;
  uint32_t ph = 0;
  for (int it = it0; it < nq && ok; ++it, ph ^= 1) {
    const int qb = it * TB;
    {  // lse and delta of the query tile (rows past the segment are never visible)
      const int c = tid & (TB - 1), q = qb + c;
      const float* src = tid < TB ? lse : delta;
      const float v = q < L ? __ldg(src + (int64_t)h * T + seg0 + q) : 0.f;
      if (tid < TB) sL[c] = v * LOG2E_B;
      else sD[c] = v;
    }
    // every wait's outcome is agreed on by the whole CTA, so that all threads leave together
    if (!__syncthreads_and(mbar_wait(bar_load, ph))) {
      if (tid == 0) report_status(status, FL_DEV_TIMEOUT_FULL);
      ok = false;
      break;
    }
    // ---- S^T = K Q^T, dP^T = V dO^T
    if (tid == 0) {
      tc_fence_after();
      const uint32_t ak = smem_u32(sK), av = smem_u32(sV), bq = smem_u32(sQ), bo = smem_u32(sdO);
#pragma unroll
      for (int kk = 0; kk < HDT / 16; ++kk) umma_bf16(tmem, desc_k(ak, kk), desc_k(bq, kk), IDESC_S, kk > 0);
#pragma unroll
      for (int kk = 0; kk < HDT / 16; ++kk) umma_bf16(tmem + 128, desc_k(av, kk), desc_k(bo, kk), IDESC_S, kk > 0);
      umma_commit(bar_mma1);
    }
    if (!__syncthreads_and(mbar_wait(bar_mma1, ph))) {
      if (tid == 0) report_status(status, FL_DEV_TIMEOUT_ACC_FULL);
      ok = false;
      break;
    }
    tc_fence_after();
    // ---- P^T and dS^T of key row r for queries qh * 64 .. + 63, in two halves of 32
    {
      const int q0 = qb + qh * 64;
      // key k is visible to queries [qfirst, qlim): causal from k, all of them for a context key
      const int qlim = key_ok ? min(L, q0 + 64) : q0;
      const int qfirst = k <= clast ? q0 : max(q0, k);
#pragma unroll 1
      for (int hf = 0; hf < 2; ++hf) {
        uint32_t sr[32], dr[32];
        tmem_ld32(t_lane + qh * 64 + 32 * hf, sr);
        tmem_ld32(t_lane + 128 + qh * 64 + 32 * hf, dr);
        tmem_ld_wait();
        const float4* L4 = reinterpret_cast<const float4*>(sL + qh * 64 + 32 * hf);
        const float4* D4 = reinterpret_cast<const float4*>(sD + qh * 64 + 32 * hf);
#pragma unroll
        for (int c8 = 0; c8 < 4; ++c8) {
          const float4 la = L4[2 * c8], lb = L4[2 * c8 + 1], da = D4[2 * c8], db = D4[2 * c8 + 1];
          const float lq[8] = {la.x, la.y, la.z, la.w, lb.x, lb.y, lb.z, lb.w};
          const float dq[8] = {da.x, da.y, da.z, da.w, db.x, db.y, db.z, db.w};
          float p[8], ds[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const int c = 8 * c8 + e, q = q0 + 32 * hf + c;
            const bool vis = q >= qfirst && q < qlim;
            const float pv = vis ? exp2_hw(fmaf(__uint_as_float(sr[c]), scale_log2, -lq[e])) : 0.f;
            p[e] = pv;
            ds[e] = pv * (__uint_as_float(dr[c]) - dq[e]);
          }
          put_chunk8(sP, qh, r, 4 * hf + c8, p);
          put_chunk8(sdS, qh, r, 4 * hf + c8, ds);
        }
      }
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    // ---- dV += P^T dO, dK += dS^T Q
    if (tid == 0) {
      tc_fence_after();
      const uint32_t ap = smem_u32(sP), as = smem_u32(sdS), bq = smem_u32(sQ), bo = smem_u32(sdO);
      const bool acc = it > it0;
#pragma unroll
      for (int kk = 0; kk < TB / 16; ++kk)
        umma_bf16(tmem + 256, desc_k(ap, kk), desc_mn(bo, kk), IDESC_G, (acc || kk > 0) ? 1u : 0u);
#pragma unroll
      for (int kk = 0; kk < TB / 16; ++kk)
        umma_bf16(tmem + 384, desc_k(as, kk), desc_mn(bq, kk), IDESC_G, (acc || kk > 0) ? 1u : 0u);
      umma_commit(bar_mma2);
    }
    if (!__syncthreads_and(mbar_wait(bar_mma2, ph))) {
      if (tid == 0) report_status(status, FL_DEV_TIMEOUT_ACC_EMPTY);
      ok = false;
      break;
    }
    tc_fence_after();
    // ---- the next query tile into the freed buffers
    if (tid == 0 && it + 1 < nq) {
      mbar_arrive_expect_tx(bar_load, 2 * TILE);
      issue_q(it + 1);
    }
  }

  // ---- dK (scaled, rotated back) and dV: thread (r, qh) takes dims qh * 64 .. + 63 of key
  // row r from TMEM, stages the bf16 rows in the freed K (dK) and V (dV) buffers (16-byte
  // chunk j of row r at position j ^ (r & 15)), then the CTA writes whole rows with
  // coalesced 16-byte stores; the bias column sums are taken from the staged rows (the
  // values stored).  The freed P / dS buffers (64 KB) hold the rotary table rows of the
  // tile's keys.
  if (ok && it0 < nq) {
    // rotary rows: region 0 (position) and, with GLM block positions, region 1; entry e of
    // row rr at e ^ (rr & 31), loaded with coalesced reads
    float2* rt = reinterpret_cast<float2*>(sP);
    const int nreg = rope_tab ? (gpos2 ? 2 : 1) : 0;
    for (int reg = 0; reg < nreg; ++reg) {  // warp w loads rows w, w + 8, ...: 16 in flight
      const int32_t* gp = reg == 0 ? gpos : gpos2;
      int pos[TB / 8];
#pragma unroll
      for (int j = 0; j < TB / 8; ++j) {
        const int kk = min(kb + warp + 8 * j, L - 1);
        pos[j] = gp ? __ldg(gp + seg0 + kk) : kk;
      }
      float2 cs[TB / 8];
#pragma unroll
      for (int j = 0; j < TB / 8; ++j) cs[j] = __ldg(rope_tab + (int64_t)pos[j] * 32 + lane);
#pragma unroll
      for (int j = 0; j < TB / 8; ++j) {
        const int rr = warp + 8 * j;
        rt[(reg * TB + rr) * 32 + (lane ^ (rr & 31))] = cs[j];
      }
    }
    __syncthreads();
#pragma unroll 1
    for (int part = 0; part < 2; ++part) {  // 0: dK, 1: dV
      uint8_t* stage = part ? sV : sK;
      uint32_t vr[64];
      tmem_ld32(t_lane + (part ? 256 : 384) + qh * 64, *reinterpret_cast<uint32_t(*)[32]>(vr));
      tmem_ld32(t_lane + (part ? 256 : 384) + qh * 64 + 32, *reinterpret_cast<uint32_t(*)[32]>(vr + 32));
      tmem_ld_wait();
      float* v = reinterpret_cast<float*>(vr);
#pragma unroll
      for (int c = 0; c < 64; ++c) v[c] = __uint_as_float(vr[c]) * (part ? 1.f : scale);
      if (part == 0 && qh < nreg && key_ok) inverse_rope_row(v, rt + (qh * TB + r) * 32, r & 31);
#pragma unroll
      for (int c8 = 0; c8 < 8; ++c8) {
        const int jc = qh * 8 + c8;
        *reinterpret_cast<uint4*>(stage + r * 256 + ((jc ^ (r & 15)) << 4)) =
            make_uint4(pack_bf16x2(v[8 * c8], v[8 * c8 + 1]), pack_bf16x2(v[8 * c8 + 2], v[8 * c8 + 3]),
                       pack_bf16x2(v[8 * c8 + 4], v[8 * c8 + 5]), pack_bf16x2(v[8 * c8 + 6], v[8 * c8 + 7]));
      }
      const int col = (part ? 2 * H : H) + blockIdx.y * HDT;
      __syncthreads();  // the tile is staged
      if (dbias) staged_colsum(stage, min(TB, L - kb), dbias + col, tid);
      // 128 rows x 16 chunks: consecutive threads write consecutive chunks of a row
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int idx = tid + 256 * i, row = idx >> 4, jc = idx & 15;
        if (kb + row < L) {
          const uint4 w = *reinterpret_cast<const uint4*>(stage + row * 256 + ((jc ^ (row & 15)) << 4));
          *reinterpret_cast<uint4*>(dqkv + ((int64_t)seg0 + kb + row) * 3 * H + col + jc * 8) = w;
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// dQ: one CTA (8 warps) per (128-query tile, head); thread (w, lane) owns query row
// r = 32 (w % 4) + lane and takes key half w / 4 of every key tile.  Per 128-key tile j
// the queries see (the prefix tile first, then the segment's own keys):
//   TMA: K_j and V_j (Q and dO once);  S = Q K_j^T -> TMEM [0, 128), dP = dO V_j^T ->
//   TMEM [128, 256);  threads: dS = P (dP - delta_q), P = exp2(S scale log2e - lse_q
//   log2e) on the visible keys, bf16 into shared memory as a K-major operand (rows =
//   queries, K = keys);  dQ += dS K_j -> TMEM [256, 384) (K_j as an MN-major operand).
// Epilogue as in the dK / dV kernel: dQ * scale, inverse rotary rotation(s), coalesced bf16
// rows, q column sums for the bias gradient.  Shared memory: five tiles used of the
// kernels' common allocation.
__global__ void __launch_bounds__(256, 1) attn_bwd_dq_tc_kernel(
    const __grid_constant__ CUtensorMap tm_qkv, const __grid_constant__ CUtensorMap tm_do,
    const __grid_constant__ CUtensorMap tm_pk, const __grid_constant__ CUtensorMap tm_pv, int T, int H,
    const int32_t* __restrict__ cu, const uint32_t* __restrict__ tiles, const float* __restrict__ lse,
    const float* __restrict__ delta, const float2* __restrict__ rope_tab, float scale, float scale_log2, int Lp,
    bf16* __restrict__ dqkv, const int32_t* __restrict__ ctxs, const int32_t* __restrict__ gpos,
    const int32_t* __restrict__ gpos2, float* __restrict__ dbias, int* status) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;
  uint8_t* sdO = smem + TILE;
  uint8_t* sK = smem + 2 * TILE;
  uint8_t* sV = smem + 3 * TILE;
  uint8_t* sdS = smem + 4 * TILE;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + 6 * TILE + 2 * TB * 4);
  uint64_t* bar_load = bars;
  uint64_t* bar_mma1 = bars + 1;
  uint64_t* bar_mma2 = bars + 2;
  uint32_t* holder = reinterpret_cast<uint32_t*>(bars + 4);

  // the 128-row tile list: (segment, query tile)
  const int s = int(tiles[blockIdx.x] >> 16), idx = int(tiles[blockIdx.x] & 0xFFFFu);
  const int h = blockIdx.y;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int quarter = warp & 3, kh = warp >> 2;
  const int r = quarter * 32 + lane;  // this thread's query row (TMEM lane)
  const int seg0 = cu[s], L = cu[s + 1] - seg0;
  const int q0 = idx * TB;
  const int q = q0 + r;
  const bool q_ok = q < L;
  const int npt = Lp > 0 ? 1 : 0;  // at most one prefix tile (Lp <= 128)
  const int clast = (ctxs ? min(max(ctxs[s], 0), L) : 0) - 1;
  const int n_kv = npt + max(idx, clast >= 0 ? clast / TB : 0) + 1;
  const float lse2 = q_ok ? __ldg(lse + (int64_t)h * T + seg0 + q) * LOG2E_B : 0.f;
  const float dl = q_ok ? __ldg(delta + (int64_t)h * T + seg0 + q) : 0.f;
  const int ulim = q_ok ? max(q, clast) : -1;  // last own key visible to the row

  if (tid == 0) {
    mbar_init(bar_load, 1);
    mbar_init(bar_mma1, 1);
    mbar_init(bar_mma2, 1);
    fence_mbar_init();
    tma_prefetch_desc(&tm_qkv);
    tma_prefetch_desc(&tm_do);
  }
  if (warp == 0) {
    tmem_alloc(holder, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *holder;
  const uint32_t t_lane = tmem + (uint32_t(quarter * 32) << 16);

  auto issue_kv = [&](int j) {  // one elected thread
    if (j < npt) {
      tma_load_2d(sK, &tm_pk, bar_load, h * HDT, 0);
      tma_load_2d(sK + BOX, &tm_pk, bar_load, h * HDT + 64, 0);
      tma_load_2d(sV, &tm_pv, bar_load, h * HDT, 0);
      tma_load_2d(sV + BOX, &tm_pv, bar_load, h * HDT + 64, 0);
    } else {
      const int row = seg0 + (j - npt) * TB;
      tma_load_2d(sK, &tm_qkv, bar_load, H + h * HDT, row);
      tma_load_2d(sK + BOX, &tm_qkv, bar_load, H + h * HDT + 64, row);
      tma_load_2d(sV, &tm_qkv, bar_load, 2 * H + h * HDT, row);
      tma_load_2d(sV + BOX, &tm_qkv, bar_load, 2 * H + h * HDT + 64, row);
    }
  };
  if (tid == 0) {
    mbar_arrive_expect_tx(bar_load, 4 * TILE);
    tma_load_2d(sQ, &tm_qkv, bar_load, h * HDT, seg0 + q0);
    tma_load_2d(sQ + BOX, &tm_qkv, bar_load, h * HDT + 64, seg0 + q0);
    tma_load_2d(sdO, &tm_do, bar_load, h * HDT, seg0 + q0);
    tma_load_2d(sdO + BOX, &tm_do, bar_load, h * HDT + 64, seg0 + q0);
    issue_kv(0);
  }

  constexpr uint32_t IDESC_S = umma_idesc_bf16(TB, TB, false, false);
  constexpr uint32_t IDESC_G = umma_idesc_bf16(TB, HDT, false, true);
  bool ok = true;
  uint32_t ph = 0;
  for (int j = 0; j < n_kv && ok; ++j, ph ^= 1) {
    if (!__syncthreads_and(mbar_wait(bar_load, ph))) {
      if (tid == 0) report_status(status, FL_DEV_TIMEOUT_FULL);
      ok = false;
      break;
    }
    // ---- S = Q K_j^T, dP = dO V_j^T
    if (tid == 0) {
      tc_fence_after();
      const uint32_t aq = smem_u32(sQ), ao = smem_u32(sdO), bk = smem_u32(sK), bv = smem_u32(sV);
#pragma unroll
      for (int kk = 0; kk < HDT / 16; ++kk) umma_bf16(tmem, desc_k(aq, kk), desc_k(bk, kk), IDESC_S, kk > 0);
#pragma unroll
      for (int kk = 0; kk < HDT / 16; ++kk) umma_bf16(tmem + 128, desc_k(ao, kk), desc_k(bv, kk), IDESC_S, kk > 0);
      umma_commit(bar_mma1);
    }
    if (!__syncthreads_and(mbar_wait(bar_mma1, ph))) {
      if (tid == 0) report_status(status, FL_DEV_TIMEOUT_ACC_FULL);
      ok = false;
      break;
    }
    tc_fence_after();
    // ---- dS of query row r for keys kh * 64 .. + 63 of the tile, in two halves of 32
    {
      const bool prefix = j < npt;
      const int u0 = (prefix ? 0 : (j - npt) * TB) + kh * 64;  // first key of the half
      const int uend = prefix ? (q_ok ? Lp : 0) : ulim + 1;    // keys [u0, uend) are visible
#pragma unroll 1
      for (int hf = 0; hf < 2; ++hf) {
        uint32_t sr[32], dr[32];
        tmem_ld32(t_lane + kh * 64 + 32 * hf, sr);
        tmem_ld32(t_lane + 128 + kh * 64 + 32 * hf, dr);
        tmem_ld_wait();
#pragma unroll
        for (int c8 = 0; c8 < 4; ++c8) {
          float ds[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const int c = 8 * c8 + e;
            const bool vis = u0 + 32 * hf + c < uend;
            const float pv = vis ? exp2_hw(fmaf(__uint_as_float(sr[c]), scale_log2, -lse2)) : 0.f;
            ds[e] = pv * (__uint_as_float(dr[c]) - dl);
          }
          put_chunk8(sdS, kh, r, 4 * hf + c8, ds);
        }
      }
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    // ---- dQ += dS K_j
    if (tid == 0) {
      tc_fence_after();
      const uint32_t as = smem_u32(sdS), bk = smem_u32(sK);
#pragma unroll
      for (int kk = 0; kk < TB / 16; ++kk)
        umma_bf16(tmem + 256, desc_k(as, kk), desc_mn(bk, kk), IDESC_G, (j > 0 || kk > 0) ? 1u : 0u);
      umma_commit(bar_mma2);
    }
    if (!__syncthreads_and(mbar_wait(bar_mma2, ph))) {
      if (tid == 0) report_status(status, FL_DEV_TIMEOUT_ACC_EMPTY);
      ok = false;
      break;
    }
    tc_fence_after();
    if (tid == 0 && j + 1 < n_kv) {
      mbar_arrive_expect_tx(bar_load, 2 * TILE);
      issue_kv(j + 1);
    }
  }

  // ---- dQ (scaled, rotated back): thread (r, kh) takes dims kh * 64 .. + 63 of query row r,
  // staged in the freed K buffer and written as whole coalesced rows, the bias column sums
  // taken from the staged rows; the rotary rows of the tile's queries in the freed V buffer
  // (32 KB: one region) or, with GLM block positions, V and dO (64 KB).
  if (ok) {
    const int nreg = rope_tab ? (gpos2 ? 2 : 1) : 0;
    for (int reg = 0; reg < nreg; ++reg) {  // warp w loads rows w, w + 8, ...: 16 in flight
      float2* rtr = reg == 0 ? reinterpret_cast<float2*>(sV) : reinterpret_cast<float2*>(sdO);
      const int32_t* gp = reg == 0 ? gpos : gpos2;
      int pos[TB / 8];
#pragma unroll
      for (int jj = 0; jj < TB / 8; ++jj) {
        const int qq = min(q0 + warp + 8 * jj, L - 1);
        pos[jj] = gp ? __ldg(gp + seg0 + qq) : qq;
      }
      float2 cs[TB / 8];
#pragma unroll
      for (int jj = 0; jj < TB / 8; ++jj) cs[jj] = __ldg(rope_tab + (int64_t)pos[jj] * 32 + lane);
#pragma unroll
      for (int jj = 0; jj < TB / 8; ++jj) {
        const int rr = warp + 8 * jj;
        rtr[rr * 32 + (lane ^ (rr & 31))] = cs[jj];
      }
    }
    __syncthreads();
    uint32_t vr[64];
    tmem_ld32(t_lane + 256 + kh * 64, *reinterpret_cast<uint32_t(*)[32]>(vr));
    tmem_ld32(t_lane + 256 + kh * 64 + 32, *reinterpret_cast<uint32_t(*)[32]>(vr + 32));
    tmem_ld_wait();
    float* v = reinterpret_cast<float*>(vr);
#pragma unroll
    for (int c = 0; c < 64; ++c) v[c] = __uint_as_float(vr[c]) * scale;
    if (kh < nreg && q_ok)
      inverse_rope_row(v, reinterpret_cast<float2*>(kh == 0 ? sV : sdO) + r * 32, r & 31);
#pragma unroll
    for (int c8 = 0; c8 < 8; ++c8) {
      const int jc = kh * 8 + c8;
      *reinterpret_cast<uint4*>(sK + r * 256 + ((jc ^ (r & 15)) << 4)) =
          make_uint4(pack_bf16x2(v[8 * c8], v[8 * c8 + 1]), pack_bf16x2(v[8 * c8 + 2], v[8 * c8 + 3]),
                     pack_bf16x2(v[8 * c8 + 4], v[8 * c8 + 5]), pack_bf16x2(v[8 * c8 + 6], v[8 * c8 + 7]));
    }
    const int col = blockIdx.y * HDT;
    __syncthreads();  // the tile is staged
    if (dbias) staged_colsum(sK, min(TB, L - q0), dbias + col, tid);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int id = tid + 256 * i, row = id >> 4, jc = id & 15;
      if (q0 + row < L) {
        const uint4 w = *reinterpret_cast<const uint4*>(sK + row * 256 + ((jc ^ (row & 15)) << 4));
        *reinterpret_cast<uint4*>(dqkv + ((int64_t)seg0 + q0 + row) * 3 * H + col + jc * 8) = w;
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

}  // namespace

int fl_launch_attn_bwd_dkv_tc(int T, int nh, const void* qkv, const void* dout, const float* lse, const float* delta,
                              const int32_t* cu, const uint32_t* tiles, int n_tiles, const float* rope_tab,
                              void* dqkv, const AttnGlm& glm, float* dbias, int* status, cudaStream_t st) {
  static bool attr = false;
  if (!attr) {
    FL_CUDA_TRY(cudaFuncSetAttribute(attn_bwd_dkv_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM));
    attr = true;
  }
  const int H = nh * HDT;
  CUtensorMap tq, tdo;
  if (int rc = fl_gemm::make_map(&tq, qkv, (uint64_t)3 * H, (uint64_t)T, 3 * (int64_t)H, 128)) return rc;
  if (int rc = fl_gemm::make_map(&tdo, dout, (uint64_t)H, (uint64_t)T, H, 128)) return rc;
  const float scale = 1.f / sqrtf((float)HDT);
  attn_bwd_dkv_tc_kernel<<<dim3(n_tiles, nh), 256, SMEM, st>>>(
      tq, tdo, T, H, cu, tiles, lse, delta, reinterpret_cast<const float2*>(rope_tab), scale, scale * LOG2E_B,
      (bf16*)dqkv, glm.ctx, glm.pos, glm.pos2, dbias, status);
  FL_CUDA_TRY(cudaGetLastError());
  return FL_OK;
}

int fl_launch_attn_bwd_dq_tc(int T, int nh, const void* qkv, const void* dout, const float* lse, const float* delta,
                             const int32_t* cu, const uint32_t* tiles, int n_tiles, const float* rope_tab, void* dqkv,
                             const AttnPrefix& pre, const AttnGlm& glm, float* dbias, int* status, cudaStream_t st) {
  static bool attr = false;
  if (!attr) {
    FL_CUDA_TRY(cudaFuncSetAttribute(attn_bwd_dq_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM));
    attr = true;
  }
  const int H = nh * HDT;
  CUtensorMap tq, tdo, tpk, tpv;
  if (int rc = fl_gemm::make_map(&tq, qkv, (uint64_t)3 * H, (uint64_t)T, 3 * (int64_t)H, 128)) return rc;
  if (int rc = fl_gemm::make_map(&tdo, dout, (uint64_t)H, (uint64_t)T, H, 128)) return rc;
  if (pre.len > 0) {
    if (int rc = fl_gemm::make_map(&tpk, pre.k, (uint64_t)H, (uint64_t)pre.len, H, 128)) return rc;
    if (int rc = fl_gemm::make_map(&tpv, pre.v, (uint64_t)H, (uint64_t)pre.len, H, 128)) return rc;
  } else {
    tpk = tq;
    tpv = tq;
  }
  const float scale = 1.f / sqrtf((float)HDT);
  attn_bwd_dq_tc_kernel<<<dim3(n_tiles, nh), 256, SMEM, st>>>(
      tq, tdo, tpk, tpv, T, H, cu, tiles, lse, delta, reinterpret_cast<const float2*>(rope_tab), scale,
      scale * LOG2E_B, pre.len, (bf16*)dqkv, glm.ctx, glm.pos, glm.pos2, dbias, status);
  FL_CUDA_TRY(cudaGetLastError());
  return FL_OK;
}
