// Attention backward on the 5th-generation tensor cores, head_dim 64 or 128: dQ, dK / dV
// of the segment's own keys, and dK / dV of the P-tuning prefix keys (the gradient of
// App. A's softmax(Q K'^T / sqrt(d_h)) V', causal or with a bidirectional GLM context).
//
// Shared layout of both kernels: 128-row tiles; operands arrive by TMA as 64-column
// 128-byte-swizzled boxes; the score-side products (S, dP or their transposes) sit in
// TMEM columns [0, 256); the probabilities / score gradients the threads derive from them
// are stored back into TMEM (bf16, two per 32-bit column) over the values already read,
// and feed the next products as A operands read from TMEM.  That leaves shared memory to
// double-buffer the tiles the CTA walks through, so their loads overlap the work on the
// previous tile.
//
// Both kernels are persistent: one CTA per SM (226 KB of shared memory at head_dim 128,
// 512 TMEM columns) walks work units u = blockIdx.x, + gridDim.x, ...  Each of the next
// unit's tiles is loaded as soon as its buffer has had its last use in the current unit,
// so they arrive while the unit's last products run and its output is staged (in a tile
// of its own) and written; a whole tile of output rows leaves by bulk tensor stores
// (TMA), which the next unit's epilogue waits for only before it stages again.  Per-row
// values that a unit needs later (the next tile's lse / delta, the rotary rows of the
// epilogue, the descriptor of the unit after next) are read while products run.
//
// dK / dV: unit = (128-key tile, head).  Warp w reads TMEM lanes 32 (w % 4) .. + 31, so
// thread (w, lane) owns key row r = 32 (w % 4) + lane, and takes query half w / 4 of every
// query tile.  Per 128-query tile i that sees the key tile:
//   TMA: Q_i and dO_i into the buffer pair (i % 2), the next tile's while this one works;
//   S^T = K Q_i^T -> TMEM [0, 128)      dP^T = V dO_i^T -> TMEM [128, 256);
//   threads: P^T = exp2(S^T scale log2e - lse_q log2e) where key r is visible to query q,
//            dS^T = P^T (dP^T - delta_q), bf16 over the S^T / dP^T values just read;
//   dV += P^T dO_i -> TMEM [256, 256 + hd)   dK += dS^T Q_i -> TMEM [256 + hd, 256 + 2 hd)
//            (A from TMEM, dO_i and Q_i as MN-major operands).
// Epilogue: dK * scale, the inverse rotary rotation(s), bf16 rows of dqkv and the k / v
// column sums for the QKV bias gradient; the prefix variant (PREFIX: the unit's keys are
// the prefix of its head, its query tiles a slice of the call's tile list) adds dK * scale
// and dV into the fp32 prefix gradients instead.
//
// dQ: unit = (128-query tile, head); thread (w, lane) owns query row r = 32 (w % 4) + lane
// and key half w / 4 of every key tile.  Per key tile j (the prefix tile first, then the
// segment's own keys), K_j / V_j double-buffered:
//   S = Q K_j^T -> TMEM [0, 128), dP = dO V_j^T -> TMEM [128, 256);
//   threads: dS = P (dP - delta_q), P = exp2(S scale log2e - lse_q log2e) on the visible
//            keys, bf16 over the S values just read;
//   dQ += dS K_j -> TMEM [256, 256 + hd) (A from TMEM, K_j as an MN-major operand).
// Epilogue as in dK / dV: dQ * scale, inverse rotary rotation(s), coalesced bf16 rows, q
// column sums.
//
// Every mbarrier wait is bounded (2 s): on expiry the CTA records a status code, lets what
// it armed land and leaves its remaining work undone.
#include <cuda.h>
#include <cuda_runtime.h>

#include <cmath>

#include "../../include/flglm_kernels.h"
#include "common.cuh"
#include "gemm_tc.cuh"
#include "kernels.cuh"
#include "ptx.cuh"
#include "waits.cuh"

namespace {

typedef __nv_bfloat16 bf16;
constexpr int TB = 128;            // keys and queries per tile (UMMA M and N)
constexpr int BOX = 64 * 128 * 2;  // one 64-column x 128-row bf16 box: 16 KB
constexpr float LOG2E_B = 1.4426950408889634f;

template <int HD>
struct BwdCfg {
  static constexpr int NB = HD / 64;     // boxes per tile row
  static constexpr int TILE = NB * BOX;  // one 128 x HD bf16 tile
  static constexpr int CH = HD / 8;      // 16-byte chunks per staged bf16 row
  static constexpr int E = HD / 4;       // rotary (cos, sin) entries per position
  // six operand tiles, a staging tile for the output rows, lse / delta of one query tile;
  // padded at head_dim 64 so that one CTA (512 TMEM columns) has an SM to itself
  static constexpr int USED = 7 * TILE + 2 * TB * 4 + 128 /*barriers, holder*/ + 1024 /*alignment*/;
  static constexpr int SMEM = USED > 120 * 1024 ? USED : 120 * 1024;
};

FL_DEV uint64_t desc_k(uint32_t base, int kk) { return smem_desc_sw128(base + (kk >> 2) * BOX + (kk & 3) * 32, 16, 1024); }
FL_DEV uint64_t desc_mn(uint32_t base, int kk) { return smem_desc_sw128(base + kk * 2048, BOX, 1024); }

// TMEM column (relative to the region's start) of the bf16 operand's k-step kk (16
// columns of the 128-wide product): thread half g = kk / 4 wrote its columns 64 g .. + 63
// as two groups of 32 values at 64 g + 16 hf (hf = (kk / 2) % 2), 8 columns per k-step.
FL_DEV uint32_t a_col(int kk) { return (kk >> 2) * 64 + ((kk >> 1) & 1) * 16 + (kk & 1) * 8; }

// The rotary table row of one token's position, (cos, sin) of pairs 2j, 2j + 1 in cs[j]:
// read from global memory (the table is small and L2-resident) while the unit's last
// products run, applied in the epilogue.
template <int HD>
struct RopeRow {
  float4 cs[HD / 8];
};
template <int HD>
FL_DEV void rope_load(RopeRow<HD>& rr, const float2* __restrict__ row) {
  const float4* r4 = reinterpret_cast<const float4*>(row);
#pragma unroll
  for (int j = 0; j < HD / 8; ++j) rr.cs[j] = __ldg(r4 + j);
}
// Inverse rotary rotation of one rotary region held by a thread: HD/2 consecutive dims,
// pairs (i, i + HD/4), angle (cos, sin) of pair i from the token's table row.
template <int HD>
FL_DEV void inverse_rope_row(float* v, const RopeRow<HD>& rr) {
  constexpr int Q = HD / 4;
#pragma unroll
  for (int j = 0; j < Q / 2; ++j) {
    const int i = 2 * j;  // pairs i and i + 1
    float x1 = v[i], x2 = v[i + Q];
    v[i] = x1 * rr.cs[j].x + x2 * rr.cs[j].y;
    v[i + Q] = x2 * rr.cs[j].x - x1 * rr.cs[j].y;
    x1 = v[i + 1];
    x2 = v[i + 1 + Q];
    v[i + 1] = x1 * rr.cs[j].z + x2 * rr.cs[j].w;
    v[i + 1 + Q] = x2 * rr.cs[j].z - x1 * rr.cs[j].w;
  }
}

// 2^x by the hardware instruction (PTX ex2.approx.ftz.f32): the probabilities it feeds are
// rounded to bf16 for the tensor cores.
FL_DEV float exp2_hw(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Staged bf16 tile in the layout of 128-byte-swizzled TMA boxes of 64 columns x 128 rows:
// 16-byte chunk j of row r in box j / 8, at chunk (j % 8) ^ (r % 8) of the box's row r.
template <int HD>
FL_DEV uint8_t* stage_chunk(uint8_t* stage, int r, int j) {
  return stage + (j >> 3) * (TB * 128) + r * 128 + (((j & 7) ^ (r & 7)) << 4);
}

// 2-D tiled store of one box from shared memory to global memory (bulk-group completion).
FL_DEV void tma_store_2d(const CUtensorMap* m, const void* src, int x, int y) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.tile.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
                   reinterpret_cast<uint64_t>(m)),
               "r"(smem_u32(src)), "r"(x), "r"(y)
               : "memory");
}
FL_DEV void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// The committed bulk stores have read their shared memory (it may be written again).
FL_DEV void bulk_wait_read() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
// The committed bulk stores are complete.
FL_DEV void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// Adds the column sums of a staged tile over its first `rows` rows to out[0..HD); called by
// all 256 threads.  Warp wp takes the HD/64 16-byte chunks wp*HD/64 ..: LPC = 32*64/HD
// lanes per chunk, lane l reading rows l % LPC, + LPC, ... (8 consecutive lanes read 8
// consecutive rows of one chunk: distinct swizzled 16-byte slots, no bank conflict), then
// a butterfly over the chunk's lanes and one atomic per column.
template <int HD>
FL_DEV void staged_colsum(uint8_t* stage, int rows, float* out, int tid) {
  constexpr int CPW = HD / 64, LPC = 32 / CPW;
  const int lane = tid & 31, jc = (tid >> 5) * CPW + lane / LPC, r0 = lane % LPC;
  float acc[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) acc[e] = 0.f;
#pragma unroll
  for (int i = 0; i < TB / LPC; ++i) {
    const int row = r0 + LPC * i;
    if (row < rows) {
      const uint4 q = *reinterpret_cast<const uint4*>(stage_chunk<HD>(stage, row, jc));
      const uint32_t qw[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float2 f = unpack_bf16x2(qw[e]);
        acc[2 * e] += f.x;
        acc[2 * e + 1] += f.y;
      }
    }
  }
#pragma unroll
  for (int off = LPC / 2; off > 0; off >>= 1)
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[e] += __shfl_xor_sync(0xffffffffu, acc[e], off);
  float mine = acc[0];
#pragma unroll
  for (int e = 1; e < 8; ++e)
    if (r0 == e) mine = acc[e];
  if (r0 < 8) atomicAdd(out + jc * 8 + r0, mine);
}

// dK / dV.  Non-prefix: unit u = (entry u / nh of the 128-row tile list, head u % nh), the
// entry's tile index i standing for key tile nq - 1 - i (a segment's key tile 0, seen by
// every query tile, first).
// PREFIX: unit u = (slice u / nh of the tile list cut into n_split slices, head u % nh),
// the unit's keys the Lp prefix keys of its head.
template <int HD, bool PREFIX>
__global__ void __launch_bounds__(256, 1) attn_bwd_dkv_tc_kernel(
    const __grid_constant__ CUtensorMap tm_qkv, const __grid_constant__ CUtensorMap tm_do,
    const __grid_constant__ CUtensorMap tm_pk, const __grid_constant__ CUtensorMap tm_pv,
    const __grid_constant__ CUtensorMap tm_dqkv, int T, int H,
    const int32_t* __restrict__ cu, const uint32_t* __restrict__ tiles, int n_tiles, int n_units, int n_split,
    const float* __restrict__ lse, const float* __restrict__ delta, const float2* __restrict__ rope_tab, float scale,
    float scale_log2, int Lp, bf16* __restrict__ dqkv, float* __restrict__ dpk, float* __restrict__ dpv,
    const int32_t* __restrict__ ctxs, const int32_t* __restrict__ gpos, const int32_t* __restrict__ gpos2,
    float* __restrict__ dbias, int dbias_segs, int64_t dbias_rstride, int* status) {
  constexpr int NB = BwdCfg<HD>::NB, TILE = BwdCfg<HD>::TILE, CH = BwdCfg<HD>::CH, E = BwdCfg<HD>::E;
  pdl_wait();  // the previous kernel on the stream has completed (see fl_launch)
  pdl_trigger();
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sK = smem;
  uint8_t* sV = smem + TILE;
  uint8_t* sQ = smem + 2 * TILE;   // [2]
  uint8_t* sdO = smem + 4 * TILE;  // [2]
  uint8_t* sST = smem + 6 * TILE;  // staging of the bf16 output rows
  float* sL = reinterpret_cast<float*>(smem + 7 * TILE);  // [128] lse * log2e of the query tile
  float* sD = sL + TB;                                    // [128] delta of the query tile
  uint64_t* bars = reinterpret_cast<uint64_t*>(sD + TB);
  uint64_t* bar_kv = bars;
  uint64_t* bar_q = bars + 1;  // [2]
  uint64_t* bar_mma1 = bars + 3;
  uint64_t* bar_mma2 = bars + 4;
  uint32_t* holder = reinterpret_cast<uint32_t*>(bars + 6);

  const int nh = H / HD;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int quarter = warp & 3, qh = warp >> 2;
  const int r = quarter * 32 + lane;  // this thread's key row (TMEM lane)
  const int nreg = rope_tab ? (gpos2 ? 2 : 1) : 0;  // rotary regions of a head

  // a unit: its head, keys (segment start and length, first key kb), the last context key
  // of the segment (GLM; -1 when causal), its query tiles [it0, it_end), and the QKV bias
  // gradient of the segment's replica
  struct Unit {
    int h, seg0, L, kb, clast, it0, it_end;
    float* db;
  };
  auto unit_t = [&](int u, uint32_t t) {
    Unit w;
    w.h = u % nh;
    if constexpr (PREFIX) {
      const int per = (n_tiles + n_split - 1) / n_split;
      w.it0 = (u / nh) * per;
      w.it_end = min(n_tiles, w.it0 + per);
      w.seg0 = w.L = w.kb = 0;
      w.clast = -1;
      w.db = nullptr;
    } else {
      const int s = int(t >> 16), idx = int(t & 0xFFFFu);
      w.seg0 = cu[s];
      w.L = cu[s + 1] - w.seg0;
      const int nq = (w.L + TB - 1) / TB;
      const int kt = nq - 1 - idx;
      w.kb = kt * TB;
      w.clast = (ctxs ? min(max(ctxs[s], 0), w.L) : 0) - 1;
      w.it0 = w.kb <= w.clast ? 0 : kt;  // a tile holding context keys is seen by every query
      w.it_end = nq;
      w.db = dbias ? dbias + (dbias_segs > 0 ? (int64_t)(s / dbias_segs) * dbias_rstride : 0) : nullptr;
    }
    return w;
  };
  auto tile_word = [&](int u) { return PREFIX ? 0u : tiles[u / nh]; };
  auto unit = [&](int u) { return unit_t(u, tile_word(u)); };
  // a query tile of unit w: its first token, the position of that token in its segment,
  // valid rows
  auto qtile = [&](const Unit& w, int it, int& row0, int& qpos0, int& valid) {
    if constexpr (PREFIX) {
      const int s = int(tiles[it] >> 16), idx = int(tiles[it] & 0xFFFFu);
      const int sb = cu[s];
      qpos0 = idx * TB;
      row0 = sb + qpos0;
      valid = min(TB, cu[s + 1] - sb - qpos0);
    } else {
      qpos0 = it * TB;
      row0 = w.seg0 + qpos0;
      valid = min(TB, w.L - qpos0);
    }
  };

  if (tid == 0) {
    for (int i = 0; i < 5; ++i) mbar_init(bars + i, 1);
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

  BarTrack tkv, tq0, tq1, tm1, tm2;
  auto issue_q = [&](const Unit& w, int it, int b) {  // one elected thread: Q_it, dO_it into pair b
    int row0, qpos0, valid;
    qtile(w, it, row0, qpos0, valid);
    (b ? tq1 : tq0).pend = true;
    mbar_arrive_expect_tx(bar_q + b, 2 * TILE);
#pragma unroll
    for (int x = 0; x < NB; ++x) {
      tma_load_2d(sQ + b * TILE + x * BOX, &tm_qkv, bar_q + b, w.h * HD + 64 * x, row0);
      tma_load_2d(sdO + b * TILE + x * BOX, &tm_do, bar_q + b, w.h * HD + 64 * x, row0);
    }
  };
  auto issue_kv = [&](const Unit& w) {  // one elected thread: the unit's K and V
    tkv.pend = true;
    mbar_arrive_expect_tx(bar_kv, 2 * TILE);
#pragma unroll
    for (int x = 0; x < NB; ++x) {
      if constexpr (PREFIX) {
        tma_load_2d(sK + x * BOX, &tm_pk, bar_kv, w.h * HD + 64 * x, 0);
        tma_load_2d(sV + x * BOX, &tm_pv, bar_kv, w.h * HD + 64 * x, 0);
      } else {
        tma_load_2d(sK + x * BOX, &tm_qkv, bar_kv, H + w.h * HD + 64 * x, w.seg0 + w.kb);
        tma_load_2d(sV + x * BOX, &tm_qkv, bar_kv, 2 * H + w.h * HD + 64 * x, w.seg0 + w.kb);
      }
    }
  };

  constexpr uint32_t IDESC_S = umma_idesc_bf16(TB, TB, false, false);
  constexpr uint32_t IDESC_G = umma_idesc_bf16(TB, HD, false, true);
  bool ok = true;
  int u = blockIdx.x;
  Unit w = u < n_units ? unit(u) : Unit{};
  Unit wn = u + (int)gridDim.x < n_units ? unit(u + gridDim.x) : Unit{};
  // the thread's lse (tid < 128) or delta value of the next query tile, loaded a tile early
  auto stat_of = [&](const Unit& x, int it) {
    int row0, qpos0, valid;
    qtile(x, it, row0, qpos0, valid);
    const int c = tid & (TB - 1);
    const float* src = tid < TB ? lse : delta;
    return c < valid ? __ldg(src + (int64_t)x.h * T + row0 + c) : 0.f;
  };
  float pf = (u < n_units && w.it0 < w.it_end) ? stat_of(w, w.it0) : 0.f;
  RopeRow<HD> rrow;
  if (tid == 0 && u < n_units && w.it0 < w.it_end) {
    issue_kv(w);
    issue_q(w, w.it0, 0);
    if (w.it0 + 1 < w.it_end) issue_q(w, w.it0 + 1, 1);
  }
  while (u < n_units && ok) {
    const int k = w.kb + r;  // the key inside its segment (or the prefix)
    const bool key_ok = PREFIX ? r < Lp : k < w.L;
    const bool work = w.it0 < w.it_end;
    // the next unit: its K / V load once this unit's last S^T / dP^T products have read K
    // and V, its first query tile once buffer pair 0 has had its last use here
    const int un = u + gridDim.x;
    const bool next = un < n_units && wn.it0 < wn.it_end;
    Unit wnn = Unit{};  // the unit after next: its tile word read while the first score
    uint32_t tnn = 0;   // products run, the rest while the first gradient products run
    // every wait's outcome is agreed on by the whole CTA, so that all threads leave together
    if (work && !track_wait_all(bar_kv, tkv)) {
      if (tid == 0) report_status(status, FL_DEV_TIMEOUT_FULL);
      ok = false;
      break;
    }
    for (int it = w.it0; it < w.it_end && ok; ++it) {
      const int b = (it - w.it0) & 1;
      int row0, qpos0, valid;
      qtile(w, it, row0, qpos0, valid);
      {  // lse and delta of the query tile (rows past its segment are never visible)
        const int c = tid & (TB - 1);
        if (tid < TB) sL[c] = pf * LOG2E_B;  // the previous tile's readers passed a barrier since
        else sD[c] = pf;
      }
      if (!track_wait_all(bar_q + b, b ? tq1 : tq0)) {
        if (tid == 0) report_status(status, FL_DEV_TIMEOUT_FULL);
        ok = false;
        break;
      }
      // ---- S^T = K Q^T, dP^T = V dO^T (the previous dV / dK products, which read these
      // columns, have completed)
      if (tid == 0) {
        tc_fence_after();
        const uint32_t ak = smem_u32(sK), av = smem_u32(sV), bq = smem_u32(sQ + b * TILE),
                       bo = smem_u32(sdO + b * TILE);
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) umma_bf16(tmem, desc_k(ak, kk), desc_k(bq, kk), IDESC_S, kk > 0);
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) umma_bf16(tmem + 128, desc_k(av, kk), desc_k(bo, kk), IDESC_S, kk > 0);
        tm1.pend = true;
        umma_commit(bar_mma1);
      }
      // while the products run: the next tile's statistics, the unit after next
      if (it + 1 < w.it_end) pf = stat_of(w, it + 1);
      else if (next) pf = stat_of(wn, wn.it0);
      if (it == w.it0 && un + (int)gridDim.x < n_units) tnn = tile_word(un + gridDim.x);
      if (!track_wait_all(bar_mma1, tm1)) {
        if (tid == 0) report_status(status, FL_DEV_TIMEOUT_ACC_FULL);
        ok = false;
        break;
      }
      tc_fence_after();
      if (tid == 0 && next && it + 1 == w.it_end) issue_kv(wn);
      // ---- P^T and dS^T of key row r for queries qh * 64 .. + 63, in two groups of 32,
      // each written (bf16 pairs) into the 16 columns at 64 qh + 16 hf it has just read
      {
        const int q0 = qpos0 + qh * 64;
        // key k is visible to queries [qfirst, qlim) of the tile's segment
        int qlim, qfirst;
        if constexpr (PREFIX) {
          qlim = key_ok ? qpos0 + valid : q0;
          qfirst = q0;
        } else {
          qlim = key_ok ? min(w.L, q0 + 64) : q0;
          qfirst = k <= w.clast ? q0 : max(q0, k);
        }
        const float* Lb = sL;
        const float* Db = sD;
#pragma unroll 1
        for (int hf = 0; hf < 2; ++hf) {
          uint32_t sr[32], dr[32];
          tmem_ld32(t_lane + qh * 64 + 32 * hf, sr);
          tmem_ld32(t_lane + 128 + qh * 64 + 32 * hf, dr);
          tmem_ld_wait();
          const float4* L4 = reinterpret_cast<const float4*>(Lb + qh * 64 + 32 * hf);
          const float4* D4 = reinterpret_cast<const float4*>(Db + qh * 64 + 32 * hf);
          uint32_t pp[16], dd[16];
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
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              pp[4 * c8 + e] = pack_bf16x2(p[2 * e], p[2 * e + 1]);
              dd[4 * c8 + e] = pack_bf16x2(ds[2 * e], ds[2 * e + 1]);
            }
          }
          tmem_st16(t_lane + qh * 64 + 16 * hf, pp);
          tmem_st16(t_lane + 128 + qh * 64 + 16 * hf, dd);
        }
      }
      tmem_st_wait();
      tc_fence_before();
      __syncthreads();
      // ---- dV += P^T dO, dK += dS^T Q (A from TMEM); then the tile after next into this
      // buffer pair once both products have read it
      if (tid == 0) {
        tc_fence_after();
        const uint32_t bq = smem_u32(sQ + b * TILE), bo = smem_u32(sdO + b * TILE);
        const bool acc = it > w.it0;
#pragma unroll
        for (int kk = 0; kk < TB / 16; ++kk)
          umma_bf16_ts(tmem + 256, tmem + a_col(kk), desc_mn(bo, kk), IDESC_G, (acc || kk > 0) ? 1u : 0u);
#pragma unroll
        for (int kk = 0; kk < TB / 16; ++kk)
          umma_bf16_ts(tmem + 256 + HD, tmem + 128 + a_col(kk), desc_mn(bq, kk), IDESC_G, (acc || kk > 0) ? 1u : 0u);
        tm2.pend = true;
        umma_commit(bar_mma2);
      }
      if (it == w.it0 && un + (int)gridDim.x < n_units) wnn = unit_t(un + gridDim.x, tnn);
      if (!PREFIX && it + 1 == w.it_end && qh < nreg && key_ok) {  // the key's rotary row, for the epilogue
        const int32_t* gp = qh == 0 ? gpos : gpos2;
        rope_load<HD>(rrow, rope_tab + (int64_t)(gp ? __ldg(gp + w.seg0 + k) : k) * E);
      }
      if (!track_wait_all(bar_mma2, tm2)) {
        if (tid == 0) report_status(status, FL_DEV_TIMEOUT_ACC_EMPTY);
        ok = false;
        break;
      }
      tc_fence_after();
      if (tid == 0) {
        if (it + 2 < w.it_end) {
          issue_q(w, it + 2, b);
        } else if (next) {  // pair b's last use in this unit: the next unit's tile of pair b
          if (wn.it0 + b < wn.it_end) issue_q(wn, wn.it0 + b, b);
          if (w.it0 + 1 == w.it_end && wn.it0 + 1 < wn.it_end) issue_q(wn, wn.it0 + 1, 1);  // pair 1 unused here
        }
      }
    }
    if (!ok) break;

    // ---- every product of the unit is complete: its dK / dV leave while the next unit's
    // tiles load
    if (tid == 0 && next && !work) {
      issue_kv(wn);
      issue_q(wn, wn.it0, 0);
      if (wn.it0 + 1 < wn.it_end) issue_q(wn, wn.it0 + 1, 1);
    }
    if (work) {
      if constexpr (PREFIX) {
        // ---- dK * scale and dV added into the fp32 prefix gradients: thread (r, qh) adds
        // dims qh * HD/2 .. + HD/2 - 1 of prefix key r
#pragma unroll 1
        for (int part = 0; part < 2; ++part) {  // 0: dK, 1: dV
          uint32_t vr[HD / 2];
#pragma unroll
          for (int c = 0; c < HD / 2; c += 32)
            tmem_ld32(t_lane + (part ? 256 : 256 + HD) + qh * (HD / 2) + c,
                      *reinterpret_cast<uint32_t(*)[32]>(vr + c));
          tmem_ld_wait();
          if (key_ok) {
            const float f = part ? 1.f : scale;
            float* dst = (part ? dpv : dpk) + (int64_t)r * H + w.h * HD + qh * (HD / 2);
#pragma unroll
            for (int c = 0; c < HD / 2; c += 4)
              red_add_v4(dst + c, __uint_as_float(vr[c]) * f, __uint_as_float(vr[c + 1]) * f,
                         __uint_as_float(vr[c + 2]) * f, __uint_as_float(vr[c + 3]) * f);
          }
        }
      } else {
        // ---- dV, then dK (scaled, rotated back): thread (r, qh) takes dims qh * HD/2 .. +
        // HD/2 - 1 of key row r from TMEM and stages the bf16 rows; a tile inside the
        // segment leaves by bulk tensor stores, a ragged last tile by coalesced 16-byte
        // stores of its valid rows; the bias column sums are taken from the staged rows
        // (the values stored)
#pragma unroll 1
        for (int pi = 0; pi < 2; ++pi) {
          const int part = 1 - pi;  // dV, then dK
          uint8_t* stage = sST;
          uint32_t vr[HD / 2];
#pragma unroll
          for (int c = 0; c < HD / 2; c += 32)
            tmem_ld32(t_lane + (part ? 256 : 256 + HD) + qh * (HD / 2) + c,
                      *reinterpret_cast<uint32_t(*)[32]>(vr + c));
          tmem_ld_wait();
          float* v = reinterpret_cast<float*>(vr);
#pragma unroll
          for (int c = 0; c < HD / 2; ++c) v[c] = __uint_as_float(vr[c]) * (part ? 1.f : scale);
          if (part == 0 && qh < nreg && key_ok) inverse_rope_row<HD>(v, rrow);  // rotary region qh
          // the staging tile is free once the previous bulk store has read it
          if (tid == 0) bulk_wait_read();
          __syncthreads();
#pragma unroll
          for (int c8 = 0; c8 < HD / 16; ++c8)
            *reinterpret_cast<uint4*>(stage_chunk<HD>(stage, r, qh * (HD / 16) + c8)) =
                make_uint4(pack_bf16x2(v[8 * c8], v[8 * c8 + 1]), pack_bf16x2(v[8 * c8 + 2], v[8 * c8 + 3]),
                           pack_bf16x2(v[8 * c8 + 4], v[8 * c8 + 5]), pack_bf16x2(v[8 * c8 + 6], v[8 * c8 + 7]));
          const int col = (part ? 2 * H : H) + w.h * HD;
          const bool full = w.kb + TB <= w.L;  // a whole tile of the segment: TMA stores
          if (full) fence_proxy_async_smem();  // the staged rows, visible to the bulk copies
          __syncthreads();  // the tile is staged
          if (full && tid == 0) {
#pragma unroll
            for (int x = 0; x < NB; ++x) tma_store_2d(&tm_dqkv, stage + x * (TB * 128), col + 64 * x, w.seg0 + w.kb);
            bulk_commit();
          }
          if (w.db) staged_colsum<HD>(stage, min(TB, w.L - w.kb), w.db + col, tid);
          if (!full) {
            // 128 rows x CH chunks: consecutive threads write consecutive chunks of a row
#pragma unroll
            for (int i = 0; i < TB * CH / 256; ++i) {
              const int id = tid + 256 * i, row = id / CH, jc = id % CH;
              if (w.kb + row < w.L)
                *reinterpret_cast<uint4*>(dqkv + ((int64_t)w.seg0 + w.kb + row) * 3 * H + col + jc * 8) =
                    *reinterpret_cast<const uint4*>(stage_chunk<HD>(stage, row, jc));
            }
          }
          __syncthreads();  // the staged rows have been read (the bulk store reads them on)
        }
      }
    }
    // the dK / dV columns are loaded before the next unit's products overwrite them
    tc_fence_before();
    __syncthreads();
    u = un;
    w = wn;
    wn = wnn;
  }
  if (tid == 0) bulk_wait_all();  // this CTA's bulk stores are complete before it leaves
  if (!ok && tid == 0) {  // a wait gave up: let what this CTA armed land before leaving
    track_drain(bar_kv, tkv);
    track_drain(bar_q, tq0);
    track_drain(bar_q + 1, tq1);
    track_drain(bar_mma1, tm1);
    track_drain(bar_mma2, tm2);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// dQ.  Unit u = (entry u / nh of the 128-row tile list, head u % nh).
template <int HD>
__global__ void __launch_bounds__(256, 1) attn_bwd_dq_tc_kernel(
    const __grid_constant__ CUtensorMap tm_qkv, const __grid_constant__ CUtensorMap tm_do,
    const __grid_constant__ CUtensorMap tm_pk, const __grid_constant__ CUtensorMap tm_pv,
    const __grid_constant__ CUtensorMap tm_dqkv, int T, int H,
    const int32_t* __restrict__ cu, const uint32_t* __restrict__ tiles, int n_units, const float* __restrict__ lse,
    const float* __restrict__ delta, const float2* __restrict__ rope_tab, float scale, float scale_log2, int Lp,
    bf16* __restrict__ dqkv, const int32_t* __restrict__ ctxs, const int32_t* __restrict__ gpos,
    const int32_t* __restrict__ gpos2, float* __restrict__ dbias, int dbias_segs, int64_t dbias_rstride, int* status) {
  constexpr int NB = BwdCfg<HD>::NB, TILE = BwdCfg<HD>::TILE, CH = BwdCfg<HD>::CH, E = BwdCfg<HD>::E;
  pdl_wait();  // the previous kernel on the stream has completed (see fl_launch)
  pdl_trigger();
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;
  uint8_t* sdO = smem + TILE;
  uint8_t* sK = smem + 2 * TILE;  // [2]
  uint8_t* sV = smem + 4 * TILE;  // [2]
  uint8_t* sST = smem + 6 * TILE;  // staging of the bf16 output rows
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + 7 * TILE + 2 * TB * 4);
  uint64_t* bar_qdo = bars;
  uint64_t* bar_kv = bars + 1;  // [2]
  uint64_t* bar_mma1 = bars + 3;
  uint64_t* bar_mma2 = bars + 4;
  uint32_t* holder = reinterpret_cast<uint32_t*>(bars + 6);

  const int nh = H / HD;
  const int tid = threadIdx.x, warp = tid >> 5;
  const int quarter = warp & 3, kh = warp >> 2;
  const int r = quarter * 32 + (tid & 31);  // this thread's query row (TMEM lane)
  const int npt = Lp > 0 ? 1 : 0;           // at most one prefix tile (Lp <= 128)
  const int nreg = rope_tab ? (gpos2 ? 2 : 1) : 0;

  // a unit: its head, segment, first query q0, last context key (-1 when causal), key
  // tiles (the prefix tile first), and the QKV bias gradient of the segment's replica
  struct Unit {
    int h, seg0, L, q0, clast, n_kv;
    float* db;
  };
  auto unit = [&](int u) {
    Unit w;
    const uint32_t t = tiles[u / nh];
    const int s = int(t >> 16), idx = int(t & 0xFFFFu);
    w.h = u % nh;
    w.seg0 = cu[s];
    w.L = cu[s + 1] - w.seg0;
    w.q0 = idx * TB;
    w.clast = (ctxs ? min(max(ctxs[s], 0), w.L) : 0) - 1;
    w.n_kv = npt + max(idx, w.clast >= 0 ? w.clast / TB : 0) + 1;
    w.db = dbias ? dbias + (dbias_segs > 0 ? (int64_t)(s / dbias_segs) * dbias_rstride : 0) : nullptr;
    return w;
  };
  // the thread's row statistics in unit w: lse * log2e and delta
  auto row_stats = [&](const Unit& w, float& lse2, float& dl) {
    const bool q_ok = w.q0 + r < w.L;
    lse2 = q_ok ? __ldg(lse + (int64_t)w.h * T + w.seg0 + w.q0 + r) * LOG2E_B : 0.f;
    dl = q_ok ? __ldg(delta + (int64_t)w.h * T + w.seg0 + w.q0 + r) : 0.f;
  };

  if (tid == 0) {
    for (int i = 0; i < 5; ++i) mbar_init(bars + i, 1);
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

  BarTrack tqdo, tkv0, tkv1, tm1, tm2;
  auto issue_kv = [&](const Unit& w, int j, int b) {  // one elected thread: K_j, V_j into pair b
    (b ? tkv1 : tkv0).pend = true;
    mbar_arrive_expect_tx(bar_kv + b, 2 * TILE);
#pragma unroll
    for (int x = 0; x < NB; ++x) {
      if (j < npt) {
        tma_load_2d(sK + b * TILE + x * BOX, &tm_pk, bar_kv + b, w.h * HD + 64 * x, 0);
        tma_load_2d(sV + b * TILE + x * BOX, &tm_pv, bar_kv + b, w.h * HD + 64 * x, 0);
      } else {
        const int row = w.seg0 + (j - npt) * TB;
        tma_load_2d(sK + b * TILE + x * BOX, &tm_qkv, bar_kv + b, H + w.h * HD + 64 * x, row);
        tma_load_2d(sV + b * TILE + x * BOX, &tm_qkv, bar_kv + b, 2 * H + w.h * HD + 64 * x, row);
      }
    }
  };
  auto issue_qdo = [&](const Unit& w) {  // one elected thread: the unit's Q and dO
    tqdo.pend = true;
    mbar_arrive_expect_tx(bar_qdo, 2 * TILE);
#pragma unroll
    for (int x = 0; x < NB; ++x) {
      tma_load_2d(sQ + x * BOX, &tm_qkv, bar_qdo, w.h * HD + 64 * x, w.seg0 + w.q0);
      tma_load_2d(sdO + x * BOX, &tm_do, bar_qdo, w.h * HD + 64 * x, w.seg0 + w.q0);
    }
  };

  constexpr uint32_t IDESC_S = umma_idesc_bf16(TB, TB, false, false);
  constexpr uint32_t IDESC_G = umma_idesc_bf16(TB, HD, false, true);
  bool ok = true;
  int u = blockIdx.x;
  Unit w = u < n_units ? unit(u) : Unit{};
  float lse2 = 0.f, dl = 0.f;
  if (u < n_units) row_stats(w, lse2, dl);
  RopeRow<HD> rrow;
  if (tid == 0 && u < n_units) {
    issue_qdo(w);
    issue_kv(w, 0, 0);
    if (w.n_kv > 1) issue_kv(w, 1, 1);
  }
  while (u < n_units && ok) {
    const int q = w.q0 + r;
    const bool q_ok = q < w.L;
    const int ulim = q_ok ? max(q, w.clast) : -1;  // last own key visible to the row
    // the next unit: its Q / dO load once this unit's last S / dP products have read them,
    // its first key / value tile once buffer pair 0 has had its last use here
    const int un = u + gridDim.x;
    const Unit wn = un < n_units ? unit(un) : Unit{};
    const bool next = un < n_units;
    // every wait's outcome is agreed on by the whole CTA, so that all threads leave together
    if (!track_wait_all(bar_qdo, tqdo)) {
      if (tid == 0) report_status(status, FL_DEV_TIMEOUT_FULL);
      ok = false;
      break;
    }
    for (int j = 0; j < w.n_kv && ok; ++j) {
      const int b = j & 1;
      if (!track_wait_all(bar_kv + b, b ? tkv1 : tkv0)) {
        if (tid == 0) report_status(status, FL_DEV_TIMEOUT_FULL);
        ok = false;
        break;
      }
      // ---- S = Q K_j^T, dP = dO V_j^T (the previous dQ product, which read these
      // columns, has completed)
      if (tid == 0) {
        tc_fence_after();
        const uint32_t aq = smem_u32(sQ), ao = smem_u32(sdO), bk = smem_u32(sK + b * TILE),
                       bv = smem_u32(sV + b * TILE);
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) umma_bf16(tmem, desc_k(aq, kk), desc_k(bk, kk), IDESC_S, kk > 0);
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) umma_bf16(tmem + 128, desc_k(ao, kk), desc_k(bv, kk), IDESC_S, kk > 0);
        tm1.pend = true;
        umma_commit(bar_mma1);
      }
      if (!track_wait_all(bar_mma1, tm1)) {
        if (tid == 0) report_status(status, FL_DEV_TIMEOUT_ACC_FULL);
        ok = false;
        break;
      }
      tc_fence_after();
      if (tid == 0 && next && j + 1 == w.n_kv) issue_qdo(wn);
      // ---- dS of query row r for keys kh * 64 .. + 63 of the tile, in two groups of 32,
      // each written (bf16 pairs) into the 16 S columns at 64 kh + 16 hf it has just read
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
          uint32_t dd[16];
#pragma unroll
          for (int c2 = 0; c2 < 16; ++c2) {
            float ds[2];
#pragma unroll
            for (int e = 0; e < 2; ++e) {
              const int c = 2 * c2 + e;
              const bool vis = u0 + 32 * hf + c < uend;
              const float pv = vis ? exp2_hw(fmaf(__uint_as_float(sr[c]), scale_log2, -lse2)) : 0.f;
              ds[e] = pv * (__uint_as_float(dr[c]) - dl);
            }
            dd[c2] = pack_bf16x2(ds[0], ds[1]);
          }
          tmem_st16(t_lane + kh * 64 + 16 * hf, dd);
        }
      }
      tmem_st_wait();
      tc_fence_before();
      __syncthreads();
      // ---- dQ += dS K_j (A from TMEM); then the tile after next into this buffer pair
      // once both products have read it
      if (tid == 0) {
        tc_fence_after();
        const uint32_t bk = smem_u32(sK + b * TILE);
#pragma unroll
        for (int kk = 0; kk < TB / 16; ++kk)
          umma_bf16_ts(tmem + 256, tmem + a_col(kk), desc_mn(bk, kk), IDESC_G, (j > 0 || kk > 0) ? 1u : 0u);
        tm2.pend = true;
        umma_commit(bar_mma2);
      }
      if (j + 1 == w.n_kv && kh < nreg && q_ok) {  // the query's rotary row, for the epilogue
        const int32_t* gp = kh == 0 ? gpos : gpos2;
        rope_load<HD>(rrow, rope_tab + (int64_t)(gp ? __ldg(gp + w.seg0 + q) : q) * E);
      }
      if (!track_wait_all(bar_mma2, tm2)) {
        if (tid == 0) report_status(status, FL_DEV_TIMEOUT_ACC_EMPTY);
        ok = false;
        break;
      }
      tc_fence_after();
      if (tid == 0) {
        if (j + 2 < w.n_kv) {
          issue_kv(w, j + 2, b);
        } else if (next) {  // pair b's last use in this unit: the next unit's tile of pair b
          if (b < wn.n_kv) issue_kv(wn, b, b);
          if (w.n_kv == 1 && wn.n_kv > 1) issue_kv(wn, 1, 1);  // pair 1 unused here
        }
      }
    }
    if (!ok) break;

    // ---- every product of the unit is complete: its dQ leaves while the next unit's tiles
    // load
    float lse2n = 0.f, dln = 0.f;
    if (next) row_stats(wn, lse2n, dln);
    // ---- dQ (scaled, rotated back): thread (r, kh) takes dims kh * HD/2 .. + HD/2 - 1 of
    // query row r, staged and written by bulk tensor stores (coalesced row stores for a
    // ragged last tile), the bias column sums taken from the staged rows
    {
      uint8_t* stage = sST;
      uint32_t vr[HD / 2];
#pragma unroll
      for (int c = 0; c < HD / 2; c += 32)
        tmem_ld32(t_lane + 256 + kh * (HD / 2) + c, *reinterpret_cast<uint32_t(*)[32]>(vr + c));
      tmem_ld_wait();
      float* v = reinterpret_cast<float*>(vr);
#pragma unroll
      for (int c = 0; c < HD / 2; ++c) v[c] = __uint_as_float(vr[c]) * scale;
      if (kh < nreg && q_ok) inverse_rope_row<HD>(v, rrow);  // rotary region kh
      // the staging tile is free once the previous bulk store has read it
      if (tid == 0) bulk_wait_read();
      __syncthreads();
#pragma unroll
      for (int c8 = 0; c8 < HD / 16; ++c8)
        *reinterpret_cast<uint4*>(stage_chunk<HD>(stage, r, kh * (HD / 16) + c8)) =
            make_uint4(pack_bf16x2(v[8 * c8], v[8 * c8 + 1]), pack_bf16x2(v[8 * c8 + 2], v[8 * c8 + 3]),
                       pack_bf16x2(v[8 * c8 + 4], v[8 * c8 + 5]), pack_bf16x2(v[8 * c8 + 6], v[8 * c8 + 7]));
      const int col = w.h * HD;
      const bool full = w.q0 + TB <= w.L;  // a whole tile of the segment: TMA stores
      if (full) fence_proxy_async_smem();
      __syncthreads();  // the tile is staged
      if (full && tid == 0) {
#pragma unroll
        for (int x = 0; x < NB; ++x) tma_store_2d(&tm_dqkv, stage + x * (TB * 128), col + 64 * x, w.seg0 + w.q0);
        bulk_commit();
      }
      if (w.db) staged_colsum<HD>(stage, min(TB, w.L - w.q0), w.db + col, tid);
      if (!full) {
#pragma unroll
        for (int i = 0; i < TB * CH / 256; ++i) {
          const int id = tid + 256 * i, row = id / CH, jc = id % CH;
          if (w.q0 + row < w.L)
            *reinterpret_cast<uint4*>(dqkv + ((int64_t)w.seg0 + w.q0 + row) * 3 * H + col + jc * 8) =
                *reinterpret_cast<const uint4*>(stage_chunk<HD>(stage, row, jc));
        }
      }
    }
    // the staged rows have been read and the dQ columns loaded before the next unit's
    // epilogue and products reuse them
    tc_fence_before();
    __syncthreads();
    u = un;
    w = wn;
    lse2 = lse2n;
    dl = dln;
  }
  if (tid == 0) bulk_wait_all();  // this CTA's bulk stores are complete before it leaves
  if (!ok && tid == 0) {  // a wait gave up: let what this CTA armed land before leaving
    track_drain(bar_qdo, tqdo);
    track_drain(bar_kv, tkv0);
    track_drain(bar_kv + 1, tkv1);
    track_drain(bar_mma1, tm1);
    track_drain(bar_mma2, tm2);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

template <int HD>
int launch_bwd_tc(int T, int nh, const void* qkv, const void* dout, const float* lse, const float* delta,
                  const int32_t* cu, const uint32_t* tiles, int n_tiles, const float* rope_tab, void* dqkv,
                  const AttnPrefix& pre, const AttnGlm& glm, float* dbias, int* status, cudaStream_t st,
                  int dbias_segs, int64_t dbias_rstride) {
  FL_CUDA_TRY(fl_func_smem((const void*)attn_bwd_dq_tc_kernel<HD>, BwdCfg<HD>::SMEM));
  FL_CUDA_TRY(fl_func_smem((const void*)attn_bwd_dkv_tc_kernel<HD, false>, BwdCfg<HD>::SMEM));
  FL_CUDA_TRY(fl_func_smem((const void*)attn_bwd_dkv_tc_kernel<HD, true>, BwdCfg<HD>::SMEM));
  const int H = nh * HD;
  CUtensorMap tq, tdo, tpk, tpv, tdq;
  if (int rc = fl_gemm::make_map(&tq, qkv, (uint64_t)3 * H, (uint64_t)T, 3 * (int64_t)H, 128)) return rc;
  if (int rc = fl_gemm::make_map(&tdq, dqkv, (uint64_t)3 * H, (uint64_t)T, 3 * (int64_t)H, 128)) return rc;
  if (int rc = fl_gemm::make_map(&tdo, dout, (uint64_t)H, (uint64_t)T, H, 128)) return rc;
  if (pre.len > 0) {
    if (int rc = fl_gemm::make_map(&tpk, pre.k, (uint64_t)H, (uint64_t)pre.len, H, 128)) return rc;
    if (int rc = fl_gemm::make_map(&tpv, pre.v, (uint64_t)H, (uint64_t)pre.len, H, 128)) return rc;
  } else {
    tpk = tq;
    tpv = tq;
  }
  const float scale = 1.f / sqrtf((float)HD);
  const float2* tab = reinterpret_cast<const float2*>(rope_tab);
  // persistent: one CTA per SM (512 TMEM columns each) walks the (tile, head) units
  const int n_units = n_tiles * nh;
  const int grid = n_units < fl_sm_count() ? n_units : fl_sm_count();
  if (n_units > 0) {
    FL_CUDA_TRY(fl_launch(attn_bwd_dq_tc_kernel<HD>, dim3(grid), dim3(256), BwdCfg<HD>::SMEM, st, tq, tdo, tpk, tpv,
                          tdq, T, H, cu, tiles, n_units, lse, delta, tab, scale, scale * LOG2E_B, pre.len, (bf16*)dqkv,
                          glm.ctx, glm.pos, glm.pos2, dbias, dbias_segs, dbias_rstride, status));
    FL_CUDA_TRY(fl_launch(attn_bwd_dkv_tc_kernel<HD, false>, dim3(grid), dim3(256), BwdCfg<HD>::SMEM, st, tq, tdo,
                          tpk, tpv, tdq, T, H, cu, tiles, n_tiles, n_units, 0, lse, delta, tab, scale, scale * LOG2E_B, 0,
                          (bf16*)dqkv, (float*)nullptr, (float*)nullptr, glm.ctx, glm.pos, glm.pos2, dbias,
                          dbias_segs, dbias_rstride, status));
  }
  if (pre.len > 0 && n_tiles > 0) {
    // the prefix keys of each head against slices of the query tiles, about one CTA per SM
    int nsplit = (fl_sm_count() + nh - 1) / nh;
    if (nsplit > n_tiles) nsplit = n_tiles;
    if (nsplit < 1) nsplit = 1;
    FL_CUDA_TRY(fl_launch(attn_bwd_dkv_tc_kernel<HD, true>, dim3(nsplit * nh), dim3(256), BwdCfg<HD>::SMEM, st, tq,
                          tdo, tpk, tpv, tdq, T, H, cu, tiles, n_tiles, nsplit * nh, nsplit, lse, delta, tab, scale,
                          scale * LOG2E_B, pre.len, (bf16*)dqkv, pre.dk, pre.dv, glm.ctx, glm.pos, glm.pos2,
                          (float*)nullptr, 0, (int64_t)0, status));
  }
  return FL_OK;
}

}  // namespace

int fl_launch_attn_bwd_tc(int T, int nh, int hd, const void* qkv, const void* dout, const float* lse,
                          const float* delta, const int32_t* cu, const uint32_t* tiles, int n_tiles,
                          const float* rope_tab, void* dqkv, const AttnPrefix& pre, const AttnGlm& glm, float* dbias,
                          int* status, cudaStream_t st, int dbias_segs, int64_t dbias_rstride) {
  if (hd == 128)
    return launch_bwd_tc<128>(T, nh, qkv, dout, lse, delta, cu, tiles, n_tiles, rope_tab, dqkv, pre, glm, dbias,
                              status, st, dbias_segs, dbias_rstride);
  if (hd == 64)
    return launch_bwd_tc<64>(T, nh, qkv, dout, lse, delta, cu, tiles, n_tiles, rope_tab, dqkv, pre, glm, dbias,
                             status, st, dbias_segs, dbias_rstride);
  return fl_internal_error(FL_ERR_UNSUPPORTED, "attention: head_dim %d", hd);
}
