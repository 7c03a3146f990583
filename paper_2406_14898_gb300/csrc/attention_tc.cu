// Attention forward on the 5th-generation tensor cores, head_dim 64 or 128 (App. A:
// softmax(Q K'^T / sqrt(d_h)) V', K' / V' = optional P-tuning prefix then the segment's own
// keys, causal within the segment or with a bidirectional GLM context; §3.3 segments are
// never mixed), with both tile contractions on tcgen05 and their accumulators in TMEM.
//
// Persistent CTAs (4 warps, two per SM) walk the (128-query tile, head) units; the next
// unit's Q and first K / V tiles load while a unit's output is written.  Thread i owns
// query row i, which is TMEM lane i.  Per 128-key tile j:
//   TMA: K_j and V_j (128 rows x head_dim, 64-column 128-byte-swizzled boxes; Q once),
//        each on its own barrier;
//   S = Q K_j^T     -> TMEM columns [0, 128)   (tcgen05.mma, both operands in shared memory);
//        K_j's buffer is free once S is complete: K_{j+1} is loaded right away;
//   softmax: the thread's S row (masked max, exp2, row sum); P (bf16, two per 32-bit
//        column) is stored back into the first 64 columns of S; the O row is rescaled when
//        the running max moved;
//   O += P V_j      -> TMEM columns [128, 128 + head_dim) (A = P read from TMEM, V_j as an
//        MN-major operand); then V_{j+1} is loaded.
// Shared memory: three tiles (96 KB at head_dim 128); 256 TMEM columns: two CTAs per SM
// overlap each other's copies and softmax.  Every mbarrier wait is bounded (2 s): on
// expiry the CTA records a status code and leaves its remaining work undone.
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
constexpr int TB = 128;            // queries and keys per tile (UMMA M; N of S; K of P V)
constexpr int BOX = 64 * 128 * 2;  // one 64-column x 128-row bf16 box: 16 KB
constexpr float LOG2E_T = 1.4426950408889634f;
constexpr float LN2_T = 0.6931471805599453f;

template <int HD>
struct FwdCfg {
  static constexpr int NB = HD / 64;      // boxes per tile row
  static constexpr int TILE = NB * BOX;   // one 128 x HD bf16 tile
  // 3 tiles; at head_dim 64 padded so that no more than two CTAs (256 TMEM columns each)
  // share an SM
  static constexpr int USED = 3 * TILE + 1024 /*barriers, holder*/ + 1024 /*alignment*/;
  static constexpr int SMEM = USED > 80 * 1024 ? USED : 80 * 1024;
};

// K-major operand (rows x HD columns in 64-column swizzled boxes): descriptor of k-step kk.
FL_DEV uint64_t desc_kmajor(uint32_t base, int kk) {
  return smem_desc_sw128(base + (kk >> 2) * BOX + (kk & 3) * 32, 16, 1024);
}
// MN-major operand (K = the tile's 128 rows, N = its HD columns): descriptor of k-step kk.
FL_DEV uint64_t desc_mnmajor(uint32_t base, int kk) { return smem_desc_sw128(base + kk * 2048, BOX, 1024); }

template <int HD>
__global__ void __launch_bounds__(128) attn_fwd_tc_kernel(
    const __grid_constant__ CUtensorMap tm_qkv, const __grid_constant__ CUtensorMap tm_pk,
    const __grid_constant__ CUtensorMap tm_pv, int T, int H, int n_heads, const int32_t* __restrict__ cu,
    const uint32_t* __restrict__ tiles, int n_units, bf16* __restrict__ O, float* __restrict__ lse,
    float scale_log2, int Lp, const int32_t* __restrict__ ctxs, int* status) {
  constexpr int NB = FwdCfg<HD>::NB, TILE = FwdCfg<HD>::TILE;
  pdl_wait();  // the previous kernel on the stream has completed (see fl_launch)
  pdl_trigger();
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;
  uint8_t* sK = smem + TILE;
  uint8_t* sV = smem + 2 * TILE;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + 3 * TILE);
  uint64_t* bar_q = bars;
  uint64_t* bar_k = bars + 1;
  uint64_t* bar_v = bars + 2;
  uint64_t* bar_s = bars + 3;
  uint64_t* bar_pv = bars + 4;
  uint32_t* holder = reinterpret_cast<uint32_t*>(bars + 6);
  const int tid = threadIdx.x, warp = tid >> 5;
  const int npt = Lp > 0 ? 1 : 0;  // at most one prefix tile (Lp <= 128)

  // A work unit u is (entry u / n_heads of the 128-row tile list, head u % n_heads): the
  // list's longest segments first, each segment's tiles together (last tile first).
  struct Unit {
    int h, seg0, L, q0, clast, n_kv;
  };
  auto unit_t = [&](int u, uint32_t t) {
    Unit w;
    const int s = int(t >> 16), idx = int(t & 0xFFFFu);
    w.h = u % n_heads;
    w.seg0 = cu[s];
    w.L = cu[s + 1] - w.seg0;
    w.q0 = idx * TB;
    w.clast = (ctxs ? min(max(ctxs[s], 0), w.L) : 0) - 1;
    w.n_kv = npt + max(idx, w.clast >= 0 ? w.clast / TB : 0) + 1;
    return w;
  };
  auto unit = [&](int u) { return unit_t(u, tiles[u / n_heads]); };

  if (tid == 0) {
    for (int i = 0; i < 5; ++i) mbar_init(bars + i, 1);
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

  BarTrack tq, tk, tv, ts, tpv;
  // one elected thread: the key (part 0) or value (part 1) tile j of unit w into its buffer
  auto issue = [&](const Unit& w, int j, int part) {
    uint8_t* dst = part ? sV : sK;
    uint64_t* bar = part ? bar_v : bar_k;
    (part ? tv : tk).pend = true;
    mbar_arrive_expect_tx(bar, TILE);
    if (j < npt) {
      const CUtensorMap* m = part ? &tm_pv : &tm_pk;
#pragma unroll
      for (int b = 0; b < NB; ++b) tma_load_2d(dst + b * BOX, m, bar, w.h * HD + 64 * b, 0);
    } else {
      const int row = w.seg0 + (j - npt) * TB;
#pragma unroll
      for (int b = 0; b < NB; ++b)
        tma_load_2d(dst + b * BOX, &tm_qkv, bar, (1 + part) * H + w.h * HD + 64 * b, row);
    }
  };
  auto issue_unit = [&](const Unit& w) {  // Q and the first key / value tiles of a unit
    tq.pend = true;
    mbar_arrive_expect_tx(bar_q, TILE);
#pragma unroll
    for (int b = 0; b < NB; ++b) tma_load_2d(sQ + b * BOX, &tm_qkv, bar_q, w.h * HD + 64 * b, w.seg0 + w.q0);
    issue(w, 0, 0);
    issue(w, 0, 1);
  };

  constexpr uint32_t IDESC_S = umma_idesc_bf16(TB, TB, false, false);
  constexpr uint32_t IDESC_PV = umma_idesc_bf16(TB, HD, false, true);
  bool ok = true;
  int u = blockIdx.x;
  Unit w = u < n_units ? unit(u) : Unit{};
  Unit wn = u + (int)gridDim.x < n_units ? unit(u + gridDim.x) : Unit{};
  if (tid == 0 && u < n_units) issue_unit(w);
  while (u < n_units && ok) {
    const int q = w.q0 + tid;  // this thread's query row (inside the segment)
    const int un = u + gridDim.x, unn = un + gridDim.x;
    // the descriptor of the unit after next, read in two steps while products run
    Unit wnn = Unit{};
    uint32_t tnn = 0;
    float m_run = -INFINITY, l_run = 0.f;
    // every wait's outcome is agreed on by the whole CTA, so that all threads leave together
    if (!track_wait_all(bar_q, tq)) {
      if (tid == 0) report_status(status, FL_DEV_TIMEOUT_FULL);
      ok = false;
      break;
    }
    for (int j = 0; j < w.n_kv && ok; ++j) {
      if (!track_wait_all(bar_k, tk)) {
        if (tid == 0) report_status(status, FL_DEV_TIMEOUT_FULL);
        ok = false;
        break;
      }
      // ---- S = Q K_j^T (the previous P V, which read the S columns, has completed)
      if (tid == 0) {
        tc_fence_after();
        const uint32_t aq = smem_u32(sQ), bk = smem_u32(sK);
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk)
          umma_bf16(tmem, desc_kmajor(aq, kk), desc_kmajor(bk, kk), IDESC_S, kk > 0);
        ts.pend = true;
        umma_commit(bar_s);
      }
      if (j == 0 && unn < n_units) tnn = tiles[unn / n_heads];
      if (!track_wait_all(bar_s, ts)) {
        if (tid == 0) report_status(status, FL_DEV_TIMEOUT_ACC_FULL);
        ok = false;
        break;
      }
      tc_fence_after();
      if (tid == 0 && j + 1 < w.n_kv) issue(w, j + 1, 0);  // K_j has been read
      // ---- the thread's S row, read once (4 x 32 columns, one wait)
      const bool prefix = j < npt;
      const int kb = prefix ? 0 : (j - npt) * TB;  // first key of the tile inside its sequence
      const int klim = prefix ? Lp - 1 : min(w.L - 1, max(q, w.clast));  // last visible key
      const bool full = kb + TB - 1 <= klim;       // every key of the tile visible to this row
      uint32_t r[TB];
      tmem_ld32(t_s, *reinterpret_cast<uint32_t(*)[32]>(r));
      tmem_ld32(t_s + 32, *reinterpret_cast<uint32_t(*)[32]>(r + 32));
      tmem_ld32(t_s + 64, *reinterpret_cast<uint32_t(*)[32]>(r + 64));
      tmem_ld32(t_s + 96, *reinterpret_cast<uint32_t(*)[32]>(r + 96));
      tmem_ld_wait();
      // masked row max; invisible keys become -inf
      float mt = -INFINITY;
#pragma unroll
      for (int e = 0; e < TB; ++e) {
        float x = __uint_as_float(r[e]) * scale_log2;
        if (!full && kb + e > klim) x = -INFINITY;
        r[e] = __float_as_uint(x);
        mt = fmaxf(mt, x);
      }
      const float m_new = fmaxf(m_run, mt);
      const float mref = m_new == -INFINITY ? 0.f : m_new;
      const float corr = exp2f(m_run - mref);  // 0 on the first tile (m_run = -inf)
      // ---- P = exp2(S - m), bf16 pairs (keys 2c, 2c + 1 in column c) into S's columns [0, 64)
      float lt = 0.f;
#pragma unroll
      for (int c = 0; c < TB / 2; ++c) {
        const float p0 = exp2f(__uint_as_float(r[2 * c]) - mref);
        const float p1 = exp2f(__uint_as_float(r[2 * c + 1]) - mref);
        lt += p0 + p1;
        r[c] = pack_bf16x2(p0, p1);
      }
      tmem_st32(t_s, *reinterpret_cast<uint32_t(*)[32]>(r));
      tmem_st32(t_s + 32, *reinterpret_cast<uint32_t(*)[32]>(r + 32));
      l_run = l_run * corr + lt;
      m_run = m_new;
      // ---- rescale the O rows when a row max moved (not before the first P V); TMEM
      // loads and stores are warp-wide, so the whole warp takes part (factor 1 elsewhere)
      if (j > 0 && __any_sync(0xffffffffu, corr != 1.f)) {
#pragma unroll 1
        for (int c = 0; c < HD; c += 32) {
          uint32_t o[32];
          tmem_ld32(t_o + c, o);
          tmem_ld_wait();
#pragma unroll
          for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * corr);
          tmem_st32(t_o + c, o);
        }
      }
      tmem_st_wait();
      tc_fence_before();
      if (!track_wait_all(bar_v, tv)) {
        if (tid == 0) report_status(status, FL_DEV_TIMEOUT_FULL);
        ok = false;
        break;
      }
      // ---- O += P V_j
      if (tid == 0) {
        tc_fence_after();
        const uint32_t bv = smem_u32(sV);
#pragma unroll
        for (int kk = 0; kk < TB / 16; ++kk)
          umma_bf16_ts(tmem + 128, tmem + kk * 8, desc_mnmajor(bv, kk), IDESC_PV, (j > 0 || kk > 0) ? 1u : 0u);
        tpv.pend = true;
        umma_commit(bar_pv);
      }
      if (j == 0 && unn < n_units) wnn = unit_t(unn, tnn);
      if (!track_wait_all(bar_pv, tpv)) {
        if (tid == 0) report_status(status, FL_DEV_TIMEOUT_ACC_EMPTY);
        ok = false;
        break;
      }
      tc_fence_after();
      if (tid == 0 && j + 1 < w.n_kv) issue(w, j + 1, 1);  // V_j has been read
    }
    if (!ok) break;
    // ---- every product of the unit is complete and Q / K / V are free: the next unit's
    // first tiles load while this one's O leaves
    if (tid == 0 && un < n_units) issue_unit(wn);
    // ---- O / l and the log-sum-exp (every lane reads TMEM, all of the row at once; rows
    // past the segment end store nothing)
    const bool valid = q < w.L;
    const float inv = valid ? 1.f / l_run : 0.f;
    bf16* orow = O + (int64_t)(w.seg0 + (valid ? q : 0)) * H + w.h * HD;
    {
      uint32_t o[HD];
#pragma unroll
      for (int c = 0; c < HD; c += 32) tmem_ld32(t_o + c, *reinterpret_cast<uint32_t(*)[32]>(o + c));
      tmem_ld_wait();
      if (valid) {
#pragma unroll
        for (int v = 0; v < HD / 8; ++v)
          *reinterpret_cast<uint4*>(orow + 8 * v) = make_uint4(
              pack_bf16x2(__uint_as_float(o[8 * v]) * inv, __uint_as_float(o[8 * v + 1]) * inv),
              pack_bf16x2(__uint_as_float(o[8 * v + 2]) * inv, __uint_as_float(o[8 * v + 3]) * inv),
              pack_bf16x2(__uint_as_float(o[8 * v + 4]) * inv, __uint_as_float(o[8 * v + 5]) * inv),
              pack_bf16x2(__uint_as_float(o[8 * v + 6]) * inv, __uint_as_float(o[8 * v + 7]) * inv));
      }
    }
    if (valid) lse[(int64_t)w.h * T + w.seg0 + q] = (m_run + log2f(l_run)) * LN2_T;
    // the O columns are read before the next unit's first P V overwrites them
    tc_fence_before();
    u = un;
    w = wn;
    wn = wnn;
  }
  if (!ok && tid == 0) {  // a wait gave up: let what this CTA armed land before leaving
    track_drain(bar_q, tq);
    track_drain(bar_k, tk);
    track_drain(bar_v, tv);
    track_drain(bar_s, ts);
    track_drain(bar_pv, tpv);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, 256);
  }
}

template <int HD>
int launch_fwd_tc(int T, int nh, const void* qkv, const int32_t* cu, const uint32_t* tiles, int n_tiles, void* o,
                  float* lse, const AttnPrefix& pre, const AttnGlm& glm, int* status, cudaStream_t st) {
  FL_CUDA_TRY(fl_func_smem((const void*)attn_fwd_tc_kernel<HD>, FwdCfg<HD>::SMEM));
  const int H = nh * HD;
  CUtensorMap tq, tpk, tpv;
  if (int rc = fl_gemm::make_map(&tq, qkv, (uint64_t)3 * H, (uint64_t)T, 3 * (int64_t)H, 128)) return rc;
  if (pre.len > 0) {
    if (int rc = fl_gemm::make_map(&tpk, pre.k, (uint64_t)H, (uint64_t)pre.len, H, 128)) return rc;
    if (int rc = fl_gemm::make_map(&tpv, pre.v, (uint64_t)H, (uint64_t)pre.len, H, 128)) return rc;
  } else {
    tpk = tq;
    tpv = tq;
  }
  const float scale_log2 = (1.f / sqrtf((float)HD)) * LOG2E_T;
  // persistent: two CTAs per SM walk the (tile, head) units
  const int n_units = n_tiles * nh;
  const int grid = n_units < 2 * fl_sm_count() ? n_units : 2 * fl_sm_count();
  FL_CUDA_TRY(fl_launch(attn_fwd_tc_kernel<HD>, dim3(grid), dim3(128), FwdCfg<HD>::SMEM, st, tq, tpk, tpv, T, H, nh,
                        cu, tiles, n_units, (bf16*)o, lse, scale_log2, pre.len, glm.ctx, status));
  return FL_OK;
}

}  // namespace

int fl_launch_attn_fwd_tc(int T, int nh, int hd, const void* qkv, const int32_t* cu, const uint32_t* tiles,
                          int n_tiles, void* o, float* lse, const AttnPrefix& pre, const AttnGlm& glm, int* status,
                          cudaStream_t st) {
  if (hd == 128) return launch_fwd_tc<128>(T, nh, qkv, cu, tiles, n_tiles, o, lse, pre, glm, status, st);
  if (hd == 64) return launch_fwd_tc<64>(T, nh, qkv, cu, tiles, n_tiles, o, lse, pre, glm, status, st);
  return fl_internal_error(FL_ERR_UNSUPPORTED, "attention: head_dim %d", hd);
}
