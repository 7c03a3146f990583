// Persistent tcgen05 GEMM for sm_103a with fused epilogues.
//
// D[M,N] = epilogue(A . B^T): bf16 operands staged by TMA (128-byte swizzle) into a
// STAGES-deep shared-memory ring, one elected thread issues tcgen05.mma kind::f16
// (M=128, N=BN, K=16) into a double-buffered fp32 TMEM accumulator, and four
// epilogue warps drain TMEM with tcgen05.ld while the next tile's main loop runs.
// An epilogue warp owns 32 rows of the tile (its TMEM lane quarter); it moves each 32x64
// fp32 chunk through 8 KB of shared memory so that, row by row, its lanes handle
// consecutive column pairs and every global load and store of the epilogue is coalesced.
//
// Operand majorness is a template parameter: K-major operands are [rows, K] row-major
// (one TMA box of 64 x rows per stage), MN-major operands are [K, rows] row-major
// (rows/64 boxes of 64 x BK per stage).  The three GEMM families of a transformer
// block map onto it as
//   forward  X[T,K]  . W[N,K]^T          A K-major,  B K-major
//   dgrad    dY[T,N] . W[N,K]            A K-major,  B MN-major
//   wgrad    dY[T,N]^T . X[T,K]          A MN-major, B MN-major  (fp32 accumulate)
//
// Warp roles (192 threads): warp 0 TMA producer, warp 1 TMEM owner + MMA issuer,
// warps 2..5 epilogue (warp w reads TMEM lanes 32*(w%4) .. +31).
#pragma once
#include <cuda.h>
#include <atomic>
#include <cstdio>
#include <mutex>

#include "../../include/flglm_kernels.h"
#include "common.cuh"
#include "ptx.cuh"

namespace fl_gemm {

constexpr int BM = 128;
constexpr int BK = 64;  // one 128-byte swizzle row of bf16
constexpr int UMMA_K = 16;
// Bytes of operand panels kept resident per raster group: 32 MB while K <= 8192, 48 MB for
// the longer panels of K = 12288 / 16384 (measured on GB300 at the stack26 shapes: DRAM
// reads of the up-projection 827 -> 554 MB and the weight gradients 8-10 us faster at 32
// MB; the K = 16384 / 12288 data gradients and down-projection best at 48 MB).
constexpr double L2_GROUP_BUDGET = 48.0 * (1 << 20);
constexpr double L2_GROUP_BUDGET_SHORT_K = 32.0 * (1 << 20);
constexpr int NUM_THREADS = 192;

template <int BN>
struct Cfg {
  static constexpr int STAGES = (BN == 256) ? 4 : 6;
  static constexpr int A_BYTES = BM * BK * 2;
  static constexpr int B_BYTES = BN * BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int TMEM_COLS = 2 * BN;  // double-buffered accumulator
  static constexpr int STAGING_BYTES = 4 * 32 * 64 * 4;  // one 32x64 fp32 chunk per epilogue warp
  static constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 256 /*barriers*/ + STAGING_BYTES + 1024 /*align*/;
};

struct Epi {
  int mode;
  const float* bias;
  const __nv_bfloat16* aux;
  int64_t ld_aux;
  float alpha;
  __nv_bfloat16* aux_out;
  int64_t ld_aux_out;
  void* D;
  int64_t ldd;
  const int32_t* pos;
  const int32_t* pos2;     // GLM block positions (second rotary half) or null
  const float2* rope_tab;  // [pos][rotary_dim/2]
  int rope_cols;           // 2*H: columns that hold q and k
  int head_dim, rotary_dim;
  int aux_f32, d_f32;
  const float *ln_mean, *ln_rstd, *ln_gamma, *ln_beta;  // residual = LayerNorm(aux) when ln_mean
  float *adam_m, *adam_v;
  float lr, b1, b2, eps, wd, inv_bc1, inv_bc2;
  float* colsum;  // GELU_BWD: column sums of D added here (bias gradient of the up-projection)
  // launch of several problems: element offsets of problem r's pointers from problem 0's
  // (entry 0 unused, always 0): D, aux, aux_out, bias / colsum, the per-row arrays (pos,
  // pos2, LayerNorm statistics), LayerNorm gain / shift, Adam moments
  int64_t o_d[FL_GEMM_MAX_BATCH], o_aux[FL_GEMM_MAX_BATCH], o_aux_out[FL_GEMM_MAX_BATCH],
      o_bias[FL_GEMM_MAX_BATCH], o_row[FL_GEMM_MAX_BATCH], o_lnp[FL_GEMM_MAX_BATCH], o_adam[FL_GEMM_MAX_BATCH];
};

// The operands of the problems of one launch: A and B of problem r with their leading
// dimensions (tensor maps are built from these on the host).
struct Problems {
  int n;
  const void* A[FL_GEMM_MAX_BATCH];
  const void* B[FL_GEMM_MAX_BATCH];
  int64_t lda[FL_GEMM_MAX_BATCH], ldb[FL_GEMM_MAX_BATCH];
};

// Tensor maps of the A and B operands of up to FL_GEMM_MAX_BATCH problems (a kernel
// parameter: TMA reads each map from parameter space).
struct GemmMaps {
  CUtensorMap a[FL_GEMM_MAX_BATCH];
  CUtensorMap b[FL_GEMM_MAX_BATCH];
};

// Epilogue families: each kernel instantiation carries only its family's code, which keeps
// the kernel small enough for the instruction cache (the MMA-issuing warp shares it).
enum { FAM_PLAIN = 0, FAM_GELU = 1, FAM_RESID = 2, FAM_ROPE = 3, FAM_ADAMW = 4, FAM_COUNT };
__host__ __device__ constexpr int family_of(int mode) {
  return (mode == FL_EPI_BIAS_GELU || mode == FL_EPI_GELU_BWD) ? FAM_GELU
         : (mode == FL_EPI_BIAS_RESID || mode == FL_EPI_RESID) ? FAM_RESID
         : mode == FL_EPI_BIAS_ROPE                            ? FAM_ROPE
         : mode == FL_EPI_ADAMW                                ? FAM_ADAMW
                                                               : FAM_PLAIN;
}

FL_DEV float4 ld_quad(const float* p) { return __ldg(reinterpret_cast<const float4*>(p)); }
FL_DEV float4 ld_quad(const __nv_bfloat16* p) {
  const uint2 u = __ldg(reinterpret_cast<const uint2*>(p));
  const float2 a = unpack_bf16x2(u.x), b = unpack_bf16x2(u.y);
  return make_float4(a.x, a.y, b.x, b.y);
}
FL_DEV void st_quad(float* p, float4 v) { *reinterpret_cast<float4*>(p) = v; }
FL_DEV void st_quad(__nv_bfloat16* p, float4 v) {
  *reinterpret_cast<uint2*>(p) = make_uint2(pack_bf16x2(v.x, v.y), pack_bf16x2(v.z, v.w));
}

// Epilogue of one 32-row x 64-column chunk held in `stage` (row r, float4 slot j stored at
// slot j ^ (r & 15)).  Half-warp h = lane / 16 takes the rows of parity h; lane l handles
// columns n0 + 4 (l % 16) .. + 3, so every warp-wide access covers two 64-column rows
// (256 B of bf16 or 512 B of fp32).  Rows go in batches of RB row pairs: all global loads of
// a batch are issued before any of its arithmetic.
// Entry r of a per-problem offset array (constant indices only: no local copy of the
// parameter struct).
FL_DEV int64_t prob_off(const int64_t (&o)[FL_GEMM_MAX_BATCH], int r) {
  static_assert(FL_GEMM_MAX_BATCH == 4, "prob_off selects among four problems");
  return r == 0 ? 0 : r == 1 ? o[1] : r == 2 ? o[2] : o[3];
}

template <int FAM>
FL_DEV void epilogue_chunk(const Epi& e, int r, const float* stage, int row0, int rows, int n0, int lane) {
  // problem r of a multi-problem launch: element offsets of its pointers (0 for r = 0)
  const int64_t od = prob_off(e.o_d, r), oaux = prob_off(e.o_aux, r), oauxo = prob_off(e.o_aux_out, r),
                ob = prob_off(e.o_bias, r), orow = prob_off(e.o_row, r), olnp = prob_off(e.o_lnp, r),
                oad = prob_off(e.o_adam, r);
  constexpr int RB = (FAM == FAM_GELU || FAM == FAM_ROPE) ? 16 : 8;  // row pairs per batch
  const int h = lane >> 4, cl = lane & 15;
  const int n = n0 + 4 * cl;
  const float4 bias = e.bias ? ld_quad(e.bias + ob + n) : make_float4(0.f, 0.f, 0.f, 0.f);
  const bool ln = FAM == FAM_RESID && e.ln_mean != nullptr;
  float4 lng = make_float4(1.f, 1.f, 1.f, 1.f), lnb = make_float4(0.f, 0.f, 0.f, 0.f);
  if (ln) {
    lng = ld_quad(e.ln_gamma + olnp + n);
    lnb = ld_quad(e.ln_beta + olnp + n);
  }
  // RoPE: a chunk of q/k columns that holds rotary dims.  Dims [0, rotary_dim) of a head
  // turn by pos; with GLM block positions, dims [rotary_dim, 2 rotary_dim) turn by pos2
  // (same frequencies and pairing).  Each rotary region is 32 or 64 columns aligned inside
  // the 64-column chunk, so a column's partner is pair_xor lanes away.
  const int hoff = n0 % e.head_dim;
  const bool rope = FAM == FAM_ROPE && n0 < e.rope_cols && (hoff == 0 || e.pos2 != nullptr);
  const int half = e.rotary_dim >> 1;
  const int pair_xor = half >> 2;  // lane distance of the partner columns (8 or 4)
  const int col = 4 * cl;
  const int region = (hoff + col) / e.rotary_dim;  // 0: rotated by pos, 1: by pos2
  const int rcol = hoff + col - region * e.rotary_dim;
  const bool rotated = rope && (region == 0 || (region == 1 && e.pos2 != nullptr));
  const int32_t* rpos_src = region == 0 ? e.pos : e.pos2;
  const bool first = rcol < half;
  const bool gelu_bwd = FAM == FAM_GELU && e.mode == FL_EPI_GELU_BWD;
  const bool colsum = FAM == FAM_GELU && gelu_bwd && e.colsum != nullptr;
  float cs[4] = {0.f, 0.f, 0.f, 0.f};  // this lane's column sums over its rows of the chunk
  const bool accum = FAM == FAM_PLAIN && e.mode == FL_EPI_ACCUM_F32;
  const bool out_f32 = e.mode == FL_EPI_STORE_F32 || e.d_f32;
#pragma unroll 1
  for (int pb = 0; 2 * pb < rows; pb += RB) {
    float4 acc[RB], aux[RB], am[RB], av[RB];
    float rmu[RB], rrs[RB];
    int rpos[RB];
    // ---- loads of the batch
#pragma unroll
    for (int i = 0; i < RB; ++i) {
      const int rr = 2 * (pb + i) + h;
      acc[i] = *reinterpret_cast<const float4*>(stage + (rr & 31) * 64 + 4 * (cl ^ (rr & 15)));
      aux[i] = am[i] = av[i] = make_float4(0.f, 0.f, 0.f, 0.f);
      rmu[i] = 0.f;
      rrs[i] = 1.f;
      rpos[i] = 0;
      if (rr < rows) {
        const int m = row0 + rr;
        const int64_t off = (int64_t)m * e.ldd + n + od;
        if constexpr (FAM == FAM_RESID) {
          const int64_t oa = (int64_t)m * e.ld_aux + n;
          aux[i] = e.aux_f32 ? ld_quad(reinterpret_cast<const float*>(e.aux) + oaux + oa) : ld_quad(e.aux + oaux + oa);
          if (ln) {
            rmu[i] = __ldg(e.ln_mean + orow + m);
            rrs[i] = __ldg(e.ln_rstd + orow + m);
          }
        } else if constexpr (FAM == FAM_ADAMW) {
          aux[i] = *reinterpret_cast<const float4*>(reinterpret_cast<const float*>(e.D) + off);  // w
          am[i] = *reinterpret_cast<const float4*>(e.adam_m + (off - od + oad));
          av[i] = *reinterpret_cast<const float4*>(e.adam_v + (off - od + oad));
        } else {
          if (gelu_bwd) aux[i] = ld_quad(e.aux + oaux + (int64_t)m * e.ld_aux + n);
          if (accum) aux[i] = *reinterpret_cast<const float4*>(reinterpret_cast<const float*>(e.D) + off);
          if (FAM == FAM_ROPE && rotated) rpos[i] = __ldg(rpos_src + orow + m);
        }
      }
    }
    // ---- arithmetic and stores of the batch
#pragma unroll
    for (int i = 0; i < RB; ++i) {
      const int rr = 2 * (pb + i) + h;
      float y[4] = {acc[i].x + bias.x, acc[i].y + bias.y, acc[i].z + bias.z, acc[i].w + bias.w};
      if (FAM == FAM_ROPE && rope) {  // uniform across the warp: every lane takes part in the shuffles
        float p[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) p[q] = __shfl_xor_sync(0xffffffffu, y[q], pair_xor);
        if (rotated && rr < rows) {
          const int ii = first ? rcol : rcol - half;
          const float2* tab = e.rope_tab + (int64_t)rpos[i] * half + ii;
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const float2 cs = __ldg(tab + q);
            y[q] = first ? y[q] * cs.x - p[q] * cs.y : y[q] * cs.x + p[q] * cs.y;
          }
        }
      }
      if (rr >= rows) continue;
      const int m = row0 + rr;
      const int64_t off = (int64_t)m * e.ldd + n + od;
      const float a4[4] = {aux[i].x, aux[i].y, aux[i].z, aux[i].w};
      if constexpr (FAM == FAM_RESID) {
        const float g4[4] = {lng.x, lng.y, lng.z, lng.w}, b4[4] = {lnb.x, lnb.y, lnb.z, lnb.w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float r = ln ? (a4[q] - rmu[i]) * rrs[i] * g4[q] + b4[q] : a4[q];  // LayerNorm(aux) in fp32
          y[q] = fmaf(e.alpha, r, y[q]);
        }
      } else if constexpr (FAM == FAM_GELU) {
        if (gelu_bwd) {
#pragma unroll
          for (int q = 0; q < 4; ++q) y[q] *= gelu_tanh_grad(a4[q]);
          if (colsum) {
#pragma unroll
            for (int q = 0; q < 4; ++q) cs[q] += y[q];
          }
        } else {
          st_quad(e.aux_out + oauxo + (int64_t)m * e.ld_aux_out + n, make_float4(y[0], y[1], y[2], y[3]));
#pragma unroll
          for (int q = 0; q < 4; ++q) y[q] = gelu_tanh(y[q]);
        }
      }
      if constexpr (FAM == FAM_ADAMW) {
        // AdamW on the four weights with g = y: the formula of adamw_kernel
        float w[4] = {aux[i].x, aux[i].y, aux[i].z, aux[i].w};
        float mm[4] = {am[i].x, am[i].y, am[i].z, am[i].w};
        float vv[4] = {av[i].x, av[i].y, av[i].z, av[i].w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          mm[q] = e.b1 * mm[q] + (1.f - e.b1) * y[q];
          vv[q] = e.b2 * vv[q] + (1.f - e.b2) * y[q] * y[q];
          const float mh = mm[q] * e.inv_bc1;
          const float vh = vv[q] * e.inv_bc2;
          w[q] = w[q] - e.lr * (mh / (sqrtf(vh) + e.eps) + e.wd * w[q]);
        }
        st_quad(reinterpret_cast<float*>(e.D) + off, make_float4(w[0], w[1], w[2], w[3]));
        st_quad(e.adam_m + (off - od + oad), make_float4(mm[0], mm[1], mm[2], mm[3]));
        st_quad(e.adam_v + (off - od + oad), make_float4(vv[0], vv[1], vv[2], vv[3]));
        st_quad(e.aux_out + oauxo + (int64_t)m * e.ld_aux_out + n, make_float4(w[0], w[1], w[2], w[3]));
      } else if (accum) {
        st_quad(reinterpret_cast<float*>(e.D) + off, make_float4(a4[0] + y[0], a4[1] + y[1], a4[2] + y[2], a4[3] + y[3]));
      } else if (out_f32) {
        st_quad(reinterpret_cast<float*>(e.D) + off, make_float4(y[0], y[1], y[2], y[3]));
      } else {
        st_quad(reinterpret_cast<__nv_bfloat16*>(e.D) + off, make_float4(y[0], y[1], y[2], y[3]));
      }
    }
  }
  if (colsum) {  // the two half-warps hold the same columns for rows of either parity
#pragma unroll
    for (int q = 0; q < 4; ++q) cs[q] += __shfl_xor_sync(0xffffffffu, cs[q], 16);
    if (h == 0 && rows > 0) red_add_v4(e.colsum + ob + n, cs[0], cs[1], cs[2], cs[3]);
  }
}

// Tile order.  Tiles are taken in groups of `gsz` panels of one operand: along m
// (gsz m-blocks, m fastest) every group streams B once while its A panels stay in L2;
// along n the roles swap.  The host picks the side and size that minimise DRAM reads.
struct Raster {
  int gsz;
  int along_n;
};
// Problem r of a batched launch and the tile's coordinates inside it: the problems' tile
// ranges follow each other, each in its own raster order.
FL_DEV void batch_tile(int tile, int num_m, int num_n, Raster rs, int& r, int& mb, int& nb);

FL_DEV void tile_coords(int tile, int num_m, int num_n, Raster r, int& mb, int& nb) {
  if (!r.along_n) {
    const int group = r.gsz * num_n;
    const int g = tile / group;
    const int first = g * r.gsz;
    const int gm = min(num_m - first, r.gsz);
    const int local = tile - g * group;
    mb = first + local % gm;
    nb = local / gm;
  } else {
    const int group = r.gsz * num_m;
    const int g = tile / group;
    const int first = g * r.gsz;
    const int gn = min(num_n - first, r.gsz);
    const int local = tile - g * group;
    nb = first + local % gn;
    mb = local / gn;
  }
}

FL_DEV void batch_tile(int tile, int num_m, int num_n, Raster rs, int& r, int& mb, int& nb) {
  const int per = num_m * num_n;
  r = tile / per;
  tile_coords(tile - r * per, num_m, num_n, rs, mb, nb);
}

template <int BN, bool A_MN, bool B_MN, int FAM>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    gemm_tc_kernel(const __grid_constant__ GemmMaps maps, Epi epi, int M, int N, int K, int batch, Raster raster,
                   int* status) {
  using C = Cfg<BN>;
  constexpr int STAGES = C::STAGES;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + STAGES * C::A_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * C::STAGE_BYTES);
  uint64_t* full = bars;
  uint64_t* empty = bars + STAGES;
  uint64_t* acc_full = bars + 2 * STAGES;
  uint64_t* acc_empty = acc_full + 2;
  uint64_t* drain = acc_empty + 2;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(drain + 1);
  float* staging = reinterpret_cast<float*>(smem + STAGES * C::STAGE_BYTES + 256);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int num_m = (M + BM - 1) / BM;
  const int num_n = N / BN;
  const int num_tiles = batch * num_m * num_n;
  const int num_k = (K + BK - 1) / BK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&acc_full[a], 1);
      mbar_init(&acc_empty[a], 128);
    }
    mbar_init(drain, 1);
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    for (int r = 0; r < batch; ++r) {
      tma_prefetch_desc(&maps.a[r]);
      tma_prefetch_desc(&maps.b[r]);
    }
  }
  if (warp == 1) {
    tmem_alloc(tmem_holder, C::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;
  pdl_wait();  // the previous kernel's outputs (operands, epilogue inputs) are complete
  pdl_trigger();

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------------ TMA producer
      int stage = 0;
      uint32_t phase = 0;
      uint32_t armed = 0, last_par = 0;  // per-stage bit masks for the teardown drain
      bool ok = true;
      for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x) {
        int r, mb, nb;
        batch_tile(tile, num_m, num_n, raster, r, mb, nb);
        const CUtensorMap* tmA = &maps.a[r];
        const CUtensorMap* tmB = &maps.b[r];
        for (int kb = 0; kb < num_k; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1)) {
            report_status(status, FL_DEV_TIMEOUT_EMPTY);
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&full[stage], C::STAGE_BYTES);
          armed |= 1u << stage;
          last_par = (last_par & ~(1u << stage)) | (phase << stage);
          const int k0 = kb * BK;
          uint8_t* a_dst = sA + stage * C::A_BYTES;
          uint8_t* b_dst = sB + stage * C::B_BYTES;
          if (!A_MN) {
            tma_load_2d(a_dst, tmA, &full[stage], k0, mb * BM);
          } else {
#pragma unroll
            for (int j = 0; j < BM / 64; ++j) tma_load_2d(a_dst + j * 64 * BK * 2, tmA, &full[stage], mb * BM + 64 * j, k0);
          }
          if (!B_MN) {
            tma_load_2d(b_dst, tmB, &full[stage], k0, nb * BN);
          } else {
#pragma unroll
            for (int j = 0; j < BN / 64; ++j) tma_load_2d(b_dst + j * 64 * BK * 2, tmB, &full[stage], nb * BN + 64 * j, k0);
          }
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      // Drain: every armed stage's copies must have landed before shared memory is released.
      for (int s = 0; s < STAGES; ++s)
        if (armed & (1u << s))
          if (!mbar_wait(&full[s], (last_par >> s) & 1)) report_status(status, FL_DEV_TIMEOUT_DRAIN);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------------------ MMA issuer
      constexpr uint32_t IDESC = umma_idesc_bf16(BM, BN, A_MN, B_MN);
      int stage = 0;
      uint32_t phase = 0;
      int local = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x, ++local) {
        const int acc = local & 1;
        const uint32_t acc_par = (local >> 1) & 1;
        if (!mbar_wait(&acc_empty[acc], acc_par ^ 1)) {
          report_status(status, FL_DEV_TIMEOUT_ACC_EMPTY);
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * BN;
        for (int kb = 0; kb < num_k; ++kb) {
          if (!mbar_wait(&full[stage], phase)) {
            report_status(status, FL_DEV_TIMEOUT_FULL);
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_base = smem_u32(sA + stage * C::A_BYTES);
          const uint32_t b_base = smem_u32(sB + stage * C::B_BYTES);
#pragma unroll
          for (int kk = 0; kk < BK / UMMA_K; ++kk) {
            // K-major: next 16 elements are 32 bytes further along the swizzled row.
            // MN-major: next 16 k-rows are 16 * 128 bytes further.
            const uint64_t adesc = A_MN ? smem_desc_sw128(a_base + kk * 2048, BK * 128, 1024)
                                        : smem_desc_sw128(a_base + kk * 32, 16, 1024);
            const uint64_t bdesc = B_MN ? smem_desc_sw128(b_base + kk * 2048, BK * 128, 1024)
                                        : smem_desc_sw128(b_base + kk * 32, 16, 1024);
            umma_bf16(d_tmem, adesc, bdesc, IDESC, (kb | kk) != 0 ? 1u : 0u);
          }
          umma_commit(&empty[stage]);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (ok) umma_commit(&acc_full[acc]);
      }
      // Drain: all MMAs issued by this thread complete before TMEM is released.
      umma_commit(drain);
      if (!mbar_wait(drain, 0)) report_status(status, FL_DEV_TIMEOUT_DRAIN);
    }
  } else {
    // -------------------------------------------------------------- epilogue warps
    const int quarter = warp & 3;
    float* stage = staging + (warp - 2) * 32 * 64;
    float4* my = reinterpret_cast<float4*>(stage + lane * 64);
    int local = 0;
    for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x, ++local) {
      int r, mb, nb;
      batch_tile(tile, num_m, num_n, raster, r, mb, nb);
      const int acc = local & 1;
      const uint32_t acc_par = (local >> 1) & 1;
      if (!mbar_wait(&acc_full[acc], acc_par)) {
        report_status(status, FL_DEV_TIMEOUT_ACC_FULL);
        break;
      }
      tc_fence_after();
      const int row0 = mb * BM + quarter * 32;
      const int rows = M - row0 < 32 ? M - row0 : 32;  // may be <= 0 for the ragged last tile
      const uint32_t t_row = tmem_base + (uint32_t(quarter * 32) << 16) + acc * BN;
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 64) {
        uint32_t r0[32], r1[32];
        tmem_ld32(t_row + c0, r0);
        tmem_ld32(t_row + c0 + 32, r1);
        tmem_ld_wait();
        if (c0 + 64 == BN) {  // accumulator fully read: the MMA may reuse it
          tc_fence_before();
          mbar_arrive(&acc_empty[acc]);
        }
        // this lane's row -> shared memory, float4 slot j at j ^ (row & 15)
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          my[j ^ (lane & 15)] = make_float4(__uint_as_float(r0[4 * j]), __uint_as_float(r0[4 * j + 1]),
                                            __uint_as_float(r0[4 * j + 2]), __uint_as_float(r0[4 * j + 3]));
          my[(8 + j) ^ (lane & 15)] = make_float4(__uint_as_float(r1[4 * j]), __uint_as_float(r1[4 * j + 1]),
                                                  __uint_as_float(r1[4 * j + 2]), __uint_as_float(r1[4 * j + 3]));
        }
        __syncwarp();
        if (rows > 0) epilogue_chunk<FAM>(epi, r, stage, row0, rows, nb * BN + c0, lane);
        __syncwarp();
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_base, C::TMEM_COLS);
  }
}

// ------------------------------------------------------------------ CTA-pair kernel
// A cluster of two CTAs on two SMs computes one 256 x 256 tile with tcgen05.mma
// .cta_group::2.  Each CTA stages its own 128 rows of A and 128 columns of B (32 KB per
// k-block, against 48 KB for a 128 x 256 tile on one SM, which leaves room for a 6-deep
// ring); the even CTA issues 256 x 256 x 16 MMAs that read both CTAs' stages and write
// accumulator rows 0..127 into its own TMEM and rows 128..255 into the odd CTA's; each
// CTA's four epilogue warps drain their own half exactly as in gemm_tc_kernel.
// Barriers: both producers' loads complete on the even CTA's full[s]; the MMA commits
// arrive on empty[s] and acc_full[a] of both CTAs; every epilogue warp of the pair
// arrives once on the even CTA's acc_empty[a].
constexpr int PAIR_BM = 256, PAIR_BN = 256;
struct CfgPair {
  static constexpr int STAGES = 6;
  static constexpr int A_BYTES = 128 * BK * 2;  // this CTA's 128 rows of A
  static constexpr int B_BYTES = 128 * BK * 2;  // this CTA's 128 columns of B
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int TMEM_COLS = 2 * PAIR_BN;  // double-buffered 256-column accumulator
  static constexpr int STAGING_BYTES = 4 * 32 * 64 * 4;
  static constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 256 /*barriers*/ + STAGING_BYTES + 1024 /*align*/;
};

template <bool A_MN, bool B_MN, int FAM>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    gemm_pair_kernel(const __grid_constant__ GemmMaps maps, Epi epi, int M, int N, int K, int batch, Raster raster,
                     int* status) {
  using C = CfgPair;
  constexpr int STAGES = C::STAGES;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + STAGES * C::A_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * C::STAGE_BYTES);
  uint64_t* full = bars;
  uint64_t* empty = bars + STAGES;
  uint64_t* acc_full = bars + 2 * STAGES;
  uint64_t* acc_empty = acc_full + 2;
  uint64_t* drain = acc_empty + 2;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(drain + 1);
  float* staging = reinterpret_cast<float*>(smem + STAGES * C::STAGE_BYTES + 256);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  const int pair = blockIdx.x >> 1, n_pairs = gridDim.x >> 1;
  const int num_m = (M + PAIR_BM - 1) / PAIR_BM;
  const int num_n = N / PAIR_BN;
  const int num_tiles = batch * num_m * num_n;
  const int num_k = (K + BK - 1) / BK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);   // the even CTA's producer (expect_tx of both CTAs' bytes)
      mbar_init(&empty[s], 1);  // one MMA commit
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&acc_full[a], 1);
      mbar_init(&acc_empty[a], 8);  // four epilogue warps in each CTA
    }
    mbar_init(drain, 1);
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    for (int r = 0; r < batch; ++r) {
      tma_prefetch_desc(&maps.a[r]);
      tma_prefetch_desc(&maps.b[r]);
    }
  }
  if (warp == 1) {
    tmem_alloc_pair(tmem_holder, C::TMEM_COLS);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync();  // both CTAs' barriers initialised and TMEM allocated
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;
  pdl_wait();  // the previous kernel's outputs (operands, epilogue inputs) are complete
  pdl_trigger();

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------------ TMA producer (both CTAs)
      const uint32_t full0 = mapa_shared(smem_u32(full), 0);  // the even CTA's full[0]
      int stage = 0;
      uint32_t phase = 0;
      uint32_t armed = 0, last_par = 0;  // per-stage bit masks for the teardown drain
      bool ok = true;
      for (int tile = pair; tile < num_tiles && ok; tile += n_pairs) {
        int r, mb, nb;
        batch_tile(tile, num_m, num_n, raster, r, mb, nb);
        const CUtensorMap* tmA = &maps.a[r];
        const CUtensorMap* tmB = &maps.b[r];
        const int m0 = mb * PAIR_BM + int(rank) * 128, n0 = nb * PAIR_BN + int(rank) * 128;
        for (int kb = 0; kb < num_k; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1)) {
            report_status(status, FL_DEV_TIMEOUT_EMPTY);
            ok = false;
            break;
          }
          if (leader) mbar_arrive_expect_tx(&full[stage], 2 * C::STAGE_BYTES);
          armed |= 1u << stage;
          last_par = (last_par & ~(1u << stage)) | (phase << stage);
          const uint32_t fb = full0 + 8u * stage;
          const int k0 = kb * BK;
          uint8_t* a_dst = sA + stage * C::A_BYTES;
          uint8_t* b_dst = sB + stage * C::B_BYTES;
          if (!A_MN) {
            tma_load_2d_pair(a_dst, tmA, fb, k0, m0);
          } else {
            tma_load_2d_pair(a_dst, tmA, fb, m0, k0);
            tma_load_2d_pair(a_dst + 64 * BK * 2, tmA, fb, m0 + 64, k0);
          }
          if (!B_MN) {
            tma_load_2d_pair(b_dst, tmB, fb, k0, n0);
          } else {
            tma_load_2d_pair(b_dst, tmB, fb, n0, k0);
            tma_load_2d_pair(b_dst + 64 * BK * 2, tmB, fb, n0 + 64, k0);
          }
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      // Drain: a stage loaded in phase p is released (empty phase p completes) only after
      // the MMAs that read it, and so after its copies landed.
      for (int s = 0; s < STAGES; ++s)
        if (armed & (1u << s))
          if (!mbar_wait(&empty[s], (last_par >> s) & 1)) report_status(status, FL_DEV_TIMEOUT_DRAIN);
    }
  } else if (warp == 1) {
    if (leader && lane == 0) {
      // ------------------------------------------------------------ MMA issuer (even CTA)
      constexpr uint32_t IDESC = umma_idesc_bf16(PAIR_BM, PAIR_BN, A_MN, B_MN);
      int stage = 0;
      uint32_t phase = 0;
      int local = 0;
      bool ok = true;
      for (int tile = pair; tile < num_tiles && ok; tile += n_pairs, ++local) {
        const int acc = local & 1;
        const uint32_t acc_par = (local >> 1) & 1;
        if (!mbar_wait(&acc_empty[acc], acc_par ^ 1)) {
          report_status(status, FL_DEV_TIMEOUT_ACC_EMPTY);
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * PAIR_BN;
        for (int kb = 0; kb < num_k; ++kb) {
          if (!mbar_wait(&full[stage], phase)) {
            report_status(status, FL_DEV_TIMEOUT_FULL);
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_base = smem_u32(sA + stage * C::A_BYTES);
          const uint32_t b_base = smem_u32(sB + stage * C::B_BYTES);
#pragma unroll
          for (int kk = 0; kk < BK / UMMA_K; ++kk) {
            const uint64_t adesc = A_MN ? smem_desc_sw128(a_base + kk * 2048, BK * 128, 1024)
                                        : smem_desc_sw128(a_base + kk * 32, 16, 1024);
            const uint64_t bdesc = B_MN ? smem_desc_sw128(b_base + kk * 2048, BK * 128, 1024)
                                        : smem_desc_sw128(b_base + kk * 32, 16, 1024);
            umma_bf16_pair(d_tmem, adesc, bdesc, IDESC, (kb | kk) != 0 ? 1u : 0u);
          }
          umma_commit_pair(&empty[stage], 3);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (ok) umma_commit_pair(&acc_full[acc], 3);
      }
      // Drain: all MMAs issued by this thread (and their arrivals) complete before the pair
      // releases TMEM and shared memory.
      umma_commit_pair(drain, 1);
      if (!mbar_wait(drain, 0)) report_status(status, FL_DEV_TIMEOUT_DRAIN);
    }
  } else {
    // -------------------------------------------------------------- epilogue warps (both CTAs)
    const int quarter = warp & 3;
    float* stage = staging + (warp - 2) * 32 * 64;
    float4* my = reinterpret_cast<float4*>(stage + lane * 64);
    const uint32_t acc_empty0 = mapa_shared(smem_u32(acc_empty), 0);
    int local = 0;
    for (int tile = pair; tile < num_tiles; tile += n_pairs, ++local) {
      int r, mb, nb;
      batch_tile(tile, num_m, num_n, raster, r, mb, nb);
      const int acc = local & 1;
      const uint32_t acc_par = (local >> 1) & 1;
      if (!mbar_wait(&acc_full[acc], acc_par)) {
        report_status(status, FL_DEV_TIMEOUT_ACC_FULL);
        break;
      }
      tc_fence_after();
      const int row0 = mb * PAIR_BM + int(rank) * 128 + quarter * 32;
      const int rows = M - row0 < 32 ? M - row0 : 32;  // may be <= 0 for the ragged last tile
      const uint32_t t_row = tmem_base + (uint32_t(quarter * 32) << 16) + acc * PAIR_BN;
#pragma unroll 1
      for (int c0 = 0; c0 < PAIR_BN; c0 += 64) {
        uint32_t r0[32], r1[32];
        tmem_ld32(t_row + c0, r0);
        tmem_ld32(t_row + c0 + 32, r1);
        tmem_ld_wait();
        if (c0 + 64 == PAIR_BN) {  // accumulator fully read: the MMA may reuse it
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_cluster(acc_empty0 + 8u * acc);
        }
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          my[j ^ (lane & 15)] = make_float4(__uint_as_float(r0[4 * j]), __uint_as_float(r0[4 * j + 1]),
                                            __uint_as_float(r0[4 * j + 2]), __uint_as_float(r0[4 * j + 3]));
          my[(8 + j) ^ (lane & 15)] = make_float4(__uint_as_float(r1[4 * j]), __uint_as_float(r1[4 * j + 1]),
                                                  __uint_as_float(r1[4 * j + 2]), __uint_as_float(r1[4 * j + 3]));
        }
        __syncwarp();
        if (rows > 0) epilogue_chunk<FAM>(epi, r, stage, row0, rows, nb * PAIR_BN + c0, lane);
        __syncwarp();
      }
    }
  }

  tc_fence_before();
  cluster_sync();  // neither CTA leaves while the pair's MMAs or arrivals may still touch it
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, C::TMEM_COLS);
  }
}

// ------------------------------------------------------------------ host side

typedef CUresult (*PFN_encodeTiled)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                    const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                    CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

inline PFN_encodeTiled get_encode_fn() {
  static PFN_encodeTiled fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_encodeTiled>(p);
  });
  return fn;
}

// 2-D bf16 tensor [outer, inner] (inner contiguous, row stride ld elements), box {64, box_outer}.
inline int make_map(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer, int64_t ld, uint32_t box_outer) {
  PFN_encodeTiled enc = get_encode_fn();
  if (!enc) return fl_internal_error(FL_ERR_CUDA, "cuTensorMapEncodeTiled is not available");
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {cuuint64_t(ld) * 2};
  cuuint32_t box[2] = {64, box_outer};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS)
    return fl_internal_error(FL_ERR_INVALID_ARG, "tensor map encode failed (%d): inner %llu outer %llu ld %lld", (int)r,
                             (unsigned long long)inner, (unsigned long long)outer, (long long)ld);
  return FL_OK;
}

inline int num_sms() { return fl_sm_count(); }

// Row-group raster that minimises DRAM reads for tiles of bm x bn (see Raster).
inline Raster pick_raster(int M, int N, int K, int bm, int bn) {
  const int num_m = (M + bm - 1) / bm, num_n = N / bn;
  const double pa = double(bm) * K * 2, pb = double(bn) * K * 2;
  const double budget = K <= 8192 ? L2_GROUP_BUDGET_SHORT_K : L2_GROUP_BUDGET;
  int gm = (int)(budget / pa), gn = (int)(budget / pb);
  gm = gm < 1 ? 1 : (gm > num_m ? num_m : gm);
  gn = gn < 1 ? 1 : (gn > num_n ? num_n : gn);
  const double cost_m = pa * num_m + pb * num_n * ((num_m + gm - 1) / gm);
  const double cost_n = pb * num_n + pa * num_m * ((num_n + gn - 1) / gn);
  Raster r;
  r.along_n = cost_n < cost_m ? 1 : 0;
  r.gsz = r.along_n ? gn : gm;
  return r;
}

template <int BN, bool A_MN, bool B_MN, int FAM>
int launch(const fl_gemm_args* a, const Problems& pr, const Epi& epi, int* status, cudaStream_t st) {
  using C = Cfg<BN>;
  auto kern = gemm_tc_kernel<BN, A_MN, B_MN, FAM>;
  FL_CUDA_TRY(fl_func_smem((const void*)kern, C::SMEM_BYTES));
  GemmMaps maps;
  const int batch = pr.n;
  for (int r = 0; r < batch; ++r) {
    int rc;
    // A(m,k): K-major -> [M rows, K inner]; MN-major -> [K rows, M inner]
    if (!A_MN) rc = make_map(&maps.a[r], pr.A[r], a->K, a->M, pr.lda[r], BM);
    else rc = make_map(&maps.a[r], pr.A[r], a->M, a->K, pr.lda[r], BK);
    if (rc) return rc;
    if (!B_MN) rc = make_map(&maps.b[r], pr.B[r], a->K, a->N, pr.ldb[r], BN);
    else rc = make_map(&maps.b[r], pr.B[r], a->N, a->K, pr.ldb[r], BK);
    if (rc) return rc;
  }
  const int num_m = (a->M + BM - 1) / BM, num_n = a->N / BN;
  const int tiles = batch * num_m * num_n;
  const int grid = tiles < num_sms() ? tiles : num_sms();
  const Raster r = pick_raster(a->M, a->N, a->K, BM, BN);
  FL_CUDA_TRY(fl_launch(gemm_tc_kernel<BN, A_MN, B_MN, FAM>, dim3(grid), dim3(NUM_THREADS), C::SMEM_BYTES, st, maps,
                        epi, a->M, a->N, a->K, batch, r, status));
  return FL_OK;
}

// CTA pairs the current device keeps resident at once for the pair kernel (0 if it cannot
// run there); queried once per device (each of the first 64 devices caches its answer).
template <bool A_MN, bool B_MN, int FAM>
int pair_slots() {
  constexpr int MAX_DEV = 64;
  static std::atomic<int> cache[MAX_DEV];  // slots + 1; 0: not queried yet
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  const bool cached = dev >= 0 && dev < MAX_DEV;
  if (cached) {
    const int c = cache[dev].load(std::memory_order_relaxed);
    if (c > 0) return c - 1;
  }
  auto kern = gemm_pair_kernel<A_MN, B_MN, FAM>;
  int slots = 0;
  if (fl_func_smem((const void*)kern, CfgPair::SMEM_BYTES) == cudaSuccess) {
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.gridDim = dim3(2 * num_sms());
    cfg.blockDim = dim3(NUM_THREADS);
    cfg.dynamicSmemBytes = CfgPair::SMEM_BYTES;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) == cudaSuccess && n > 0) slots = n;
  }
  cudaGetLastError();  // a refused query leaves the single-SM kernel in use
  if (cached) cache[dev].store(slots + 1, std::memory_order_relaxed);
  return slots;
}

template <bool A_MN, bool B_MN, int FAM>
int launch_pair(const fl_gemm_args* a, const Problems& pr, const Epi& epi, int* status, cudaStream_t st) {
  auto kern = gemm_pair_kernel<A_MN, B_MN, FAM>;
  const int slots = pair_slots<A_MN, B_MN, FAM>();
  if (slots <= 0) return fl_internal_error(FL_ERR_CUDA, "gemm: the CTA-pair kernel cannot be resident");
  GemmMaps maps;
  const int batch = pr.n;
  for (int r = 0; r < batch; ++r) {
    int rc;
    // each CTA loads 128 rows of A and 128 columns of B per k-block
    if (!A_MN) rc = make_map(&maps.a[r], pr.A[r], a->K, a->M, pr.lda[r], 128);
    else rc = make_map(&maps.a[r], pr.A[r], a->M, a->K, pr.lda[r], BK);
    if (rc) return rc;
    if (!B_MN) rc = make_map(&maps.b[r], pr.B[r], a->K, a->N, pr.ldb[r], 128);
    else rc = make_map(&maps.b[r], pr.B[r], a->N, a->K, pr.ldb[r], BK);
    if (rc) return rc;
  }
  const int tiles = batch * ((a->M + PAIR_BM - 1) / PAIR_BM) * (a->N / PAIR_BN);
  const int pairs = tiles < slots ? tiles : slots;
  const Raster r = pick_raster(a->M, a->N, a->K, PAIR_BM, PAIR_BN);
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // see pdl_wait
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.gridDim = dim3(2 * pairs);
  cfg.blockDim = dim3(NUM_THREADS);
  cfg.dynamicSmemBytes = CfgPair::SMEM_BYTES;
  cfg.stream = st;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  FL_CUDA_TRY(cudaLaunchKernelEx(&cfg, kern, maps, epi, a->M, a->N, a->K, batch, r, status));
  return FL_OK;
}

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

// Every (layout, family) pair for the CTA-pair kernel and both single-SM tile widths; the three operand layouts are
// instantiated in separate translation units so that the build compiles them in parallel.
#define FL_GEMM_INSTANTIATE(AMN, BMN)                                                              \
  template int pair_slots<AMN, BMN, FAM_PLAIN>();                                                      \
  template int pair_slots<AMN, BMN, FAM_GELU>();                                                       \
  template int pair_slots<AMN, BMN, FAM_RESID>();                                                      \
  template int pair_slots<AMN, BMN, FAM_ROPE>();                                                       \
  template int pair_slots<AMN, BMN, FAM_ADAMW>();                                                      \
  template int launch_pair<AMN, BMN, FAM_PLAIN>(const fl_gemm_args*, const Problems&, const Epi&, int*, cudaStream_t); \
  template int launch_pair<AMN, BMN, FAM_GELU>(const fl_gemm_args*, const Problems&, const Epi&, int*, cudaStream_t);  \
  template int launch_pair<AMN, BMN, FAM_RESID>(const fl_gemm_args*, const Problems&, const Epi&, int*, cudaStream_t); \
  template int launch_pair<AMN, BMN, FAM_ROPE>(const fl_gemm_args*, const Problems&, const Epi&, int*, cudaStream_t);  \
  template int launch_pair<AMN, BMN, FAM_ADAMW>(const fl_gemm_args*, const Problems&, const Epi&, int*, cudaStream_t); \
  template int launch<256, AMN, BMN, FAM_PLAIN>(const fl_gemm_args*, const Problems&, const Epi&, int*, cudaStream_t); \
  template int launch<128, AMN, BMN, FAM_PLAIN>(const fl_gemm_args*, const Problems&, const Epi&, int*, cudaStream_t); \
  template int launch<256, AMN, BMN, FAM_GELU>(const fl_gemm_args*, const Problems&, const Epi&, int*, cudaStream_t);  \
  template int launch<128, AMN, BMN, FAM_GELU>(const fl_gemm_args*, const Problems&, const Epi&, int*, cudaStream_t);  \
  template int launch<256, AMN, BMN, FAM_RESID>(const fl_gemm_args*, const Problems&, const Epi&, int*, cudaStream_t); \
  template int launch<128, AMN, BMN, FAM_RESID>(const fl_gemm_args*, const Problems&, const Epi&, int*, cudaStream_t); \
  template int launch<256, AMN, BMN, FAM_ROPE>(const fl_gemm_args*, const Problems&, const Epi&, int*, cudaStream_t);  \
  template int launch<128, AMN, BMN, FAM_ROPE>(const fl_gemm_args*, const Problems&, const Epi&, int*, cudaStream_t);  \
  template int launch<256, AMN, BMN, FAM_ADAMW>(const fl_gemm_args*, const Problems&, const Epi&, int*, cudaStream_t); \
  template int launch<128, AMN, BMN, FAM_ADAMW>(const fl_gemm_args*, const Problems&, const Epi&, int*, cudaStream_t);

}  // namespace fl_gemm

