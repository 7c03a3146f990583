// Persistent tcgen05 GEMM for sm_103a with fused epilogues.
//
// D[M,N] = epilogue(A . B^T): bf16 operands staged by TMA (128-byte swizzle) into a
// STAGES-deep shared-memory ring, one elected thread issues tcgen05.mma kind::f16
// (M=128, N=BN, K=16) into a double-buffered fp32 TMEM accumulator, and four
// epilogue warps drain TMEM with tcgen05.ld while the next tile's main loop runs.
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
#include <cuda.h>
#include <cstdio>
#include <mutex>

#include "../../include/flglm_kernels.h"
#include "common.cuh"
#include "ptx.cuh"

namespace {

constexpr int BM = 128;
constexpr int BK = 64;  // one 128-byte swizzle row of bf16
constexpr int UMMA_K = 16;
constexpr double L2_GROUP_BUDGET = 48.0 * (1 << 20);  // bytes of operand panels kept resident per group
constexpr int NUM_THREADS = 192;

template <int BN>
struct Cfg {
  static constexpr int STAGES = (BN == 256) ? 4 : 6;
  static constexpr int A_BYTES = BM * BK * 2;
  static constexpr int B_BYTES = BN * BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int TMEM_COLS = 2 * BN;  // double-buffered accumulator
  static constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 1024 /*align*/ + 256 /*barriers*/;
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
  const float2* rope_tab;  // [pos][rotary_dim/2]
  int rope_cols;           // 2*H: columns that hold q and k
  int head_dim, rotary_dim;
  int aux_f32, d_f32;
  const float *ln_mean, *ln_rstd, *ln_gamma, *ln_beta;  // residual = LayerNorm(aux) when ln_mean
};

FL_DEV void store_bf16x64(__nv_bfloat16* dst, const float* v) {
  uint4* d = reinterpret_cast<uint4*>(dst);
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    uint4 w;
    w.x = pack_bf16x2(v[8 * j + 0], v[8 * j + 1]);
    w.y = pack_bf16x2(v[8 * j + 2], v[8 * j + 3]);
    w.z = pack_bf16x2(v[8 * j + 4], v[8 * j + 5]);
    w.w = pack_bf16x2(v[8 * j + 6], v[8 * j + 7]);
    d[j] = w;
  }
}
FL_DEV void load_bf16x64(const __nv_bfloat16* src, float* v) {
  const uint4* s = reinterpret_cast<const uint4*>(src);
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    uint4 w = __ldg(s + j);
    float2 a = unpack_bf16x2(w.x), b = unpack_bf16x2(w.y), c = unpack_bf16x2(w.z), d = unpack_bf16x2(w.w);
    v[8 * j + 0] = a.x; v[8 * j + 1] = a.y; v[8 * j + 2] = b.x; v[8 * j + 3] = b.y;
    v[8 * j + 4] = c.x; v[8 * j + 5] = c.y; v[8 * j + 6] = d.x; v[8 * j + 7] = d.y;
  }
}

// Applies the epilogue to 64 consecutive columns [n0, n0+64) of row m.
FL_DEV void epilogue64(const Epi& e, int m, int n0, float* v) {
  if (e.bias) {
    const float4* b4 = reinterpret_cast<const float4*>(e.bias + n0);
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      float4 b = __ldg(b4 + j);
      v[4 * j] += b.x; v[4 * j + 1] += b.y; v[4 * j + 2] += b.z; v[4 * j + 3] += b.w;
    }
  }
  switch (e.mode) {
    case FL_EPI_BIAS_GELU: {
      __nv_bfloat16* u = e.aux_out + (int64_t)m * e.ld_aux_out + n0;
      store_bf16x64(u, v);
#pragma unroll
      for (int j = 0; j < 64; ++j) v[j] = gelu_tanh(v[j]);
      break;
    }
    case FL_EPI_BIAS_RESID:
    case FL_EPI_RESID: {
      float r[64];
      if (e.aux_f32) {
        const float4* a4 = reinterpret_cast<const float4*>(reinterpret_cast<const float*>(e.aux) + (int64_t)m * e.ld_aux + n0);
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const float4 q = __ldg(a4 + j);
          r[4 * j] = q.x; r[4 * j + 1] = q.y; r[4 * j + 2] = q.z; r[4 * j + 3] = q.w;
        }
      } else {
        load_bf16x64(e.aux + (int64_t)m * e.ld_aux + n0, r);
      }
      if (e.ln_mean) {  // residual = LayerNorm(aux), recomputed in fp32
        const float mu = __ldg(e.ln_mean + m), rs = __ldg(e.ln_rstd + m);
        const float4* g4 = reinterpret_cast<const float4*>(e.ln_gamma + n0);
        const float4* b4 = reinterpret_cast<const float4*>(e.ln_beta + n0);
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const float4 g = __ldg(g4 + j), b = __ldg(b4 + j);
          r[4 * j] = (r[4 * j] - mu) * rs * g.x + b.x;
          r[4 * j + 1] = (r[4 * j + 1] - mu) * rs * g.y + b.y;
          r[4 * j + 2] = (r[4 * j + 2] - mu) * rs * g.z + b.z;
          r[4 * j + 3] = (r[4 * j + 3] - mu) * rs * g.w + b.w;
        }
      }
#pragma unroll
      for (int j = 0; j < 64; ++j) v[j] = fmaf(e.alpha, r[j], v[j]);
      break;
    }
    case FL_EPI_GELU_BWD: {
      float u[64];
      load_bf16x64(e.aux + (int64_t)m * e.ld_aux + n0, u);
#pragma unroll
      for (int j = 0; j < 64; ++j) v[j] *= gelu_tanh_grad(u[j]);
      break;
    }
    case FL_EPI_BIAS_ROPE: {
      if (n0 < e.rope_cols && (n0 % e.head_dim) == 0) {
        const int half = e.rotary_dim >> 1;
        const float2* tab = e.rope_tab + (int64_t)__ldg(e.pos + m) * half;
        if (half == 32) {
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            float2 cs = __ldg(tab + i);
            float x1 = v[i], x2 = v[i + 32];
            v[i] = x1 * cs.x - x2 * cs.y;
            v[i + 32] = x2 * cs.x + x1 * cs.y;
          }
        } else {  // half == 16
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            float2 cs = __ldg(tab + i);
            float x1 = v[i], x2 = v[i + 16];
            v[i] = x1 * cs.x - x2 * cs.y;
            v[i + 16] = x2 * cs.x + x1 * cs.y;
          }
        }
      }
      break;
    }
    default:
      break;
  }
  if (e.mode == FL_EPI_ACCUM_F32) {
    float4* d = reinterpret_cast<float4*>(reinterpret_cast<float*>(e.D) + (int64_t)m * e.ldd + n0);
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      float4 o = d[j];
      o.x += v[4 * j]; o.y += v[4 * j + 1]; o.z += v[4 * j + 2]; o.w += v[4 * j + 3];
      d[j] = o;
    }
  } else if (e.mode == FL_EPI_STORE_F32 || e.d_f32) {
    float4* d = reinterpret_cast<float4*>(reinterpret_cast<float*>(e.D) + (int64_t)m * e.ldd + n0);
#pragma unroll
    for (int j = 0; j < 16; ++j) d[j] = make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
  } else {
    store_bf16x64(reinterpret_cast<__nv_bfloat16*>(e.D) + (int64_t)m * e.ldd + n0, v);
  }
}

// Tile order.  Tiles are taken in groups of `gsz` panels of one operand: along m
// (gsz m-blocks, m fastest) every group streams B once while its A panels stay in L2;
// along n the roles swap.  The host picks the side and size that minimise DRAM reads.
struct Raster {
  int gsz;
  int along_n;
};
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

template <int BN, bool A_MN, bool B_MN>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, Epi epi,
                   int M, int N, int K, Raster raster, int* status) {
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

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int num_m = (M + BM - 1) / BM;
  const int num_n = N / BN;
  const int num_tiles = num_m * num_n;
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
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
  }
  if (warp == 1) {
    tmem_alloc(tmem_holder, C::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------------ TMA producer
      int stage = 0;
      uint32_t phase = 0;
      uint32_t armed = 0, last_par = 0;  // per-stage bit masks for the teardown drain
      bool ok = true;
      for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x) {
        int mb, nb;
        tile_coords(tile, num_m, num_n, raster, mb, nb);
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
            tma_load_2d(a_dst, &tmA, &full[stage], k0, mb * BM);
          } else {
#pragma unroll
            for (int j = 0; j < BM / 64; ++j) tma_load_2d(a_dst + j * 64 * BK * 2, &tmA, &full[stage], mb * BM + 64 * j, k0);
          }
          if (!B_MN) {
            tma_load_2d(b_dst, &tmB, &full[stage], k0, nb * BN);
          } else {
#pragma unroll
            for (int j = 0; j < BN / 64; ++j) tma_load_2d(b_dst + j * 64 * BK * 2, &tmB, &full[stage], nb * BN + 64 * j, k0);
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
    const int row = quarter * 32 + lane;
    int local = 0;
    for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x, ++local) {
      int mb, nb;
      tile_coords(tile, num_m, num_n, raster, mb, nb);
      const int acc = local & 1;
      const uint32_t acc_par = (local >> 1) & 1;
      if (!mbar_wait(&acc_full[acc], acc_par)) {
        report_status(status, FL_DEV_TIMEOUT_ACC_FULL);
        break;
      }
      tc_fence_after();
      const int m = mb * BM + row;
      const uint32_t t_row = tmem_base + (uint32_t(quarter * 32) << 16) + acc * BN;
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 64) {
        uint32_t r0[32], r1[32];
        tmem_ld32(t_row + c0, r0);
        tmem_ld32(t_row + c0 + 32, r1);
        tmem_ld_wait();
        const int n0 = nb * BN + c0;
        if (m < M) {
          float v[64];
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            v[j] = __uint_as_float(r0[j]);
            v[32 + j] = __uint_as_float(r1[j]);
          }
          epilogue64(epi, m, n0, v);
        }
      }
      tc_fence_before();
      mbar_arrive(&acc_empty[acc]);
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

// ------------------------------------------------------------------ host side

typedef CUresult (*PFN_encodeTiled)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                    const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                    CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

PFN_encodeTiled get_encode_fn() {
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
int make_map(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer, int64_t ld, uint32_t box_outer) {
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

int num_sms() {
  static int n = 0;
  if (!n) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 148;
  }
  return n;
}

template <int BN, bool A_MN, bool B_MN>
int launch(const fl_gemm_args* a, const Epi& epi, int* status, cudaStream_t st) {
  using C = Cfg<BN>;
  auto kern = gemm_tc_kernel<BN, A_MN, B_MN>;
  static bool attr_set = false;  // per instantiation; the attribute is per device function
  if (!attr_set) {
    FL_CUDA_TRY(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM_BYTES));
    attr_set = true;
  }
  CUtensorMap ta, tb;
  int rc;
  // A(m,k): K-major -> [M rows, K inner]; MN-major -> [K rows, M inner]
  if (!A_MN) rc = make_map(&ta, a->A, a->K, a->M, a->lda, BM);
  else rc = make_map(&ta, a->A, a->M, a->K, a->lda, BK);
  if (rc) return rc;
  if (!B_MN) rc = make_map(&tb, a->B, a->K, a->N, a->ldb, BN);
  else rc = make_map(&tb, a->B, a->N, a->K, a->ldb, BK);
  if (rc) return rc;
  const int num_m = (a->M + BM - 1) / BM, num_n = a->N / BN;
  const int tiles = num_m * num_n;
  const int grid = tiles < num_sms() ? tiles : num_sms();
  // DRAM reads of the two orders: the grouped operand once, the other once per group
  const double pa = double(BM) * a->K * 2, pb = double(BN) * a->K * 2;
  int gm = (int)(L2_GROUP_BUDGET / pa), gn = (int)(L2_GROUP_BUDGET / pb);
  gm = gm < 1 ? 1 : (gm > num_m ? num_m : gm);
  gn = gn < 1 ? 1 : (gn > num_n ? num_n : gn);
  const double cost_m = pa * num_m + pb * num_n * ((num_m + gm - 1) / gm);
  const double cost_n = pb * num_n + pa * num_m * ((num_n + gn - 1) / gn);
  Raster r;
  r.along_n = cost_n < cost_m ? 1 : 0;
  r.gsz = r.along_n ? gn : gm;
  gemm_tc_kernel<BN, A_MN, B_MN><<<grid, NUM_THREADS, C::SMEM_BYTES, st>>>(ta, tb, epi, a->M, a->N, a->K, r, status);
  FL_CUDA_TRY(cudaGetLastError());
  return FL_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

}  // namespace

extern "C" int fl_k_gemm(const fl_gemm_args* a, int* status, void* stream) {
  if (!a || !a->A || !a->B || !a->D) return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: null pointer");
  if (a->M < 0 || a->N <= 0 || a->K <= 0) return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: bad sizes");
  if (a->M == 0) return FL_OK;
  if (a->N % 128) return fl_internal_error(FL_ERR_UNSUPPORTED, "gemm: N=%d is not a multiple of 128", a->N);
  if (a->epilogue < 0 || a->epilogue >= FL_EPI_COUNT) return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: epilogue");
  if ((a->lda % 8) || (a->ldb % 8) || (a->ldd % 8) || !aligned16(a->A) || !aligned16(a->B) || !aligned16(a->D))
    return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: leading dims must be multiples of 8 and pointers 16-byte aligned");
  if (a->a_mn_major && a->lda < a->M) return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: lda < M");
  if (!a->a_mn_major && a->lda < a->K) return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: lda < K");
  if (a->b_mn_major && a->ldb < a->N) return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: ldb < N");
  if (!a->b_mn_major && a->ldb < a->K) return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: ldb < K");
  if (a->a_mn_major && (a->M % 8)) return fl_internal_error(FL_ERR_UNSUPPORTED, "gemm: MN-major A needs M % 8 == 0");
  const int mode = a->epilogue;
  if ((mode == FL_EPI_BIAS_RESID || mode == FL_EPI_RESID || mode == FL_EPI_GELU_BWD) &&
      (!a->aux || (a->ld_aux % 8) || !aligned16(a->aux)))
    return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: epilogue needs an aligned aux tensor");
  if ((a->aux_dtype != FL_DT_BF16 && a->aux_dtype != FL_DT_F32) || (a->d_dtype != FL_DT_BF16 && a->d_dtype != FL_DT_F32))
    return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: aux/d dtype");
  if (a->aux_dtype == FL_DT_F32 && !(mode == FL_EPI_BIAS_RESID || mode == FL_EPI_RESID))
    return fl_internal_error(FL_ERR_UNSUPPORTED, "gemm: fp32 aux only for the residual epilogues");
  if (a->d_dtype == FL_DT_F32 && !(mode == FL_EPI_STORE || mode == FL_EPI_BIAS_RESID || mode == FL_EPI_RESID))
    return fl_internal_error(FL_ERR_UNSUPPORTED, "gemm: fp32 D only for STORE and the residual epilogues");
  if (a->ln_mean && (!a->ln_rstd || !a->ln_gamma || !a->ln_beta || !aligned16(a->ln_gamma) || !aligned16(a->ln_beta) ||
                     !(mode == FL_EPI_BIAS_RESID || mode == FL_EPI_RESID)))
    return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: LayerNorm residual needs mean, rstd, gamma, beta");
  if (mode == FL_EPI_BIAS_GELU && (!a->aux_out || (a->ld_aux_out % 8) || !aligned16(a->aux_out)))
    return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: GeLU epilogue needs aux_out");
  if (mode == FL_EPI_BIAS_ROPE) {
    if (!a->pos || !a->rope_tab || a->head_dim <= 0 || a->head_dim % 64 ||
        !(a->rotary_dim == 32 || a->rotary_dim == 64) || a->rotary_dim > a->head_dim)
      return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: RoPE epilogue arguments");
  }
  if (a->bias && !aligned16(a->bias)) return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: bias alignment");

  Epi e;
  e.mode = mode;
  e.bias = a->bias;
  e.aux = reinterpret_cast<const __nv_bfloat16*>(a->aux);
  e.ld_aux = a->ld_aux;
  e.alpha = a->alpha;
  e.aux_out = reinterpret_cast<__nv_bfloat16*>(a->aux_out);
  e.ld_aux_out = a->ld_aux_out;
  e.D = a->D;
  e.ldd = a->ldd;
  e.pos = a->pos;
  e.rope_tab = reinterpret_cast<const float2*>(a->rope_tab);
  e.rope_cols = 2 * a->n_heads * a->head_dim;
  e.head_dim = a->head_dim > 0 ? a->head_dim : 64;
  e.rotary_dim = a->rotary_dim;
  e.aux_f32 = a->aux_dtype == FL_DT_F32;
  e.d_f32 = a->d_dtype == FL_DT_F32 && mode != FL_EPI_ACCUM_F32;
  e.ln_mean = a->ln_mean;
  e.ln_rstd = a->ln_rstd;
  e.ln_gamma = a->ln_gamma;
  e.ln_beta = a->ln_beta;

  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  // Tile width: 256 columns unless 128 gives clearly fewer idle SM slots in the last wave.
  bool wide = (a->N % 256) == 0;
  if (wide) {
    const int sms = num_sms();
    const long t256 = (long)((a->M + BM - 1) / BM) * (a->N / 256);
    const long t128 = 2 * t256;
    const double eff256 = double(t256) / double(((t256 + sms - 1) / sms) * sms);
    const double eff128 = double(t128) / double(((t128 + sms - 1) / sms) * sms);
    if (eff128 > eff256 * 1.15) wide = false;
  }
  const bool amn = a->a_mn_major != 0, bmn = a->b_mn_major != 0;
  if (!amn && !bmn) return wide ? launch<256, false, false>(a, e, status, st) : launch<128, false, false>(a, e, status, st);
  if (!amn && bmn) return wide ? launch<256, false, true>(a, e, status, st) : launch<128, false, true>(a, e, status, st);
  if (amn && bmn) return wide ? launch<256, true, true>(a, e, status, st) : launch<128, true, true>(a, e, status, st);
  return fl_internal_error(FL_ERR_UNSUPPORTED, "gemm: MN-major A with K-major B is not built");
}
