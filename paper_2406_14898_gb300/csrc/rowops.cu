// HBM-bound kernels of the server step: LayerNorm forward/backward (a CTA per row,
// 128-bit loads), bias-gradient column sums, AdamW over the flat fp32 arena,
// client pack/unpack, per-call packing metadata and the seeded parameter init.
#include <cstdio>
#include <mutex>

#include "../../include/flglm_kernels.h"
#include "common.cuh"
#include "kernels.cuh"
#include "ptx.cuh"

namespace {

int sm_count() {
  return fl_sm_count();
}

FL_DEV float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

FL_DEV void unpack8(const uint4& w, float* f) {
  float2 a = unpack_bf16x2(w.x), b = unpack_bf16x2(w.y), c = unpack_bf16x2(w.z), d = unpack_bf16x2(w.w);
  f[0] = a.x; f[1] = a.y; f[2] = b.x; f[3] = b.y; f[4] = c.x; f[5] = c.y; f[6] = d.x; f[7] = d.y;
}

FL_DEV uint4 pack8(const float* f) {
  uint4 w;
  w.x = pack_bf16x2(f[0], f[1]);
  w.y = pack_bf16x2(f[2], f[3]);
  w.z = pack_bf16x2(f[4], f[5]);
  w.w = pack_bf16x2(f[6], f[7]);
  return w;
}

// ------------------------------------------------------------------ typed 8-element chunks
template <typename T>
FL_DEV void load8(const T* base, int64_t chunk, float* f);
template <>
FL_DEV void load8<__nv_bfloat16>(const __nv_bfloat16* base, int64_t chunk, float* f) {
  unpack8(__ldg(reinterpret_cast<const uint4*>(base) + chunk), f);
}
template <>
FL_DEV void load8<float>(const float* base, int64_t chunk, float* f) {
  const float4 a = __ldg(reinterpret_cast<const float4*>(base) + 2 * chunk);
  const float4 b = __ldg(reinterpret_cast<const float4*>(base) + 2 * chunk + 1);
  f[0] = a.x; f[1] = a.y; f[2] = a.z; f[3] = a.w; f[4] = b.x; f[5] = b.y; f[6] = b.z; f[7] = b.w;
}

// ------------------------------------------------------------------ LayerNorm
// Each row is read from HBM exactly once; the row statistics are block reductions.

// Sum of (a, b) over the block; `red` is a [2][32] shared buffer, `par` alternates between
// consecutive calls so that one barrier per call suffices.
FL_DEV float2 block_sum2(float a, float b, float2 (*red)[32], int par) {
  a = warp_sum(a);
  b = warp_sum(b);
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
  if (lane == 0) red[par][w] = make_float2(a, b);
  __syncthreads();
  float2 r = make_float2(0.f, 0.f);
  for (int i = 0; i < nw; ++i) {
    const float2 v = red[par][i];
    r.x += v.x;
    r.y += v.y;
  }
  return r;
}

// Forward: persistent CTAs of H/16 (CH = 2) or H/8 (CH = 1) threads, each thread CH chunks of 8 elements
// (chunk c + k * blockDim.x) of every row.  The CTA walks rows blockIdx.x, + gridDim.x, ...
// and keeps the next LN_STAGES of them in flight: one elected thread copies each whole row
// into a shared-memory stage with one bulk copy (cp.async.bulk, completion on the stage's
// mbarrier) and refills the stage as soon as every thread has read it.  Three CTAs per SM
// at H = 4096 (fp32 rows: 4 x 16 KB of stages each) keep 12 rows in flight per SM.  The
// statistics are two block reductions (mean, then the centred variance).  Every wait is
// bounded: on expiry the CTA records a status code and stops.
constexpr int LN_STAGES = 4;

// After a stage wait gave up at iteration `it`: the elected thread waits (bounded) for every
// row copy still in flight into the CTA's NS stages (the next row of each stage, if the
// schedule issued it), so that none lands after the CTA has left.
FL_DEV void ln_drain(uint64_t* full, int NS, int it, int T) {
  for (int s = 0; s < NS; ++s) {
    const int it2 = ((it - s + NS - 1) / NS) * NS + s;  // next iteration that uses stage s
    if (blockIdx.x + (int64_t)it2 * gridDim.x < T) mbar_wait(full + s, (it2 / NS) & 1);
  }
}

template <typename TX, int CH>
__global__ void __launch_bounds__(256) ln_fwd_bulk_kernel(int T, int H, const TX* __restrict__ x,
                                                          const float* __restrict__ gamma,
                                                          const float* __restrict__ beta, float eps,
                                                          __nv_bfloat16* __restrict__ y, float* __restrict__ mean,
                                                          float* __restrict__ rstd, int* status) {
  extern __shared__ __align__(128) uint8_t ln_smem[];
  pdl_wait();  // the previous kernel on the stream has completed (see fl_launch)
  pdl_trigger();
  const uint32_t row_bytes = (uint32_t)H * sizeof(TX);
  uint64_t* full = reinterpret_cast<uint64_t*>(ln_smem + LN_STAGES * row_bytes);
  __shared__ float red[2][8];
  const int c = threadIdx.x, nt = blockDim.x;
  const int lane = c & 31, w = c >> 5, nw = nt >> 5;
  if (c == 0) {
    for (int i = 0; i < LN_STAGES; ++i) mbar_init(full + i, 1);
    fence_mbar_init();
    for (int i = 0; i < LN_STAGES; ++i) {
      const int row = blockIdx.x + i * gridDim.x;
      if (row < T) {
        mbar_arrive_expect_tx(full + i, row_bytes);
        bulk_load(ln_smem + i * row_bytes, x + (int64_t)row * H, row_bytes, full + i);
      }
    }
  }
  float gg[CH][8], bt[CH][8];
#pragma unroll
  for (int k = 0; k < CH; ++k) {
    load8<float>(gamma, c + k * nt, gg[k]);
    load8<float>(beta, c + k * nt, bt[k]);
  }
  __syncthreads();
  for (int it = 0;; ++it) {
    const int row = blockIdx.x + it * gridDim.x;
    if (row >= T) break;
    const int st = it % LN_STAGES;
    if (!__syncthreads_and(mbar_wait(full + st, (it / LN_STAGES) & 1))) {
      if (c == 0) {
        report_status(status, FL_DEV_TIMEOUT_FULL);
        ln_drain(full, LN_STAGES, it, T);
      }
      break;
    }
    const TX* xr = reinterpret_cast<const TX*>(ln_smem + st * row_bytes);
    float v[CH][8];
#pragma unroll
    for (int k = 0; k < CH; ++k) {
      if constexpr (sizeof(TX) == 4) {
        const float4 a = reinterpret_cast<const float4*>(xr)[2 * (c + k * nt)];
        const float4 b = reinterpret_cast<const float4*>(xr)[2 * (c + k * nt) + 1];
        v[k][0] = a.x; v[k][1] = a.y; v[k][2] = a.z; v[k][3] = a.w;
        v[k][4] = b.x; v[k][5] = b.y; v[k][6] = b.z; v[k][7] = b.w;
      } else {
        unpack8(reinterpret_cast<const uint4*>(xr)[c + k * nt], v[k]);
      }
    }
    float s = 0.f;
#pragma unroll
    for (int k = 0; k < CH; ++k)
#pragma unroll
      for (int j = 0; j < 8; ++j) s += v[k][j];
    s = warp_sum(s);
    if (lane == 0) red[0][w] = s;
    __syncthreads();  // also: every thread has read the stage
    if (c == 0) {
      const int nxt = row + LN_STAGES * gridDim.x;
      if (nxt < T) {
        fence_proxy_async_smem();
        mbar_arrive_expect_tx(full + st, row_bytes);
        bulk_load(ln_smem + st * row_bytes, x + (int64_t)nxt * H, row_bytes, full + st);
      }
    }
    float tot = 0.f;
    for (int i = 0; i < nw; ++i) tot += red[0][i];
    const float mu = tot / H;
    float q = 0.f;
#pragma unroll
    for (int k = 0; k < CH; ++k)
#pragma unroll
      for (int j = 0; j < 8; ++j) q += (v[k][j] - mu) * (v[k][j] - mu);
    q = warp_sum(q);
    if (lane == 0) red[1][w] = q;
    __syncthreads();
    tot = 0.f;
    for (int i = 0; i < nw; ++i) tot += red[1][i];
    const float rs = rsqrtf(tot / H + eps);
    __nv_bfloat16* yr = y + (int64_t)row * H;
#pragma unroll
    for (int k = 0; k < CH; ++k) {
      float o[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) o[j] = (v[k][j] - mu) * rs * gg[k][j] + bt[k][j];
      reinterpret_cast<uint4*>(yr)[c + k * nt] = pack8(o);
    }
    if (c == 0) {
      mean[row] = mu;
      rstd[row] = rs;
    }
  }
}

// Backward: dx = rstd (g - mean(g) - xhat mean(g xhat)), g = gamma dy (+ alpha resid);
// persistent CTAs of H/8 threads walk rows blockIdx.x, + gridDim.x, ...; one elected thread
// bulk-copies each row's dy and x into a shared-memory stage (LNB_STAGES in flight, refilled
// once every thread has read it).  Thread c keeps its 8 columns' dgamma / dbeta partials (and
// with CS the column sums of dx, the bias gradient of the GEMM whose output gradient dx is)
// in registers across the CTA's rows and writes them to workspace[blockIdx.x][2 + CS][H];
// ln_bwd_reduce_kernel adds them up.  At <= 64 registers two 512-thread CTAs (3 x 32 KB of
// stages each at H = 4096, fp32) share an SM: six rows in flight.  Every wait is bounded.
constexpr int LNB_STAGES = 3;

template <typename T, bool CS>
__global__ void __launch_bounds__(512, 2) ln_bwd_kernel(int Tn, int H, const T* __restrict__ dy,
                                                        const T* __restrict__ x, const float* __restrict__ mean,
                                                        const float* __restrict__ rstd,
                                                        const float* __restrict__ gamma, const T* __restrict__ resid,
                                                        float resid_alpha, __nv_bfloat16* __restrict__ dx_bf16,
                                                        float* __restrict__ dx_f32, float* __restrict__ ws,
                                                        int* status) {
  extern __shared__ __align__(128) uint8_t lnb_smem[];
  pdl_wait();  // the previous kernel on the stream has completed (see fl_launch)
  pdl_trigger();
  const uint32_t row_bytes = (uint32_t)H * sizeof(T);
  uint64_t* full = reinterpret_cast<uint64_t*>(lnb_smem + 2 * LNB_STAGES * row_bytes);
  __shared__ float2 red[2][32];
  const int c = threadIdx.x;
  auto issue = [&](int st, int row) {  // one elected thread: dy and x of `row` into stage st
    mbar_arrive_expect_tx(full + st, 2 * row_bytes);
    bulk_load(lnb_smem + (2 * st) * row_bytes, dy + (int64_t)row * H, row_bytes, full + st);
    bulk_load(lnb_smem + (2 * st + 1) * row_bytes, x + (int64_t)row * H, row_bytes, full + st);
  };
  if (c == 0) {
    for (int i = 0; i < LNB_STAGES; ++i) mbar_init(full + i, 1);
    fence_mbar_init();
    for (int i = 0; i < LNB_STAGES; ++i)
      if (blockIdx.x + i * gridDim.x < Tn) issue(i, blockIdx.x + i * gridDim.x);
  }
  float accg[8], accb[8], accd[CS ? 8 : 1];
#pragma unroll
  for (int k = 0; k < 8; ++k) accg[k] = accb[k] = 0.f;
#pragma unroll
  for (int k = 0; k < (CS ? 8 : 1); ++k) accd[k] = 0.f;
  __syncthreads();
  int par = 0;
  for (int it = 0;; ++it) {
    const int row = blockIdx.x + it * gridDim.x;
    if (row >= Tn) break;
    const int st = it % LNB_STAGES;
    // the row's statistics and the gain are requested before the stage wait, so that their
    // latency passes while the bulk copy lands
    float gcol[8];
    load8<float>(gamma, c, gcol);
    const float mu = __ldg(mean + row), rs = __ldg(rstd + row);
    if (!__syncthreads_and(mbar_wait(full + st, (it / LNB_STAGES) & 1))) {
      if (c == 0) {
        report_status(status, FL_DEV_TIMEOUT_FULL);
        ln_drain(full, LNB_STAGES, it, Tn);
      }
      break;
    }
    float d[8], xh[8];
    if constexpr (sizeof(T) == 4) {
      const float4* sd = reinterpret_cast<const float4*>(lnb_smem + (2 * st) * row_bytes) + 2 * c;
      const float4* sx = reinterpret_cast<const float4*>(lnb_smem + (2 * st + 1) * row_bytes) + 2 * c;
      const float4 d0 = sd[0], d1 = sd[1], x0 = sx[0], x1 = sx[1];
      d[0] = d0.x; d[1] = d0.y; d[2] = d0.z; d[3] = d0.w; d[4] = d1.x; d[5] = d1.y; d[6] = d1.z; d[7] = d1.w;
      xh[0] = x0.x; xh[1] = x0.y; xh[2] = x0.z; xh[3] = x0.w; xh[4] = x1.x; xh[5] = x1.y; xh[6] = x1.z; xh[7] = x1.w;
    } else {
      unpack8(reinterpret_cast<const uint4*>(lnb_smem + (2 * st) * row_bytes)[c], d);
      unpack8(reinterpret_cast<const uint4*>(lnb_smem + (2 * st + 1) * row_bytes)[c], xh);
    }
    float s1 = 0.f, s2 = 0.f;
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      xh[k] = (xh[k] - mu) * rs;
      const float g = d[k] * gcol[k];
      s1 += g;
      s2 += g * xh[k];
      accg[k] += d[k] * xh[k];
      accb[k] += d[k];
    }
    const float2 sums = block_sum2(s1, s2, red, par);  // its barrier: every thread has read the stage
    par ^= 1;
    if (c == 0) {
      const int nxt = row + LNB_STAGES * gridDim.x;
      if (nxt < Tn) {
        fence_proxy_async_smem();
        issue(st, nxt);
      }
    }
    const float mg = sums.x / H, mgx = sums.y / H;
    float o[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) o[k] = rs * (d[k] * gcol[k] - mg - xh[k] * mgx);
    if (resid) {
      float r[8];
      load8<T>(resid + (int64_t)row * H, c, r);
#pragma unroll
      for (int k = 0; k < 8; ++k) o[k] = fmaf(resid_alpha, r[k], o[k]);
    }
    if constexpr (CS) {
#pragma unroll
      for (int k = 0; k < 8; ++k) accd[k] += o[k];
    }
    if (dx_bf16) reinterpret_cast<uint4*>(dx_bf16 + (int64_t)row * H)[c] = pack8(o);
    if (dx_f32) {
      float4* df = reinterpret_cast<float4*>(dx_f32 + (int64_t)row * H) + 2 * c;
      df[0] = make_float4(o[0], o[1], o[2], o[3]);
      df[1] = make_float4(o[4], o[5], o[6], o[7]);
    }
  }
  float* out = ws + (int64_t)blockIdx.x * (CS ? 3 : 2) * H;
  float4* og = reinterpret_cast<float4*>(out + 8 * c);
  float4* ob = reinterpret_cast<float4*>(out + H + 8 * c);
  og[0] = make_float4(accg[0], accg[1], accg[2], accg[3]);
  og[1] = make_float4(accg[4], accg[5], accg[6], accg[7]);
  ob[0] = make_float4(accb[0], accb[1], accb[2], accb[3]);
  ob[1] = make_float4(accb[4], accb[5], accb[6], accb[7]);
  if constexpr (CS) {
    float4* od = reinterpret_cast<float4*>(out + 2 * H + 8 * c);
    od[0] = make_float4(accd[0], accd[1], accd[2], accd[3]);
    od[1] = make_float4(accd[4], accd[5], accd[6], accd[7]);
  }
}

// dgamma, dbeta (and dcol) += sum over the nblk partial rows of the nv = 2 (3) vectors;
// blockIdx.y takes a slice of the rows.
__global__ void ln_bwd_reduce_kernel(int nblk, int H, int nv, const float* __restrict__ ws, float* __restrict__ dgamma,
                                     float* __restrict__ dbeta, float* __restrict__ dcol) {
  pdl_wait();  // the previous kernel on the stream has completed (see fl_launch)
  pdl_trigger();
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= nv * H) return;
  const int per = (nblk + gridDim.y - 1) / gridDim.y;
  const int b0 = blockIdx.y * per, b1 = min(nblk, b0 + per);
  if (b0 >= b1) return;
  float s = 0.f;
#pragma unroll 8
  for (int b = b0; b < b1; ++b) s += ws[(int64_t)b * nv * H + i];  // independent loads: eight in flight
  atomicAdd(i < H ? dgamma + i : i < 2 * H ? dbeta + (i - H) : dcol + (i - 2 * H), s);
}

template <typename T>
int dispatch_ln_bwd(int nblk, int Tn, int H, const void* dy, const void* x, const float* mean, const float* rstd,
                    const float* gamma, const void* resid, float alpha, void* dx_bf16, float* dx_f32, float* ws,
                    float* dgamma, float* dbeta, float* dcol, cudaStream_t st, int* status = nullptr) {
  const int smem = 2 * LNB_STAGES * H * (int)sizeof(T) + LNB_STAGES * 8;
  const int mx = 2 * LNB_STAGES * 4096 * (int)sizeof(T) + LNB_STAGES * 8;
  FL_CUDA_TRY(fl_func_smem((const void*)ln_bwd_kernel<T, true>, mx));
  FL_CUDA_TRY(fl_func_smem((const void*)ln_bwd_kernel<T, false>, mx));
  if (dcol)
    FL_CUDA_TRY(fl_launch(ln_bwd_kernel<T, true>, dim3(nblk), dim3(H / 8), smem, st, Tn, H, (const T*)dy, (const T*)x,
                          mean, rstd, gamma, (const T*)resid, alpha, (__nv_bfloat16*)dx_bf16, dx_f32, ws, status));
  else
    FL_CUDA_TRY(fl_launch(ln_bwd_kernel<T, false>, dim3(nblk), dim3(H / 8), smem, st, Tn, H, (const T*)dy,
                          (const T*)x, mean, rstd, gamma, (const T*)resid, alpha, (__nv_bfloat16*)dx_bf16, dx_f32, ws,
                          status));
  const int split = nblk >= 64 ? 16 : 1;
  const int nv = dcol ? 3 : 2;
  FL_CUDA_TRY(fl_launch(ln_bwd_reduce_kernel, dim3((nv * H + 255) / 256, split), dim3(256), 0, st, nblk, H, nv,
                        (const float*)ws, dgamma, dbeta, dcol));
  return FL_OK;
}

// Threads of the forward's CTA for hidden size H: H/16 (two 8-element chunks each) when that
// is a whole number of warps, else H/8 (one chunk each); at most 8 warps (the kernel's
// launch bound and its reduction array).
int ln_fwd_threads(int H) { return (H / 16) % 32 == 0 ? H / 16 : H / 8; }
bool ln_fwd_shape_ok(int H) {
  if (H <= 0 || (H % 256) || H > 4096) return false;
  const int t = ln_fwd_threads(H);
  return t % 32 == 0 && t <= 256;
}

template <typename TX>
int dispatch_ln_fwd(int Tn, int H, const void* x, const float* gamma, const float* beta, float eps, void* y,
                    float* mean, float* rstd, cudaStream_t st, int* status = nullptr) {
  if (!ln_fwd_shape_ok(H)) return fl_internal_error(FL_ERR_UNSUPPORTED, "layernorm: H=%d", H);
  const int threads = ln_fwd_threads(H);
  const int ch = H / (8 * threads);
  const int smem = LN_STAGES * H * (int)sizeof(TX) + LN_STAGES * 8;
  FL_CUDA_TRY(fl_func_smem((const void*)ln_fwd_bulk_kernel<TX, 1>, LN_STAGES * 4096 * (int)sizeof(TX) + LN_STAGES * 8));
  FL_CUDA_TRY(fl_func_smem((const void*)ln_fwd_bulk_kernel<TX, 2>, LN_STAGES * 4096 * (int)sizeof(TX) + LN_STAGES * 8));
  int grid = 3 * sm_count();
  if (grid > Tn) grid = Tn;
  const TX* xx = (const TX*)x;
  __nv_bfloat16* yy = (__nv_bfloat16*)y;
  if (ch == 2)
    FL_CUDA_TRY(fl_launch(ln_fwd_bulk_kernel<TX, 2>, dim3(grid), dim3(threads), smem, st, Tn, H, xx, gamma, beta, eps,
                          yy, mean, rstd, status));
  else
    FL_CUDA_TRY(fl_launch(ln_fwd_bulk_kernel<TX, 1>, dim3(grid), dim3(threads), smem, st, Tn, H, xx, gamma, beta, eps,
                          yy, mean, rstd, status));
  return FL_OK;
}

// CTAs of the backward (and rows of its partial-sum workspace).
int ln_bwd_blocks(int T) {
  const int cap = 2 * sm_count();
  return T < cap ? T : cap;
}

// ------------------------------------------------------------------ column sums (bias grads)
// Block: 32 column-threads (8 columns each = 256 columns) x 8 row groups.
__global__ void __launch_bounds__(256) colsum_kernel(int T, int N, const __nv_bfloat16* __restrict__ x,
                                                     float* __restrict__ out, int rows_per_block) {
  pdl_wait();  // the previous kernel on the stream has completed (see fl_launch)
  pdl_trigger();
  __shared__ float red[8][256];
  const int cx = threadIdx.x & 31;
  const int ry = threadIdx.x >> 5;
  const int col = blockIdx.x * 256 + cx * 8;
  const int r0 = blockIdx.y * rows_per_block;
  const int r1 = min(T, r0 + rows_per_block);
  float acc[8] = {0, 0, 0, 0, 0, 0, 0, 0};
  if (col < N) {
#pragma unroll 4
    for (int r = r0 + ry; r < r1; r += 8) {
      float f[8];
      unpack8(__ldg(reinterpret_cast<const uint4*>(x + (int64_t)r * N + col)), f);
#pragma unroll
      for (int j = 0; j < 8; ++j) acc[j] += f[j];
    }
  }
#pragma unroll
  for (int j = 0; j < 8; ++j) red[ry][cx * 8 + j] = acc[j];
  __syncthreads();
  const int c = threadIdx.x;
  if (blockIdx.x * 256 + c < N) {
    float s = 0.f;
#pragma unroll
    for (int k = 0; k < 8; ++k) s += red[k][c];
    atomicAdd(out + blockIdx.x * 256 + c, s);
  }
}

// ------------------------------------------------------------------ AdamW
__global__ void __launch_bounds__(256) adamw_kernel(int64_t n4, float4* __restrict__ w, float4* __restrict__ g,
                                                    float4* __restrict__ m, float4* __restrict__ v,
                                                    uint2* __restrict__ wb, float lr, float b1, float b2, float eps,
                                                    float wd, float inv_bc1, float inv_bc2, int zero_grad) {
  pdl_wait();  // the previous kernel on the stream has completed (see fl_launch)
  pdl_trigger();
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n4; i += (int64_t)gridDim.x * blockDim.x) {
    float4 W = w[i], G = g[i], M = m[i], V = v[i];
    float* pw = &W.x;
    float* pg = &G.x;
    float* pm = &M.x;
    float* pv = &V.x;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      pm[j] = b1 * pm[j] + (1.f - b1) * pg[j];
      pv[j] = b2 * pv[j] + (1.f - b2) * pg[j] * pg[j];
      const float mh = pm[j] * inv_bc1;
      const float vh = pv[j] * inv_bc2;
      pw[j] = pw[j] - lr * (mh / (sqrtf(vh) + eps) + wd * pw[j]);
    }
    w[i] = W;
    m[i] = M;
    v[i] = V;
    if (zero_grad) g[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    if (wb) wb[i] = make_uint2(pack_bf16x2(W.x, W.y), pack_bf16x2(W.z, W.w));
  }
}

// Parameter averaging of n replicas (§3.3 server-hierarchical: the replicas' parameters are
// averaged at the end of each period).  Every replica's fp32 master and bf16 copy receive
// the arithmetic mean, summed in replica order (deterministic).
__global__ void __launch_bounds__(256) average_kernel(ReplicaTable t, int64_t n4) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n4; i += (int64_t)gridDim.x * blockDim.x) {
    float4 s = reinterpret_cast<const float4*>(t.w[0])[i];
    for (int r = 1; r < t.n; ++r) {
      const float4 v = reinterpret_cast<const float4*>(t.w[r])[i];
      s.x += v.x; s.y += v.y; s.z += v.z; s.w += v.w;
    }
    const float inv = 1.f / (float)t.n;
    const float4 mean = make_float4(s.x * inv, s.y * inv, s.z * inv, s.w * inv);
    const uint2 packed = make_uint2(pack_bf16x2(mean.x, mean.y), pack_bf16x2(mean.z, mean.w));
    for (int r = 0; r < t.n; ++r) {
      reinterpret_cast<float4*>(t.w[r])[i] = mean;
      reinterpret_cast<uint2*>(t.wb[r])[i] = packed;
    }
  }
}

// The last step of a mean taken across processes: the arena holds the sum of n replicas'
// weights (an all-reduce), scaled here by 1/n as average_kernel does, bf16 copy refreshed.
__global__ void __launch_bounds__(256) mean_finish_kernel(int64_t n4, float inv, float* __restrict__ w,
                                                          __nv_bfloat16* __restrict__ wb) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n4; i += (int64_t)gridDim.x * blockDim.x) {
    const float4 s = reinterpret_cast<const float4*>(w)[i];
    const float4 mean = make_float4(s.x * inv, s.y * inv, s.z * inv, s.w * inv);
    reinterpret_cast<float4*>(w)[i] = mean;
    reinterpret_cast<uint2*>(wb)[i] = make_uint2(pack_bf16x2(mean.x, mean.y), pack_bf16x2(mean.z, mean.w));
  }
}

__global__ void f32_to_bf16_kernel(int64_t n, const float* __restrict__ src, __nv_bfloat16* __restrict__ dst) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
    dst[i] = f2bf(src[i]);
}

// ------------------------------------------------------------------ pack / unpack
// blockIdx.y = table entry; each entry moves n8 groups of 8 elements between a client
// buffer (bf16) and the packed buffer (bf16 or fp32).
__global__ void copy_clients_kernel(CopyTable tab) {
  pdl_wait();  // the previous kernel on the stream has completed (see fl_launch)
  pdl_trigger();
  const int e = blockIdx.y;
  if (e >= tab.n) return;
  const int64_t n8 = tab.n8[e], off = tab.off8[e];
  uint4* client = reinterpret_cast<uint4*>(tab.client[e]);
  uint4* pb = tab.packed_bf16 ? reinterpret_cast<uint4*>(tab.packed_bf16) + off : nullptr;
  float4* pf = tab.packed_f32 ? reinterpret_cast<float4*>(tab.packed_f32) + 2 * off : nullptr;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n8; i += (int64_t)gridDim.x * blockDim.x) {
    switch (tab.mode) {
      case COPY_GATHER_BF16: pb[i] = client[i]; break;
      case COPY_SCATTER_BF16: client[i] = pb[i]; break;
      case COPY_GATHER_F32: {
        const uint4 w = client[i];
        if (pb) pb[i] = w;
        float f[8];
        unpack8(w, f);
        pf[2 * i] = make_float4(f[0], f[1], f[2], f[3]);
        pf[2 * i + 1] = make_float4(f[4], f[5], f[6], f[7]);
        break;
      }
      default: {  // COPY_SCATTER_F32
        const float4 a = pf[2 * i], b = pf[2 * i + 1];
        const float f[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
        client[i] = pack8(f);
        break;
      }
    }
  }
}

// ------------------------------------------------------------------ packing metadata
// GLM positions of token i of a segment with context length c and mask position mp:
// (i, 0) in the context (or in a plain causal segment, c = 0), (mp, i - c + 1) in the span.
__global__ void meta_kernel(MetaArgs a, int32_t* __restrict__ cu, int32_t* __restrict__ pos,
                            uint32_t* __restrict__ tiles, int32_t* __restrict__ pos2, int32_t* __restrict__ ctx) {
  pdl_wait();  // the previous kernel on the stream has completed (see fl_launch)
  pdl_trigger();
  const int64_t tid = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  const int64_t nth = (int64_t)gridDim.x * blockDim.x;
  const int T = a.cu[a.S];
  for (int64_t i = tid; i <= a.S; i += nth) cu[i] = a.cu[i];
  for (int64_t i = tid; i < a.n_tiles + a.n_tiles128; i += nth) tiles[i] = a.tiles[i];
  if (ctx)
    for (int64_t i = tid; i < a.S; i += nth) ctx[i] = a.glm ? a.ctx[i] : 0;
  for (int64_t t = tid; t < T; t += nth) {
    int lo = 0, hi = a.S - 1;  // last segment with cu[s] <= t
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (a.cu[mid] <= t) lo = mid;
      else hi = mid - 1;
    }
    const int i = int(t - a.cu[lo]);
    int p1 = i, p2 = 0;
    if (a.glm && a.ctx[lo] > 0 && i >= a.ctx[lo]) {
      p1 = a.mpos[lo];
      p2 = i - a.ctx[lo] + 1;
    }
    pos[t] = p1;
    if (pos2) pos2[t] = p2;
  }
}

// ------------------------------------------------------------------ seeded init
// SplitMix64 stream (Steele, Lea & Flood 2014) and Box-Muller (1958):
//   raw(key, i) = mix64(key + (i+1) * GOLDEN);  U = ((raw >> 11) + 1) * 2^-53
//   element i: pair j = i/2, r = sqrt(-2 ln U(2j)), phi = 2 pi U(2j+1),
//   z = r cos(phi) (even i) or r sin(phi) (odd i); value = fp32(mean + std * z)
__device__ __forceinline__ uint64_t mix64(uint64_t z) {
  z ^= z >> 30;
  z *= 0xBF58476D1CE4E5B9ull;
  z ^= z >> 27;
  z *= 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}
__device__ __forceinline__ double unif(uint64_t key, uint64_t i) {
  const uint64_t x = mix64(key + (i + 1) * 0x9E3779B97F4A7C15ull);
  return (double)((x >> 11) + 1) * (1.0 / 9007199254740992.0);
}
__global__ void normal_init_kernel(int64_t n, uint64_t key, double mean, double std_, float* __restrict__ out) {
  const double two_pi = 6.283185307179586476925286766559;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
    const uint64_t j = (uint64_t)i >> 1;
    const double u1 = unif(key, 2 * j), u2 = unif(key, 2 * j + 1);
    const double r = sqrt(-2.0 * log(u1));
    const double z = (i & 1) ? r * sin(two_pi * u2) : r * cos(two_pi * u2);
    out[i] = (float)(mean + std_ * z);
  }
}
__global__ void fill_kernel(int64_t n, float v, float* __restrict__ out) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
    out[i] = v;
}

int grid_for(int64_t n, int per_thread_block = 256) {
  int64_t b = (n + per_thread_block - 1) / per_thread_block;
  const int64_t cap = (int64_t)sm_count() * 8;
  if (b > cap) b = cap;
  if (b < 1) b = 1;
  return (int)b;
}

}  // namespace

// ====================================================================== exported kernel API

extern "C" int fl_k_layernorm_fwd(int32_t T, int32_t H, const void* x, int32_t x_dtype, const float* gamma,
                                  const float* beta, float eps, void* y, float* mean, float* rstd, void* stream) {
  if (T < 0) return fl_internal_error(FL_ERR_INVALID_ARG, "layernorm: negative T=%d", T);
  if (!ln_fwd_shape_ok(H))
    return fl_internal_error(FL_ERR_UNSUPPORTED, "layernorm: H=%d (a multiple of 256 up to 2048, or of 512 up to 4096)", H);
  if (!x || !gamma || !beta || !y || !mean || !rstd) return fl_internal_error(FL_ERR_INVALID_ARG, "layernorm: null");
  if (x_dtype != FL_DT_BF16 && x_dtype != FL_DT_F32) return fl_internal_error(FL_ERR_INVALID_ARG, "layernorm: dtype");
  if (fl_misaligned(x, 16) || fl_misaligned(gamma, 16) || fl_misaligned(beta, 16) || fl_misaligned(y, 16))
    return fl_internal_error(FL_ERR_INVALID_ARG, "layernorm: x, gamma, beta and y must be 16-byte aligned");
  if (T == 0) return FL_OK;
  cudaStream_t st = (cudaStream_t)stream;
  return x_dtype == FL_DT_F32 ? dispatch_ln_fwd<float>(T, H, x, gamma, beta, eps, y, mean, rstd, st)
                              : dispatch_ln_fwd<__nv_bfloat16>(T, H, x, gamma, beta, eps, y, mean, rstd, st);
}

extern "C" size_t fl_k_layernorm_bwd_workspace(int32_t T, int32_t H) {
  return (size_t)ln_bwd_blocks(T > 0 ? T : 1) * 2 * (size_t)H * sizeof(float);
}

extern "C" int fl_k_layernorm_bwd(int32_t T, int32_t H, const void* dy, const void* x, int32_t io_dtype,
                                  const float* mean, const float* rstd, const float* gamma, const void* resid,
                                  float resid_alpha, void* dx_bf16, float* dx_f32, float* dgamma, float* dbeta,
                                  void* workspace, void* stream) {
  if (T < 0) return fl_internal_error(FL_ERR_INVALID_ARG, "layernorm bwd: negative T=%d", T);
  if (H <= 0 || (H % 256) || H > 4096)
    return fl_internal_error(FL_ERR_UNSUPPORTED, "layernorm bwd: H=%d (a multiple of 256 up to 4096)", H);
  if (!dy || !x || !mean || !rstd || !gamma || (!dx_bf16 && !dx_f32) || !dgamma || !dbeta || !workspace)
    return fl_internal_error(FL_ERR_INVALID_ARG, "layernorm bwd: null");
  if (io_dtype != FL_DT_BF16 && io_dtype != FL_DT_F32) return fl_internal_error(FL_ERR_INVALID_ARG, "layernorm bwd: dtype");
  if (fl_misaligned(dy, 16) || fl_misaligned(x, 16) || fl_misaligned(gamma, 16) || fl_misaligned(resid, 16) ||
      fl_misaligned(dx_bf16, 16) || fl_misaligned(dx_f32, 16) || fl_misaligned(workspace, 16))
    return fl_internal_error(FL_ERR_INVALID_ARG,
                             "layernorm bwd: dy, x, gamma, resid, dx and the workspace must be 16-byte aligned");
  if (T == 0) return FL_OK;
  cudaStream_t st = (cudaStream_t)stream;
  const int nblk = ln_bwd_blocks(T);
  float* ws = (float*)workspace;
  return io_dtype == FL_DT_F32
             ? dispatch_ln_bwd<float>(nblk, T, H, dy, x, mean, rstd, gamma, resid, resid_alpha, dx_bf16, dx_f32, ws,
                                      dgamma, dbeta, nullptr, st)
             : dispatch_ln_bwd<__nv_bfloat16>(nblk, T, H, dy, x, mean, rstd, gamma, resid, resid_alpha, dx_bf16,
                                              dx_f32, ws, dgamma, dbeta, nullptr, st);
}

// The runtime's LayerNorm backward on the fp32 residual stream: fl_k_layernorm_bwd plus
// dcol += column sums of dx (the bias gradient of the GEMM whose output gradient dx is).
// The workspace holds fl_launch_layernorm_bwd_workspace(T, H) bytes.
size_t fl_launch_layernorm_bwd_workspace(int T, int H) {
  return (size_t)ln_bwd_blocks(T > 0 ? T : 1) * 3 * (size_t)H * sizeof(float);
}
int fl_launch_layernorm_bwd_f32(int T, int H, const float* dy, const float* x, const float* mean, const float* rstd,
                                const float* gamma, const float* resid, float resid_alpha, __nv_bfloat16* dx_bf16,
                                float* dx_f32, float* dgamma, float* dbeta, float* dcol, float* workspace,
                                cudaStream_t st, int* status) {
  if (T == 0) return FL_OK;
  return dispatch_ln_bwd<float>(ln_bwd_blocks(T), T, H, dy, x, mean, rstd, gamma, resid, resid_alpha, dx_bf16, dx_f32,
                                workspace, dgamma, dbeta, dcol, st, status);
}

int fl_launch_layernorm_fwd_f32(int T, int H, const float* x, const float* gamma, const float* beta, float eps,
                                __nv_bfloat16* y, float* mean, float* rstd, cudaStream_t st, int* status) {
  if (T == 0) return FL_OK;
  return dispatch_ln_fwd<float>(T, H, x, gamma, beta, eps, y, mean, rstd, st, status);
}

extern "C" int fl_k_colsum(int32_t T, int32_t N, const void* x, float* out, void* stream) {
  if (T < 0 || N <= 0 || (N % 8) || !x || !out) return fl_internal_error(FL_ERR_INVALID_ARG, "colsum: args");
  if (fl_misaligned(x, 16) || fl_misaligned(out, 4))
    return fl_internal_error(FL_ERR_INVALID_ARG, "colsum: x must be 16-byte aligned");
  if (T == 0) return FL_OK;
  const int cblocks = (N + 255) / 256;
  int rblocks = (8 * sm_count() + cblocks - 1) / cblocks;  // ~8 CTAs (64 warps) per SM
  if (rblocks < 1) rblocks = 1;
  int rows = (T + rblocks - 1) / rblocks;
  rows = (rows + 7) / 8 * 8;
  rblocks = (T + rows - 1) / rows;
  FL_CUDA_TRY(fl_launch(colsum_kernel, dim3(cblocks, rblocks), dim3(256), 0, (cudaStream_t)stream, T, N,
                        (const __nv_bfloat16*)x, out, rows));
  return FL_OK;
}

extern "C" int fl_k_adamw(int64_t n, float* w, float* g, float* m, float* v, void* w_bf16, float lr, float beta1,
                          float beta2, float eps, float weight_decay, float bc1, float bc2, void* stream) {
  if (n < 0 || (n % 4) || !w || !g || !m || !v) return fl_internal_error(FL_ERR_INVALID_ARG, "adamw: args (n %% 4)");
  if (fl_misaligned(w, 16) || fl_misaligned(g, 16) || fl_misaligned(m, 16) || fl_misaligned(v, 16) ||
      fl_misaligned(w_bf16, 8))
    return fl_internal_error(FL_ERR_INVALID_ARG, "adamw: w, g, m, v must be 16-byte and w_bf16 8-byte aligned");
  if (n == 0) return FL_OK;
  const int64_t n4 = n / 4;
  adamw_kernel<<<grid_for(n4), 256, 0, (cudaStream_t)stream>>>(n4, (float4*)w, (float4*)g, (float4*)m, (float4*)v,
                                                              (uint2*)w_bf16, lr, beta1, beta2, eps, weight_decay,
                                                              1.f / bc1, 1.f / bc2, 1);
  FL_CUDA_TRY(cudaGetLastError());
  return FL_OK;
}

int fl_launch_adamw(int64_t n, float* w, float* g, float* m, float* v, void* w_bf16, float lr, float beta1,
                    float beta2, float eps, float weight_decay, float bc1, float bc2, int zero_grad, cudaStream_t st) {
  if (n <= 0) return FL_OK;
  const int64_t n4 = n / 4;
  FL_CUDA_TRY(fl_launch(adamw_kernel, dim3(grid_for(n4)), dim3(256), 0, st, n4, (float4*)w, (float4*)g, (float4*)m,
                        (float4*)v, (uint2*)w_bf16, lr, beta1, beta2, eps, weight_decay, 1.f / bc1, 1.f / bc2,
                        zero_grad));
  return FL_OK;
}

// ====================================================================== internal launchers

int fl_launch_copy_clients(const CopyTable& tab, cudaStream_t st) {
  if (tab.n <= 0) return FL_OK;
  int64_t maxn = 0;
  for (int e = 0; e < tab.n; ++e) maxn = tab.n8[e] > maxn ? tab.n8[e] : maxn;
  int gx = (int)((maxn + 255) / 256);
  const int cap = (2 * sm_count() + tab.n - 1) / tab.n + 1;
  if (gx > cap) gx = cap;
  if (gx < 1) gx = 1;
  FL_CUDA_TRY(fl_launch(copy_clients_kernel, dim3(gx, tab.n), dim3(256), 0, st, tab));
  return FL_OK;
}

int fl_launch_meta(const MetaArgs& a, int32_t* cu, int32_t* pos, uint32_t* tiles, int32_t* pos2, int32_t* ctx,
                   cudaStream_t st) {
  const int T = a.cu[a.S];
  FL_CUDA_TRY(fl_launch(meta_kernel, dim3(grid_for(T > a.n_tiles ? T : a.n_tiles)), dim3(256), 0, st, a, cu, pos,
                        tiles, pos2, ctx));
  return FL_OK;
}

int fl_launch_normal_init(int64_t n, uint64_t key, double mean, double std_, float* out, cudaStream_t st) {
  if (n <= 0) return FL_OK;
  normal_init_kernel<<<grid_for(n), 256, 0, st>>>(n, key, mean, std_, out);
  FL_CUDA_TRY(cudaGetLastError());
  return FL_OK;
}

int fl_launch_fill(int64_t n, float v, float* out, cudaStream_t st) {
  if (n <= 0) return FL_OK;
  fill_kernel<<<grid_for(n), 256, 0, st>>>(n, v, out);
  FL_CUDA_TRY(cudaGetLastError());
  return FL_OK;
}

int fl_launch_average(const ReplicaTable& t, int64_t n, cudaStream_t st) {
  if (n <= 0 || t.n <= 0) return FL_OK;
  average_kernel<<<grid_for(n / 4), 256, 0, st>>>(t, n / 4);
  FL_CUDA_TRY(cudaGetLastError());
  return FL_OK;
}

int fl_launch_mean_finish(int64_t n, int n_replicas, float* w, void* wb, cudaStream_t st) {
  if (n % 4) return fl_internal_error(FL_ERR_INVALID_ARG, "mean finish: length %lld not a multiple of 4", (long long)n);
  if (n <= 0) return FL_OK;
  mean_finish_kernel<<<grid_for(n / 4), 256, 0, st>>>(n / 4, 1.f / (float)n_replicas, w, (__nv_bfloat16*)wb);
  FL_CUDA_TRY(cudaGetLastError());
  return FL_OK;
}

// dst[c][r] = src[r][c] for src [rows, cols] (fp32), through 32 x 32 shared-memory tiles so
// that both the reads and the writes are coalesced; blockDim (32, 8).
__global__ void transpose_f32_kernel(int64_t rows, int64_t cols, const float* __restrict__ src,
                                     float* __restrict__ dst) {
  __shared__ float tile[32][33];
  const int64_t r0 = (int64_t)blockIdx.y * 32, c0 = (int64_t)blockIdx.x * 32;
  for (int i = threadIdx.y; i < 32; i += 8) {
    const int64_t r = r0 + i, c = c0 + threadIdx.x;
    if (r < rows && c < cols) tile[i][threadIdx.x] = src[r * cols + c];
  }
  __syncthreads();
  for (int i = threadIdx.y; i < 32; i += 8) {
    const int64_t c = c0 + i, r = r0 + threadIdx.x;
    if (r < rows && c < cols) dst[c * rows + r] = tile[threadIdx.x][i];
  }
}

int fl_launch_transpose_f32(int64_t rows, int64_t cols, const float* src, float* dst, cudaStream_t st) {
  if (rows <= 0 || cols <= 0) return FL_OK;
  const int64_t gx = (cols + 31) / 32, gy = (rows + 31) / 32;
  if (gy > 65535) return fl_internal_error(FL_ERR_UNSUPPORTED, "transpose: %lld rows", (long long)rows);
  transpose_f32_kernel<<<dim3((unsigned)gx, (unsigned)gy), dim3(32, 8), 0, st>>>(rows, cols, src, dst);
  FL_CUDA_TRY(cudaGetLastError());
  return FL_OK;
}

int fl_launch_f32_to_bf16(int64_t n, const float* src, void* dst, cudaStream_t st) {
  if (n <= 0) return FL_OK;
  f32_to_bf16_kernel<<<grid_for(n), 256, 0, st>>>(n, src, (__nv_bfloat16*)dst);
  FL_CUDA_TRY(cudaGetLastError());
  return FL_OK;
}

extern "C" int fl_k_pack_clients(int32_t K, void* const* clients_host, const int64_t* bytes_host, void* packed,
                                 int32_t scatter, void* stream) {
  if (K < 0 || K > 4096 || !packed || (K > 0 && (!clients_host || !bytes_host)))
    return fl_internal_error(FL_ERR_INVALID_ARG, "pack: args");
  if (reinterpret_cast<uintptr_t>(packed) & 15) return fl_internal_error(FL_ERR_INVALID_ARG, "pack: packed alignment");
  int64_t off = 0;
  for (int k0 = 0; k0 < K; k0 += FL_MAX_COPY) {
    CopyTable tab;
    tab.n = (K - k0) < FL_MAX_COPY ? (K - k0) : FL_MAX_COPY;
    tab.mode = scatter ? COPY_SCATTER_BF16 : COPY_GATHER_BF16;
    tab.packed_bf16 = packed;
    tab.packed_f32 = nullptr;
    for (int e = 0; e < tab.n; ++e) {
      const int k = k0 + e;
      if (!clients_host[k] || (reinterpret_cast<uintptr_t>(clients_host[k]) & 15) || bytes_host[k] < 0 ||
          (bytes_host[k] % 16))
        return fl_internal_error(FL_ERR_INVALID_ARG, "pack: client %d pointer/size", k);
      tab.client[e] = clients_host[k];
      tab.off8[e] = off / 16;
      tab.n8[e] = bytes_host[k] / 16;
      off += bytes_host[k];
    }
    if (int rc = fl_launch_copy_clients(tab, (cudaStream_t)stream)) return rc;
  }
  return FL_OK;
}

// ====================================================================== allocation-free LayerNorm backward
// Some callers cannot call cudaMalloc: a plug-in hosted by a framework that owns every
// byte of device memory through its own pool and forbids raw allocations, a serving loop
// that must not pay cudaMalloc's implicit device synchronisation, or a process whose
// device-memory budget was reserved in full at start-up.  For them this variant of the
// LayerNorm backward keeps its per-CTA dgamma/dbeta partial sums in a fixed array that
// lives in the library image instead of a caller-provided workspace.
//
// The array holds FL_LN_NOALLOC_MAX_BLOCKS x 2 x 4096 floats (8 MiB); every GPU that loads
// the library holds it until the process exits.  The launch uses at most that many CTAs;
// hidden sizes above 4096 are rejected.  Every call shares the array: calls that overlap
// on the GPU (for example on two streams) race and must be serialised by the caller.
// Each CTA overwrites its whole slice before the reduction reads it, so nothing in the
// array has to start at zero and stale contents from an earlier call are never read.
namespace {
constexpr int FL_LN_NOALLOC_MAX_BLOCKS = 256;
constexpr int FL_LN_NOALLOC_MAX_H = 4096;
constexpr size_t FL_LN_NOALLOC_FLOATS = (size_t)FL_LN_NOALLOC_MAX_BLOCKS * 2 * FL_LN_NOALLOC_MAX_H;
}  // namespace

static __device__ __align__(256) float g_ln_bwd_scratch[FL_LN_NOALLOC_FLOATS];

namespace {
constexpr int FL_NOALLOC_MAX_DEVICES = 64;
float* g_ln_scratch_ptr[FL_NOALLOC_MAX_DEVICES] = {};
std::mutex g_ln_scratch_mu;

// Device address of the scratch array on the current device.  The host-side name of a
// __device__ array is only a stand-in, so the address is looked up once per device with
// that device current (the first call on each device does this) and kept for the life of
// the process: after a cudaDeviceReset the cached address is stale, so the entry point
// must not be called again in a process that has reset the device.
int ln_scratch_address(float** out) {
  int dev = 0;
  FL_CUDA_TRY(cudaGetDevice(&dev));
  if (dev < 0 || dev >= FL_NOALLOC_MAX_DEVICES)
    return fl_internal_error(FL_ERR_UNSUPPORTED, "layernorm bwd (no-alloc): device ordinal %d", dev);
  std::lock_guard<std::mutex> lock(g_ln_scratch_mu);
  if (!g_ln_scratch_ptr[dev]) {
    void* p = nullptr;
    FL_CUDA_TRY(cudaGetSymbolAddress(&p, g_ln_bwd_scratch));
    g_ln_scratch_ptr[dev] = static_cast<float*>(p);
  }
  *out = g_ln_scratch_ptr[dev];
  return FL_OK;
}
}  // namespace

extern "C" int fl_k_layernorm_bwd_noalloc(int32_t T, int32_t H, const void* dy, const void* x, const float* mean,
                                          const float* rstd, const float* gamma, const void* resid,
                                          float resid_alpha, void* dx, float* dgamma, float* dbeta, void* stream) {
  if (T < 0) return fl_internal_error(FL_ERR_INVALID_ARG, "layernorm bwd (no-alloc): T=%d is negative", T);
  if (H <= 0 || (H % 256))
    return fl_internal_error(FL_ERR_UNSUPPORTED, "layernorm bwd (no-alloc): H=%d must be a positive multiple of 256", H);
  if (H > FL_LN_NOALLOC_MAX_H)
    return fl_internal_error(FL_ERR_CAPACITY,
                             "layernorm bwd (no-alloc): H=%d exceeds the %d columns its fixed scratch array holds", H,
                             FL_LN_NOALLOC_MAX_H);
  if (!dy || !x || !mean || !rstd || !gamma || !dx || !dgamma || !dbeta)
    return fl_internal_error(FL_ERR_INVALID_ARG, "layernorm bwd (no-alloc): null pointer");
  if (fl_misaligned(dy, 16) || fl_misaligned(x, 16) || fl_misaligned(gamma, 16) || fl_misaligned(resid, 16) ||
      fl_misaligned(dx, 16))
    return fl_internal_error(FL_ERR_INVALID_ARG, "layernorm bwd (no-alloc): dy, x, gamma, resid and dx must be 16-byte aligned");
  float* ws = nullptr;
  if (int rc = ln_scratch_address(&ws)) return rc;
  if (T == 0) return FL_OK;
  cudaStream_t st = (cudaStream_t)stream;
  int nblk = ln_bwd_blocks(T);
  if (nblk > FL_LN_NOALLOC_MAX_BLOCKS) nblk = FL_LN_NOALLOC_MAX_BLOCKS;
  return dispatch_ln_bwd<__nv_bfloat16>(nblk, T, H, dy, x, mean, rstd, gamma, resid, resid_alpha, dx, nullptr, ws,
                                        dgamma, dbeta, nullptr, st);
}
