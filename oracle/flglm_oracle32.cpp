// fp32 CPU oracle of the FL-GLM server block stack (forward + backward + AdamW).
//
// TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and bench.py's
// cpu_baseline / --impl reference legs load this library; the CUDA library never does,
// and the two share no code, header, table or constant.
//
// The same definitions as the fp64 oracle (flglm_oracle.py), written out in plain C++ in
// single precision: every sum runs over its index in order (a dot product in k order, a
// column sum in token order), nothing is blocked, fused or reordered beyond that, no BLAS.
// OpenMP splits independent outputs (rows, columns, (segment, head) pairs) over the host
// cores; it never splits a sum.
//
//   §3.1 (Model Split): the server maps each client's smashed data h_0 through its blocks
//     and back-propagates the client's gradient w.r.t. its output;
//   §3.3 (client-batch): the clients' rows are stacked into one batch without mixing, so
//     every (client, row) is its own causal segment (cu_seqlens);
//   the block (the ChatGLM-6B reading; the paper prints no block internals):
//     a = LN1(x); qkv = a Wqkv^T + bqkv; q, k <- RoPE (dims [0, rotary_dim) of each head,
//     pairs (i, i + rotary_dim/2), angle p base^(-2i/rotary_dim), p = index in the segment)
//     o = softmax(q k^T / sqrt(d_h) + causal mask) v        (App. A scale)
//     h = alpha res1 + o Wd^T + bd,   res1 = a (residual_from_ln = 1) or x (0)
//     m = LN2(h); y = alpha res2 + gelu(m W1^T + b1) W2^T + b2,  res2 = m or h
//     LN: biased variance, gelu: tanh form;
//   §4.1.4: Adam as AdamW with bias correction (decoupled decay, default 0).
// The backward is the exact chain rule of the above.
#include <omp.h>

#include <cmath>
#include <cstdint>
#include <cstring>
#include <vector>

extern "C" {

typedef struct {
  int32_t hidden, n_heads, head_dim, ffn_hidden, rotary_dim;
  float rope_base, ln_eps, alpha;
  int32_t residual_from_ln;
} flo_shape;

}  // extern "C"

namespace {

using Vec = std::vector<float>;

// C[M,N] = A[M,K] W[N,K]^T (+ bias[N]): every C[m,n] is the dot product of row m of A and
// row n of W summed over k in order, then the bias.  The threads split the rows of W.
void matmul_nt(const float* A, const float* W, const float* bias, float* C, int M, int N, int K) {
#pragma omp parallel for schedule(static)
  for (int n = 0; n < N; ++n) {
    const float* w = W + (size_t)n * K;
    for (int m = 0; m < M; ++m) {
      const float* a = A + (size_t)m * K;
      float s = 0.f;
      for (int k = 0; k < K; ++k) s += a[k] * w[k];
      C[(size_t)m * N + n] = bias ? s + bias[n] : s;
    }
  }
}

// C[M,K] = A[M,N] B[N,K]: every C[m,k] summed over n in order.  The threads split the
// columns k (each walks the rows of B once).
void matmul_nn(const float* A, const float* B, float* C, int M, int N, int K) {
#pragma omp parallel
  {
    const int nt = omp_get_num_threads(), it = omp_get_thread_num();
    const int k0 = (int)((int64_t)K * it / nt), k1 = (int)((int64_t)K * (it + 1) / nt);
    for (int m = 0; m < M; ++m)
      for (int k = k0; k < k1; ++k) C[(size_t)m * K + k] = 0.f;
    for (int n = 0; n < N; ++n) {
      const float* b = B + (size_t)n * K;
      for (int m = 0; m < M; ++m) {
        const float a = A[(size_t)m * N + n];
        float* c = C + (size_t)m * K;
        for (int k = k0; k < k1; ++k) c[k] += a * b[k];
      }
    }
  }
}

// G[N,K] += A[M,N]^T B[M,K]: the product summed over the M tokens in order, then added to
// the accumulator (a weight gradient).
void matmul_tn_acc(const float* A, const float* B, float* G, int M, int N, int K) {
#pragma omp parallel
  {
    Vec t(K);
#pragma omp for schedule(static)
    for (int n = 0; n < N; ++n) {
      for (int k = 0; k < K; ++k) t[k] = 0.f;
      for (int m = 0; m < M; ++m) {
        const float a = A[(size_t)m * N + n];
        const float* b = B + (size_t)m * K;
        for (int k = 0; k < K; ++k) t[k] += a * b[k];
      }
      float* g = G + (size_t)n * K;
      for (int k = 0; k < K; ++k) g[k] += t[k];
    }
  }
}

// g[N] += column sums of A[M,N] (summed over the rows in order): a bias gradient.
void colsum_acc(const float* A, float* g, int M, int N) {
#pragma omp parallel for schedule(static)
  for (int n = 0; n < N; ++n) {
    float s = 0.f;
    for (int m = 0; m < M; ++m) s += A[(size_t)m * N + n];
    g[n] += s;
  }
}

// Row LayerNorm (biased variance): y = (x - mu) rstd gamma + beta.
void layer_norm_fwd(const float* x, const float* gamma, const float* beta, float eps, float* y, float* mu,
                    float* rstd, int T, int H) {
#pragma omp parallel for schedule(static)
  for (int t = 0; t < T; ++t) {
    const float* r = x + (size_t)t * H;
    float s = 0.f;
    for (int i = 0; i < H; ++i) s += r[i];
    const float m = s / H;
    float v = 0.f;
    for (int i = 0; i < H; ++i) v += (r[i] - m) * (r[i] - m);
    const float rs = 1.f / std::sqrt(v / H + eps);
    mu[t] = m;
    rstd[t] = rs;
    for (int i = 0; i < H; ++i) y[(size_t)t * H + i] = (r[i] - m) * rs * gamma[i] + beta[i];
  }
}

// dx = rstd (g - mean(g) - xhat mean(g xhat)), g = gamma dy; dgamma += sum_t dy xhat,
// dbeta += sum_t dy.
void layer_norm_bwd(const float* dy, const float* x, const float* mu, const float* rstd, const float* gamma,
                    float* dx, float* dgamma, float* dbeta, int T, int H) {
#pragma omp parallel for schedule(static)
  for (int t = 0; t < T; ++t) {
    const float* d = dy + (size_t)t * H;
    const float* r = x + (size_t)t * H;
    float sg = 0.f, sgx = 0.f;
    for (int i = 0; i < H; ++i) {
      const float g = d[i] * gamma[i];
      const float xh = (r[i] - mu[t]) * rstd[t];
      sg += g;
      sgx += g * xh;
    }
    const float mg = sg / H, mgx = sgx / H;
    for (int i = 0; i < H; ++i) {
      const float xh = (r[i] - mu[t]) * rstd[t];
      dx[(size_t)t * H + i] = rstd[t] * (d[i] * gamma[i] - mg - xh * mgx);
    }
  }
#pragma omp parallel for schedule(static)
  for (int i = 0; i < H; ++i) {
    float sg = 0.f, sb = 0.f;
    for (int t = 0; t < T; ++t) {
      const float d = dy[(size_t)t * H + i];
      const float xh = (x[(size_t)t * H + i] - mu[t]) * rstd[t];
      sg += d * xh;
      sb += d;
    }
    dgamma[i] += sg;
    dbeta[i] += sb;
  }
}

// Rotary encoding in place on the q or k part of a [T, 3H] row block (column offset
// `col`): pairs (i, i + half) of dims [0, rotary_dim) of every head, position = index in
// the own segment; inverse = rotation by the negative angle.
void rope(float* qkv, int col, const std::vector<int>& pos, const Vec& cs, const Vec& sn, const flo_shape& sh,
          int T, bool inverse, int ld) {
  const int half = sh.rotary_dim / 2;
#pragma omp parallel for schedule(static)
  for (int t = 0; t < T; ++t)
    for (int h = 0; h < sh.n_heads; ++h) {
      float* v = qkv + (size_t)t * ld + col + h * sh.head_dim;
      for (int i = 0; i < half; ++i) {
        const float c = cs[(size_t)pos[t] * half + i];
        const float s = inverse ? -sn[(size_t)pos[t] * half + i] : sn[(size_t)pos[t] * half + i];
        const float x1 = v[i], x2 = v[i + half];
        v[i] = x1 * c - x2 * s;
        v[i + half] = x2 * c + x1 * s;
      }
    }
}

float gelu(float u) {
  const float c = 0.7978845608028654f, a = 0.044715f;
  return 0.5f * u * (1.f + std::tanh(c * (u + a * u * u * u)));
}
float gelu_grad(float u) {
  const float c = 0.7978845608028654f, a = 0.044715f;
  const float t = std::tanh(c * (u + a * u * u * u));
  return 0.5f * (1.f + t) + 0.5f * u * (1.f - t * t) * c * (1.f + 3.f * a * u * u);
}

// Softmax probabilities of query t of one segment and head (causal: keys 0..t), into p.
// qkv rows of the segment start at `base`; the scores are (q . k_u) / sqrt(d_h).
void probs(const float* qkv, int ld, int H, int hd, int h, int t, float scale, float* p, float* lse) {
  const float* q = qkv + (size_t)t * ld + h * hd;
  float mx = -INFINITY;
  for (int u = 0; u <= t; ++u) {
    const float* k = qkv + (size_t)u * ld + H + h * hd;
    float s = 0.f;
    for (int d = 0; d < hd; ++d) s += q[d] * k[d];
    p[u] = s * scale;
    mx = std::fmax(mx, p[u]);
  }
  float l = 0.f;
  for (int u = 0; u <= t; ++u) {
    p[u] = std::exp(p[u] - mx);
    l += p[u];
  }
  for (int u = 0; u <= t; ++u) p[u] /= l;
  if (lse) *lse = mx + std::log(l);
}

struct Saved {
  Vec x, a, mu1, rs1, qkv, o, h, m, mu2, rs2, u, g;
};

struct Block {
  const float *Wqkv, *bqkv, *Wd, *bd, *W1, *b1, *W2, *b2, *g1, *be1, *g2, *be2;
};

void block_fwd(const Block& P, const float* x, float* y, Saved& sv, const flo_shape& sh, int T, int S,
               const int32_t* cu, const std::vector<int>& pos, const Vec& cs, const Vec& sn) {
  const int H = sh.hidden, F = sh.ffn_hidden, nh = sh.n_heads, hd = sh.head_dim;
  const size_t TH = (size_t)T * H;
  sv.x.assign(x, x + TH);
  sv.a.resize(TH);
  sv.mu1.resize(T);
  sv.rs1.resize(T);
  layer_norm_fwd(x, P.g1, P.be1, sh.ln_eps, sv.a.data(), sv.mu1.data(), sv.rs1.data(), T, H);
  sv.qkv.resize(3 * TH);
  matmul_nt(sv.a.data(), P.Wqkv, P.bqkv, sv.qkv.data(), T, 3 * H, H);
  rope(sv.qkv.data(), 0, pos, cs, sn, sh, T, false, 3 * H);
  rope(sv.qkv.data(), H, pos, cs, sn, sh, T, false, 3 * H);
  sv.o.assign(TH, 0.f);
  const float scale = 1.f / std::sqrt((float)hd);
#pragma omp parallel
  {
    Vec p;
#pragma omp for schedule(dynamic)
    for (int sh_ = 0; sh_ < S * nh; ++sh_) {
      const int s = sh_ / nh, h = sh_ % nh;
      const int a0 = cu[s], L = cu[s + 1] - cu[s];
      p.resize(L > 0 ? L : 1);
      const float* seg = sv.qkv.data() + (size_t)a0 * 3 * H;
      for (int t = 0; t < L; ++t) {
        probs(seg, 3 * H, H, hd, h, t, scale, p.data(), nullptr);
        float* o = sv.o.data() + (size_t)(a0 + t) * H + h * hd;
        for (int u = 0; u <= t; ++u) {
          const float* v = seg + (size_t)u * 3 * H + 2 * H + h * hd;
          for (int d = 0; d < hd; ++d) o[d] += p[u] * v[d];
        }
      }
    }
  }
  const float al = sh.alpha;
  sv.h.resize(TH);
  matmul_nt(sv.o.data(), P.Wd, P.bd, sv.h.data(), T, H, H);
  const float* res1 = sh.residual_from_ln ? sv.a.data() : x;
  for (size_t i = 0; i < TH; ++i) sv.h[i] = al * res1[i] + sv.h[i];
  sv.m.resize(TH);
  sv.mu2.resize(T);
  sv.rs2.resize(T);
  layer_norm_fwd(sv.h.data(), P.g2, P.be2, sh.ln_eps, sv.m.data(), sv.mu2.data(), sv.rs2.data(), T, H);
  sv.u.resize((size_t)T * F);
  matmul_nt(sv.m.data(), P.W1, P.b1, sv.u.data(), T, F, H);
  sv.g.resize((size_t)T * F);
  for (size_t i = 0; i < (size_t)T * F; ++i) sv.g[i] = gelu(sv.u[i]);
  matmul_nt(sv.g.data(), P.W2, P.b2, y, T, H, F);
  const float* res2 = sh.residual_from_ln ? sv.m.data() : sv.h.data();
  for (size_t i = 0; i < TH; ++i) y[i] = al * res2[i] + y[i];
}

void block_bwd(const Block& P, float* const* G, const Saved& sv, const float* dy, float* dx, const flo_shape& sh,
               int T, int S, const int32_t* cu, const std::vector<int>& pos, const Vec& cs, const Vec& sn) {
  const int H = sh.hidden, F = sh.ffn_hidden, nh = sh.n_heads, hd = sh.head_dim;
  const size_t TH = (size_t)T * H;
  const float al = sh.alpha;
  // FFN down: y = alpha res2 + g W2^T + b2
  matmul_tn_acc(dy, sv.g.data(), G[6], T, H, F);
  colsum_acc(dy, G[7], T, H);
  Vec du((size_t)T * F);
  matmul_nn(dy, P.W2, du.data(), T, H, F);
  for (size_t i = 0; i < (size_t)T * F; ++i) du[i] = du[i] * gelu_grad(sv.u[i]);
  matmul_tn_acc(du.data(), sv.m.data(), G[4], T, F, H);
  colsum_acc(du.data(), G[5], T, F);
  Vec dm(TH);
  matmul_nn(du.data(), P.W1, dm.data(), T, F, H);
  if (sh.residual_from_ln)
    for (size_t i = 0; i < TH; ++i) dm[i] = dm[i] + al * dy[i];
  Vec dh(TH);
  layer_norm_bwd(dm.data(), sv.h.data(), sv.mu2.data(), sv.rs2.data(), P.g2, dh.data(), G[10], G[11], T, H);
  if (!sh.residual_from_ln)
    for (size_t i = 0; i < TH; ++i) dh[i] = dh[i] + al * dy[i];
  // attention output projection: h = alpha res1 + o Wd^T + bd
  matmul_tn_acc(dh.data(), sv.o.data(), G[2], T, H, H);
  colsum_acc(dh.data(), G[3], T, H);
  Vec dO(TH);
  matmul_nn(dh.data(), P.Wd, dO.data(), T, H, H);
  // attention: dV = P^T dO, dP = dO V^T, dS = P (dP - rowsum(dP P)), dQ = dS K / sqrt(d_h),
  // dK = dS^T Q / sqrt(d_h); gradients w.r.t. the rotated q, k
  Vec dqkv(3 * TH, 0.f);
  const float scale = 1.f / std::sqrt((float)hd);
#pragma omp parallel
  {
    Vec p, dp;
#pragma omp for schedule(dynamic)
    for (int sh_ = 0; sh_ < S * nh; ++sh_) {
      const int s = sh_ / nh, h = sh_ % nh;
      const int a0 = cu[s], L = cu[s + 1] - cu[s];
      p.resize(L > 0 ? L : 1);
      dp.resize(L > 0 ? L : 1);
      const float* seg = sv.qkv.data() + (size_t)a0 * 3 * H;
      float* dseg = dqkv.data() + (size_t)a0 * 3 * H;
      for (int t = 0; t < L; ++t) {
        probs(seg, 3 * H, H, hd, h, t, scale, p.data(), nullptr);
        const float* d_o = dO.data() + (size_t)(a0 + t) * H + h * hd;
        float rs = 0.f;
        for (int u = 0; u <= t; ++u) {
          const float* v = seg + (size_t)u * 3 * H + 2 * H + h * hd;
          float x = 0.f;
          for (int d = 0; d < hd; ++d) x += d_o[d] * v[d];
          dp[u] = x;
          rs += x * p[u];
        }
        const float* q = seg + (size_t)t * 3 * H + h * hd;
        float* dq = dseg + (size_t)t * 3 * H + h * hd;
        for (int u = 0; u <= t; ++u) {
          const float ds = p[u] * (dp[u] - rs);
          const float* k = seg + (size_t)u * 3 * H + H + h * hd;
          float* dk = dseg + (size_t)u * 3 * H + H + h * hd;
          float* dv = dseg + (size_t)u * 3 * H + 2 * H + h * hd;
          for (int d = 0; d < hd; ++d) {
            dq[d] += ds * k[d];
            dk[d] += ds * q[d];
            dv[d] += p[u] * d_o[d];
          }
        }
      }
      for (int t = 0; t < L; ++t) {
        float* r = dseg + (size_t)t * 3 * H + h * hd;
        for (int d = 0; d < hd; ++d) {
          r[d] *= scale;
          r[H + d] *= scale;
        }
      }
    }
  }
  rope(dqkv.data(), 0, pos, cs, sn, sh, T, true, 3 * H);
  rope(dqkv.data(), H, pos, cs, sn, sh, T, true, 3 * H);
  matmul_tn_acc(dqkv.data(), sv.a.data(), G[0], T, 3 * H, H);
  colsum_acc(dqkv.data(), G[1], T, 3 * H);
  Vec da(TH);
  matmul_nn(dqkv.data(), P.Wqkv, da.data(), T, 3 * H, H);
  if (sh.residual_from_ln)
    for (size_t i = 0; i < TH; ++i) da[i] = da[i] + al * dh[i];
  layer_norm_bwd(da.data(), sv.x.data(), sv.mu1.data(), sv.rs1.data(), P.g1, dx, G[8], G[9], T, H);
  if (!sh.residual_from_ln)
    for (size_t i = 0; i < TH; ++i) dx[i] = dx[i] + al * dh[i];
}

}  // namespace

extern "C" {

// Threads the oracle's parallel loops use (OpenMP's current maximum).
int flo_threads(void) { return omp_get_max_threads(); }

// One server call on the fp32 oracle: the packed tokens x [T, H] (segment s = rows
// [cu[s], cu[s+1])) through n_blocks blocks to y [T, H]; then dy [T, H] back to dx [T, H],
// the weight gradients added into grads.  params / grads: n_blocks x 12 pointers in the
// order Wqkv [3H,H], bqkv [3H], Wd [H,H], bd [H], W1 [F,H], b1 [F], W2 [H,F], b2 [H],
// gamma1, beta1, gamma2, beta2 [H] (fp32, row-major).  Returns 0, or -1 on a bad argument.
int flo_server_fwd_bwd(const flo_shape* shp, int32_t n_blocks, const float* const* params, float* const* grads,
                       int32_t S, const int32_t* cu, const float* x, const float* dy, float* y, float* dx) {
  if (!shp || n_blocks < 1 || !params || !grads || S < 1 || !cu || !x || !dy || !y || !dx) return -1;
  const flo_shape sh = *shp;
  if (sh.hidden != sh.n_heads * sh.head_dim || sh.rotary_dim < 2 || sh.rotary_dim % 2 ||
      sh.rotary_dim > sh.head_dim || cu[0] != 0)
    return -1;
  for (int s = 0; s < S; ++s)
    if (cu[s + 1] < cu[s]) return -1;
  const int T = cu[S], H = sh.hidden;
  if (T < 1) return -1;
  std::vector<int> pos(T);
  int max_pos = 0;
  for (int s = 0; s < S; ++s)
    for (int t = cu[s]; t < cu[s + 1]; ++t) {
      pos[t] = t - cu[s];
      max_pos = pos[t] > max_pos ? pos[t] : max_pos;
    }
  // rotation angles p base^(-2i/rotary_dim), evaluated in double and rounded to fp32
  const int half = sh.rotary_dim / 2;
  Vec cs((size_t)(max_pos + 1) * half), sn((size_t)(max_pos + 1) * half);
  for (int p = 0; p <= max_pos; ++p)
    for (int i = 0; i < half; ++i) {
      const double ang = p * std::pow((double)sh.rope_base, -2.0 * i / sh.rotary_dim);
      cs[(size_t)p * half + i] = (float)std::cos(ang);
      sn[(size_t)p * half + i] = (float)std::sin(ang);
    }
  std::vector<Saved> saved(n_blocks);
  Vec cur(x, x + (size_t)T * H), nxt((size_t)T * H);
  for (int b = 0; b < n_blocks; ++b) {
    const float* const* p = params + 12 * b;
    const Block P{p[0], p[1], p[2], p[3], p[4], p[5], p[6], p[7], p[8], p[9], p[10], p[11]};
    block_fwd(P, cur.data(), nxt.data(), saved[b], sh, T, S, cu, pos, cs, sn);
    cur.swap(nxt);
  }
  std::memcpy(y, cur.data(), sizeof(float) * T * H);
  cur.assign(dy, dy + (size_t)T * H);
  for (int b = n_blocks - 1; b >= 0; --b) {
    const float* const* p = params + 12 * b;
    const Block P{p[0], p[1], p[2], p[3], p[4], p[5], p[6], p[7], p[8], p[9], p[10], p[11]};
    block_bwd(P, grads + 12 * b, saved[b], cur.data(), nxt.data(), sh, T, S, cu, pos, cs, sn);
    saved[b] = Saved();
    cur.swap(nxt);
  }
  std::memcpy(dx, cur.data(), sizeof(float) * T * H);
  return 0;
}

// AdamW with bias correction at step t >= 1 (§4.1.4): m = b1 m + (1-b1) g,
// v = b2 v + (1-b2) g^2, w -= lr (m/(1-b1^t) / (sqrt(v/(1-b2^t)) + eps) + wd w).
int flo_adamw(int64_t n, float* w, const float* g, float* m, float* v, int32_t t, float lr, float b1, float b2,
              float eps, float wd) {
  if (n < 0 || t < 1 || (n > 0 && (!w || !g || !m || !v))) return -1;
  const float c1 = 1.f - std::pow(b1, (float)t), c2 = 1.f - std::pow(b2, (float)t);
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i) {
    m[i] = b1 * m[i] + (1.f - b1) * g[i];
    v[i] = b2 * v[i] + (1.f - b2) * g[i] * g[i];
    const float mh = m[i] / c1, vh = v[i] / c2;
    w[i] = w[i] - lr * (mh / (std::sqrt(vh) + eps) + wd * w[i]);
  }
  return 0;
}

}  // extern "C"
