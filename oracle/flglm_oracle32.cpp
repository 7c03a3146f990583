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
//   App. A (P-tuning v2): optional trainable prefix keys / values per block, K' =
//     [prefix_key : key], V' = [prefix_value : value], seen by every query, not rotated;
//     their gradients are summed over every segment;
//   §4.1.1 (GLM blank infilling): optional per-segment context length c and mask-token
//     position; own key u is seen by query t when u <= t or u < c (bidirectional context,
//     causal span); positions are two-dimensional (context token t: (t, 0); span token t:
//     (mask position, t - c + 1)), the second position rotating dims [rotary_dim,
//     2 rotary_dim) of each head with the same frequencies;
//   §4.1.4: Adam as AdamW with bias correction (decoupled decay, default 0);
//   §3.1 client parts (one client's round with the server's blocks left out): bottom =
//     Embedding + Block_0, top = Block_{N-1} + final LayerNorm + bias-free LM head +
//     cross-entropy, the mean over the tokens that carry a target (label >= 0).
// The backward is the exact chain rule of the above.
#include <omp.h>

#include <algorithm>
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
// `col`): pairs (i, i + half) of dims [dim0, dim0 + rotary_dim) of every head, by the angle
// of pos[t]; inverse = rotation by the negative angle.
void rope(float* qkv, int col, int dim0, const std::vector<int>& pos, const Vec& cs, const Vec& sn,
          const flo_shape& sh, int T, bool inverse, int ld) {
  const int half = sh.rotary_dim / 2;
#pragma omp parallel for schedule(static)
  for (int t = 0; t < T; ++t)
    for (int h = 0; h < sh.n_heads; ++h) {
      float* v = qkv + (size_t)t * ld + col + h * sh.head_dim + dim0;
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

// The keys one segment's queries see for one head: the Lp prefix rows (pk / pv [Lp, H],
// null when Lp = 0) then the segment's own rows (q | k | v at `seg`, row stride ld); c is
// the segment's GLM context length (0: plainly causal).  Key j < Lp is prefix row j, key
// Lp + u own row u.
struct Keys {
  const float* seg;
  int ld, H, hd, h, L, c;
  const float* pk;
  const float* pv;
  int Lp;
  // keys 0 .. n(t) - 1 are the ones query t sees: every prefix key and the own keys u <= t,
  // or u < c in the GLM context
  int n(int t) const { return Lp + 1 + (c - 1 > t ? (c - 1 < L - 1 ? c - 1 : L - 1) : t); }
  const float* k(int j) const { return j < Lp ? pk + (size_t)j * H + h * hd : seg + (size_t)(j - Lp) * ld + H + h * hd; }
  const float* v(int j) const {
    return j < Lp ? pv + (size_t)j * H + h * hd : seg + (size_t)(j - Lp) * ld + 2 * H + h * hd;
  }
  const float* q(int t) const { return seg + (size_t)t * ld + h * hd; }
};

// Softmax probabilities of query t over its visible keys 0 .. K.n(t) - 1, into p; the
// scores are (q . k'_j) / sqrt(d_h).
void probs(const Keys& K, int t, float scale, float* p) {
  const float* q = K.q(t);
  const int n = K.n(t);
  float mx = -INFINITY;
  for (int j = 0; j < n; ++j) {
    const float* k = K.k(j);
    float s = 0.f;
    for (int d = 0; d < K.hd; ++d) s += q[d] * k[d];
    p[j] = s * scale;
    mx = std::fmax(mx, p[j]);
  }
  float l = 0.f;
  for (int j = 0; j < n; ++j) {
    p[j] = std::exp(p[j] - mx);
    l += p[j];
  }
  for (int j = 0; j < n; ++j) p[j] /= l;
}

struct Saved {
  Vec x, a, mu1, rs1, qkv, o, h, m, mu2, rs2, u, g;
};

struct Block {
  const float *Wqkv, *bqkv, *Wd, *bd, *W1, *b1, *W2, *b2, *g1, *be1, *g2, *be2;
};

// Positions of a call: pos[t] rotates dims [0, rotary_dim) of every head; with GLM
// segments (glm), pos2[t] rotates dims [rotary_dim, 2 rotary_dim); ctx[s] is segment s's
// context length (all 0 without GLM).
struct Positions {
  std::vector<int> pos, pos2, ctx;
  bool glm = false;
  Vec cs, sn;  // (cos, sin) of position p, pair i at p * rotary_dim / 2 + i
};

void rope_all(float* qkv, const Positions& ps, const flo_shape& sh, int T, bool inverse) {
  for (int col : {0, sh.hidden}) {
    rope(qkv, col, 0, ps.pos, ps.cs, ps.sn, sh, T, inverse, 3 * sh.hidden);
    if (ps.glm) rope(qkv, col, sh.rotary_dim, ps.pos2, ps.cs, ps.sn, sh, T, inverse, 3 * sh.hidden);
  }
}

void block_fwd(const Block& P, const float* x, float* y, Saved& sv, const flo_shape& sh, int T, int S,
               const int32_t* cu, const Positions& ps, const float* pk, const float* pv, int Lp) {
  const int H = sh.hidden, F = sh.ffn_hidden, nh = sh.n_heads, hd = sh.head_dim;
  const size_t TH = (size_t)T * H;
  sv.x.assign(x, x + TH);
  sv.a.resize(TH);
  sv.mu1.resize(T);
  sv.rs1.resize(T);
  layer_norm_fwd(x, P.g1, P.be1, sh.ln_eps, sv.a.data(), sv.mu1.data(), sv.rs1.data(), T, H);
  sv.qkv.resize(3 * TH);
  matmul_nt(sv.a.data(), P.Wqkv, P.bqkv, sv.qkv.data(), T, 3 * H, H);
  rope_all(sv.qkv.data(), ps, sh, T, false);
  sv.o.assign(TH, 0.f);
  const float scale = 1.f / std::sqrt((float)hd);
#pragma omp parallel
  {
    Vec p;
#pragma omp for schedule(dynamic)
    for (int sh_ = 0; sh_ < S * nh; ++sh_) {
      const int s = sh_ / nh, h = sh_ % nh;
      const int a0 = cu[s], L = cu[s + 1] - cu[s];
      const Keys K{sv.qkv.data() + (size_t)a0 * 3 * H, 3 * H, H, hd, h, L, ps.ctx[s], pk, pv, Lp};
      p.resize(Lp + (L > 0 ? L : 1));
      for (int t = 0; t < L; ++t) {
        probs(K, t, scale, p.data());
        float* o = sv.o.data() + (size_t)(a0 + t) * H + h * hd;
        for (int j = 0; j < K.n(t); ++j) {
          const float* v = K.v(j);
          for (int d = 0; d < hd; ++d) o[d] += p[j] * v[d];
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

// dpk / dpv (with a prefix): fp32 [Lp, H] accumulators of the prefix gradients, summed
// over the segments in order.
void block_bwd(const Block& P, float* const* G, const Saved& sv, const float* dy, float* dx, const flo_shape& sh,
               int T, int S, const int32_t* cu, const Positions& ps, const float* pk, const float* pv, int Lp,
               float* dpk, float* dpv) {
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
  // prefix gradients of each (segment, head), added in segment order after the loop
  std::vector<Vec> dpre(Lp > 0 ? (size_t)S * nh : 0);
#pragma omp parallel
  {
    Vec p, dp;
#pragma omp for schedule(dynamic)
    for (int sh_ = 0; sh_ < S * nh; ++sh_) {
      const int s = sh_ / nh, h = sh_ % nh;
      const int a0 = cu[s], L = cu[s + 1] - cu[s];
      const Keys K{sv.qkv.data() + (size_t)a0 * 3 * H, 3 * H, H, hd, h, L, ps.ctx[s], pk, pv, Lp};
      p.resize(Lp + (L > 0 ? L : 1));
      dp.resize(Lp + (L > 0 ? L : 1));
      float* dseg = dqkv.data() + (size_t)a0 * 3 * H;
      float* dpkv = nullptr;  // [2][Lp][hd]: this (segment, head)'s prefix key and value gradients
      if (Lp > 0) {
        dpre[sh_].assign((size_t)2 * Lp * hd, 0.f);
        dpkv = dpre[sh_].data();
      }
      for (int t = 0; t < L; ++t) {
        probs(K, t, scale, p.data());
        const int n = K.n(t);
        const float* d_o = dO.data() + (size_t)(a0 + t) * H + h * hd;
        float rs = 0.f;
        for (int j = 0; j < n; ++j) {
          const float* v = K.v(j);
          float x = 0.f;
          for (int d = 0; d < hd; ++d) x += d_o[d] * v[d];
          dp[j] = x;
          rs += x * p[j];
        }
        const float* q = K.q(t);
        float* dq = dseg + (size_t)t * 3 * H + h * hd;
        for (int j = 0; j < n; ++j) {
          const float ds = p[j] * (dp[j] - rs);
          const float* k = K.k(j);
          float* dk = j < Lp ? dpkv + (size_t)j * hd : dseg + (size_t)(j - Lp) * 3 * H + H + h * hd;
          float* dv = j < Lp ? dpkv + (size_t)(Lp + j) * hd : dseg + (size_t)(j - Lp) * 3 * H + 2 * H + h * hd;
          for (int d = 0; d < hd; ++d) {
            dq[d] += ds * k[d];
            dk[d] += ds * q[d];
            dv[d] += p[j] * d_o[d];
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
      for (int i = 0; i < Lp * hd; ++i) dpkv[i] *= scale;
    }
  }
  for (int s = 0; s < S; ++s)
    for (int h = 0; h < nh; ++h)
      for (int j = 0; j < Lp; ++j)
        for (int d = 0; d < hd; ++d) {
          const float* g = dpre[(size_t)s * nh + h].data();
          dpk[(size_t)j * H + h * hd + d] += g[(size_t)j * hd + d];
          dpv[(size_t)j * H + h * hd + d] += g[(size_t)(Lp + j) * hd + d];
        }
  rope_all(dqkv.data(), ps, sh, T, true);
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

// Positions and rotary tables of a call: segment s = rows [cu[s], cu[s+1]), with GLM
// context lengths ctx / mask positions mask_pos (null: plain segments; null mask_pos: c - 1).
// Returns false on a bad argument.
bool make_positions(const flo_shape& sh, int S, const int32_t* cu, const int32_t* ctx, const int32_t* mask_pos,
                    Positions& ps) {
  const int T = cu[S];
  ps = Positions();
  ps.glm = ctx != nullptr;
  ps.pos.resize(T);
  ps.pos2.assign(T, 0);
  ps.ctx.assign(S, 0);
  int max_pos = 0;
  for (int s = 0; s < S; ++s) {
    const int L = cu[s + 1] - cu[s];
    const int c = ctx ? ctx[s] : 0;
    const int mp = !ctx ? 0 : mask_pos ? mask_pos[s] : c - 1;
    if (c < 0 || c > L || (c > 0 && (mp < 0 || mp >= c))) return false;
    ps.ctx[s] = c;
    for (int t = 0; t < L; ++t) {
      const bool span = c > 0 && t >= c;
      ps.pos[cu[s] + t] = span ? mp : t;
      ps.pos2[cu[s] + t] = span ? t - c + 1 : 0;
      max_pos = std::max(max_pos, std::max(ps.pos[cu[s] + t], ps.pos2[cu[s] + t]));
    }
  }
  // rotation angles p base^(-2i/rotary_dim), evaluated in double and rounded to fp32
  const int half = sh.rotary_dim / 2;
  ps.cs.resize((size_t)(max_pos + 1) * half);
  ps.sn.resize((size_t)(max_pos + 1) * half);
  for (int p = 0; p <= max_pos; ++p)
    for (int i = 0; i < half; ++i) {
      const double ang = p * std::pow((double)sh.rope_base, -2.0 * i / sh.rotary_dim);
      ps.cs[(size_t)p * half + i] = (float)std::cos(ang);
      ps.sn[(size_t)p * half + i] = (float)std::sin(ang);
    }
  return true;
}

}  // namespace

extern "C" {

// Threads the oracle's parallel loops use (OpenMP's current maximum).
int flo_threads(void) { return omp_get_max_threads(); }

// One server call on the fp32 oracle: the packed tokens x [T, H] (segment s = rows
// [cu[s], cu[s+1])) through n_blocks blocks to y [T, H]; then dy [T, H] back to dx [T, H],
// the weight gradients added into grads.  params / grads: n_blocks x 12 pointers in the
// order Wqkv [3H,H], bqkv [3H], Wd [H,H], bd [H], W1 [F,H], b1 [F], W2 [H,F], b2 [H],
// gamma1, beta1, gamma2, beta2 [H] (fp32, row-major).
// ctx / mask_pos (int32 [S] each, or null): GLM segments (§4.1.1), context length c in
// [0, L_s] and mask-token position in [0, c) (null mask_pos: c - 1); needs rotary_dim =
// head_dim / 2.  prefix_len in 0..: with prefix_len > 0, prefixes / prefix_grads hold
// n_blocks x 2 pointers to the fp32 [prefix_len, H] prefix keys and values of each block
// (App. A) and their gradient accumulators.  Returns 0, or -1 on a bad argument.
int flo_server_fwd_bwd_ext(const flo_shape* shp, int32_t n_blocks, const float* const* params, float* const* grads,
                           int32_t S, const int32_t* cu, const int32_t* ctx, const int32_t* mask_pos,
                           int32_t prefix_len, const float* const* prefixes, float* const* prefix_grads,
                           const float* x, const float* dy, float* y, float* dx) {
  if (!shp || n_blocks < 1 || !params || !grads || S < 1 || !cu || !x || !dy || !y || !dx) return -1;
  if (prefix_len < 0 || (prefix_len > 0 && (!prefixes || !prefix_grads))) return -1;
  const flo_shape sh = *shp;
  if (sh.hidden != sh.n_heads * sh.head_dim || sh.rotary_dim < 2 || sh.rotary_dim % 2 ||
      sh.rotary_dim > sh.head_dim || cu[0] != 0)
    return -1;
  if (ctx && 2 * sh.rotary_dim != sh.head_dim) return -1;
  for (int s = 0; s < S; ++s)
    if (cu[s + 1] < cu[s]) return -1;
  const int T = cu[S], H = sh.hidden;
  if (T < 1) return -1;
  Positions ps;
  if (!make_positions(sh, S, cu, ctx, mask_pos, ps)) return -1;
  const int Lp = prefix_len;
  auto pre = [&](int b, int i) { return Lp > 0 ? prefixes[2 * b + i] : nullptr; };
  std::vector<Saved> saved(n_blocks);
  Vec cur(x, x + (size_t)T * H), nxt((size_t)T * H);
  for (int b = 0; b < n_blocks; ++b) {
    const float* const* p = params + 12 * b;
    const Block P{p[0], p[1], p[2], p[3], p[4], p[5], p[6], p[7], p[8], p[9], p[10], p[11]};
    block_fwd(P, cur.data(), nxt.data(), saved[b], sh, T, S, cu, ps, pre(b, 0), pre(b, 1), Lp);
    cur.swap(nxt);
  }
  std::memcpy(y, cur.data(), sizeof(float) * T * H);
  cur.assign(dy, dy + (size_t)T * H);
  for (int b = n_blocks - 1; b >= 0; --b) {
    const float* const* p = params + 12 * b;
    const Block P{p[0], p[1], p[2], p[3], p[4], p[5], p[6], p[7], p[8], p[9], p[10], p[11]};
    block_bwd(P, grads + 12 * b, saved[b], cur.data(), nxt.data(), sh, T, S, cu, ps, pre(b, 0), pre(b, 1), Lp,
              Lp > 0 ? prefix_grads[2 * b] : nullptr, Lp > 0 ? prefix_grads[2 * b + 1] : nullptr);
    saved[b] = Saved();
    cur.swap(nxt);
  }
  std::memcpy(dx, cur.data(), sizeof(float) * T * H);
  return 0;
}

// The server call without GLM segments or a prefix.
int flo_server_fwd_bwd(const flo_shape* shp, int32_t n_blocks, const float* const* params, float* const* grads,
                       int32_t S, const int32_t* cu, const float* x, const float* dy, float* y, float* dx) {
  return flo_server_fwd_bwd_ext(shp, n_blocks, params, grads, S, cu, nullptr, nullptr, 0, nullptr, nullptr, x, dy,
                                y, dx);
}

// One client's round of §3.1 with the server's blocks left out (the bottom's output handed
// straight to the top): tokens / labels int32 [b * L] (b rows of L tokens; a label < 0
// carries no target); x = Embedding(tokens), h0 = Block_0(x), z = Block_{N-1}(h0),
// logits = LN_f(z) head^T, loss = the mean over the tokens with a target of
// -log softmax(logits)[label]; then the chain rule back to the embedding table.
// Both blocks see the rows as b segments of length L (GLM: ctx / mask_pos [b] as in
// flo_server_fwd_bwd_ext) and, with prefix_len > 0, their own prefixes (bottom[12..13],
// top[12..13]).  Parameters: embed [V, H], bottom / top 12 (+ 2) pointers in the server
// order, lnf_gamma / lnf_beta [H], head [V, H]; their gradients are ADDED into g_embed,
// g_bottom, g_top (same counts), g_lnf (2 pointers) and g_head.  *loss receives the loss.
// Returns 0, or -1 on a bad argument (a token outside [0, vocab), a label >= vocab).
int flo_client_round(const flo_shape* shp, int32_t vocab, int32_t b, int32_t L, const int32_t* tokens,
                     const int32_t* labels, const int32_t* ctx, const int32_t* mask_pos, int32_t prefix_len,
                     const float* embed, const float* const* bottom, const float* const* top, const float* lnf_gamma,
                     const float* lnf_beta, const float* head, float* g_embed, float* const* g_bottom,
                     float* const* g_top, float* const* g_lnf, float* g_head, float* loss) {
  if (!shp || vocab < 1 || b < 1 || L < 1 || !tokens || !labels || prefix_len < 0 || !embed || !bottom || !top ||
      !lnf_gamma || !lnf_beta || !head || !g_embed || !g_bottom || !g_top || !g_lnf || !g_head || !loss)
    return -1;
  const flo_shape sh = *shp;
  if (sh.hidden != sh.n_heads * sh.head_dim || sh.rotary_dim < 2 || sh.rotary_dim % 2 ||
      sh.rotary_dim > sh.head_dim || (ctx && 2 * sh.rotary_dim != sh.head_dim))
    return -1;
  const int S = b, T = b * L, H = sh.hidden, V = vocab, Lp = prefix_len;
  for (int t = 0; t < T; ++t)
    if (tokens[t] < 0 || tokens[t] >= V || labels[t] >= V) return -1;
  std::vector<int32_t> cu(S + 1);
  for (int s = 0; s <= S; ++s) cu[s] = s * L;
  Positions ps;
  if (!make_positions(sh, S, cu.data(), ctx, mask_pos, ps)) return -1;
  const Block Pb{bottom[0], bottom[1], bottom[2], bottom[3], bottom[4], bottom[5],
                 bottom[6], bottom[7], bottom[8], bottom[9], bottom[10], bottom[11]};
  const Block Pt{top[0], top[1], top[2], top[3], top[4], top[5], top[6], top[7], top[8], top[9], top[10], top[11]};
  const float* bpk = Lp ? bottom[12] : nullptr;
  const float* bpv = Lp ? bottom[13] : nullptr;
  const float* tpk = Lp ? top[12] : nullptr;
  const float* tpv = Lp ? top[13] : nullptr;
  // forward: embedding rows, the two blocks, final LayerNorm, LM head
  Vec x((size_t)T * H), h0((size_t)T * H), z((size_t)T * H), zn((size_t)T * H), mu(T), rs(T);
  for (int t = 0; t < T; ++t)
    std::memcpy(x.data() + (size_t)t * H, embed + (size_t)tokens[t] * H, sizeof(float) * H);
  Saved svb, svt;
  block_fwd(Pb, x.data(), h0.data(), svb, sh, T, S, cu.data(), ps, bpk, bpv, Lp);
  block_fwd(Pt, h0.data(), z.data(), svt, sh, T, S, cu.data(), ps, tpk, tpv, Lp);
  layer_norm_fwd(z.data(), lnf_gamma, lnf_beta, sh.ln_eps, zn.data(), mu.data(), rs.data(), T, H);
  Vec logits((size_t)T * V);
  matmul_nt(zn.data(), head, nullptr, logits.data(), T, V, H);
  // cross-entropy over the rows with a target, and its gradient w.r.t. the logits
  int n = 0;
  for (int t = 0; t < T; ++t) n += labels[t] >= 0;
  const float inv_n = 1.f / (float)(n > 0 ? n : 1);
  Vec row_loss(T, 0.f);
#pragma omp parallel for schedule(static)
  for (int t = 0; t < T; ++t) {
    float* r = logits.data() + (size_t)t * V;
    if (labels[t] < 0) {
      for (int v = 0; v < V; ++v) r[v] = 0.f;
      continue;
    }
    float mx = -INFINITY;
    for (int v = 0; v < V; ++v) mx = std::fmax(mx, r[v]);
    float l = 0.f;
    for (int v = 0; v < V; ++v) l += std::exp(r[v] - mx);
    const float lse = mx + std::log(l);
    row_loss[t] = lse - r[labels[t]];
    for (int v = 0; v < V; ++v) r[v] = std::exp(r[v] - lse);
    r[labels[t]] -= 1.f;
    for (int v = 0; v < V; ++v) r[v] *= inv_n;
  }
  float sum = 0.f;
  for (int t = 0; t < T; ++t) sum += row_loss[t];
  *loss = sum * inv_n;
  // backward: LM head, final LayerNorm, top block, bottom block, embedding rows
  const float* dlog = logits.data();
  matmul_tn_acc(dlog, zn.data(), g_head, T, V, H);
  Vec dzn((size_t)T * H), dz((size_t)T * H), dh0((size_t)T * H), dx((size_t)T * H);
  matmul_nn(dlog, head, dzn.data(), T, V, H);
  layer_norm_bwd(dzn.data(), z.data(), mu.data(), rs.data(), lnf_gamma, dz.data(), g_lnf[0], g_lnf[1], T, H);
  block_bwd(Pt, g_top, svt, dz.data(), dh0.data(), sh, T, S, cu.data(), ps, tpk, tpv, Lp, Lp ? g_top[12] : nullptr,
            Lp ? g_top[13] : nullptr);
  block_bwd(Pb, g_bottom, svb, dh0.data(), dx.data(), sh, T, S, cu.data(), ps, bpk, bpv, Lp,
            Lp ? g_bottom[12] : nullptr, Lp ? g_bottom[13] : nullptr);
  for (int t = 0; t < T; ++t) {  // rows of repeated tokens accumulate in token order
    float* g = g_embed + (size_t)tokens[t] * H;
    const float* d = dx.data() + (size_t)t * H;
    for (int i = 0; i < H; ++i) g[i] += d[i];
  }
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
