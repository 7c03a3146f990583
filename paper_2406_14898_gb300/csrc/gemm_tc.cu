// fl_k_gemm: argument checks, epilogue set-up and dispatch to the instantiation of the
// operand layout, tile width and epilogue family (kernels: gemm_tc.cuh; instantiations:
// gemm_inst_fwd.cu, gemm_inst_dgrad.cu, gemm_inst_wgrad.cu).
#include <cstring>

#include "gemm_tc.cuh"

namespace fl_gemm {
#define FL_GEMM_EXTERN(AMN, BMN, FAM)                                                                   \
  extern template int pair_slots<AMN, BMN, FAM>();                                                      \
  extern template int launch_pair<AMN, BMN, FAM>(const fl_gemm_args*, const Problems&, const Epi&, int*, cudaStream_t);  \
  extern template int launch<256, AMN, BMN, FAM>(const fl_gemm_args*, const Problems&, const Epi&, int*, cudaStream_t); \
  extern template int launch<128, AMN, BMN, FAM>(const fl_gemm_args*, const Problems&, const Epi&, int*, cudaStream_t);
#define FL_GEMM_EXTERN_ALL(AMN, BMN)                                                                   \
  FL_GEMM_EXTERN(AMN, BMN, FAM_PLAIN) FL_GEMM_EXTERN(AMN, BMN, FAM_GELU) FL_GEMM_EXTERN(AMN, BMN, FAM_RESID) \
  FL_GEMM_EXTERN(AMN, BMN, FAM_ROPE) FL_GEMM_EXTERN(AMN, BMN, FAM_ADAMW)
FL_GEMM_EXTERN_ALL(false, false)
FL_GEMM_EXTERN_ALL(false, true)
FL_GEMM_EXTERN_ALL(true, true)

// Tile shape: 0 = 128 x 128 on one SM, 1 = 128 x 256 on one SM, 2 = 256 x 256 on a CTA pair.
template <bool AMN, bool BMN>
int dispatch_layout(int fam, int shape, const fl_gemm_args* a, const Problems& pr, const Epi& e, int* status,
                    cudaStream_t st) {
  if (shape == 2) {
    switch (fam) {
      case FAM_GELU: return launch_pair<AMN, BMN, FAM_GELU>(a, pr, e, status, st);
      case FAM_RESID: return launch_pair<AMN, BMN, FAM_RESID>(a, pr, e, status, st);
      case FAM_ROPE: return launch_pair<AMN, BMN, FAM_ROPE>(a, pr, e, status, st);
      case FAM_ADAMW: return launch_pair<AMN, BMN, FAM_ADAMW>(a, pr, e, status, st);
      default: return launch_pair<AMN, BMN, FAM_PLAIN>(a, pr, e, status, st);
    }
  }
  const bool wide = shape == 1;
  switch (fam) {
    case FAM_GELU: return wide ? launch<256, AMN, BMN, FAM_GELU>(a, pr, e, status, st) : launch<128, AMN, BMN, FAM_GELU>(a, pr, e, status, st);
    case FAM_RESID: return wide ? launch<256, AMN, BMN, FAM_RESID>(a, pr, e, status, st) : launch<128, AMN, BMN, FAM_RESID>(a, pr, e, status, st);
    case FAM_ROPE: return wide ? launch<256, AMN, BMN, FAM_ROPE>(a, pr, e, status, st) : launch<128, AMN, BMN, FAM_ROPE>(a, pr, e, status, st);
    case FAM_ADAMW: return wide ? launch<256, AMN, BMN, FAM_ADAMW>(a, pr, e, status, st) : launch<128, AMN, BMN, FAM_ADAMW>(a, pr, e, status, st);
    default: return wide ? launch<256, AMN, BMN, FAM_PLAIN>(a, pr, e, status, st) : launch<128, AMN, BMN, FAM_PLAIN>(a, pr, e, status, st);
  }
}

int dispatch_fam(int fam, int shape, bool amn, bool bmn, const fl_gemm_args* a, const Problems& pr, const Epi& e,
                 int* status, cudaStream_t st) {
  if (!amn && !bmn) return dispatch_layout<false, false>(fam, shape, a, pr, e, status, st);
  if (!amn && bmn) return dispatch_layout<false, true>(fam, shape, a, pr, e, status, st);
  return dispatch_layout<true, true>(fam, shape, a, pr, e, status, st);
}

int pair_slots_for(int fam, bool amn, bool bmn) {
#define FL_SLOTS(AMN, BMN)                                          \
  switch (fam) {                                                    \
    case FAM_GELU: return pair_slots<AMN, BMN, FAM_GELU>();         \
    case FAM_RESID: return pair_slots<AMN, BMN, FAM_RESID>();       \
    case FAM_ROPE: return pair_slots<AMN, BMN, FAM_ROPE>();         \
    case FAM_ADAMW: return pair_slots<AMN, BMN, FAM_ADAMW>();       \
    default: return pair_slots<AMN, BMN, FAM_PLAIN>();              \
  }
  if (!amn && !bmn) { FL_SLOTS(false, false) }
  if (!amn && bmn) { FL_SLOTS(false, true) }
  FL_SLOTS(true, true)
#undef FL_SLOTS
}
}  // namespace fl_gemm

using namespace fl_gemm;

namespace {

// Checks one problem's arguments (everything but the batch fields).
int check_args(const fl_gemm_args* a) {
  if (!a || !a->A || !a->B || !a->D) return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: null pointer");
  if (a->M < 0 || a->N <= 0 || a->K <= 0) return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: bad sizes");
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
  if ((mode == FL_EPI_BIAS_GELU || mode == FL_EPI_ADAMW) &&
      (!a->aux_out || (a->ld_aux_out % 8) || !aligned16(a->aux_out)))
    return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: epilogue needs an aligned aux_out");
  if (mode == FL_EPI_ADAMW && (!a->adam_m || !a->adam_v || !aligned16(a->adam_m) || !aligned16(a->adam_v) ||
                               a->bias || (a->ldd % 4)))
    return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: AdamW epilogue needs aligned moments and no bias");
  if (mode == FL_EPI_BIAS_ROPE) {
    if (!a->pos || !a->rope_tab || a->head_dim <= 0 || a->head_dim % 64 ||
        !(a->rotary_dim == 32 || a->rotary_dim == 64) || a->rotary_dim > a->head_dim)
      return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: RoPE epilogue arguments");
    if (a->pos2 && 2 * a->rotary_dim != a->head_dim)
      return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: 2D rotary needs rotary_dim = head_dim / 2");
  } else if (a->pos2) {
    return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: block positions only with the RoPE epilogue");
  }
  if (a->bias && !aligned16(a->bias)) return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: bias alignment");
  if (fl_misaligned(a->rope_tab, 8) || fl_misaligned(a->pos, 4) || fl_misaligned(a->pos2, 4) ||
      fl_misaligned(a->ln_mean, 4) || fl_misaligned(a->ln_rstd, 4))
    return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: rope_tab must be 8-byte and per-row arrays 4-byte aligned");
  if (a->colsum && mode != FL_EPI_GELU_BWD)
    return fl_internal_error(FL_ERR_UNSUPPORTED, "gemm: column sums only with the GeLU-backward epilogue");
  if (a->colsum && !aligned16(a->colsum))
    return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: colsum must be 16-byte aligned");
  if (a->tile < FL_TILE_AUTO || a->tile > FL_TILE_256x256_PAIR)
    return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: tile %d", a->tile);
  if (a->tile >= FL_TILE_128x256 && (a->N % 256))
    return fl_internal_error(FL_ERR_UNSUPPORTED, "gemm: 256-column tiles need N %% 256 == 0 (N=%d)", a->N);
  if (a->a_mn_major && !a->b_mn_major)
    return fl_internal_error(FL_ERR_UNSUPPORTED, "gemm: MN-major A with K-major B is not built");
  return FL_OK;
}

// The epilogue of problem 0 (offsets of the other problems zero).
Epi make_epi(const fl_gemm_args* a) {
  const int mode = a->epilogue;
  Epi e;
  memset(&e, 0, sizeof e);
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
  e.pos2 = a->pos2;
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
  e.adam_m = a->adam_m;
  e.adam_v = a->adam_v;
  e.lr = a->lr;
  e.b1 = a->beta1;
  e.b2 = a->beta2;
  e.eps = a->eps;
  e.wd = a->weight_decay;
  e.inv_bc1 = a->inv_bc1;
  e.inv_bc2 = a->inv_bc2;
  e.colsum = a->colsum;
  return e;
}

bool d_is_f32(const fl_gemm_args* a) {
  const int mode = a->epilogue;
  return a->d_dtype == FL_DT_F32 || mode == FL_EPI_STORE_F32 || mode == FL_EPI_ACCUM_F32 || mode == FL_EPI_ADAMW;
}

// Tile shape for the launch (see fl_k_gemm) and the dispatch.
int run(const fl_gemm_args* a, const Problems& pr, const Epi& e, int* status, cudaStream_t st) {
  const bool amn = a->a_mn_major != 0, bmn = a->b_mn_major != 0;
  const int fam = family_of(a->epilogue);
  const int batch = pr.n;
  if (a->tile == FL_TILE_256x256_PAIR && pair_slots_for(fam, amn, bmn) <= 0)
    return fl_internal_error(FL_ERR_UNSUPPORTED, "gemm: this device cannot hold the CTA-pair kernel");
  if (a->tile != FL_TILE_AUTO) return dispatch_fam(fam, a->tile - 1, amn, bmn, a, pr, e, status, st);
  // Tile shape: 256 columns (on a CTA pair where the device can hold pairs) unless
  // 128 x 128 tiles give clearly fewer idle SM slots in the last wave.
  int shape = 0;
  if ((a->N % 256) == 0) {
    const int sms = num_sms();
    const int pairs = pair_slots_for(fam, amn, bmn);
    const long t128 = (long)batch * ((a->M + BM - 1) / BM) * (a->N / 128);
    const double eff128 = double(t128) / double(((t128 + sms - 1) / sms) * sms);
    double eff_wide;
    if (pairs > 0) {
      const long tp = (long)batch * ((a->M + PAIR_BM - 1) / PAIR_BM) * (a->N / PAIR_BN);
      eff_wide = double(tp) / double(((tp + pairs - 1) / pairs) * pairs);
      shape = 2;
    } else {
      const long t256 = (long)batch * ((a->M + BM - 1) / BM) * (a->N / 256);
      eff_wide = double(t256) / double(((t256 + sms - 1) / sms) * sms);
      shape = 1;
    }
    if (eff128 > eff_wide * 1.15) shape = 0;
  }
  return dispatch_fam(fam, shape, amn, bmn, a, pr, e, status, st);
}

// Element offset of p from p0 (both null, or both in the same address space; elem bytes).
int64_t elem_off(const void* p, const void* p0, int elem) {
  return (reinterpret_cast<intptr_t>(p) - reinterpret_cast<intptr_t>(p0)) / elem;
}

}  // namespace

extern "C" int fl_k_gemm(const fl_gemm_args* a, int* status, void* stream) {
  if (int rc = check_args(a)) return rc;
  if (a->M == 0) return FL_OK;
  if (a->batch < 0 || a->batch > FL_GEMM_MAX_BATCH)
    return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: batch %d outside 0..%d", a->batch, FL_GEMM_MAX_BATCH);
  const int batch = a->batch > 1 ? a->batch : 1;
  if (batch > 1) {
    // every problem's pointers keep the 16-byte alignment of the first problem's: strides in
    // bf16 elements multiples of 8, in fp32 elements multiples of 4 (and of 4 for the
    // per-row int32 / fp32 arrays read one element at a time)
    const bool d32 = d_is_f32(a);
    if ((a->a_bstride % 8) || (a->b_bstride % 8) || (a->d_bstride % (d32 ? 4 : 8)) ||
        (a->aux && (a->aux_bstride % (a->aux_dtype == FL_DT_F32 ? 4 : 8))) || (a->aux_out && (a->aux_out_bstride % 8)) ||
        ((a->bias || a->colsum) && (a->bias_bstride % 4)) || (a->ln_mean && (a->lnp_bstride % 4)) ||
        (a->adam_m && (a->adam_bstride % 4)))
      return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: batch strides break the 16-byte alignment");
  }
  Epi e = make_epi(a);
  Problems pr;
  memset(&pr, 0, sizeof pr);
  pr.n = batch;
  for (int r = 0; r < batch; ++r) {
    pr.A[r] = static_cast<const __nv_bfloat16*>(a->A) + r * a->a_bstride;
    pr.B[r] = static_cast<const __nv_bfloat16*>(a->B) + r * a->b_bstride;
    pr.lda[r] = a->lda;
    pr.ldb[r] = a->ldb;
    e.o_d[r] = r * a->d_bstride;
    e.o_aux[r] = r * a->aux_bstride;
    e.o_aux_out[r] = r * a->aux_out_bstride;
    e.o_bias[r] = r * a->bias_bstride;
    e.o_row[r] = r * a->row_bstride;
    e.o_lnp[r] = r * a->lnp_bstride;
    e.o_adam[r] = r * a->adam_bstride;
  }
  return run(a, pr, e, status, reinterpret_cast<cudaStream_t>(stream));
}

extern "C" int fl_k_gemm_multi(const fl_gemm_args* probs, int32_t n, int* status, void* stream) {
  if (!probs || n < 1 || n > FL_GEMM_MAX_BATCH)
    return fl_internal_error(FL_ERR_INVALID_ARG, "gemm multi: need 1..%d problems", FL_GEMM_MAX_BATCH);
  const fl_gemm_args* a = probs;
  for (int r = 0; r < n; ++r) {
    const fl_gemm_args* q = probs + r;
    if (int rc = check_args(q)) return rc;
    if (q->batch > 1) return fl_internal_error(FL_ERR_INVALID_ARG, "gemm multi: problem %d has batch %d", r, q->batch);
    // one shape, layout, epilogue and set of scalars; output leading dimensions shared
    const bool same = q->M == a->M && q->N == a->N && q->K == a->K && q->a_mn_major == a->a_mn_major &&
                      q->b_mn_major == a->b_mn_major && q->epilogue == a->epilogue && q->ldd == a->ldd &&
                      q->ld_aux == a->ld_aux && q->ld_aux_out == a->ld_aux_out && q->aux_dtype == a->aux_dtype &&
                      q->d_dtype == a->d_dtype && q->alpha == a->alpha && q->lr == a->lr && q->beta1 == a->beta1 &&
                      q->beta2 == a->beta2 && q->eps == a->eps && q->weight_decay == a->weight_decay &&
                      q->inv_bc1 == a->inv_bc1 && q->inv_bc2 == a->inv_bc2 && q->n_heads == a->n_heads &&
                      q->head_dim == a->head_dim && q->rotary_dim == a->rotary_dim && q->rope_tab == a->rope_tab &&
                      q->tile == a->tile;
    if (!same) return fl_internal_error(FL_ERR_INVALID_ARG, "gemm multi: problem %d differs in shape or epilogue", r);
    // each optional operand present in every problem or in none
    const bool present = (!q->aux == !a->aux) && (!q->aux_out == !a->aux_out) && (!q->bias == !a->bias) &&
                         (!q->colsum == !a->colsum) && (!q->pos == !a->pos) && (!q->pos2 == !a->pos2) &&
                         (!q->ln_mean == !a->ln_mean) && (!q->adam_m == !a->adam_m);
    if (!present) return fl_internal_error(FL_ERR_INVALID_ARG, "gemm multi: problem %d lacks an operand", r);
  }
  if (a->M == 0) return FL_OK;
  Epi e = make_epi(a);
  Problems pr;
  memset(&pr, 0, sizeof pr);
  pr.n = n;
  const int d_el = d_is_f32(a) ? 4 : 2, aux_el = a->aux_dtype == FL_DT_F32 ? 4 : 2;
  for (int r = 0; r < n; ++r) {
    const fl_gemm_args* q = probs + r;
    pr.A[r] = q->A;
    pr.B[r] = q->B;
    pr.lda[r] = q->lda;
    pr.ldb[r] = q->ldb;
    // offsets from problem 0's pointers: every pointer is 16-byte aligned, so each offset
    // keeps the vector alignment the epilogue relies on
    e.o_d[r] = elem_off(q->D, a->D, d_el);
    e.o_aux[r] = a->aux ? elem_off(q->aux, a->aux, aux_el) : 0;
    e.o_aux_out[r] = a->aux_out ? elem_off(q->aux_out, a->aux_out, 2) : 0;
    e.o_bias[r] = a->bias ? elem_off(q->bias, a->bias, 4) : a->colsum ? elem_off(q->colsum, a->colsum, 4) : 0;
    if (a->bias && a->colsum && elem_off(q->colsum, a->colsum, 4) != e.o_bias[r])
      return fl_internal_error(FL_ERR_INVALID_ARG, "gemm multi: bias and colsum offsets differ");
    e.o_row[r] = a->pos ? elem_off(q->pos, a->pos, 4) : a->ln_mean ? elem_off(q->ln_mean, a->ln_mean, 4) : 0;
    if ((a->pos2 && elem_off(q->pos2, a->pos2, 4) != e.o_row[r]) ||
        (a->ln_mean && (elem_off(q->ln_mean, a->ln_mean, 4) != e.o_row[r] ||
                        elem_off(q->ln_rstd, a->ln_rstd, 4) != e.o_row[r])))
      return fl_internal_error(FL_ERR_INVALID_ARG, "gemm multi: per-row operand offsets differ");
    e.o_lnp[r] = a->ln_gamma ? elem_off(q->ln_gamma, a->ln_gamma, 4) : 0;
    if (a->ln_gamma && elem_off(q->ln_beta, a->ln_beta, 4) != e.o_lnp[r])
      return fl_internal_error(FL_ERR_INVALID_ARG, "gemm multi: LayerNorm gain and shift offsets differ");
    e.o_adam[r] = a->adam_m ? elem_off(q->adam_m, a->adam_m, 4) : 0;
    if (a->adam_m && elem_off(q->adam_v, a->adam_v, 4) != e.o_adam[r])
      return fl_internal_error(FL_ERR_INVALID_ARG, "gemm multi: Adam moment offsets differ");
  }
  return run(a, pr, e, status, reinterpret_cast<cudaStream_t>(stream));
}
