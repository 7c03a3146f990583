// fl_k_gemm: argument checks, epilogue set-up and dispatch to the instantiation of the
// operand layout, tile width and epilogue family (kernels: gemm_tc.cuh; instantiations:
// gemm_inst_fwd.cu, gemm_inst_dgrad.cu, gemm_inst_wgrad.cu).
#include "gemm_tc.cuh"

namespace fl_gemm {
#define FL_GEMM_EXTERN(AMN, BMN, FAM)                                                                   \
  extern template int pair_slots<AMN, BMN, FAM>();                                                      \
  extern template int launch_pair<AMN, BMN, FAM>(const fl_gemm_args*, const Epi&, int*, cudaStream_t);  \
  extern template int launch<256, AMN, BMN, FAM>(const fl_gemm_args*, const Epi&, int*, cudaStream_t); \
  extern template int launch<128, AMN, BMN, FAM>(const fl_gemm_args*, const Epi&, int*, cudaStream_t);
#define FL_GEMM_EXTERN_ALL(AMN, BMN)                                                                   \
  FL_GEMM_EXTERN(AMN, BMN, FAM_PLAIN) FL_GEMM_EXTERN(AMN, BMN, FAM_GELU) FL_GEMM_EXTERN(AMN, BMN, FAM_RESID) \
  FL_GEMM_EXTERN(AMN, BMN, FAM_ROPE) FL_GEMM_EXTERN(AMN, BMN, FAM_ADAMW)
FL_GEMM_EXTERN_ALL(false, false)
FL_GEMM_EXTERN_ALL(false, true)
FL_GEMM_EXTERN_ALL(true, true)

// Tile shape: 0 = 128 x 128 on one SM, 1 = 128 x 256 on one SM, 2 = 256 x 256 on a CTA pair.
template <bool AMN, bool BMN>
int dispatch_layout(int fam, int shape, const fl_gemm_args* a, const Epi& e, int* status, cudaStream_t st) {
  if (shape == 2) {
    switch (fam) {
      case FAM_GELU: return launch_pair<AMN, BMN, FAM_GELU>(a, e, status, st);
      case FAM_RESID: return launch_pair<AMN, BMN, FAM_RESID>(a, e, status, st);
      case FAM_ROPE: return launch_pair<AMN, BMN, FAM_ROPE>(a, e, status, st);
      case FAM_ADAMW: return launch_pair<AMN, BMN, FAM_ADAMW>(a, e, status, st);
      default: return launch_pair<AMN, BMN, FAM_PLAIN>(a, e, status, st);
    }
  }
  const bool wide = shape == 1;
  switch (fam) {
    case FAM_GELU: return wide ? launch<256, AMN, BMN, FAM_GELU>(a, e, status, st) : launch<128, AMN, BMN, FAM_GELU>(a, e, status, st);
    case FAM_RESID: return wide ? launch<256, AMN, BMN, FAM_RESID>(a, e, status, st) : launch<128, AMN, BMN, FAM_RESID>(a, e, status, st);
    case FAM_ROPE: return wide ? launch<256, AMN, BMN, FAM_ROPE>(a, e, status, st) : launch<128, AMN, BMN, FAM_ROPE>(a, e, status, st);
    case FAM_ADAMW: return wide ? launch<256, AMN, BMN, FAM_ADAMW>(a, e, status, st) : launch<128, AMN, BMN, FAM_ADAMW>(a, e, status, st);
    default: return wide ? launch<256, AMN, BMN, FAM_PLAIN>(a, e, status, st) : launch<128, AMN, BMN, FAM_PLAIN>(a, e, status, st);
  }
}

int dispatch_fam(int fam, int shape, bool amn, bool bmn, const fl_gemm_args* a, const Epi& e, int* status,
                 cudaStream_t st) {
  if (!amn && !bmn) return dispatch_layout<false, false>(fam, shape, a, e, status, st);
  if (!amn && bmn) return dispatch_layout<false, true>(fam, shape, a, e, status, st);
  return dispatch_layout<true, true>(fam, shape, a, e, status, st);
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
  if (a->colsum && mode != FL_EPI_GELU_BWD)
    return fl_internal_error(FL_ERR_UNSUPPORTED, "gemm: column sums only with the GeLU-backward epilogue");
  if (a->colsum && !aligned16(a->colsum))
    return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: colsum must be 16-byte aligned");
  if (a->batch < 0 || a->batch > FL_GEMM_MAX_BATCH)
    return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: batch %d outside 0..%d", a->batch, FL_GEMM_MAX_BATCH);
  const int batch = a->batch > 1 ? a->batch : 1;
  if (batch > 1) {
    // every problem's pointers keep the 16-byte alignment of the first problem's: strides in
    // bf16 elements multiples of 8, in fp32 elements multiples of 4 (and of 4 for the
    // per-row int32 / fp32 arrays read one element at a time)
    const bool d32 = a->d_dtype == FL_DT_F32 || mode == FL_EPI_STORE_F32 || mode == FL_EPI_ACCUM_F32 ||
                     mode == FL_EPI_ADAMW;
    if ((a->a_bstride % 8) || (a->b_bstride % 8) || (a->d_bstride % (d32 ? 4 : 8)) ||
        (a->aux && (a->aux_bstride % (a->aux_dtype == FL_DT_F32 ? 4 : 8))) || (a->aux_out && (a->aux_out_bstride % 8)) ||
        ((a->bias || a->colsum) && (a->bias_bstride % 4)) || (a->ln_mean && (a->lnp_bstride % 4)) ||
        (a->adam_m && (a->adam_bstride % 4)))
      return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: batch strides break the 16-byte alignment");
  }

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
  e.bs_d = a->d_bstride;
  e.bs_aux = a->aux_bstride;
  e.bs_aux_out = a->aux_out_bstride;
  e.bs_bias = a->bias_bstride;
  e.bs_row = a->row_bstride;
  e.bs_lnp = a->lnp_bstride;
  e.bs_adam = a->adam_bstride;

  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const bool amn = a->a_mn_major != 0, bmn = a->b_mn_major != 0;
  if (amn && !bmn) return fl_internal_error(FL_ERR_UNSUPPORTED, "gemm: MN-major A with K-major B is not built");
  const int fam = family_of(mode);
  if (a->tile < FL_TILE_AUTO || a->tile > FL_TILE_256x256_PAIR)
    return fl_internal_error(FL_ERR_INVALID_ARG, "gemm: tile %d", a->tile);
  if (a->tile >= FL_TILE_128x256 && (a->N % 256))
    return fl_internal_error(FL_ERR_UNSUPPORTED, "gemm: 256-column tiles need N %% 256 == 0 (N=%d)", a->N);
  if (a->tile == FL_TILE_256x256_PAIR && pair_slots_for(fam, amn, bmn) <= 0)
    return fl_internal_error(FL_ERR_UNSUPPORTED, "gemm: this device cannot hold the CTA-pair kernel");
  if (a->tile != FL_TILE_AUTO) return dispatch_fam(fam, a->tile - 1, amn, bmn, a, e, status, st);
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
  return dispatch_fam(fam, shape, amn, bmn, a, e, status, st);
}
