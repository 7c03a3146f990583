"""The oracle's pins catch plausible mistakes (CPU only).

Each case plants one mistake in the fp64 oracle (a wrapper around one of its functions,
swapped in for the test's duration: a dropped term, a sign, a wrong operand or index, a
wrong constant) and runs the pins of `test_oracle_pins.py` that should notice it; at least
one of them must fail with an assertion.  The same pins pass on the unmodified oracle (in
`test_oracle_pins.py`), so each failure here is the planted mistake's: a pin set that
passed with the mistake in place could not tell the oracle from the mistake.
"""
import math

import numpy as np
import pytest

import test_oracle_pins as P
from oracle import flglm_oracle as O


def _ln_beta_dropped(orig):
    return lambda x, g, b, eps: orig(x, g, np.zeros_like(b), eps)


def _ln_eps_dropped(orig):
    return lambda x, g, b, eps: orig(x, g, b, 0.0)


def _ln_bwd_dgamma_sign(orig):
    def f(*a):
        dx, dg, db = orig(*a)
        return dx, -dg, db
    return f


def _ln_bwd_gamma_ignored(orig):
    return lambda dy, x, mu, rstd, gamma: orig(dy, x, mu, rstd, np.ones_like(gamma))


def _gelu_erf(orig):
    from scipy.special import erf
    return lambda u: 0.5 * u * (1.0 + erf(u / math.sqrt(2.0)))


def _gelu_grad_at_output(orig):
    return lambda u: orig(O.gelu(u))


def _attn_scale_over_d(orig):
    def f(q, k, v, cu, *a, **kw):
        return orig(q / math.sqrt(q.shape[-1]), k, v, cu, *a, **kw)
    return f


def _attn_segments_mixed(orig):
    def f(q, k, v, cu, *a, **kw):
        kw.pop("ctx", None)
        return orig(q, k, v, np.array([0, q.shape[0]], np.int32), *a, **kw)
    return f


def _mask_sees_next_token(orig):
    def f(L, Lp, c=0):
        m = orig(L, Lp, c).copy()
        for t in range(L - 1):
            m[t, Lp + t + 1] = True
        return m
    return f


def _mask_prefix_causal(orig):
    def f(L, Lp, c=0):
        m = orig(L, Lp, c).copy()
        m[:, :Lp] = np.tril(np.ones((L, Lp), bool))
        return m
    return f


def _glm_context_causal(orig):
    return lambda ctx, s: 0


def _glm_block_position_from_zero(orig):
    def f(L, c, mask_pos):
        p1, p2 = orig(L, c, mask_pos)
        p2 = p2.copy()
        p2[p2 > 0] -= 1
        return p1, p2
    return f


def _attn_bwd_dk_dv_swapped(orig):
    def f(*a, **kw):
        r = list(orig(*a, **kw))
        r[1], r[2] = r[2], r[1]
        return tuple(r)
    return f


def _attn_bwd_dq_unscaled(orig):
    def f(do, q, *a, **kw):
        r = list(orig(do, q, *a, **kw))
        r[0] = r[0] * math.sqrt(q.shape[-1])
        return tuple(r)
    return f


def _rope_direction(orig):
    return lambda x, cos, sin, rd, inverse=False: orig(x, cos, -sin, rd, inverse)


def _rope_base(orig):
    return lambda pos, rd, base: orig(pos, rd, math.sqrt(base))


def _rope_interleaved_pairs(orig):
    def f(x, cos, sin, rd, inverse=False):
        # rotate (2i, 2i + 1) instead of (i, i + rd/2): permute into rotate-half order and back
        perm = np.concatenate([np.arange(0, rd, 2), np.arange(1, rd, 2), np.arange(rd, x.shape[-1])])
        inv = np.argsort(perm)
        return orig(x[..., perm], cos, sin, rd, inverse)[..., inv]
    return f


def _rope_no_inverse(orig):
    return lambda x, pk, rd, base, inverse=False: orig(x, pk, rd, base, False)


def _pack_seq_major(orig):
    def f(ts):
        H = ts[0].shape[-1]
        return np.concatenate([t.transpose(1, 0, 2).reshape(-1, H) for t in ts], axis=0)
    return f


def _wgrad_mean_over_tokens(orig):
    def f(params, saved, dy, pk, sh):
        dx, grads = orig(params, saved, dy, pk, sh)
        return dx, [[g / dy.shape[0] for g in blk] for blk in grads]
    return f


def _adamw_no_bias_correction(orig):
    return lambda w, g, m, v, t, lr, b1, b2, eps, wd: orig(w, g, m, v, 10 ** 9, lr, b1, b2, eps, wd)


def _adamw_coupled_decay(orig):
    return lambda w, g, m, v, t, lr, b1, b2, eps, wd: orig(w, g + wd * w, m, v, t, lr, b1, b2, eps, 0.0)


def _alpha_ignored(orig):
    def f(cfg):
        sh = orig(cfg)
        sh.alpha = 1.0
        return sh
    return f


def _embedding_bwd_overwrites(orig):
    def f(dX, tokens, vocab):
        dE = np.zeros((vocab, dX.shape[1]))
        dE[tokens] = dX  # a repeated token keeps one occurrence's gradient, not the sum
        return dE
    return f


def _ce_mean_over_all_rows(orig):
    def f(logits, labels):
        loss, d = orig(logits, labels)
        n, T = int((labels >= 0).sum()), labels.shape[0]
        return (loss * n / T, d * n / T) if n else (loss, d)
    return f


def _ce_ignored_rows_keep_gradient(orig):
    def f(logits, labels):
        loss, d = orig(logits, labels)
        d = d.copy()
        ign = labels < 0
        if ign.any() and (~ign).any():
            sm = np.exp(logits[ign] - logits[ign].max(-1, keepdims=True))
            d[ign] = sm / sm.sum(-1, keepdims=True) / int((~ign).sum())
        return loss, d
    return f


def _prefix_grads_halved(orig):
    def f(*a, **kw):
        r = list(orig(*a, **kw))
        if len(r) == 5:  # a prefix: dq, dk, dv, dprefix_k, dprefix_v
            r[3], r[4] = 0.5 * r[3], 0.5 * r[4]
        return tuple(r)
    return f


def _glm_context_one_short(orig):
    return lambda ctx, s: max(orig(ctx, s) - 1, 0)


def _rope_2d_second_half_fixed(orig):
    def f(x, pk, rd, base, inverse=False):
        out = orig(x, pk, rd, base, inverse)
        if pk.pos2 is not None:
            out = out.copy()
            out[..., rd:] = x[..., rd:]  # block position ignored
        return out
    return f


FD = lambda: P.test_finite_difference_gradients(1)  # noqa: E731

# (mistake, oracle attribute, mutant factory, pins that should catch it)
CASES = [
    ("LayerNorm drops beta", "layer_norm_fwd", _ln_beta_dropped, [P.test_layer_norm_matches_torch_and_row_stats]),
    ("LayerNorm drops eps", "layer_norm_fwd", _ln_eps_dropped, [P.test_layer_norm_matches_torch_and_row_stats]),
    ("LayerNorm backward: dgamma sign", "layer_norm_bwd", _ln_bwd_dgamma_sign, [FD]),
    ("LayerNorm backward: gamma left out of dx", "layer_norm_bwd", _ln_bwd_gamma_ignored, [FD]),
    ("GeLU in the erf form", "gelu", _gelu_erf, [P.test_gelu_matches_torch_tanh_form]),
    ("GeLU derivative taken at the output", "gelu_grad", _gelu_grad_at_output, [FD]),
    ("softmax scale 1/d_h", "attention_fwd", _attn_scale_over_d,
     [P.test_attention_matches_torch_sdpa_per_segment, P.test_attention_brute_force_global_mask]),
    ("segments attend to each other", "attention_fwd", _attn_segments_mixed,
     [P.test_attention_matches_torch_sdpa_per_segment, P.test_causality_and_segment_isolation]),
    ("causal mask admits the next token", "_mask", _mask_sees_next_token,
     [P.test_attention_matches_torch_sdpa_per_segment]),
    ("prefix keys masked causally", "_mask", _mask_prefix_causal, [P.test_prefix_attention_matches_torch_sdpa]),
    ("GLM context not bidirectional", "_ctx", _glm_context_causal,
     [lambda: P.test_glm_attention_matches_torch_sdpa(0), P.test_glm_context_is_bidirectional_and_span_causal]),
    ("GLM block positions from 0", "glm_positions", _glm_block_position_from_zero,
     [P.test_glm_positions_worked_example]),
    ("attention backward: dK and dV swapped", "attention_bwd", _attn_bwd_dk_dv_swapped, [FD]),
    ("attention backward: dQ without the softmax scale", "attention_bwd", _attn_bwd_dq_unscaled, [FD]),
    ("RoPE turns the other way", "rope_rotate", _rope_direction, [P.test_rope_properties]),
    ("RoPE frequency base", "rope_cos_sin", _rope_base, [P.test_rope_properties]),
    ("RoPE pairs adjacent dims", "rope_rotate", _rope_interleaved_pairs, [P.test_rope_properties]),
    ("backward without the inverse rotation", "rope_2d", _rope_no_inverse, [FD]),
    ("pack takes a client's rows token by token", "pack", _pack_seq_major,
     [P.test_pack_unpack_roundtrip_and_metadata]),
    ("weight gradients averaged over tokens", "stack_bwd", _wgrad_mean_over_tokens, [FD]),
    ("AdamW without bias correction", "adamw_update", _adamw_no_bias_correction,
     [P.test_adamw_first_step_closed_form, P.test_adamw_matches_torch_over_steps]),
    ("AdamW with coupled (L2) decay", "adamw_update", _adamw_coupled_decay,
     [P.test_adamw_first_step_closed_form, P.test_adamw_matches_torch_over_steps]),
    ("embedding gradient overwrites repeated tokens", "embedding_bwd", _embedding_bwd_overwrites,
     [P.test_embedding_matches_torch]),
    ("cross-entropy averaged over rows without a target", "cross_entropy", _ce_mean_over_all_rows,
     [P.test_cross_entropy_matches_torch, P.test_cross_entropy_uniform_closed_form]),
    ("cross-entropy gradient on rows without a target", "cross_entropy", _ce_ignored_rows_keep_gradient,
     [P.test_cross_entropy_matches_torch, P.test_cross_entropy_uniform_closed_form]),
    ("prefix gradients halved", "attention_bwd", _prefix_grads_halved,
     [lambda: P.test_finite_difference_prefix_gradients(1)]),
    ("GLM context one token short", "_ctx", _glm_context_one_short,
     [lambda: P.test_glm_attention_matches_torch_sdpa(0), P.test_glm_context_is_bidirectional_and_span_causal]),
    ("2D rotary ignores the block position", "rope_2d", _rope_2d_second_half_fixed,
     [P.test_rope_2d_properties]),
    ("residual scale alpha ignored", "BlockShape.of", _alpha_ignored,
     [lambda: P.test_zero_weight_block_closed_form(1), lambda: P.test_zero_weight_block_closed_form(0)]),
]


@pytest.mark.parametrize("name,attr,factory,pins", CASES, ids=[c[0] for c in CASES])
def test_pins_catch_planted_mistake(monkeypatch, name, attr, factory, pins):
    if attr == "BlockShape.of":
        monkeypatch.setattr(O.BlockShape, "of", staticmethod(factory(O.BlockShape.of)))
    else:
        monkeypatch.setattr(O, attr, factory(getattr(O, attr)))
    failed = []
    for pin in pins:
        try:
            pin()
        except AssertionError:
            failed.append(pin)
    assert failed, f"no pin noticed: {name}"

