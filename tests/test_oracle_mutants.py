"""Planted mistakes in the oracle must each fail at least one pin (no GPU).

Every entry patches one plausible mistake into a copy of oracle/cb_oracle.c (a
dropped term, a wrong sign, index or exponent, a transposed operand, a wrong
tie-break), builds it with gcc, and runs the pins of tests/oracle_pins.py on
it.  A mutant that passes every pin would mean the pins cannot see that
mistake.  All mutants keep every memory access in bounds for the pins' sizes.
"""
import concurrent.futures as cf
import os
import tempfile

import pytest

import oracle
import oracle_pins

MUTANTS = [
    ("gqa_mapping_in_attention", "load_keys_transposed(dm, K, l, h / G)", "load_keys_transposed(dm, K, l, h % dm->n_kv_heads)"),
    ("gqa_mapping_in_score", "const int h = g * G + j;", "const int h = j * Hkv + g;"),
    ("scale_dropped", "z[t] *= scale;", "z[t] *= 1.0;"),
    ("softmax_sign", "a[t] = exp(z[t] - M);", "a[t] = exp(M - z[t]);"),
    ("softmax_not_normalised", "for (int64_t t = 0; t < T; ++t) a[t] /= Z;", "(void)Z;"),
    ("q_operand_transposed", "(int64_t)r * dm->q_tok + (int64_t)h * dm->q_head", "(int64_t)h * dm->q_tok + (int64_t)r * dm->q_head"),
    ("k_dim_reversed", "bf16_to_double(base[t * dm->k_pos + k])", "bf16_to_double(base[t * dm->k_pos + (d - 1 - k)])"),
    ("k_position_shifted", "bf16_to_double(base[t * dm->k_pos + k])", "bf16_to_double(base[((t + 1) % T) * dm->k_pos + k])"),
    ("group_mean_missing_1_over_G", "br[t] += a[t] / G;", "br[t] += a[t];"),
    ("layer_term_over_kv_heads", "Us[t] += a[t] / ((double)m * Hq);", "Us[t] += a[t] / ((double)m * Hkv);"),
    ("numerator_unpooled", "cbo_pool(br, pooled, T, pool_w);", "cbo_pool(br, pooled, T, 1);"),
    ("denominator_unpooled", "cbo_pool(bbar, pooled, T, pool_w);", "cbo_pool(bbar, pooled, T, 1);"),
    ("numerator_power_fixed_2", "Ns[t] += pow(pooled[t], p) / m;", "Ns[t] += pooled[t] * pooled[t] / m;"),
    ("denominator_power_dropped", "Ds[t] = p_inf ? pooled[t] : pow(pooled[t], p);", "Ds[t] = pooled[t];"),
    ("numerator_sum_not_mean", "Ns[t] += pow(pooled[t], p) / m;", "Ns[t] += pow(pooled[t], p);"),
    ("mean_query_attention_unpooled", "cbo_pool(Usum, Qv, T, pool_w);", "cbo_pool(Usum, Qv, T, 1);"),
    ("correction_exponent", "pow(Nsum[t] / Dsum[t], 1.0 / (p - 1.0))", "pow(Nsum[t] / Dsum[t], 1.0 / p)"),
    ("correction_ratio_inverted", "pow(Nsum[t] / Dsum[t], 1.0 / (p - 1.0))", "pow(Dsum[t] / Nsum[t], 1.0 / (p - 1.0))"),
    ("strength_exponent_dropped", "if (S) S[t] = Qv[t] * pow(c, alpha);", "if (S) S[t] = Qv[t] * c;"),
    ("zero_denominator_gives_0", "pow(Nsum[t] / Dsum[t], 1.0 / (p - 1.0))) : 1.0;", "pow(Nsum[t] / Dsum[t], 1.0 / (p - 1.0))) : 0.0;"),
    ("p_inf_groups_summed", "Nsum[t] = n_s > Nsum[t] ? n_s : Nsum[t];", "Nsum[t] += n_s;"),
    ("p_inf_denominator_groups_summed", "Dsum[t] = d_s > Dsum[t] ? d_s : Dsum[t];", "Dsum[t] += d_s;"),
    ("p_inf_tokens_averaged", "Ns[t] = pooled[t] > Ns[t] ? pooled[t] : Ns[t];", "Ns[t] += pooled[t] / m;"),
    ("p_inf_denominator_squared", "Ds[t] = p_inf ? pooled[t] : pow(pooled[t], p);", "Ds[t] = p_inf ? pooled[t] * pooled[t] : pow(pooled[t], p);"),
    ("p_inf_ratio_inverted", "(p_inf ? Nsum[t] / Dsum[t] :", "(p_inf ? Dsum[t] / Nsum[t] :"),
    ("pool_window_too_wide", "int64_t half = w / 2;", "int64_t half = w / 2 + 1;"),
    ("pool_window_shifted", "int64_t hi = t + half > T - 1 ? T - 1 : t + half;", "int64_t hi = t + half + 1 > T - 1 ? T - 1 : t + half + 1;"),
    ("pool_min_not_max", "if (x[u] > mx) mx = x[u];", "if (x[u] < mx) mx = x[u];"),
    ("span_tie_favours_later", "return a->j < b->j ? -1 : (a->j > b->j ? 1 : 0);", "return a->j > b->j ? -1 : (a->j < b->j ? 1 : 0);"),
    ("first_position_not_raised", "Sp[0] = mx;", "(void)mx;"),
    ("partial_argmax_over_selected", "if (!sel[t] && (c < 0 || Sp[t] > Sp[c])) c = t;", "if (c < 0 || Sp[t] > Sp[c]) c = t;"),
    ("partial_takes_span_start", "near[n].dist = t > c ? t - c : c - t;", "near[n].dist = t;"),
    ("nearest_tie_to_higher_index", "return a->t < b->t ? -1 : (a->t > b->t ? 1 : 0);", "return a->t > b->t ? -1 : (a->t < b->t ? 1 : 0);"),
    ("latent_tail_off_by_one", "if (t < n_sink || t >= T - n_latent) { sel[t] = 1; ++count; }", "if (t < n_sink || t > T - n_latent) { sel[t] = 1; ++count; }"),
    ("short_span_mean_over_full_width", "rank[j].mean = acc / (double)(hi - lo);", "rank[j].mean = acc / (double)span_w;"),
    ("short_span_mean_over_full_width_f32", "rank[j].mean = (double)(acc / (float)(hi - lo));", "rank[j].mean = (double)(acc / (float)span_w);"),
    ("ranking_ascending", "if (a->mean > b->mean) return -1;\n    if (a->mean < b->mean) return 1;", "if (a->mean < b->mean) return -1;\n    if (a->mean > b->mean) return 1;"),
    ("compact_offset_dropped", "int64_t dst = (int64_t)l * o_layer + (int64_t)g * o_head + (off + j) * d;", "int64_t dst = (int64_t)l * o_layer + (int64_t)g * o_head + j * d;"),
    ("gather_offset_dropped", "memcpy(out + (off + j) * out_stride, src + (int64_t)idx[j] * src_stride, (size_t)row_bytes);", "memcpy(out + j * out_stride, src + (int64_t)idx[j] * src_stride, (size_t)row_bytes);"),
    ("gather_row_shifted", "memcpy(out + (off + j) * out_stride, src + (int64_t)idx[j] * src_stride, (size_t)row_bytes);", "memcpy(out + (off + j) * out_stride, src + (int64_t)(idx[j] + (idx[j] + 1 < T)) * src_stride, (size_t)row_bytes);"),
    ("self_keys_not_causal", "for (int u = 0; u <= r; ++u) Z += exp(", "for (int u = 0; u < dm->m; ++u) Z += exp("),
    ("self_keys_unscaled", "    return z * scale;\n}", "    return z;\n}"),
    ("unpage_pages_in_order", "const int64_t page = pages[t / P], row", "const int64_t page = t / P, row"),
    ("unpage_row_dropped", "page * s_page + row * s_pos + g * s_head", "page * s_page + g * s_head"),
    ("unpage_layer_stride_dropped", "pool + l * s_layer + page * s_page", "pool + page * s_page"),
    ("unpage_head_stride_dropped", "row * s_pos + g * s_head;", "row * s_pos;"),
    ("self_keys_wrong_group", "(int64_t)g * dm->s_head;", "(int64_t)((g + 1) % dm->n_kv_heads) * dm->s_head;"),
    ("rope_sign_flipped", "k_out[dst + a] = double_to_bf16(xa * cos(phi) - xb * sin(phi));", "k_out[dst + a] = double_to_bf16(xa * cos(phi) + xb * sin(phi));"),
    ("rope_halves_paired_as_interleaved", "const int a = style == 0 ? k : 2 * k, b = style == 0 ? k + half : 2 * k + 1;", "const int a = 2 * k, b = 2 * k + 1;"),
    ("rope_theta_exponent", "const double phi = delta * pow(base, -2.0 * k / d);", "const double phi = delta * pow(base, -1.0 * k / d);"),
    ("rope_offset_dropped", "const double delta = (double)(pos0 + off + j - idx[j]);", "const double delta = (double)(pos0 + j - idx[j]);"),
    ("compact_v_from_k", "memcpy(v_out + dst, V + src, sizeof(uint16_t) * (size_t)d);", "memcpy(v_out + dst, K + src, sizeof(uint16_t) * (size_t)d);"),
]


def _build(args):
    name, old, new, src, outdir = args
    if src.count(old) != 1:
        return name, None, "snippet occurs %d times" % src.count(old)
    path = os.path.join(outdir, name + ".c")
    with open(path, "w") as f:
        f.write(src.replace(old, new))
    so = os.path.join(outdir, "lib_" + name + ".so")
    oracle.build(path, so, force=True)
    return name, so, None


@pytest.fixture(scope="module")
def mutant_libs():
    with open(oracle._SRC) as f:
        src = f.read()
    outdir = tempfile.mkdtemp(prefix="cbo_mutants_")
    with cf.ThreadPoolExecutor(max_workers=os.cpu_count() or 4) as ex:
        res = list(ex.map(_build, [(n, o, nw, src, outdir) for n, o, nw in MUTANTS]))
    return {n: (so, err) for n, so, err in res}


@pytest.mark.parametrize("name", [m[0] for m in MUTANTS])
def test_mutant_is_caught(mutant_libs, name):
    so, err = mutant_libs[name]
    assert err is None, err
    o = oracle.Oracle(so)
    caught = []
    for pin in oracle_pins.ALL_PINS:
        try:
            pin(o)
        except (AssertionError, RuntimeError, ValueError):
            caught.append(pin.__name__)
    assert caught, "no pin catches the planted mistake %r" % name
