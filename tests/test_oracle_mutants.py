"""Each plausible mistake planted in a copy of the oracle must trip a pin.

The mutation is applied to a temporary copy of oracle/spire_oracle.c, which is
compiled on the CPU; the real oracle is never modified.  A mutant that passes
every pin would mean the pins cannot tell that mistake from the definition.
"""
import os
import shutil
import subprocess
import tempfile

import pytest

import oracle
import oracle_pins

SRC = os.path.join(os.path.dirname(oracle.__file__), "spire_oracle.c")

# (id, text in the oracle, replacement) -- one plausible mistake each.
MUTATIONS = [
    ("no_causal_offset", "int64_t n_i = L - c->k + i;", "int64_t n_i = L - c->k;"),
    ("causal_off_by_one", "int64_t n_i = L - c->k + i;", "int64_t n_i = L - c->k + i + 1;"),
    ("gqa_modulo", "int32_t g = h / group;", "int32_t g = h % c->Hkv;"),
    ("page_index_no_table",
     "int64_t page = c->block_table[(int64_t)b * c->max_pages + j / c->page_size];",
     "int64_t page = (int64_t)b * c->max_pages + j / c->page_size;"),
    ("page_slot_wrong", "int64_t slot = j % c->page_size;", "int64_t slot = j / c->page_size;"),
    ("exp2_not_exp", "double p = exp(scores[j] - m);", "double p = exp2(scores[j] - m);"),
    ("scale_dropped", "s *= scale;", "s *= 1.0;"),
    ("no_normalise", "out[d] /= l;", "out[d] /= 1.0;"),
    ("transposed_qk", "s += bf16_to_double(q[d]) * bf16_to_double(keys[j][d]);",
     "s += bf16_to_double(q[d]) * bf16_to_double(vals[j][d]);"),
    ("window_off_by_one", "return p < n_sink || p >= t - window;",
     "return p < n_sink || p > t - window;"),
    ("sinks_dropped", "return p < n_sink || p >= t - window;", "return p >= t - window;"),
    ("window_one_extra", "return p < n_sink || p >= t - window;",
     "return p < n_sink || p >= t - window - 1;"),
    ("ring_no_sink_offset", "return n_sink + (p - n_sink) % window;",
     "return (p - n_sink) % window;"),
    ("ring_reads_k_as_v",
     "vals[n] = base + ((((int64_t)b * 2 + 1) * c->Hkv + g) * S + s) * c->D;",
     "vals[n] = base + ((((int64_t)b * 2 + 0) * c->Hkv + g) * S + s) * c->D;"),
    ("query_row_stride", "const uint16_t *qi = c->q + (((int64_t)b * rows + i) * c->Hq + h) * c->D;",
     "const uint16_t *qi = c->q + (((int64_t)b * rows) * c->Hq + h) * c->D;"),
    ("mix_not_normalised", "m[((int64_t)i * B + b) * d_model + c] = s / z;",
     "m[((int64_t)i * B + b) * d_model + c] = s;"),
    ("mix_linear_not_exp", "a[l] = exp(w[(int64_t)i * n_act + l] - wmax);",
     "a[l] = 1.0 + w[(int64_t)i * n_act + l] - wmax;"),
    ("rope_sign", "k[d] = a0 * cs - a1 * sn;", "k[d] = a0 * cs + a1 * sn;"),
    ("rope_frequency", "pow(rope_theta, -2.0 * d / D)", "pow(rope_theta, -1.0 * d / D)"),
    ("rope_adjacent_pairs", "double a0 = k[d], a1 = k[d + D / 2];",
     "double a0 = k[d], a1 = k[d ^ 1];"),
    ("append_k_v_swapped", "const double *src = y + ((int64_t)kvi * Hkv + g) * D;",
     "const double *src = y + ((int64_t)(1 - kvi) * Hkv + g) * D;"),
    ("append_slot_is_position_mod_s",
     "int64_t dst_slot = oracle_draft_slot(p, n_sink, window);",
     "int64_t dst_slot = p % S;"),
    ("round_truncates", "double r = ldexp(nearbyint(ldexp(v, -q)), q);",
     "double r = ldexp(trunc(ldexp(v, -q)), q);"),
    ("round_ties_away", "double r = ldexp(nearbyint(ldexp(v, -q)), q);",
     "double r = ldexp(round(ldexp(v, -q)), q);"),
    ("accept_ratio_inverted", "float uq = u[(int64_t)b * k + j] * qv;",
     "float uq = u[(int64_t)b * k + j] * pv; pv = qv;"),
    ("residual_sign", "float w = use_residual ? p[v] - q[v] : p[v];",
     "float w = use_residual ? q[v] - p[v] : p[v];"),
    ("bonus_from_last_draft_row", "const float *pj = p + ((int64_t)b * (k + 1) + j) * V;",
     "const float *pj = p + ((int64_t)b * (k + 1) + (j < k ? j : k - 1)) * V;"),
    ("race_multiplies", "float s = w / e;", "float s = w * e;"),
    ("race_argmin", "if (key > best) {", "if (best == 0 || key < best) {"),
    ("accepted_tokens_reversed", "o[i] = x[(int64_t)b * k + i];",
     "o[i] = x[(int64_t)b * k + (j - 1 - i)];"),
    ("magicdec_delta_sign", "rotate_pairs(k_cache + row, (double)(c - p), D, theta, kc + c * D);",
     "rotate_pairs(k_cache + row, (double)(p - c), D, theta, kc + c * D);"),
    ("magicdec_query_text_position",
     "rotate_pairs(q + ((int64_t)b * Hq + h) * D, (double)(n - 1), D, theta, qe);",
     "rotate_pairs(q + ((int64_t)b * Hq + h) * D, (double)(t - 1), D, theta, qe);"),
    ("magicdec_window_start", "int64_t w0 = ok ? (t - window > s ? t - window : s) : 0;",
     "int64_t w0 = ok ? (t - window + 1 > s ? t - window + 1 : s) : 0;"),
    ("magicdec_no_sinks", "int64_t s = ok ? (t < n_sink ? t : n_sink) : 0;", "int64_t s = 0;"),
    ("magicdec_pair_partner",
     "double a0 = bf16_to_double(src[d]), a1 = bf16_to_double(src[d + D / 2]);",
     "double a0 = bf16_to_double(src[d]), a1 = bf16_to_double(src[d ^ 1]);"),
]


@pytest.fixture(scope="module")
def workdir():
    d = tempfile.mkdtemp(prefix="spire_mutants_")
    yield d
    shutil.rmtree(d, ignore_errors=True)


@pytest.mark.parametrize("mid,old,new", MUTATIONS, ids=[m[0] for m in MUTATIONS])
def test_mutant_is_caught(mid, old, new, workdir):
    text = open(SRC).read()
    assert text.count(old) == 1, "mutation anchor must occur exactly once: %r" % old
    src = os.path.join(workdir, mid + ".c")
    so = os.path.join(workdir, mid + ".so")
    with open(src, "w") as f:
        f.write(text.replace(old, new))
    subprocess.run(["gcc", "-std=c11", "-O2", "-fPIC", "-shared", "-pthread", "-o", so, src,
                    "-lm"], check=True)
    lib = oracle.load(so)
    caught = []
    for pin in oracle_pins.ALL_PINS:
        try:
            pin(lib)
        except (AssertionError, ValueError):
            caught.append(pin.__name__)
    assert caught, "mutant %s passed every pin" % mid
