"""Planted mistakes in the oracle fail its pins (no GPU).

Each mutant is a copy of oracle/mk_oracle.c with one plausible mistake (a
dropped term, a wrong sign or index, a swapped operand, an off-by-one mask,
the wrong logarithm, a wrong output index), compiled to a temporary library.
The pin suite in oracle_pin_checks.py must reject every one of them; the real
oracle passes it (test_oracle_pins.py)."""
import os

import pytest

import oracle
import oracle_pin_checks as pins

SRC = os.path.join(os.path.dirname(oracle.__file__), "mk_oracle.c")

MUTANTS = {
    "drop_scale": ("double s = p->scale * dot;", "double s = dot;"),
    "sign_of_max": ("double w = exp(s_buf[j] - m);", "double w = exp(s_buf[j] + m);"),
    "lse_without_max": ("*lse_out = m + log(l);", "*lse_out = log(l);"),
    "lse_log2": ("*lse_out = m + log(l);", "*lse_out = m + log2(l);"),
    "no_normalisation": ("        o_row[d] /= l;\n    *lse_out", "        o_row[d] *= 1.0;\n    *lse_out"),
    "causal_excludes_diagonal": ("int n_keys = p->causal ? (i + 1 < L ? i + 1 : L) : L;",
                                 "int n_keys = p->causal ? (i < L ? i : L) : L;"),
    "causal_ignored": ("int n_keys = p->causal ? (i + 1 < L ? i + 1 : L) : L;",
                       "int n_keys = L;"),
    "gqa_interleaved_groups": ("const int g = h / group;", "const int g = h % p->Hkv;"),
    "keys_read_from_values": ("/* |K_i| */\n\n    double m = -INFINITY;\n    for (int j = 0; j < n_keys; ++j) {\n        const uint16_t *kj = p->k + ",
                              "/* |K_i| */\n\n    double m = -INFINITY;\n    for (int j = 0; j < n_keys; ++j) {\n        const uint16_t *kj = p->v + "),
    "values_read_from_keys": ("const uint16_t *vj = p->v + ((tok0 + j) * p->Hkv + g) * (int64_t)D;\n        double w",
                              "const uint16_t *vj = p->k + ((tok0 + j) * p->Hkv + g) * (int64_t)D;\n        double w"),
    "query_row_offset": ("const uint16_t *qi = p->q + ((tok0 + i) * p->Hq + h) * (int64_t)D;\n    int n_keys",
                         "const uint16_t *qi = p->q + ((tok0 + i) * p->Hq + 0) * (int64_t)D;\n    int n_keys"),
    "varlen_lse_index": ("int64_t lse_idx = p->cu ? (int64_t)h * p->S + tok0 + i",
                         "int64_t lse_idx = p->cu ? (int64_t)h * p->S + i"),
    "weights_not_accumulated": ("        l += w;\n", "        l = w;\n"),
    "last_dim_dropped": ("for (int d = 0; d < D; ++d)\n            dot += bf16_bits_to_f64(qi[d]) * bf16_bits_to_f64(kj[d]);\n        double s",
                         "for (int d = 0; d + 1 < D; ++d)\n            dot += bf16_bits_to_f64(qi[d]) * bf16_bits_to_f64(kj[d]);\n        double s"),
    "decode_slot_from_page_index": (
        "const int64_t row = (page * job->page_size + j % job->page_size) * job->Hkv + g;\n            const uint16_t *kr",
        "const int64_t row = (page * job->page_size + j / job->page_size) * job->Hkv + g;\n            const uint16_t *kr"),
    "decode_interleaved_groups": ("h = (int)(t % job->Hq), g = h / G;", "h = (int)(t % job->Hq), g = h % job->Hkv;"),
    "decode_drop_scale": ("s_buf[j] = job->scale * acc;\n            if (s_buf[j] > m)\n                m = s_buf[j];\n        }\n        double l = 0.0;\n        for (int j = 0; j < L; ++j) {\n            const double e = exp(s_buf[j] - m);\n            l += e;",
                          "s_buf[j] = acc;\n            if (s_buf[j] > m)\n                m = s_buf[j];\n        }\n        double l = 0.0;\n        for (int j = 0; j < L; ++j) {\n            const double e = exp(s_buf[j] - m);\n            l += e;"),
    "decode_lse_log2": ("            orow[d] /= l;\n        job->lse[t] = m + log(l);\n    }\n    free(s_buf);\n    return NULL;\n}\n\nint mk_oracle_decode_paged_f64",
                        "            orow[d] /= l;\n        job->lse[t] = m + log2(l);\n    }\n    free(s_buf);\n    return NULL;\n}\n\nint mk_oracle_decode_paged_f64"),
    "mla_lse_log2": ("            orow[d] /= l;\n        job->lse[t] = m + log(l);\n    }\n    free(s_buf);\n    return NULL;\n}\n\nint mk_oracle_mla_decode_f64",
                     "            orow[d] /= l;\n        job->lse[t] = m + log2(l);\n    }\n    free(s_buf);\n    return NULL;\n}\n\nint mk_oracle_mla_decode_f64"),
    "bwd_drop_delta": ("const double dS = P * (dp_buf[j] - delta);\n                    const uint16_t *kj",
                       "const double dS = P * dp_buf[j];\n                    const uint16_t *kj"),
    "bwd_delta_sign": ("delta += s_buf[j] * dp;", "delta -= s_buf[j] * dp;"),
    "bwd_dk_without_scale": ("dkj[d] += p->scale * dS * bf16_bits_to_f64(qi[d]);",
                             "dkj[d] += dS * bf16_bits_to_f64(qi[d]);"),
    "bwd_dk_from_keys": ("dkj[d] += p->scale * dS * bf16_bits_to_f64(qi[d]);",
                         "dkj[d] += p->scale * dS * bf16_bits_to_f64(kj[d]);"),
    "bwd_dq_from_queries": ("dqi[d] += p->scale * dS * bf16_bits_to_f64(kj[d]);\n                        dkj",
                            "dqi[d] += p->scale * dS * bf16_bits_to_f64(qi[d]);\n                        dkj"),
    "bwd_dv_uses_ds": ("dvj[d] += P * bf16_bits_to_f64(doi[d]);", "dvj[d] += dS * bf16_bits_to_f64(doi[d]);"),
    "bwd_dv_uses_queries": ("dvj[d] += P * bf16_bits_to_f64(doi[d]);", "dvj[d] += P * bf16_bits_to_f64(qi[d]);"),
    "bwd_dp_from_keys": ("const uint16_t *vj = p->v + ((tok0 + j) * p->Hkv + g) * (int64_t)D;\n        double dp",
                         "const uint16_t *vj = p->k + ((tok0 + j) * p->Hkv + g) * (int64_t)D;\n        double dp"),
    "bwd_probs_without_lse": ("s_buf[j] = exp(s_buf[j] - lse);", "s_buf[j] = exp(s_buf[j]);"),
    "bwd_first_head_only": ("for (int h = g * group; h < (g + 1) * group; ++h) {\n            for (int i = 0; i < L; ++i) {",
                            "for (int h = g * group; h < g * group + 1; ++h) {\n            for (int i = 0; i < L; ++i) {"),
    "bwd_causal_excludes_diagonal": ("return p->causal ? (i + 1 < L ? i + 1 : L) : L; /* |K_i| */",
                                     "return p->causal ? (i < L ? i : L) : L; /* |K_i| */"),
    "bwd_dq_rows_drop_scale": ("dqi[d] += p->scale * dS * bf16_bits_to_f64(kj[d]);\n        }\n    }",
                               "dqi[d] += dS * bf16_bits_to_f64(kj[d]);\n        }\n    }"),
    "mla_values_from_suffix": ("orow[d] += e * bf16_bits_to_f64(cj[d]);",
                               "orow[d] += e * bf16_bits_to_f64(cj[d + (job->Dqk - job->Dv)]);"),
    "mla_rope_dropped": ("for (int d = 0; d < job->Dqk; ++d)\n                acc += bf16_bits_to_f64(qr[d]) * bf16_bits_to_f64(cj[d]);",
                         "for (int d = 0; d < job->Dv; ++d)\n                acc += bf16_bits_to_f64(qr[d]) * bf16_bits_to_f64(cj[d]);"),
    "mla_drop_scale": ("s_buf[j] = job->scale * acc;\n            if (s_buf[j] > m)\n                m = s_buf[j];\n        }\n        double l = 0.0;\n        for (int j = 0; j < L; ++j) {\n            const double e = exp(s_buf[j] - m);\n            const uint16_t *cj = mla_row",
                       "s_buf[j] = acc;\n            if (s_buf[j] > m)\n                m = s_buf[j];\n        }\n        double l = 0.0;\n        for (int j = 0; j < L; ++j) {\n            const double e = exp(s_buf[j] - m);\n            const uint16_t *cj = mla_row"),
    "mla_slot_from_page_index": ("return job->cache + (page * job->page_size + j % job->page_size) * (int64_t)job->Dqk;",
                                 "return job->cache + (page * job->page_size + j / job->page_size) * (int64_t)job->Dqk;"),
    "bwd_ranges_skip_first_row": ("for (int i = p->causal ? j0 : 0; i < L; ++i) {",
                                  "for (int i = p->causal ? j0 + 1 : 0; i < L; ++i) {"),
}


@pytest.fixture(scope="module")
def source():
    with open(SRC) as f:
        return f.read()


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(tmp_path, source, name):
    old, new = MUTANTS[name]
    assert source.count(old) == 1, f"mutation site for {name} not found exactly once"
    src = tmp_path / f"mutant_{name}.c"
    src.write_text(source.replace(old, new))
    lib = oracle.load(oracle.compile_oracle(str(src), str(tmp_path / f"libmutant_{name}.so")))
    failures = []
    for check in pins.ALL_CHECKS:
        try:
            check(lib)
        except AssertionError as e:
            failures.append(f"{check.__name__}: {e}")
    assert failures, f"mutant {name} passed every pin"
