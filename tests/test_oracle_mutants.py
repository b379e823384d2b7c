"""Plant plausible mistakes in copies of the oracle and check that the pins catch each.

Every mutant is a one-line textual change of ``oracle/oracle.c`` (a dropped term, a wrong
sign, a transposed operand, a wrong index or rounding), compiled on the CPU into a
temporary library.  The pins must reject every one of them.
"""

import os

import pytest

import oracle
import oracle_pins

SRC = os.path.join(os.path.dirname(oracle.__file__), "oracle.c")

MUTANTS = {
    "ef_sign": ("s[j] = xr[j] + er[j];", "s[j] = xr[j] - er[j];"),
    "ef_residual_dropped": ("er[j] = s[j] - c[j];", "er[j] = s[j];"),
    "tie_order_reversed": ("return (a->j < b->j) ? -1 : (a->j > b->j);\n}\n\nstatic int by_index_asc",
                           "return (a->j > b->j) ? -1 : (a->j < b->j);\n}\n\nstatic int by_index_asc"),
    "magnitude_ignores_sign": ("work[j].mag = fabsf(x[j]);", "work[j].mag = x[j];"),
    "payload_not_index_sorted": ("qsort(work, (size_t)k, sizeof(orc_entry), by_index_asc);", ""),
    "ef21_update_dropped_term": ("gr[idx[i]] = gr[idx[i]] + vals[i];", "gr[idx[i]] = vals[i];"),
    "ef21_delta_transposed": ("d[j] = xr[j] - gr[j];", "d[j] = gr[j] - xr[j];"),
    "aqsgd_wrong_row": ("int64_t stored = sample_ids[i] * rows_per_sample + r;",
                        "int64_t stored = i * rows_per_sample + r;"),
    "round_floor": ("qf = rintf(t); /* nearest, ties to even */", "qf = floorf(t);"),
    "round_half_up": ("qf = rintf(t); /* nearest, ties to even */", "qf = floorf(t + 0.5f);"),
    "inv_transposed": ("float inv = levels / range;", "float inv = range / levels;"),
    "levels_off_by_one": ("float levels = (float)((1u << bits) - 1u);",
                          "float levels = (float)(1u << bits);"),
    "max_transposed": ("if (total_less(mx, xr[j])) mx = xr[j];",
                       "if (total_less(xr[j], mx)) mx = xr[j];"),
    "straddle_dropped": ("if (off + bits > 32) row_codes[w + 1] |= q >> (32 - off);", ""),
    "dequant_min_dropped": ("yr[j] = minv[r] + q * scale[r];", "yr[j] = q * scale[r];"),
    "stochastic_no_noise": ("qf = floorf(t + u);", "qf = floorf(t);"),
    "splitmix_counter": ("uint64_t z = seed + (counter + 1u) * GAMMA;",
                         "uint64_t z = seed + counter * GAMMA;"),
    "uniform_halves_swapped": ("(i & 1u) ? (uint32_t)(z >> 32) : (uint32_t)(z & 0xffffffffu)",
                               "(i & 1u) ? (uint32_t)(z & 0xffffffffu) : (uint32_t)(z >> 32)"),
    "signed_zero_min": ("return signbit(a) && !signbit(b);", "return 0;"),
    "efmix_buffer_share_from_input": ("work[m].mag = fabsf(er[j]);", "work[m].mag = fabsf(xr[j]);"),
    "efmix_shares_overlap": ("            if (!taken[j]) {\n                work[m].mag",
                             "            if (1) {\n                work[m].mag"),
    "aqsgd_quant_delta_transposed": ("d[logical * row_len + j] = x[logical * row_len + j] - br[j];",
                                     "d[logical * row_len + j] = br[j] - x[logical * row_len + j];"),
    "aqsgd_quant_update_dropped": ("for (int64_t j = 0; j < row_len; ++j) br[j] = br[j] + dh[logical * row_len + j];\n        }\n    free(dh);\n    free(d);",
                                   "for (int64_t j = 0; j < row_len; ++j) br[j] = dh[logical * row_len + j];\n        }\n    free(dh);\n    free(d);"),
    "gather_row_offset_dropped": ("vals[r * k + i] = g[r * row_len + idx[r * k + i]];",
                                  "vals[r * k + i] = g[idx[r * k + i]];"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_reject_mutant(name, tmp_path):
    old, new = MUTANTS[name]
    src = open(SRC).read()
    assert src.count(old) == 1, name
    mut_src = tmp_path / "oracle.c"
    mut_src.write_text(src.replace(old, new))
    (tmp_path / "oracle.h").write_text(open(os.path.join(os.path.dirname(SRC), "oracle.h")).read())
    lib_path = oracle.build(force=True, src=str(mut_src), out=str(tmp_path / "libmut.so"))
    lib = oracle.load(lib_path)
    failed = []
    for pin in oracle_pins.ALL_PINS:
        try:
            pin(lib)
        except AssertionError:
            failed.append(pin.__name__)
            break
    assert failed, "mutant %s passed every pin" % name
