"""Every plausible mistake planted in a copy of the oracle is caught by some pin.

Each mutant is a textual edit of ``oracle/oracle.c`` (a dropped term, a wrong
sign, index or operand), compiled to a temporary library and checked against
the pins of ``oracle_pins.py`` in a child process (a mutant that reads out of
bounds may crash; a crash counts as caught).  The real oracle is never edited.
"""
import os
import subprocess
import sys
import tempfile


ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SOURCE = os.path.join(ROOT, "oracle", "oracle.c")

MUTANTS = {
    "scale_dropped": [("s[j] = scale * dot;", "s[j] = dot;")],
    "scale_twice": [("s[j] = scale * dot;", "s[j] = scale * scale * dot;")],
    "k_transposed": [("bf16_to_f64(k[kj * D + d])", "bf16_to_f64(k[(size_t)d * L + kj])")],
    "dot_skips_first_dim": [("for (int d = 0; d < D; ++d)\n            dot",
                             "for (int d = 1; d < D; ++d)\n            dot")],
    "lse_drops_max": [("*lse = m + log(l);", "*lse = log(l);")],
    "lse_log2": [("*lse = m + log(l);", "*lse = m + log2(l);")],
    "exp_sign": [("exp(s[j] - m)", "exp(m - s[j])")],
    "no_max_shift": [("exp(s[j] - m)", "exp(s[j])"), ("*lse = m + log(l);", "*lse = log(l);")],
    "min_not_max": [("if (s[j] > m)", "if (s[j] < m)")],
    "not_normalised": [("double p = exp(s[j] - m) / l;", "double p = exp(s[j] - m);")],
    "v_dims_reversed": [("bf16_to_f64(v[vj * D + d])", "bf16_to_f64(v[vj * D + (D - 1 - d)])")],
    "varlen_off_by_one": [("int L = kv_lens[b];", "int L = kv_lens[b] + 1;")],
    "varlen_wrong_sample": [("valid_len(kv_lens, b, Skv)", "valid_len(kv_lens, 0, Skv)")],
    "rows_ignore_head": [("rows[bh * nrows + r]", "rows[r]")],
    "q_ignores_head": [("((size_t)bh * Sq + i) * D", "((size_t)i) * D")],
    "k_ignores_head": [("k + (size_t)bh * Skv * D", "k")],
    "v_ignores_head": [("v + (size_t)bh * Skv * D", "v")],
    "seg_not_equal": [("if (kseg[j] == seg)", "if (kseg[j] != seg)")],
    "seg_keys_of_sample_0": [("kv_seg + (size_t)b * Skv", "kv_seg")],
    "seg_first_query_id": [("q_seg[(size_t)b * Sq + i]", "q_seg[(size_t)b * Sq]")],
    "seg_query_ids_of_sample_0": [("q_seg[(size_t)b * Sq + i]", "q_seg[i]")],
    "seg_drops_last_key": [("for (int j = 0; j < Skv; ++j)\n                if (kseg",
                            "for (int j = 0; j < Skv - 1; ++j)\n                if (kseg")],
    "seg_k_by_position": [("const size_t kj = (size_t)(idx ? idx[j] : j);", "const size_t kj = (size_t)j;")],
    "seg_v_by_position": [("const size_t vj = (size_t)(idx ? idx[j] : j);", "const size_t vj = (size_t)j;")],
    "seg_probs_by_position": [("pr[idx[e]] = ps[e];", "pr[e] = ps[e];")],
    "rope_sign": [("yr[ia] = xa * cos(phi) - xb * sin(phi);", "yr[ia] = xa * cos(phi) + xb * sin(phi);")],
    "rope_direction": [("yr[ia] = xa * cos(phi) - xb * sin(phi);", "yr[ia] = xa * cos(phi) + xb * sin(phi);"),
                       ("yr[ib] = xa * sin(phi) + xb * cos(phi);", "yr[ib] = -xa * sin(phi) + xb * cos(phi);")],
    "rope_freq_exponent": [("pow(theta, -2.0 * i / da)", "pow(theta, -1.0 * i / da)")],
    "rope_raster_h": [("(g / Wp) % Hp", "g % Hp")],
    "rope_t_from_w": [("g / ((long)Hp * Wp)", "g / Wp")],
    "rope_pairs_swapped": [("(interleaved ? 2 * i : i)", "(interleaved ? i : 2 * i)"),
                           ("(interleaved ? 2 * i + 1 : i + da / 2)", "(interleaved ? i + da / 2 : 2 * i + 1)")],
    "rope_base_fixed": [("            base += da;\n        }\n    }\n    return 0;", "        }\n    }\n    return 0;")],
    "rope_offset_ignored": [("const long g = s - s0;", "const long g = s;")],
    "win_h_from_raw_index": [("ph = (i / Wp) % Hp", "ph = i % Hp")],
    "win_t_from_rows": [("const int pt = i / (Hp * Wp)", "const int pt = i / Wp")],
    "win_no_inward_shift": [("        if (start > last_start)\n            start = last_start;\n", "")],
    "win_truncated_radius": [("*hi = p + k / 2 < L - 1 ? p + k / 2 : L - 1;", "*hi = p + k / 2 - 1 < L - 1 ? p + k / 2 - 1 : L - 1;")],
    "win_key_index_axes": [("idx[n++] = (tt * Hp + hh) * Wp + ww;", "idx[n++] = (tt * Wp + hh) * Hp + ww;")],
    "win_w_axis_uses_h_size": [("axis_window(pw, Wp, kw,", "axis_window(pw, Wp, kh,")],
    "win_neighbourhood_one_past": [("*hi = start + k - 1 < L - 1 ? start + k - 1 : L - 1;",
                                    "*hi = start + k < L - 1 ? start + k : L - 1;")],
    "win_truncated_lo_clamped_to_one": [("*lo = p - k / 2 > 0 ? p - k / 2 : 0;", "*lo = p - k / 2 > 0 ? p - k / 2 : 1;")],
    "win_border_rule_inverted": [("    if (neighbourhood) {\n        int start", "    if (!neighbourhood) {\n        int start")],
    "rope_passthrough_zeroed": [("            yr[d] = bf16_to_f64(xr[d]);", "            yr[d] = 0.0;")],
    "rope_turns_tokens_after_grid": [("if (g < 0 || g >= grid)", "if (g < 0)")],
    "empty_row_lse_zero": [("*lse = -INFINITY;", "*lse = 0.0;")],
}

CHILD = r"""
import sys, traceback
sys.path.insert(0, sys.argv[2]); sys.path.insert(0, sys.argv[3])
import oracle, oracle_pins
orc = oracle.Oracle(sys.argv[1])
failed = []
for pin in oracle_pins.ALL_PINS:
    try:
        pin(orc)
    except Exception:
        failed.append(pin.__name__)
print("FAILED:" + ",".join(failed))
"""


def _mutate(text, edits):
    for old, new in edits:
        assert old in text, f"mutation anchor not found: {old!r}"
        text = text.replace(old, new)
    return text


def test_real_oracle_passes_in_child(tmp_path):
    import oracle
    lib = oracle.build(output=str(tmp_path / "liboracle_real.so"))
    out = subprocess.run([sys.executable, "-c", CHILD, lib, ROOT, os.path.join(ROOT, "tests")],
                         capture_output=True, text=True, timeout=300)
    assert out.returncode == 0, out.stderr
    assert "FAILED:\n" in out.stdout or out.stdout.strip() == "FAILED:", out.stdout


def test_every_mutant_is_caught():
    import oracle
    text = open(SOURCE).read()
    procs = {}
    with tempfile.TemporaryDirectory() as tmp:
        for name, edits in MUTANTS.items():
            src = os.path.join(tmp, f"{name}.c")
            with open(src, "w") as f:
                f.write(_mutate(text, edits))
            lib = oracle.build(source=src, output=os.path.join(tmp, f"lib{name}.so"))
            procs[name] = subprocess.Popen(
                [sys.executable, "-c", CHILD, lib, ROOT, os.path.join(ROOT, "tests")],
                stdout=subprocess.PIPE, stderr=subprocess.PIPE, text=True,
                env={**os.environ, "OMP_NUM_THREADS": "1"})
        survivors = []
        for name, p in procs.items():
            out, err = p.communicate(timeout=600)
            caught = p.returncode != 0
            if not caught:
                line = [ln for ln in out.splitlines() if ln.startswith("FAILED:")]
                caught = bool(line) and line[-1] != "FAILED:"
            if not caught:
                survivors.append(name)
    assert not survivors, f"mutants not caught by any pin: {survivors}"
