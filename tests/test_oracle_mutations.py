"""Planted mistakes in the oracle (CPU only).

Each mutant is a copy of the oracle's C sources with one plausible error in
one function: a flipped sign, a dropped term or factor, a wrong exponent,
rounding mode, bias or index, an off-by-one budget or order. It is compiled on
its own, and the oracle's pin tests (which check it against the paper's
printed values, closed forms, brute force and invariants, never against the
CUDA library) run against it in a subprocess. Every mutant must fail at least
one pin. A control run of an unmodified copy must pass them all.
"""
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
ORACLE = os.path.join(ROOT, "oracle")
SOURCES = ["numerics.c", "recurrence.c", "codec.c", "plan.c", "batch.c", "calib.c"]
PINS = ["tests/test_oracle_numerics.py", "tests/test_oracle_recurrence.py", "tests/test_oracle_codec.py",
        "tests/test_oracle_plan.py", "tests/test_oracle_step.py"]

DELTA_W = ("            S[i * OR_D + j] = (float)(P[i * OR_D + j] +\n"
           "                                      (double)beta * (double)k[i] * ((double)v[j] - u[j]));")
STEP_W = ("            X[i * OR_D + j] = (float)(S[i * OR_D + j] +\n"
          "                                      (double)beta * (double)k[i] * ((double)v[j] - u[j]));\n"
          "    for (int j = 0; j < OR_D; j++) {                           /* readout before requantization */")
STEP_Y = ("    for (int j = 0; j < OR_D; j++) {                           /* readout before requantization */\n"
          "        double acc = 0.0;\n"
          "        for (int i = 0; i < OR_D; i++)\n"
          "            acc += (double)q[i] * (double)X[i * OR_D + j];")
INTB_W = ("            X[i * OR_D + j] = (float)(S[i * OR_D + j] +\n"
          "                                      (double)beta * (double)k[i] * ((double)v[j] - u[j]));\n"
          "    for (int j = 0; j < OR_D; j++) {\n"
          "        double acc = 0.0;")
READOUT = ("    for (int j = 0; j < OR_D; j++) {                              /* readout S^T q */\n"
           "        double acc = 0.0;\n"
           "        for (int i = 0; i < OR_D; i++)\n"
           "            acc += (double)q[i] * (double)S[i * OR_D + j];")

# (id, file, original text, mutated text)
MUTANTS = [
    ("delta_sign", "recurrence.c", DELTA_W, DELTA_W.replace("((double)v[j] - u[j])", "(u[j] - (double)v[j])")),
    ("retrieval_ungated", "recurrence.c", "            acc += (double)k[i] * P[i * OR_D + j];",
     "            acc += (double)k[i] * (double)S[i * OR_D + j];"),
    ("readout_before_update", "recurrence.c", READOUT,
     READOUT.replace("(double)q[i] * (double)S[i * OR_D + j]", "(double)q[i] * P[i * OR_D + j]")),
    ("row_impact_gate_dropped", "recurrence.c",
     "        g[i] = d * ((double)q[i] - (double)beta * (double)k[i] * kq);",
     "        g[i] = ((double)q[i] - (double)beta * (double)k[i] * kq);"),
    ("exact_read_own_state", "recurrence.c",
     "            acc += (double)k[i] * (d * (double)Sref[i * OR_D + j]);",
     "            acc += (double)k[i] * (d * (double)S[i * OR_D + j]);"),
    ("step_delta_sign", "codec.c", STEP_W, STEP_W.replace("((double)v[j] - u[j])", "(u[j] - (double)v[j])")),
    ("step_readout_source", "codec.c", STEP_Y,
     STEP_Y.replace("(double)q[i] * (double)X[i * OR_D + j]", "(double)k[i] * (double)X[i * OR_D + j]")),
    ("intb_step_delta_sign", "codec.c", INTB_W, INTB_W.replace("((double)v[j] - u[j])", "(u[j] - (double)v[j])")),
    ("ls_weight_w_not_w2", "codec.c", "                double w2 = (double)w[i] * (double)w[i];",
     "                double w2 = (double)w[i];"),
    ("row_factor_exponent", "codec.c", "        double t = sqrt(m) / sqrt((double)w[i]);",
     "        double t = sqrt(m) * sqrt((double)w[i]);"),
    ("column_start_without_qmax", "codec.c",
     "                double a = fabs((double)X[i * OR_D + j]) / (rz[i] * qmax_of(rb[i]));",
     "                double a = fabs((double)X[i * OR_D + j]) / rz[i];"),
    ("codes_floored", "codec.c", "    return clampd(rne_div((double)x, r_zs * c), -qm, qm);",
     "    return clampd(floor((double)x / (r_zs * c)), -qm, qm);"),
    ("code_ties_to_odd", "codec.c", "    if (2.0 * fabs(e) == d && fmod(n, 2.0) != 0.0)",
     "    if (2.0 * fabs(e) == d && fmod(n, 2.0) == 0.0)"),
    ("code_clip_qmax_plus_one", "codec.c", "    return clampd(rne_div((double)x, r_zs * c), -qm, qm);",
     "    return clampd(rne_div((double)x, r_zs * c), -qm - 1, qm + 1);"),
    ("offset_binary_bias", "codec.c",
     "            put_code(page, unit_kind, rb, off, i, j, (unsigned)(qv + (1 << (b - 1))));",
     "            put_code(page, unit_kind, rb, off, i, j, (unsigned)(qv + (1 << (b - 1)) - 1));"),
    ("final_codes_unrounded_c", "codec.c",
     "            int qv = (int)level(X[i * OR_D + j], rz, c16[j], qmax_of(b));",
     "            int qv = (int)level(X[i * OR_D + j], rz, c[j], qmax_of(b));"),
    ("temporal_scale_qmax", "codec.c",
     "            double s16 = or_fp16_round(clampd((float)((double)amax / qm), F16_MIN_NORMAL, F16_MAX));",
     "            double s16 = or_fp16_round(clampd((float)((double)amax / (qm + 1)), F16_MIN_NORMAL, F16_MAX));"),
    ("intb_scale_qmax", "codec.c", "        float s = (float)((double)amax / qm);",
     "        float s = (float)((double)amax / (qm + 1));"),
    ("fp16_ties_away", "numerics.c",
     "    double n = nearbyint(a / quantum);    /* exact quotient; default mode is ties-to-even */",
     "    double n = round(a / quantum);"),
    ("lifetime_factor_two", "plan.c", "        L += exp(2.0 * j * ell);", "        L += exp(j * ell);"),
    ("row_weight_exponent", "plan.c", "    const double half_gamma = 0.125;", "    const double half_gamma = 0.25;"),
    ("dp_predecessor", "plan.c", "                double val = cost[(size_t)u * n_cand + k] + Fn[c - a];",
     "                double val = cost[(size_t)u * n_cand + k] + Fn[c];"),
    ("lagrangian_price", "plan.c", "            double val = cost[(size_t)u * n_cand + k] + lam * cands[k];",
     "            double val = cost[(size_t)u * n_cand + k] + lam;"),
    ("repair_slack_off_by_one", "plan.c", "                if (db <= 0 || db > slack)",
     "                if (db <= 0 || db >= slack)"),
    ("pivots_lowest_risk", "plan.c", "            if (!pivot[u] && (best < 0 || risk[u] > risk[best]))",
     "            if (!pivot[u] && (best < 0 || risk[u] < risk[best]))"),
    ("pivot_budget_16", "plan.c", "(long long)nominal * n_units - 8LL * n_piv",
     "(long long)nominal * n_units - 16LL * n_piv"),
    ("slot_stride_128", "plan.c", "    *slot_stride = (off + 255) / 256 * 256;",
     "    *slot_stride = (off + 127) / 128 * 128;"),
    ("gqa_interleaved", "batch.c", "    int hk = h / (Hv / Hk);\n    const float *g = gate_per_row ? gate + ((size_t)b * Hv + h) * OR_D : gate",
     "    int hk = h % Hk;\n    const float *g = gate_per_row ? gate + ((size_t)b * Hv + h) * OR_D : gate"),
    ("slot_ignored", "batch.c", "    return pool + (uint64_t)slots[b] * stride + head_off[h];",
     "    return pool + (uint64_t)b * stride + head_off[h];"),
    ("batch_recurrence_interleaved", "recurrence.c",
     "            int hk = h / grp;\n            const float *g = gate_per_row ? gate + ((size_t)b * Hv + h) * OR_D\n"
     "                                          : gate + (size_t)b * Hv + h;\n            or_delta_step_f32(",
     "            int hk = h % Hk;\n            const float *g = gate_per_row ? gate + ((size_t)b * Hv + h) * OR_D\n"
     "                                          : gate + (size_t)b * Hv + h;\n            or_delta_step_f32("),
    ("omega_abs_not_square", "calib.c", "                omega_sum[(size_t)h * OR_D + i] += gi[i] * gi[i];",
     "                omega_sum[(size_t)h * OR_D + i] += fabs(gi[i]);"),
    ("logret_without_log", "calib.c", "                logret_sum[h] += log((double)g[0]);",
     "                logret_sum[h] += (double)g[0];"),
    ("logret_row_without_log", "calib.c", "                    logret_sum[(size_t)h * OR_D + i] += log((double)g[i]);",
     "                    logret_sum[(size_t)h * OR_D + i] += (double)g[i];"),
    ("distortion_head_unweighted", "calib.c",
     "                        double w2 = (double)w[i] * (double)w[i], ei = 0.0;",
     "                        double w2 = 1.0, ei = 0.0;"),
    ("distortion_row_per_element_sum", "calib.c", "                        acc[((size_t)h * OR_D + i) * (n_cand + 1) + k] += ei / OR_D;",
     "                        acc[((size_t)h * OR_D + i) * (n_cand + 1) + k] += ei;"),
    ("row_codebook_spacing", "codec.c",
     "static int zs_of(int unit_kind, int b) { return unit_kind == OR_UNIT_ROW ? 1 << (8 - b) : 1; }",
     "static int zs_of(int unit_kind, int b) { return unit_kind == OR_UNIT_ROW ? 1 << (7 - b) : 1; }"),
    ("zero_denominator_divides", "codec.c", "            if (den > 0.0)\n                c[j] =",
     "            if (den >= 0.0)\n                c[j] ="),
    ("row_scale_floor_zero", "codec.c", "        r[i] = or_fp16_round(clampd(t, F16_MIN_NORMAL, F16_MAX));",
     "        r[i] = or_fp16_round(clampd(t, 0.0, F16_MAX));"),
    ("extra_fit_iteration", "codec.c", "    for (int it = 0; it < fit_iters; it++) {\n        for (int j = 0; j < OR_D; j++) {\n            double num",
     "    for (int it = 0; it <= fit_iters; it++) {\n        for (int j = 0; j < OR_D; j++) {\n            double num"),
    ("pivot_rows_in_fit", "codec.c", "        in_fit[i] = (b != OR_PIVOT_BITS);", "        in_fit[i] = 1;"),
    ("bits_msb_first", "codec.c", "        if ((u >> t) & 1u)\n            row[p >> 3] |=",
     "        if ((u >> (b - 1 - t)) & 1u)\n            row[p >> 3] |="),
    ("rows_stored_ascending", "codec.c", "            if (rb[r] > b || (rb[r] == b && r < i))",
     "            if (rb[r] < b || (rb[r] == b && r < i))"),
    ("band_of_row", "codec.c", "        int w = j / 16, l = 8 * ((j / 4) % 4) + i / 16;",
     "        int w = j / 16, l = 8 * ((j / 4) % 4) + i % 8;"),
    ("pieces_contiguous_per_lane", "codec.c", "(size_t)(word / 4) * 512 + 16 * (size_t)l +",
     "(size_t)(word / 4) * 16 + 16 * (size_t)l +"),
    ("code_bits_msb_first", "codec.c", "        if ((u >> t) & 1u)\n            *p |= (uint8_t)(1u << bit);",
     "        if ((u >> (rb[i] - 1 - t)) & 1u)\n            *p |= (uint8_t)(1u << bit);"),
    ("fp16_subnormal_scale", "numerics.c", "        return s | (uint16_t)(a / ldexp(1.0, -24));   /* subnormal: fraction counts 2^-24 */",
     "        return s | (uint16_t)(a / ldexp(1.0, -23));   /* subnormal: fraction counts 2^-24 */"),
    ("row_pivot_risk_without_fp16", "plan.c",
     "            risk[u] = L[u] * (dist[(size_t)u * (n_cand + 1) + kn] -\n                              dist[(size_t)u * (n_cand + 1) + n_cand]);",
     "            risk[u] = L[u] * (dist[(size_t)u * (n_cand + 1) + kn] -\n                              0.0 * dist[(size_t)u * (n_cand + 1) + n_cand]);"),
    ("dp_ties_narrower", "plan.c", "            if (cands[order[b]] > cands[order[a]]) {",
     "            if (cands[order[b]] < cands[order[a]]) {"),
]


CFLAGS = ["-O2", "-std=c11", "-fPIC", "-fopenmp", "-ffp-contract=off"]


@pytest.fixture(scope="module")
def objects(tmp_path_factory):
    """The unmodified sources compiled once; a mutant recompiles only its file."""
    d = str(tmp_path_factory.mktemp("oracle_objs"))
    for f in SOURCES + ["oracle.h"]:
        shutil.copy(os.path.join(ORACLE, f), d)
    for f in SOURCES:
        subprocess.run(["gcc", "-c"] + CFLAGS + ["-o", os.path.join(d, f + ".o"), os.path.join(d, f)],
                       check=True)
    return d


def _build(objs, dst, edit=None):
    os.makedirs(dst, exist_ok=True)
    parts = [os.path.join(objs, f + ".o") for f in SOURCES]
    if edit:
        fname, old, new = edit
        src = open(os.path.join(objs, fname)).read()
        assert src.count(old) == 1, f"mutation site not unique in {fname}: {old!r}"
        path = os.path.join(dst, fname)
        open(path, "w").write(src.replace(old, new))
        obj = os.path.join(dst, fname + ".o")
        subprocess.run(["gcc", "-c"] + CFLAGS + ["-I", objs, "-o", obj, path], check=True)
        parts[SOURCES.index(fname)] = obj
    so = os.path.join(dst, "liboracle.so")
    subprocess.run(["gcc", "-shared", "-fopenmp", "-o", so] + parts + ["-lm"], check=True)
    return so


def _run_pins(so):
    env = dict(os.environ, STEPQ_ORACLE_LIB=so, OMP_NUM_THREADS="2")
    return subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                           "-m", "not gpu"] + PINS, cwd=ROOT, env=env, capture_output=True, text=True,
                          timeout=900)


def test_unmodified_copy_passes_the_pins(objects, tmp_path):
    r = _run_pins(_build(objects, str(tmp_path / "control")))
    assert r.returncode == 0, r.stdout[-3000:]


@pytest.mark.parametrize("mid,fname,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_planted_mistake_fails_a_pin(objects, tmp_path, mid, fname, old, new):
    r = _run_pins(_build(objects, str(tmp_path / mid), (fname, old, new)))
    assert r.returncode == 1, f"{mid} passed every pin:\n{r.stdout[-3000:]}"
