"""The oracle pins are sensitive: plausible mistakes planted in a temporary
copy of the oracle source (on the CPU) make at least one pin fail.  Mistakes
in the channel RMS normalisation, the per-head parameters and the signed
channel outputs are checked against their own pin files."""
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

MUTANTS = {
    "dropped 1/sqrt(M) scale": (
        "const double s = 1.0 / sqrt((double)p->M);\n    for (int i = 0; i < p->M; ++i) {\n        double u = project(p, i, x);",
        "const double s = 1.0;\n    for (int i = 0; i < p->M; ++i) {\n        double u = project(p, i, x);"),
    "dropped projection bias": ("double u = p->b[i];", "double u = 0.0;"),
    "channel-major feature order": ("out[i * p->L + l]", "out[l * p->M + i]"),
    "wrong sign of d(den)": ("dden[i] = -dot / den;", "dden[i] = dot / den;"),
    "exclusive causal mask": ("int jmax = causal ? i + 1 : len;", "int jmax = causal ? i : len;"),
    "fc2 weight gradient without activation": (
        "g->dw2[(size_t)l * p->hid + k] += term(dy * act_f(p->act, a));",
        "g->dw2[(size_t)l * p->hid + k] += term(dy);"),
    "eps dropped from the linear form": (
        "double den = eps;\n        for (int f = 0; f < D; ++f) den += phq[f] * z[f];",
        "double den = 0;\n        for (int f = 0; f < D; ++f) den += phq[f] * z[f];"),
    "transposed state index": (
        "for (int f = 0; f < D; ++f) num += phq[f] * S[(size_t)f * dv + c];",
        "for (int f = 0; f < D; ++f) num += phq[f] * S[(size_t)c * D + f];"),
    "inner ReLU mask inverted in backward": ("if (p->act == 0 && !(a > 0.0)) continue;", "if (p->act == 0 && a > 0.0) continue;"),
    "shared fc1 read per channel": ("return (size_t)(p->shared ? 0 : l) * p->hid;", "return (size_t)l * p->hid;"),
    "shared fc1 gradient not summed over channels": (
        "g->dw1[fc1_row(p, l) + k] += term(dh * u);", "g->dw1[(size_t)l * p->hid + k] += term(dh * u);"),
}

CH_RMS_PINS = "tests/test_oracle_ch_rms.py"
CH_RMS_MUTANTS = {
    "channel RMS: scale term dropped from the backward": (
        "if (p->chs) dy = dy * p->chs[l] + (kappa ? kappa[l] * y : 0.0);", "if (p->chs) dy = dy * p->chs[l];"),
    "channel RMS: mean over rows only": ("*count = rows * p->M;", "*count = rows;"),
    "channel RMS: scale not clamped at 1": ("s[l] = r < 1.0 ? r : 1.0;", "s[l] = r;"),
    "channel RMS: padded rows in the statistics": (
        "for (int bh = 0; bh < BH; ++bh) rows += head_len(lengths, bh / H, n);\n    *count",
        "for (int bh = 0; bh < BH; ++bh) rows += n;\n    *count"),
    "channel RMS: key statistics taken from the queries": (
        "ch_rms_scales(p, K, B, H, n, lengths, sk, sk + L, sk + 2 * L);",
        "ch_rms_scales(p, Q, B, H, n, lengths, sk, sk + L, sk + 2 * L);"),
    "channel RMS: sign of the scale derivative": (
        "? -p->ch_rms_target / ((rms + CH_RMS_EPS) * (rms + CH_RMS_EPS)) / (N * rms) * a",
        "? p->ch_rms_target / ((rms + CH_RMS_EPS) * (rms + CH_RMS_EPS)) / (N * rms) * a"),
}


PER_HEAD_PINS = "tests/test_oracle_per_head.py"
PER_HEAD_MUTANTS = {
    "per-head parameters of the wrong head": (
        "const oracle_phi vq = head_view(&sm.pq, bh % H), vk = head_view(&sm.pk, bh % H);\n        attn_fwd_head(",
        "const oracle_phi vq = head_view(&sm.pq, (bh + 1) % H), vk = head_view(&sm.pk, (bh + 1) % H);\n"
        "        attn_fwd_head("),
    "per-head gradients summed over every head": (
        "if (G == 1 || bh % H == h) acc +=", "if (1) acc +="),
}

SIGNED_PINS = "tests/test_oracle_signed.py"
SIGNED_MUTANTS = {
    "signed outputs still through the outer ReLU": ("return p->signed_out ? y : relu(y);", "return relu(y);"),
    "signed outputs: backward still masks by the outer ReLU": (
        "if (!p->signed_out && !(y > 0.0)) continue;", "if (!(y > 0.0)) continue;"),
}

VARIANT_PINS = "tests/test_oracle_variants.py"
VARIANT_MUTANTS = {
    "GELU: tanh-free form with a wrong argument": (
        "case 1: return 0.5 * a * (1.0 + erf(a / sqrt(2.0)));", "case 1: return 0.5 * a * (1.0 + erf(a));"),
    "GELU derivative without the density term": (
        " + a * exp(-0.5 * a * a) / sqrt(2.0 * ORACLE_PI);", ";"),
    "SiLU derivative taken as the logistic function": ("return sg * (1.0 + a * (1.0 - sg));", "return sg;"),
    "tanh derivative with the wrong sign": ("return 1.0 - t * t;", "return 1.0 + t * t;"),
    "envelope gate without its bias": ("double a = p->be[l];", "double a = 0.0;"),
    "envelope gate derivative without h (1 - h)": (
        "const double dpre = dE[l] * chcoef(p, l) * h[l] * (1.0 - h[l]);", "const double dpre = dE[l] * chcoef(p, l);"),
    "envelope gradient does not reach dX": ("dx[c] += dpre * p->We[(size_t)l * d + c];", ""),
    "coefficient gradient without the gate": (
        "if (p->coef) g->dcoef[l] += term(dE[l] * h[l]);", "if (p->coef) g->dcoef[l] += term(dE[l]);"),
    "coefficient missing from the feature": (
        "* gate(p, l, x) * chcoef(p, l) * channel_out", "* gate(p, l, x) * channel_out"),
    "coefficient missing from the chain rule into the MLP": (
        "double dy = dphi * s * h[l] * chcoef(p, l);", "double dy = dphi * s * h[l];"),
}

WEIGHTS_PINS = "tests/test_oracle_weights.py"
WEIGHTS_MUTANTS = {
    "weights: eps dropped from the normaliser": (
        "double den = eps;\n            for (int j = 0; j < jmax; ++j) {\n                double kij",
        "double den = 0.0;\n            for (int j = 0; j < jmax; ++j) {\n                double kij"),
    "weights: exclusive causal mask": (
        "const int jmax = causal ? i + 1 : len;", "const int jmax = causal ? i : len;"),
    "teacher: 1/sqrt(d) scale dropped": ("ar[j] = s / sqrt((double)d);", "ar[j] = s;"),
}

ALL = {**{k: (v, "tests/test_oracle_pins.py") for k, v in MUTANTS.items()},
       **{k: (v, WEIGHTS_PINS) for k, v in WEIGHTS_MUTANTS.items()},
       **{k: (v, VARIANT_PINS) for k, v in VARIANT_MUTANTS.items()},
       **{k: (v, SIGNED_PINS) for k, v in SIGNED_MUTANTS.items()},
       **{k: (v, CH_RMS_PINS) for k, v in CH_RMS_MUTANTS.items()},
       **{k: (v, PER_HEAD_PINS) for k, v in PER_HEAD_MUTANTS.items()}}


@pytest.mark.parametrize("name", sorted(ALL))
def test_planted_mistake_is_caught(name, tmp_path):
    src = open(os.path.join(ROOT, "oracle", "luna_oracle.c")).read()
    (a, b), pins = ALL[name]
    assert a in src, f"mutation site for {name!r} not found"
    work = tmp_path / "w"
    shutil.copytree(os.path.join(ROOT, "oracle"), work / "oracle", ignore=shutil.ignore_patterns("_build", "__pycache__"))
    shutil.copytree(os.path.join(ROOT, "synth"), work / "synth", ignore=shutil.ignore_patterns("__pycache__"))
    shutil.copytree(os.path.join(ROOT, "tests"), work / "tests", ignore=shutil.ignore_patterns("__pycache__"))
    (work / "oracle" / "luna_oracle.c").write_text(src.replace(a, b, 1))
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider",
                        pins], cwd=str(work), capture_output=True, text=True, timeout=600)
    assert r.returncode != 0, f"mutant {name!r} survived the pins:\n{r.stdout[-2000:]}"
