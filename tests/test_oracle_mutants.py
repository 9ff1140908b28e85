"""Each plausible mistake, planted in a temporary copy of the oracle's C source
(never in the oracle itself), must trip at least one pin of oracle_pins.py.

This shows that the pins constrain every part of the oracle: the feature map,
its W orientation, the softmax scale, the gate, the shared normaliser, the
commit, the GQA head mapping, the in-block mask, the per-head and per-request
indexing of every route and the training form's forward and gradients.  Mutants run in a
subprocess, so a mutant that crashes counts as caught without harming the
test process.
"""
import os
import subprocess
import sys

import pytest

from oracle import SOURCE, build_oracle

HERE = os.path.dirname(os.path.abspath(__file__))

# (name, exact text in the oracle source, replacement)
MUTANTS = [
    ("softmax scale 1/d", "s /= sqrt((double)d);", "s /= (double)d;"),
    ("softmax scale dropped", "s /= sqrt((double)d);", "s /= 1.0;"),
    ("phi negative half sign", "out[F + f] = exp(-u[f]) / sum_neg;", "out[F + f] = exp(u[f]) / sum_neg;"),
    ("phi negative normaliser sign", "sum_neg += exp(-u[f]);", "sum_neg += exp(u[f]);"),
    ("phi W transposed", "acc += x[e] * W[(size_t)e * F + f];", "acc += x[e] * W[((size_t)f * d + e) % ((size_t)d * F)];"),
    ("phi halves swapped", "out[f] = exp(u[f]) / sum_pos;\n        out[F + f] = exp(-u[f]) / sum_neg;",
     "out[F + f] = exp(u[f]) / sum_pos;\n        out[f] = exp(-u[f]) / sum_neg;"),
    ("gate sign", "return 1.0 / (1.0 + exp(-alpha));", "return 1.0 / (1.0 + exp(alpha));"),
    ("gate dropped in numerator", "o[e] = (w * sm_num[e] + lin_num[e]) / den;", "o[e] = (sm_num[e] + lin_num[e]) / den;"),
    ("gate on the wrong branch", "const double den = w * sm_den + lin_den;", "const double den = sm_den + w * lin_den;"),
    ("separate normalisers", "o[e] = (w * sm_num[e] + lin_num[e]) / den;",
     "o[e] = w * sm_num[e] / sm_den + (lin_den > 0 ? lin_num[e] / lin_den : 0.0);"),
    ("z not accumulated", "z[f] += phi[f];", "z[f] += 0.0 * phi[f];"),
    ("lin_den ignores phi(q)", "lin_den += phi_q[f] * z[f];", "lin_den += z[f];"),
    ("state read transposed", "lin_num[e] += phi_q[f] * S[(size_t)f * d + e];",
     "lin_num[e] += phi_q[f] * S[((size_t)e * P2 + f) % ((size_t)P2 * d)];"),
    ("commit drops last token", "for (int t = 0; t < c->T; ++t) {", "for (int t = 0; t < c->T - 1; ++t) {"),
    ("causal mask inside the block", "(size_t)c->Hkv * d, B, d, sm_num, &sm_den);",
     "(size_t)c->Hkv * d, i + 1, d, sm_num, &sm_den);"),
    ("GQA mapping modulo", "return h / G;", "return h % Hkv;"),
    ("prefix route skips last token", "for (int t = 0; t < P; ++t) {", "for (int t = 0; t + 1 < P; ++t) {"),
    ("value index shifted", "for (int e = 0; e < d; ++e) sm_num[e] += a * v[e];",
     "for (int e = 0; e < d; ++e) sm_num[e] += a * v[(e + 1) % d];"),
    # training form (Stage 1): forward over a sequence and the gradient of W, alpha
    ("train forward never commits", "        /* block n commits after its own readout */\n        for (int t = 0; t < B; ++t) {",
     "        /* block n commits after its own readout */\n        for (int t = 0; t < B && n < 0; ++t) {"),
    ("train forward commits one block late", "for (int n = 0; n < n_blk; ++n) {\n        const size_t t0 = (size_t)s * c->L + (size_t)n * B;   /* first token of block n */",
     "for (int n = 0; n < n_blk; ++n) {\n        const size_t t0 = (size_t)s * c->L + (size_t)(n > 0 ? n - 1 : 0) * B;   /* first token of block n */"),
    ("train prefix states not carried over", "for (size_t i = 0; i < st; ++i) Sn[i] = Sn[i - st];",
     "for (size_t i = 0; i < st; ++i) Sn[i] = 0.0 * Sn[i - st];"),
    ("train dD sign", "const double dD = -go / D;", "const double dD = go / D;"),
    ("train z gradient dropped", "double acc_f = z[f] * dD;", "double acc_f = 0.0 * dD;"),
    ("train phi backward negative half sign", "- phi[F + f] * (gphi[F + f] - dot_neg);",
     "+ phi[F + f] * (gphi[F + f] - dot_neg);"),
    ("train key side uses its own block", "const double *dS = dSpre + (size_t)(m + 1) * st;",
     "const double *dS = dSpre + (size_t)m * st;"),
    ("train key gradient ignores values", "acc_f += acc[(size_t)f * d + e] * v[e];",
     "acc_f += acc[(size_t)f * d + e];"),
    ("train dalpha without the sigmoid slope", "dalpha[h] = a * w * (1.0 - w);", "dalpha[h] = a;"),
    ("train state gradient of own block", "dS[(size_t)f * d + e] += phi[f] * dN[e];",
     "dS[(size_t)f * d + e] += phi[f] * dN[(e + 1) % d];"),
    ("train backward query heads of group 0", "const int h = g * G + hl;", "const int h = hl;"),
    ("train backward drops the key-side W gradient", "phi_backward_add(k, phi, gphi, d, F, du, dW);",
     "if (0) phi_backward_add(k, phi, gphi, d, F, du, dW);"),
    ("train backward drops the query-side W gradient", "phi_backward_add(q, phi, gphi, d, F, du, dW);",
     "if (0) phi_backward_add(q, phi, gphi, d, F, du, dW);"),
    ("train dalpha without the softmax denominator", "dw += dD * sm_den;", "dw += 0.0 * sm_den;"),
    ("train backward prefix state includes its own block", "const size_t t0 = (size_t)s * c->L + (size_t)(n - 1) * B;",
     "const size_t t0 = (size_t)s * c->L + (size_t)n * B;"),
    ("train forward every sequence reads the first", "const size_t t0 = (size_t)s * c->L + (size_t)n * B;   /* first token of block n */",
     "const size_t t0 = (size_t)0 * s * c->L + (size_t)n * B;   /* first token of block n */"),
    ("fan-out: threads after the first start one unit late",
     "for (long u = a->tid; u < a->n_units; u += a->n_threads) {",
     "for (long u = a->tid + (a->tid > 0); u < a->n_units; u += a->n_threads) {"),
    # head and request indexing of the inference routes
    ("commit uses state head 0's W", "const double *Wg = c->W ? c->W + (size_t)g * d * F : NULL;\n    for (int t = 0; t < c->T; ++t) {",
     "const double *Wg = c->W ? c->W + (size_t)0 * g * d * F : NULL;\n    for (int t = 0; t < c->T; ++t) {"),
    ("step uses state head 0's W", "const double *Wg = c->W ? c->W + (size_t)g * d * F : NULL;\n\n    double *u = scratch;",
     "const double *Wg = c->W ? c->W + (size_t)0 * g * d * F : NULL;\n\n    double *u = scratch;"),
    ("commit into state head 0", "double *S = c->S + ((size_t)r * c->Hkv + g) * P2 * d;\n    double *z = c->z",
     "double *S = c->S + ((size_t)r * c->Hkv + 0 * g) * P2 * d;\n    double *z = c->z"),
    ("prefix values of the mirrored head", "const double *vt = c->Vp + (((size_t)r * c->P_max + t) * c->Hkv + g) * d;",
     "const double *vt = c->Vp + (((size_t)r * c->P_max + t) * c->Hkv + (c->Hkv - 1 - g)) * d;"),
    ("prefix kernel over phi+ only", "for (int f = 0; f < P2; ++f) kern += phi_q[f] * phi_k[f];",
     "for (int f = 0; f < P2 / 2; ++f) kern += phi_q[f] * phi_k[f];"),
    ("state readout over phi+ only", "for (int f = 0; f < P2; ++f) {\n        for (int e = 0; e < d; ++e) lin_num[e] += phi_q[f] * S[(size_t)f * d + e];",
     "for (int f = 0; f < P2 / 2; ++f) {\n        for (int e = 0; e < d; ++e) lin_num[e] += phi_q[f] * S[(size_t)f * d + e];"),
    ("block keys of the next request", "const size_t kv0 = ((size_t)r * B * c->Hkv + g) * d;",
     "const size_t kv0 = ((size_t)((r + 1) % c->n_req) * B * c->Hkv + g) * d;"),
    ("query row reversed", "const double *q = c->Q + (((size_t)r * B + i) * c->Hq + h) * d;",
     "const double *q = c->Q + (((size_t)r * B + (B - 1 - i)) * c->Hq + h) * d;"),
    ("output of the next query head", "merge(w, sm_num, sm_den, lin_num, lin_den, d, c->O + (((size_t)r * B + i) * c->Hq + h) * d);",
     "merge(w, sm_num, sm_den, lin_num, lin_den, d, c->O + (((size_t)r * B + i) * c->Hq + (h + 1) % c->Hq) * d);"),
    ("feature map with head 0's W", "const double *Wg = W + (size_t)(h / group) * d * F;",
     "const double *Wg = W + (size_t)0 * (h / group) * d * F;"),
    ("feature map W by head modulo", "const double *Wg = W + (size_t)(h / group) * d * F;",
     "const double *Wg = W + (size_t)(h % n_kv_heads) * d * F;"),
    ("gate of the first head of the group", "const double w = gate(c->alpha[h]);\n\n    for (int i = 0; i < B; ++i) {",
     "const double w = gate(c->alpha[g * (c->Hq / c->Hkv)]);\n\n    for (int i = 0; i < B; ++i) {"),
]


@pytest.mark.parametrize("name,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_mutant_is_caught(tmp_path, name, old, new):
    src = open(SOURCE).read()
    assert src.count(old) == 1, f"mutation site for '{name}' not found exactly once"
    mutant_src = tmp_path / "mutant.c"
    mutant_src.write_text(src.replace(old, new))
    lib = build_oracle(str(mutant_src), str(tmp_path / "libmutant.so"))
    proc = subprocess.run([sys.executable, os.path.join(HERE, "oracle_pins.py"), lib],
                          capture_output=True, text=True, timeout=300)
    caught = proc.returncode != 0 or "FAIL" in proc.stdout
    assert caught, f"mutant '{name}' passed every pin:\n{proc.stdout}\n{proc.stderr}"


def test_unmutated_copy_passes(tmp_path):
    """Control: the same harness on an unmodified copy reports no failure."""
    lib = build_oracle(SOURCE, str(tmp_path / "libcontrol.so"))
    proc = subprocess.run([sys.executable, os.path.join(HERE, "oracle_pins.py"), lib],
                          capture_output=True, text=True, timeout=300)
    assert proc.returncode == 0 and "FAIL" not in proc.stdout and "DONE" in proc.stdout, proc.stdout
