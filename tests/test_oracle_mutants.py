"""Plant plausible mistakes in copies of the oracle source and check that the pins
catch each one (CPU only).  The committed oracle is never modified: each mutant is
a rewritten copy compiled into a temporary directory."""
import os

import pytest

import oracle
from oracle_pins import ALL_PINS

# (what the mistake is, text in estp_oracle.c, replacement)
MUTANTS = [
    ("entropy in bits", "H -= p * log(p);", "H -= p * log2(p);"),
    ("output rows_from off by one", "for (int64_t i = c->row_from; i < T; i++) {",
     "for (int64_t i = c->row_from + 1; i < T; i++) {"),
    ("entropy sign", "H -= p * log(p);", "H += p * log(p);"),
    ("entropy unnormalised", "double p = e[v] / s;", "double p = e[v];"),
    ("entropy ignores row stride", "int64_t off = r * c->ld;", "int64_t off = r * c->V;"),
    ("bf16 widening shift", "[idx] << 16;", "[idx] << 15;"),
    ("lm-head dot drops the last coordinate",
     "for (int64_t k = 0; k < c->D; ++k) dot +=", "for (int64_t k = 0; k < c->D - 1; ++k) dot +="),
    ("lm-head W transposed", "load_elem(c->W, c->dtype, v * c->ldw + k)",
     "load_elem(c->W, c->dtype, k * c->V + v)"),
    ("lm-head entropy sign", "H += -p * log(p);", "H += p * log(p);"),
    ("scores unscaled", "s[j] = c->scale * dot;", "s[j] = dot;"),
    ("row sums instead of column sums", "col[j] += exp(s[j] - m) / Z;",
     "col[i] += exp(s[j] - m) / Z;"),
    ("softmax unnormalised", "col[j] += exp(s[j] - m) / Z;", "col[j] += exp(s[j] - m);"),
    ("GQA head mapping", "int g = h / (c->Hq / c->Hkv);", "int g = h % c->Hkv;"),
    ("K head ignored", "((t0 + t) * c->Hkv + g)", "((t0 + t) * c->Hkv + 0)"),
    ("Q prompt offset dropped", "((t0 + t) * c->Hq + h)", "((t) * c->Hq + h)"),
    ("self term never excluded", "if (c->exclude_self && j == i) continue;", ""),
    ("lse sign", "m + log(Z);", "m - log(Z);"),
    ("output scores unscaled", "s[j] = dot * c->scale;", "s[j] = dot;"),
    ("output weights unnormalised", "const double a = exp(s[j] - m) / Z;",
     "const double a = exp(s[j] - m);"),
    ("output reads the key rows as values", "v[t * d + x] = load_elem(c->V,",
     "v[t * d + x] = load_elem(c->K,"),
    ("output ignores the GQA map", "const int64_t row_kv = (t0 + t) * (int64_t)c->Hkv + g;",
     "const int64_t row_kv = (t0 + t) * (int64_t)c->Hkv + 0;"),
    ("output drops the diagonal", "for (int64_t j = 0; j <= i; ++j) {\n            const double a",
     "for (int64_t j = 0; j < i; ++j) {\n            const double a"),
    ("rows_from off by one", "for (int64_t i = c->row_from; i < T; ++i) {",
     "for (int64_t i = c->row_from + 1; i < T; ++i) {"),
    ("causal count divisor", "if (divisor == ORACLE_DIV_LENGTH) n = (double)N;",
     "if (divisor == ORACLE_DIV_LENGTH) n = (double)(N - j);"),
    ("head mean dropped", "(n * (double)n_layers * (double)n_heads)", "(n * (double)n_layers)"),
    ("causal count keeps the diagonal", "(double)(N - j - (exclude_self ? 1 : 0))",
     "(double)(N - j)"),
    ("causal count off by one", "(double)(N - j - (exclude_self ? 1 : 0))",
     "(double)(N - j + 1 - (exclude_self ? 1 : 0))"),
    ("no-divisor variant divides by N", "else n = 1.0;", "else n = (double)N;"),
    ("temperature ignored", "w[i] = T / alpha;", "w[i] = T;"),
    ("lambdas swapped", "lambda1 * S[t0 + i] + lambda2 * H[t0 + i]",
     "lambda1 * H[t0 + i] + lambda2 * S[t0 + i]"),
    ("pool weights unnormalised", "double e = exp(w[i] - M) / Z;", "double e = exp(w[i] - M);"),
    ("pool ignores row stride", "(t0 + i) * ldh + x", "(t0 + i) * D + x"),
    ("head bias dropped", "double acc = bias ? (double)bias[k] : 0.0;", "double acc = 0.0;"),
    ("head W transposed", "W[(int64_t)k * D + x]", "W[(int64_t)x * K + k]"),
    ("expectation over bin index", "y += p * (double)centers[k];", "y += p * (double)k;"),
    ("MSE gradient without its factor 2", "(1.0 - lambda3) * 2.0 * err", "(1.0 - lambda3) * err"),
    ("CE gradient sign", "(lambda3 * (p_hat[k] - p) +", "(lambda3 * (p - p_hat[k]) +"),
    ("MSE not averaged over the batch", "(1.0 - lambda3) * mse / (double)B;",
     "(1.0 - lambda3) * mse;"),
    ("soft label decays with the squared distance",
     "const double p = exp(-fabs((double)(k - i))) / norm;",
     "const double p = exp(-(double)((k - i) * (k - i))) / norm;"),
    ("gradient not divided by the batch size", "((double)centers[k] - yh[b])) / (double)B;",
     "((double)centers[k] - yh[b]));"),
    ("feature gradient through W transposed", "g += (double)wk[x] * dz[k];",
     "g += (double)W[x * K + k] * dz[k];"),
    ("MLP without its ReLU", "u[(int64_t)b * F + f] = a > 0.0 ? a : 0.0;",
     "u[(int64_t)b * F + f] = a;"),
    ("MLP first layer transposed", "(double)W1[(int64_t)f * D + x] * pooled",
     "(double)W1[(int64_t)x * F + f] * pooled"),
    ("MLP gradient passes switched-off units", "if (!(u[q] > 0.0)) du[q] = 0.0;", ""),
    ("MLP input gradient through W1 transposed", "(double)W1[(int64_t)f * D + x] * du",
     "(double)W1[(int64_t)x * F + f] * du"),
    ("MLP first-layer bias gradient averaged", "grad_b1[f] = g;", "grad_b1[f] = g / (double)B;"),
]


@pytest.mark.parametrize("what,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_mutant_is_caught(what, old, new, tmp_path):
    src = oracle.source_text()
    assert src.count(old) == 1, f"mutation site for '{what}' must occur exactly once"
    so = oracle.compile_source(src.replace(old, new), str(tmp_path / "liboracle_mut.so"))
    failed = []
    with oracle.use_library(so):
        for pin in ALL_PINS:
            try:
                pin()
            except AssertionError:
                failed.append(pin.__name__)
    assert failed, f"no pin catches the planted mistake '{what}'"
