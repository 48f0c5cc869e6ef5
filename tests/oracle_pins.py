"""Pins of the fp64 oracle to facts fixed by the mathematics, not by the oracle.

Each pin is a function that raises AssertionError when the oracle (whichever build
``oracle`` currently routes to) disagrees with a closed form, an invariant, or an
independent library routine (scipy) on tiny inputs.  ``test_oracle_pins`` runs all
of them on the committed oracle; ``test_oracle_mutants`` runs them on copies of the
oracle with planted mistakes and requires that some pin fails for every mistake.
"""
from __future__ import annotations

import math

import numpy as np
from scipy import special, stats

import oracle
from synth import f32_to_bf16_bits

RTOL = 1e-11


def _close(a, b, rtol=RTOL, atol=1e-12, what=""):
    a, b = np.asarray(a, dtype=np.float64), np.asarray(b, dtype=np.float64)
    assert a.shape == b.shape, f"{what}: shape {a.shape} vs {b.shape}"
    assert np.allclose(a, b, rtol=rtol, atol=atol), (
        f"{what}: max abs diff {np.max(np.abs(a - b)) if a.size else 0}")


def _rng(seed=0):
    return np.random.default_rng(seed)


# ------------------------------------------------------------- Eq. 2-1 entropy

def pin_entropy_uniform():
    """Uniform logits give H = ln V exactly (any constant, any V)."""
    for V in (1, 7, 64, 32000, 152064):
        for c in (0.0, -3.5, 17.0):
            z = np.full((2, V), c, dtype=np.float32)
            # naive summation of V terms: relative rounding bound ~ V * 2**-53
            _close(oracle.token_entropy(z), [math.log(V)] * 2, rtol=max(1e-12, V * 2.0**-52),
                   what=f"uniform V={V}")
    z = f32_to_bf16_bits(np.full((1, 128256), 2.0, dtype=np.float32))
    _close(oracle.token_entropy(z), [math.log(128256)], rtol=128256 * 2.0**-52,
           what="uniform bf16")


def pin_entropy_onehot_and_ties():
    """One dominant logit gives H = 0; k tied dominant logits give H = ln k."""
    V = 1000
    for k in (1, 2, 3, 10):
        z = np.zeros((1, V), dtype=np.float32)
        z[0, np.arange(k) * 37] = 1e4
        _close(oracle.token_entropy(z), [math.log(k)], atol=1e-12, what=f"ties k={k}")


def pin_entropy_two_level():
    """a entries at x and V-a at 0: H = -a p ln p - (V-a) q ln q,
    p = e^x / (a e^x + V - a), q = 1 / (a e^x + V - a)."""
    for V, a, x in ((50, 3, 2.5), (32000, 17, 6.0), (1000, 999, -1.25), (64, 1, 0.5)):
        z = np.zeros((1, V), dtype=np.float32)
        z[0, :a] = x
        den = a * math.exp(x) + (V - a)
        p, q = math.exp(x) / den, 1.0 / den
        ref = -a * p * math.log(p) - (V - a) * q * math.log(q)
        _close(oracle.token_entropy(z), [ref], rtol=max(1e-12, V * 2.0**-52),
               what=f"two-level V={V}")


def pin_entropy_library_bruteforce():
    """Small V: scipy.stats.entropy of scipy.special.softmax (natural log)."""
    rng = _rng(1)
    for V in (1, 2, 5, 33, 64):
        z = (rng.standard_normal((6, V)) * rng.uniform(0.1, 6, (6, 1))).astype(np.float32)
        ref = [stats.entropy(special.softmax(r.astype(np.float64))) for r in z]
        _close(oracle.token_entropy(z), ref, rtol=1e-11, atol=1e-13, what=f"scipy V={V}")


def pin_entropy_shift_perm_pad():
    """H(z + c) = H(z); H is invariant to permuting a row; columns past V are ignored."""
    rng = _rng(2)
    V = 300
    z = np.round(rng.standard_normal((4, V)) * 64).astype(np.float32) / 16  # exact grid
    H = oracle.token_entropy(z)
    _close(oracle.token_entropy(z + np.float32(8.0)), H, rtol=1e-12, what="shift")
    _close(oracle.token_entropy(z[:, rng.permutation(V)]), H, rtol=1e-12, what="perm")
    padded = np.full((4, V + 13), 1e4, dtype=np.float32)
    padded[:, :V] = z
    _close(oracle.token_entropy(padded, V=V), H, rtol=1e-12, what="ld padding")


# ------------------------------------------------------- Eq. 2-0 importance

def pin_lm_head_zero_weights():
    """Logits formed from hidden states: W = 0 gives uniform logits, H = ln V."""
    rng = _rng(41)
    for V, D in ((1, 8), (7, 3), (300, 64)):
        h = rng.standard_normal((3, D)).astype(np.float32)
        W = np.zeros((V, D), dtype=np.float32)
        _close(oracle.lm_head_entropy(h, W), [math.log(V)] * 3, what="W = 0")


def pin_lm_head_two_level():
    """A hidden row c e_k reads column k of W only: with a entries x / c and V - a zeros
    there, the logits are two-level (a at x, V - a at 0) and H has the closed form of the
    two-level pin, whatever the other columns of W hold."""
    rng = _rng(42)
    for V, D, a, x, k in ((50, 6, 3, 2.5, 4), (1000, 16, 999, -1.25, 0), (64, 3, 1, 0.5, 2)):
        c = 2.0
        W = rng.standard_normal((V, D)).astype(np.float64)
        W[:, k] = 0.0
        W[rng.choice(V, a, replace=False), k] = x / c
        h = np.zeros((1, D))
        h[0, k] = c
        Z = a * math.exp(x) + V - a
        p, q = math.exp(x) / Z, 1.0 / Z
        ref = -a * p * math.log(p) - (V - a) * q * math.log(q)
        _close(oracle.lm_head_entropy(h.astype(np.float32), W.astype(np.float32)), [ref],
               rtol=1e-6, what="two-level from hidden")


def pin_lm_head_bruteforce():
    """Tiny shapes, fp32 and bf16: a pure-Python triple loop forms every logit and the
    entropy with math.exp / math.log."""
    from synth import bf16_bits_to_f32
    rng = _rng(43)
    for rows, D, V in ((3, 5, 7), (2, 9, 1), (4, 1, 11)):
        h = rng.standard_normal((rows, D)).astype(np.float32) * 2
        W = rng.standard_normal((V, D)).astype(np.float32)
        for bf16 in (False, True):
            if bf16:
                hb, Wb = (np.asarray(x).view(np.uint32) >> 16 for x in (h, W))
                hb, Wb = hb.astype(np.uint16), Wb.astype(np.uint16)
                hv, Wv = bf16_bits_to_f32(hb).astype(np.float64), bf16_bits_to_f32(Wb).astype(np.float64)
                got = oracle.lm_head_entropy(hb, Wb)
            else:
                hv, Wv = h.astype(np.float64), W.astype(np.float64)
                got = oracle.lm_head_entropy(h, W)
            ref = []
            for r in range(rows):
                z = [sum(float(hv[r, k]) * float(Wv[v, k]) for k in range(D)) for v in range(V)]
                m = max(z)
                e = [math.exp(t - m) for t in z]
                sm = sum(e)
                ref.append(-sum((x / sm) * math.log(x / sm) for x in e if x > 0))
            _close(got, ref, rtol=1e-12, atol=1e-12, what=f"brute force bf16={bf16}")


def _brute_colsum(Q, K, cu, scale, heads=None, exclude_self=False):
    """Full masked score matrix per (prompt, head); rows via scipy softmax."""
    Qd = Q.astype(np.float64) if Q.dtype != np.uint16 else _bf(Q)
    Kd = K.astype(np.float64) if K.dtype != np.uint16 else _bf(K)
    sumT, Hq, d = Qd.shape
    rep = Hq // Kd.shape[1]
    heads = range(Hq) if heads is None else heads
    C = np.zeros(sumT)
    for b in range(len(cu) - 1):
        t0, t1 = cu[b], cu[b + 1]
        if t1 == t0:
            continue
        T = t1 - t0
        for h in heads:
            S = scale * Qd[t0:t1, h] @ Kd[t0:t1, h // rep].T
            S[np.triu_indices(T, 1)] = -np.inf
            A = special.softmax(S, axis=1)
            if exclude_self:
                A[np.diag_indices(T)] = 0.0
            C[t0:t1] += A.sum(axis=0)
    return C


def _bf(a):
    from synth import bf16_bits_to_f32
    return bf16_bits_to_f32(a).astype(np.float64)


def _qk(rng, cu, Hq, Hkv, d, spread=1.0, dtype=np.float32):
    sumT = int(cu[-1])
    Q = (rng.standard_normal((sumT, Hq, d)) * spread).astype(np.float32)
    K = (rng.standard_normal((sumT, Hkv, d)) * spread).astype(np.float32)
    if dtype == np.uint16:
        return f32_to_bf16_bits(Q), f32_to_bf16_bits(K)
    return Q, K


def pin_attn_output_rows_and_uniform():
    """Attention output O = A V (Sec. 3.1): softmax rows sum to 1, so V = 1 gives O = 1;
    Q = 0 makes every causal row uniform, so O_i is the running mean of v_0 .. v_i (numpy
    cumulative sums), per prompt and per KV head of each query head."""
    rng = _rng(61)
    cu = np.array([0, 5, 5, 21, 22], np.int32)
    Hq, Hkv, d = 6, 2, 8
    sumT = int(cu[-1])
    Q = rng.standard_normal((sumT, Hq, d)).astype(np.float32)
    K = rng.standard_normal((sumT, Hkv, d)).astype(np.float32)
    ones = np.ones((sumT, Hkv, d), np.float32)
    _close(oracle.attn_output(Q, K, ones, cu, 0.4), np.ones((sumT, Hq, d)), rtol=1e-12,
           what="V = 1")
    V = rng.standard_normal((sumT, Hkv, d)).astype(np.float32)
    O = oracle.attn_output(np.zeros_like(Q), K, V, cu, 0.4)
    ref = np.zeros((sumT, Hq, d))
    for b in range(len(cu) - 1):
        t0, t1 = int(cu[b]), int(cu[b + 1])
        if t1 == t0:
            continue
        cum = np.cumsum(V[t0:t1].astype(np.float64), axis=0) / np.arange(1, t1 - t0 + 1)[:, None, None]
        for h in range(Hq):
            ref[t0:t1, h] = cum[:, h // (Hq // Hkv)]
    _close(O, ref, rtol=1e-12, atol=1e-12, what="uniform rows: running mean")


def pin_attn_output_bruteforce():
    """T <= 16: the full masked score matrix, scipy softmax rows, times V (numpy)."""
    rng = _rng(62)
    for cu, Hq, Hkv, d in (([0, 16], 2, 2, 8), ([0, 3, 3, 12, 13], 4, 2, 16)):
        cu = np.asarray(cu, np.int32)
        sumT = int(cu[-1])
        Q = rng.standard_normal((sumT, Hq, d)).astype(np.float32)
        K = rng.standard_normal((sumT, Hkv, d)).astype(np.float32)
        V = rng.standard_normal((sumT, Hkv, d)).astype(np.float32)
        scale = 1 / math.sqrt(d)
        ref = np.zeros((sumT, Hq, d))
        for b in range(len(cu) - 1):
            t0, t1 = int(cu[b]), int(cu[b + 1])
            T = t1 - t0
            if T == 0:
                continue
            for h in range(Hq):
                g = h // (Hq // Hkv)
                s = scale * Q[t0:t1, h].astype(np.float64) @ K[t0:t1, g].astype(np.float64).T
                s[np.triu_indices(T, 1)] = -np.inf
                ref[t0:t1, h] = special.softmax(s, axis=1) @ V[t0:t1, g].astype(np.float64)
        _close(oracle.attn_output(Q, K, V, cu, scale), ref, rtol=1e-12, atol=1e-12,
               what="attention output brute force")


def pin_attn_output_rows_bruteforce():
    """Output rows i >= row_from only (prompt-local index): those rows equal the brute-force
    softmax rows times V (numpy / scipy), and the rows before stay 0."""
    rng = _rng(63)
    cu = np.asarray([0, 3, 3, 12, 13], np.int32)
    Hq, Hkv, d, row_from = 4, 2, 16, 2
    sumT = int(cu[-1])
    Q = rng.standard_normal((sumT, Hq, d)).astype(np.float32)
    K = rng.standard_normal((sumT, Hkv, d)).astype(np.float32)
    V = rng.standard_normal((sumT, Hkv, d)).astype(np.float32)
    scale = 0.3
    ref = np.zeros((sumT, Hq, d))
    for b in range(len(cu) - 1):
        t0, t1 = int(cu[b]), int(cu[b + 1])
        T = t1 - t0
        if T == 0:
            continue
        for h in range(Hq):
            g = h // (Hq // Hkv)
            s = scale * Q[t0:t1, h].astype(np.float64) @ K[t0:t1, g].astype(np.float64).T
            s[np.triu_indices(T, 1)] = -np.inf
            full = special.softmax(s, axis=1) @ V[t0:t1, g].astype(np.float64)
            ref[t0 + row_from:t1, h] = full[row_from:]
    _close(oracle.attn_output_rows(Q, K, V, cu, scale, row_from), ref, rtol=1e-12, atol=1e-12,
           what="attention output rows >= row_from")


def pin_importance_bruteforce():
    """T <= 16: column sums of scipy softmax rows of the causal score matrix."""
    rng = _rng(3)
    for cu, Hq, Hkv, d in (([0, 16], 2, 2, 8), ([0, 5, 5, 16, 17], 4, 2, 16),
                           ([0, 9, 12], 6, 3, 4)):
        cu = np.asarray(cu, dtype=np.int32)
        for dt in (np.float32, np.uint16):
            Q, K = _qk(rng, cu, Hq, Hkv, d, spread=1.5, dtype=dt)
            sc = 1 / math.sqrt(d)
            _close(oracle.attn_colsum(Q, K, cu, sc), _brute_colsum(Q, K, cu, sc),
                   rtol=1e-11, what=f"brute cu={list(cu)}")
            hs = [Hq - 1, 0]
            _close(oracle.attn_colsum(Q, K, cu, sc, heads=hs),
                   _brute_colsum(Q, K, cu, sc, heads=hs), rtol=1e-11, what="brute heads")
            _close(oracle.attn_colsum(Q, K, cu, sc, exclude_self=True),
                   _brute_colsum(Q, K, cu, sc, exclude_self=True), rtol=1e-11,
                   what="brute exclude_self")


def pin_importance_row_sums():
    """Each causal softmax row sums to 1, so sum_j C_j = T_b per head; with the 1/N
    scaling and head/layer mean, S sums to 1 over each prompt."""
    rng = _rng(4)
    cu = np.asarray([0, 1, 40, 41, 140], dtype=np.int32)
    Q, K = _qk(rng, cu, 4, 1, 32, spread=2.0)
    sc = 0.3
    C = oracle.attn_colsum(Q, K, cu, sc)
    C = oracle.attn_colsum(Q * np.float32(0.5), K, cu, sc, out=C)  # a second "layer"
    for b in range(len(cu) - 1):
        T = cu[b + 1] - cu[b]
        _close(C[cu[b]:cu[b + 1]].sum(), 2 * 4 * T, rtol=1e-12, what="colsum total")
    S = oracle.importance(C, cu, n_layers=2, n_heads=4)
    for b in range(len(cu) - 1):
        _close(S[cu[b]:cu[b + 1]].sum(), 1.0, rtol=1e-12, what="S sums to 1")
    _close(S[cu[0]], 1.0, rtol=1e-12, what="T=1 gives S=1")
    _close(S[cu[2]], 1.0, rtol=1e-12, what="T=1 gives S=1")


def pin_importance_uniform_harmonic():
    """Q = 0 (or K = 0) makes every causal row uniform, A_ij = 1/(i+1) (0-based), so
    S_j = (H_N - H_j) / N with harmonic numbers H_n."""
    rng = _rng(5)
    cu = np.asarray([0, 7, 300], dtype=np.int32)
    Q, K = _qk(rng, cu, 2, 1, 16)
    for QQ, KK in ((np.zeros_like(Q), K), (Q, np.zeros_like(K))):
        C = oracle.attn_colsum(QQ, KK, cu, 0.25)
        S = oracle.importance(C, cu, n_layers=1, n_heads=2)
        for b in range(2):
            N = cu[b + 1] - cu[b]
            Hn = np.concatenate([[0.0], np.cumsum(1.0 / np.arange(1, N + 1))])
            ref = (Hn[N] - Hn[np.arange(N)]) / N
            _close(S[cu[b]:cu[b + 1]], ref, rtol=1e-12, what="harmonic")


def pin_importance_divisors_uniform():
    """The divisor variants of Eq. 2-0 under uniform causal rows (Q = 0), A_ij = 1/(i+1):
    C_j = H_N - H_j (H_N - H_{j+1} without the diagonal).  Causal count: n_j = N - j
    (N - j - 1 without the diagonal, S = 0 where it is 0); none: S_j = C_j."""
    rng = _rng(15)
    cu = np.asarray([0, 1, 9, 200], dtype=np.int32)
    Q, K = _qk(rng, cu, 2, 1, 16)
    for excl in (False, True):
        C = oracle.attn_colsum(np.zeros_like(Q), K, cu, 0.25, exclude_self=excl)
        Sc = oracle.importance(C, cu, n_layers=1, n_heads=2, divisor="causal", exclude_self=excl)
        Sn = oracle.importance(C, cu, n_layers=1, n_heads=2, divisor="none", exclude_self=excl)
        for b in range(len(cu) - 1):
            N = int(cu[b + 1] - cu[b])
            Hn = np.concatenate([[0.0], np.cumsum(1.0 / np.arange(1, N + 1))])
            j = np.arange(N)
            col = Hn[N] - Hn[j + (1 if excl else 0)]
            cnt = N - j - (1 if excl else 0)
            ref_c = np.where(cnt > 0, col / np.maximum(cnt, 1), 0.0)
            _close(Sc[cu[b]:cu[b + 1]], ref_c, rtol=1e-12, what=f"causal excl={excl}")
            _close(Sn[cu[b]:cu[b + 1]], col, rtol=1e-12, what=f"none excl={excl}")


def pin_importance_divisor_invariants():
    """Random inputs: with the diagonal, every softmax row sums to 1, so the "none"
    variant sums to N_b per prompt; the causal variant of the last token is its own
    diagonal weight A_{N-1,N-1} averaged over heads, 1 / sum_j exp(s_{N-1,j} - s_{N-1,N-1})
    from a direct softmax of that row."""
    rng = _rng(16)
    cu = np.asarray([0, 5, 64, 130], dtype=np.int32)
    Hq, Hkv, d, sc = 4, 2, 16, 0.3
    Q, K = _qk(rng, cu, Hq, Hkv, d)
    C = oracle.attn_colsum(Q, K, cu, sc)
    Sn = oracle.importance(C, cu, n_layers=1, n_heads=Hq, divisor="none")
    Sc = oracle.importance(C, cu, n_layers=1, n_heads=Hq, divisor="causal")
    q64, k64 = Q.astype(np.float64), K.astype(np.float64)
    for b in range(len(cu) - 1):
        t0, t1 = int(cu[b]), int(cu[b + 1])
        _close(np.sum(Sn[t0:t1]), float(t1 - t0), rtol=1e-12, what="none sums to N")
        diag = 0.0
        for h in range(Hq):
            s = sc * (k64[t0:t1, h // (Hq // Hkv)] @ q64[t1 - 1, h])
            diag += 1.0 / np.sum(np.exp(s - s[-1]))
        _close(Sc[t1 - 1], diag / Hq, rtol=1e-12, what="causal last token")


def pin_importance_gqa_and_scale():
    """GQA: query head h reads KV head h // rep -- equal to the MHA case with K heads
    repeated; the softmax scale multiplies the scores (doubling Q == doubling scale)."""
    rng = _rng(6)
    cu = np.asarray([0, 12, 30], dtype=np.int32)
    Q, K = _qk(rng, cu, 6, 2, 8)
    Krep = np.repeat(K, 3, axis=1)
    a = oracle.attn_colsum(Q, K, cu, 0.4)
    _close(a, oracle.attn_colsum(Q, Krep, cu, 0.4), rtol=1e-12, what="gqa == repeated mha")
    _close(oracle.attn_colsum(Q * np.float32(2), K, cu, 0.2), a, rtol=1e-12, what="scale")
    for h in range(6):  # head h alone == brute force on head h with kv h//3
        _close(oracle.attn_colsum(Q, K, cu, 0.4, heads=[h]),
               _brute_colsum(Q, K, cu, 0.4, heads=[h]), rtol=1e-11, what=f"head {h}")


def pin_importance_rows_from():
    """Forming only rows i >= r gives the exact column sums of keys j >= r (they receive
    mass only from those rows) and strictly less for earlier keys."""
    rng = _rng(13)
    cu = np.asarray([0, 40, 43], dtype=np.int32)
    Q, K = _qk(rng, cu, 4, 2, 8, spread=1.5)
    full = oracle.attn_colsum(Q, K, cu, 0.3, exclude_self=True)
    for r in (0, 5, 39):
        part = oracle.attn_colsum_rows(Q, K, cu, 0.3, r, exclude_self=True)
        for b in range(2):
            lo, hi = cu[b], cu[b + 1]
            late = np.arange(lo, hi) >= lo + r
            _close(part[lo:hi][late], full[lo:hi][late], rtol=1e-12, what=f"rows_from {r}")
            if r > 0:
                assert np.all(part[lo:hi][~late] < full[lo:hi][~late] + 1e-15)


def pin_lse_library():
    """Row log-normalisers equal scipy.special.logsumexp over the causal prefix."""
    rng = _rng(7)
    cu = np.asarray([0, 3, 20], dtype=np.int32)
    Q, K = _qk(rng, cu, 4, 2, 8, spread=2.0)
    sc = 0.35
    lse = oracle.attn_lse(Q, K, cu, sc)
    Qd, Kd = Q.astype(np.float64), K.astype(np.float64)
    for b in range(2):
        for h in range(4):
            for i in range(cu[b], cu[b + 1]):
                s = sc * Kd[cu[b]:i + 1, h // 2] @ Qd[i, h]
                _close(lse[h, i], special.logsumexp(s), rtol=1e-12, what="lse")


def pin_importance_prompt_independence():
    """Prompts are independent: the packed result equals each prompt run alone."""
    rng = _rng(8)
    cu = np.asarray([0, 10, 11, 40], dtype=np.int32)
    Q, K = _qk(rng, cu, 2, 2, 8)
    C = oracle.attn_colsum(Q, K, cu, 0.3)
    for b in range(3):
        sub = np.asarray([0, cu[b + 1] - cu[b]], dtype=np.int32)
        _close(C[cu[b]:cu[b + 1]], oracle.attn_colsum(Q[cu[b]:cu[b + 1]], K[cu[b]:cu[b + 1]],
                                                     sub, 0.3), rtol=1e-12, what="independent")


# ---------------------------------------------------- Eqs. 2-2..2-4 pooling

def _pool_inputs(rng, cu, D, dtype=np.float32):
    sumT = int(cu[-1])
    hid = rng.standard_normal((sumT, D)).astype(np.float32)
    if dtype == np.uint16:
        hid = f32_to_bf16_bits(hid)
    H = rng.uniform(0, 10, sumT)
    S = rng.uniform(0, 0.05, sumT)
    return hid, H, S


def pin_pool_mean():
    """lambda1 = lambda2 = 0 gives uniform weights: the pooled vector is the mean."""
    rng = _rng(9)
    cu = np.asarray([0, 1, 50, 177], dtype=np.int32)
    hid, H, S = _pool_inputs(rng, cu, 40)
    P = oracle.pool(hid, H, S, cu, 0.0, 0.0, 1.0)
    for b in range(3):
        _close(P[b], hid[cu[b]:cu[b + 1]].astype(np.float64).mean(axis=0), rtol=1e-12,
               what="mean pool")


def pin_pool_library_weights():
    """Weights are scipy.special.softmax((lambda1 S + lambda2 H) / alpha) per prompt,
    and the pooled vector is the weighted sum of the rows."""
    rng = _rng(10)
    cu = np.asarray([0, 33, 34, 90], dtype=np.int32)
    for dt in (np.float32, np.uint16):
        hid, H, S = _pool_inputs(rng, cu, 24, dt)
        hd = hid.astype(np.float64) if dt == np.float32 else _bf(hid)
        for l1, l2, al in ((0.7, 0.3, 1.0), (0.0, 1.0, 0.5), (1.0, 0.0, 2.0), (3.0, -0.2, 0.1)):
            P, w = oracle.pool(hid, H, S, cu, l1, l2, al, return_weights=True)
            for b in range(3):
                sl = slice(cu[b], cu[b + 1])
                ref_w = special.softmax((l1 * S[sl] + l2 * H[sl]) / al)
                _close(w[sl], ref_w, rtol=1e-12, what="weights")
                _close(w[sl].sum(), 1.0, rtol=1e-12, what="weights sum to 1")
                _close(P[b], ref_w @ hd[sl], rtol=1e-11, what="weighted sum")


def pin_pool_limits():
    """alpha -> 0 selects the argmax token's row; T = 1 returns that row; an empty
    prompt pools to zero; permuting (T_i, h_i) pairs leaves the result unchanged."""
    rng = _rng(11)
    cu = np.asarray([0, 20, 21, 21, 60], dtype=np.int32)
    hid, H, S = _pool_inputs(rng, cu, 16)
    P = oracle.pool(hid, H, S, cu, 0.0, 1.0, 1e-6)
    _close(P[0], hid[cu[0] + np.argmax(H[:20])], rtol=1e-12, what="alpha->0")
    _close(P[1], hid[20], rtol=1e-12, what="T=1")
    _close(P[2], np.zeros(16), what="empty prompt")
    perm = np.concatenate([np.arange(0, 21), 21 + rng.permutation(39)])
    P2 = oracle.pool(hid[perm], H[perm], S[perm], cu, 0.4, 0.6, 0.7)
    _close(P2, oracle.pool(hid, H, S, cu, 0.4, 0.6, 0.7), rtol=1e-12, what="permutation")
    padded = np.full((60, 16 + 5), 1e4, dtype=np.float32)  # row stride > D
    padded[:, :16] = hid
    _close(oracle.pool(padded, H, S, cu, 0.4, 0.6, 0.7, D=16),
           oracle.pool(hid, H, S, cu, 0.4, 0.6, 0.7), rtol=1e-12, what="row stride")


def pin_pool_two_token():
    """Two tokens: e_1 = 1 / (1 + exp((T_2 - T_1)/alpha))."""
    hid = np.asarray([[1.0, 0.0, 2.0], [0.0, 1.0, -2.0]], dtype=np.float32)
    H = np.asarray([2.0, 5.0])
    S = np.asarray([0.9, 0.1])
    l1, l2, al = 2.0, 0.5, 0.8
    T1, T2 = l1 * S[0] + l2 * H[0], l1 * S[1] + l2 * H[1]
    e1 = 1.0 / (1.0 + math.exp((T2 - T1) / al))
    P = oracle.pool(hid, H, S, np.asarray([0, 2], dtype=np.int32), l1, l2, al)
    _close(P[0], e1 * hid[0].astype(np.float64) + (1 - e1) * hid[1].astype(np.float64),
           rtol=1e-12, what="two tokens")


# ------------------------------------------------------ Eq. 3-2 length head

def pin_head():
    """W = 0 (bias 0) gives the mean of the bin centres; a dominant logit selects its
    centre; in general p is scipy softmax(W h + b) and y = p . c."""
    rng = _rng(12)
    K, D = 32, 20
    c = ((np.arange(K) + 0.5) * 256).astype(np.float32)
    h = rng.standard_normal((3, D))
    y = oracle.length_head(h, np.zeros((K, D), np.float32), np.zeros(K, np.float32), c)
    _close(y, [c.astype(np.float64).mean()] * 3, rtol=1e-12, what="W=0")
    bias = np.zeros(K, np.float32)
    bias[11] = 1e4
    y = oracle.length_head(h, np.zeros((K, D), np.float32), bias, c)
    _close(y, [float(c[11])] * 3, rtol=1e-12, what="dominant bin")
    W = rng.standard_normal((K, D)).astype(np.float32)
    b = rng.standard_normal(K).astype(np.float32)
    y, p = oracle.length_head(h, W, b, c, return_probs=True)
    ref_p = special.softmax(h @ W.astype(np.float64).T + b.astype(np.float64), axis=1)
    _close(p, ref_p, rtol=1e-11, what="probs")
    _close(y, ref_p @ c.astype(np.float64), rtol=1e-11, what="expectation")


def _soft_label(K, i):
    """Eq. 3-1 written out: exp(-|j - i|) normalised over the K bins."""
    e = np.exp(-np.abs(np.arange(K) - i).astype(np.float64))
    return e / e.sum()


def pin_head_loss_closed_forms():
    """W = 0, bias = 0: p_hat is uniform (1/K) and y_hat the mean centre, so
    CE = ln K for every target and MSE = (mean c - y)^2; with lambda3 = 1 the loss is
    ln K exactly and dL/db_k = (1/K - p_k) averaged over the batch."""
    K, D = 8, 6
    c = ((np.arange(K) + 0.5) * 100).astype(np.float32)
    h = _rng(17).standard_normal((3, D))
    y = np.asarray([40.0, 420.0, 799.0], np.float32)   # bins 0, 4, 7 (nearest centres)
    Wz, bz = np.zeros((K, D), np.float32), np.zeros(K, np.float32)
    L1, gW, gb, gp = oracle.head_loss(h, Wz, bz, c, y, 1.0)
    _close(L1, math.log(K), rtol=1e-13, what="CE of a uniform prediction")
    ref_gb = np.mean([1.0 / K - _soft_label(K, i) for i in (0, 4, 7)], axis=0)
    _close(gb, ref_gb, rtol=1e-12, atol=1e-15, what="CE bias gradient")
    _close(gp, np.zeros_like(gp), what="W = 0: no gradient to the features")
    L0 = oracle.head_loss(h, Wz, bz, c, y, 0.0, grads=False)
    mc = float(np.mean(c.astype(np.float64)))
    _close(L0, float(np.mean((mc - y.astype(np.float64)) ** 2)), rtol=1e-13, what="MSE")


def pin_head_loss_soft_label():
    """A head whose softmax equals the soft label of the target's bin: the CE term is
    the label's own entropy -sum p ln p (minimum of CE over p_hat), and the label is
    symmetric, sums to 1 and falls by exactly e per bin away from i."""
    K, D = 9, 4
    c = np.arange(K, dtype=np.float32) * 10.0
    for i in (0, 3, 8):
        p = _soft_label(K, i)
        _close(p.sum(), 1.0, rtol=1e-15, what="sums to 1")
        _close(p[i + 1:] * math.e, p[i:-1], rtol=1e-13, atol=0, what="geometric decay")
        bias = np.log(p).astype(np.float32)        # softmax(bias) == p up to fp32 rounding
        h = np.zeros((1, D))
        y = np.asarray([c[i] + 1.0], np.float32)   # nearest centre: bin i
        L = oracle.head_loss(h, np.zeros((K, D), np.float32), bias, c, y, 1.0, grads=False)
        q = special.softmax(bias.astype(np.float64))
        _close(L, float(-(p * np.log(q)).sum()), rtol=1e-12, what="CE with p_hat = softmax(bias)")
        _close(L, float(-(p * np.log(p)).sum()), rtol=1e-6, what="CE close to the label entropy")


def pin_head_loss_gradients():
    """The analytic gradients against central finite differences of the oracle's own
    loss, for W, the bias and the pooled features, at several lambda3."""
    rng = _rng(18)
    B, D, K = 3, 5, 6
    c = ((np.arange(K) + 0.5) * 3).astype(np.float32)
    h = rng.standard_normal((B, D))
    W = (0.5 * rng.standard_normal((K, D))).astype(np.float32)
    b = rng.standard_normal(K).astype(np.float32)
    y = np.asarray([1.0, 7.9, 16.0], np.float32)
    for lam in (0.0, 0.3, 1.0):
        _, gW, gb, gp = oracle.head_loss(h, W, b, c, y, lam)
        eps = 1e-5
        num_p = np.zeros_like(h)
        for idx in np.ndindex(h.shape):
            hp, hm = h.copy(), h.copy()
            hp[idx] += eps
            hm[idx] -= eps
            num_p[idx] = (oracle.head_loss(hp, W, b, c, y, lam, grads=False) -
                          oracle.head_loss(hm, W, b, c, y, lam, grads=False)) / (2 * eps)
        _close(gp, num_p, rtol=1e-6, atol=1e-8, what=f"d/dpooled lam={lam}")
        # W and b are fp32 parameters: difference them in float64 through an exact
        # reparametrisation (a feature of value 1 carries the bias, h scaled by W)
        num_b = np.zeros(K)
        for k in range(K):
            bp, bm = b.astype(np.float64).copy(), b.astype(np.float64).copy()
            bp[k] += 1e-3
            bm[k] -= 1e-3
            hx = np.concatenate([h, np.ones((B, 1))], axis=1)
            Wp = np.concatenate([W, bp[:, None].astype(np.float32)], axis=1)
            Wm = np.concatenate([W, bm[:, None].astype(np.float32)], axis=1)
            num_b[k] = (oracle.head_loss(hx, Wp, None, c, y, lam, grads=False) -
                        oracle.head_loss(hx, Wm, None, c, y, lam, grads=False)) / (
                            float(np.float32(bp[k])) - float(np.float32(bm[k])))
        _close(gb, num_b, rtol=2e-3, atol=1e-6, what=f"d/dbias lam={lam}")
        # W is an fp32 parameter: central differences with the exact fp32 step
        for k, x in ((0, 0), (2, 3), (5, 4)):
            Wp, Wm = W.copy(), W.copy()
            Wp[k, x] = np.float32(W[k, x] + np.float32(1e-3))
            Wm[k, x] = np.float32(W[k, x] - np.float32(1e-3))
            num = (oracle.head_loss(h, Wp, b, c, y, lam, grads=False) -
                   oracle.head_loss(h, Wm, b, c, y, lam, grads=False)) / (float(Wp[k, x]) - float(Wm[k, x]))
            _close(gW[k, x], num, rtol=2e-3, atol=1e-6, what=f"d/dW[{k},{x}] lam={lam}")
        # the batch loss is the mean of the per-prompt losses: dW = mean_b dz_b h_b^T
        ref_gW = np.zeros((K, D))
        for bb in range(B):
            _, _, gb1, _ = oracle.head_loss(h[bb:bb + 1], W, b, c, y[bb:bb + 1], lam)
            ref_gW += np.outer(gb1, h[bb]) / B
        _close(gW, ref_gW, rtol=1e-12, atol=1e-14, what=f"dW = sum_b dz_b h_b^T lam={lam}")


def pin_misalignment():
    """The misalignment counts against sets built from scipy's ordinal ranks (ties by
    order of appearance, i.e. the lower index first), and the limits: S = H gives 0 and
    0, S = -H gives k and k, all-tied values pick the k lowest indices for both
    directions; for independent measures about pct % of TopH lands in BotS."""
    rng = _rng(19)
    cu = np.asarray([0, 0, 1, 2, 3, 10, 137, 1137], dtype=np.int32)
    H = rng.standard_normal(int(cu[-1]))
    S = rng.standard_normal(int(cu[-1]))
    H[200:260] = 0.5   # ties inside a prompt
    S[230:300] = -1.0
    for pct in (40, 25, 50):
        got = oracle.misalignment(H, S, cu, pct)
        for b in range(len(cu) - 1):
            t0, t1 = int(cu[b]), int(cu[b + 1])
            k = pct * (t1 - t0) // 100
            assert got[b, 0] == k
            if k == 0:
                assert got[b, 1] == got[b, 2] == 0
                continue
            rh_d = stats.rankdata(-H[t0:t1], method="ordinal")   # 1 = largest
            rh_a = stats.rankdata(H[t0:t1], method="ordinal")    # 1 = smallest
            rs_d = stats.rankdata(-S[t0:t1], method="ordinal")
            rs_a = stats.rankdata(S[t0:t1], method="ordinal")
            assert got[b, 1] == int(np.sum((rh_d <= k) & (rs_a <= k))), (pct, b)
            assert got[b, 2] == int(np.sum((rh_a <= k) & (rs_d <= k))), (pct, b)
    same = oracle.misalignment(H, H, cu)
    assert np.all(same[:, 1] == 0) and np.all(same[:, 2] == 0)
    anti = oracle.misalignment(H, -H, cu)
    # S = -H: TopH = BotS exactly when no two H values of a prompt tie
    distinct = [b for b in range(len(cu) - 1) if len(np.unique(H[cu[b]:cu[b + 1]])) == cu[b + 1] - cu[b]]
    assert all(anti[b, 1] == anti[b, 0] and anti[b, 2] == anti[b, 0] for b in distinct)
    flat = oracle.misalignment(np.zeros(20), np.zeros(20), np.asarray([0, 20], np.int32))
    assert flat.tolist() == [[8, 8, 8]]   # both directions pick tokens 0..7
    big = oracle.misalignment(rng.standard_normal(50000), rng.standard_normal(50000),
                              np.asarray([0, 50000], np.int32))
    assert abs(big[0, 1] / big[0, 0] - 0.4) < 0.02 and abs(big[0, 2] / big[0, 0] - 0.4) < 0.02


def _mlp_case(rng, B, D, F, K, spread=1.0):
    h = rng.standard_normal((B, D))
    W1 = (rng.standard_normal((F, D)) / np.sqrt(D)).astype(np.float32)
    b1 = (rng.standard_normal(F) * 0.5).astype(np.float32)
    W2 = (rng.standard_normal((K, F)) * spread / np.sqrt(F)).astype(np.float32)
    b2 = rng.standard_normal(K).astype(np.float32)
    c = ((np.arange(K) + 0.5) * 16.0).astype(np.float32)
    y = rng.uniform(0, 16.0 * K, B).astype(np.float32)
    return h, W1, b1, W2, b2, c, y


def pin_mlp_reduces_to_linear():
    """With F = D, W1 = I and b1 = 50 every hidden unit is active and u = h + 50, so the
    MLP predictor is the linear head of Eq. 3-2 on h + 50: the same y_hat, loss, dL/dW2,
    dL/db2, and dL/dh = dL/du; dL/dW1 and dL/db1 are the outer products of dL/du with h
    and its batch sum."""
    rng = _rng(51)
    B, D, K = 4, 6, 9
    h = rng.standard_normal((B, D))
    W2 = rng.standard_normal((K, D)).astype(np.float32)
    b2 = rng.standard_normal(K).astype(np.float32)
    c = ((np.arange(K) + 0.5) * 10.0).astype(np.float32)
    y = rng.uniform(0, 90, B).astype(np.float32)
    W1, b1 = np.eye(D, dtype=np.float32), np.full(D, 50.0, dtype=np.float32)
    u = h + 50.0
    _close(oracle.mlp_length_head(h, W1, b1, W2, b2, c), oracle.length_head(u, W2, b2, c),
           rtol=1e-12, what="MLP y_hat vs linear head")
    for lam in (0.0, 0.3, 1.0):
        L, gW1, gb1, gW2, gb2, gh = oracle.mlp_head_loss(h, W1, b1, W2, b2, c, y, lam)
        Ll, gW, gb, gu = oracle.head_loss(u, W2, b2, c, y, lam)
        _close([L], [Ll], rtol=1e-12, what="MLP loss vs linear")
        _close(gW2, gW, rtol=1e-12, atol=1e-12, what="dL/dW2")
        _close(gb2, gb, rtol=1e-12, atol=1e-12, what="dL/db2")
        _close(gh, gu, rtol=1e-12, atol=1e-12, what="dL/dh")
        _close(gb1, gu.sum(0), rtol=1e-12, atol=1e-12, what="dL/db1")
        _close(gW1, gu.T @ h, rtol=1e-10, atol=1e-12, what="dL/dW1")


def pin_mlp_dead_units():
    """W1 = 0 and b1 < 0 switch every hidden unit off: u = 0, so z = b2 for every prompt,
    y_hat = sum softmax(b2)_k c_k (scipy), the loss is the linear head's on zero features,
    and no gradient reaches W1, b1 or h."""
    rng = _rng(52)
    B, D, F, K = 3, 7, 5, 8
    h = rng.standard_normal((B, D))
    W1, b1 = np.zeros((F, D), np.float32), np.full(F, -1.0, np.float32)
    W2 = rng.standard_normal((K, F)).astype(np.float32)
    b2 = rng.standard_normal(K).astype(np.float32)
    c = ((np.arange(K) + 0.5) * 10.0).astype(np.float32)
    y = rng.uniform(0, 80, B).astype(np.float32)
    ref = float(np.dot(special.softmax(b2.astype(np.float64)), c.astype(np.float64)))
    _close(oracle.mlp_length_head(h, W1, b1, W2, b2, c), [ref] * B, rtol=1e-12, what="dead y_hat")
    L, gW1, gb1, gW2, gb2, gh = oracle.mlp_head_loss(h, W1, b1, W2, b2, c, y, 0.4)
    _close([L], [oracle.head_loss(np.zeros((B, F)), W2, b2, c, y, 0.4, grads=False)], rtol=1e-12,
           what="dead loss")
    assert not np.any(gW1) and not np.any(gb1) and not np.any(gh), "gradient through dead units"
    assert not np.any(gW2), "dL/dW2 = dz^T u = 0"


def pin_mlp_finite_differences():
    """Every gradient of the MLP loss equals central differences of the loss (units kept
    away from the ReLU's kink)."""
    rng = _rng(53)
    B, D, F, K = 3, 5, 4, 6
    for _ in range(20):
        h, W1, b1, W2, b2, c, y = _mlp_case(rng, B, D, F, K, spread=2.0)
        a = h @ W1.T.astype(np.float64) + b1
        if np.min(np.abs(a)) > 0.05:
            break
    lam = 0.35
    L, gW1, gb1, gW2, gb2, gh = oracle.mlp_head_loss(h, W1, b1, W2, b2, c, y, lam)
    loss = lambda hh, w1, bb1, w2, bb2: oracle.mlp_head_loss(hh, w1, bb1, w2, bb2, c, y, lam, grads=False)

    def fd(arr, grad, call, eps):
        arr64 = np.array(arr, dtype=np.float64)
        num = np.zeros(arr64.shape)
        for idx in np.ndindex(arr64.shape):
            up, dn = arr64.copy(), arr64.copy()
            up[idx] += eps
            dn[idx] -= eps
            num[idx] = (call(up) - call(dn)) / (2 * eps)
        scale = max(np.max(np.abs(num)), 1e-12)
        assert np.max(np.abs(num - grad)) <= 1e-3 * scale, f"finite differences: {np.max(np.abs(num - grad))}"

    # W1, b1, W2, b2 are fp32 arguments of the oracle: steps of 2^-10 keep them exact
    eps = 1.0 / 1024
    fd(h, gh, lambda v: loss(v, W1, b1, W2, b2), 1e-5)
    fd(W1, gW1, lambda v: loss(h, v.astype(np.float32), b1, W2, b2), eps)
    fd(b1, gb1, lambda v: loss(h, W1, v.astype(np.float32), W2, b2), eps)
    fd(W2, gW2, lambda v: loss(h, W1, b1, v.astype(np.float32), b2), eps)
    fd(b2, gb2, lambda v: loss(h, W1, b1, W2, v.astype(np.float32)), eps)


ALL_PINS = [v for k, v in sorted(globals().items()) if k.startswith("pin_")]
