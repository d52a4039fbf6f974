"""Pins of the fp64 oracle to facts fixed by the paper and by mathematics.

Each ``pin_*`` function runs one check against an oracle build (``lib=None``
is the real oracle) and raises AssertionError when the oracle disagrees.
They are collected by test_oracle_pins.py (the real oracle must pass all of
them) and test_oracle_mutants.py (every deliberately broken build must fail at
least one of them).

What pins what:
  * Eq. 1 + causal mask      -> torch float64 scaled_dot_product_attention
                                (gamma = 1, and window >= N where A* = A).
  * sink + window set W(i)   -> closed-form counts |W(i)| and mean key index
                                under uniform scores (Q = 0).
  * Eq. 6 / Alg. 1 Delta     -> closed forms with K = 0 (prefix / window means),
                                window = 1 (S_i = v_i), constant V, and the
                                sampled-row identity A^V_{k gamma} = ~AV_k.
  * GQA head mapping         -> explicit repetition of the KV heads.
  * Lemma 1                  -> the appendix inequality on every sample,
                                and both of its sides in closed form under
                                uniform scores (Q = 0).
  * whole-matrix restatement -> the numpy brute force (oracle/brute.py).
  * Eq. 2 decoding           -> the dense causal row at the token's position
                                and torch scaled_dot_product_attention.
  * RoPE                     -> identity at position 0, the unit-vector closed
                                form, pair norms, relative-position scores.
  * Delta smoothing          -> reductions to Eq. 6 (EMA beta = 1, filter
    (appendix Interpolation,    (1, 0, 0), linear at gamma = 1), fixed points
     Alg. 2)                    of a constant Delta, the EMA step response,
                                exactness of linear interpolation on affine
                                Delta sequences, the filter's transfer function
                                (impulse response summed against w^k) and its
                                steady-state lag 6 (alpha - 1) / gamma on a
                                cubic input (final-value theorem).
"""
import numpy as np
import torch

import oracle
from oracle import brute

TOL = 1e-12


def rand_bits(seed, shape, scale=1.0):
    g = torch.Generator().manual_seed(seed)
    x = (torch.randn(shape, generator=g, dtype=torch.float32) * scale).to(torch.bfloat16)
    return x.view(torch.int16).numpy().view(np.uint16)


def const_bits(shape, value):
    x = torch.full(shape, value, dtype=torch.float32).to(torch.bfloat16)
    return x.view(torch.int16).numpy().view(np.uint16)


def f64(bits):
    return oracle.bf16_bits_to_f64(bits)


def _sdpa_causal(Qb, Kb, Vb):
    Q, K, V = (torch.from_numpy(f64(x)) for x in (Qb, Kb, Vb))
    G = Q.shape[1] // K.shape[1]
    K = K.repeat_interleave(G, dim=1)
    V = V.repeat_interleave(G, dim=1)
    return torch.nn.functional.scaled_dot_product_attention(Q, K, V, is_causal=True).numpy()


def _w_count(i, n_sink, window):
    """Closed form |W(i)|: the band of min(i+1, window) keys ending at i plus
    the sinks that lie before the band."""
    band_start = max(0, i - window + 1)
    return min(i + 1, window) + min(n_sink, band_start)


def _w_index_sum(i, n_sink, window):
    """Closed form sum of the key indices in W(i) (arithmetic series)."""
    a = max(0, i - window + 1)
    band = (a + i) * (i - a + 1) // 2
    s = min(n_sink, a)
    return band + s * (s - 1) // 2


# --------------------------------------------------------------------------
def pin_gamma1_is_sdpa(lib=None):
    """gamma = 1: every row is sampled, Eq. 6 gives dense causal attention."""
    for (B, Hq, Hkv, N, d, s, w) in [(1, 2, 2, 45, 16, 2, 7), (2, 4, 2, 33, 8, 0, 3)]:
        Q, K, V = rand_bits(1, (B, Hq, N, d)), rand_bits(2, (B, Hkv, N, d)), rand_bits(3, (B, Hkv, N, d))
        A = oracle.delta_attn(Q, K, V, s, w, 1, lib=lib)["A"]
        ref = _sdpa_causal(Q, K, V)
        assert np.abs(A - ref).max() <= TOL, "gamma=1 must equal dense causal attention"


def pin_full_window_is_sdpa(lib=None):
    """window >= N: W(i) = C(i), so A* = A and the output is dense attention."""
    B, Hq, Hkv, N, d = 1, 4, 2, 40, 16
    Q, K, V = rand_bits(4, (B, Hq, N, d), 2.0), rand_bits(5, (B, Hkv, N, d), 2.0), rand_bits(6, (B, Hkv, N, d))
    for s, w, gamma in [(0, N, 8), (3, N + 5, 5), (1, N, 64)]:
        out = oracle.delta_attn(Q, K, V, s, w, gamma, lib=lib)
        ref = _sdpa_causal(Q, K, V)
        assert np.abs(out["A"] - ref).max() <= TOL
        assert np.abs(out["S"] - ref).max() <= TOL, "A*V must be dense when window >= N"


def pin_zero_keys_closed_form(lib=None):
    """K = 0: every score is 0, softmax is uniform over the key set, so
    D_i = mean_{j<=i} v_j and S_i = mean_{j in W(i)} v_j (no exponentials)."""
    B, Hq, Hkv, N, d = 1, 2, 1, 50, 8
    Q = rand_bits(7, (B, Hq, N, d))
    K = np.zeros((B, Hkv, N, d), np.uint16)
    V = rand_bits(8, (B, Hkv, N, d))
    Vf = f64(V)[0, 0]
    pre = np.concatenate([np.zeros((1, d)), np.cumsum(Vf, axis=0)])
    for s, w, gamma in [(2, 6, 4), (0, 1, 3), (5, 13, 7), (1, 3, 16)]:
        out = oracle.delta_attn(Q, K, V, s, w, gamma, lib=lib)
        for h in range(Hq):
            for i in range(N):
                a = max(0, i - w + 1)
                cnt = (i - a + 1) + min(s, a)
                S_i = (pre[i + 1] - pre[a] + pre[min(s, a)]) / cnt
                assert np.abs(out["S"][0, h, i] - S_i).max() <= TOL
                ks = (i // gamma) * gamma
                aks = max(0, ks - w + 1)
                S_k = (pre[ks + 1] - pre[aks] + pre[min(s, aks)]) / ((ks - aks + 1) + min(s, aks))
                D_k = pre[ks + 1] / (ks + 1)
                assert np.abs(out["A"][0, h, i] - (S_i + D_k - S_k)).max() <= TOL


def pin_window1_no_sink(lib=None):
    """window = 1, n_sink = 0: S_i = v_i, so A^V_i = v_i + D_{k gamma} - v_{k gamma}."""
    B, Hq, Hkv, N, d = 1, 2, 2, 37, 16
    Q, K, V = rand_bits(9, (B, Hq, N, d)), rand_bits(10, (B, Hkv, N, d)), rand_bits(11, (B, Hkv, N, d))
    gamma = 6
    out = oracle.delta_attn(Q, K, V, 0, 1, gamma, lib=lib)
    dense = _sdpa_causal(Q, K, V)
    Vf = f64(V)
    for h in range(Hq):
        assert np.abs(out["S"][0, h] - Vf[0, h]).max() <= TOL
        for i in range(N):
            ks = (i // gamma) * gamma
            want = Vf[0, h, i] + dense[0, h, ks] - Vf[0, h, ks]
            assert np.abs(out["A"][0, h, i] - want).max() <= TOL


def pin_constant_values(lib=None):
    """v_j = c for all j: every softmax average is c, Delta = 0."""
    B, Hq, Hkv, N, d = 1, 2, 2, 30, 8
    Q, K = rand_bits(12, (B, Hq, N, d), 3.0), rand_bits(13, (B, Hkv, N, d), 3.0)
    V = const_bits((B, Hkv, N, d), 0.375)
    out = oracle.delta_attn(Q, K, V, 2, 5, 4, lib=lib)
    assert np.abs(out["A"] - 0.375).max() <= TOL


def pin_mask_structure(lib=None):
    """Q = 0 gives uniform weights over the key set.  With v_j[0] = 1,
    v_j[1] = [j < n_sink], v_j[2] = j / 64 the sparse output exposes the set:
    S_i[1] = (#sinks in W(i)) / |W(i)|, S_i[2] = mean index / 64."""
    N, d = 64, 8
    Q = np.zeros((1, 1, N, d), np.uint16)
    K = rand_bits(14, (1, 1, N, d))
    for s, w in [(4, 8), (0, 5), (3, 1), (10, 6), (2, 64)]:
        Vf = np.zeros((1, 1, N, d), np.float32)
        Vf[0, 0, :, 0] = 1.0
        Vf[0, 0, :, 1] = (np.arange(N) < s)
        Vf[0, 0, :, 2] = np.arange(N) / 64.0
        V = torch.from_numpy(Vf).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
        out = oracle.delta_attn(Q, K, V, s, w, 4, lib=lib)
        for i in range(N):
            cnt = _w_count(i, s, w)
            sinks_in = min(s, i + 1)
            S = out["S"][0, 0, i]
            assert abs(S[0] - 1.0) <= TOL
            assert abs(S[1] - sinks_in / cnt) <= TOL, (i, s, w)
            assert abs(S[2] - _w_index_sum(i, s, w) / 64.0 / cnt) <= TOL, (i, s, w)


def pin_sampled_rows_are_dense(lib=None):
    """Eq. 6 at i = k gamma: A^V = A*V + ~AV - A*V = the dense row; and row 0
    attends to itself only, so A^V_0 = v_0."""
    B, Hq, Hkv, N, d = 1, 4, 2, 53, 16
    Q, K, V = rand_bits(15, (B, Hq, N, d)), rand_bits(16, (B, Hkv, N, d)), rand_bits(17, (B, Hkv, N, d))
    gamma = 8
    out = oracle.delta_attn(Q, K, V, 2, 9, gamma, lib=lib)
    dense = _sdpa_causal(Q, K, V)
    assert np.abs(out["A"][:, :, ::gamma] - dense[:, :, ::gamma]).max() <= TOL
    Vf = f64(V)
    for h in range(Hq):
        assert np.abs(out["A"][0, h, 0] - Vf[0, h // 2, 0]).max() <= TOL
    assert out["max_dev"] <= TOL, "softmax rows must sum to 1"


def pin_gqa_repeat(lib=None):
    """GQA: Hkv = 2 with Hq = 4 equals Hkv = 4 with each KV head repeated."""
    B, Hq, Hkv, N, d = 2, 4, 2, 41, 16
    Q, K, V = rand_bits(18, (B, Hq, N, d)), rand_bits(19, (B, Hkv, N, d)), rand_bits(20, (B, Hkv, N, d))
    a = oracle.delta_attn(Q, K, V, 3, 7, 5, lib=lib)["A"]
    Kr = np.ascontiguousarray(np.repeat(K, 2, axis=1))
    Vr = np.ascontiguousarray(np.repeat(V, 2, axis=1))
    b = oracle.delta_attn(Q, Kr, Vr, 3, 7, 5, lib=lib)["A"]
    assert np.abs(a - b).max() <= TOL


def pin_lemma1(lib=None):
    """Appendix, Lemma 1: |Delta - sum_{omitted} a_j v_j| <= H/(H+T) max_W |v_j|,
    on every sample of a problem with scaled sinks."""
    B, Hq, Hkv, N, d = 1, 2, 1, 96, 16
    Q, K, V = rand_bits(21, (B, Hq, N, d), 1.5), rand_bits(22, (B, Hkv, N, d), 1.5), rand_bits(23, (B, Hkv, N, d))
    nontrivial = 0
    for h in range(Hq):
        for k in range(0, N // 8):
            lhs, rhs, frac = oracle.lemma1(Q, K, V, 2, 16, 8, 0, h, k, lib=lib)
            assert np.all(lhs <= rhs * (1 + 1e-9) + TOL), (h, k)
            nontrivial += frac > 0.05
    assert nontrivial > 0


def pin_lemma1_uniform(lib=None):
    """Lemma 1's terms in closed form.  With Q = 0 every score is 0, so over
    the causal set C(i) (i + 1 keys) and the sparse set W(i): H = |C \\ W|,
    T = |W|, H/(H+T) = 1 - |W|/(i+1); Delta minus the omitted-key term is
    mean_W(v) (|W|/(i+1) - 1), so lhs = H/(H+T) |mean_W(v)|, and
    rhs = H/(H+T) max_W |v|.  V carries large values on keys outside W(i), so
    a maximum taken over any other set than W(i) shows."""
    B, Hq, Hkv, N, d = 1, 2, 1, 80, 8
    n_sink, window, gamma = 2, 9, 8
    Q = const_bits((B, Hq, N, d), 0.0)
    K = rand_bits(24, (B, Hkv, N, d))
    v = f64(rand_bits(25, (B, Hkv, N, d)))
    v[0, 0, n_sink:N - window] *= 16.0   # keys omitted by every late row
    V = torch.from_numpy(v.astype(np.float32)).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    vv = f64(V)[0, 0]
    checked = 0
    for h in range(Hq):
        for k in range(N // gamma):
            i = k * gamma
            j = np.arange(i + 1)
            w_set = (j < n_sink) | (j > i - window)
            frac = 1.0 - w_set.sum() / (i + 1.0)
            lhs, rhs, f = oracle.lemma1(Q, K, V, n_sink, window, gamma, 0, h, k, lib=lib)
            assert abs(f - frac) <= TOL, (h, k, f, frac)
            assert np.abs(lhs - frac * np.abs(vv[j[w_set]].mean(axis=0))).max() <= TOL, (h, k)
            assert np.abs(rhs - frac * np.abs(vv[j[w_set]]).max(axis=0)).max() <= TOL, (h, k)
            checked += frac > 0
    assert checked > 0


def pin_lemma1_brute(lib=None):
    """Lemma 1's terms equal the whole-matrix restatement (oracle/brute.py)
    on random inputs with scaled sinks."""
    B, Hq, Hkv, N, d = 2, 4, 2, 70, 16
    Q, K, V = rand_bits(26, (B, Hq, N, d), 1.5), rand_bits(27, (B, Hkv, N, d), 1.5), rand_bits(28, (B, Hkv, N, d))
    K[:, :, :3] = rand_bits(29, (B, Hkv, 3, d), 8.0)
    Qf, Kf, Vf = f64(Q), f64(K), f64(V)
    for (n_sink, window, gamma) in ((3, 10, 7), (0, 1, 5), (4, 64, 16)):
        for b in range(B):
            for h in range(Hq):
                for k in range((N + gamma - 1) // gamma):
                    lhs, rhs, f = oracle.lemma1(Q, K, V, n_sink, window, gamma, b, h, k, lib=lib)
                    bl, br, bf = brute.lemma1_terms(Qf, Kf, Vf, n_sink, window, gamma, b, h, k)
                    assert abs(f - bf) <= TOL and np.abs(lhs - bl).max() <= TOL and np.abs(rhs - br).max() <= TOL, \
                        (n_sink, window, gamma, b, h, k)


def pin_brute_force(lib=None):
    """The direct per-row evaluation equals the whole-matrix restatement of
    Alg. 1 (numpy) on small problems, over a sweep of gamma, window, sinks,
    GQA ratio, both output modes and the dense tail."""
    cases = []
    for gamma in (1, 2, 3, 5, 16, 64):
        for window in (1, 2, 7, 64):
            for n_sink in (0, 1, 4):
                cases.append((gamma, window, n_sink))
    seed = 100
    for idx, (gamma, window, n_sink) in enumerate(cases):
        G = (1, 2, 4)[idx % 3]
        Hkv = 1 + (idx % 2)
        Hq = Hkv * G
        N = (64, 37, 50)[idx % 3]
        d = 8
        seed += 1
        Q, K, V = rand_bits(seed, (1, Hq, N, d), 1.5), rand_bits(seed + 1000, (1, Hkv, N, d), 1.5), \
            rand_bits(seed + 2000, (1, Hkv, N, d))
        mode = "recompute" if idx % 7 == 3 else "delta"
        tail = 5 if idx % 11 == 4 else 0
        A_b, S_b, _ = brute.delta_attn(f64(Q), f64(K), f64(V), n_sink, window, gamma, mode=mode, tail_dense=tail)
        out = oracle.delta_attn(Q, K, V, n_sink, window, gamma, mode=mode, tail_dense=tail, lib=lib)
        assert np.abs(out["A"] - A_b).max() <= TOL, (gamma, window, n_sink, mode, tail)
        assert np.abs(out["S"] - S_b).max() <= TOL


def pin_rows_agree(lib=None):
    """oracle_rows (per-row) agrees with the box evaluation."""
    B, Hq, Hkv, N, d = 2, 4, 2, 70, 16
    Q, K, V = rand_bits(30, (B, Hq, N, d)), rand_bits(31, (B, Hkv, N, d)), rand_bits(32, (B, Hkv, N, d))
    full = oracle.delta_attn(Q, K, V, 3, 11, 9, lib=lib)
    rng = np.random.default_rng(0)
    bhi = np.stack([rng.integers(0, B, 40), rng.integers(0, Hq, 40), rng.integers(0, N, 40)], 1)
    r = oracle.rows(Q, K, V, 3, 11, 9, bhi, lib=lib)
    for t, (b, h, i) in enumerate(bhi):
        assert np.abs(r["A"][t] - full["A"][b, h, i]).max() <= TOL
        assert np.abs(r["S"][t] - full["S"][b, h, i]).max() <= TOL
        assert np.abs(r["D_sample"][t] - full["D"][b, h, i // 9]).max() <= TOL


def pin_smooth_reductions(lib=None):
    """Smoothing forms that reduce to plain Eq. 6 or to each other: EMA with
    beta = 1 and the filter with (1, 0, 0) give the repeated Delta; at gamma = 1
    linear interpolation gives Delta itself and the filter with (alpha, 0, 0)
    is the EMA with beta = alpha; a constant Delta is a fixed point of every
    form; the box evaluation with smoothing "none" is the Eq. 6 box."""
    rng = np.random.default_rng(7)
    n_s, g, N, d = 9, 5, 43, 4
    delta = rng.standard_normal((n_s, d))
    plain = np.repeat(delta, g, axis=0)[:N]
    for kind, par in (("ema", (1.0,)), ("abg", (1.0, 0.0, 0.0)), ("none", ())):
        assert np.abs(oracle.smooth_seq(kind, par, delta, n_s, g, (0, N), lib=lib) - plain).max() <= TOL, kind
    assert np.abs(oracle.smooth_seq("linear", (), delta, n_s, 1, (0, n_s), lib=lib) - delta).max() <= TOL
    a = oracle.smooth_seq("abg", (0.3, 0.0, 0.0), delta, n_s, 1, (0, n_s), lib=lib)
    b = oracle.smooth_seq("ema", (0.3,), delta, n_s, 1, (0, n_s), lib=lib)
    assert np.abs(a - b).max() <= TOL
    const = np.tile(rng.standard_normal((1, d)), (n_s, 1))
    for kind, par in (("linear", ()), ("ema", (0.37,)), ("abg", (0.2, 0.05, 0.0035)), ("abg", (0.5, 0.4, 0.1))):
        out = oracle.smooth_seq(kind, par, const, n_s, g, (3, N), lib=lib)
        assert np.abs(out - const[0]).max() <= 1e-12, kind
    Q, K, V = rand_bits(40, (1, 2, 45, 8)), rand_bits(41, (1, 1, 45, 8)), rand_bits(42, (1, 1, 45, 8))
    ref = oracle.delta_attn(Q, K, V, 2, 6, 4, lib=lib)["A"]
    got = oracle.delta_attn(Q, K, V, 2, 6, 4, smooth="ema", smooth_params=(1.0,), lib=lib)["A"]
    assert np.abs(got - ref).max() <= TOL


def _abg_transfer(al, be, ga, w):
    """Transfer function from the filter input to its position output at
    z^-1 = w, from the state-space form of Alg. 2 (x_k = M x_{k-1} + g y_k):
    (2a + (2b + c - 4a) w + (2a - 2b + c) w^2) /
    (2 + (2a + 2b + c - 6) w + (6 - 4a - 2b + c) w^2 + (2a - 2) w^3)."""
    num = 2 * al + (2 * be + ga - 4 * al) * w + (2 * al - 2 * be + ga) * w ** 2
    den = 2 + (2 * al + 2 * be + ga - 6) * w + (6 - 4 * al - 2 * be + ga) * w ** 2 + (2 * al - 2) * w ** 3
    return num / den


def pin_smooth_closed_forms(lib=None):
    """EMA step response 1 - (1 - beta)^(i - gamma + 1); linear interpolation
    exact on an affine Delta sequence (held after the last sample); the
    filter's impulse response summed against w^k equals w H(w); the filter
    tracks a cubic with the constant lag 6 (alpha - 1) / gamma."""
    g, n_s, beta = 4, 10, 0.3
    step = np.zeros((n_s, 1))
    step[1:] = 1.0
    e = oracle.smooth_seq("ema", (beta,), step, n_s, g, (0, n_s * g), lib=lib)[:, 0]
    i = np.arange(n_s * g)
    want = np.where(i < g, 0.0, 1.0 - (1.0 - beta) ** np.maximum(i - g + 1, 0))
    assert np.abs(e - want).max() <= TOL
    aff = (0.25 + 0.5 * np.arange(n_s))[:, None] * np.array([[1.0, -2.0]])
    lin = oracle.smooth_seq("linear", (), aff, n_s, g, (0, n_s * g), lib=lib)
    want = (0.25 + 0.5 * np.minimum(i / g, n_s - 1))[:, None] * np.array([[1.0, -2.0]])
    assert np.abs(lin - want).max() <= TOL
    for (al, be, ga) in ((0.2, 0.05, 0.0035), (0.5, 0.4, 0.1), (0.1, 5e-3, 1.66e-4)):
        n = 400
        imp = np.zeros((n, 1))
        imp[1] = 1.0
        o = oracle.smooth_seq("abg", (al, be, ga), imp, n, 1, (0, n), lib=lib)[:, 0]
        w = 0.5
        assert abs(np.sum(o * w ** np.arange(n)) - w * _abg_transfer(al, be, ga, w)) <= 1e-12, (al, be, ga)
    al, be, ga = 0.2, 0.05, 0.0035
    n = 3000
    cubic = (np.arange(n, dtype=np.float64) ** 3 * 1e-6)[:, None]
    o = oracle.smooth_seq("abg", (al, be, ga), cubic, n, 1, (0, n), lib=lib)[:, 0]
    lag = o[-1] - cubic[-1, 0]
    assert abs(lag - 6e-6 * (al - 1) / ga) <= 1e-6 * abs(lag), lag


def pin_smooth_brute(lib=None):
    """The smoothed prefill (direct per-row evaluation) equals the whole-matrix
    numpy restatement with its own smoothing forms, over gamma, window, GQA,
    the three forms and the dense tail."""
    seed = 500
    for idx, (gamma, window, kind, par) in enumerate((
            (4, 7, "linear", ()), (3, 16, "ema", (0.5,)), (5, 2, "abg", (0.2, 0.05, 0.0035)),
            (1, 5, "ema", (0.75,)), (16, 9, "linear", ()), (7, 64, "abg", (0.1, 5e-3, 1.66e-4)))):
        seed += 3
        Hkv, G = 1 + idx % 2, (1, 2, 4)[idx % 3]
        N, d = (61, 40, 53)[idx % 3], 8
        Q, K, V = rand_bits(seed, (1, Hkv * G, N, d), 1.5), rand_bits(seed + 1, (1, Hkv, N, d), 1.5), \
            rand_bits(seed + 2, (1, Hkv, N, d))
        tail = 6 if idx % 2 else 0
        A_b, _, _ = brute.delta_attn(f64(Q), f64(K), f64(V), 2, window, gamma, tail_dense=tail, smooth_kind=kind,
                                     smooth_params=par)
        got = oracle.delta_attn(Q, K, V, 2, window, gamma, tail_dense=tail, smooth=kind, smooth_params=par,
                                lib=lib)["A"]
        assert np.abs(got - A_b).max() <= TOL, (gamma, window, kind)
        r0 = N // 3
        part = oracle.delta_attn(Q, K, V, 2, window, gamma, rows=(r0, N), tail_dense=tail, smooth=kind,
                                 smooth_params=par, lib=lib)["A"]
        assert np.abs(part - A_b[:, :, r0:]).max() <= TOL


def pin_decode(lib=None):
    """Eq. 2 decoding of the token at position i over keys 0..i equals the
    dense causal row i (Eq. 1, gamma = 1) and torch's scaled_dot_product_attention
    of that single query over the same keys; a cache longer than n_keys is
    ignored past n_keys."""
    B, Hq, Hkv, N, d = 2, 4, 2, 50, 16
    Q, K, V = rand_bits(60, (B, Hq, N, d)), rand_bits(61, (B, Hkv, N, d)), rand_bits(62, (B, Hkv, N, d))
    dense = oracle.delta_attn(Q, K, V, 0, 1, 1, lib=lib)["A"]
    for pos in ((0, 0), (7, 49), (31, 12)):
        q = np.ascontiguousarray(np.stack([Q[b, :, pos[b]] for b in range(B)]))
        out, dev = oracle.decode(q, K, V, [pos[0] + 1, pos[1] + 1], lib=lib)
        assert dev <= 1e-12
        for b in range(B):
            assert np.abs(out[b] - dense[b, :, pos[b]]).max() <= TOL, pos
            n = pos[b] + 1
            Qt = torch.from_numpy(f64(q[b]))[None, :, None, :]
            Kt = torch.from_numpy(f64(K[b, :, :n])).repeat_interleave(Hq // Hkv, dim=0)[None]
            Vt = torch.from_numpy(f64(V[b, :, :n])).repeat_interleave(Hq // Hkv, dim=0)[None]
            ref = torch.nn.functional.scaled_dot_product_attention(Qt, Kt, Vt).numpy()[0, :, 0]
            assert np.abs(out[b] - ref).max() <= TOL


def pin_rope(lib=None):
    """RoPE: position 0 is the identity; a unit vector on channel c rotates into
    (cos a, sin a) on channels (c, c + d/2) with a = pos base^(-2c/d) (the
    pairing and the sign); each pair keeps its norm; and the score of two
    rotated vectors depends only on the difference of their positions."""
    d, base = 16, 10000.0
    X = rand_bits(70, (1, 1, 5, d))
    assert np.array_equal(oracle.rope(X[:, :, :1], base, 0, lib=lib), X[:, :, :1])
    for c in (0, 3, 7):
        for pos in (1, 5, 123):
            e = np.zeros((1, 1, 1, d), np.float32)
            e[..., c] = 1.0
            eb = torch.from_numpy(e).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
            r = oracle.rope(eb, base, pos, rounded=False, lib=lib)[0, 0, 0]
            a = pos * base ** (-2.0 * c / d)
            want = np.zeros(d)
            want[c], want[c + d // 2] = np.cos(a), np.sin(a)
            assert np.abs(r - want).max() <= 1e-12, (c, pos)
    r = oracle.rope(X, base, 37, rounded=False, lib=lib)[0, 0]
    x = f64(X)[0, 0]
    assert np.abs(r[:, :d // 2] ** 2 + r[:, d // 2:] ** 2 - x[:, :d // 2] ** 2 - x[:, d // 2:] ** 2).max() <= 1e-12
    q, k = rand_bits(71, (1, 1, 1, d)), rand_bits(72, (1, 1, 1, d))
    for (m, n) in ((10, 3), (1000, 993), (50007, 50000)):
        s = np.dot(oracle.rope(q, base, m, rounded=False, lib=lib).ravel(),
                   oracle.rope(k, base, n, rounded=False, lib=lib).ravel())
        s0 = np.dot(oracle.rope(q, base, 7, rounded=False, lib=lib).ravel(),
                    oracle.rope(k, base, 0, rounded=False, lib=lib).ravel())
        assert abs(s - s0) <= 1e-9, (m, n)
    rb = oracle.rope(X, base, 37, lib=lib)
    rt = torch.from_numpy(r.astype(np.float32)).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.abs(f64(rb)[0, 0] - f64(rt)).max() <= 2.0 ** -7 * np.abs(r).max()


ALL_PINS = [pin_gamma1_is_sdpa, pin_full_window_is_sdpa, pin_zero_keys_closed_form,
            pin_window1_no_sink, pin_constant_values, pin_mask_structure,
            pin_sampled_rows_are_dense, pin_gqa_repeat, pin_lemma1, pin_lemma1_uniform, pin_rows_agree,
            pin_smooth_reductions, pin_smooth_closed_forms, pin_decode, pin_rope]
# The brute-force restatements are listed separately: the mutant test shows the
# other pins catch every planted mistake without them.
BRUTE_PINS = [pin_brute_force, pin_smooth_brute, pin_lemma1_brute]
