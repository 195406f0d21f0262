"""Scalar-loop restatement of the compactor forward, for tiny inputs (test infrastructure only).

TEST INFRASTRUCTURE: imported only by tests. It recomputes the per-layer compactor of
Sec. 2.1 / App. A with explicit Python loops over every index and the `math` module, without
NumPy broadcasting or library matrix products, so that an axis, transpose or broadcasting
mistake in oracle/still_oracle.py shows up as a disagreement. Intended sizes: N <= 64,
t <= 8, d <= 8, d_l <= 16. Same readings as the vectorised oracle (see its header).
"""
from __future__ import annotations

import math


def _matvec_row(x, W, col0, ncols):
    """y[j] = sum_k x[k] * W[k][col0 + j] for j < ncols (x @ W restricted to a column block)."""
    return [sum(x[k] * W[k][col0 + j] for k in range(len(x))) for j in range(ncols)]


def _rot_pairs(vec, p, base, sign):
    w = len(vec)
    h = w // 2
    out = [0.0] * w
    for m in range(h):
        a = sign * p * base ** (-2.0 * m / w)
        c, s = math.cos(a), math.sin(a)
        out[m] = vec[m] * c - vec[m + h] * s
        out[m + h] = vec[m] * s + vec[m + h] * c
    return out


def _rms(vec, eps):
    ms = sum(v * v for v in vec) / len(vec)
    return [v / math.sqrt(ms + eps) for v in vec]


def _l2(vec, eps):
    nrm = math.sqrt(sum(v * v for v in vec))
    return [v / max(nrm, eps) for v in vec]


def _softmax(row):
    mx = max(row)
    e = [math.exp(v - mx) for v in row]
    s = sum(e)
    return [v / s for v in e]


def _gelu(x):
    return 0.5 * x * (1.0 + math.erf(x / math.sqrt(2.0)))


def _attend(Qrows, Krows, Vrows, scale):
    out = []
    for q in Qrows:
        logits = [scale * sum(q[m] * k[m] for m in range(len(q))) for k in Krows]
        a = _softmax(logits)
        out.append([sum(a[n] * Vrows[n][f] for n in range(len(Krows)))
                    for f in range(len(Vrows[0]))])
    return out


def _w(W, name, b):
    return W[name if b == 0 else f"{name}@{b}"]


def compact_head_brute(Kh, Vh, Zh, W, cfg, kpos):
    """Lists-of-lists version of one KV-head's compaction. Returns (C_k, C_v) as lists."""
    D, d, t, N = cfg.D, cfg.d, len(Zh), len(Kh)
    pmin, pmax = min(kpos), max(kpos)
    qpos = [pmin + (pmax - pmin) * j / (t - 1) if t > 1 else pmin for j in range(t)]
    X = []
    for n in range(N):
        kx = _rot_pairs(list(Kh[n]), kpos[n], cfg.theta, -1.0) if cfg.rope_fix else list(Kh[n])
        X.append(kx + list(Vh[n]))
    Z = [list(r) for r in Zh]
    for b in range(cfg.n_blocks):
        if b == 0 or cfg.cross_every_block:
            Zn = [_rms(r, cfg.rms_eps) for r in Z]
            Wq, bq, Wk, bk = _w(W, "Wq", b), _w(W, "bq", b), _w(W, "Wk", b), _w(W, "bk", b)
            Wv, Wo = _w(W, "Wv", b), _w(W, "Wo", b)
            cat = [[] for _ in range(t)]
            for i in range(cfg.n_c):
                q = []
                for j in range(t):
                    v = _matvec_row(Zn[j], Wq, i * D, D)
                    v = _l2([v[m] + bq[i * D + m] for m in range(D)], cfg.l2_eps)
                    q.append(_rot_pairs(v, qpos[j], cfg.theta_c, 1.0) if cfg.compactor_rope else v)
                k, vv = [], []
                for n in range(N):
                    v = _matvec_row(X[n], Wk, i * D, D)
                    v = _l2([v[m] + bk[i * D + m] for m in range(D)], cfg.l2_eps)
                    k.append(_rot_pairs(v, kpos[n], cfg.theta_c, 1.0) if cfg.compactor_rope else v)
                    vv.append(_matvec_row(X[n], Wv, i * D, D))
                head = _attend(q, k, vv, cfg.scale)
                for j in range(t):
                    cat[j] += head[j]
            for j in range(t):
                upd = _matvec_row(cat[j], Wo, 0, D)
                Z[j] = [Z[j][f] + upd[f] for f in range(D)]
        if cfg.self_attn:
            Zn = [_rms(r, cfg.rms_eps) for r in Z]
            Sq, sbq, Sk, sbk = _w(W, "Sq", b), _w(W, "sbq", b), _w(W, "Sk", b), _w(W, "sbk", b)
            Sv, So = _w(W, "Sv", b), _w(W, "So", b)
            cat = [[] for _ in range(t)]
            for i in range(cfg.n_s):
                q = [_l2([a + c for a, c in zip(_matvec_row(Zn[j], Sq, i * D, D),
                                                sbq[i * D:(i + 1) * D])], cfg.l2_eps)
                     for j in range(t)]
                k = [_l2([a + c for a, c in zip(_matvec_row(Zn[j], Sk, i * D, D),
                                                sbk[i * D:(i + 1) * D])], cfg.l2_eps)
                     for j in range(t)]
                v = [_matvec_row(Zn[j], Sv, i * D, D) for j in range(t)]
                head = _attend(q, k, v, cfg.scale)
                for j in range(t):
                    cat[j] += head[j]
            for j in range(t):
                upd = _matvec_row(cat[j], So, 0, D)
                Z[j] = [Z[j][f] + upd[f] for f in range(D)]
        if cfg.F:
            W1, W2 = _w(W, "W1", b), _w(W, "W2", b)
            for j in range(t):
                zn = _rms(Z[j], cfg.rms_eps)
                g = [_gelu(v) for v in _matvec_row(zn, W1, 0, cfg.F)]
                upd = _matvec_row(g, W2, 0, D)
                Z[j] = [Z[j][f] + upd[f] for f in range(D)]
    Ck, Cv = [], []
    for j in range(t):
        zo = _rms(Z[j], cfg.rms_eps) if cfg.final_norm else Z[j]
        ck = _matvec_row(zo, W["Wkey"], 0, d)
        Ck.append(_rot_pairs(ck, qpos[j], cfg.theta, 1.0) if cfg.rope_fix else ck)
        Cv.append(_matvec_row(zo, W["Wval"], 0, d))
    return Ck, Cv
