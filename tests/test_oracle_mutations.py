"""Mutation check of the oracle's pins (CPU): each case plants one plausible mistake in a copy
of the oracle's source, loads that copy as a separate module and runs every pin of
test_oracle_pins.py against it. A pin set that lets a planted mistake through is too weak to
vouch for the oracle, so every mutant must fail at least one pin, and the unmutated copy must
pass them all.

The oracle file on disk is never modified: the mutant is compiled from a string."""
import inspect
import os
import sys
import types

import pytest

import test_oracle_pins as P

SRC_PATH = os.path.join(os.path.dirname(__file__), os.pardir, "oracle", "still_oracle.py")

# (what the mistake is, the oracle's text, the mistaken text)
MUTANTS = [
    # compactor sublayers (App. A)
    ("key bias dropped",
     "k = l2norm(X @ Wk[:, cols] + bk[cols], cfg.l2_eps)",
     "k = l2norm(X @ Wk[:, cols], cfg.l2_eps)"),
    ("value projection given the key bias",
     "v = X @ Wv[:, cols]                                        # [N, D], no bias",
     "v = X @ Wv[:, cols] + bk[cols]"),
    ("cross-attention heads concatenated in reverse",
     "return np.concatenate(heads, axis=-1) @ Wo ",
     "return np.concatenate(heads[::-1], axis=-1) @ Wo "),
    ("self-attention scores transposed",
     "heads.append(softmax_rows(cfg.scale * (q @ k.T)) @ v)",
     "heads.append(softmax_rows(cfg.scale * (k @ q.T)) @ v)"),
    ("self-attention values projected by the key weights",
     "v = Zn @ Sv[:, cols]",
     "v = Zn @ Sk[:, cols]"),
    ("self-attention output projection by the value weights",
     "return np.concatenate(heads, axis=-1) @ So",
     "return np.concatenate(heads, axis=-1) @ Sv.T"),
    ("self-attention query bias dropped",
     "q = l2norm(Zn @ Sq[:, cols] + sbq[cols], cfg.l2_eps)",
     "q = l2norm(Zn @ Sq[:, cols], cfg.l2_eps)"),
    ("FFN without its pre-norm",
     "Z = Z + ffn(rmsnorm(Z, cfg.rms_eps), W, b)",
     "Z = Z + ffn(Z, W, b)"),
    ("self-attention residual dropped",
     "Z = Z + self_attention(rmsnorm(Z, cfg.rms_eps), W, b, cfg)",
     "Z = self_attention(rmsnorm(Z, cfg.rms_eps), W, b, cfg)"),
    ("cross-attention in every block regardless of the configuration",
     "if b == 0 or cfg.cross_every_block:",
     "if True:"),
    ("final RMSNorm always on",
     "Zout = rmsnorm(Z, cfg.rms_eps) if cfg.final_norm else Z",
     "Zout = rmsnorm(Z, cfg.rms_eps)"),
    # primitives
    ("tanh-approximate GELU",
     "return 0.5 * x * (1.0 + erf(x / np.sqrt(2.0)))",
     "return 0.5 * x * (1.0 + np.tanh(np.sqrt(2.0 / np.pi) * (x + 0.044715 * x ** 3)))"),
    ("RMSNorm over the sum instead of the mean",
     "return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps)",
     "return x / np.sqrt(np.sum(x * x, axis=-1, keepdims=True) + eps)"),
    ("L2 norm by the squared norm",
     "return x / np.maximum(np.linalg.norm(x, axis=-1, keepdims=True), eps)",
     "return x / np.maximum(np.linalg.norm(x, axis=-1, keepdims=True) ** 2, eps)"),
    ("softmax normalised over the wrong axis",
     "return e / e.sum(axis=-1, keepdims=True)",
     "return e / e.sum(axis=0, keepdims=True)"),
    # RoPE and positions (Sec. 2.2; App. A, App. B)
    ("RoPE inverse with the wrong sign",
     "return np.concatenate([a * c + b * s, -a * s + b * c], axis=-1)",
     "return np.concatenate([a * c - b * s, a * s + b * c], axis=-1)"),
    ("frequency index shifted by one",
     "omega = base ** (-2.0 * m / width)",
     "omega = base ** (-2.0 * (m + 1) / width)"),
    ("query positions past the last key",
     "qpos = linspace_positions(pmin, pmax, t)",
     "qpos = linspace_positions(pmin, pmax + 1, t)"),
    ("query positions exclude the last key position",
     "return np.linspace(pmin, pmax, t, dtype=np.float64)",
     "return np.linspace(pmin, pmax, t, endpoint=False, dtype=np.float64)"),
    ("keys un-rotated one position off",
     "Kx = unrope(Kh, kpos, cfg.theta) if cfg.rope_fix else Kh",
     "Kx = unrope(Kh, kpos + 1, cfg.theta) if cfg.rope_fix else Kh"),
    ("C_k re-rotated with the compactor's base",
     "Ck = rope(Ck, opos, cfg.theta)                 # back into",
     "Ck = rope(Ck, opos, cfg.theta_c)                 # back into"),
    # accounting (App. J, App. B, App. D)
    ("budget floored instead of rounded",
     "return (2 * N + c) // (2 * c)",
     "return N // c"),
    ("position offset without the compact length",
     "return logical_len - t",
     "return logical_len"),
    ("parameter count without W_O",
     "ca = D * n_c * D + 2 * (2 * d * n_c * D) + n_c * D * D",
     "ca = D * n_c * D + 2 * (2 * d * n_c * D)"),
    ("KV bytes for K only",
     "return 2 * L * H * d * b * S",
     "return L * H * d * b * S"),
    # lookahead schedule (Sec. 2.3)
    ("prefill past without the raw chunk",
     "past = compacted_before * t + ct",
     "past = compacted_before * t"),
    ("retained cache without the lookahead chunk",
     "retained_after = compacted_after * t + raw_after",
     "retained_after = compacted_after * t"),
    ("prefill starts one chunk early",
     "prefill = ((k + 1) * ct, ct)",
     "prefill = (k * ct, ct)"),
    # beta head and biased attention (App. A, App. B)
    ("saturation without beta_max",
     "beta = beta_max * np.tanh(beta / beta_max)",
     "beta = np.tanh(beta)"),
    ("mass-matching offset inverted",
     "beta = beta + np.log(T / t) + (log_x if mass_match == 2 else 0.0)",
     "beta = beta + np.log(t / T) + (log_x if mass_match == 2 else 0.0)"),
    ("bias subtracted",
     "scale * (q @ Ck.T) + beta[None, :], scale * (q @ Kfix.T)",
     "scale * (q @ Ck.T) - beta[None, :], scale * (q @ Kfix.T)"),
    ("bias moved to the uncompacted entries",
     "scale * (q @ Ck.T) + beta[None, :], scale * (q @ Kfix.T)",
     "scale * (q @ Ck.T), scale * (q @ Kfix.T) + beta.mean()"),
    ("value rows in the wrong order",
     "return softmax_rows(logits) @ np.concatenate([Cv, Vfix], axis=0)",
     "return softmax_rows(logits) @ np.concatenate([Vfix, Cv], axis=0)"),
]


def _source():
    with open(SRC_PATH) as f:
        return f.read()


def _load(src, name):
    mod = types.ModuleType(name)
    mod.__file__ = SRC_PATH
    sys.modules[name] = mod  # dataclass processing looks the module up by name
    try:
        exec(compile(src, f"<{name}>", "exec"), mod.__dict__)
    finally:
        del sys.modules[name]
    return mod


def _pins():
    """Every pin of test_oracle_pins.py as (id, function, kwargs), parametrised cases expanded."""
    out = []
    for name, fn in inspect.getmembers(P, inspect.isfunction):
        if not name.startswith("test_"):
            continue
        marks = [m for m in getattr(fn, "pytestmark", []) if m.name == "parametrize"]
        needed = list(inspect.signature(fn).parameters)
        if not marks:
            assert not needed, f"{name} takes fixtures {needed}"
            out.append((name, fn, {}))
            continue
        assert len(marks) == 1, name
        argnames, values = marks[0].args[0], marks[0].args[1]
        names = [a.strip() for a in argnames.split(",")] if isinstance(argnames, str) else list(argnames)
        assert sorted(names) == sorted(needed), (name, names, needed)
        for v in values:
            vals = tuple(v) if len(names) > 1 else (v,)
            out.append((f"{name}{vals}", fn, dict(zip(names, vals))))
    return out


def _failing_pins(mod):
    saved = P.O
    P.O = mod
    failed = []
    try:
        for pid, fn, kw in _pins():
            try:
                fn(**kw)
            except Exception as e:  # noqa: BLE001 - an assertion or a crash both catch it
                failed.append((pid, type(e).__name__))
    finally:
        P.O = saved
    return failed


def test_unmutated_copy_passes_every_pin():
    assert len(_pins()) >= 30
    assert _failing_pins(_load(_source(), "still_oracle_copy")) == []


@pytest.mark.filterwarnings("ignore::RuntimeWarning")
@pytest.mark.parametrize("what,orig,mutant", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_planted_mistake_fails_a_pin(what, orig, mutant):
    src = _source()
    assert src.count(orig) == 1, f"oracle text not found once: {orig!r}"
    failed = _failing_pins(_load(src.replace(orig, mutant), "still_oracle_mutant"))
    # caught by a failed assertion, not only by a crash of the mutated code
    assert any(kind == "AssertionError" for _, kind in failed), f"no pin catches: {what} {failed}"
