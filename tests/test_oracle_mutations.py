"""The oracle's pins catch plausible mistakes.  Each case plants one mistake
in a copy of the oracle's source (a dropped term, a wrong sign, an off-by-one
window, a missing normaliser, a reversed index, the wrong logarithm...), runs
the pins of tests/test_oracle.py against that copy, and requires at least one
of them to fail.  CPU only; the oracle itself is never modified."""

import inspect
import os
import types

import pytest

import tests.test_oracle as pins

ORACLE = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "oracle",
                      "spo_oracle.py")
GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")

# (name, text in the oracle, replacement): each text occurs exactly once
MUTATIONS = [
    ("logits: temperature dropped", "return float(inv_temp) * (np.asarray(H", "return (np.asarray(H"),
    ("lse: max shift dropped", "lse_r = m + np.log(s)", "lse_r = np.log(s)"),
    ("entropy: sign", "ent[rows] = lse_r - (p * z).sum(axis=1)",
     "ent[rows] = lse_r + (p * z).sum(axis=1)"),
    ("logp: sign of lse", "logp[rows] = z[np.arange(rows.size), tgt[rows]] - lse_r",
     "logp[rows] = z[np.arange(rows.size), tgt[rows]] + lse_r"),
    ("window: off by one", "(earlier < window)", "(earlier <= window)"),
    ("token select: ignore index dropped",
     "eligible = (np.asarray(mask).astype(np.int64) == 1) & (np.asarray(tgt).astype(np.int64) >= 0)",
     "eligible = np.asarray(mask).astype(np.int64) == 1"),
    ("advantage: always population std", "dof = (n - 1) if std_mode == STD_UNBIASED else n",
     "dof = n"),
    ("advantage: eps dropped", "adv[idx] = (rg - mu) / (sigma + eps)",
     "adv[idx] = (rg - mu) / sigma"),
    ("advantage: zero-variance rule dropped",
     "        if rg.max() == rg.min():\n            continue\n        mu = rg.sum() / n",
     "        mu = rg.sum() / n"),
    ("advantage f32: wrong count in the mean", "mu = f(acc / f(n))", "mu = f(acc / f(n + 1))"),
    ("advantage f32: pairwise sum (np.sum) for the sequential one",
     "        acc = f(0.0)\n        for i in idx:\n            acc = f(acc + r[i])",
     "        acc = f(np.sum(r[idx]))"),
    ("advantage f32: members summed in descending index",
     "        for i in idx:\n            acc = f(acc + r[i])",
     "        for i in reversed(idx):\n            acc = f(acc + r[i])"),
    ("advantage f32: fused multiply-add in the sum of squares", "ss = f(ss + f(dv * dv))",
     "ss = f(float(ss) + float(dv) * float(dv))"),
    ("KL: sign of delta", "kl = np.exp(delta) - delta - 1.0", "kl = np.exp(delta) + delta - 1.0"),
    ("surrogate: max for min", "surr = np.minimum(rho * A, clipped * A)",
     "surr = np.maximum(rho * A, clipped * A)"),
    ("clip: upper bound", "clipped = np.clip(rho, 1.0 - clip_eps, 1.0 + clip_eps)",
     "clipped = np.clip(rho, 1.0 - clip_eps, 1.0 + 2.0 * clip_eps)"),
    ("clip gradient: negative-advantage branch dropped",
     "binds = ((A > 0) & (rho > 1.0 + clip_eps)) | ((A < 0) & (rho < 1.0 - clip_eps))",
     "binds = (A > 0) & (rho > 1.0 + clip_eps)"),
    ("KL gradient: sign", "dkl = 1.0 - np.exp(delta)", "dkl = np.exp(delta) - 1.0"),
    ("aggregation: group size dropped", "w = 1.0 / (n_nonempty * size[gid[i]] * n_tok[i])",
     "w = 1.0 / (n_nonempty * n_tok[i])"),
    ("token aggregation: wrong normaliser", "c[lm == 1] = 1.0 / total", "c[lm == 1] = 1.0 / T"),
    ("backward: lse without the max", "lse = m + np.log(np.exp(z - m[:, None]).sum(axis=1))",
     "lse = np.log(np.exp(z - m[:, None]).sum(axis=1))"),
    ("backward: one-hot sign",
     "onehot[np.arange(rows.size), tgt[rows]] = 1.0\n    G = inv_temp * g[rows][:, None] * (onehot - p)",
     "onehot[np.arange(rows.size), tgt[rows]] = 1.0\n    G = inv_temp * g[rows][:, None] * (p - onehot)"),
    ("backward: dW rows reversed", "    dW = G.T @ H[rows]\n    return dH, dW\n\n\ndef policy_loss_bwd_slice",
     "    dW = (G.T @ H[rows])[::-1]\n    return dH, dW\n\n\ndef policy_loss_bwd_slice"),
    ("slice merge: maxima not aligned", "S = (s * np.exp(m - M)).sum()", "S = s.sum()"),
    ("slice record: missing target marked 0", "zt = np.full(rows.size, -np.inf)",
     "zt = np.zeros(rows.size)"),
    ("slice backward: offset forgotten", "local = tgt[rows] - v_offset\n    hit = np.nonzero",
     "local = tgt[rows]\n    hit = np.nonzero"),
    ("reward: stability sign", 'r += -q["alpha_cv"] * c[i]', 'r += q["alpha_cv"] * c[i]'),
    ("reward: natural log for log2", "ls = math.log2(S[i]) if S[i] > 0 else -math.inf",
     "ls = math.log(S[i]) if S[i] > 0 else -math.inf"),
    ("reward: speedup counted before all tests pass", "if p[i] >= 1.0:", "if p[i] > 0.5:"),
    ("ranker: first ReLU dropped", "h1 = np.maximum(a1, 0.0)", "h1 = a1"),
    ("ranker: z-score sign",
     "x = (np.asarray(phi, dtype=np.float64) - np.asarray(mu, dtype=np.float64))",
     "x = (np.asarray(phi, dtype=np.float64) + np.asarray(mu, dtype=np.float64))"),
]


def _calls():
    """Every pin of tests/test_oracle.py as (name, zero-argument callable)."""
    out = []
    for name, fn in inspect.getmembers(pins, inspect.isfunction):
        if not name.startswith("test_") or fn.__module__ != pins.__name__:
            continue
        variants = [{}]
        for mark in getattr(fn, "pytestmark", []):
            if mark.name != "parametrize":
                continue
            argnames = mark.args[0]
            names = [a.strip() for a in argnames.split(",")] if isinstance(argnames, str) \
                else list(argnames)
            values = [v.values if hasattr(v, "values") else (v if len(names) > 1 else (v,))
                      for v in mark.args[1]]
            variants = [dict(base, **dict(zip(names, v))) for base in variants for v in values]
        takes_golden = "golden_dir" in inspect.signature(fn).parameters
        for kw in variants:
            kw = dict(kw, golden_dir=GOLDEN) if takes_golden else kw
            out.append((name, lambda fn=fn, kw=kw: fn(**kw)))
    return out


def _mutant(text, replacement):
    src = open(ORACLE).read()
    assert src.count(text) == 1, f"mutation text occurs {src.count(text)} times"
    mod = types.ModuleType("spo_oracle_mutant")
    exec(compile(src.replace(text, replacement), ORACLE, "exec"), mod.__dict__)
    return mod


@pytest.mark.parametrize("name,text,replacement", MUTATIONS, ids=[m[0] for m in MUTATIONS])
def test_pins_catch_the_mistake(name, text, replacement, monkeypatch):
    monkeypatch.setattr(pins, "O", _mutant(text, replacement))
    for pin, call in _calls():
        try:
            call()
        except Exception:
            return      # caught
    pytest.fail(f"no pin fails when the oracle has: {name}")


def test_unmodified_oracle_passes_every_pin():
    for pin, call in _calls():
        call()
