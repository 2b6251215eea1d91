"""The oracle's pins catch plausible mistakes.

Each case plants one mistake in a copy of ``oracle/`` (a dropped term, a wrong
sign, a swapped threshold, a transposed operand, an off-by-one) and runs the
pin tests against that copy in a child process; the pins must fail.  The
mistakes are planted in the oracle, on the CPU, never in the kernels.
"""

import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

PIN_TESTS = ["test_oracle_logprob.py", "test_oracle_loss.py", "test_oracle_ewma.py",
             "test_oracle_diagnostics.py"]

# (file, original text, mutated text, what the mistake is)
MUTATIONS = [
    ("loss.py", "lse = M + np.log(np.exp(z - M[:, None]).sum(axis=1))",
     "lse = np.log(np.exp(z - M[:, None]).sum(axis=1))", "drop the max shift in lse"),
    ("loss.py", "logp[rows] = z[rows, ids[rows]] - lse[rows]",
     "logp[rows] = lse[rows] - z[rows, ids[rows]]", "sign of the log-probability"),
    ("loss.py", "log_rd = lo_ - lm", "log_rd = lm - lo_", "r_d inverted (mu/pi_old)"),
    ("loss.py", "log_rs = np.where(valid, lt - lo_, 0.0)",
     "log_rs = np.where(valid, lo_ - lt, 0.0)", "r_s inverted"),
    ("loss.py", "in_band = (p.rd_lo <= r_d) & (r_d <= p.rd_hi)",
     "in_band = (p.rd_lo < r_d) & (r_d < p.rd_hi)", "exclusive band"),
    ("loss.py", "mis = np.where(A >= 0, r_s <= 1.0 + p.eps_high, r_s >= 1.0 - p.eps_low)",
     "mis = np.where(A >= 0, r_s <= 1.0 + p.eps_low, r_s >= 1.0 - p.eps_high)",
     "eps_low / eps_high swapped"),
    ("loss.py", "mis = np.where(A >= 0, r_s <= 1.0 + p.eps_high, r_s >= 1.0 - p.eps_low)",
     "mis = np.where(A > 0, r_s <= 1.0 + p.eps_high, r_s >= 1.0 - p.eps_low)",
     "A = 0 in the wrong branch"),
    ("loss.py", "mis = np.where(A >= 0, r_s <= 1.0 + p.eps_high, r_s >= 1.0 - p.eps_low)",
     "mis = np.where(A >= 0, r_s >= 1.0 - p.eps_low, r_s <= 1.0 + p.eps_high)",
     "clip sides swapped between advantage signs"),
    ("loss.py", "w_d = r_d if p.rd_weight else np.ones(T)",
     "w_d = np.ones(T) if p.rd_weight else r_d", "role of r_d swapped"),
    ("loss.py", "s = np.minimum(r_s * A, np.clip(r_s, 1.0 - p.eps_low, 1.0 + p.eps_high) * A)",
     "s = np.maximum(r_s * A, np.clip(r_s, 1.0 - p.eps_low, 1.0 + p.eps_high) * A)",
     "max instead of min in the surrogate"),
    ("loss.py", "loss_t = np.where(keep, -w_d * s, 0.0)", "loss_t = np.where(keep, w_d * s, 0.0)",
     "loss sign"),
    ("loss.py", "g = np.where(active, -p.grad_scale * w_d * r_s * A / N, 0.0)",
     "g = np.where(active, -p.grad_scale * w_d * A / N, 0.0)", "gradient misses r_s"),
    ("loss.py", "g = np.where(active, -p.grad_scale * w_d * r_s * A / N, 0.0)",
     "g = np.where(keep, -p.grad_scale * w_d * r_s * A / N, 0.0)", "gradient ignores the clip"),
    ("loss.py", "out[rows] = -g[rows, None] * np.exp(z[rows] - np.asarray(lse)[rows, None])",
     "out[rows] = g[rows, None] * np.exp(z[rows] - np.asarray(lse)[rows, None])",
     "softmax term sign in dlogits"),
    ("loss.py", "out[rows, ids[rows]] += g[rows]", "out[rows, ids[rows] - 1] += g[rows]",
     "one-hot at the wrong index"),
    ("loss.py", "N = int(p.denom) if p.denom > 0 else int(np.sum(valid))",
     "N = int(p.denom) if p.denom > 0 else int(valid.size)", "masked tokens in the denominator"),
    ("ewma.py", "a = beta * w_prev / w", "a = beta / w", "recursion drops w_prev"),
    ("ewma.py", "w = 1.0 + beta * w_prev", "w = beta + w_prev", "weight recursion"),
    ("ewma.py", "streak = streak + 1 if rho < tau else 0", "streak = streak + 1 if rho <= tau else 0",
     "reset threshold inclusive"),
    ("ewma.py", "return beta / (1.0 - beta)", "return 1.0 / (1.0 - beta)", "center of mass"),
    ("ewma.py", "z = (z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)",
     "z = (z ^ (z >> np.uint64(26))) * np.uint64(0x94D049BB133111EB)", "generator shift"),
    ("ewma.py", "r = np.uint64(0x7FFF) + lsb", "r = np.uint64(0x8000)", "ties away from even"),
    ("proxies.py", "return alpha * lm + (1.0 - alpha) * lt", "return (1.0 - alpha) * lm + alpha * lt",
     "log-linear weights transposed"),
    ("proxies.py", "return np.log(alpha * np.exp(lm) + (1.0 - alpha) * np.exp(lt))",
     "return np.log(alpha * np.exp(lt) + (1.0 - alpha) * np.exp(lm))",
     "arithmetic proxy weights transposed"),
    ("diagnostics.py", "return (np.exp(lq) * (lq - lp)).sum(axis=1)",
     "return (np.exp(lp) * (lq - lp)).sum(axis=1)", "KL weighted by the wrong distribution"),
    ("diagnostics.py", "return -(np.exp(lp) * lp).sum(axis=1)",
     "return (np.exp(lp) * lp).sum(axis=1)", "entropy sign"),
    ("ewma.py", "b = 1.0 / w", "b = 1.0 / (w + 1.0)", "new-parameter weight off by one"),
    ("ewma.py", "new = th.copy() if reset else a * tp + b * th",
     "new = tp.copy() if reset else a * tp + b * th", "a reset keeps the old proximal parameters"),
    ("ewma.py", "out = ((u + r) >> np.uint64(16)) & np.uint64(0xFFFF)",
     "out = ((u + r + np.uint64(0x8000)) >> np.uint64(16)) & np.uint64(0xFFFF)",
     "rounding offset added on top of the random bits"),
    ("ewma.py", "fix = (np.abs(d) == half) & (d * e > 0)",
     "fix = (np.abs(d) == half) & (d * e < 0)", "float32 FMA midpoint resolved the wrong way"),
    ("loss.py", "flags = (in_band * FLAG_IN_BAND + (~mis) * FLAG_CLIPPED",
     "flags = (in_band * FLAG_IN_BAND + mis * FLAG_CLIPPED", "clip flag inverted"),
    ("loss.py", "n_rd_out=int(np.sum(valid & ~in_band))", "n_rd_out=int(np.sum(~in_band))",
     "out-of-band count includes masked tokens"),
    ("loss.py", "    ok = (ids >= 0) & (ids < V)\n", "    ok = (ids >= 0) & (ids <= V + 1)\n",
     "token ids past the vocabulary accepted"),
    ("ewma.py", "n_valid > 0 and streak >= min_streak", "n_valid > 0 and streak > min_streak",
     "reset one low step late"),
    ("ewma.py", "EwmaState(w=1.0, streak=0, n_resets=state.n_resets + 1)",
     "EwmaState(w=0.0, streak=0, n_resets=state.n_resets + 1)", "a reset empties the history weight"),
    ("diagnostics.py", "return z - (M + np.log(np.exp(z - M).sum(axis=1, keepdims=True)))",
     "return z - np.log(np.exp(z - M).sum(axis=1, keepdims=True))", "log-softmax without its shift"),
    ("ewma.py", "np.where(nan, quiet, np.where(special, trunc, out))", "out",
     "inf and NaN rounded like finite values"),
    ("ewma.py", "np.where(nan, quiet, np.where(special, trunc, out))", "np.where(special, trunc, out)",
     "NaN truncated (a low payload becomes inf)"),
    ("loss.py", "bad_ids = int(np.sum(m & ~ok))", "bad_ids = int(np.sum(~ok))",
     "masked tokens counted as bad ids"),
    ("loss.py", "loss = loss_sum / N if N > 0 else 0.0", "loss = loss_sum / N if N > 0 else np.nan",
     "empty batch gives NaN"),
    ("loss.py", "    valid = m & ok\n", "    valid = m\n", "bad ids kept as valid tokens"),
    ("loss.py", "dist_rs = np.where(A >= 0, np.abs(log_rs - np.log1p(p.eps_high))",
     "dist_rs = np.where(A >= 0, np.abs(log_rs - np.log1p(p.eps_low))",
     "clip-distance measured to the wrong edge"),
]


@pytest.fixture(scope="module")
def sandbox(tmp_path_factory):
    base = tmp_path_factory.mktemp("mut")
    shutil.copytree(os.path.join(ROOT, "tests"), base / "tests")
    return base


@pytest.mark.parametrize("fname,orig,mut,what", MUTATIONS, ids=[m[3] for m in MUTATIONS])
def test_pins_catch_planted_mistake(sandbox, fname, orig, mut, what):
    src = os.path.join(ROOT, "oracle", fname)
    text = open(src).read()
    assert text.count(orig) == 1, f"mutation anchor not found once in {fname}: {orig}"
    dst = sandbox / "oracle"
    if dst.exists():
        shutil.rmtree(dst)
    shutil.copytree(os.path.join(ROOT, "oracle"), dst)
    (dst / fname).write_text(text.replace(orig, mut))
    env = dict(os.environ, PYTHONPATH=str(sandbox))
    tests = [str(sandbox / "tests" / t) for t in PIN_TESTS]
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                        "--rootdir", str(sandbox), *tests], cwd=str(sandbox), env=env,
                       capture_output=True, text=True, timeout=300)
    assert r.returncode != 0, f"pins did not catch: {what}\n{r.stdout[-1500:]}"
