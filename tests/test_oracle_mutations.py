"""The oracle's pins catch plausible mistakes (CPU).

Each mutant plants one mistake -- a dropped term, a wrong sign, index or
operand, a relaxed comparison, a swapped tie-break -- in a copy of oracle/
and runs the pin tests that cover the function against that copy, in a
subprocess; every mutant must make them fail.  An unmutated copy must pass
the same tests, so a failure is the mistake's doing and not the harness's.
The library is not involved: the copy holds oracle/, synth/, the pin test
files, tests/conftest.py and tests/golden/ only."""

import os
import shutil
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

PLANNER = "tests/test_oracle_planner.py"
DIT = "tests/test_oracle_dit.py"
LEGAL = "tests/test_oracle_legality.py"
VARIANTS = "tests/test_oracle_variants.py"
RESPONSE = "tests/test_oracle_response.py"
GUIDANCE = "tests/test_oracle_guidance.py"
DRIFT = "tests/test_oracle_drift_trace.py"

# (name, file under oracle/, text, replacement, pin test files)
MUTANTS = [
    # Eq. 2
    ("L1 instead of L2 step length", "planner.py",
     "L = L + math.sqrt(dx * dx + dy * dy)", "L = L + abs(dx) + abs(dy)", [PLANNER]),
    ("heading change not wrapped", "planner.py",
     "T = T + abs(wrap(float(poses[t][2]) - float(poses[t - 1][2])))",
     "T = T + abs(float(poses[t][2]) - float(poses[t - 1][2]))", [PLANNER]),
    ("wrap seam left at -pi", "planner.py",
     "    if r == -math.pi:\n        r = math.pi\n", "", [PLANNER]),
    # Sec. 3.1 anchors
    ("median test not strict", "planner.py",
     "if Ts[i] > med and Ls[i] > L0 and Ts[i] > T0:",
     "if Ts[i] >= med and Ls[i] > L0 and Ts[i] > T0:", [PLANNER]),
    ("low anchor ties to the last clip", "planner.py",
     "        if s < best:\n            best, i0 = s, i",
     "        if s <= best:\n            best, i0 = s, i", [PLANNER]),
    ("moving anchor by sum instead of product", "planner.py",
     "p = zL[i] * zT[i]", "p = zL[i] + zT[i]", [PLANNER]),
    ("median of an even count is the lower middle", "planner.py",
     "return (s[n // 2 - 1] + s[n // 2]) / 2.0", "return s[n // 2 - 1]", [PLANNER]),
    # Eq. 3-4
    ("Theta normalised by the L anchors", "planner.py",
     'zT = (T - anc["T0"]) / max(anc["T1"] - anc["T0"], eps)',
     'zT = (T - anc["T0"]) / max(anc["L1"] - anc["L0"], eps)', [PLANNER]),
    ("support gate without the upper bound on zL", "planner.py",
     "return 0.0 <= zL <= 1.0 and 0.0 <= zT <= 1.0", "return 0.0 <= zL and 0.0 <= zT <= 1.0",
     [PLANNER]),
    ("intensity divided by 2 instead of sqrt 2", "planner.py",
     "return math.sqrt(zL * zL + zT * zT) / math.sqrt(2.0)",
     "return math.sqrt(zL * zL + zT * zT) / 2.0", [PLANNER]),
    # Eq. 8-9
    ("interpolation not one-sided", "planner.py",
     "out[j][h] = a + D * max(b - a, 0.0)", "out[j][h] = a + D * (b - a)", [PLANNER]),
    ("no monotone envelope", "planner.py",
     "run = max(run, qt[j][h])", "run = qt[j][h]", [PLANNER]),
    # Eq. 10-11, backtracking
    ("transition charged at the old age", "planner.py",
     "cand = cur[n][h] + c[k - h][h + 1]", "cand = cur[n][h] + c[k - h][h]", [PLANNER]),
    ("legality read at the current step", "planner.py",
     "if not legal(k + 1, h + 1):", "if not legal(k, h + 1):", [PLANNER]),
    ("budget test strict", "planner.py",
     "if v < INF and v <= tau:", "if v < INF and v < tau:", [PLANNER]),
    ("terminal age ties to the largest age", "planner.py",
     "        if row[hh] < best:\n            best, h = row[hh], hh",
     "        if row[hh] <= best:\n            best, h = row[hh], hh", [PLANNER]),
    # Eq. 12 and the controller
    ("acceptance ignores the running charge", "planner.py",
     "return d_obs <= dbar + eps and charge + c_inc <= tau",
     "return d_obs <= dbar + eps and c_inc <= tau", [PLANNER]),
    ("acceptance ignores the drift threshold", "planner.py",
     "return d_obs <= dbar + eps and charge + c_inc <= tau",
     "return charge + c_inc <= tau", [DIT]),
    ("drift normalised by the reference input", "planner.py",
     "den = math.sqrt(float(np.sum(a * a)))", "den = math.sqrt(float(np.sum(b * b)))", [PLANNER]),
    ("replan ignores the spent charge", "controller.py",
     'P.plan_suffix(tabs["c"], K, H, k, tau - S["C"], legal)',
     'P.plan_suffix(tabs["c"], K, H, k, tau, legal)', [PLANNER]),
    ("anchor drift normalised by the earlier input", "controller.py",
     "d[j][l] = P.drift(us[j + l], us[j], eps)", "d[j][l] = P.drift(us[j], us[j + l], eps)",
     [DRIFT]),
    ("anchor drift one step early", "controller.py",
     "d[j][l] = P.drift(us[j + l], us[j], eps)", "d[j][l] = P.drift(us[j + l - 1], us[j], eps)",
     [DRIFT]),
    ("checked drift normalised by the refresh input", "controller.py",
     'd_obs = P.drift(u_k, S["u_ref"], eps)', 'd_obs = P.drift(S["u_ref"], u_k, eps)', [DRIFT]),
    ("refresh does not reset the cache age", "controller.py",
     'S["j"], S["age"], S["r"], S["u_ref"] = k, 0, r, u',
     'S["j"], S["r"], S["u_ref"] = k, r, u', [DIT]),
    # Table 3 / Table 1 variants, Sec. 3.2 legality
    ("even schedule shifted by one step", "planner.py",
     "want = K > 1 and (k - 1) * n // (K - 1) > (k - 2) * n // (K - 1)",
     "want = K > 1 and k * n // (K - 1) > (k - 1) * n // (K - 1)", [VARIANTS]),
    ("expert boundary off by one", "planner.py",
     "(j <= expert_boundary) != (k <= expert_boundary)",
     "(j < expert_boundary) != (k < expert_boundary)", [LEGAL]),
    ("segments indexed from step 0", "planner.py",
     "(j - 1) // segment_len != (k - 1) // segment_len",
     "j // segment_len != k // segment_len", [LEGAL]),
    ("translation-only variant gates on Theta", "planner.py",
     "return (1, zL) if 0.0 <= zL <= 1.0 else (0, 0.0)",
     "return (1, zL) if 0.0 <= zT <= 1.0 else (0, 0.0)", [VARIANTS]),
    # the DiT (Eq. 1) and the sampler
    ("LayerNorm epsilon 1e-5", "dit.py", "LN_EPS = 1e-6", "LN_EPS = 1e-5", [DIT]),
    ("GELU cubic coefficient", "dit.py",
     "(x + 0.044715 * x ** 3)", "(x + 0.04715 * x ** 3)", [DIT]),
    ("attention scaled by 1/dh", "dit.py",
     "p = softmax(q[hd] @ k[hd].T / math.sqrt(dh))", "p = softmax(q[hd] @ k[hd].T / dh)", [DIT]),
    ("k and v planes swapped", "dit.py",
     "k = qkv[:, d:2 * d].reshape", "k = qkv[:, 2 * d:].reshape", [DIT]),
    ("scale applied without the 1 +", "dit.py",
     'a = layer_norm(h) * (1.0 + mod["scale1"]) + mod["shift1"]',
     'a = layer_norm(h) * mod["scale1"] + mod["shift1"]', [DIT]),
    ("MLP residual gated by the attention gate", "dit.py",
     'h = h + mod["gate2"] * linear(m, wb["w_2"], wb["b_2"])',
     'h = h + mod["gate1"] * linear(m, wb["w_2"], wb["b_2"])', [DIT]),
    ("Euler step with the wrong sign", "dit.py",
     "return f64(x) + (float(sigma_next) - float(sigma_k)) * f64(v)",
     "return f64(x) + (float(sigma_k) - float(sigma_next)) * f64(v)", [DIT]),
    ("cached feature is h_L instead of h_L - u", "dit.py",
     "return v, u, hL - u", "return v, u, hL", [DIT]),
    ("timestep features of sigma instead of 1000 sigma", "dit.py",
     "t = 1000.0 * float(sigma)", "t = float(sigma)", [DIT]),
    ("final shift and scale swapped", "dit.py",
     "return blocks, dict(shift=f[0], scale=f[1])", "return blocks, dict(shift=f[1], scale=f[0])",
     [DIT]),
    ("pose heading not wrapped", "dit.py",
     "out[t, 2] = _wrap(p[t, 2] - p[0, 2])", "out[t, 2] = p[t, 2] - p[0, 2]", [DIT]),
    ("guidance around the conditional branch", "controller.py",
     "return v_u + cfg_scale * (v_c - v_u)", "return v_c + cfg_scale * (v_c - v_u)", [GUIDANCE]),
    # Eq. 6-7 responses
    ("LayerNorm tangent without the projection term", "response.py",
     "return (dx - dx.mean(axis=-1, keepdims=True) - y * (y * dx).mean(axis=-1, keepdims=True)) / sig",
     "return (dx - dx.mean(axis=-1, keepdims=True)) / sig", [RESPONSE]),
    ("GELU derivative of the cubic term", "response.py",
     "(1.0 + 3.0 * c * x * x)", "(1.0 + c * x * x)", [RESPONSE]),
    ("softmax tangent without the row sum", "response.py",
     "dp = p * (ds - (p * ds).sum(axis=1, keepdims=True))", "dp = p * ds", [RESPONSE]),
    ("perturbation injected without the step size", "response.py",
     "dx = (float(sig[t]) - float(sig[t - 1])) * f64(e)", "dx = f64(e)", [RESPONSE]),
    ("response normalised by x_K instead of the terminal latent", "response.py",
     "den = float(np.linalg.norm(xs[K + 1])) + eps", "den = float(np.linalg.norm(xs[K])) + eps",
     [RESPONSE]),
]


def _copy_tree(dst, mutant=None):
    shutil.copytree(os.path.join(ROOT, "oracle"), os.path.join(dst, "oracle"),
                    ignore=shutil.ignore_patterns("__pycache__"))
    shutil.copytree(os.path.join(ROOT, "synth"), os.path.join(dst, "synth"),
                    ignore=shutil.ignore_patterns("__pycache__"))
    os.makedirs(os.path.join(dst, "tests"))
    shutil.copytree(os.path.join(ROOT, "tests", "golden"), os.path.join(dst, "tests", "golden"))
    for f in ("conftest.py", "test_oracle_planner.py", "test_oracle_dit.py",
              "test_oracle_legality.py", "test_oracle_variants.py", "test_oracle_response.py",
              "test_oracle_guidance.py", "test_oracle_drift_trace.py"):
        shutil.copy(os.path.join(ROOT, "tests", f), os.path.join(dst, "tests", f))
    if mutant is not None:
        _, fname, old, new, _ = mutant
        p = os.path.join(dst, "oracle", fname)
        with open(p) as fh:
            src = fh.read()
        assert src.count(old) == 1, f"mutation site not unique in {fname}: {old!r}"
        with open(p, "w") as fh:
            fh.write(src.replace(old, new))


def _run(dst, files):
    env = dict(os.environ, PYTHONPATH=dst, PYTHONDONTWRITEBYTECODE="1")
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                        "-m", "not gpu", *files], cwd=dst, env=env, capture_output=True,
                       text=True, timeout=600)
    return r.returncode, (r.stdout + r.stderr)[-1500:]


def test_mutation_sites_exist_once():
    for m in MUTANTS:
        with open(os.path.join(ROOT, "oracle", m[1])) as fh:
            assert fh.read().count(m[2]) == 1, m[0]


def test_every_planted_mistake_fails_a_pin(tmp_path):
    pytest.importorskip("torch")

    def job(i):
        dst = str(tmp_path / f"m{i}")
        if i < 0:
            _copy_tree(dst)
            return i, _run(dst, sorted({f for m in MUTANTS for f in m[4]}))
        _copy_tree(dst, MUTANTS[i])
        return i, _run(dst, MUTANTS[i][4])

    with ThreadPoolExecutor(max(2, min(8, os.cpu_count() or 2))) as ex:
        res = dict(ex.map(job, [-1] + list(range(len(MUTANTS)))))
    rc, out = res[-1]
    assert rc == 0, "the unmutated copy must pass its pins:\n" + out
    survivors = [MUTANTS[i][0] for i in range(len(MUTANTS)) if res[i][0] == 0]
    broken = [(MUTANTS[i][0], res[i][1]) for i in range(len(MUTANTS)) if res[i][0] not in (0, 1)]
    assert not broken, broken
    assert not survivors, "mistakes no pin catches: " + "; ".join(survivors)
