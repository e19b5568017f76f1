"""Strength of the oracle's pins.

Each entry of MUTANTS is a plausible mistake (a dropped term, a wrong sign,
index, constant or bound, a transposed operand, a reading swapped for its
alternative).  It is planted in a copy of the oracle in a temporary
directory, on the CPU, and the oracle's pin tests (tests/test_oracle_*.py,
copied beside it) are run against that copy: every mutant must make at
least one pin fail.  The unmodified copy must pass, so a failure can only
come from the planted mistake.  Nothing here touches the oracle in the tree
or the CUDA path.

Mistakes with no observable effect are not listed: reversing the shuffle's
index tie-break, for one, changes nothing, because the 64-bit keys of one
iteration do not collide at any size the path handles (the shuffle pin
checks that they are distinct).
"""
import glob
import os
import shutil
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
C = "edp_oracle.c"

# (name, oracle file, text as it stands, the mistake)
MUTANTS = [
    # Philox4x32-10 and the draw assembly (Salmon et al.)
    ("philox-weyl-constant", C, "k0 += PHILOX_W0;", "k0 += PHILOX_W1;"),
    ("philox-nine-rounds", C, "for (int r = 0; r < 10; ++r)", "for (int r = 0; r < 9; ++r)"),
    ("philox-multiplier-swap", C, "(uint64_t)PHILOX_M0 * (uint64_t)x0",
     "(uint64_t)PHILOX_M1 * (uint64_t)x0"),
    ("u64-word-order", C, "return ((uint64_t)o[1] << 32) | (uint64_t)o[0];",
     "return ((uint64_t)o[0] << 32) | (uint64_t)o[1];"),
    ("u64-counter-layout", C,
     "uint32_t c[4] = {j, (uint32_t)round, stream, (uint32_t)(round >> 32)};",
     "uint32_t c[4] = {j, stream, (uint32_t)round, (uint32_t)(round >> 32)};"),
    ("mulhi-shift", C, "return (uint64_t)(p >> 64);", "return (uint64_t)(p >> 63);"),
    # logical ring
    ("ring-slot-off-by-one", C, "return (total - size + k) % cap;",
     "return (total - size + k + 1) % cap;"),
    ("ring-offset-off-by-one", C, "return (slot + cap - oldest) % cap;",
     "return (slot + cap - oldest + 1) % cap;"),
    ("ring-write-slot", C, "uint64_t slot = (total + j) % cap;",
     "uint64_t slot = (total + j + 1) % cap;"),
    # priorities and the deferred newest leaf
    ("defer-resolves-to-new-q", C,
     "if (id >= 1 && cap >= 2) leaves[(id - 1) % cap] = *pending;",
     "if (id >= 1 && cap >= 2) leaves[(id - 1) % cap] = qj;"),
    ("defer-off", C, "leaves[slot] = 0;\n      *pending = qj;",
     "leaves[slot] = qj;\n      *pending = qj;"),
    ("default-not-running-max", C, "    if (qj > *qmax) *qmax = qj;\n", ""),
    ("update-first-wins", C, "for (uint64_t p = 0; p < n; ++p) {\n    if (idx[p] < 0",
     "for (uint64_t p = n; p-- > 0;) {\n    if (idx[p] < 0"),
    ("update-newest-not-pending", C, "*pending = q[p];\n    else",
     "leaves[s] = q[p];\n    else"),
    ("update-stale-slot-kept", C, "    if (k >= size) continue;\n", ""),
    ("td-floor", C, "double r = nearbyint(p);", "double r = floor(p);"),
    ("td-no-abs", C, "pow(fabs(td) + eps, alpha)", "pow(td + eps, alpha)"),
    ("td-scale", C, "* 1048576.0;", "* 1048575.0;"),
    ("td-no-eps", C, "pow(fabs(td) + eps, alpha)", "pow(fabs(td), alpha)"),
    # samplers
    ("uniform-stream", C, "uint64_t u = orc_philox_u64(seed, k, round, 0);",
     "uint64_t u = orc_philox_u64(seed, k, round, 1);"),
    ("uniform-range", C, "uint64_t off = orc_mulhi64(u, n_valid);",
     "uint64_t off = orc_mulhi64(u, n_valid + 1);"),
    ("stratum-ceil", C, "unsigned __int128 hi = ((unsigned __int128)S * (k + 1)) / B;",
     "unsigned __int128 hi = ((unsigned __int128)S * (k + 1) + B - 1) / B;"),
    ("stratum-no-offset", C, "return (uint64_t)lo + orc_mulhi64(u, (uint64_t)(hi - lo));",
     "return orc_mulhi64(u, (uint64_t)(hi - lo));"),
    ("scan-closed-interval", C, "if (t < prefix + leaves[i]) break;",
     "if (t <= prefix + leaves[i]) break;"),
    ("scan-stream", C,
     "uint64_t t = orc_stratum_target(S, B, k, orc_philox_u64(seed, k, round, 1));\n"
     "    uint64_t prefix = 0;",
     "uint64_t t = orc_stratum_target(S, B, k, orc_philox_u64(seed, k, round, 0));\n"
     "    uint64_t prefix = 0;"),
    ("bisect-bound", C, "if (prefix[mid + 1] > t)", "if (prefix[mid + 1] >= t)"),
    ("isw-inverted", C, "pow((double)qmin / (double)q[k], beta)",
     "pow((double)q[k] / (double)qmin, beta)"),
    ("isw-batch-max", C, "if (q[k] < qmin) qmin = q[k];", "if (q[k] > qmin) qmin = q[k];"),
    ("isw-no-beta", C, "pow((double)qmin / (double)q[k], beta)",
     "((double)qmin / (double)q[k])"),
    # byte -> float transforms
    ("unit-256", C, "float den = 255.0f;", "float den = 256.0f;"),
    ("unit-reciprocal", C, "return num / den;", "return num * (1.0f / den);"),
    ("bf16-ties-away", C, "u += 0x7FFFu + lsb;", "u += 0x8000u;"),
    ("bf16-truncate", C, "u += 0x7FFFu + lsb;", "u += 0u;"),
    ("norm-sign", C, "float t = x - mean;", "float t = mean - x;"),
    ("norm-times-std", C, "float y = t / stdv;", "float y = t * stdv;"),
    # frame stacks
    ("stack-anchor-done-counts", C, "for (int64_t o = j; !zero && o < anchor_off; ++o)",
     "for (int64_t o = j; !zero && o <= anchor_off; ++o)"),
    ("stack-repeat-oldest", C, "int zero = (j < 0);",
     "int zero = 0;\n    if (j < 0) j = 0;"),
    ("stack-ignores-done", C,
     "for (int64_t o = j; !zero && o < anchor_off; ++o)",
     "for (int64_t o = j; 0 && o < anchor_off; ++o)"),
    ("next-obs-same-anchor", C, "stack_at(frames, done, cap, total, F, K, k + 1, next_obs);",
     "stack_at(frames, done, cap, total, F, K, k, next_obs);"),
    ("stack-frame-order", C, "float *dst = out + (uint64_t)m * F;",
     "float *dst = out + (uint64_t)(K - 1 - m) * F;"),
    ("dqn-reward-of-next", C, "if (rew_out) rew_out[b] = reward[s];\n    if (done_out)",
     "if (rew_out) rew_out[b] = reward[(s + 1) % cap];\n    if (done_out)"),
    ("dqn-action-of-next", C, "if (act_out) act_out[b] = action[s];",
     "if (act_out) act_out[b] = action[(s + 1) % cap];"),
    # on-policy and multimodal delivery
    ("hwc-channel-order", C, "hwc[((uint64_t)y * W + x) * C + c]",
     "hwc[((uint64_t)y * W + x) * C + (C - 1 - c)]"),
    ("hwc-transposed", C, "chw[((uint64_t)c * H + y) * W + x]",
     "chw[((uint64_t)c * W + x) * H + y]"),
    ("ppo-scalars-by-slot", C, "if (adv_out) adv_out[b] = adv_src[k];",
     "if (adv_out) adv_out[b] = adv_src[s];"),
    ("ppo-return-is-advantage", C, "if (ret_out) ret_out[b] = ret_src[k];",
     "if (ret_out) ret_out[b] = adv_src[k];"),
    ("mm-channel-stats-swapped", C,
     "out[c * HW + p] = orc_norm_bf16(chw[c * HW + p], mean[c], stdv[c]);",
     "out[c * HW + p] = orc_norm_bf16(chw[c * HW + p], mean[C - 1 - c], stdv[C - 1 - c]);"),
    ("mm-tokens-of-previous", C, "memcpy(tok_out + (uint64_t)b * L, tok_ring + s * L, (size_t)L * 4);",
     "memcpy(tok_out + (uint64_t)b * L, tok_ring + (s ? s - 1 : 0) * L, (size_t)L * 4);"),
    ("mm-reward-of-previous", C, "if (rew_out) rew_out[b] = reward[s];\n  }\n}\n\n/* ---",
     "if (rew_out) rew_out[b] = reward[s ? s - 1 : 0];\n  }\n}\n\n/* ---"),
    # GAE and normalisation (Schulman et al.)
    ("gae-no-done-cut", C, "        if (d[at]) break;\n", ""),
    ("gae-no-lambda", C, "coef *= gamma * lambda;", "coef *= gamma;"),
    ("gae-bootstrap-unmasked", C,
     "gamma * (double)v[(uint64_t)(u + 1) * E + e] * nd", "gamma * (double)v[(uint64_t)(u + 1) * E + e]"),
    ("gae-value-sign", C, "                       (double)v[at];",
     "                       0.0 * (double)v[at];"),
    ("gae-return-next-value", C, "ret[o] = A + (double)v[o];", "ret[o] = A + (double)v[o + E];"),
    ("normalize-biased-std", C, "sqrt(ss / (double)(n - 1))", "sqrt(ss / (double)n)"),
    ("normalize-no-eps", C, "out[i] = (a[i] - mean) / (sd + 1e-8);", "out[i] = (a[i] - mean) / sd;"),
    # shuffle
    ("perm-descending", C, "if (x->key != y->key) return x->key < y->key ? -1 : 1;",
     "if (x->key != y->key) return x->key < y->key ? 1 : -1;"),
    ("perm-stream", C, "v[j].key = orc_philox_u64(seed, j, iteration, 2);",
     "v[j].key = orc_philox_u64(seed, j, iteration, 1);"),
    # two-tier placement map
    ("tier-boundary", C, "} else if (L >= total - in_hbm) {", "} else if (L > total - in_hbm) {"),
    ("tier-host-slot", C, "*slot = L % (cap - cap_h);", "*slot = L % cap_h;"),
    ("tier-evicted-kept", C, "if (L >= total || L < total - size) {", "if (L >= total) {"),
    # more row lookups, bounds and clamps
    ("philox-key-bumped-first", C, "    if (r > 0) {\n      k0 += PHILOX_W0;",
     "    if (r >= 0) {\n      k0 += PHILOX_W0;"),
    ("philox-key-word-swap", C, "uint32_t n0 = (uint32_t)(p1 >> 32) ^ x1 ^ k0;",
     "uint32_t n0 = (uint32_t)(p1 >> 32) ^ x1 ^ k1;"),
    ("leaf-sum-drops-last", C, "for (uint64_t i = lo; i < hi; ++i) s += leaves[i];",
     "for (uint64_t i = lo; i + 1 < hi; ++i) s += leaves[i];"),
    ("scan-q-of-next", C, "qout[k] = leaves[i];", "qout[k] = leaves[(i + 1) % cap];"),
    ("bisect-prefix-offset", C, "  prefix[0] = 0;\n", "  prefix[0] = 1;\n"),
    ("td-clamp-low", C, "if (!(r >= 1.0)) r = 1.0;", "if (!(r >= 0.0)) r = 0.0;"),
    ("td-clamp-high", C, "if (r > 4294967295.0) r = 4294967295.0;",
     "if (r > 4294967294.0) r = 4294967294.0;"),
    ("dqn-done-of-next", C, "if (done_out) done_out[b] = done[s];",
     "if (done_out) done_out[b] = done[(s + 1) % cap];"),
    ("ppo-image-of-previous", C,
     "orc_hwc_to_chw_bf16(obs_ring + s * F, H, W, C, obs_out + (uint64_t)b * F);",
     "orc_hwc_to_chw_bf16(obs_ring + (s ? s - 1 : 0) * F, H, W, C, obs_out + (uint64_t)b * F);"),
    ("mm-image-of-previous", C, "orc_norm_chw_bf16(obs_ring + s * F, C, HW, mean, stdv,",
     "orc_norm_chw_bf16(obs_ring + (s ? s - 1 : 0) * F, C, HW, mean, stdv,"),
    ("normalize-mean-n-minus-1", C, "double mean = s / (double)n;",
     "double mean = s / (double)(n - 1);"),
    ("tier-hbm-window-always-full", C, "uint64_t in_hbm = total < cap_h ? total : cap_h;",
     "uint64_t in_hbm = cap_h;"),
    ("sched-iteration-max", "sched.py", "return a, b, a + b", "return a, b, max(a, b)"),
    ("sched-overlap-always", "sched.py", "    if overlap:\n", "    if True:\n"),
    ("sched-rollout-not-counted", "sched.py", "t = t_neighbour + per_unit(t_of_g, g)",
     "t = per_unit(t_of_g, g)"),
    ("place-first-candidate-skipped", "place.py", "for i, o in enumerate(opts):",
     "for i, o in list(enumerate(opts))[1:]:"),
    # the Python marshalling in front of the C oracle
    ("wrap-uniform-seed-round-swapped", "oracle.py",
     "lib().orc_sample_uniform(cap, total, n_valid, B, seed, round_,",
     "lib().orc_sample_uniform(cap, total, n_valid, B, round_, seed,"),
    ("wrap-ppo-adv-ret-swapped", "oracle.py",
     "_p(idx, C.c_int64), B, _p(adv, C.c_float),\n                          _p(ret, C.c_float),",
     "_p(idx, C.c_int64), B, _p(ret, C.c_float),\n                          _p(adv, C.c_float),"),
    ("wrap-gae-gamma-lambda-swapped", "oracle.py", "                  gamma, lam, _p(adv, C.c_double)",
     "                  lam, gamma, _p(adv, C.c_double)"),
    ("wrap-normalize-std-as-mean", "oracle.py", "return out, float(m[0]), float(s[0])",
     "return out, float(s[0]), float(m[0])"),
    ("wrap-ingest-defer-dropped", "oracle.py",
     "lib().orc_ingest_leaves(_p(st.leaves, C.c_uint32), st.cap, total, st.defer,\n"
     "                            _p(qq, C.c_uint32)",
     "lib().orc_ingest_leaves(_p(st.leaves, C.c_uint32), st.cap, total, 0,\n"
     "                            _p(qq, C.c_uint32)"),
    ("wrap-dqn-reward-as-action", "oracle.py", "_p(action, C.c_int32), _p(reward, C.c_float), cap,",
     "_p(action, C.c_int32), _p(action, C.c_float), cap,"),
    ("wrap-ring-write-rec", "oracle.py", "rec = ring.nbytes // cap", "rec = ring.nbytes // cap // ring.itemsize"),
    ("wrap-isw-beta-fixed", "oracle.py", "lib().orc_is_weights(_p(q, C.c_uint32), len(q), beta,",
     "lib().orc_is_weights(_p(q, C.c_uint32), len(q), 0.4,"),
    # group-relative advantages and packing (Python)
    ("grpo-population-std", "llm.py", "/ (n - 1) if n > 1 else 0.0", "/ n if n > 1 else 0.0"),
    ("grpo-eps-inside-sqrt", "llm.py", "den = math.sqrt(var) + float(np.float32(eps))",
     "den = math.sqrt(var + float(np.float32(eps)))"),
    ("grpo-not-centred", "llm.py", "np.float32((v - mean) / den)", "np.float32(v / den)"),
    ("pack-value-of-next", "llm.py", "vals.append(np.full(len(seg), seq_value[s] if",
     "vals.append(np.full(len(seg), seq_value[(s + 1) % n_seq] if"),
    ("pack-offsets-not-cumulative", "llm.py", "off.append(off[-1] + len(seg))",
     "off.append(len(seg))"),
    ("pack-out-of-range-wraps", "llm.py", "        if 0 <= s < n_seq:\n            seg",
     "        if True:\n            s %= n_seq\n            seg"),
    # placement model (Python)
    ("place-share-inverted", "place.py", "h = 1.0 if opt[\"mem\"] >= need else opt[\"mem\"] / need",
     "h = 1.0 if opt[\"mem\"] >= need else 1.0 - opt[\"mem\"] / need"),
    ("place-tie-last-wins", "place.py", "        if t < t_min:", "        if t <= t_min:"),
    ("place-capacity-ignored", "place.py", "    if need > mem:\n", "    if False:\n"),
    ("place-one-leg", "place.py", "return x / opt[\"bw_in\"] + leg_out", "return leg_out"),
    ("place-second-tier-ignored", "place.py",
     "mem = opt[\"mem\"] + opt[\"mem2\"] if two else opt[\"mem\"]", "mem = opt[\"mem\"]"),
    # scheduling model (Python)
    ("sched-gamma-fraction", "sched.py", "return 1.0 if g >= 1 else 1.0 - g",
     "return 1.0 if g >= 1 else g"),
    ("sched-hide-max", "sched.py", "min(t_neighbour, per_unit(t_of_g, g))",
     "max(t_neighbour, per_unit(t_of_g, g))"),
    ("sched-sync-dropped", "sched.py", "t = t + (t_sync - hide(t_neighbour, g, t_of_g, contention))",
     "t = t - hide(t_neighbour, g, t_of_g, contention)"),
    ("sched-contention-ignored", "sched.py", "return (1.0 - contention) * (", "return ("),
    ("sched-tie-last-wins", "sched.py", "if best is None or t < best[-1]:",
     "if best is None or t <= best[-1]:"),
    ("sched-per-unit-times", "sched.py", "return t_of_g / g", "return t_of_g * g"),
    ("sched-granularities-by-four", "sched.py", "        k *= 2\n", "        k *= 4\n"),
]

PIN_TESTS = sorted(glob.glob(os.path.join(ROOT, "tests", "test_oracle_*.py")))


def _tree(dst, mutant):
    """A copy of the oracle and its pin tests, with the mistake planted."""
    os.makedirs(os.path.join(dst, "oracle"))
    for f in sorted(os.listdir(os.path.join(ROOT, "oracle"))):
        if f.endswith((".py", ".c")):
            shutil.copy(os.path.join(ROOT, "oracle", f), os.path.join(dst, "oracle", f))
    os.makedirs(os.path.join(dst, "tests"))
    for f in PIN_TESTS + [os.path.join(ROOT, "tests", "conftest.py")]:
        shutil.copy(f, os.path.join(dst, "tests"))
    shutil.copytree(os.path.join(ROOT, "tests", "golden"), os.path.join(dst, "tests", "golden"))
    shutil.copy(os.path.join(ROOT, "pytest.ini"), dst)
    if mutant is None:
        return
    _, fname, old, new = mutant
    path = os.path.join(dst, "oracle", fname)
    src = open(path).read()
    assert src.count(old) == 1, "%s: the text to mutate must occur once" % mutant[0]
    open(path, "w").write(src.replace(old, new))


def _run(base, mutant):
    name = "unmodified" if mutant is None else mutant[0]
    dst = os.path.join(base, name)
    _tree(dst, mutant)
    env = dict(os.environ, OMP_NUM_THREADS="1", PYTHONDONTWRITEBYTECODE="1")
    env.pop("PYTHONPATH", None)
    # build first, so a mutant that does not compile is reported as such
    b = subprocess.run([sys.executable, "-c", "import oracle; oracle.lib()"],
                       cwd=dst, env=env, capture_output=True, text=True, timeout=300)
    if b.returncode != 0:
        return name, "build", b.returncode, b.stdout[-2000:] + b.stderr[-2000:]
    p = subprocess.run([sys.executable, "-m", "pytest", "tests", "-x", "-q", "-m", "not gpu"],
                       cwd=dst, env=env, capture_output=True, text=True, timeout=600)
    return name, "pins", p.returncode, p.stdout[-3000:] + p.stderr[-1000:]


@pytest.fixture(scope="module")
def runs(tmp_path_factory):
    base = str(tmp_path_factory.mktemp("mutants"))
    jobs = [None] + MUTANTS
    with ThreadPoolExecutor(max_workers=max(1, min(8, os.cpu_count() or 1))) as ex:
        res = list(ex.map(lambda m: _run(base, m), jobs))
    return {r[0]: r[1:] for r in res}


def test_names_are_unique():
    names = [m[0] for m in MUTANTS]
    assert len(names) == len(set(names))


def test_unmodified_copy_passes(runs):
    stage, rc, out = runs["unmodified"]
    assert (stage, rc) == ("pins", 0), out


@pytest.mark.parametrize("name", [m[0] for m in MUTANTS])
def test_pins_catch_mutant(runs, name):
    stage, rc, out = runs[name]
    assert stage == "pins", "mutant does not build:\n" + out
    # 1: a pin failed (not a crash, a collection error or an interrupt)
    assert rc == 1, "no pin caught %s (pytest exit %d):\n%s" % (name, rc, out)
