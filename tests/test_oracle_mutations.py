"""Planted mistakes in the oracle must fail its pins.

Each case copies the oracle, the tests and the package's Python files into a temporary directory. It then plants
one plausible mistake in the copied oracle: a flipped comparison, a reversed order, a dropped offset or term, a
wrong index or operator. The oracle's pin tests run against the copy in a fresh interpreter. The pins are strong
enough only if every planted mistake makes at least one of them fail. Nothing here touches the GPU or the CUDA
library.
"""
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

PINS = ["tests/test_oracle_pins.py"]
LSH = ["tests/test_oracle_lsh.py"]
ENS = ["tests/test_oracle_ensemble.py"]
CAL = ["tests/test_oracle_calibration.py"]
SPEC = ["tests/test_oracle_speculative.py"]
SHARDS = ["tests/test_oracle_shards.py"]

# (id, oracle file, text, planted replacement, pin files that must catch it)
MUTATIONS = [
    ("key-threshold-exclusive", "lookup.py", "ok[b] & (s[b] >= self.tau_c)", "ok[b] & (s[b] > self.tau_c)", PINS),
    ("ties-by-id-descending", "lookup.py", "np.lexsort((j, -s))", "np.lexsort((-j, -s))", PINS),
    ("candidates-ascending", "lookup.py", "np.lexsort((j, -s))", "np.lexsort((j, s))", PINS),
    ("block-offset-dropped", "lookup.py", "self.add_scores(self.q @ K.T, j0)", "self.add_scores(self.q @ K.T, 0)",
     PINS),
    ("best-score-minimum", "lookup.py", "np.where(ok, s, -np.inf).max(axis=1)", "np.where(ok, s, np.inf).min(axis=1)",
     PINS),
    ("lookahead-threshold-exclusive", "lookup.py", "emb_ok = r >= params.tau_a", "emb_ok = r > params.tau_a", PINS),
    ("token-threshold-exclusive", "lookup.py", "tok_ok = m >= tmin", "tok_ok = m > tmin", PINS),
    ("both-mode-is-or", "lookup.py", "return emb_ok & tok_ok", "return emb_ok | tok_ok", PINS),
    ("token-positions-reversed", "lookup.py", "np.asarray(t_ids, dtype=np.int64)[None, :]",
     "np.asarray(t_ids, dtype=np.int64)[None, ::-1]", PINS),
    ("prefix-check-reads-key-rows", "lookup.py", "lambda j: store.prefix[j], lambda j: store.ids[j])",
     "lambda j: store.key[j], lambda j: store.ids[j])", PINS),
    ("last-passing-served", "lookup.py", "served = int(hits[0])", "served = int(hits[-1])", PINS),
    ("hit-key-score-of-top-candidate", "lookup.py", "res.key_score[b] = cs[served]", "res.key_score[b] = cs[0]",
     PINS),
    ("candidate-cut-off-by-one", "lookup.py", "nc = min(c, n_above)", "nc = min(c - 1, n_above)", PINS),
    ("shown-prefix-score-of-top-candidate", "lookup.py", "res.prefix_score[b] = r[shown]",
     "res.prefix_score[b] = r[0]", PINS),
    ("margin-drops-threshold-gap", "lookup.py", "gaps.append(cs[served] - tau_c)",
     "gaps.append(np.inf)", PINS),
    ("literal-margin-drops-top-two-gap", "lookup.py", "lit.append(s_sorted[0] - s_sorted[1])", "pass", PINS),
    ("literal-margin-drops-threshold-distance", "lookup.py",
     "lit = [abs(kc.best[b] - tau_c)] if np.isfinite(kc.best[b]) else []", "lit = []", PINS),
    ("margin-push-out-only-from-the-last-slot", "lookup.py",
     "            if n_above > c:\n                # j* pushed past the cut",
     "            if n_above > c and served == c - 1:\n                # j* pushed past the cut", PINS),
    ("margin-ignores-later-failing-candidates", "lookup.py",
     "gaps.append(max(cs[served] - cs[i], flip(rm[i], m[i])))", "pass", PINS),
    ("margin-ignores-entries-below-threshold", "lookup.py", "gaps.append(cs[-1] - kc.below[b])",
     "gaps.append(np.inf)", PINS),
    ("margin-ignores-entries-past-the-cut", "lookup.py",
     "gaps.append(key if oke[t] else max(key, flip(rme[t], me[t])))", "pass", PINS),
    ("margin-past-the-cut-all-passing", "lookup.py",
     "gaps.append(key if oke[t] else max(key, flip(rme[t], me[t])))", "gaps.append(key)", PINS),
    ("below-threshold-best-of-all-scores", "lookup.py", "np.where(ok & (s < self.tau_c), s, -np.inf)",
     "np.where(ok, s, -np.inf)", PINS),
    ("ensemble-any-model-passes", "lookup.py", "emb_ok = np.all(r >= np.array(", "emb_ok = np.any(r >= np.array(",
     ENS),
    ("ensemble-thresholds-reversed", "lookup.py", "np.array([t for _, _, t in segments])[None, :]",
     "np.array([t for _, _, t in segments])[None, ::-1]", ENS),
    ("miss-key-score-minus-infinity", "lookup.py", "key_score=kc.best.copy()", "key_score=np.full(B, -np.inf)",
     PINS),
    ("reject-shows-last-candidate", "lookup.py", "shown = int(hits[0]) if hits.size else 0",
     "shown = int(hits[0]) if hits.size else nc - 1", PINS),
    ("token-mismatches-counted", "lookup.py", "== np.asarray(t_ids, dtype=np.int64)[None, :]).sum(axis=1)",
     "!= np.asarray(t_ids, dtype=np.int64)[None, :]).sum(axis=1)", PINS),
    ("prefix-score-negated", "lookup.py", "        r = P @ p\n", "        r = -(P @ p)\n", PINS),
    ("widen-shift-15", "bf16.py", "<< np.uint32(16)", "<< np.uint32(15)", PINS),
    ("rounding-ties-away", "bf16.py", "((dropped == half) & ((kept & np.uint64(1)) == np.uint64(1)))",
     "(dropped == half)", PINS),
    ("nan-not-quieted", "bf16.py", "r = np.where(is_nan, kept | np.uint64(0x0040), r)", "r = np.where(is_nan, kept, r)",
     PINS),
    ("hyperplanes-reversed", "lsh.py", "widen(rows_bits) @ widen(hyperplanes_bits).T",
     "widen(rows_bits) @ widen(hyperplanes_bits)[::-1].T", LSH),
    ("signature-sign-strict", "lsh.py", "return p >= 0.0, np.abs(p) < amb", "return p > 0.0, np.abs(p) < amb", LSH),
    ("hamming-drops-factor-two", "lsh.py", "- 2 * (a @ b.T)", "- (a @ b.T)", LSH),
    ("radius-exclusive", "lsh.py", "admitted=hd <= self.radius", "admitted=hd < self.radius", LSH),
    ("lsh-block-offset-dropped", "lsh.py", "self.kc.add_scores(s, j0,", "self.kc.add_scores(s, 0,", LSH),
    ("ambiguity-ignores-query-bits", "lsh.py", "slack = self.q_amb.sum(axis=1)[:, None] +",
     "slack = 0 * self.q_amb.sum(axis=1)[:, None] +", LSH),
    ("nearest-rank-floor", "calibrate.py", "math.ceil(percentile / 100.0 * v.size)",
     "math.floor(percentile / 100.0 * v.size)", CAL),
    ("cap-is-max", "calibrate.py", "return min(cap, p), p", "return max(cap, p), p", CAL),
    ("acceptance-strict", "speculative.py", "pf[b, n] >= pg[b, n]", "pf[b, n] > pg[b, n]", SPEC),
    ("served-queries-verified", "speculative.py", "out[np.asarray(status) == HIT] = -1",
     "out[np.asarray(status) == HIT] = out[np.asarray(status) == HIT]", SPEC),
    ("serve-loop-appends-hits", "serve.py", "miss = np.nonzero(res.status != HIT)[0]",
     "miss = np.nonzero(res.status == HIT)[0]", PINS),
    ("merge-ties-by-id-descending", "shards.py", "pool.sort(key=lambda e: (-e[0], e[1]))",
     "pool.sort(key=lambda e: (-e[0], -e[1]))", SHARDS),
    ("merge-drops-shard-base", "shards.py", "base + int(res.cand_id[b, i])", "int(res.cand_id[b, i])", SHARDS),
    ("merge-counts-last-shard-only", "shards.py", "out.n_above[b] += res.n_above[b]", "out.n_above[b] = res.n_above[b]",
     SHARDS),
    ("merge-best-from-key-scores", "shards.py",
     "best = max(best, res.cand_score[b, 0] if nc else res.key_score[b])", "best = max(best, res.key_score[b])",
     SHARDS),
]


def _copy_tree(dst: str) -> None:
    skip = shutil.ignore_patterns("__pycache__", "_build", "csrc", "c_client", "*.so", "*.o")
    for name in ("oracle", "tests", "paper_2608_01718_gb300"):
        shutil.copytree(os.path.join(ROOT, name), os.path.join(dst, name), ignore=skip)


@pytest.mark.parametrize("name,path,text,planted,pins", MUTATIONS, ids=[m[0] for m in MUTATIONS])
def test_planted_mistake_fails_a_pin(tmp_path, name, path, text, planted, pins):
    dst = str(tmp_path)
    _copy_tree(dst)
    target = os.path.join(dst, "oracle", path)
    with open(target) as f:
        src = f.read()
    assert src.count(text) == 1, f"{name}: the text to replace must occur exactly once in oracle/{path}"
    with open(target, "w") as f:
        f.write(src.replace(text, planted))
    env = dict(os.environ, PYTHONDONTWRITEBYTECODE="1")
    run = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider", *pins],
                         cwd=dst, env=env, capture_output=True, text=True, timeout=600)
    out = run.stdout + run.stderr
    assert run.returncode == 1 and " failed" in out, f"{name} was not caught by {pins}:\n{out[-2000:]}"


def test_unmutated_copy_passes_the_pins(tmp_path):
    """The harness itself: the same copy without a planted mistake passes every pin file."""
    dst = str(tmp_path)
    _copy_tree(dst)
    files = sorted({f for m in MUTATIONS for f in m[4]})
    run = subprocess.run([sys.executable, "-m", "pytest", "-q", "-p", "no:cacheprovider", *files], cwd=dst,
                         env=dict(os.environ, PYTHONDONTWRITEBYTECODE="1"), capture_output=True, text=True,
                         timeout=600)
    assert run.returncode == 0, (run.stdout + run.stderr)[-2000:]
