"""Mutation check of the oracle's pins (run by hand: ``python tests/oracle_mutants.py``).

Each mutant below is a plausible one-token mistake in the float64 oracle -- a
dropped term, a wrong sign or index, an off-by-one, a wrong tie rule.  For
every mutant the script copies the repository's ``oracle/``, ``tests/`` and
the Python package into a temporary directory, applies the mistake to the
copy of the oracle (never to the repository), and runs the oracle's pin tests
(``tests/test_oracle_*.py``, CPU only).  A mutant is *caught* when at least
one pin fails (a per-test timeout counts: a mistake that makes the oracle
loop forever fails that way).  The script prints one line per mutant with the
pins that caught it and exits non-zero if any mutant survives.

Not collected by pytest (the file name does not start with ``test_``): it
runs the whole pin suite once per mutant, about a quarter of an hour on 8
cores (the chi-square losslessness pins take most of it).
"""

import concurrent.futures as cf
import glob
import os
import shutil
import subprocess
import sys
import tempfile

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

# (oracle file, snippet, replacement, what the mistake is)
MUTANTS = [
 # tree
 ("tree.py", "                if j != -1:\n                    edges += 1", "                edges += 1", "depth counts the root edge (off by one)"),
 ("tree.py", "            pos[b, i] = prefix_len[b] + edges", "            pos[b, i] = prefix_len[b] + edges + 1", "pos one too far"),
 ("tree.py", "            pos[b, i] = prefix_len[b] + edges", "            pos[b, i] = edges", "pos without the prefix"),
 ("tree.py", "                bits |= 1 << j\n                j = int(parents[b, j])", "                j = int(parents[b, j])\n                if j != -1: bits |= 1 << j", "ancestor set without self"),
 ("tree.py", "        if p < 0 or p >= i:", "        if p < 0 or p > i:", "validity allows self-parent"),
 # rope
 ("attention.py", "    out[..., :half] = lo * c - hi * s", "    out[..., :half] = lo * c + hi * s", "rope sign flipped (low half)"),
 ("attention.py", "    out[..., half:] = hi * c + lo * s", "    out[..., half:] = hi * c - lo * s", "rope sign flipped (high half)"),
 ("attention.py", "    theta = np.power(float(base), -2.0 * j / d)", "    theta = np.power(float(base), -1.0 * j / d)", "rope frequency exponent -j/d"),
 ("attention.py", "    theta = np.power(float(base), -2.0 * j / d)", "    theta = np.power(float(base), -2.0 * (j + 1) / d)", "rope frequency index shifted"),
 ("attention.py", "    c = np.cos(ang)[:, None, :]\n    s = np.sin(ang)[:, None, :]", "    s = np.cos(ang)[:, None, :]\n    c = np.sin(ang)[:, None, :]", "rope cos and sin swapped"),
 # attention
 ("attention.py", "    scale = 1.0 / np.sqrt(d)", "    scale = 1.0", "no softmax scale"),
 ("attention.py", "                s_tree = np.where(allowed, s_tree, -np.inf)", "                pass", "no tree mask"),
 ("attention.py", "                s_tree = (Q @ kr[:, g, :].T) * scale", "                s_tree = (Q @ k_new[b, :, g, :].T) * scale", "tree keys unrotated"),
 ("attention.py", "            Kp = np.asarray(cacheK[b, g, :P, :], dtype=np.float64)", "            Kp = np.asarray(cacheK[b, g, :max(P - 1, 0), :], dtype=np.float64)", "prefix keys one short"),
 ("attention.py", "                h = g * G + hl", "                h = hl * Hkv + g", "GQA head mapping interleaved"),
 ("attention.py", "        qr = rope_rotate(q[b], pos[b], rope_base)", "        qr = np.asarray(q[b], dtype=np.float64)", "queries unrotated"),
 ("attention.py", "            allowed[i, ancestor_list(anc[b, i], N)] = True", "            allowed[i, :i + 1] = True", "causal mask instead of the ancestor mask"),
 ("attention.py", "                out[b, :, h, :] = p[:, :P] @ Vp + p[:, P:] @ v_new[b, :, g, :]", "                out[b, :, h, :] = p[:, :P] @ Vp", "tree values dropped"),
 ("attention.py", "            treeV[b, g] = v_new[b, :, g, :]", "            treeV[b, g] = kr[:, g, :]", "tree V scratch holds keys"),
 # lm head
 ("lmhead.py", "        best = int(np.argmax(logits[r]))", "        best = int(len(logits[r]) - 1 - np.argmax(logits[r][::-1]))", "argmax ties toward the highest id"),
 ("lmhead.py", "    order = np.argsort(-logits, axis=1, kind=\"stable\")[:, :k]", "    order = np.argsort(-logits, axis=1, kind=\"stable\")[:, 1:k + 1]", "top-k drops the best"),
 ("lmhead.py", "    order = np.argsort(-logits, axis=1, kind=\"stable\")[:, :k]", "    order = (logits.shape[1] - 1 - np.argsort(-logits[:, ::-1], axis=1, kind=\"stable\"))[:, :k]", "top-k ties toward the higher id"),
 ("lmhead.py", "    lse = m + np.log(np.exp(logits - m[:, None]).sum(axis=1))", "    lse = np.log(np.exp(logits - m[:, None]).sum(axis=1))", "log-sum-exp without the max"),
 ("lmhead.py", "    return np.asarray(h, dtype=np.float64) @ np.asarray(W, dtype=np.float64).T", "    return np.asarray(h, dtype=np.float64) @ np.asarray(W, dtype=np.float64)[:, ::-1].T", "LM head hidden index reversed"),
 # greedy acceptance
 ("accept.py", "            if ok and len(chains[i]) > len(chains[best]):", "            if ok and len(chains[i]) >= len(chains[best]):", "greedy ties toward the largest index"),
 ("accept.py", "            ok = all(int(tokens[b, j]) == int(choice[b, parents[b, j]]) for j in chains[i][1:])", "            ok = all(int(tokens[b, j]) == int(choice[b, j]) for j in chains[i][1:])", "match against the node's own choice"),
 ("accept.py", "            ok = all(int(tokens[b, j]) == int(choice[b, parents[b, j]]) for j in chains[i][1:])", "            ok = int(tokens[b, chains[i][-1]]) == int(choice[b, parents[b, chains[i][-1]]]) if i else True", "only the last edge checked"),
 ("accept.py", "        out_tokens[b] = _pad([int(tokens[b, j]) for j in p[1:]] + [int(choice[b, best])], D + 1)", "        out_tokens[b] = _pad([int(tokens[b, j]) for j in p[1:]] + [int(choice[b, p[-2] if len(p) > 1 else best])], D + 1)", "bonus token from the parent's choice"),
 ("accept.py", "        if max(len(c) for c in chains) - 1 > D:", "        if max(len(c) for c in chains) > D:", "depth bound off by one"),
 # compaction
 ("compact.py", "                    cacheK[layer, b, h, P + t, :] = treeK[layer, b, h, src, :]", "                    cacheK[layer, b, h, P + t - 1, :] = treeK[layer, b, h, src, :]", "compaction one row early (K)"),
 ("compact.py", "                    cacheV[layer, b, h, P + t, :] = treeV[layer, b, h, src, :]", "                    cacheV[layer, b, h, P + t, :] = treeV[layer, b, h, t, :]", "compaction copies tree rows in node order (V)"),
 ("compact.py", "        if P + n > S_max:", "        if P + n >= S_max:", "capacity check off by one"),
 ("compact.py", "        new_len[b] = P + n", "        new_len[b] = P + n - 1", "new length one short"),
]



def run(idx, base):
    fname, old, new, desc = MUTANTS[idx]
    d = os.path.join(base, f"m{idx}")
    os.makedirs(d)
    ign = shutil.ignore_patterns("_build", "__pycache__", "*.so", "*.o")
    for sub in ("oracle", "tests", "paper_2502_11018_gb300"):
        shutil.copytree(os.path.join(ROOT, sub), os.path.join(d, sub), ignore=ign)
    path = os.path.join(d, "oracle", fname)
    text = open(path).read()
    if text.count(old) != 1:
        return idx, "ANCHOR MISSING", []
    open(path, "w").write(text.replace(old, new))
    pins = sorted(glob.glob(os.path.join(d, "tests", "test_oracle_*.py")))
    r = subprocess.run([sys.executable, "-m", "pytest", *pins, "-q", "-m", "not gpu", "-p", "no:cacheprovider",
                        "--tb=no", "--timeout=60"], cwd=d, capture_output=True, text=True)
    failed = [ln.split()[1] for ln in r.stdout.splitlines() if ln.startswith("FAILED")]
    shutil.rmtree(d)
    return idx, ("caught" if failed else "SURVIVED"), failed


def main():
    base = tempfile.mkdtemp(prefix="oracle_mutants_")
    survived = 0
    try:
        with cf.ThreadPoolExecutor(max(1, min(8, os.cpu_count() or 1))) as ex:
            for idx, res, failed in ex.map(lambda i: run(i, base), range(len(MUTANTS))):
                fname, _, _, desc = MUTANTS[idx]
                names = sorted({f.split("::")[-1].split("[")[0] for f in failed})
                print(f"{idx:2d} {fname:13s} {res:8s} {desc}: {len(failed)} failing pins ({', '.join(names[:4])})")
                survived += res != "caught"
    finally:
        shutil.rmtree(base, ignore_errors=True)
    print(f"{len(MUTANTS) - survived} of {len(MUTANTS)} mutants caught")
    return 1 if survived else 0


if __name__ == "__main__":
    sys.exit(main())
