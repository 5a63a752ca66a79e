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
runs the whole pin suite once per mutant, about twenty minutes on 8 cores
(the chi-square losslessness pins take most of it).
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
 # temperature sampling acceptance
 ("accept.py", "    return np.maximum(p - q, 0.0)", "    return np.abs(p - q)", "residual |p - q| instead of max(p - q, 0)"),
 ("accept.py", "                ratio = p[x] / qx\n                min_margin", "                ratio = qx / max(p[x], 1e-300)\n                min_margin", "acceptance ratio inverted"),
 ("accept.py", "                if s > 0.0:\n                    p = r / s\n            if nxt is None:", "                if s > 0.0:\n                    p = r\n            if nxt is None:", "residual not renormalised"),
 ("accept.py", "            for c in _children(parents[b], u):\n                x = int(tokens[b, c])\n                qx = 1.0 if q is None else q[x]\n                if qx == 0.0:", "            for c in reversed(_children(parents[b], u)):\n                x = int(tokens[b, c])\n                qx = 1.0 if q is None else q[x]\n                if qx == 0.0:", "children tried in decreasing index order"),
 ("accept.py", "    z = np.asarray(x, dtype=np.float64) / T", "    z = np.asarray(x, dtype=np.float64)", "temperature ignored"),
 ("accept.py", "                v, m = _inverse_cdf(p, float(u_res[b, u]))", "                v, m = _inverse_cdf(_softmax(target_logits[b, u], temperature), float(u_res[b, u]))", "bonus drawn from the target, not the residual"),
 # training objective
 ("tat.py", "        out[r] = 1 if ahead < k else 0", "        out[r] = 1 if ahead <= k else 0", "predictable mask top-(k+1)"),
 ("tat.py", "((logits[r] == lx) & (ids < x))", "((logits[r] == lx) & (ids > x))", "predictable mask tie rule reversed"),
 ("tat.py", "        out[r] = lse - logits[r, int(tokens[r])]", "        out[r] = lse - logits[r].max()", "token loss against the argmax"),
 ("tat.py", "        lse = m + np.log(np.exp(logits[r] - m).sum())", "        lse = np.log(np.exp(logits[r] - m).sum())", "token loss log-sum-exp without the max"),
 ("tat.py", "    return np.abs(fd - ft).sum(axis=1)", "    return ((fd - ft) ** 2).sum(axis=1)", "feature loss squared, not L1"),
 ("tat.py", "                v *= int(mbar_prev[j - 1][b][t - n + j])", "                v *= int(mbar_prev[j - 1][b][t - n + j + 1])", "alignment chain shifted by one position"),
 ("tat.py", "            if t - n + 1 < 0:", "            if t - n < 0:", "alignment start bound off by one"),
 ("tat.py", "    ell = (lam_tok * token_loss(rows_logits, rows_tok)\n           + lam_feat * feature_loss(", "    ell = (lam_feat * token_loss(rows_logits, rows_tok)\n           + lam_tok * feature_loss(", "loss weights swapped"),
 ("tat.py", "        seq_loss[b] = num / den if den > 0 else 0.0", "        seq_loss[b] = num / T if den > 0 else 0.0", "pass loss divided by the length, not the mask sum"),
 # decoder layer
 ("layer.py", "    ms = (x * x).mean(axis=1, keepdims=True)", "    ms = (x * x).sum(axis=1, keepdims=True)", "RMSNorm over the sum, not the mean"),
 ("layer.py", "    return z / (1.0 + np.exp(-z))", "    return 1.0 / (1.0 + np.exp(-z))", "sigmoid instead of silu"),
 ("layer.py", "    return silu(linear(x, Wg)) * linear(x, Wu)", "    return linear(x, Wg) * silu(linear(x, Wu))", "silu on the up projection"),
 ("layer.py", "    h = h + linear(o.reshape(B * N, Hq * d), w[\"Wo\"])", "    h = linear(o.reshape(B * N, Hq * d), w[\"Wo\"])", "attention residual dropped"),
 ("layer.py", "    x = rmsnorm(h, w[\"mlp_norm\"], eps)", "    x = rmsnorm(h, w[\"attn_norm\"], eps)", "MLP norm with the attention norm's gain"),
 ("layer.py", "    k = linear(x, w[\"Wk\"]).reshape(B, N, Hkv, d)", "    k = linear(x, w[\"Wv\"]).reshape(B, N, Hkv, d)", "keys projected with Wv"),
 # Token-Guided Fusion
 ("tgf.py", "    var = ((x - mu) ** 2).mean(axis=1, keepdims=True)", "    var = ((x - mu) ** 2).sum(axis=1, keepdims=True) / (x.shape[1] - 1)", "layer norm with the sample variance"),
 ("tgf.py", "    h = linear(np.concatenate([F, x], axis=1), w[\"Wm\"]) + w[\"bm\"]", "    h = linear(np.concatenate([x, F], axis=1), w[\"Wm\"]) + w[\"bm\"]", "Eq. 6 concatenation order swapped"),
 ("tgf.py", "    o = linear(silu(z), w[\"Wd\"]) + w[\"bd\"] + h", "    o = linear(silu(z), w[\"Wd\"]) + w[\"bd\"]", "Eq. 8 residual dropped"),
 ("tgf.py", "layernorm(h, w[\"g_h\"], w[\"b_h\"], eps)", "layernorm(h, w[\"g_x\"], w[\"b_x\"], eps)", "Eq. 7 norm of h with the token norm's gain"),
 ("tgf.py", "    z = linear(zin, w[\"Wu\"]) + w[\"bu\"]", "    z = linear(zin, w[\"Wu\"])", "Eq. 7 bias dropped"),
 # draft tree
 ("draft_tree.py", "            pool[\"score\"].append(pool[\"score\"][pid] + lp[t])", "            pool[\"score\"].append(pool[\"score\"][pid] + np.exp(lp[t]))", "scores add probabilities, not log-probabilities"),
 ("draft_tree.py", "            pool[\"score\"].append(pool[\"score\"][pid] + lp[t])", "            pool[\"score\"].append(lp[t])", "scores not cumulative"),
 ("draft_tree.py", "    order = np.lexsort((np.arange(x.size), -x))", "    order = np.lexsort((-np.arange(x.size), -x))", "expansion top-k ties toward the higher id"),
 ("draft_tree.py", "    order = np.lexsort((np.array(ids), -sc))", "    order = np.lexsort((-np.array(ids), -sc))", "selection ties toward the later pool node"),
 ("draft_tree.py", "    kept, gap = best(pool, range(1, len(pool[\"token\"])), N - 1)", "    kept, gap = best(pool, range(1, len(pool[\"token\"])), N - 2)", "rerank keeps one node too few"),
 # indexing across layers and sequences
 ("attention.py", "            Kp = np.asarray(cacheK[b, g, :P, :], dtype=np.float64)", "            Kp = np.asarray(cacheK[0, g, :P, :], dtype=np.float64)", "every sequence reads sequence 0's prefix keys"),
 ("compact.py", "        for layer in range(L):", "        for layer in range(1):", "only the first layer committed"),
 ("tree.py", "                anc[b, i] = np.uint64(1) << np.uint64(i)", "                anc[b, i] = np.uint64(1)", "an invalid tree's nodes all see the root"),
 # the step composition
 ("step.py", "                                   as_f64(inp.v_new[layer]), as_f64(inp.cacheK[layer]),", "                                   as_f64(inp.v_new[layer]), as_f64(inp.cacheK[0]),", "every layer reads layer 0's key cache"),
 ("step.py", "        o, tk, tv = tree_attention(as_f64(inp.q[layer]),", "        o, tk, tv = tree_attention(as_f64(inp.q[L - 1 - layer]),", "layers' queries in reverse order"),
 ("step.py", "                                   as_f64(inp.cacheV[layer]), prefix_len, pos, anc,", "                                   as_f64(inp.cacheV[layer]), prefix_len, depth, anc,", "RoPE at depths, not positions"),
 ("step.py", "                                          path, alen, prefix_len, st)", "                                          path, alen, prefix_len + 1, st)", "commit one row late"),
 ("step.py", "        ck, cv, new_len, st2 = kv_compact(np.stack(treeK), np.stack(treeV),", "        ck, cv, new_len, st2 = kv_compact(np.stack(treeK[::-1]), np.stack(treeV),", "keys committed into the wrong layers"),
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
    # One thread per run: parallel runs with a full BLAS / OpenMP pool each
    # oversubscribe the cores badly enough to time out fast tests.
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1")
    r = subprocess.run([sys.executable, "-m", "pytest", *pins, "-q", "-m", "not gpu", "-p", "no:cacheprovider",
                        "--tb=no", "--timeout=120"], cwd=d, capture_output=True, text=True, env=env)
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
