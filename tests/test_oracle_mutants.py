"""The oracle's pins catch plausible mistakes.  Each case below plants one mistake in a copy of the
oracle's C++ source (a dropped term, a wrong sign, a swapped index or operand, a transposed weight,
a rule applied one step off), builds that copy on the CPU and runs the oracle's pin tests
(tests/test_oracle.py) against it: every mutant must fail at least one of them, and the unmodified
copy must pass them all.  Nothing here touches the CUDA library or a GPU.
"""
import concurrent.futures as cf
import os
import re
import shutil
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

# (name, file, original text, planted text, occurrence: 0 = the only one, k = the k-th of several)
MUTANTS = [
    # propagation forward (Eq. 1 with per-type weights and biases)
    ("fwd: W_p transposed", "oracle.cpp",
     "s += E[(size_t)u * H + hi] * W[((size_t)p * H + hi) * H + ho];",
     "s += E[(size_t)u * H + hi] * W[((size_t)p * H + ho) * H + hi];", 0),
    ("fwd: bias dropped", "oracle.cpp",
     "double s = b ? b[(size_t)p * H + ho] : 0.0;", "double s = 0.0;", 0),
    ("fwd: message sent against the edge", "oracle.cpp",
     "const double* m = &M[((size_t)e_type[e] * N + e_src[e]) * H];\n"
     "    double* y = &Y[(size_t)e_dst[e] * H];",
     "const double* m = &M[((size_t)e_type[e] * N + e_dst[e]) * H];\n"
     "    double* y = &Y[(size_t)e_src[e] * H];", 0),
    ("fwd: edge type ignored", "oracle.cpp",
     "const double* m = &M[((size_t)e_type[e] * N + e_src[e]) * H];",
     "const double* m = &M[((size_t)0 * N + e_src[e]) * H];", 0),
    ("fwd: messages averaged over types", "oracle.cpp",
     "for (int32_t h = 0; h < H; ++h) y[h] += m[h];",
     "for (int32_t h = 0; h < H; ++h) y[h] += m[h] / P;", 0),
    # propagation backward
    ("bwd: dE with W_p instead of W_p^T", "oracle.cpp",
     "for (int32_t ho = 0; ho < H; ++ho) s += g[ho] * W[((size_t)p * H + hi) * H + ho];",
     "for (int32_t ho = 0; ho < H; ++ho) s += g[ho] * W[((size_t)p * H + ho) * H + hi];", 0),
    ("bwd: dW_p transposed", "oracle.cpp",
     "dW[((size_t)p * H + hi) * H + ho] += E[(size_t)u * H + hi] * g[ho];",
     "dW[((size_t)p * H + hi) * H + ho] += E[(size_t)u * H + ho] * g[hi];", 0),
    ("bwd: db dropped", "oracle.cpp",
     "for (int32_t ho = 0; ho < H; ++ho) db[(size_t)p * H + ho] += g[ho];",
     "for (int32_t ho = 0; ho < H; ++ho) db[(size_t)p * H + ho] += 0.0 * g[ho];", 0),
    ("bwd: gradient gathered along the edge", "oracle.cpp",
     "double* g = &dM[((size_t)e_type[e] * N + e_src[e]) * H];\n"
     "    const double* y = &dY[(size_t)e_dst[e] * H];",
     "double* g = &dM[((size_t)e_type[e] * N + e_dst[e]) * H];\n"
     "    const double* y = &dY[(size_t)e_src[e] * H];", 0),
    # GRU forward (reading c4)
    ("gru: reset gate outside the hidden term", "oracle.cpp",
     "double nn = std::tanh(gi[2 * H + h] + r * gh[2 * H + h]);",
     "double nn = std::tanh(r * (gi[2 * H + h] + gh[2 * H + h]));", 1),
    ("gru: z and 1 - z swapped", "oracle.cpp",
     "Hn[(size_t)i * H + h] = (1.0 - z) * nn + z * Hs[(size_t)i * H + h];",
     "Hn[(size_t)i * H + h] = z * nn + (1.0 - z) * Hs[(size_t)i * H + h];", 0),
    ("gru: r and z gate rows swapped", "oracle.cpp",
     "double r = sigmoid(gi[h] + gh[h]);\n      double z = sigmoid(gi[H + h] + gh[H + h]);\n"
     "      double nn = std::tanh(gi[2 * H + h] + r * gh[2 * H + h]);\n"
     "      Hn[",
     "double z = sigmoid(gi[h] + gh[h]);\n      double r = sigmoid(gi[H + h] + gh[H + h]);\n"
     "      double nn = std::tanh(gi[2 * H + h] + r * gh[2 * H + h]);\n"
     "      Hn[", 0),
    ("gru: W_ih transposed", "oracle.cpp",
     "a += W_ih[(size_t)o * H + h] * X[(size_t)i * H + h];",
     "a += W_ih[(size_t)h * 3 * H + o] * X[(size_t)i * H + h];", 0),
    ("gru: padding rows not zeroed", "oracle.cpp",
     "for (int32_t h = 0; h < H; ++h) Hn[(size_t)i * H + h] = 0.0;\n      continue;",
     "(void)0;", 0),
    # GRU backward (hand-derived)
    ("gru bwd: r missing from the hidden n-gate gradient", "oracle.cpp",
     "dgh[2 * H + h] = dan * r;", "dgh[2 * H + h] = dan;", 0),
    ("gru bwd: dz sign", "oracle.cpp",
     "double dz = g * (hs[h] - nn);", "double dz = g * (nn - hs[h]);", 0),
    ("gru bwd: direct state path dropped", "oracle.cpp",
     "dh[h] = g * z;", "dh[h] = 0.0 * g * z;", 0),
    ("gru bwd: tanh derivative", "oracle.cpp",
     "double dan = dn * (1.0 - nn * nn);", "double dan = dn * (1.0 - nn);", 0),
    ("gru bwd: sigmoid derivative of r", "oracle.cpp",
     "double dar = dr * r * (1.0 - r);", "double dar = dr * r;", 0),
    ("gru bwd: dW_hh against the input instead of the state", "oracle.cpp",
     "dW_hh[(size_t)o * H + h] += dgh[o] * hs[h];", "dW_hh[(size_t)o * H + h] += dgh[o] * x[h];",
     0),
    # GGNN steps
    ("ggnn bwd: direct state gradient dropped between steps", "oracle.cpp",
     "for (size_t i = 0; i < NH; ++i) g[i] = dHs[i] + dEp[i];",
     "for (size_t i = 0; i < NH; ++i) g[i] = dEp[i];", 0),
    ("ggnn bwd: weight gradient of one step only", "oracle.cpp",
     "for (size_t i = 0; i < dWt.size(); ++i) dW[i] += dWt[i];",
     "for (size_t i = 0; i < dWt.size(); ++i) dW[i] = dWt[i];", 0),
    ("ggnn fwd: messages from the initial state at every step", "oracle.cpp",
     "orc_propagate_fwd(N, P, H, n_edges, e_dst, e_src, e_type, Es + t * NH, W, b, Ys + t * NH);",
     "orc_propagate_fwd(N, P, H, n_edges, e_dst, e_src, e_type, Es, W, b, Ys + t * NH);", 0),
    # RCM (reading c8)
    ("rcm: Cuthill-McKee order not reversed", "oracle.cpp",
     "std::reverse(order.begin(), order.end());", "(void)0;", 0),
    ("rcm: ties broken by descending id", "oracle.cpp",
     "return da != db ? da < db : a < b;", "return da != db ? da < db : a > b;", 0),
    ("rcm: neighbours by descending degree", "oracle.cpp",
     "return da != db ? da < db : a < b;", "return da != db ? da > db : a < b;", 0),
    ("rcm: no pseudo-peripheral search", "oracle.cpp",
     "if (lx.size() > levels.size()) {", "if (false && lx.size() > levels.size()) {", 0),
    ("rcm: keep-if-better inverted", "oracle.cpp",
     "if (orc_bandwidth(n, m, src, dst, pos.data()) > orc_bandwidth(n, m, src, dst, nullptr))",
     "if (orc_bandwidth(n, m, src, dst, pos.data()) < orc_bandwidth(n, m, src, dst, nullptr))", 0),
    ("bandwidth: position map ignored", "oracle.cpp",
     "int64_t i = pos ? pos[dst[e]] : dst[e];", "int64_t i = dst[e];", 0),
    # layout (Eq. 3 and the coverage rule; readings c6, c9, c10)
    ("layout: super-diagonal blocks dropped", "oracle.cpp",
     "if (!via_super && (d < -1 || d > 1)) { ++dropped; continue; }",
     "if (!via_super && (d < -1 || d > 0)) { ++dropped; continue; }", 0),
    ("layout: blocks two apart kept", "oracle.cpp",
     "if (!via_super && (d < -1 || d > 1)) { ++dropped; continue; }",
     "if (!via_super && (d < -2 || d > 2)) { ++dropped; continue; }", 0),
    ("layout: bit order within a byte reversed", "oracle.cpp",
     "masks[byte] |= (uint8_t)(1u << (cc % 8));", "masks[byte] |= (uint8_t)(1u << (7 - cc % 8));",
     0),
    ("layout: upper and lower diagonals swapped", "oracle.cpp",
     "size_t byte = ((((size_t)k * 3 + (size_t)(d + 1)) * P + t) * S + r) * (S / 8) + cc / 8;",
     "size_t byte = ((((size_t)k * 3 + (size_t)(1 - d)) * P + t) * S + r) * (S / 8) + cc / 8;", 0),
    ("layout: rows and columns of a tile swapped", "oracle.cpp",
     "int64_t r = i % S, cc = j % S;", "int64_t r = j % S, cc = i % S;", 0),
    ("layout: packing skips a graph that does not fit instead of stopping", "oracle.cpp",
     "if (!stopped && next_pos + n <= cap) {", "if (next_pos + n <= cap) {", 0),
    ("layout: duplicate edges kept", "oracle.cpp",
     "edges.erase(std::unique(edges.begin(), edges.end()), edges.end());", "(void)0;", 0),
    ("supernodes: lowest degree first", "oracle.cpp",
     "return nb[a].size() != nb[b].size() ? nb[a].size() > nb[b].size() : a < b;",
     "return nb[a].size() != nb[b].size() ? nb[a].size() < nb[b].size() : a < b;", 0),
    # reachability (Section 4)
    ("reach: followed along the edges instead of against them", "oracle.cpp",
     "if (in[dst[e]]) next[src[e]] = 1;", "if (in[src[e]]) next[dst[e]] = 1;", 0),
    ("reach: one step short", "oracle.cpp",
     "for (int32_t k = 1; k <= T; ++k) {", "for (int32_t k = 1; k < T; ++k) {", 0),
    # readout and Adam
    ("readout: graph sum instead of mean", "oracle.cpp",
     "for (int32_t h = 0; h < H; ++h) pool[h] /= count[g];", "(void)0;", 0),
    ("adam: no bias correction of the first moment", "oracle.cpp",
     "param[i] -= lr * (m[i] / c1) / (std::sqrt(v[i] / c2) + eps);",
     "param[i] -= lr * m[i] / (std::sqrt(v[i] / c2) + eps);", 0),
    # the multi-threaded variant must agree with the oracle to the last bit
    ("parallel oracle: sigmoid of the negated argument", "oracle_par.cpp",
     "double sigmoid_p(double x) { return 1.0 / (1.0 + std::exp(-x)); }",
     "double sigmoid_p(double x) { return 1.0 / (1.0 + std::exp(x)); }", 0),
    # summation order alone: the same terms added in another order must not pass as bit-equal
    ("parallel oracle: a target's messages summed last edge first", "oracle_par.cpp",
     "    for (int64_t i = off[v]; i < off[v + 1]; ++i) {\n      const int64_t e = ids[(size_t)i];",
     "    for (int64_t i = off[v]; i < off[v + 1]; ++i) {\n"
     "      const int64_t e = ids[(size_t)(off[v] + off[v + 1] - 1 - i)];", 0),
    ("parallel oracle: dE summed over the types in descending order", "oracle_par.cpp",
     "      for (int32_t p = 0; p < P; ++p) {\n        const double* g = &dM[((size_t)p * N + u) * H];",
     "      for (int32_t p = P - 1; p >= 0; --p) {\n"
     "        const double* g = &dM[((size_t)p * N + u) * H];", 0),
]


def _plant(text, old, new, occurrence):
    starts = [m.start() for m in re.finditer(re.escape(old), text)]
    if occurrence == 0:
        assert len(starts) == 1, f"expected one occurrence, found {len(starts)}: {old[:60]}"
        at = starts[0]
    else:
        assert len(starts) >= occurrence, f"fewer than {occurrence} occurrences: {old[:60]}"
        at = starts[occurrence - 1]
    return text[:at] + new + text[at + len(old):]


def _tree(base, mutant):
    """A copy of the oracle (one mistake planted unless `mutant` is None) beside a copy of its pin
    tests; the package of seeded input generators is linked, not copied."""
    os.makedirs(base)
    shutil.copytree(os.path.join(ROOT, "oracle"), os.path.join(base, "oracle"),
                    ignore=shutil.ignore_patterns("*.so", "*.so.tmp*", "__pycache__"))
    os.makedirs(os.path.join(base, "tests"))
    for f in ("conftest.py", "test_oracle.py"):
        shutil.copy(os.path.join(ROOT, "tests", f), os.path.join(base, "tests", f))
    shutil.copytree(os.path.join(ROOT, "tests", "golden"), os.path.join(base, "tests", "golden"))
    os.symlink(os.path.join(ROOT, "paper_1906_11786_gb300"),
               os.path.join(base, "paper_1906_11786_gb300"))
    if mutant is not None:
        _, fname, old, new, occ = mutant
        p = os.path.join(base, "oracle", fname)
        src = open(p).read()
        open(p, "w").write(_plant(src, old, new, occ))


def _run(base):
    """Build the copy's oracle, then run its pin tests; (return code, first failing test)."""
    env = dict(os.environ, PYTHONPATH=base, PYTHONDONTWRITEBYTECODE="1", OMP_NUM_THREADS="2")
    b = subprocess.run([sys.executable, "-c", "import oracle; oracle.build()"], cwd=base, env=env,
                       capture_output=True, text=True, timeout=300)
    if b.returncode != 0:
        return b.returncode, "build failed: " + b.stderr[-300:]
    r = subprocess.run([sys.executable, "-m", "pytest", os.path.join(base, "tests", "test_oracle.py"),
                        "-x", "-q", "-p", "no:cacheprovider", "-m", "not gpu"],
                       cwd=base, env=env, capture_output=True, text=True, timeout=600)
    failed = re.findall(r"FAILED \S+::(\S+)", r.stdout)
    return r.returncode, (failed[0] if failed else r.stdout[-300:])


def test_every_planted_mistake_fails_a_pin(tmp_path):
    names = [m[0] for m in MUTANTS]
    assert len(set(names)) == len(names)
    jobs = {"control": None}
    jobs.update({m[0]: m for m in MUTANTS})
    bases = {}
    for i, (name, m) in enumerate(jobs.items()):
        bases[name] = str(tmp_path / f"m{i:02d}")
        _tree(bases[name], m)
    with cf.ThreadPoolExecutor(max_workers=max(2, min(8, os.cpu_count() or 2))) as ex:
        res = dict(zip(jobs, ex.map(lambda n: _run(bases[n]), jobs)))
    rc, info = res.pop("control")
    assert rc == 0, f"the unmodified copy of the oracle fails its pins: {info}"
    survivors = {n: info for n, (rc, info) in res.items() if rc == 0}
    assert not survivors, f"mistakes no pin catches: {sorted(survivors)}"
    broken = {n: info for n, (rc, info) in res.items() if info.startswith("build failed")}
    assert not broken, f"mutants that do not compile (fix the case, not the oracle): {broken}"
    for n, (rc, info) in sorted(res.items()):
        print(f"{n:70s} -> {info}")
