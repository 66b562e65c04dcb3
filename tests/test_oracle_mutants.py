"""Planted mistakes in the oracles must fail at least one of their pins (CPU).

Construction oracle: each case copies ``oracle/dart_oracle.c``, changes one
spot the way a plausible slip would (a swapped concatenation, a dropped term,
a wrong index or drafter row, a reversed tie-break, ...), compiles the copy
and points the oracle's ctypes wrapper at it for the duration of the test,
then runs every pin of ``test_oracle_pins.py``.  Tree-attention oracle: the
same with a changed copy of ``oracle/tree_attn.py`` loaded as a module and
the pins of ``test_attn_oracle_pins.py``.  A planted mistake that passes
every pin would mean the pins cannot tell that part of an oracle from a
wrong one.  The oracle sources themselves carry no switches for this.
"""
import importlib.util
import inspect
import itertools
import os
import shutil
import subprocess

import pytest

import oracle
import test_attn_oracle_pins as attn_pins
import test_oracle_pins as pins
from oracle import tree_attn

# (name, exact text of the oracle, planted replacement)
MUTANTS = [
    ("head: [E[t]; h_p] instead of [h_p; E[t]]",
     "        x[j] = hp[j];\n        x[d + j] = wval(E, dt, (size_t)tok * d + j);",
     "        x[d + j] = hp[j];\n        x[j] = wval(E, dt, (size_t)tok * d + j);"),
    ("head: residual h_p dropped",
     "r[i] = hp[i] + wdot(Wo, dt, (size_t)i * d, a, d);",
     "r[i] = wdot(Wo, dt, (size_t)i * d, a, d);"),
    ("head: RMSNorm epsilon dropped",
     "sqrt(ss / d + c->rms_eps)",
     "sqrt(ss / d)"),
    ("head: ReLU instead of SiLU",
     "a[i] = u / (1.0 + exp(-u));",
     "a[i] = u > 0.0 ? u : 0.0;"),
    ("scoring: temperature not applied",
     "z[v] = ((double)dlog_row[v] + wdot(E, dt, (size_t)v * d, h, d)) / Tp;",
     "z[v] = ((double)dlog_row[v] + wdot(E, dt, (size_t)v * d, h, d));"),
    ("scoring: drafter row of position d instead of d-1",
     "const float *row = Dlog + ((size_t)s * L + dep - 1) * V;",
     "const float *row = Dlog + ((size_t)s * L + (dep < L ? dep : dep - 1)) * V;"),
    ("Eq. 5: depth bonus beta dropped",
     "cand[ncand].score = pscore[p] + logq[idx[j]] + c->beta; /* Eq. 5 */",
     "cand[ncand].score = pscore[p] + logq[idx[j]]; /* Eq. 5 */"),
    ("Eq. 5: parent's path score not accumulated",
     "cand[ncand].score = pscore[p] + logq[idx[j]] + c->beta; /* Eq. 5 */",
     "cand[ncand].score = logq[idx[j]] + c->beta; /* Eq. 5 */"),
    ("state update: child state from the first parent",
     "orc_head(c, Wi, Wo, E, hs + (size_t)cand[r].p * d, cand[r].tok,",
     "orc_head(c, Wi, Wo, E, hs, cand[r].tok,"),
    ("top-k: ties by token desc",
     "return a > b || (a == b && ia < ib);",
     "return a > b || (a == b && ia > ib);"),
    ("frontier: ties by parent slot desc",
     "if (a->p != b->p) return a->p < b->p ? -1 : 1;",
     "if (a->p != b->p) return a->p > b->p ? -1 : 1;"),
    ("pruning: ties by node id desc",
     "return a->id < b->id ? -1 : (a->id > b->id);",
     "return a->id > b->id ? -1 : (a->id < b->id);"),
    ("emission: position id = pos_offset + depth - 1",
     "o_pos[o] = c->pos_offset + dep;",
     "o_pos[o] = c->pos_offset + dep - 1;"),
    ("emission: mask row holds the parent only",
     "            a = o_par[(size_t)s * B + a];",
     "            a = -1;"),
    ("heap: ties popped by node id desc",
     "((a).score == (b).score && (a).id < (b).id))",
     "((a).score == (b).score && (a).id > (b).id))"),
    ("candidate set: the K smallest drafter logits",
     "for (int v = 0; v < c->V; v++) x[v] = (double)dlog_row[v];",
     "for (int v = 0; v < c->V; v++) x[v] = -(double)dlog_row[v];"),
    ("candidate set: left in rank order instead of token order",
     "    qsort(cand, (size_t)c->cand_k, sizeof(int), int_cmp);\n",
     ""),
    ("chain: the state advanced with depth 1's token at every depth",
     "orc_head(c, Wi, Wo, E, h, y, t);",
     "orc_head(c, Wi, Wo, E, h, ltok[0], t);"),
    ("DDTree: a node's offers scored with its own depth's marginal",
     "if (dep < L) memcpy(olq + (size_t)(n + 1) * B, llq + (size_t)dep * B, sizeof(double) * (size_t)B);",
     "if (dep < L) memcpy(olq + (size_t)(n + 1) * B, llq + (size_t)(dep - 1) * B, sizeof(double) * (size_t)B);"),
    ("sequential heap: children scored at the parent's state",
     "child_logq_all(c, E, dl + (size_t)dep * V, hn, lq);",
     "child_logq_all(c, E, dl + (size_t)dep * V, hs + (size_t)(p + 1) * d, lq);"),
    ("sequential heap: children scored with the parent's drafter row",
     "child_logq_all(c, E, dl + (size_t)dep * V, hn, lq);",
     "child_logq_all(c, E, dl + (size_t)(dep - 1) * V, hn, lq);"),
    ("best-first offers: depth bonus dropped",
     "+ llq[(size_t)(p + 1) * lstride + next[p + 1]] + c->beta;",
     "+ llq[(size_t)(p + 1) * lstride + next[p + 1]];"),
    ("pop-order emission: mask row holds the node only",
     "for (int a = i; a >= 0; a = par[a]) row[a / 64] |= 1ull << (a % 64);",
     "row[i / 64] |= 1ull << (i % 64);"),
    ("teacher-forced state: every step from the first token",
     "    for (int i = 0; i < len; i++) {\n        orc_head(c, Wi, Wo, E, h, path[i], t);\n        memcpy(h, t, sizeof(double) * (size_t)d);\n    }\n    memcpy(h_out",
     "    for (int i = 0; i < len; i++) {\n        orc_head(c, Wi, Wo, E, h, path[0], t);\n        memcpy(h, t, sizeof(double) * (size_t)d);\n    }\n    memcpy(h_out"),
    ("teacher-forced children: drafter row of the prefix's last position",
     "const float *row = Dlog_seq + (size_t)len * V;",
     "const float *row = Dlog_seq + (size_t)(len > 0 ? len - 1 : 0) * V;"),
    ("teacher-forced scores: beta not added",
     "s += lq[path[i]] + c->beta;",
     "s += lq[path[i]];"),
    ("restricted q~: normalised over the full vocabulary",
     "    double lse = orc_log_softmax(z, K, lq);\n    free(z);",
     "    double *zf = (double *)malloc(sizeof(double) * (size_t)c->V);\n"
     "    double *lf = (double *)malloc(sizeof(double) * (size_t)c->V);\n"
     "    orc_child_logits(c, E, dlog_row, h, zf);\n"
     "    double lse = orc_log_softmax(zf, c->V, lf);\n"
     "    for (int i = 0; i < K; i++) lq[i] = z[i] - lse < 0.0 ? z[i] - lse : 0.0;\n"
     "    free(zf);\n    free(lf);\n    free(z);"),
]


# the tree-attention oracle (numpy): (name, exact text, planted replacement)
ATTN_MUTANTS = [
    ("RoPE: rotation by -angle",
     "return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)",
     "return np.concatenate([x1 * c + x2 * s, x2 * c - x1 * s], axis=-1)"),
    ("RoPE: frequencies theta^(-t/dh)",
     "inv_freq = float(theta) ** (-2.0 * np.arange(half, dtype=np.float64) / dh)",
     "inv_freq = float(theta) ** (-1.0 * np.arange(half, dtype=np.float64) / dh)"),
    ("GQA: query head h reads kv head h % Hkv",
     "g = h // G",
     "g = h % Hkv"),
    ("positions: pos_offset + depth - 1",
     "pos = pos_offset + np.asarray(depths[s], dtype=np.int64)",
     "pos = pos_offset + np.asarray(depths[s], dtype=np.int64) - 1"),
    ("logits: scale dropped",
     "logits = scale * (keys @ qi)",
     "logits = keys @ qi"),
    ("path: the node itself left out",
     "    j = int(i)\n    while j >= 0:",
     "    j = int(parents[i])\n    while j >= 0:"),
    ("context: keys and values left out",
     "keys = np.concatenate([k_ctx[s, :, g], kt], axis=0)\n"
     "                vals = np.concatenate([v_ctx[s, :, g], v_tree[s, path, g]], axis=0)",
     "keys = kt\n                vals = v_tree[s, path, g]"),
    ("context: values of kv head 0",
     "vals = np.concatenate([v_ctx[s, :, g], v_tree[s, path, g]], axis=0)",
     "vals = np.concatenate([v_ctx[s, :, 0], v_tree[s, path, g]], axis=0)"),
    ("query not rotated",
     "qi = rope(q[s, i, h], pos[i], rope_theta)",
     "qi = q[s, i, h]"),
    ("tree keys rotated at the query's position",
     "kt = rope(k_tree[s, path, g], pos[path], rope_theta)",
     "kt = rope(k_tree[s, path, g], pos[i], rope_theta)"),
]


def pin_cases(module=pins):
    """(id, function, kwargs) for every pin, parametrisations expanded."""
    out = []
    for name, fn in inspect.getmembers(module, inspect.isfunction):
        if not name.startswith("test_") or fn.__module__ != module.__name__:
            continue
        marks = [m for m in getattr(fn, "pytestmark", []) if m.name == "parametrize"]
        grids = []
        for m in marks:
            names = [a.strip() for a in m.args[0].split(",")] if isinstance(m.args[0], str) else list(m.args[0])
            vals = [v if len(names) > 1 else (v,) for v in m.args[1]]
            grids.append([dict(zip(names, v)) for v in vals])
        params = set(inspect.signature(fn).parameters)
        for combo in itertools.product(*grids) if grids else [()]:
            kw = {}
            for part in combo:
                kw.update(part)
            if set(kw) != params:
                continue  # needs a fixture: not a pure pin
            out.append((f"{name}{sorted(kw.items()) if kw else ''}", fn, kw))
    return out


def build_mutant(tmp_path, old, new):
    src = open(oracle._SRC).read()
    assert src.count(old) == 1, "the planted spot must occur exactly once in the oracle"
    msrc = tmp_path / "dart_oracle_mut.c"
    msrc.write_text(src.replace(old, new))
    mlib = tmp_path / "libdart_oracle_mut.so"
    cmd = ["gcc", "-O2", "-std=c11", "-shared", "-fPIC", str(msrc), "-o", str(mlib), "-lm"]
    r = subprocess.run(cmd[:1] + ["-fopenmp"] + cmd[1:], capture_output=True)
    if r.returncode != 0:
        subprocess.run(cmd, check=True, capture_output=True)
    return msrc, mlib


def failing_pins(module=pins):
    failed = []
    for cid, fn, kw in pin_cases(module):
        try:
            fn(**kw)
        except Exception as e:  # an assertion, or a crash on nonsense output
            failed.append(f"{cid}: {type(e).__name__}")
    return failed


@pytest.mark.skipif(shutil.which("gcc") is None, reason="gcc not available")
def test_unmodified_oracle_passes_every_pin():
    assert len(pin_cases()) >= 25
    assert failing_pins() == []


@pytest.mark.skipif(shutil.which("gcc") is None, reason="gcc not available")
@pytest.mark.parametrize("name,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_planted_mistake_fails_a_pin(tmp_path, monkeypatch, name, old, new):
    msrc, mlib = build_mutant(tmp_path, old, new)
    monkeypatch.setattr(oracle, "_SRC", str(msrc))
    monkeypatch.setattr(oracle, "_LIB", str(mlib))
    monkeypatch.setattr(oracle, "_lib", None)
    failed = failing_pins()
    print(name, "->", failed)
    assert failed, f"planted mistake passed every pin: {name}"


def test_unmodified_attention_oracle_passes_every_pin():
    assert len(pin_cases(attn_pins)) >= 8
    assert failing_pins(attn_pins) == []


@pytest.mark.parametrize("name,old,new", ATTN_MUTANTS, ids=[m[0] for m in ATTN_MUTANTS])
def test_planted_attention_mistake_fails_a_pin(tmp_path, monkeypatch, name, old, new):
    src = open(tree_attn.__file__).read()
    assert src.count(old) == 1, "the planted spot must occur exactly once in the oracle"
    path = tmp_path / "tree_attn_mut.py"
    path.write_text(src.replace(old, new))
    spec = importlib.util.spec_from_file_location("tree_attn_mut", path)
    mut = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mut)
    monkeypatch.setattr(attn_pins, "ta", mut)
    failed = failing_pins(attn_pins)
    print(name, "->", failed)
    assert failed, f"planted mistake passed every pin: {name}"
