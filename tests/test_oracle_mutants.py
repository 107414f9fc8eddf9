"""Plant one plausible mistake at a time in a copy of the oracle (on the CPU) and
check that the pins catch it.  This is evidence that the pins constrain every
part of the oracle: a dropped term, a wrong index or alignment, a swapped
operand, a wrong crop offset or push order."""
import importlib.util
import os
import shutil
import sys

import pytest

import oracle_pins as pins

ORACLE_DIR = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "oracle")

MUTANTS = [
    ("gqa_mapping", "attention.c", "const int32_t kvh = h / group;", "const int32_t kvh = h % jb->hkv;"),
    ("causal_off_by_one", "attention.c", "j <= a; ++j", "j < a; ++j"),
    ("dropped_scale", "attention.c", "s *= jb->scale;", ""),
    ("top_left_alignment", "attention.c", "const int64_t a = jb->n_keys - jb->n_q + i;", "const int64_t a = i;"),
    ("value_from_keys", "attention.c", "const uint16_t *vrow = jb->v +", "const uint16_t *vrow = jb->k +"),
    ("unnormalised", "attention.c", "o[c] /= den;", "o[c] /= 1.0;"),
    ("keys_head_major", "attention.c", "jb->k + (j * jb->hkv + kvh) * (int64_t)d",
     "jb->k + (kvh * jb->n_keys + j) * (int64_t)d"),
    ("query_from_output_row", "attention.c", "jb->q + (i * jb->hq + h) * (int64_t)d",
     "jb->q + (r * jb->hq + h) * (int64_t)d"),
    ("output_head_major", "attention.c", "jb->out + (r * jb->hq + h) * (int64_t)d",
     "jb->out + (h * jb->n_rows + r) * (int64_t)d"),
    ("crop_keeps_tau", "kvcache.py", "new_len = tau - 1\n", "new_len = min(tau, n)\n"),
    ("push_ascending", "kvcache.py", "for p in reversed(pages):", "for p in pages:"),
    ("slot_shift", "kvcache.py", "page, slot = tbl[pos // self.ps], pos % self.ps",
     "page, slot = tbl[pos // self.ps], (pos + 1) % self.ps"),
    ("counter_not_reset", "kvcache.py", "self.length[seq] = new_len\n        self.appended[seq] = 0\n",
     "self.length[seq] = new_len\n"),
    ("cow_skipped", "kvcache.py", "cow = n > 0 and old % self.ps != 0 and self.refs[tbl[-1]] > 1",
     "cow = False"),
    ("fork_no_ref", "kvcache.py", "        for p in self.table[s]:\n            self.refs[p] += 1\n", ""),
    ("checkpoint_le_tau", "kvcache.py", "cands = [b for b in self.checkpoints[seq] if b < tau]",
     "cands = [b for b in self.checkpoints[seq] if b <= tau]"),
]


def _load_mutant(tmp_path, name, fname, old, new):
    dst = tmp_path / f"oracle_mut_{name}"
    shutil.copytree(ORACLE_DIR, dst, ignore=shutil.ignore_patterns("*.so", "__pycache__"))
    path = dst / fname
    src = path.read_text()
    assert old in src, f"mutation anchor for {name} not found"
    path.write_text(src.replace(old, new))
    spec = importlib.util.spec_from_file_location(f"oracle_mut_{name}", dst / "__init__.py",
                                                  submodule_search_locations=[str(dst)])
    mod = importlib.util.module_from_spec(spec)
    sys.modules[spec.name] = mod
    spec.loader.exec_module(mod)
    return mod


def _pins_fail(mod):
    checks = [lambda: pins.pin_bruteforce(mod, full=False), lambda: pins.pin_closed_forms(mod),
              lambda: pins.pin_splice(mod), lambda: pins.pin_corollary(mod),
              lambda: pins.pin_bookkeeping(mod, n_ops=150), lambda: pins.pin_fork(mod, n_ops=150)]
    caught = 0
    for chk in checks:
        try:
            chk()
        except Exception:  # an assertion or any failure counts as caught
            caught += 1
    return caught


@pytest.mark.parametrize("name,fname,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_pins_catch_planted_mistake(tmp_path, name, fname, old, new):
    mod = _load_mutant(tmp_path, name, fname, old, new)
    assert _pins_fail(mod) >= 1, f"no pin caught mutant {name}"


PROV_MUTANTS = [
    ("edges_reversed", "for p in rec[\"parents\"]:\n                ch[p].append(a)",
     "for p in rec[\"parents\"]:\n                ch[a].append(p)"),
    ("closure_without_source", "seen = {s}\n        frontier = [s]", "seen = set()\n        frontier = [s]"),
    ("tau_zero_based", "return min(self.art[a][\"begin\"] for a in self.taint_closure(s)) + 1",
     "return min(self.art[a][\"begin\"] for a in self.taint_closure(s))"),
    ("source_not_root", "return min(roots, key=lambda a: (self.art[a][\"begin\"], a))",
     "return max(carriers, key=lambda a: (self.art[a][\"begin\"], a))"),
]


@pytest.mark.parametrize("name,old,new", PROV_MUTANTS, ids=[m[0] for m in PROV_MUTANTS])
def test_provenance_pins_catch_planted_mistake(tmp_path, name, old, new):
    import test_oracle_provenance as tp
    src = open(os.path.join(ORACLE_DIR, "provenance.py")).read()
    assert old in src, name
    path = tmp_path / f"prov_mut_{name}.py"
    path.write_text(src.replace(old, new))
    spec = importlib.util.spec_from_file_location(f"prov_mut_{name}", path)
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    caught = 0
    for chk in (lambda: _prov_episode(tp, mod), lambda: _prov_random(tp, mod)):
        try:
            chk()
        except Exception:
            caught += 1
    assert caught >= 1, f"no pin caught provenance mutant {name}"


def _prov_episode(tp, mod):
    ep = tp.load_episode()
    g = tp.build(mod.OracleProvenance(), ep["artifacts"])
    q = ep["query"]
    s = g.locate_source(q["z"])
    assert s == q["source"] and g.taint_closure(s) == q["closure"] and g.first_entry(s) == q["tau"]


def _prov_random(tp, mod):
    for seed in range(6):
        arts = tp.random_dag(seed, 60)
        g = tp.build(mod.OracleProvenance(), arts)
        s = g.locate_source(9)
        assert g.taint_closure(s) == tp.brute_closure(arts, s)
        assert not any(9 in g.art[p]["sources"] for p in g.art[s]["parents"])


SCHED_MUTANTS = [
    ("independent_turns_decoded", "_KNOWN = {SELECTIVE: (0, 1), PREFIX_CACHE: (0,)}",
     "_KNOWN = {SELECTIVE: (0,), PREFIX_CACHE: (0,)}"),
    ("trailing_run_dropped", "    if run > 0:\n        units.append(run)\n    return units", "    return units"),
    ("decode_turn_one_pass", "units.extend([1] * n)", "units.append(n)"),
    ("known_turns_not_merged",
     "            run += n                      # known tokens extend the current prefill run\n",
     "            if run > 0:\n                units.append(run)\n            run = n\n"),
    ("values_from_keys", "cache.append(seqs[i], k_bits[:, lo:hi], v_bits[:, lo:hi])",
     "cache.append(seqs[i], k_bits[:, lo:hi], k_bits[:, lo:hi])"),
    ("progress_ignored", "lo = int(cu_tok[i]) + done[i]", "lo = int(cu_tok[i])"),
]


@pytest.mark.parametrize("name,old,new", SCHED_MUTANTS, ids=[m[0] for m in SCHED_MUTANTS])
def test_schedule_pins_catch_planted_mistake(tmp_path, name, old, new):
    import test_oracle_schedule as ts
    mod = _load_mutant(tmp_path, name, "schedule.py", old, new)
    caught = 0
    for chk in (lambda: ts.pin_golden(mod.schedule), lambda: ts.pin_bruteforce_and_count(mod.schedule),
                lambda: ts.pin_degenerate(mod.schedule), lambda: ts.pin_workload_monotone(mod.schedule),
                lambda: ts.pin_execution(mod, seeds=range(3))):
        try:
            chk()
        except Exception:
            caught += 1
    assert caught >= 1, f"no pin caught schedule mutant {name}"
