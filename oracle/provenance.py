"""Oracle: provenance-graph queries of Alg. 1 (lines 1-3), by their definitions.

TEST INFRASTRUCTURE ONLY (see the package docstring).  Written from the paper;
shares no code with the C++ library.

The runtime records artifacts (Sec. 3.4(a)): each has an id, a type, parents
(the artifacts it was computed from), the source ids it carries, the token
span it occupies in the session and its turn, and whether it committed an
external side effect.  Edges run parent -> child.

  LocateSource(z)   the artifact through which z entered: among artifacts
                    that carry z in their own source ids, the one that no
                    parent carrying z precedes; several such -> the earliest
                    token_begin, then the smallest id
  TaintClosure(s)   I(z): every artifact reachable from s along parent ->
                    child edges, s included (Lemma 2: reachability closure)
  FirstEntry(s)     tau: the 1-based position of the first token held by an
                    artifact of the closure (min token_begin + 1); every
                    position before it is clean (Lemma 1, Lemma 2(ii))
"""
from __future__ import annotations


class ProvError(Exception):
    def __init__(self, kind, msg):
        super().__init__(f"{kind}: {msg}")
        self.kind = kind


class OracleProvenance:
    def __init__(self):
        self.art = {}  # id -> dict

    def add(self, aid, type_=0, parents=(), source_ids=(), token_begin=0, token_end=0, turn=0, committed=False):
        if aid in self.art:
            raise ProvError("invalid", f"duplicate artifact {aid}")
        for p in parents:
            if p not in self.art:
                raise ProvError("invalid", f"unknown parent {p}")
        if token_end < token_begin or token_begin < 0:
            raise ProvError("invalid", "bad token span")
        self.art[aid] = dict(type=type_, parents=list(parents), sources=set(source_ids), begin=token_begin,
                             end=token_end, turn=turn, committed=bool(committed))

    def children(self):
        ch = {a: [] for a in self.art}
        for a, rec in self.art.items():
            for p in rec["parents"]:
                ch[p].append(a)
        return ch

    def locate_source(self, z):
        carriers = [a for a, r in self.art.items() if z in r["sources"]]
        if not carriers:
            raise ProvError("range", f"no artifact carries {z}")
        roots = [a for a in carriers if not any(z in self.art[p]["sources"] for p in self.art[a]["parents"])]
        return min(roots, key=lambda a: (self.art[a]["begin"], a))

    def taint_closure(self, s):
        if s not in self.art:
            raise ProvError("range", f"unknown artifact {s}")
        ch = self.children()
        seen = {s}
        frontier = [s]
        while frontier:
            nxt = []
            for a in frontier:
                for c in ch[a]:
                    if c not in seen:
                        seen.add(c)
                        nxt.append(c)
            frontier = nxt
        return sorted(seen)

    def first_entry(self, s):
        return min(self.art[a]["begin"] for a in self.taint_closure(s)) + 1

    def committed_in(self, closure):
        return sum(1 for a in closure if self.art[a]["committed"])
