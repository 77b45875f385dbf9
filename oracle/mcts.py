"""Reference Monte Carlo tree search over transformation sequences (CPU).

TEST INFRASTRUCTURE ONLY: used by the tests to check the library's search
step by step; the product never imports it.

Follows Sec. 3.2 of the paper in its own order and notation:
  * tree T = <V, E>: nodes are programs P, edges transformations tau;
  * selection: descend from the root by
        UCT(P_i) = Q(P_i)/N(P_i) + c * sqrt(ln N(P_{i-1}) / N(P_i));
  * expansion: propose a transformation for the selected leaf P_i and apply
    it, P_{i+1} = tau(P_i); a program already in the tree is not added
    (acyclicity). B children per expansion (Sec. 4.1: B = 2, c = sqrt(2));
  * rollout: P_sim = (tau_q o ... o tau_1)(P_{i+1}) with random legal tau;
    the reward of P_{i+1} is the objective of P_sim, here a measurement;
  * backpropagation: Q(P_A) += Q(P_{i+1}), N(P_A) += 1 for every ancestor
    P_A (including P_{i+1} itself).
The proposal is the non-LLM policy the paper falls back to (App. G): a
transformation drawn uniformly from the valid set.

Readings where the paper is silent (shared with the library's
documentation, written here independently): unvisited children are taken
first in child order and UCT ties go to the lower index; horizon T = 8,
rollout q = 2; the reward of a program is t(P0)/t(P) (failed = 0); a newly
added node and its P_sim are both measured and measurements are cached per
program; random numbers come from the published splitmix64 sequence
draw(n) = mix(mix(seed) + (n + 1) * 0x9E3779B97F4A7C15), an index in [0, m)
being ((draw >> 11) * m) >> 53.
"""
from __future__ import annotations

import math

_MASK = (1 << 64) - 1


def _mix(z: int) -> int:
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _MASK
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _MASK
    return z ^ (z >> 31)


class Node:
    def __init__(self, program, parent, depth):
        self.program = program
        self.parent = parent
        self.depth = depth
        self.children = []
        self.expanded = False
        self.Q = 0.0
        self.N = 0
        self.sim = program


class MCTS:
    """space: list of transforms; apply(program, tau) -> program or None (illegal)."""

    def __init__(self, root, space, apply, seed=0, c=math.sqrt(2.0), B=2, T=8, q=2, max_tries=64):
        self.space, self.apply = space, apply
        self.c, self.B, self.T, self.q, self.max_tries = c, B, T, q, max_tries
        self.key = _mix(seed & _MASK)
        self.n = 0
        self.nodes = [Node(root, None, 0)]
        self.where = {root: 0}
        self.reward = {}
        self.pending = []
        self.awaiting = []
        self.t0 = None

    def _draw(self):
        self.n += 1
        return _mix((self.key + self.n * 0x9E3779B97F4A7C15) & _MASK)

    def _index(self, m):
        return ((self._draw() >> 11) * m) >> 53

    def _random_tau(self):
        return self.space[self._index(len(self.space))]

    def _backprop(self, i, r):
        while i is not None:
            self.nodes[i].Q += r
            self.nodes[i].N += 1
            i = self.nodes[i].parent

    def _expandable(self, i):
        nd = self.nodes[i]
        return not nd.expanded and nd.depth < self.T

    def _open(self, i):
        return self._expandable(i) or any(self._open(c) for c in self.nodes[i].children)

    def _uct(self, child, parent):
        ch, pa = self.nodes[child], self.nodes[parent]
        return ch.Q / ch.N + self.c * math.sqrt(math.log(pa.N) / ch.N)

    def _select(self):
        if not self._open(0):
            return None
        i = 0
        while not self._expandable(i):
            best, best_v = None, -math.inf
            for ch in self.nodes[i].children:
                if not self._open(ch):
                    continue
                if self.nodes[ch].N == 0:
                    best = ch
                    break
                v = self._uct(ch, i)
                if v > best_v:
                    best, best_v = ch, v
            if best is None:
                return None
            i = best
        return i

    def step(self, times):
        """times: measured ms (None = failed) of the previous batch, in order."""
        assert len(times) == len(self.pending)
        for p, t in zip(self.pending, times):
            if self.t0 is None:
                self.t0 = t
            self.reward[p] = (self.t0 / t) if t else 0.0
        self.pending = []
        for i in self.awaiting:
            self._backprop(i, self.reward[self.nodes[i].sim])
        self.awaiting = []
        if self.t0 is None:
            self.pending.append(self.nodes[0].program)
            self.awaiting.append(0)
            return list(self.pending)

        def want(p):
            if p not in self.reward and p not in self.pending:
                self.pending.append(p)

        for _ in range(4096):
            if self.pending:
                break
            leaf = self._select()
            if leaf is None:
                break
            self.nodes[leaf].expanded = True
            kids = []
            tries = 0
            while len(kids) < self.B and tries < self.max_tries:
                tries += 1
                p = self.apply(self.nodes[leaf].program, self._random_tau())
                if p is None or p in self.where:
                    continue
                self.where[p] = len(self.nodes)
                self.nodes.append(Node(p, leaf, self.nodes[leaf].depth + 1))
                self.nodes[leaf].children.append(len(self.nodes) - 1)
                kids.append(len(self.nodes) - 1)
            for k in kids:
                p = self.nodes[k].program
                for _q in range(self.q):
                    for _t in range(self.max_tries):
                        nxt = self.apply(p, self._random_tau())
                        if nxt is not None:
                            p = nxt
                            break
                self.nodes[k].sim = p
                want(self.nodes[k].program)
                if p != self.nodes[k].program:
                    want(p)
                self.awaiting.append(k)
            if not self.pending:
                for i in self.awaiting:
                    self._backprop(i, self.reward[self.nodes[i].sim])
                self.awaiting = []
        return list(self.pending)

    def best(self):
        return max(self.reward.items(), key=lambda kv: kv[1]) if self.reward else None
