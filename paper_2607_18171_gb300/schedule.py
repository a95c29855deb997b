"""Deployment period and latency calculator for streaming pipelines (App. A).

The paper models a streaming application as a pipeline graph (App. A.1.2): a set of
operations that each run once per batch, edges (u, v, lam) meaning batch j of v waits
for batch j - lam of u, entry operations gated by the batch's arrival time
R_j = (j + 1) T, and an output map o(k) naming the operation whose completion releases
chunk k of a batch. A deployment assigns every operation to a resource (one GPU or a
GPU group), gives per-operation times tau_v and per-edge lags kappa, and runs each
resource through a fixed cyclic order of its operations.

This module computes, for such a graph and deployment:

* the earliest-start schedule under the cyclic orders (start S and completion C of
  every instance over a finite horizon of batches);
* the smallest feasible display offset d0* = sup_{j,k} (Y_jk - j T - k Delta), with
  Y_jk = C_{j,o(k)} and Delta = T / N (Lemma A.1, "display offset");
* the path lower bound w(P) + (1 - Lambda(P)) T - k Delta for a path P from an entry to
  o(k) (Lemma A.2, "path bound");
* the sustainable period T_min = max over resources of the per-batch load
  W_r = sum of tau_v on r (Lemma A.3, "resource load"), together with the
  cross-batch self-edge terms tau_v + kappa_{v,v,1} that App. A.3 and A.4 add;
* the closed forms of App. A.3 (DiT -> VAE, co-located vs disaggregated) and App. A.4
  (n denoising steps, sequence parallel vs stage pipeline over per-step KV caches),
  and the peak displayed frame rate N / T_min.

It is host-side arithmetic over a handful of numbers; measured per-chunk kernel times
(for example the per-step attention times of a frt_steps group) are its inputs.
"""

from __future__ import annotations

import argparse
import json
from dataclasses import dataclass, field
from typing import Dict, Iterable, List, Mapping, Optional, Sequence, Tuple

Edge = Tuple[str, str, int]   # (u, v, lam): batch j of v waits for batch j - lam of u


@dataclass(frozen=True)
class PipelineGraph:
    """The static template of App. A.1.2: operations, edges, entries, output map."""

    ops: Tuple[str, ...]
    edges: Tuple[Edge, ...]
    entry: Tuple[str, ...]
    output: Tuple[str, ...]          # o(k) for k = 0 .. N - 1

    def __post_init__(self):
        names = set(self.ops)
        if len(names) != len(self.ops):
            raise ValueError("operation names must be unique")
        for u, v, lam in self.edges:
            if u not in names or v not in names:
                raise ValueError(f"edge ({u}, {v}, {lam}) names an unknown operation")
            if lam not in (0, 1):
                raise ValueError("edge batch shift must be 0 or 1")
        if not self.entry or any(e not in names for e in self.entry):
            raise ValueError("entry operations must be known and non-empty")
        if not self.output or any(o not in names for o in self.output):
            raise ValueError("output map must name known operations")

    @property
    def n_chunks(self) -> int:
        return len(self.output)


@dataclass
class Deployment:
    """A deployment plan with its timing data (App. A.1.2).

    assign: operation -> resource; tau: operation -> processing time on that
    assignment; kappa: edge -> synchronisation lag (missing edges lag 0); order:
    resource -> cyclic per-batch order of its operations (default: the template order
    of the operations assigned to it).
    """

    assign: Dict[str, str]
    tau: Dict[str, float]
    kappa: Dict[Edge, float] = field(default_factory=dict)
    order: Dict[str, Tuple[str, ...]] = field(default_factory=dict)

    def lag(self, e: Edge) -> float:
        return float(self.kappa.get(e, 0.0))

    def cyclic_order(self, graph: PipelineGraph) -> Dict[str, Tuple[str, ...]]:
        res: Dict[str, List[str]] = {}
        for v in graph.ops:
            if v not in self.assign:
                raise ValueError(f"operation {v} has no resource")
            if self.tau.get(v, -1.0) < 0:
                raise ValueError(f"operation {v} needs a non-negative processing time")
            res.setdefault(self.assign[v], []).append(v)
        out: Dict[str, Tuple[str, ...]] = {}
        for r, ops in res.items():
            given = self.order.get(r)
            if given is not None:
                if sorted(given) != sorted(ops):
                    raise ValueError(f"order of resource {r} must list exactly its operations")
                out[r] = tuple(given)
            else:
                out[r] = tuple(ops)
        for e, k in self.kappa.items():
            if k < 0:
                raise ValueError(f"lag of edge {e} is negative")
        return out


@dataclass
class Schedule:
    start: Dict[Tuple[int, str], float]
    finish: Dict[Tuple[int, str], float]
    batches: int
    period: float
    n_chunks: int
    output: Tuple[str, ...]

    def ready(self, j: int, k: int) -> float:
        """Y_jk: completion of o(k) in batch j (App. A.1.3)."""
        return self.finish[(j, self.output[k])]


def arrival(j: int, T: float) -> float:
    """R_j = (j + 1) T: batch j is complete once its last action has arrived (App. A.1.1)."""
    return (j + 1) * T


def simulate(graph: PipelineGraph, dep: Deployment, T: float, batches: int) -> Schedule:
    """Earliest-start schedule of `batches` batches under the deployment's cyclic orders.

    Every instance (j, v) starts as soon as (i) its resource has finished the instance
    before it in the cyclic order, (ii) for an entry operation, R_j has passed, and
    (iii) every edge (u, v, lam) has C_{j-lam,u} + kappa behind it. Raises ValueError
    when a cyclic order contradicts an intra-batch edge (no feasible schedule).
    """
    if T <= 0 or batches < 1:
        raise ValueError("period must be positive and batches >= 1")
    orders = dep.cyclic_order(graph)
    preds: Dict[str, List[Edge]] = {v: [] for v in graph.ops}
    for e in graph.edges:
        preds[e[1]].append(e)
    entry = set(graph.entry)
    S: Dict[Tuple[int, str], float] = {}
    C: Dict[Tuple[int, str], float] = {}
    free = {r: 0.0 for r in orders}
    for j in range(batches):
        pos = {r: 0 for r in orders}
        remaining = sum(len(o) for o in orders.values())
        while remaining:
            progressed = False
            for r, seq in orders.items():
                while pos[r] < len(seq):
                    v = seq[pos[r]]
                    t = free[r]
                    ok = True
                    for (u, _, lam) in preds[v]:
                        jj = j - lam
                        if jj < 0:
                            continue
                        if (jj, u) not in C:
                            ok = False
                            break
                        t = max(t, C[(jj, u)] + dep.lag((u, v, lam)))
                    if not ok:
                        break
                    if v in entry:
                        t = max(t, arrival(j, T))
                    S[(j, v)] = t
                    C[(j, v)] = t + float(dep.tau[v])
                    free[r] = C[(j, v)]
                    pos[r] += 1
                    remaining -= 1
                    progressed = True
            if not progressed:
                raise ValueError("cyclic orders contradict the intra-batch edges")
    return Schedule(S, C, batches, T, graph.n_chunks, graph.output)


def offsets(sched: Schedule) -> List[float]:
    """Per batch j: max_k (Y_jk - j T - k Delta), Delta = T / N."""
    T, N = sched.period, sched.n_chunks
    delta = T / N
    return [max(sched.ready(j, k) - j * T - k * delta for k in range(N))
            for j in range(sched.batches)]


def display_offset(sched: Schedule) -> float:
    """d0* over the simulated horizon (Lemma A.1): the smallest offset d0 with
    d0 + j T + k Delta >= Y_jk for every simulated chunk."""
    return max(offsets(sched))


def display_feasible(sched: Schedule, d0: float, tol: float = 1e-12) -> bool:
    """Whether the constant-rate display schedule d_jk = d0 + j T + k Delta meets every
    simulated chunk (the feasibility condition that Lemma A.1 characterises)."""
    T, N = sched.period, sched.n_chunks
    delta = T / N
    return all(d0 + j * T + k * delta >= sched.ready(j, k) - tol
               for j in range(sched.batches) for k in range(N))


def path_weight(path: Sequence[Edge], dep: Deployment) -> Tuple[float, int]:
    """(w(P), Lambda(P)) of a path given as its edges (Lemma A.2)."""
    if not path:
        raise ValueError("a path needs at least one edge; use path_bound_single for one node")
    for a, b in zip(path, path[1:]):
        if a[1] != b[0]:
            raise ValueError("path edges do not chain")
    nodes = [path[0][0]] + [e[1] for e in path]
    w = sum(float(dep.tau[v]) for v in nodes) + sum(dep.lag(e) for e in path)
    return w, sum(e[2] for e in path)


def path_bound(path: Sequence[Edge], dep: Deployment, T: float, k: int, N: int) -> float:
    """Lemma A.2: d0* >= w(P) + (1 - Lambda(P)) T - k Delta for a path from an entry
    operation to o(k)."""
    w, lam = path_weight(path, dep)
    return w + (1 - lam) * T - k * (T / N)


def simple_paths(graph: PipelineGraph, target: str) -> List[Tuple[Edge, ...]]:
    """Every path from an entry operation to `target` that visits no operation twice.
    A zero-length path (target is itself an entry) is returned as ()."""
    out_edges: Dict[str, List[Edge]] = {v: [] for v in graph.ops}
    for e in graph.edges:
        if e[0] != e[1]:
            out_edges[e[0]].append(e)
    found: List[Tuple[Edge, ...]] = []

    def walk(v: str, seen: frozenset, acc: Tuple[Edge, ...]):
        if v == target:
            found.append(acc)
        for e in out_edges[v]:
            if e[1] not in seen:
                walk(e[1], seen | {e[1]}, acc + (e,))

    for s in graph.entry:
        walk(s, frozenset({s}), ())
    return found


def best_path_bound(graph: PipelineGraph, dep: Deployment, T: float) -> float:
    """The largest Lemma A.2 bound over all chunks k and all simple entry paths to o(k)."""
    N = graph.n_chunks
    best = float("-inf")
    for k in range(N):
        for p in simple_paths(graph, graph.output[k]):
            if p:
                b = path_bound(p, dep, T, k, N)
            else:
                b = float(dep.tau[graph.output[k]]) + T - k * (T / N)
            best = max(best, b)
    return best


def resource_load(graph: PipelineGraph, dep: Deployment) -> Dict[str, float]:
    """W_r = sum of tau_v over the operations assigned to r (Lemma A.3)."""
    dep.cyclic_order(graph)
    load: Dict[str, float] = {}
    for v in graph.ops:
        load[dep.assign[v]] = load.get(dep.assign[v], 0.0) + float(dep.tau[v])
    return load


def t_min(graph: PipelineGraph, dep: Deployment) -> float:
    """Sustainable period: the largest per-batch resource load (Lemma A.3), and for each
    cross-batch self-edge (v, v, 1) the time tau_v + kappa_{v,v,1} between consecutive
    instances of v that App. A.3 and A.4 add to it."""
    t = max(resource_load(graph, dep).values())
    for e in graph.edges:
        if e[0] == e[1] and e[2] == 1:
            t = max(t, float(dep.tau[e[0]]) + dep.lag(e))
    return t


def frame_rate(N: int, period: float) -> float:
    """Peak displayed chunk rate N / T_min (Lemma A.3)."""
    return N / period


# ---- App. A.3: actions -> DiT -> VAE --------------------------------------------------

def dit_vae_graph(N: int) -> PipelineGraph:
    """Operations D (DiT) and V (VAE decode); D -> V within a batch, each stage waits
    for its own previous batch; D is gated by arrival; every chunk leaves from V."""
    return PipelineGraph(ops=("D", "V"),
                         edges=(("D", "V", 0), ("D", "D", 1), ("V", "V", 1)),
                         entry=("D",), output=("V",) * N)


def dit_vae_colocated(tau_d: float, tau_v: float, kappa_dd: float = 0.0,
                      kappa_vv: float = 0.0) -> Deployment:
    """Both stages on one G-GPU resource, run D then V per batch; no D -> V lag."""
    return Deployment(assign={"D": "col", "V": "col"}, tau={"D": tau_d, "V": tau_v},
                      kappa={("D", "D", 1): kappa_dd, ("V", "V", 1): kappa_vv},
                      order={"col": ("D", "V")})


def dit_vae_disaggregated(tau_d: float, tau_v: float, kappa_dv: float = 0.0,
                          kappa_dd: float = 0.0, kappa_vv: float = 0.0) -> Deployment:
    """D on an X-GPU resource, V on a disjoint Y-GPU resource; D -> V may lag."""
    return Deployment(assign={"D": "dit", "V": "vae"}, tau={"D": tau_d, "V": tau_v},
                      kappa={("D", "V", 0): kappa_dv, ("D", "D", 1): kappa_dd,
                             ("V", "V", 1): kappa_vv})


def dit_vae_metrics(dep: Deployment, T: float) -> Tuple[float, float]:
    """Closed forms of App. A.3: d0* = T + tau_D + kappa_DV + tau_V (the D -> V path at
    k = 0, met by the earliest-start schedule at a sustainable T), and T_min = the
    resource loads and self-edge terms. Returns (d0*, T_min)."""
    td, tv = float(dep.tau["D"]), float(dep.tau["V"])
    d0 = T + td + dep.lag(("D", "V", 0)) + tv
    terms = [td + dep.lag(("D", "D", 1)), tv + dep.lag(("V", "V", 1))]
    if dep.assign["D"] == dep.assign["V"]:
        terms.append(td + tv)
    return d0, max(terms)


# ---- App. A.4: n denoising steps, SP vs stage PP ----------------------------------------

def denoise_graph(n: int, N: int) -> PipelineGraph:
    """Steps Q1..Qn chained within a batch; each step waits only for the same step of the
    previous batch (its own KV cache), which is what makes the stage pipeline legal."""
    if n < 1:
        raise ValueError("n >= 1")
    ops = tuple(f"Q{i}" for i in range(1, n + 1))
    edges = tuple((ops[i], ops[i + 1], 0) for i in range(n - 1)) + tuple((q, q, 1) for q in ops)
    return PipelineGraph(ops=ops, edges=edges, entry=(ops[0],), output=(ops[-1],) * N)


def sp_deployment(n: int, tq_sp: float) -> Deployment:
    """All n steps on one n-GPU sequence-parallel resource, each taking T_Q^SP(n)."""
    ops = tuple(f"Q{i}" for i in range(1, n + 1))
    return Deployment(assign={q: "sp" for q in ops}, tau={q: tq_sp for q in ops},
                      order={"sp": ops})


def pp_deployment(n: int, tq: float, kappas: Optional[Sequence[float]] = None) -> Deployment:
    """Step i on GPU i, each taking the single-GPU time T_Q; kappas[i] lags Q_{i+1} -> Q_{i+2}."""
    ops = tuple(f"Q{i}" for i in range(1, n + 1))
    kap = list(kappas) if kappas is not None else [0.0] * (n - 1)
    if len(kap) != n - 1:
        raise ValueError("need n - 1 lags")
    return Deployment(assign={q: f"gpu{i}" for i, q in enumerate(ops)}, tau={q: tq for q in ops},
                      kappa={(ops[i], ops[i + 1], 0): kap[i] for i in range(n - 1)})


def sp_metrics(n: int, tq_sp: float, T: float) -> Tuple[float, float]:
    """App. A.4, SP: d0* = T + n T_Q^SP(n), T_min = n T_Q^SP(n)."""
    return T + n * tq_sp, n * tq_sp


def pp_metrics(n: int, tq: float, T: float, kappas: Optional[Sequence[float]] = None) -> Tuple[float, float]:
    """App. A.4, PP: d0* = T + n T_Q + sum of the intra-batch lags, T_min = T_Q."""
    kap = list(kappas) if kappas is not None else [0.0] * (n - 1)
    return T + n * tq + sum(kap), tq


def main(argv: Optional[Iterable[str]] = None) -> None:
    """Print SP-vs-PP latency and period for a measured single-GPU step time."""
    ap = argparse.ArgumentParser(description="App. A period/latency calculator")
    ap.add_argument("--tq-ms", type=float, required=True,
                    help="single-GPU time of one denoising step for one batch, ms")
    ap.add_argument("--steps", type=int, default=4, help="denoising steps n (= GPUs)")
    ap.add_argument("--chunks", type=int, default=4, help="output chunks N per batch")
    ap.add_argument("--sp-speedup", type=float, default=None,
                    help="T_Q / T_Q^SP(n); default n (linear)")
    ap.add_argument("--lag-ms", type=float, default=0.0, help="PP inter-stage lag, ms")
    a = ap.parse_args(list(argv) if argv is not None else None)
    n, tq = a.steps, a.tq_ms
    tq_sp = tq / (a.sp_speedup if a.sp_speedup else n)
    kap = [a.lag_ms] * (n - 1)
    _, t_sp = sp_metrics(n, tq_sp, 1.0)
    _, t_pp = pp_metrics(n, tq, 1.0, kap)
    rows = {}
    for name, tmin, fn in (("sp", t_sp, lambda T: sp_metrics(n, tq_sp, T)),
                           ("pp", t_pp, lambda T: pp_metrics(n, tq, T, kap))):
        d0, _ = fn(tmin)
        rows[name] = {"T_min_ms": tmin, "d0_at_T_min_ms": d0,
                      "chunks_per_s": frame_rate(a.chunks, tmin / 1e3)}
    print(json.dumps(rows))


if __name__ == "__main__":
    main()
