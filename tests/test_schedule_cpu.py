"""Pins for the App. A period/latency calculator.

The simulator (earliest-start cyclic schedule) and the closed forms of App. A.3/A.4 are
two independent formulations; each is checked against the other and against the
inequalities of Lemmas A.1-A.3, on random timings and on one worked example whose
numbers are computed by hand below.
"""

import itertools
import math

import numpy as np
import pytest

from paper_2607_18171_gb300 import schedule as sc

BATCHES = 40


def _close(a, b, tol=1e-9):
    return abs(a - b) <= tol * max(1.0, abs(a), abs(b))


# ---- App. A.3: DiT -> VAE --------------------------------------------------------------

@pytest.mark.parametrize("trial", range(40))
def test_dit_vae_colocated_matches_closed_form(trial):
    rng = np.random.default_rng([31, trial])
    td, tv = rng.uniform(0.05, 1.0, 2)
    kdd, kvv = rng.uniform(0.0, 0.5, 2) * (rng.random(2) < 0.5)
    N = int(rng.integers(1, 9))
    g = sc.dit_vae_graph(N)
    dep = sc.dit_vae_colocated(td, tv, kdd, kvv)
    d0_cf, tmin_cf = sc.dit_vae_metrics(dep, 1.0)
    assert _close(sc.t_min(g, dep), tmin_cf)
    assert _close(tmin_cf, max(td + tv, td + kdd, tv + kvv))
    T = tmin_cf * (1.0 + rng.uniform(0.0, 0.5))
    s = sc.simulate(g, dep, T, BATCHES)
    d0_cf, _ = sc.dit_vae_metrics(dep, T)
    assert _close(sc.display_offset(s), d0_cf)
    assert _close(d0_cf, T + td + tv)


@pytest.mark.parametrize("trial", range(40))
def test_dit_vae_disaggregated_matches_closed_form(trial):
    rng = np.random.default_rng([32, trial])
    td, tv, kdv = rng.uniform(0.05, 1.0, 3)
    kdd, kvv = rng.uniform(0.0, 0.5, 2) * (rng.random(2) < 0.5)
    N = int(rng.integers(1, 9))
    g = sc.dit_vae_graph(N)
    dep = sc.dit_vae_disaggregated(td, tv, kdv, kdd, kvv)
    _, tmin_cf = sc.dit_vae_metrics(dep, 1.0)
    assert _close(sc.t_min(g, dep), tmin_cf)
    assert _close(tmin_cf, max(td + kdd, tv + kvv))
    T = tmin_cf * (1.0 + rng.uniform(0.0, 0.5))
    s = sc.simulate(g, dep, T, BATCHES)
    d0_cf, _ = sc.dit_vae_metrics(dep, T)
    assert _close(sc.display_offset(s), d0_cf)
    assert _close(d0_cf, T + td + kdv + tv)


@pytest.mark.parametrize("trial", range(20))
def test_colocation_latency_and_disaggregation_period(trial):
    """Prop. 'co-location is latency-optimal' and 'disaggregation can be throughput-optimal'
    on random splits: with tau_col <= tau_pipe, d0*(col) <= d0*(pipe) at a T both sustain;
    the best split's T_min is the min over splits."""
    rng = np.random.default_rng([33, trial])
    td_c, tv_c = rng.uniform(0.05, 0.5, 2)
    splits = []
    for _ in range(4):
        td_p = td_c * rng.uniform(1.0, 3.0)
        tv_p = tv_c * rng.uniform(1.0, 3.0)
        splits.append(sc.dit_vae_disaggregated(td_p, tv_p, rng.uniform(0.0, 0.1)))
    col = sc.dit_vae_colocated(td_c, tv_c)
    g = sc.dit_vae_graph(4)
    T = max([sc.t_min(g, col)] + [sc.t_min(g, d) for d in splits]) * 1.1
    d_col = sc.display_offset(sc.simulate(g, col, T, BATCHES))
    for d in splits:
        assert d_col <= sc.display_offset(sc.simulate(g, d, T, BATCHES)) + 1e-12
    best = min(splits, key=lambda d: sc.t_min(g, d))
    assert all(sc.t_min(g, best) <= sc.t_min(g, d) for d in splits)


def test_dit_vae_worked_example():
    """Hand-computed: tau_D = 0.3, tau_V = 0.2 co-located; 0.3 and 0.25 disaggregated with
    no lag; N = 4 chunks per batch, requested period T = 0.5.
    Co-located:    d0* = 0.5 + 0.3 + 0.2 = 1.0,   T_min = 0.3 + 0.2 = 0.5, 4 / 0.5 = 8 chunks/s.
    Disaggregated: d0* = 0.5 + 0.3 + 0.25 = 1.05, T_min = max(0.3, 0.25) = 0.3, 13.33 chunks/s."""
    g = sc.dit_vae_graph(4)
    col = sc.dit_vae_colocated(0.3, 0.2)
    pipe = sc.dit_vae_disaggregated(0.3, 0.25)
    assert _close(sc.display_offset(sc.simulate(g, col, 0.5, BATCHES)), 1.0)
    assert _close(sc.display_offset(sc.simulate(g, pipe, 0.5, BATCHES)), 1.05)
    assert _close(sc.t_min(g, col), 0.5) and _close(sc.t_min(g, pipe), 0.3)
    assert _close(sc.frame_rate(4, sc.t_min(g, col)), 8.0)
    assert _close(sc.frame_rate(4, sc.t_min(g, pipe)), 40.0 / 3.0)
    # the first chunk binds: Y_00 = R_0 + tau_D + tau_V = 0.5 + 0.5 and d0* - Y_00 = 0
    s = sc.simulate(g, col, 0.5, 3)
    assert _close(s.ready(0, 0), 1.0) and _close(s.start[(1, "D")], 1.0)


# ---- App. A.4: SP vs stage PP ----------------------------------------------------------

@pytest.mark.parametrize("n", [1, 2, 3, 4, 6])
@pytest.mark.parametrize("trial", range(6))
def test_sp_pp_match_closed_forms(n, trial):
    rng = np.random.default_rng([34, n, trial])
    tq = float(rng.uniform(0.05, 0.5))
    tq_sp = tq / rng.uniform(1.0, n) if n > 1 else tq        # sublinear: T_Q <= n T_Q^SP
    kap = list(rng.uniform(0.0, 0.05, n - 1))
    N = int(rng.integers(1, 6))
    g = sc.denoise_graph(n, N)
    sp, pp = sc.sp_deployment(n, tq_sp), sc.pp_deployment(n, tq, kap)
    _, tsp = sc.sp_metrics(n, tq_sp, 1.0)
    _, tpp = sc.pp_metrics(n, tq, 1.0, kap)
    assert _close(sc.t_min(g, sp), tsp) and _close(sc.t_min(g, pp), tpp)
    assert tpp <= tsp + 1e-12                                   # PP period <= SP period
    T = max(tsp, tpp) * (1.0 + rng.uniform(0.0, 0.3))
    d_sp = sc.display_offset(sc.simulate(g, sp, T, BATCHES))
    d_pp = sc.display_offset(sc.simulate(g, pp, T, BATCHES))
    assert _close(d_sp, sc.sp_metrics(n, tq_sp, T)[0])
    assert _close(d_pp, sc.pp_metrics(n, tq, T, kap)[0])
    assert d_sp <= d_pp + 1e-12                                 # SP latency <= PP latency
    assert _close(d_pp - d_sp, n * (tq - tq_sp) + sum(kap))


def test_pp_runs_steps_of_different_batches_concurrently():
    """At T = T_Q the PP stages overlap: Q_i of batch j runs while Q_{i+1} runs batch j-1."""
    g = sc.denoise_graph(4, 1)
    s = sc.simulate(g, sc.pp_deployment(4, 1.0), 1.0, 8)
    for j in range(1, 8):
        for i in range(1, 4):
            a = (s.start[(j, f"Q{i}")], s.finish[(j, f"Q{i}")])
            b = (s.start[(j - 1, f"Q{i + 1}")], s.finish[(j - 1, f"Q{i + 1}")])
            assert a == b


# ---- Lemmas A.1-A.3 on random templates -------------------------------------------------

def _random_template(rng):
    m = int(rng.integers(2, 6))
    ops = tuple(f"v{i}" for i in range(m))
    edges = []
    for a, b in itertools.combinations(range(m), 2):          # forward intra-batch DAG
        if rng.random() < 0.5:
            edges.append((ops[a], ops[b], 0))
    for a in range(m):
        for b in range(m):
            if rng.random() < 0.2:
                edges.append((ops[a], ops[b], 1))
    for i in range(1, m):                                      # every op reachable from v0
        if not any(e[1] == ops[i] and e[2] == 0 for e in edges):
            edges.append((ops[int(rng.integers(0, i))], ops[i], 0))
    N = int(rng.integers(1, 5))
    out = tuple(ops[int(rng.integers(0, m))] for _ in range(N))
    g = sc.PipelineGraph(ops, tuple(sorted(set(edges))), (ops[0],), out)
    n_res = int(rng.integers(1, m + 1))
    assign = {v: f"r{int(rng.integers(0, n_res))}" for v in ops}
    tau = {v: float(rng.uniform(0.05, 1.0)) for v in ops}
    kappa = {e: float(rng.uniform(0.0, 0.3)) * (rng.random() < 0.5) for e in g.edges}
    return g, sc.Deployment(assign, tau, kappa)          # template order is topological


@pytest.mark.parametrize("trial", range(30))
def test_path_bound_and_display_offset(trial):
    """Lemma A.2 lower-bounds the simulated d0* for every entry path; Lemma A.1: the
    display schedule at d0* is feasible and one just below it is not."""
    rng = np.random.default_rng([35, trial])
    g, dep = _random_template(rng)
    T = sc.t_min(g, dep) * (1.0 + rng.uniform(0.0, 0.5)) + 1e-3
    s = sc.simulate(g, dep, T, BATCHES)
    d0 = sc.display_offset(s)
    for k in range(g.n_chunks):
        for p in sc.simple_paths(g, g.output[k]):
            if p:
                assert sc.path_bound(p, dep, T, k, g.n_chunks) <= d0 + 1e-9
    assert sc.best_path_bound(g, dep, T) <= d0 + 1e-9
    assert sc.display_feasible(s, d0)
    assert not sc.display_feasible(s, d0 - 1e-6)


@pytest.mark.parametrize("trial", range(30))
def test_resource_load_bound(trial):
    """Lemma A.3 (a necessary condition): below T_min some resource falls further behind
    every batch, so the completion of each batch's work, relative to jT, grows by at
    least (T_min - T) per batch. The lemma counts all of a batch's work as needed for
    its output; the backlog is therefore taken over every instance."""
    rng = np.random.default_rng([36, trial])
    g, dep = _random_template(rng)
    tm = sc.t_min(g, dep)
    load = sc.resource_load(g, dep)
    assert _close(sum(load.values()), sum(dep.tau.values()))
    assert tm >= max(load.values()) - 1e-12
    T = 0.9 * tm
    s = sc.simulate(g, dep, T, 300)
    backlog = [max(s.finish[(j, v)] for v in g.ops) - j * T for j in range(300)]
    assert backlog[-1] - backlog[-201] >= 200 * 0.1 * tm - 2 * tm


def test_t_min_settles_for_the_paper_deployments():
    """At T = T_min the per-batch offsets of App. A.3/A.4's deployments are constant."""
    cases = [(sc.dit_vae_graph(3), sc.dit_vae_colocated(0.3, 0.2, 0.1, 0.25)),
             (sc.dit_vae_graph(3), sc.dit_vae_disaggregated(0.3, 0.25, 0.05, 0.1, 0.0)),
             (sc.denoise_graph(4, 2), sc.sp_deployment(4, 0.1)),
             (sc.denoise_graph(4, 2), sc.pp_deployment(4, 0.3, [0.01, 0.02, 0.03]))]
    for g, dep in cases:
        off = sc.offsets(sc.simulate(g, dep, sc.t_min(g, dep), 60))
        assert max(off[5:]) - min(off[5:]) <= 1e-9


def test_self_edge_term_binds():
    """A self-edge lag longer than the resource load sets T_min (App. A.3's extra terms):
    D alone on its resource with tau = 0.2 and kappa_DD = 0.3 sustains T = 0.5, not 0.2."""
    g = sc.dit_vae_graph(2)
    dep = sc.dit_vae_disaggregated(0.2, 0.1, 0.0, kappa_dd=0.3)
    assert _close(sc.t_min(g, dep), 0.5)
    grow = sc.offsets(sc.simulate(g, dep, 0.45, 100))
    assert grow[-1] - grow[-51] > 1.0
    flat = sc.offsets(sc.simulate(g, dep, 0.5, 100))
    assert _close(flat[-1], flat[-51])


def test_validation():
    g = sc.dit_vae_graph(2)
    with pytest.raises(ValueError):
        sc.PipelineGraph(("a", "a"), (), ("a",), ("a",))
    with pytest.raises(ValueError):
        sc.PipelineGraph(("a",), (("a", "b", 0),), ("a",), ("a",))
    with pytest.raises(ValueError):
        sc.simulate(g, sc.dit_vae_colocated(0.1, 0.1), 0.0, 3)
    bad = sc.Deployment({"D": "r", "V": "r"}, {"D": 0.1, "V": 0.1}, order={"r": ("V", "D")})
    with pytest.raises(ValueError):                  # V before D contradicts D -> V
        sc.simulate(g, bad, 1.0, 2)
    with pytest.raises(ValueError):
        sc.Deployment({"D": "r"}, {"D": 0.1}).cyclic_order(g)


def test_cli(capsys):
    sc.main(["--tq-ms", "0.8", "--steps", "4", "--chunks", "3", "--sp-speedup", "2.5"])
    import json
    row = json.loads(capsys.readouterr().out)
    assert _close(row["pp"]["T_min_ms"], 0.8)
    assert _close(row["sp"]["T_min_ms"], 4 * 0.8 / 2.5)
    assert _close(row["pp"]["chunks_per_s"], 3 / 0.8e-3)
    assert math.isfinite(row["sp"]["d0_at_T_min_ms"])
