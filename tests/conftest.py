import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
for p in (ROOT, os.path.dirname(os.path.abspath(__file__))):
    if p not in sys.path:
        sys.path.insert(0, p)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built libvd.so")


@pytest.fixture(scope="session")
def orc():
    import oracle
    return oracle.load()


def pytest_terminal_summary(terminalreporter):
    """The worst score error each GPU test saw against the oracle, per rule:
    relative (over scores above 1e-6) and as a fraction of the tolerance."""
    try:
        from vd_gpu import TRAJECTORIES, WORST
    except Exception:
        return
    tr = terminalreporter
    if TRAJECTORIES:
        tr.section("free-running trajectories, CUDA path vs the oracle's own loop")
        for name, t in sorted(TRAJECTORIES.items()):
            fd = t["first_divergence"]
            tr.write_line(f"{name:<16} {t['units']} units, {t['events']} evicting events: "
                          f"{t['identical_events']} identical, first divergence "
                          f"{'none' if fd is None else f'event {fd[0]} (unit {fd[1]})'}, "
                          f"final caches share {100 * t['final_overlap']:.1f} % of their tokens")
    if not WORST:
        return
    tr.section("worst score error vs the fp64 oracle (tolerance 1e-5 relative)")
    for (test, rule), (rel, frac, count) in sorted(WORST.items()):
        tr.write_line(f"{test:<60} {rule:<8} rel {rel:.2e}  of tol {frac:.3f}  ({count} scores)")
    by_rule = {}
    for (_, rule), (rel, frac, _) in WORST.items():
        r = by_rule.setdefault(rule, [0.0, 0.0])
        r[0], r[1] = max(r[0], rel), max(r[1], frac)
    for rule, (rel, frac) in sorted(by_rule.items()):
        tr.write_line(f"overall {rule:<8} worst relative error {rel:.3e}, worst fraction of "
                      f"the tolerance {frac:.3f}")
