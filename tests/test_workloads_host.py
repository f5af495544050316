"""Host-side workload helpers (no GPU): static view schedules, the policy's
view levels, the fill's byte count and the benchmark's new flags."""
import numpy as np
import pytest

import bench
from paper_2608_01821_gb300 import workloads


@pytest.mark.parametrize("name", ["tiny", "single", "single_mixed", "ragged"])
def test_static_views_and_policy_levels(name):
    w = workloads.make(name)
    low, mid, high = workloads.policy_view_levels(w)
    assert high == 0 and low == min(2, w.n_levels - 1)
    assert mid == (w.n_levels if w.mixed else 1)
    for which, lv in (("high", high), ("mid", mid), ("low", low)):
        v = workloads.make(name)
        workloads.set_static_view(v, which)
        assert v.schedule.shape == w.schedule.shape and (v.schedule == lv).all()
        # every step of a static schedule has the same length, that of the view
        lens = {tuple(v.step_lengths(t)) for t in range(v.T)}
        assert lens == {tuple(v.seq_len(b, lv) for b in range(v.batch))}
    # views by length: coarse < mixed or level 1 < high
    assert all(w.seq_len(b, low) < w.seq_len(b, mid) < w.seq_len(b, high) for b in range(w.batch) if w.tiles[b])


def test_fill_bytes_count_every_view_blocks_text_and_the_mixed_rows():
    w = workloads.make("single")
    text = w.prompt[0] + w.resp[0]
    assert w.view_fill_bytes() == w.n_views() * text * w.C * 4
    m = workloads.make("single_mixed")
    mixed_rows = m.tiles[0] * m.view_rows_per_tile(m.n_levels)
    assert m.view_fill_bytes() == (m.n_views() * text + mixed_rows) * m.C * 4


def test_demand_prior_is_table_a_in_turn():
    w = workloads.make("ragged")
    d = workloads.request_demands(w)
    assert d[:5] == list(workloads.DEMAND_PRIOR) and d[5] == 1.0 and len(d) == w.batch
    assert np.all(np.diff(workloads.DEMAND_PRIOR) < 0)


def test_bench_parses_the_policy_and_schedule_flags(monkeypatch):
    seen = {}

    def fake_backbone(args, rank, world, local):
        seen.update(vars(args))
        return None

    monkeypatch.setattr(bench, "run_backbone", fake_backbone)
    monkeypatch.setattr(bench, "init_dist", lambda world, backend: None)
    bench.main(["--model", "full", "--policy", "--uniform-demand", "--orientation", "late", "--budget", "0.45",
                "--alpha", "0.5", "--schedule", "high", "--layers", "4", "--no-cpu-baseline"])
    assert seen["policy"] and seen["uniform_demand"] and seen["orientation"] == "late"
    assert seen["budget"] == 0.45 and seen["alpha"] == 0.5 and seen["schedule"] == "high" and seen["layers"] == 4
