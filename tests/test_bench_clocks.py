"""bench.py's clock summary keeps the nvidia-smi samples taken inside the
timed region (host wall clock), so that idle samples before it cannot hide
a throttled or clock-locked run."""
import datetime
import importlib.util
import os

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench():
    spec = importlib.util.spec_from_file_location("bench_mod", os.path.join(ROOT, "bench.py"))
    m = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(m)
    return m


def _line(t, mhz, reason="Not Active"):
    ts = datetime.datetime.fromtimestamp(t).strftime("%Y/%m/%d %H:%M:%S.%f")[:-3]
    return f"{ts}, {mhz}, 2070, 900.0, 0x0, {reason}, Not Active, Not Active, Not Active\n"


def test_rows_inside_the_region():
    b = _bench()
    t0 = 1_800_000_000.0
    lines = [_line(t0 - 0.2, 900), _line(t0 + 0.05, 2070), _line(t0 + 0.10, 2060, "Active"),
             _line(t0 + 0.4, 900)]
    rows, where = b.clock_rows_in_region(lines, t0, t0 + 0.2)
    assert where == "in region"
    assert [r[1] for r in rows] == ["2070", "2060"]
    assert rows[1][5] == "Active"


def test_short_region_takes_the_first_sample_after_its_start():
    b = _bench()
    t0 = 1_800_000_000.0
    lines = [_line(t0 - 0.03, 900), _line(t0 + 0.04, 2070), _line(t0 + 0.09, 2070)]
    rows, where = b.clock_rows_in_region(lines, t0, t0 + 0.02)
    assert where == "first after start" and len(rows) == 1 and rows[0][1] == "2070"


def test_unmarked_region_keeps_every_row():
    b = _bench()
    lines = [_line(1_800_000_000.0, 2070), "garbage\n"]
    rows, where = b.clock_rows_in_region(lines, None, None)
    assert where == "all" and len(rows) == 1
