"""Host logic of bench.py that needs no GPU: the clock summary keeps only the
nvidia-smi samples taken during the timed steps (the rule that a run's SM
clock is the median under load, with the throttle reasons seen then)."""
import datetime
import os

import bench


class _FakeProc:
    def terminate(self):
        pass

    def wait(self, timeout=None):
        return 0


def _sampler(tmp_path, rows, t0, t1):
    s = bench.ClockSampler("0")
    s.path = str(tmp_path / "clocks.csv")
    with open(s.path, "w") as f:
        for ts, sm, mx, pw, reasons in rows:
            stamp = datetime.datetime.fromtimestamp(ts).strftime("%Y/%m/%d %H:%M:%S.%f")[:-3]
            f.write(f"{stamp}, {sm}, {mx}, {pw}, " + ", ".join(reasons) + "\n")
    s.fh = open(os.devnull, "w")
    s.proc = _FakeProc()
    s.t0, s.t1 = t0, t1
    return s


def test_only_samples_inside_the_timed_steps_count(tmp_path):
    base = 1_800_000_000.0
    idle = ("Not Active",) * 4
    capped = ("Not Active", "Not Active", "Not Active", "Active")
    rows = [(base + 0.00, 2070, 2070, 150.0, idle),      # before the timed steps
            (base + 0.05, 2070, 2070, 160.0, idle),
            (base + 0.30, 1500, 2070, 900.0, capped),    # timed steps
            (base + 0.35, 1520, 2070, 910.0, capped),
            (base + 0.40, 1510, 2070, 905.0, capped),
            (base + 0.90, 2070, 2070, 140.0, ("Not Active", "Active", "Not Active", "Not Active"))]  # after
    out = _sampler(tmp_path, rows, base + 0.25, base + 0.45).stop()
    assert out["samples"] == 3
    assert out["sm_mhz"] == 1510
    assert out["sm_mhz_min"] == 1500 and out["sm_max_mhz"] == 2070
    assert out["reasons"] == ["sw_power_cap"]           # the thermal flag after the window is not counted
    assert out["window"] == "timed steps only"
    assert not os.path.exists(str(tmp_path / "clocks.csv"))


def test_falls_back_to_every_sample_and_says_so(tmp_path):
    base = 1_800_000_000.0
    rows = [(base, 2000, 2070, 200.0, ("Not Active",) * 4),
            (base + 0.05, 1800, 2070, 800.0, ("Active", "Not Active", "Not Active", "Not Active"))]
    out = _sampler(tmp_path, rows, base + 5.0, base + 6.0).stop()
    assert out["samples"] == 2 and out["sm_mhz"] == 1900
    assert out["reasons"] == ["hw_slowdown"]
    assert out["window"].startswith("whole sampler run")


def test_missing_nvidia_smi_is_reported():
    s = bench.ClockSampler("0")
    out = s.stop()
    assert out["sm_mhz"] is None and out["reasons"] == ["nvidia-smi unavailable"]


def _max_rank_main(rank, world, port, out_dir):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    got = bench._max_over_ranks(dist, 1.0 + 2.5 * rank, "cpu")
    with open(os.path.join(out_dir, f"r{rank}.txt"), "w") as f:
        f.write(repr(got))
    dist.destroy_process_group()


def test_step_time_is_the_maximum_over_ranks(tmp_path):
    """The whole-job rate divides by the slowest rank's time: every rank gets
    the maximum (two gloo ranks on the CPU); one rank keeps its own."""
    import socket

    import torch.multiprocessing as mp
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        port = s.getsockname()[1]
    mp.spawn(_max_rank_main, args=(2, port, str(tmp_path)), nprocs=2, join=True)
    for r in range(2):
        assert float(open(tmp_path / f"r{r}.txt").read()) == 3.5
    assert bench._max_over_ranks(None, 1.25, "cpu") == 1.25


def test_traffic_is_reported_only_for_the_captured_source(tmp_path, monkeypatch):
    """roofline.traffic comes from the committed ncu record while the kernel's
    source file still has the hash recorded with the capture; a changed source
    or a kernel without a record gives null."""
    import hashlib
    import json

    src = tmp_path / "k.cu"
    src.write_text("// kernel as captured\n")
    (tmp_path / "profiles").mkdir()
    rec = {"k": {"source": "k.cu", "sha256": hashlib.sha256(src.read_bytes()).hexdigest(),
                 "dram_bytes_per_launch": 123}}
    (tmp_path / "profiles" / "ncu_traffic.json").write_text(json.dumps(rec))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench._ncu_traffic("k") == 123
    assert bench._ncu_traffic("other") is None
    src.write_text("// kernel changed after the capture\n")
    assert bench._ncu_traffic("k") is None
