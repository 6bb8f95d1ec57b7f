"""Host logic of the benchmark's multi-rank path, on CPU with gloo ranks:
each rank gets its own token shard (distinct seeds), the timed region is
closed by a barrier, the reported time is the max over ranks and the value is
the whole-job rate. Also the roofline arithmetic on known numbers."""
import os
import socket

import pytest
import torch.multiprocessing as mp

import bench


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    ws, r, local = bench.dist_env()
    seed = bench.shard_seed(0, r)
    bench.barrier(ws)
    t = bench.max_over_ranks(1.0 + r, ws)
    q.put((r, ws, local, seed, t))
    dist.destroy_process_group()


def test_two_gloo_ranks_shard_and_take_the_max():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    out = sorted(q.get(timeout=10) for _ in range(2))
    assert [o[0] for o in out] == [0, 1] and all(o[1] == 2 for o in out)
    assert out[0][3] != out[1][3]                       # distinct token shards
    assert all(o[4] == 2.0 for o in out)                # max over ranks
    assert bench.whole_job_rate(65536, 2, 10, 2.0) == 65536 * 2 * 10 / 2.0


def test_roofline_arithmetic():
    cfg = {"d": 768, "k": 64, "beam": 8, "levels": 5, "children": [0, 16, 16, 16, 16]}
    work = bench.algorithmic_work(cfg, 65536, 40.0, 2)
    assert work["encode"]["bytes"] == 65536 * 2052
    assert work["encode"]["tensor_flops"] == 65536 * 4 * 2 * 8 * 16 * 768
    assert work["backward"]["bytes"] == 65536 * 5376
    # 24,576 sign applications per token; a LOP3 flips a packed bf16 pair
    assert work["encode"]["int_ops"] == 65536 * 4 * 8 * 768 / 2
    assert bench.algorithmic_work(cfg, 1, 0.0, 4)["encode"]["int_ops"] == 4 * 8 * 768  # fp32: one each
    assert work["decode"]["fp_ops"] == 65536 * (40 * 768 + 3 * 768)
    peaks = {"hbm_gbs": 6781.4, "bf16_tflops_sustained": 1714.8, "sm_max_mhz": 2070.0}
    # encode: 12,288 LOP3 per token at 152 x 64 logic ops per clock (40 us at
    # T = 65536) bind before its 786,432 tensor flops at 1714.8 TFLOP/s (30 us)
    r = bench.roofline_for("encode", work["encode"], 200e-6, peaks, "measured")
    assert r["bound"] == "alu" and r["pipe"] == "integer logic" and abs(r["peak"] - 152 * 64 * 2070e6 / 1e12) < 1e-3
    assert abs(r["frac"] - work["encode"]["int_ops"] / 200e-6 / (152 * 64 * 2070e6)) < 1e-3
    assert abs(r["t_roofline_us"] - 40.0) < 0.1
    assert "maximum SM clock" in r["peak_source"]
    # with clock samples the ALU peak follows the median clock: a kernel run at
    # 1035 MHz is held to half the issue rate
    half = bench.roofline_for("encode", work["encode"], 200e-6, peaks, "measured", clocks={"sm_mhz": 1035.0})
    assert abs(half["peak"] - r["peak"] / 2) < 1e-3 and abs(half["frac"] - 2 * r["frac"]) < 1e-3
    assert "1035 MHz" in half["peak_source"]
    r = bench.roofline_for("decode", work["decode"], 100e-6, peaks, "measured")
    assert r["bound"] == "alu" and r["pipe"] == "fp32" and abs(r["peak"] - 152 * 128 * 2070e6 / 1e12) < 1e-3
    # a pure-HBM call picks the copy bandwidth, whatever the clock
    r = bench.roofline_for("copy", {"bytes": 6781.4e9 * 1e-3}, 2e-3, peaks, "measured", clocks={"sm_mhz": 900.0})
    assert r["bound"] == "hbm" and abs(r["frac"] - 0.5) < 1e-6 and r["unit"] == "GB/s"
    assert abs(r["frac_nominal"] - 6781.4 / 2 / 7900.0) < 1e-4  # and the nominal 7.9 TB/s beside it


def test_measured_traffic_follows_the_kernel_sources(monkeypatch, tmp_path):
    # figures are read for the size they were taken at, while the kernel's
    # sources hash as recorded; any other size or a changed source gives None
    f = tmp_path / "traffic.txt"
    h = bench.kernel_source_hash("decode")
    f.write_text("# comment line\n"
                 f"decode 65536 271791872 {h}\n"
                 "backward 65536 535708928 0000000000000000\n")
    monkeypatch.setattr(bench, "TRAFFIC_FILE", str(f))
    assert bench.measured_traffic("decode", 65536) == 271791872
    assert bench.measured_traffic("decode", 32768) is None
    assert bench.measured_traffic("backward", 65536) is None  # recorded for other sources
    assert bench.measured_traffic("encode", 65536) is None    # not recorded
    monkeypatch.setattr(bench, "kernel_source_hash", lambda name: "ffffffffffffffff")
    assert bench.measured_traffic("decode", 65536) is None
    monkeypatch.setattr(bench, "TRAFFIC_FILE", str(tmp_path / "absent.txt"))
    assert bench.measured_traffic("decode", 65536) is None
