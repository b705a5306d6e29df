"""Window sharding across ranks (the multi-GPU form of the encode path): world-size-2 gloo
processes on the CPU each code their window range (with the oracle), exchange bit lengths and
payload slices, and rank 0's assembled container equals the single-process container byte for
byte."""
import os
import socket

import numpy as np
import pytest
import torch.multiprocessing as mp

import oracle as O
from paper_2409_17836_gb300 import inputs as I
from paper_2409_17836_gb300 import shard


def cfg():
    return O.OracleConfig(n_layers=1, d_model=32, n_heads=2, n_kv_heads=1, d_ffn=64, vocab=32, bf16=False, window=40,
                          cdf_bits=16, weight_seed=4, init_std=0.3)


def test_window_ranges():
    for n, w in [(10, 2), (7, 3), (3, 4), (1314, 8)]:
        r = shard.window_ranges(n, w)
        assert len(r) == w and sum(c for _, c in r) == n
        assert all(r[i][0] + r[i][1] == r[i + 1][0] for i in range(w - 1))
        assert max(c for _, c in r) - min(c for _, c in r) <= 1


def _worker(rank, world, port, out_path, n_values):
    import torch.distributed as dist

    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    c = cfg()
    vals = I.tiny_gradient(3)[:n_values]
    tok = O.serialize(vals, 0)
    n_win = -(-tok.size // c.window)
    first, count = shard.window_ranges(n_win, world)[rank]
    if count:
        codes = O.encode_windows(c, tok, first, count)
        bl = np.array([b for _, b in codes], np.uint32)
        crc = O.window_crcs(tok, c.window, first, count)
        pb = b"".join(cd for cd, _ in codes)
    else:  # more ranks than windows: this rank contributes empty parts
        bl, crc, pb = np.zeros(0, np.uint32), np.zeros(0, np.uint32), b""
    header = O.encode(c, vals)[:64]  # the single-process container's header
    res = shard.gather_container(header, bl, crc, pb)
    if rank == 0:
        with open(out_path, "wb") as f:
            f.write(res)
    else:
        assert res is None
    dist.destroy_process_group()


@pytest.mark.parametrize("world,n_values", [(2, 37), (3, 37), (4, 11)])
def test_gloo_sharded_container_equals_single_process(tmp_path, world, n_values):
    """(4, 11): 99 tokens in 3 windows over 4 ranks, so rank 3 codes nothing."""
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        port = s.getsockname()[1]
    out = tmp_path / "c.bin"
    mp.start_processes(_worker, args=(world, port, str(out), n_values), nprocs=world, start_method="spawn")
    got = out.read_bytes()
    c = cfg()
    ref = O.encode(c, I.tiny_gradient(3)[:n_values])
    assert got == ref
    h = O.parse_container(got)
    assert h["n_win"] == -(-n_values * 9 // 40)
    if world == 4:
        assert shard.window_ranges(h["n_win"], world)[3][1] == 0


def test_assemble_rejects_inconsistent_parts():
    header = bytes(64)
    bl = [np.array([9, 17], np.uint32)]  # 2 + 3 bytes of codes
    crc = [np.array([1, 2], np.uint32)]
    good = shard.assemble(header, bl, crc, [b"\x01\x02\x03\x04\x05"])
    assert len(good) == 64 + 8 + 8 + 5
    assert np.array_equal(shard.payload_offsets([9, 17, 0, 8]), [0, 2, 5, 5, 6])
    with pytest.raises(ValueError):
        shard.assemble(header, bl, crc, [b"\x01\x02\x03\x04"])  # one payload byte short
    with pytest.raises(ValueError):
        shard.assemble(header, bl, [np.array([1], np.uint32)], [b"\x01\x02\x03\x04\x05"])


def _worker_leaves(rank, world, port, out_path):
    """Rank 1 leaves before the exchange; rank 0's gather must fail within the group's timeout."""
    import datetime
    import time

    import torch.distributed as dist

    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world, timeout=datetime.timedelta(seconds=10))
    if rank == 1:
        return  # exits without joining the exchange (its sockets close with the process)
    t0 = time.monotonic()
    try:
        shard.gather_container(bytes(64), np.zeros(1, np.uint32), np.zeros(1, np.uint32), b"")
        msg = "no error"
    except Exception as e:  # the failure surfaces on the host as an exception
        msg = f"error after {time.monotonic() - t0:.1f} s: {type(e).__name__}"
    with open(out_path, "w") as f:
        f.write(msg)


def test_gloo_rank_leaving_before_exchange_is_reported(tmp_path):
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        port = s.getsockname()[1]
    out = tmp_path / "msg.txt"
    mp.start_processes(_worker_leaves, args=(2, port, str(out)), nprocs=2, start_method="spawn")
    msg = out.read_text()
    assert msg.startswith("error after"), msg
    assert float(msg.split()[2]) < 30.0, msg
