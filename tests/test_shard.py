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


def _worker(rank, world, port, out_path):
    import torch.distributed as dist

    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    c = cfg()
    vals = I.tiny_gradient(3)[:37]
    tok = O.serialize(vals, 0)
    n_win = -(-tok.size // c.window)
    first, count = shard.window_ranges(n_win, world)[rank]
    codes = O.encode_windows(c, tok, first, count)
    bl = np.array([b for _, b in codes], np.uint32)
    crc = O.window_crcs(tok, c.window, first, count)
    pb = b"".join(cd for cd, _ in codes)
    header = O.encode(c, vals)[:64]  # the single-process container's header
    res = shard.gather_container(header, bl, crc, pb)
    if rank == 0:
        with open(out_path, "wb") as f:
            f.write(res)
    dist.destroy_process_group()


@pytest.mark.parametrize("world", [2])
def test_gloo_sharded_container_equals_single_process(tmp_path, world):
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        port = s.getsockname()[1]
    out = tmp_path / "c.bin"
    mp.start_processes(_worker, args=(world, port, str(out)), nprocs=world, start_method="spawn")
    got = out.read_bytes()
    c = cfg()
    ref = O.encode(c, I.tiny_gradient(3)[:37])
    assert got == ref
    h = O.parse_container(got)
    assert h["n_win"] == -(-37 * 9 // 40)
