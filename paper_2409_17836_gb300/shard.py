"""Encoding one gradient on several GPUs: windows are independent (Sec. 4 "Compression": every
window is coded from its own BOS), so each rank codes a contiguous range of windows with no data
exchange. The one exchange step builds the container: the ranks all-gather their windows' bit
lengths and token checksums (8 bytes per window) and payload slices; an exclusive scan of the
byte lengths gives each slice's offset, and the slices are concatenated in rank order after the
header, the length table and the checksum table."""
from __future__ import annotations

import numpy as np


def window_ranges(n_win: int, world: int) -> list[tuple[int, int]]:
    """Contiguous (first, count) window ranges, sizes differing by at most one."""
    base, extra = divmod(n_win, world)
    out, w0 = [], 0
    for r in range(world):
        cnt = base + (1 if r < extra else 0)
        out.append((w0, cnt))
        w0 += cnt
    return out


def payload_offsets(bitlen_all: np.ndarray) -> np.ndarray:
    """Exclusive scan of the code byte lengths (ceil(bits / 8)), one more entry for the total."""
    nb = (np.asarray(bitlen_all, dtype=np.int64) + 7) // 8
    return np.concatenate([[0], np.cumsum(nb)])


def assemble(header: bytes, bitlen_parts: list[np.ndarray], crc_parts: list[np.ndarray],
             payload_parts: list[bytes]) -> bytes:
    """The container from the header and every rank's bit lengths, token checksums and payload
    slice (rank order)."""
    bl = np.concatenate([np.asarray(b, dtype="<u4") for b in bitlen_parts])
    crc = np.concatenate([np.asarray(c, dtype="<u4") for c in crc_parts])
    if crc.size != bl.size:
        raise ValueError("one token checksum per window expected")
    offs = payload_offsets(bl)
    body = b"".join(payload_parts)
    if len(body) != offs[-1]:
        raise ValueError("payload slices do not match their bit lengths")
    return header + bl.tobytes() + crc.tobytes() + body


def gather_container(header: bytes, bitlen: np.ndarray, crc: np.ndarray, payload: bytes, group=None) -> bytes | None:
    """Exchange step over torch.distributed: every rank contributes its range's bit lengths, token
    checksums and payload slice; rank 0 returns the assembled container, the other ranks None."""
    import torch.distributed as dist

    world = dist.get_world_size(group)
    parts: list = [None] * world
    dist.all_gather_object(parts, (np.asarray(bitlen, dtype=np.uint32), np.asarray(crc, dtype=np.uint32),
                                   bytes(payload)), group=group)
    if dist.get_rank(group) != 0:
        return None
    return assemble(header, [p[0] for p in parts], [p[1] for p in parts], [p[2] for p in parts])


def encode_sharded(ctx, values, rank: int, world: int, group=None) -> bytes | None:
    """lmgc_encode of `values` (a CUDA tensor on this rank's GPU) with the windows split over
    `world` ranks; returns the container on rank 0."""
    from . import lmgc as L

    n_win = -(-L.lmgc_serial_tokens(ctx, values.numel()) // ctx.cfg.window)
    first, count = window_ranges(n_win, world)[rank]
    if count:
        payload, bitlen, crc = L.lmgc_encode_windows(ctx, values, first, count)
        pb, bl = payload.cpu().numpy().tobytes(), bitlen.cpu().numpy().view(np.uint32)
        cr = crc.cpu().numpy().view(np.uint32)
    else:
        pb, bl, cr = b"", np.zeros(0, np.uint32), np.zeros(0, np.uint32)
    return gather_container(L.lmgc_container_header(ctx, values.numel()), bl, cr, pb, group)
