"""Oracle: the drafted frontier and the spatial dependency mask (float-free).

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

Sec. 3.1, Eq. 1: the n x n token grid is flattened in raster order after the
text prefix c, and each token conditions on c and every earlier token.
Sec. 3.3: SSD drafts with horizontal heads until the current row is complete,
then drafts up to k_v following rows at once (column-wise independence: one
token per column from the completed row above).  One verification step
therefore covers the remainder of the current row plus the k_v rows below it.

reading: a position is committed iff its flat index is below cache_len; the
frontier is the remainder of row y0 (the row holding the first uncommitted
token) plus the next k_v rows, clipped at the grid's last row.  Grid rows
are laid out with ``row_stride`` flat slots (W, or W + 1 when the backbone
emits an end-of-line token after each row); the frontier rule itself is only
defined here for row_stride == W.
"""
from __future__ import annotations

import numpy as np


def frontier(grid_h: int, grid_w: int, prefix_len: int, cache_len: int, k_v: int = 1,
             k_h: int = 0):
    """Return the drafted grid coordinates [(y, x), ...] in raster order.

    Horizontal part: (y0, x) for x = c .. W-1, where the first uncommitted
    token sits at (y0, c); with k_h > 0 only the first k_h of them (Sec. 3.3:
    k_h horizontal heads draft offsets +1 .. +k_h along the row).  Vertical
    part: rows y0+1 .. y0+k_v, all columns -- reading: only when the
    horizontal part completes the row, so the frontier stays contiguous in
    raster order.  Rows at or beyond grid_h do not exist and are dropped.
    """
    n_c = cache_len - prefix_len  # committed image tokens
    if n_c < 0 or n_c > grid_h * grid_w:
        raise ValueError("cache_len outside [prefix_len, prefix_len + H*W]")
    y0, c = divmod(n_c, grid_w)
    coords = []
    h = grid_w - c if k_h <= 0 else min(k_h, grid_w - c)
    if y0 < grid_h:
        coords += [(y0, x) for x in range(c, c + h)]            # horizontal heads
    if c + h == grid_w:
        for dy in range(1, k_v + 1):                            # vertical heads
            if y0 + dy < grid_h:
                coords += [(y0 + dy, x) for x in range(grid_w)]
    return coords


def grid_index(coords, grid_w: int) -> np.ndarray:
    """Grid index g = y * W + x of each (y, x)."""
    return np.array([y * grid_w + x for (y, x) in coords], dtype=np.int64)


def flat_position(y: int, x: int, prefix_len: int, row_stride: int) -> int:
    """Position of grid token (y, x) in the backbone's flattened sequence."""
    return prefix_len + y * row_stride + x


def coord_of_flat(pos: int, prefix_len: int, row_stride: int):
    """Inverse of flat_position for a non-prefix slot: (y, x); x == W marks the
    end-of-line slot when row_stride == W + 1.  Returns None for prefix slots."""
    if pos < prefix_len:
        return None
    return divmod(pos - prefix_len, row_stride)


def coord_mask(draft_coords, cache_len: int, prefix_len: int, row_stride: int) -> np.ndarray:
    """Visibility mask [n_d, cache_len + n_d] built from grid coordinates.

    Keys are the cache_len committed slots followed by the n_d drafts.  A
    draft at (y, x) sees a key iff the key is a text-prefix token, or the key
    sits on an earlier grid row, or on the same row at a column <= x (Eq. 1's
    conditioning set, which may include other drafts: App. "Deviation").
    """
    n_d = len(draft_coords)
    keys = []
    for s in range(cache_len):
        keys.append(coord_of_flat(s, prefix_len, row_stride))
    keys += list(draft_coords)
    m = np.zeros((n_d, cache_len + n_d), dtype=bool)
    for i, (y, x) in enumerate(draft_coords):
        for j, kc in enumerate(keys):
            if kc is None:
                m[i, j] = True
            else:
                yk, xk = kc
                m[i, j] = (yk < y) or (yk == y and xk <= x)
    return m


def flat_mask(draft_coords, cache_len: int, prefix_len: int, row_stride: int) -> np.ndarray:
    """The same mask as the flat-position predicate pos(key) <= pos(query)."""
    qpos = np.array([flat_position(y, x, prefix_len, row_stride) for (y, x) in draft_coords],
                    dtype=np.int64)
    kpos = np.concatenate([np.arange(cache_len, dtype=np.int64), qpos])
    return kpos[None, :] <= qpos[:, None]
