"""Frame and weight generators (seeded numpy; inputs only).

Frames are NHWC float32 arrays.  For bfloat16 workloads the generator rounds
them to bfloat16 storage (round to nearest even) and hands out the 16-bit
patterns; ``bf16_bits_to_f32`` gives back the exact values.
"""
from __future__ import annotations

import numpy as np


# ---------------------------------------------------------------- bf16 storage
def bf16_bits(a: np.ndarray) -> np.ndarray:
    """float32 -> bfloat16 bit patterns (uint16), round to nearest, ties to even."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    u = a.view(np.uint32).astype(np.uint64)
    bias = np.uint64(0x7FFF) + ((u >> np.uint64(16)) & np.uint64(1))
    out = ((u + bias) >> np.uint64(16)).astype(np.uint16)
    nan = np.isnan(a)
    if nan.any():
        out[nan] = 0x7FC0
    return out


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """bfloat16 bit patterns (uint16) -> exact float32 values."""
    b = np.ascontiguousarray(b, dtype=np.uint16)
    return (b.astype(np.uint32) << np.uint32(16)).view(np.float32)


def round_to_bf16(a: np.ndarray) -> np.ndarray:
    """float32 values rounded to the nearest bfloat16 value, kept as float32."""
    return bf16_bits_to_f32(bf16_bits(a))


# ------------------------------------------------------------------- weights
def he_weights(rng: np.random.Generator, c_out: int, c_in_per_group: int, k: int,
               bf16: bool) -> np.ndarray:
    """Kernel w in the paper's c_o x c_i x k_h x k_w order, N(0, var 2/(k^2 c_i))."""
    std = np.sqrt(2.0 / (k * k * c_in_per_group))
    w = (rng.standard_normal((c_out, c_in_per_group, k, k)) * std).astype(np.float32)
    return round_to_bf16(w) if bf16 else w


# ------------------------------------------------------------------ motion
def _reflect(pos: int, vel: int, size: int, extent: int):
    pos += vel
    hi = extent - size
    if pos < 0:
        pos, vel = -pos, -vel
    elif pos > hi:
        pos, vel = 2 * hi - pos, -vel
    return min(max(pos, 0), hi), vel


def moving_squares_video(seed: int, T: int, h: int, w: int, c: int, n_squares: int, size: int,
                         speed: int = 2, noise_std: float = 0.01) -> np.ndarray:
    """Static U[0,1) background, textured size x size squares moving `speed`
    px/frame in a seeded direction from {-s,0,s}^2 minus the origin
    (reflecting at the borders), and fresh N(0, noise_std) noise per frame.
    Returns float32 [T, h, w, c]."""
    rng = np.random.default_rng(seed)
    bg = rng.random((h, w, c), dtype=np.float32)
    dirs = [(dy, dx) for dy in (-speed, 0, speed) for dx in (-speed, 0, speed) if (dy, dx) != (0, 0)]
    squares = []
    for _ in range(n_squares):
        tex = rng.random((size, size, c), dtype=np.float32)
        y, x = int(rng.integers(0, h - size + 1)), int(rng.integers(0, w - size + 1))
        vy, vx = dirs[int(rng.integers(len(dirs)))]
        squares.append([tex, y, x, vy, vx])
    out = np.empty((T, h, w, c), np.float32)
    for t in range(T):
        f = bg.copy()
        for sq in squares:
            tex, y, x = sq[0], sq[1], sq[2]
            f[y:y + size, x:x + size, :] = tex
        if noise_std > 0:
            f += (rng.standard_normal(f.shape) * noise_std).astype(np.float32)
        out[t] = f
        for sq in squares:
            sq[1], sq[3] = _reflect(sq[1], sq[3], size, h)
            sq[2], sq[4] = _reflect(sq[2], sq[4], size, w)
    return out


def panning_video(seed: int, T: int, n: int, h: int, w: int, c: int, dy: int, dx: int) -> np.ndarray:
    """A camera pan: frame t of stream s is the h x w window of a seeded
    U[0,1) texture whose top-left corner is at (t * dy, t * dx) (plus a
    margin so the window stays inside), i.e. frame t at pixel p equals frame
    t-1 at p + (dy, dx).  [T, n, h, w, c] float32."""
    rng = np.random.default_rng(seed)
    H, Wd = h + T * abs(dy) + 1, w + T * abs(dx) + 1
    oy, ox = (T * abs(dy) if dy < 0 else 0), (T * abs(dx) if dx < 0 else 0)
    out = np.empty((T, n, h, w, c), np.float32)
    for s in range(n):
        tex = rng.random((H, Wd, c), dtype=np.float32)
        for t in range(T):
            y0, x0 = oy + t * dy, ox + t * dx
            out[t, s] = tex[y0:y0 + h, x0:x0 + w]
    return out


def moving_rect_video(seed: int, T: int, h: int, w: int, c: int, n_rects: int, rh: int, rw: int,
                      speed: int = 2, jitter: int = 1) -> np.ndarray:
    """Static background plus textured rh x rw rectangles moving `speed`
    px/frame with a per-frame random jitter in {-jitter..jitter}^2.
    Returns float32 [T, h, w, c]."""
    rng = np.random.default_rng(seed)
    bg = rng.random((h, w, c), dtype=np.float32)
    rects = []
    for _ in range(n_rects):
        tex = rng.random((rh, rw, c), dtype=np.float32)
        y, x = int(rng.integers(0, h - rh + 1)), int(rng.integers(0, w - rw + 1))
        ang = rng.integers(0, 8)
        vy = int(round(speed * np.sin(ang * np.pi / 4)))
        vx = int(round(speed * np.cos(ang * np.pi / 4)))
        rects.append([tex, y, x, vy, vx])
    out = np.empty((T, h, w, c), np.float32)
    for t in range(T):
        f = bg.copy()
        for rc in rects:
            f[rc[1]:rc[1] + rh, rc[2]:rc[2] + rw, :] = rc[0]
        out[t] = f
        for rc in rects:
            jy, jx = (int(v) for v in rng.integers(-jitter, jitter + 1, size=2))
            rc[1], rc[3] = _reflect(rc[1], rc[3], rh, h)
            rc[2], rc[4] = _reflect(rc[2], rc[4], rw, w)
            rc[1] = min(max(rc[1] + jy, 0), h - rh)
            rc[2] = min(max(rc[2] + jx, 0), w - rw)
    return out


def traffic_video(seed: int, T: int, h: int = 512, w: int = 512, c: int = 3, n_rects: int = 8,
                  min_side: int = 8, max_side: int = 64, min_speed: int = 1,
                  max_speed: int = 4) -> np.ndarray:
    """Traffic-like video: U[0,1) background and n_rects flat-coloured
    rectangles (sides U[min_side, max_side], speeds min..max px/frame along a
    seeded axis direction), no noise.  Returns float32 [T, h, w, c]."""
    rng = np.random.default_rng(seed)
    bg = rng.random((h, w, c), dtype=np.float32)
    cars = []
    for _ in range(n_rects):
        rh, rw = (int(v) for v in rng.integers(min_side, max_side + 1, size=2))
        colour = rng.random(c, dtype=np.float32)
        y, x = int(rng.integers(0, h - rh + 1)), int(rng.integers(0, w - rw + 1))
        sp = int(rng.integers(min_speed, max_speed + 1))
        if rng.random() < 0.5:
            vy, vx = 0, sp if rng.random() < 0.5 else -sp
        else:
            vy, vx = sp if rng.random() < 0.5 else -sp, 0
        cars.append([rh, rw, colour, y, x, vy, vx])
    out = np.empty((T, h, w, c), np.float32)
    for t in range(T):
        f = bg.copy()
        for car in cars:
            rh, rw, colour, y, x = car[:5]
            f[y:y + rh, x:x + rw, :] = colour
        out[t] = f
        for car in cars:
            car[3], car[5] = _reflect(car[3], car[5], car[0], h)
            car[4], car[6] = _reflect(car[4], car[6], car[1], w)
    return out


class block_perturbation_video:
    """Density-controlled video: U[0,1) background (no noise); at every frame
    after the first, exactly `n_changed` of the b x b blocks of each stream,
    chosen without replacement, get U[0,1) added to their interior
    (b-2) x (b-2) pixels on every channel, and the sum is stored at the frame's
    precision.  Frame 0 is the background.  Iterate to get frames in order.

    Yields (t, frame) with frame float32 [n, h, w, c] (bfloat16-exact values
    when bf16=True)."""

    def __init__(self, seed: int, T: int, n: int, h: int, w: int, c: int, block: int,
                 n_changed: int, bf16: bool = True, margin: int = 1, stream_offset: int = 0):
        self.seed, self.T, self.n, self.h, self.w, self.c = seed, T, n, h, w, c
        self.stream_offset = stream_offset
        self.block, self.n_changed, self.bf16, self.margin = block, n_changed, bf16, margin
        self.nby, self.nbx = h // block, w // block
        assert 0 <= n_changed <= self.nby * self.nbx

    def __iter__(self):
        rng = [np.random.default_rng(self.seed * 100 + self.stream_offset + s) for s in range(self.n)]
        frame = np.empty((self.n, self.h, self.w, self.c), np.float32)
        for s in range(self.n):
            frame[s] = rng[s].random((self.h, self.w, self.c), dtype=np.float32)
        if self.bf16:
            frame = round_to_bf16(frame)
        b, m = self.block, self.margin
        for t in range(self.T):
            if t > 0:
                for s in range(self.n):
                    chosen = rng[s].choice(self.nby * self.nbx, size=self.n_changed, replace=False)
                    for blk in np.sort(chosen):
                        by, bx = divmod(int(blk), self.nbx)
                        y0, x0 = by * b + m, bx * b + m
                        sl = (s, slice(y0, y0 + b - 2 * m), slice(x0, x0 + b - 2 * m), slice(None))
                        d = rng[s].random((b - 2 * m, b - 2 * m, self.c), dtype=np.float32)
                        v = frame[sl] + d
                        frame[sl] = round_to_bf16(v) if self.bf16 else v
            yield t, frame

    def frames(self) -> np.ndarray:
        out = np.empty((self.T, self.n, self.h, self.w, self.c), np.float32)
        for t, f in self:
            out[t] = f
        return out
