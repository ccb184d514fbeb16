"""Seeded synthetic boundary inputs shaped like the paper's VLM workloads.

This module only draws random tensors and lays them out; it holds none of
the compression method's arithmetic.  Both the CUDA path (through the
binding) and the CPU oracle (through the tests) read the same arrays.

Workloads (the synthetic stand-ins for the paper's models and benchmarks;
no benchmark image, prompt or checkpoint is used):

  tiny     1 image, N=64 (8x8), T=8, H=Hkv=4, d=64, D=256, K=16, fp32,
           every tensor ~ N(0,1).
  llava    LLaVA-1.5-7B shape: N=576 (24x24), T=32, H=Hkv=32, d=128,
           D=4096, K in {64,128,192}, bf16.  8 object regions (Voronoi cells
           of 8 seeded grid points); visual hidden rows and visual keys are a
           region centre ~ N(0,I) plus 0.3 N(0,I).  1-D positions replicated
           on the three position rows.
  qwen     Qwen2.5-VL-7B shape: N=1296 (36x36), T=64, H=28, Hkv=4, d=128,
           D=3584, K=257 (about 20%), bf16, 3-D M-RoPE positions.  As llava,
           plus 2 seeded "detail" tokens per region replaced by
           5 * typical-norm * unit(N(0,I)).
  doc      high-resolution document: qwen dims, N=4096 (64x64), T=128,
           K=410, bf16.  Hidden rows = Bw_i with B ~ N(0,1/32) (D x 32),
           w_i ~ N(0,I_32), and 200 seeded rows replaced by fresh N(0,I_D).
  serving  32 independent qwen-shaped images, T_b ~ U[16,256] (seeded),
           K=257 each, one call.
  multi    one prompt with two qwen-shaped images (N = 2 x 1296, each 36x36,
           one after the other), T=64, K=514 (20%), bf16; every image drawn
           like a qwen image from its own substream (seed, 0, 1000 + image).
  longdoc  the paper's long-prefix document path: qwen dims, N=15876
           (126x126), T=128, K=4096, bf16, drawn like doc (rank-32
           background, isolated rows at doc's density: 775 of them); bounded
           appearance bank with rank 128, at most 4096 clients, b = 512.
  longsmall a small long-prefix case for parity: N=1600 (40x40), T=16, H=4,
           Hkv=2, d=64, D=256, K=320, bf16, drawn like doc (80 isolated
           rows); rank 128, at most 512 clients, b = 64 (pool 256).

Values are drawn in fp32; bf16 workloads round them once to bf16 (round to
nearest even) and every consumer reads the rounded values.  Values V ~ N(0,1).
The probe input W_h = O_h P (d x 4) with O_h ~ N(0,1/D) and P orthonormal
has i.i.d. N(0,1/D) entries, and is drawn that way from seed 0.
Positions: M-RoPE visual (0, r, c), text s+k on all three rows with
s = max(gh, gw); 1-D layouts use (i, i, i) and N+k.
Seeds: numpy default_rng(1000 + workload index), one substream per image.

Historical message views (``history_view``): the text queries, keys, values
and probe of an earlier layer for the same image, drawn from their own
substreams (seed, image, 1 + view) and probe seed (0, 1 + view), so the
boundary tensors above do not change.  Where the image has object regions,
the view's visual keys follow the same regions with fresh region centres.
Dense prefix layers (``prefix_kv``): keys and values of the layers before the
boundary, N(0, 1) from substreams (seed, image, 100 + layer).
Long-prefix Rademacher map (``rademacher``): r x D entries +-1 with equal
probability from numpy default_rng(104729) (the seed of the paper's
configuration table), an input of both the CUDA path and the oracle.
"""

from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

WORKLOADS = {
    # name: (index, B, gh, gw, T, H, Hkv, d, D, K, dtype, structure, positions)
    "tiny": (0, 1, 8, 8, 8, 4, 4, 64, 256, 16, "f32", "plain", "mrope"),
    "llava": (1, 1, 24, 24, 32, 32, 32, 128, 4096, 128, "bf16", "regions", "1d"),
    "qwen": (2, 1, 36, 36, 64, 28, 4, 128, 3584, 257, "bf16", "regions+detail", "mrope"),
    "doc": (3, 1, 64, 64, 128, 28, 4, 128, 3584, 410, "bf16", "lowrank", "mrope"),
    "serving": (4, 32, 36, 36, None, 28, 4, 128, 3584, 257, "bf16", "regions+detail", "mrope"),
    # multi-image prompt: two qwen-shaped images (2 x 36 x 36 visual tokens) before the text
    "multi": (5, 1, 36, 36, 64, 28, 4, 128, 3584, 514, "bf16", "regions+detail", "mrope"),
    # long prefixes: the bounded appearance bank (LONG_PREFIX below)
    "longdoc": (6, 1, 126, 126, 128, 28, 4, 128, 3584, 4096, "bf16", "lowrank", "mrope"),
    "longsmall": (7, 1, 40, 40, 16, 4, 2, 64, 256, 320, "bf16", "lowrank", "mrope"),
}
IMAGES = {"multi": 2}  # images per boundary (1 when absent)
# bounded appearance bank of the long-prefix workloads: projection rank, most
# appearance clients, responsibility batch b (pool 4b)
LONG_PREFIX = {
    "longdoc": dict(rank=128, max_clients=4096, batch_b=512),
    "longsmall": dict(rank=128, max_clients=512, batch_b=64),
}


def rademacher(D: int, rank: int = 128, seed: int = 104729) -> np.ndarray:
    """The fixed rank x D Rademacher map of the long-prefix appearance bank:
    entries -1 or +1 with equal probability, fp32 (exact in bf16)."""
    rng = np.random.default_rng(seed)
    return (rng.integers(0, 2, size=(rank, D)).astype(np.float32) * 2.0 - 1.0).astype(np.float32)


def round_to_bf16(x: np.ndarray) -> np.ndarray:
    """fp32 -> nearest bf16 (ties to even), returned as fp32 values."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32)


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """Upper 16 bits of fp32 values that are already bf16-representable."""
    return (np.ascontiguousarray(x, dtype=np.float32).view(np.uint32) >> 16).astype(np.uint16)


@dataclass
class Image:
    hidden: np.ndarray    # [N+T, D] fp32 (bf16-representable for bf16 workloads)
    keys: np.ndarray      # [N+T, Hkv, d]
    values: np.ndarray    # [N+T, Hkv, d]
    queries: np.ndarray   # [T, H, d]
    pos: np.ndarray       # [3, N+T] int32
    T: int
    region: np.ndarray = None  # [N] object region of every visual token (region workloads)


@dataclass
class Workload:
    name: str
    index: int
    B: int
    gh: int
    gw: int
    T: list
    H: int
    Hkv: int
    d: int
    D: int
    K: int
    dtype: str
    structure: str
    positions: str
    I: int = 1  # images per boundary (a multi-image prompt when > 1)
    _cache: dict = field(default_factory=dict, repr=False)

    @property
    def Ng(self) -> int:
        """Visual tokens of one image (its grid)."""
        return self.gh * self.gw

    @property
    def N(self) -> int:
        return self.gh * self.gw * self.I

    @property
    def T_max(self) -> int:
        return max(self.T)

    @property
    def ragged(self) -> bool:
        return len(set(self.T)) > 1

    @property
    def seed(self) -> int:
        return 1000 + self.index

    def probe(self) -> np.ndarray:
        """W [H, d, 4] fp32, W_h = O_h P drawn directly as i.i.d. N(0, 1/D)."""
        rng = np.random.default_rng(0)
        return (rng.standard_normal((self.H, self.d, 4), dtype=np.float32)
                / np.float32(np.sqrt(self.D))).astype(np.float32)

    def _round(self, x):
        x = np.asarray(x, dtype=np.float32)
        return round_to_bf16(x) if self.dtype == "bf16" else x

    def _visual(self, rng, f32):
        """One image's visual hidden rows, keys, values and regions (multi-image
        prompts), drawn like the single-image rows below."""
        Ng, D, Hkv, d = self.Ng, self.D, self.Hkv, self.d
        hidden = rng.standard_normal((Ng, D), dtype=f32)
        keys = rng.standard_normal((Ng, Hkv, d), dtype=f32)
        values = rng.standard_normal((Ng, Hkv, d), dtype=f32)
        region = None
        if self.structure.startswith("regions"):
            n_reg = 8
            seeds = rng.choice(Ng, size=n_reg, replace=False)
            sr, sc = np.divmod(seeds, self.gw)
            r, c = np.divmod(np.arange(Ng), self.gw)
            dist = (r[:, None] - sr[None, :]) ** 2 + (c[:, None] - sc[None, :]) ** 2
            region = np.argmin(dist, axis=1)
            mu = rng.standard_normal((n_reg, D), dtype=f32)
            kap = rng.standard_normal((n_reg, Hkv, d), dtype=f32)
            hidden = mu[region] + f32(0.3) * rng.standard_normal((Ng, D), dtype=f32)
            keys = kap[region] + f32(0.3) * rng.standard_normal((Ng, Hkv, d), dtype=f32)
            if self.structure == "regions+detail":
                typical = float(np.mean(np.linalg.norm(hidden, axis=1)))
                for k in range(n_reg):
                    members = np.flatnonzero(region == k)
                    pick = rng.choice(members, size=min(2, members.size), replace=False)
                    for i in pick:
                        v = rng.standard_normal(D, dtype=f32)
                        hidden[i] = f32(5.0 * typical) * v / np.linalg.norm(v)
        return hidden, keys, values, region

    def _multi_image(self, b: int) -> Image:
        f32 = np.float32
        rng = np.random.default_rng([self.seed, b])
        T, D, H, Hkv, d = self.T[b], self.D, self.H, self.Hkv, self.d
        parts = [self._visual(np.random.default_rng([self.seed, b, 1000 + k]), f32)
                 for k in range(self.I)]
        hidden = np.concatenate([p[0] for p in parts] + [rng.standard_normal((T, D), dtype=f32)])
        keys = np.concatenate([p[1] for p in parts] + [rng.standard_normal((T, Hkv, d), dtype=f32)])
        values = np.concatenate([p[2] for p in parts] +
                                [rng.standard_normal((T, Hkv, d), dtype=f32)])
        queries = rng.standard_normal((T, H, d), dtype=f32)
        region = None
        if parts[0][3] is not None:  # regions numbered per image, distinct across images
            region = np.concatenate([p[3] + 8 * k for k, p in enumerate(parts)])
        N, Ng, s = self.N, self.Ng, max(self.gh, self.gw)
        pos = np.empty((3, N + T), dtype=np.int32)
        r, c = np.divmod(np.arange(Ng), self.gw)
        for k in range(self.I):  # M-RoPE: image k at temporal index k*s
            pos[0, k * Ng:(k + 1) * Ng] = k * s
            pos[1, k * Ng:(k + 1) * Ng] = k * s + r
            pos[2, k * Ng:(k + 1) * Ng] = k * s + c
        pos[:, N:] = self.I * s + np.arange(T)
        return Image(self._round(hidden), self._round(keys), self._round(values),
                     self._round(queries), pos, T, region)

    def image(self, b: int) -> Image:
        if b in self._cache:
            return self._cache[b]
        if self.I > 1:
            self._cache[b] = self._multi_image(b)
            return self._cache[b]
        rng = np.random.default_rng([self.seed, b])
        N, T, D, H, Hkv, d = self.N, self.T[b], self.D, self.H, self.Hkv, self.d
        f32 = np.float32
        hidden = rng.standard_normal((N + T, D), dtype=f32)
        keys = rng.standard_normal((N + T, Hkv, d), dtype=f32)
        values = rng.standard_normal((N + T, Hkv, d), dtype=f32)
        queries = rng.standard_normal((T, H, d), dtype=f32)
        if self.structure.startswith("regions"):
            n_reg = 8
            seeds = rng.choice(N, size=n_reg, replace=False)
            sr, sc = np.divmod(seeds, self.gw)
            r, c = np.divmod(np.arange(N), self.gw)
            dist = (r[:, None] - sr[None, :]) ** 2 + (c[:, None] - sc[None, :]) ** 2
            region = np.argmin(dist, axis=1)          # ties to the lowest region
            mu = rng.standard_normal((n_reg, D), dtype=f32)
            kap = rng.standard_normal((n_reg, Hkv, d), dtype=f32)
            hidden[:N] = mu[region] + f32(0.3) * rng.standard_normal((N, D), dtype=f32)
            keys[:N] = kap[region] + f32(0.3) * rng.standard_normal((N, Hkv, d), dtype=f32)
            if self.structure == "regions+detail":
                typical = float(np.mean(np.linalg.norm(hidden[:N], axis=1)))
                for k in range(n_reg):
                    members = np.flatnonzero(region == k)
                    pick = rng.choice(members, size=min(2, members.size), replace=False)
                    for i in pick:
                        v = rng.standard_normal(D, dtype=f32)
                        hidden[i] = f32(5.0 * typical) * v / np.linalg.norm(v)
        elif self.structure == "lowrank":
            Bm = rng.standard_normal((D, 32), dtype=f32) / f32(np.sqrt(32.0))
            w = rng.standard_normal((N, 32), dtype=f32)
            hidden[:N] = w @ Bm.T
            # isolated high-innovation rows: 200 per 4096 tokens
            iso = rng.choice(N, size=min(int(round(200 * N / 4096)), N), replace=False)
            hidden[iso] = rng.standard_normal((iso.size, D), dtype=f32)
        pos = np.empty((3, N + T), dtype=np.int32)
        if self.positions == "mrope":
            r, c = np.divmod(np.arange(N), self.gw)
            pos[0, :N] = 0
            pos[1, :N] = r
            pos[2, :N] = c
            s = max(self.gh, self.gw)
            pos[:, N:] = s + np.arange(T)
        else:
            pos[:, :N] = np.arange(N)
            pos[:, N:] = N + np.arange(T)
        img = Image(self._round(hidden), self._round(keys), self._round(values),
                    self._round(queries), pos, T,
                    region if self.structure.startswith("regions") else None)
        self._cache[b] = img
        return img

    def history_view(self, b: int, v: int) -> dict:
        """Historical view v of image b: Q [T, H, d], K and V [N+T, Hkv, d],
        W [H, d, 4] (rounded like the boundary tensors)."""
        im = self.image(b)
        rng = np.random.default_rng([self.seed, b, 1 + v])
        N, T, H, Hkv, d = self.N, self.T[b], self.H, self.Hkv, self.d
        f32 = np.float32
        q = rng.standard_normal((T, H, d), dtype=f32)
        k = rng.standard_normal((N + T, Hkv, d), dtype=f32)
        val = rng.standard_normal((N + T, Hkv, d), dtype=f32)
        if im.region is not None:
            kap = rng.standard_normal((int(im.region.max()) + 1, Hkv, d), dtype=f32)
            k[:N] = kap[im.region] + f32(0.3) * rng.standard_normal((N, Hkv, d), dtype=f32)
        w = (np.random.default_rng([0, 1 + v]).standard_normal((H, d, 4), dtype=f32)
             / f32(np.sqrt(self.D))).astype(f32)
        return dict(Q=self._round(q), K=self._round(k), V=self._round(val), W=w)

    def history_abi_arrays(self, v: int) -> dict:
        """Historical view v of every image in the C-ABI layout of gmc_views:
        keys [B][2][N+T_b][Hkv][d] (K then V), queries [B][T_b][H][d], vo_probe."""
        kv, q = [], []
        for b in range(self.B):
            hv = self.history_view(b, v)
            kv.append(np.stack([hv["K"], hv["V"]]).reshape(-1))
            q.append(hv["Q"].reshape(-1))
        conv = bf16_bits if self.dtype == "bf16" else (lambda a: np.ascontiguousarray(a, np.float32))
        return dict(keys=conv(np.concatenate(kv)), queries=conv(np.concatenate(q)),
                    vo_probe=self.history_view(0, v)["W"])

    def prefix_kv(self, b: int, layer: int) -> dict:
        """Keys and values [N+T, Hkv, d] of dense prefix layer `layer` of image b
        (the cached path keeps them at the kept rows), from their own substream
        (seed, image, 100 + layer); N(0, 1), rounded like the boundary tensors."""
        rng = np.random.default_rng([self.seed, b, 100 + layer])
        shape = (self.N + self.T[b], self.Hkv, self.d)
        return dict(K=self._round(rng.standard_normal(shape, dtype=np.float32)),
                    V=self._round(rng.standard_normal(shape, dtype=np.float32)))

    def prefix_abi_arrays(self, layer: int) -> np.ndarray:
        """Prefix layer `layer` of every image in the C-ABI layout of `keys`:
        [B][2][N+T_b][Hkv][d], K then V."""
        kv = []
        for b in range(self.B):
            pk = self.prefix_kv(b, layer)
            kv.append(np.stack([pk["K"], pk["V"]]).reshape(-1))
        conv = bf16_bits if self.dtype == "bf16" else (lambda a: np.ascontiguousarray(a, np.float32))
        return conv(np.concatenate(kv))

    def text_offsets(self) -> np.ndarray:
        return np.concatenate([[0], np.cumsum(self.T)]).astype(np.int32)

    def abi_arrays(self) -> dict:
        """Host arrays in the C-ABI layout (see include/gmc.h).

        hidden [B][N+T_b][D], keys [B][2][N+T_b][Hkv][d] (K then V),
        queries [B][T_b][H][d], pos_ids [B][3][N+T_b]; bf16 tensors as uint16
        bit patterns, fp32 ones as float32.
        """
        hid, kv, q, pos = [], [], [], []
        for b in range(self.B):
            im = self.image(b)
            hid.append(im.hidden.reshape(-1))
            kv.append(np.stack([im.keys, im.values]).reshape(-1))
            q.append(im.queries.reshape(-1))
            pos.append(im.pos.reshape(-1))
        conv = bf16_bits if self.dtype == "bf16" else (lambda a: np.ascontiguousarray(a, np.float32))
        return dict(hidden=conv(np.concatenate(hid)), keys=conv(np.concatenate(kv)),
                    queries=conv(np.concatenate(q)), pos_ids=np.concatenate(pos).astype(np.int32),
                    vo_probe=self.probe(), text_offsets=self.text_offsets())


def make(name: str, K: int | None = None, B: int | None = None, T: int | list | None = None,
         **shape) -> Workload:
    """Build a named workload; K, B, T and shape fields may be overridden for tests."""
    idx, B0, gh, gw, T0, H, Hkv, d, D, K0, dtype, structure, positions = WORKLOADS[name]
    gh = shape.pop("gh", gh)
    gw = shape.pop("gw", gw)
    H = shape.pop("H", H)
    Hkv = shape.pop("Hkv", Hkv)
    d = shape.pop("d", d)
    D = shape.pop("D", D)
    dtype = shape.pop("dtype", dtype)
    n_img = shape.pop("I", IMAGES.get(name, 1))
    structure = shape.pop("structure", structure)
    if shape:
        raise KeyError(f"unknown workload fields {sorted(shape)}")
    B = B0 if B is None else B
    if T is None:
        if T0 is None:   # serving: ragged T_b ~ U[16, 256]
            T = np.random.default_rng([1000 + idx, 999_999]).integers(16, 257, size=B).tolist()
        else:
            T = [T0] * B
    elif isinstance(T, int):
        T = [T] * B
    return Workload(name, idx, B, gh, gw, list(T), H, Hkv, d, D, K0 if K is None else K,
                    dtype, structure, positions, n_img)
