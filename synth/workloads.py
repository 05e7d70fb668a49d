"""Seeded synthetic workloads for the foreground-only block-sparse attention path.

This module only makes inputs: canvas silhouettes, the canvas Q/K/V/dO tensors
and, for the structured configurations, the block bitmap that a caller hands
to the bitmap mode of the block-mask step.  It holds none of the method's
arithmetic (no compaction, pooling, Top-K, attention or scatter); both the
fp64 oracle and the CUDA path consume what it returns.

Shapes follow the paper's multi-view sequence (Sec. 3.1): 6 noisy target
images, 6 normal-map condition images and 1 reference image, each of
side x side latent tokens after 8x VAE downsampling and 2x2 patchify
(16,384 tokens per image and 212,992 in all at 2048 resolution).  The six
view masks are shared by target view v and condition view v; the reference
image has its own mask (Sec. 3.2, "Mask Construction and Sequence
Compression").  Images are laid out one after another on the canvas, raster
order inside each image.

Random streams (numpy PCG64 seeded with ``[seed, stream]``):
mask=0, Q=1, K=2, V=3, dO=4, block fill=5, oracle row subsample=6, sampler
latent=7, sampler velocity=8, background latent tile=9, alpha renders=10.
Q/K/V/dO are drawn N(0,1) in fp32 and, for bf16 workloads, rounded to
nearest-even bf16 by torch.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import numpy as np
import torch

STREAM_MASK, STREAM_Q, STREAM_K, STREAM_V, STREAM_DO, STREAM_FILL, STREAM_ROWS = range(7)
STREAM_LATENT, STREAM_VEL, STREAM_BG, STREAM_ALPHA = 7, 8, 9, 10
ALPHA_FACTOR = 16  # alpha pixels per token side (8x VAE downsampling, 2x2 patches)

# Sampler-side latent: 16 VAE channels per 8x8 pixels, 2x2-patchified into one
# token, i.e. 64 values per token; one step of a 28-step uniform schedule.
LATENT_CHANNELS = 64
EULER_DT = -1.0 / 28.0

# The multi-view layout: images 0-5 targets, 6-11 conditions, 12 reference.
N_VIEWS = 6


def rng(seed: int, stream: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64([int(seed), int(stream)]))


def round_half_up(x: float) -> int:
    return int(math.floor(x + 0.5))


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    n_images: int          # 13 for the multi-view canvas, 2 for the tiny case
    side: int              # tokens per image side
    fg_frac: float         # foreground fraction per image
    shape: str             # 'disc' | 'ellipse' | 'blob'
    ref_full: bool         # reference image fully kept (512 config)
    heads: int
    head_dim: int
    dtype: str             # 'f32' | 'bf16'
    block: int             # b_q = b_kv
    mask_mode: str         # 'structured' | 'topk'
    density: float         # structured: target density (random fill up to it); topk: rho
    tiny_fill: Optional[float] = None  # tiny case: fixed fill probability of non-own tiles
    seed: int = 0
    text_prefix: int = 0   # text tokens of the joint MM-DiT sequence before the images (always kept)

    # ---------------------------------------------------------------- sizes
    @property
    def multiview(self) -> bool:
        return self.n_images == 2 * N_VIEWS + 1

    @property
    def tokens_per_image(self) -> int:
        return self.side * self.side

    @property
    def T(self) -> int:
        return self.text_prefix + self.n_images * self.tokens_per_image

    def image_counts(self) -> np.ndarray:
        """Foreground tokens per image (exact counts, round half up)."""
        k = round_half_up(self.fg_frac * self.tokens_per_image)
        counts = np.full(self.n_images, k, dtype=np.int64)
        if self.multiview and self.ref_full:
            counts[-1] = self.tokens_per_image
        return counts

    @property
    def N(self) -> int:
        return self.text_prefix + int(self.image_counts().sum())

    @property
    def n_tiles(self) -> int:
        return -(-self.N // self.block)

    @property
    def rho(self) -> float:
        assert self.mask_mode == "topk"
        return float(self.density)

    def with_(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)

    # ---------------------------------------------------------- silhouettes
    def _field(self, g: np.random.Generator) -> np.ndarray:
        s = self.side
        yy, xx = np.meshgrid(np.arange(s, dtype=np.float64) + 0.5,
                             np.arange(s, dtype=np.float64) + 0.5, indexing="ij")
        if self.shape == "disc":
            cy, cx = g.uniform(0.3, 0.7, size=2) * s
            return -((yy - cy) ** 2 + (xx - cx) ** 2)
        if self.shape == "ellipse":
            cy, cx = g.uniform(0.35, 0.65, size=2) * s
            th = g.uniform(0.0, math.pi)
            ratio = g.uniform(0.5, 1.0)
            u = (xx - cx) * math.cos(th) + (yy - cy) * math.sin(th)
            v = -(xx - cx) * math.sin(th) + (yy - cy) * math.cos(th)
            return -((u / 1.0) ** 2 + (v / ratio) ** 2)
        if self.shape == "blob":
            n_g = int(g.integers(3, 7))
            f = np.zeros_like(yy)
            for _ in range(n_g):
                cy, cx = g.uniform(0.2, 0.8, size=2) * s
                sig = g.uniform(0.08, 0.25) * s
                w = g.uniform(0.5, 1.0)
                f += w * np.exp(-((yy - cy) ** 2 + (xx - cx) ** 2) / (2.0 * sig * sig))
            return f
        raise ValueError(self.shape)

    def _silhouette(self, g: np.random.Generator, k: int) -> np.ndarray:
        """Keep the k tokens with the highest field value; ties -> lower raster index."""
        field = self._field(g).ravel()
        order = np.lexsort((np.arange(field.size), -field))
        m = np.zeros(field.size, dtype=np.uint8)
        m[order[:k]] = 1
        return m

    def image_masks(self) -> np.ndarray:
        """[n_images, side*side] uint8 masks: view masks shared by target/condition."""
        g = rng(self.seed, STREAM_MASK)
        counts = self.image_counts()
        masks = np.zeros((self.n_images, self.tokens_per_image), dtype=np.uint8)
        if not self.multiview:
            for v in range(self.n_images):
                masks[v] = self._silhouette(g, int(counts[v]))
            return masks
        for v in range(N_VIEWS):
            m = self._silhouette(g, int(counts[v]))
            masks[v] = m                 # target view v
            masks[N_VIEWS + v] = m       # condition view v shares it
        if self.ref_full:
            masks[-1] = 1
        else:
            masks[-1] = self._silhouette(g, int(counts[-1]))
        return masks

    def canvas_mask(self) -> np.ndarray:
        """[T] uint8: the text prefix (always kept), then the images one after another."""
        m = self.image_masks().reshape(-1)
        if self.text_prefix:
            m = np.concatenate([np.ones(self.text_prefix, np.uint8), m])
        return np.ascontiguousarray(m)

    # --------------------------------------------------------------- tensors
    def _draw(self, stream: int, rows: Optional[int] = None) -> torch.Tensor:
        """[T, H, d] N(0,1) drawn row-chunk by row-chunk, rounded to the workload dtype."""
        T = self.T if rows is None else rows
        H, d = self.heads, self.head_dim
        g = rng(self.seed, stream)
        tdtype = torch.bfloat16 if self.dtype == "bf16" else torch.float32
        out = torch.empty((T, H, d), dtype=tdtype)
        chunk = max(1, (1 << 24) // (H * d))
        for r0 in range(0, T, chunk):
            r1 = min(T, r0 + chunk)
            x = g.standard_normal(size=(r1 - r0, H, d), dtype=np.float32)
            out[r0:r1] = torch.from_numpy(x).to(tdtype)
        return out

    def q(self) -> torch.Tensor:
        return self._draw(STREAM_Q)

    def k(self) -> torch.Tensor:
        return self._draw(STREAM_K)

    def v(self) -> torch.Tensor:
        return self._draw(STREAM_V)

    def dout(self) -> torch.Tensor:
        return self._draw(STREAM_DO)

    # -------------------------------------------------------- alpha renders
    def alpha_images(self, factor: int = ALPHA_FACTOR) -> np.ndarray:
        """[V + 1, side*factor, side*factor] uint8 alpha channels of the view
        renders and the reference: a blob silhouette per image (sum of 3-6
        Gaussians, thresholded so that ~0.45 fg_frac of the pixels are opaque; the pooling and dilation bring the token mask near fg_frac),
        a two-pixel anti-aliased edge ramp, and sparse faint specks (alpha
        1-20) in the background the way renders leave them."""
        n_img = (N_VIEWS + 1) if self.multiview else self.n_images
        P = self.side * factor
        g = rng(self.seed, STREAM_ALPHA)
        yy, xx = np.meshgrid((np.arange(P, dtype=np.float64) + 0.5) / factor,
                             (np.arange(P, dtype=np.float64) + 0.5) / factor, indexing="ij")
        out = np.zeros((n_img, P, P), dtype=np.uint8)
        for i in range(n_img):
            f = np.zeros_like(yy)
            for _ in range(int(g.integers(3, 7))):
                cy, cx = g.uniform(0.2, 0.8, size=2) * self.side
                sig = g.uniform(0.08, 0.25) * self.side
                f += g.uniform(0.5, 1.0) * np.exp(-((yy - cy) ** 2 + (xx - cx) ** 2) / (2.0 * sig * sig))
            level = np.quantile(f, 1.0 - 0.45 * self.fg_frac)
            band = 2.0 * float(np.abs(np.gradient(f)[0]).mean()) + 1e-12
            a = np.clip((f - level) / band, 0.0, 1.0)
            img = np.rint(a * 255.0).astype(np.uint8)
            specks = g.random((P, P)) < 2e-4
            img[specks & (img == 0)] = g.integers(1, 21, size=int((specks & (img == 0)).sum()), dtype=np.uint8)
            out[i] = img
        return out

    # ----------------------------------------------------- sampler inputs
    def sampler_inputs(self, channels: int = LATENT_CHANNELS, dtype: torch.dtype = torch.bfloat16) -> dict:
        """Inputs of the sampler steps on the target canvas (the noisy target
        images only: the first six images of the multi-view canvas, or the whole
        canvas otherwise): its foreground mask, the canvas latent z (Gaussian
        noise), the predicted velocities of its retained tokens, one image's
        canonical background latent tile, and the step dt = t_prev - t_curr."""
        n_img = N_VIEWS if self.multiview else self.n_images
        T = n_img * self.tokens_per_image
        mask = self.canvas_mask()[self.text_prefix:self.text_prefix + T].copy()
        n = int(mask.sum())
        z = rng(self.seed, STREAM_LATENT).standard_normal((T, channels), dtype=np.float32)
        v = rng(self.seed, STREAM_VEL).standard_normal((n, channels), dtype=np.float32)
        gb = rng(self.seed, STREAM_BG)
        tile = (gb.standard_normal((1, channels), dtype=np.float32) +
                np.float32(0.1) * gb.standard_normal((self.tokens_per_image, channels), dtype=np.float32))
        conv = lambda a: torch.from_numpy(a).to(dtype)
        return {"mask": mask, "z": conv(z), "v": conv(v), "tile": conv(tile), "dt": EULER_DT,
                "period": self.tokens_per_image}

    # ------------------------------------------------- structured block bitmap
    def tile_images(self) -> list[tuple[int, int]]:
        """(first, last) image of each compacted tile, from the per-image counts.

        Compacted rows keep canvas order, so image boundaries in compacted
        order are the running sums of the per-image foreground counts.
        """
        assert self.text_prefix == 0, "the structured rule is defined for image tokens only"
        bounds = np.concatenate([[0], np.cumsum(self.image_counts())])
        out = []
        for i in range(self.n_tiles):
            r0 = i * self.block
            r1 = min(self.N, r0 + self.block) - 1
            a = int(np.searchsorted(bounds, r0, side="right") - 1)
            b = int(np.searchsorted(bounds, r1, side="right") - 1)
            out.append((a, b))
        return out

    def structural_bitmap(self) -> np.ndarray:
        """[n_tiles, n_tiles] uint8 structural pattern shared by all heads.

        Multi-view canvas: query tile i keeps key tile j when their image sets
        intersect (own view), when j holds the same-index view of the other
        modality (target v <-> condition v), or when j holds reference tokens.
        Two-view tiny case: own-view tiles only.
        """
        ti = self.tile_images()
        n = len(ti)
        sets = [set(range(a, b + 1)) for a, b in ti]
        ref = self.n_images - 1

        def partner(img: int) -> Optional[int]:
            if not self.multiview or img == ref:
                return None
            return img + N_VIEWS if img < N_VIEWS else img - N_VIEWS

        bm = np.zeros((n, n), dtype=np.uint8)
        for i in range(n):
            own = sets[i]
            part = {partner(x) for x in own} - {None}
            for j in range(n):
                kj = sets[j]
                if own & kj or part & kj or (self.multiview and ref in kj):
                    bm[i, j] = 1
        return bm

    def block_bitmap(self) -> np.ndarray:
        """[H, n_tiles, n_tiles] uint8 block bitmap for the structured configs."""
        assert self.mask_mode == "structured"
        base = self.structural_bitmap()
        n = base.shape[0]
        g = rng(self.seed, STREAM_FILL)
        if self.tiny_fill is not None:
            p = float(self.tiny_fill)
        else:
            s = float(base.mean())
            p = max(0.0, (self.density - s) / (1.0 - s)) if s < 1.0 else 0.0
        fill = g.random(size=(self.heads, n, n)) < p
        return np.ascontiguousarray(np.where(base[None] == 1, 1, fill.astype(np.uint8)).astype(np.uint8))

    def row_subsample(self, n_rows: int, frac: float) -> np.ndarray:
        """Seeded sorted subsample of compacted row indices (oracle spot checks)."""
        g = rng(self.seed, STREAM_ROWS)
        k = max(1, int(round(frac * n_rows)))
        return np.sort(g.choice(n_rows, size=k, replace=False)).astype(np.int64)


CONFIGS: dict[str, Workload] = {
    # 2 views of 16x16, ~50% discs, 1 head, d=64, fp32, b=32; own-view tiles + 25% fill.
    "tiny": Workload("tiny", n_images=2, side=16, fg_frac=0.5, shape="disc", ref_full=False,
                     heads=1, head_dim=64, dtype="f32", block=32, mask_mode="structured",
                     density=0.0, tiny_fill=0.25),
    # 13 x 32x32, 55% ellipses, reference fully kept, 24 heads, d=128, bf16, b=128, ~30%.
    "c512": Workload("c512", n_images=13, side=32, fg_frac=0.55, shape="ellipse", ref_full=True,
                     heads=24, head_dim=128, dtype="bf16", block=128, mask_mode="structured",
                     density=0.30),
    # 13 x 64x64, 45% blobs, structural rule only (~20%+), forward and backward.
    "c1024": Workload("c1024", n_images=13, side=64, fg_frac=0.45, shape="blob", ref_full=False,
                      heads=24, head_dim=128, dtype="bf16", block=128, mask_mode="structured",
                      density=0.20),
    # 13 x 128x128, 40% blobs (85,202 tokens), Top-K rule with rho = 0.12.
    "c2048": Workload("c2048", n_images=13, side=128, fg_frac=0.40, shape="blob", ref_full=False,
                      heads=24, head_dim=128, dtype="bf16", block=128, mask_mode="topk",
                      density=0.12),
    # the 2048 canvas with the joint sequence's 512 text tokens in front (the
    # token lengths of Table S1 include them): T = 213,504, N = 85,714
    "c2048t": Workload("c2048t", n_images=13, side=128, fg_frac=0.40, shape="blob", ref_full=False,
                       heads=24, head_dim=128, dtype="bf16", block=128, mask_mode="topk",
                       density=0.12, text_prefix=512),
}

SWEEP_FG = (0.20, 0.40, 0.60, 0.80)
SWEEP_RHO = (0.05, 0.10, 0.25, 0.50, 1.00)
SWEEP_BLOCK = (64, 128)


def sweep2048(fg: float, rho: float, block: int = 128) -> Workload:
    return CONFIGS["c2048"].with_(name=f"sweep2048_fg{int(fg*100)}_rho{int(rho*100)}_b{block}",
                                  fg_frac=fg, density=rho, block=block)
