"""Seeded synthetic workloads for the BMLP training path (inputs only).

This module generates inputs and labels.  It holds none of the training rule's
arithmetic and is the only code that both the CPU oracle and the GPU library
see.  The paper trains on FashionMNIST, CIFAR-10 / Imagenette AlexNet features
and a Random Prototypes set (Sec. 4.1).  None of those are available here, so
these seeded generators stand in for their shapes:

  C1  784 -> 256 -> 10             2,000 / 500 samples, 1 epoch
  C2  784 -> 1024 x3 -> 10         60,000 / 10,000, 5 epochs
  C3  3072 -> 2048 x3 -> 10        50,000 / 10,000, 3 epochs
  C4  3072 -> 4096 x4 -> 100       50,000 / 10,000, 2 epochs
  C5  8192 -> 8192 x4 -> 10        1,000,000 streamed samples, 1 pass;
                                   plus a 65,536-sample forward-only sweep

Random Prototypes (Sec. 4.1.1, ``random_prototypes``): K_0 = 1000 bits,
10 classes, each sample a class prototype with every entry flipped with
probability 0.44, all samples distinct; 10,000 training and 2,000 test samples.

Input distributions:
  "bias"  : bit j of a sample is +1 with probability p_j, p_j ~ U[0.3, 0.7]
            drawn once per feature (C1, C2, the 784-pixel FashionMNIST shape);
  "field" : a 32 x 32 x 3 image per sample; each channel is i.i.d. N(0, 1)
            smoothed by a Gaussian of length scale 3 pixels with periodic
            boundaries (FFT), thresholded at 0; flattened channel-major (C3,
            C4, the CIFAR-10 image shape);
  "iid"   : i.i.d. +-1 bits with p = 1/2 (C5).
Labels come from a fixed random +-1 teacher MLP (one hidden layer of sign
units, sign(0) = +1, argmax with ties to the lowest class).  The teacher's
sums are integers of magnitude <= 8192, which float32 and bf16-input / fp32-
accumulate matmuls represent exactly, so the labels do not depend on which
backend computes them.

Packed layout (the GPU library's input format): a sample of K bits is
ceil(K / 64) little-endian uint64 words; bit j of word w is feature 64 w + j;
a set bit means +1; pad bits are 0.
Seeds: data seed = 1000 + config number; model seed = config number.
"""
from __future__ import annotations

import dataclasses

import numpy as np


@dataclasses.dataclass(frozen=True)
class Config:
    key: str
    widths: tuple      # K_0 .. K_L
    classes: int
    n_train: int
    n_test: int
    epochs: int
    gen: str
    teacher_hidden: int
    number: int

    @property
    def data_seed(self) -> int:
        return 1000 + self.number

    @property
    def model_seed(self) -> int:
        return self.number

    @property
    def name(self) -> str:
        return "bmlp-" + "-".join(str(w) for w in self.widths) + "-%d" % self.classes


CONFIGS = {
    "C1": Config("C1", (784, 256), 10, 2000, 500, 1, "bias", 128, 1),
    "C2": Config("C2", (784, 1024, 1024, 1024), 10, 60000, 10000, 5, "bias", 512, 2),
    "C3": Config("C3", (3072, 2048, 2048, 2048), 10, 50000, 10000, 3, "field", 1024, 3),
    "C4": Config("C4", (3072, 4096, 4096, 4096, 4096), 100, 50000, 10000, 2, "field", 2048, 4),
    "C5": Config("C5", (8192, 8192, 8192, 8192, 8192), 10, 1000000, 65536, 1, "iid", 1024, 5),
}


def words(K: int) -> int:
    return (K + 63) // 64


# -- format conversion ---------------------------------------------------------

def pack(x_pm1: np.ndarray) -> np.ndarray:
    """n x K array of +-1 -> n x ceil(K/64) uint64 (set bit = +1, pad bits 0)."""
    x = np.asarray(x_pm1)
    n, K = x.shape
    nw = words(K)
    bits = np.zeros((n, nw * 64), np.uint8)
    bits[:, :K] = x > 0
    by = np.packbits(bits, axis=1, bitorder="little")
    return np.ascontiguousarray(by).view("<u8").reshape(n, nw)


def unpack(xp: np.ndarray, K: int) -> np.ndarray:
    """n x nw uint64 -> n x K int8 of +-1."""
    xp = np.ascontiguousarray(xp, dtype="<u8")
    n = xp.shape[0]
    bits = np.unpackbits(xp.view(np.uint8).reshape(n, -1), axis=1, bitorder="little")[:, :K]
    return (bits.astype(np.int8) * 2 - 1).astype(np.int8)


# -- input distributions ---------------------------------------------------------

def _bias_inputs(rng, p, n):
    return np.where(rng.random((n, p.shape[0])) < p[None, :], 1, -1).astype(np.int8)


def _field_inputs(rng, n, side=32, channels=3, scale=3.0, chunk=4096):
    f = np.fft.fftfreq(side)
    transfer = np.exp(-2.0 * (np.pi ** 2) * (scale ** 2) * (f[:, None] ** 2 + f[None, :] ** 2))
    out = np.empty((n, channels * side * side), np.int8)
    for s in range(0, n, chunk):
        b = min(chunk, n - s)
        g = rng.standard_normal((b, channels, side, side))
        sm = np.fft.ifft2(np.fft.fft2(g) * transfer).real
        out[s:s + b] = np.where(sm.reshape(b, -1) > 0, 1, -1)
    return out


def _iid_packed(rng, n, K):
    nw = words(K)
    xp = np.frombuffer(rng.bytes(n * nw * 8), dtype="<u8").reshape(n, nw).copy()
    if K % 64:
        xp[:, -1] &= np.uint64((1 << (K % 64)) - 1)
    return xp


def random_packed(seed: int, n: int, K: int) -> np.ndarray:
    """n packed rows of K i.i.d. fair +-1 values (pad bits 0), seeded."""
    return _iid_packed(np.random.default_rng(seed), n, K)


def real_patterns(seed: int, n: int, K: int, kind: str = "pixels") -> np.ndarray:
    """n x K fp32 real-valued patterns for the median-binarisation front end:
    "pixels" = integer intensities 0..255 with about 60 % zeros (an image-like
    mix with many ties), "gauss" = N(0, 1), "ties" = a pool of seven values
    including -0.0 and +0.0."""
    rng = np.random.default_rng(seed)
    if kind == "pixels":
        v = rng.integers(1, 256, (n, K)).astype(np.float32)
        return np.where(rng.random((n, K)) < 0.6, np.float32(0), v).astype(np.float32)
    if kind == "gauss":
        return rng.standard_normal((n, K)).astype(np.float32)
    if kind == "ties":
        pool = np.array([-2.0, -1.0, -0.0, 0.0, 0.5, 1.0, 3.0], np.float32)
        return pool[rng.integers(0, len(pool), (n, K))]
    raise ValueError(kind)


def pixel_bytes(seed: int, n: int, D: int, kind: str = "pixels") -> np.ndarray:
    """n x D uint8 patterns for the expansion front end: "pixels" = intensities
    1..255 with about 60 % zeros (image-like), "full" = uniform 0..255,
    "sparse" = 0/1 with 5 % ones (many exact ties z = 0 of the expansion
    sums), "saturated" = every input 255 (z = 255 times the weight row's
    sum: a tie wherever a row of an even width sums to 0)."""
    rng = np.random.default_rng(seed)
    if kind == "pixels":
        v = rng.integers(1, 256, (n, D))
        return np.where(rng.random((n, D)) < 0.6, 0, v).astype(np.uint8)
    if kind == "full":
        return rng.integers(0, 256, (n, D)).astype(np.uint8)
    if kind == "sparse":
        return (rng.random((n, D)) < 0.05).astype(np.uint8)
    if kind == "saturated":
        return np.full((n, D), 255, np.uint8)
    raise ValueError(kind)


# -- teacher -------------------------------------------------------------------

@dataclasses.dataclass
class Teacher:
    W1: np.ndarray   # K_0 x hidden, +-1
    W2: np.ndarray   # hidden x classes, +-1


def make_teacher(cfg: Config) -> Teacher:
    rng = np.random.Generator(np.random.PCG64(np.random.SeedSequence([cfg.data_seed, 1])))
    K0 = cfg.widths[0]
    W1 = np.where(rng.random((K0, cfg.teacher_hidden)) < 0.5, 1, -1).astype(np.int8)
    W2 = np.where(rng.random((cfg.teacher_hidden, cfg.classes)) < 0.5, 1, -1).astype(np.int8)
    return Teacher(W1, W2)


def teacher_labels_pm1(teacher: Teacher, x_pm1: np.ndarray, chunk: int = 8192) -> np.ndarray:
    """Labels of n x K_0 +-1 inputs (float32 matmuls, exact for these sums)."""
    W1 = teacher.W1.astype(np.float32)
    W2 = teacher.W2.astype(np.float32)
    n = x_pm1.shape[0]
    out = np.empty(n, np.int32)
    for s in range(0, n, chunk):
        xs = x_pm1[s:s + chunk].astype(np.float32)
        hid = np.where(xs @ W1 >= 0, 1.0, -1.0).astype(np.float32)
        out[s:s + chunk] = np.argmax(hid @ W2, axis=1)
    return out


def teacher_labels_packed_torch(teacher: Teacher, xp, K0: int, chunk: int = 32768):
    """Labels of packed inputs held in a torch tensor (any device), computed with
    bf16 +-1 operands and fp32 accumulation (exact for |sum| <= 8192)."""
    import torch
    dev = xp.device
    W1 = torch.from_numpy(teacher.W1.astype(np.float32)).to(dev, torch.bfloat16)
    W2 = torch.from_numpy(teacher.W2.astype(np.float32)).to(dev, torch.bfloat16)
    n, nw = xp.shape
    shifts = torch.arange(64, device=dev, dtype=torch.int64)
    out = torch.empty(n, dtype=torch.int32, device=dev)
    for s in range(0, n, chunk):
        w = xp[s:s + chunk].view(torch.int64)
        bits = (w.unsqueeze(-1) >> shifts) & 1                       # b x nw x 64
        pm = (bits.reshape(w.shape[0], nw * 64)[:, :K0] * 2 - 1).to(torch.bfloat16)
        h = torch.where((pm @ W1).float() >= 0, 1.0, -1.0).to(torch.bfloat16)
        out[s:s + chunk] = torch.argmax((h @ W2).float(), dim=1).to(torch.int32)
    return out


# -- datasets ------------------------------------------------------------------

@dataclasses.dataclass
class Split:
    xp: np.ndarray        # n x nw uint64 packed
    y: np.ndarray         # n int32
    K0: int

    def pm1(self, start: int = 0, stop: int | None = None) -> np.ndarray:
        return unpack(self.xp[start:stop], self.K0)


def _rng(cfg, tag):
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([cfg.data_seed, tag])))


def make_inputs(cfg: Config, split: str, n: int | None = None) -> np.ndarray:
    """Packed inputs of the train (tag 2) or test (tag 3) split, first n samples
    of the split's seeded stream (n defaults to the split's size)."""
    tag = 2 if split == "train" else 3
    total = cfg.n_train if split == "train" else cfg.n_test
    n = total if n is None else n
    rng = _rng(cfg, tag)
    K0 = cfg.widths[0]
    if cfg.gen == "bias":
        p = 0.3 + 0.4 * _rng(cfg, 4).random(K0)
        return pack(_bias_inputs(rng, p, n))
    if cfg.gen == "field":
        assert K0 == 3 * 32 * 32
        return pack(_field_inputs(rng, n))
    if cfg.gen == "iid":
        return _iid_packed(rng, n, K0)
    raise ValueError(cfg.gen)


def make_split(cfg: Config, split: str, n: int | None = None) -> Split:
    """Inputs and teacher labels (numpy; fine up to ~10^5 samples)."""
    xp = make_inputs(cfg, split, n)
    t = make_teacher(cfg)
    y = teacher_labels_pm1(t, unpack(xp, cfg.widths[0]))
    return Split(xp, y, cfg.widths[0])


def random_prototypes(seed: int, n_train: int = 10000, n_test: int = 2000, K0: int = 1000,
                      classes: int = 10, p: float = 0.44):
    """The Random Prototypes set of Sec. 4.1.1: one uniformly random +-1
    prototype per class; a sample of class j is prototype j with each entry
    flipped independently with probability p; a sample equal to an earlier one
    (train or test) is discarded and redrawn, so all n_train + n_test samples
    are distinct.  Sample i (train first, then test) has class i mod classes,
    so every mini-batch in dataset order mixes the classes.  Returns
    (train Split, test Split) with labels = the classes."""
    rng = np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, 77])))
    proto = np.where(rng.random((classes, K0)) < 0.5, 1, -1).astype(np.int8)
    n = n_train + n_test
    x = np.empty((n, K0), np.int8)
    y = (np.arange(n) % classes).astype(np.int32)
    seen = set()
    for i in range(n):
        while True:
            flip = rng.random(K0) < p
            v = np.where(flip, -proto[y[i]], proto[y[i]]).astype(np.int8)
            key = v.tobytes()
            if key not in seen:
                seen.add(key)
                x[i] = v
                break
    xp = pack(x)
    return Split(xp[:n_train], y[:n_train], K0), Split(xp[n_train:], y[n_train:], K0)


def small_config(widths, classes, n_train, n_test=0, gen="bias", teacher_hidden=32, number=99):
    """A config outside the table, for tests (same generators)."""
    return Config("custom", tuple(widths), classes, n_train, n_test, 1, gen, teacher_hidden, number)
