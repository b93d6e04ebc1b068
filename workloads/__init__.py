"""Seeded synthetic workloads for the DP Compress tabulate-fusion path.

This module makes INPUTS only: random embedding-net parameters, geometries,
neighbour lists and environment-matrix rows, and the upstream gradient dE/dT.
It holds none of the method's arithmetic (no net evaluation, no table, no
interval search, no fused contraction), so both the CUDA path and the oracle
can consume it without sharing any of the computation they are compared on.

The paper's own datasets are not available; every workload here is a
stand-in with the sizes, neighbour counts and per-type caps of the paper's
Cu, H2O and Al-Cu-Mg systems (Sec. III) and of the 4096-water system of its
network-size study.  The C core (wl_gen.c) is built on first use with gcc.
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess
import tempfile
from dataclasses import dataclass, field

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "wl_gen.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "libwl.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile wl_gen.c into a shared library (atomic rename, safe in parallel)."""
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    os.makedirs(_BUILD_DIR, exist_ok=True)
    fd, tmp = tempfile.mkstemp(suffix=".so", dir=_BUILD_DIR)
    os.close(fd)
    cmd = ["gcc", "-O2", "-fopenmp", "-ffp-contract=off", "-fno-fast-math", "-std=c11",
           "-shared", "-fPIC", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _get_lib():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        P = ctypes.c_void_p
        i64, i32, u64, dbl = ctypes.c_int64, ctypes.c_int, ctypes.c_uint64, ctypes.c_double
        lib.wl_normal.argtypes = [u64, i64, dbl, dbl, P]
        lib.wl_normal.restype = None
        lib.wl_uniform.argtypes = [u64, i64, dbl, dbl, P]
        lib.wl_uniform.restype = None
        lib.wl_det_log.argtypes = [dbl]
        lib.wl_det_log.restype = dbl
        lib.wl_det_cos.argtypes = [dbl]
        lib.wl_det_cos.restype = dbl
        lib.wl_switch.argtypes = [dbl, dbl, dbl, i32]
        lib.wl_switch.restype = dbl
        lib.wl_random_shell.argtypes = [u64, i32, i32, i32, dbl, dbl, dbl, dbl, i32, P, P, P]
        lib.wl_random_shell.restype = i32
        lib.wl_fcc.argtypes = [u64, i32, i32, i32, dbl, dbl, P, P]
        lib.wl_fcc.restype = i32
        lib.wl_species.argtypes = [u64, i64, i32, P, P]
        lib.wl_species.restype = None
        lib.wl_water.argtypes = [u64, i32, i32, dbl, dbl, dbl, dbl, P, P]
        lib.wl_water.restype = i64
        lib.wl_envmat.argtypes = [i64, P, P, P, i32, P, dbl, dbl, i32, P, P, P, P, P, P, i32, P, P]
        lib.wl_envmat.restype = i32
        _lib = lib
    return _lib


def _ptr(a: np.ndarray):
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(ctypes.c_void_p)


def _sub_seed(seed: int, *tags: int) -> int:
    """Derive an independent 64-bit stream seed from (seed, tags...)."""
    x = (seed * 0x9E3779B97F4A7C15 + 0x632BE59BD9B4E019) & 0xFFFFFFFFFFFFFFFF
    for t in tags:
        x = ((x ^ (t + 0x94D049BB133111EB)) * 0xBF58476D1CE4E5B9) & 0xFFFFFFFFFFFFFFFF
        x ^= x >> 31
    return x


def normal(seed: int, shape, mean: float = 0.0, std: float = 1.0) -> np.ndarray:
    n = int(np.prod(shape)) if len(shape) else 1
    out = np.empty(n, dtype=np.float64)
    _get_lib().wl_normal(seed & 0xFFFFFFFFFFFFFFFF, n, mean, std, _ptr(out))
    return out.reshape(shape)


def uniform(seed: int, shape, lo: float = 0.0, hi: float = 1.0) -> np.ndarray:
    n = int(np.prod(shape)) if len(shape) else 1
    out = np.empty(n, dtype=np.float64)
    _get_lib().wl_uniform(seed & 0xFFFFFFFFFFFFFFFF, n, lo, hi, _ptr(out))
    return out.reshape(shape)


def switch(r: float, rcs: float, rc: float, kind: int = 0) -> float:
    """Weighting function s(r): kind 0 cosine switch (workloads), 1 the paper's quintic."""
    return _get_lib().wl_switch(float(r), float(rcs), float(rc), int(kind))


def net_param_count(widths) -> int:
    return sum(widths[l] * widths[l + 1] + widths[l + 1] for l in range(len(widths) - 1))


def net_params(seed: int, widths, npair: int) -> np.ndarray:
    """Random embedding-net parameters, one row per type pair.

    Row layout, layer by layer: W_l [w_l][w_{l+1}] row-major, then b_l [w_{l+1}].
    W_l ~ N(0, 1/w_l), b_l ~ N(0, 1).
    """
    P = net_param_count(widths)
    out = np.empty((npair, P), dtype=np.float64)
    for p in range(npair):
        pos = 0
        for l in range(len(widths) - 1):
            nin, nout = widths[l], widths[l + 1]
            w = normal(_sub_seed(seed, 101, p, l, 0), (nin * nout,), 0.0, 1.0 / math.sqrt(nin))
            b = normal(_sub_seed(seed, 101, p, l, 1), (nout,), 0.0, 1.0)
            out[p, pos:pos + nin * nout] = w
            pos += nin * nout
            out[p, pos:pos + nout] = b
            pos += nout
    return out


def fitting_net(seed: int, in_width: int, hidden=(240, 240, 240), ntypes: int = 1):
    """Random fitting-net parameters, one row per centre type: widths (in_width, *hidden, 1), the
    layout of net_params (W ~ N(0, 1/fan_in), b ~ N(0, 1)).  The paper's nets are (240, 240, 240)."""
    widths = [int(in_width), *[int(h) for h in hidden], 1]
    return widths, net_params(_sub_seed(seed, 505), widths, ntypes)


@dataclass
class Workload:
    """One synthetic batch of the tabulate-fusion path, host arrays.

    s      [nloc][nnei]      f64  embedding input per neighbour row (0 on padding)
    Rt     [nloc][nnei][4]   f64  environment-matrix rows (0 on padding)
    nvalid [nloc][ntypes]    i32  real neighbours per type segment
    atype  [nloc]            i32  centre type (atoms sorted by it)
    params [npair][P]        f64  embedding-net parameters, pair = a*ntypes + b
    dT     [nloc][4][M1]     f64  upstream gradient dE/dT
    """
    name: str
    seed: int
    ntypes: int
    sel: np.ndarray
    widths: list
    M2: int
    s: np.ndarray
    Rt: np.ndarray
    nvalid: np.ndarray
    atype: np.ndarray
    params: np.ndarray
    dT: np.ndarray
    s_min: float
    s_max: float
    stride0: float = 0.01
    stride1: float = 0.1
    ext: float = 5.0
    stats: dict = field(default_factory=dict)
    pos: np.ndarray | None = None
    box: np.ndarray | None = None
    env: dict | None = None  # rcs, rc, switch kind, normalisation, nlist [nloc][nnei], image shift [nloc][nnei][3]

    @property
    def nloc(self) -> int:
        return int(self.s.shape[0])

    @property
    def nnei(self) -> int:
        return int(self.sel.sum())

    @property
    def M1(self) -> int:
        return int(self.widths[-1])

    @property
    def npair(self) -> int:
        return self.ntypes * self.ntypes

    @property
    def evals(self) -> int:
        """Valid neighbour x channel pairs: the unit of work of the path."""
        return int(self.nvalid.astype(np.int64).sum()) * self.M1

    @property
    def fill(self) -> float:
        return float(self.nvalid.astype(np.int64).sum()) / float(self.nloc * self.nnei) if self.nloc else 0.0

    def ncentre(self) -> np.ndarray:
        return np.bincount(self.atype, minlength=self.ntypes).astype(np.int64)

    def describe(self) -> dict:
        return {"workload": self.name, "seed": self.seed, "nloc": self.nloc, "ntypes": self.ntypes,
                "sel": [int(x) for x in self.sel], "nnei": self.nnei, "M1": self.M1, "M2": self.M2,
                "widths": list(self.widths), "fill": round(self.fill, 4),
                "mean_valid_neighbours": round(self.fill * self.nnei, 2),
                "stride0": self.stride0, "stride1": self.stride1, **self.stats}


def _dT(seed: int, nloc: int, M1: int) -> np.ndarray:
    return normal(_sub_seed(seed, 303), (nloc, 4, M1))


def _envmat(pos, types, box, ntypes, sel, rcs, rc, kind=0, norm=None, nthreads=0):
    lib = _get_lib()
    natoms = int(pos.shape[0])
    sel = np.ascontiguousarray(sel, dtype=np.int32)
    nnei = int(sel.sum())
    s = np.empty((natoms, nnei), dtype=np.float64)
    Rt = np.empty((natoms, nnei, 4), dtype=np.float64)
    nvalid = np.empty((natoms, ntypes), dtype=np.int32)
    stats = np.zeros(4, dtype=np.int64)
    srange = np.zeros(2, dtype=np.float64)
    nlist = np.empty((natoms, nnei), dtype=np.int32)
    shift = np.empty((natoms, nnei, 3), dtype=np.int8)
    box = np.ascontiguousarray(box, dtype=np.float64)
    normp = None
    if norm is not None:
        norm_a = np.ascontiguousarray(norm, dtype=np.float64)
        normp = _ptr(norm_a)
    rc_ = lib.wl_envmat(natoms, _ptr(np.ascontiguousarray(pos)), _ptr(np.ascontiguousarray(types, dtype=np.int32)),
                        _ptr(box), ntypes, _ptr(sel), rcs, rc, kind, normp, _ptr(s), _ptr(Rt), _ptr(nvalid),
                        _ptr(stats), _ptr(srange), nthreads, _ptr(nlist), _ptr(shift))
    if rc_ != 0:
        raise RuntimeError(f"wl_envmat failed ({rc_})")
    st = {"real_neighbours_total": int(stats[0]), "rows_dropped_by_sel": int(stats[1]),
          "max_real_neighbours": int(stats[2]), "rows_kept": int(stats[3])}
    env = {"rcs": float(rcs), "rc": float(rc), "kind": int(kind),
           "norm": None if norm is None else tuple(float(x) for x in norm), "nlist": nlist, "shift": shift}
    return s, Rt, nvalid, st, float(srange[0]), float(srange[1]), env


def tiny(seed: int = 1, nloc: int = 64, nreal: int = 24, sel: int = 32, widths=(1, 8, 16, 32), M2: int = 4,
         rmin: float = 0.9, rmax: float = 4.0, rcs: float = 0.5, rc: float = 4.0, kind: int = 0) -> Workload:
    """Random neighbour shells: nreal neighbours at r ~ U[rmin, rmax), uniform directions."""
    lib = _get_lib()
    s = np.empty((nloc, sel), dtype=np.float64)
    Rt = np.empty((nloc, sel, 4), dtype=np.float64)
    nvalid = np.empty((nloc, 1), dtype=np.int32)
    rc_ = lib.wl_random_shell(_sub_seed(seed, 1), nloc, nreal, sel, rmin, rmax, rcs, rc, kind,
                              _ptr(s), _ptr(Rt), _ptr(nvalid))
    if rc_ != 0:
        raise RuntimeError(f"wl_random_shell failed ({rc_})")
    widths = list(widths)
    valid = np.arange(sel)[None, :] < nvalid
    sv = s[valid]
    return Workload(name="tiny", seed=seed, ntypes=1, sel=np.array([sel], dtype=np.int32), widths=widths, M2=M2,
                    s=s, Rt=Rt, nvalid=nvalid, atype=np.zeros(nloc, dtype=np.int32),
                    params=net_params(_sub_seed(seed, 2), widths, 1), dT=_dT(seed, nloc, widths[-1]),
                    s_min=float(sv.min()) if sv.size else 0.0, s_max=float(sv.max()) if sv.size else 0.0,
                    stats={"rcs": rcs, "rc": rc, "nreal": nreal})


def fcc_constant_for(neigh: float, rc: float) -> float:
    """fcc lattice constant whose mean neighbour count inside rc is `neigh` (4 atoms per a^3)."""
    return (4.0 * (4.0 / 3.0) * math.pi * rc ** 3 / neigh) ** (1.0 / 3.0)


def cu(seed: int = 2, fill: float | None = 0.85, a: float | None = None, cells=(8, 8, 16), sel: int = 512,
       widths=(1, 25, 50, 100), M2: int = 16, jitter: float = 0.1, rcs: float = 2.0, rc: float = 8.0,
       name: str | None = None) -> Workload:
    """Cu-like: jittered fcc, one type.  fill=0.85 scales the lattice so ~85 % of sel rows are real."""
    lib = _get_lib()
    if a is None:
        a = fcc_constant_for(fill * sel, rc)
    nx, ny, nz = cells
    nat = 4 * nx * ny * nz
    pos = np.empty((nat, 3), dtype=np.float64)
    box = np.empty(3, dtype=np.float64)
    lib.wl_fcc(_sub_seed(seed, 1), nx, ny, nz, a, jitter, _ptr(pos), _ptr(box))
    types = np.zeros(nat, dtype=np.int32)
    sela = np.array([sel], dtype=np.int32)
    s, Rt, nvalid, st, smin, smax, env = _envmat(pos, types, box, 1, sela, rcs, rc)
    widths = list(widths)
    st.update({"lattice_constant": round(a, 6), "rcs": rcs, "rc": rc, "box": [float(x) for x in box]})
    return Workload(name=name or ("cu85" if fill else "cu"), seed=seed, ntypes=1, sel=sela,
                    widths=widths, M2=M2, s=s, Rt=Rt, nvalid=nvalid, atype=types,
                    params=net_params(_sub_seed(seed, 2), widths, 1), dT=_dT(seed, nat, widths[-1]),
                    s_min=smin, s_max=smax, stats=st, pos=pos, box=box, env=env)


def water(seed: int = 3, nmol: int = 4096, extra_o: int = 0, density: float = 0.0334, sel=(46, 92),
          widths=(1, 25, 50, 100), M2: int = 16, rcs: float = 0.5, rc: float = 6.0, r_oo_min: float = 2.5,
          r_oh: float = 0.96, angle: float = 104.5, name: str = "water", norm=None) -> Workload:
    """Water-like: random liquid-density O with an O-O exclusion, rigid H2O; types O=0, H=1."""
    lib = _get_lib()
    L = ((nmol + extra_o) / density) ** (1.0 / 3.0)
    nat = 3 * nmol + extra_o
    pos = np.empty((nat, 3), dtype=np.float64)
    types = np.empty(nat, dtype=np.int32)
    att = lib.wl_water(_sub_seed(seed, 1), nmol, extra_o, L, r_oo_min, r_oh, angle, _ptr(pos), _ptr(types))
    if att < 0:
        raise RuntimeError(f"wl_water failed ({att})")
    box = np.array([L, L, L], dtype=np.float64)
    sela = np.array(sel, dtype=np.int32)
    s, Rt, nvalid, st, smin, smax, env = _envmat(pos, types, box, 2, sela, rcs, rc, norm=norm)
    widths = list(widths)
    st.update({"box": L, "rcs": rcs, "rc": rc, "placement_attempts": int(att), "molecules": nmol,
               "extra_O": extra_o})
    return Workload(name=name, seed=seed, ntypes=2, sel=sela, widths=widths, M2=M2, s=s, Rt=Rt, nvalid=nvalid,
                    atype=types, params=net_params(_sub_seed(seed, 2), widths, 4), dT=_dT(seed, nat, widths[-1]),
                    s_min=smin, s_max=smax, stats=st, pos=pos, box=box, env=env)


def alcumg(seed: int = 4, pad: float | None = 0.3, cells=(16, 16, 32), sel=(400, 60, 40),
           frac=(0.90, 0.06, 0.04), widths=(1, 25, 50, 100), M2: int = 16, jitter: float = 0.1,
           rcs: float = 2.0, rc: float = 8.0, name: str | None = None) -> Workload:
    """Al-Cu-Mg-like: jittered fcc, three species 90/6/4 %, atoms sorted by species.

    pad = target padding fraction of the 500 rows; the lattice constant is scaled so
    that (1 - pad) * nnei real neighbours are expected.  pad=None keeps a = 4.05.
    """
    lib = _get_lib()
    sela = np.array(sel, dtype=np.int32)
    nnei = int(sela.sum())
    a = 4.05 if pad is None else fcc_constant_for((1.0 - pad) * nnei, rc)
    nx, ny, nz = cells
    nat = 4 * nx * ny * nz
    pos = np.empty((nat, 3), dtype=np.float64)
    box = np.empty(3, dtype=np.float64)
    lib.wl_fcc(_sub_seed(seed, 1), nx, ny, nz, a, jitter, _ptr(pos), _ptr(box))
    types = np.empty(nat, dtype=np.int32)
    fr = np.array(frac, dtype=np.float64)
    lib.wl_species(_sub_seed(seed, 3), nat, len(frac), _ptr(fr), _ptr(types))
    order = np.argsort(types, kind="stable")
    pos = np.ascontiguousarray(pos[order])
    types = np.ascontiguousarray(types[order])
    s, Rt, nvalid, st, smin, smax, env = _envmat(pos, types, box, 3, sela, rcs, rc)
    widths = list(widths)
    achieved_pad = 1.0 - float(nvalid.astype(np.int64).sum()) / float(nat * nnei)
    st.update({"lattice_constant": round(a, 6), "pad_target": pad, "pad_achieved": round(achieved_pad, 4),
               "rcs": rcs, "rc": rc, "box": [float(x) for x in box]})
    return Workload(name=name or (f"alcumg_pad{int(round(pad * 100))}" if pad is not None else "alcumg_a405"),
                    seed=seed, ntypes=3, sel=sela, widths=widths, M2=M2, s=s, Rt=Rt, nvalid=nvalid, atype=types,
                    params=net_params(_sub_seed(seed, 2), widths, 9), dT=_dT(seed, nat, widths[-1]),
                    s_min=smin, s_max=smax, stats=st, pos=pos, box=box, env=env)


def water_large(seed: int = 5, nmol: int = 349525, extra_o: int = 1, **kw) -> Workload:
    """Large water-like: 349,525 molecules + 1 O = 1,048,576 atoms."""
    return water(seed=seed, nmol=nmol, extra_o=extra_o, name="water_large", **kw)


def make(name: str, **kw) -> Workload:
    """Workload by name: tiny, cu85, cugeo, water, alcumg (pad=...), water_large."""
    if name == "tiny":
        return tiny(**kw)
    if name == "cu85":
        return cu(fill=0.85, name="cu85", **kw)
    if name == "cugeo":
        return cu(fill=None, a=3.6, name="cugeo", **kw)
    if name == "water":
        return water(**kw)
    if name == "alcumg":
        return alcumg(**kw)
    if name == "water_large":
        return water_large(**kw)
    raise KeyError(name)


def shard(nloc: int, rank: int, world: int) -> tuple[int, int]:
    """Contiguous atom range [lo, hi) of `rank` when nloc atoms are split over `world` ranks."""
    base, rem = divmod(nloc, world)
    lo = rank * base + min(rank, rem)
    return lo, lo + base + (1 if rank < rem else 0)


def ghost_system(w: Workload):
    """Coordinates with periodic images as extra atoms, for inputs given as positions and a neighbour list.

    Returns (coord [nall][3] f64, nlist [nloc][nnei] int32 indexing coord, -1 on padding rows,
    owner [nall] int32: the local atom each coordinate is a copy of).  Neighbour rows whose image
    shift is zero point at the local atom itself; every other (atom, shift) pair becomes one
    image, placed at r_j + shift * box.
    """
    if w.env is None or w.pos is None:
        raise ValueError(f"workload {w.name} has no positions and neighbour list")
    nl, sh = w.env["nlist"], w.env["shift"].astype(np.int64)
    nloc = w.nloc
    code = (sh[..., 0] + 1) * 9 + (sh[..., 1] + 1) * 3 + (sh[..., 2] + 1)  # 13 = no shift
    need = (nl >= 0) & (code != 13)
    key = nl.astype(np.int64) * 27 + code
    uniq, inv = np.unique(key[need], return_inverse=True)
    j_img, c_img = uniq // 27, uniq % 27
    shv = np.stack([c_img // 9 - 1, (c_img // 3) % 3 - 1, c_img % 3 - 1], axis=1).astype(np.float64)
    coord = np.concatenate([w.pos, w.pos[j_img] + shv * w.box[None, :]], axis=0)
    nlist = nl.copy()
    nlist[need] = (nloc + inv).astype(np.int32)
    owner = np.concatenate([np.arange(nloc), j_img]).astype(np.int32)
    return np.ascontiguousarray(coord), np.ascontiguousarray(nlist), owner
