"""The C ABI library loads and exports every symbol its header declares;
host-side argument checks return their codes without touching a GPU."""
import ctypes
import os
import re

import numpy as np
import pytest

from paper_2609_08443_gb300 import binding, build

HEADER = os.path.join(os.path.dirname(os.path.dirname(__file__)), "include", "sa_sketch.h")


@pytest.fixture(scope="module")
def lib():
    build.build()
    return binding.load()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(sa_[a-z_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for must in ("sa_workspace_size", "sa_sketch_fwd", "sa_sketch_bwd", "sa_get_device_error",
                 "sa_status_string"):
        assert must in names


def test_every_declared_symbol_is_exported(lib):
    for name in declared_functions():
        assert hasattr(lib, name), f"{name} declared in sa_sketch.h but not exported"


def test_status_strings(lib):
    for code in range(7):
        s = binding.sa_status_string(code)
        assert s and s != "unknown status"
    assert binding.sa_status_string(99) == "unknown status"


def test_workspace_size_rejects_bad_shapes(lib):
    assert binding.sa_workspace_size(1, 10, 1, 0, 64, 1, 0) == 0       # P = 0
    assert binding.sa_workspace_size(1, 10, 1, 4096, 64, 1, 0) == 0    # P too large
    assert binding.sa_workspace_size(1, 10, 1, 64, 12, 1, 0) == 0      # d not multiple of 8 (bf16)
    assert binding.sa_workspace_size(0, 10, 1, 64, 64, 1, 0) == 0      # B = 0
    assert binding.sa_workspace_size(1, 2**31, 1, 64, 64, 1, 0) == 0   # N too large
    a = binding.sa_workspace_size(4, 1000, 2, 256, 64, 1, 0)
    b = binding.sa_workspace_size(4, 1000, 2, 256, 64, 1, 1)
    assert a > 0 and b >= a and a % 256 == 0 and b % 256 == 0


def _fwd(lib, **kw):
    args = dict(K=256, V=512, cu=768, B=2, N=100, Q=1024, H=2, P=64, d=64, scale=0.125, dt=1,
                sketch=2048, lse=None, ws=4096, wsb=1 << 30)
    args.update(kw)
    vp = ctypes.c_void_p
    return lib.sa_sketch_fwd(vp(args["K"]), vp(args["V"]), vp(args["cu"]), args["B"], args["N"], vp(args["Q"]),
                             args["H"], args["P"], args["d"], args["scale"], args["dt"], vp(args["sketch"]),
                             vp(args["lse"]) if args["lse"] else None, vp(args["ws"]), args["wsb"], None)


def test_host_checks_return_codes_before_any_launch(lib):
    # fake, never-dereferenced addresses: only the host checks run
    assert _fwd(lib, sketch=0) == 1                      # NULL output
    assert _fwd(lib, cu=0) == 1                          # NULL offsets
    assert _fwd(lib, scale=float("nan")) == 1            # non-finite scale
    assert _fwd(lib, ws=4096 + 8) == 1                   # workspace not 256-aligned
    assert _fwd(lib, K=256 + 2) == 1                     # K not 16-byte aligned
    assert _fwd(lib, P=4096) == 2                        # unsupported P
    assert _fwd(lib, d=200) == 2                         # unsupported d
    assert _fwd(lib, dt=7) == 2                          # unknown dtype
    assert _fwd(lib, wsb=16) == 3                        # workspace too small


def test_plan_host_covers_every_tile_once(lib):
    rng = np.random.default_rng(0)
    for lens in ([0], [1], [128], [129], [0, 0, 5], list(rng.integers(0, 600, size=4100)),
                 [100000] * 3 + [0, 1, 127, 128, 129]):
        cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
        for H in (1, 8):
            for W in (1, 7, 152, 10000):
                begin = binding.sa_plan_host(cu, H, 128, W)
                tiles = H * sum((L + 127) // 128 for L in lens)
                assert begin[0] == 0 and begin[-1] == tiles
                sizes = np.diff(begin)
                assert np.all(sizes >= 0) and sizes.max() - sizes.min() <= 1


def _tiles_in_order(lens, H, T):
    """Every tile of the batch in (head, user, tile) order, written out."""
    cu = np.concatenate([[0], np.cumsum(lens)])
    rows = []
    for h in range(H):
        for b, L in enumerate(lens):
            for k in range((L + T - 1) // T):
                rows.append((b, h, cu[b] + k * T, min(T, L - k * T)))
    return np.array(rows, dtype=np.int64).reshape(-1, 4)


def test_walk_host_matches_the_tile_order(lib):
    """The kernels' walk over their ranges (search for the first tile, steps
    inside a segment, forward scan to the next segment's user) gives every tile
    of the (head, user, tile) order, including across runs of empty users longer
    than the scan (where it falls back to the search) and users cut across
    workers."""
    rng = np.random.default_rng(1)
    gaps = [0] * 9 + [5, 300, 1]                        # nine empty users in a row, then more
    cases = [[5], [0, 0, 7], [130, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 129, 0],
             gaps * 3, [0] * 20 + [1] + [0] * 20 + [256],
             list(rng.integers(0, 600, size=500)),
             [int(x) if rng.random() < 0.3 else 0 for x in rng.integers(1, 400, size=300)],
             [100000] * 2 + [0] * 17 + [1, 127, 128, 129]]
    for lens in cases:
        cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
        for H in (1, 3):
            want = _tiles_in_order(lens, H, 128)
            for W in (1, 5, 152, 777):
                user, head, tok0, ntok = binding.sa_walk_host(cu, H, 128, W)
                got = np.stack([user, head, tok0, ntok], axis=1).astype(np.int64)
                assert got.shape == want.shape and np.array_equal(got, want), (lens[:8], H, W)


def test_plan_host_rejects_bad_offsets(lib):
    with pytest.raises(binding.SketchError):
        binding.sa_plan_host(np.array([0, 5, 3], np.int32), 1, 128, 4)
    with pytest.raises(binding.SketchError):
        binding.sa_plan_host(np.array([1, 5], np.int32), 1, 128, 4)


def test_tokenwise_host_checks(lib):
    vp = ctypes.c_void_p

    def fwd(**kw):
        a = dict(K=256, V=512, cu=768, B=2, N=100, Q=1024, H=2, P=64, d=64, scale=0.125, dt=1, sketch=2048,
                 ws=4096, wsb=1 << 30)
        a.update(kw)
        return lib.sa_sketch_fwd_tokenwise(vp(a["K"]), vp(a["V"]), vp(a["cu"]), a["B"], a["N"], vp(a["Q"]), a["H"],
                                           a["P"], a["d"], a["scale"], a["dt"], vp(a["sketch"]) if a["sketch"] else None,
                                           None, vp(a["ws"]), a["wsb"], None)

    assert fwd(sketch=0) == 1
    assert fwd(ws=4096 + 8) == 1
    assert fwd(P=4096) == 2
    assert fwd(wsb=16) == 3
    bwd = lib.sa_sketch_bwd_tokenwise(vp(256), vp(512), vp(768), 2, 100, vp(1024), 2, 64, 64, 0.125, 1, None, None,
                                      None, vp(2048), vp(2304), vp(2560), vp(4096), 1 << 30, None)
    assert bwd == 1  # NULL dsketch
    a = binding.load().sa_workspace_size_tokenwise(4, 1000, 2, 256, 64, 1, 0)
    b = binding.load().sa_workspace_size_tokenwise(4, 1000, 2, 256, 64, 1, 1)
    assert a > 0 and b > a and a % 256 == 0 and b % 256 == 0
    assert binding.load().sa_workspace_size_tokenwise(1, 10, 1, 4096, 64, 1, 0) == 0


def test_chunk_plan_host(lib):
    """The user chunks of the host-buffer pipeline: consecutive users within the
    token budget, a longer user alone, every user exactly once."""
    lens = [5, 0, 7, 3, 20, 1, 1, 0, 6]
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    b = binding.sa_plan_chunks_host(cu, chunk_tokens=10)
    assert b[0] == 0 and b[-1] == len(lens) and np.all(np.diff(b) > 0)
    for c in range(len(b) - 1):
        tok = int(cu[b[c + 1]] - cu[b[c]])
        assert tok <= 10 or b[c + 1] - b[c] == 1, (c, tok)
        if c + 1 < len(b) - 1:  # a chunk closes only when the next user would overflow it
            assert tok + lens[b[c + 1]] > 10
    assert list(b) == [0, 2, 4, 5, 9]
    many = np.arange(3001, dtype=np.int32)  # 3000 one-token users: at most 1024 per chunk
    assert list(binding.sa_plan_chunks_host(many, chunk_tokens=1 << 20)) == [0, 1024, 2048, 3000]
    with pytest.raises(binding.SketchError):
        binding.sa_plan_chunks_host(np.array([0, 5, 3], dtype=np.int32))


def test_step_host_checks(lib):
    vp = ctypes.c_void_p
    cu = np.array([0, 4, 10], dtype=np.int32)
    # NULL host output and a workspace that is too small: refused before any copy
    st = lib.sa_sketch_step_host(vp(256), vp(512), cu.ctypes.data, 2, 10, vp(1024), 1, 64, 64, 0.125, 1, vp(2048),
                                 None, vp(4096), vp(8192), vp(9216), 0, vp(1 << 20), 1 << 30, None)
    assert st == 1
    st = lib.sa_sketch_step_host(vp(256), vp(512), cu.ctypes.data, 2, 10, vp(1024), 1, 64, 64, 0.125, 1, vp(2048),
                                 vp(3072), vp(4096), vp(8192), vp(9216), 0, vp(1 << 20), 16, None)
    assert st == 3
    assert lib.sa_step_host_workspace_size(cu.ctypes.data, 2, 1, 64, 64, 1, 0) > 0


def test_wait_limit_bounds(lib):
    assert lib.sa_set_wait_limit_ns(5 * 10**9) == 1  # above 4 s: SA_ERR_INVALID_ARG
    assert lib.sa_set_wait_limit_ns(3 * 10**9) == 0
    assert lib.sa_set_wait_limit_ns(0) == 0           # back to the default
