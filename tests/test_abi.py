"""Host-side checks of the C ABI: the library builds, loads and exports every
symbol include/grpo.h declares, and host-detectable errors come back as status
codes without touching a GPU."""
import ctypes
import os
import re

import numpy as np
import pytest

import paper_2507_05687_gb300 as grpo
from paper_2507_05687_gb300 import build as build_mod

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HERE = os.path.dirname(os.path.abspath(__file__))


@pytest.fixture(scope="module")
def lib():
    build_mod.build()
    return grpo.load()


def header_symbols():
    text = open(os.path.join(ROOT, "include", "grpo.h")).read()
    return sorted(set(re.findall(r"^\S.*?\b(grpo_\w+)\(", text, flags=re.M)))


def test_header_declares_the_boundary():
    syms = header_symbols()
    for name in ("grpo_group_advantages", "grpo_token_logprobs", "grpo_loss_fwd_bwd",
                 "grpo_workspace_bytes", "grpo_check_device_status", "grpo_status_string"):
        assert name in syms
    assert set(syms) == set(grpo.SIGNATURES), "binding and header disagree"


def test_every_declared_symbol_is_exported(lib):
    for name in header_symbols():
        assert hasattr(lib, name), name
    # exported with C linkage (no mangling)
    raw = ctypes.CDLL(grpo.LIB_PATH)
    for name in header_symbols():
        assert ctypes.cast(getattr(raw, name), ctypes.c_void_p).value


def test_status_strings(lib):
    for code, name in ((0, "GRPO_OK"), (1, "GRPO_ERR_INVALID_ARG"), (2, "GRPO_ERR_WORKSPACE"),
                       (5, "GRPO_ERR_TIMEOUT"), (6, "GRPO_ERR_UNSUPPORTED")):
        assert grpo.status_string(code) == name


def test_workspace_sizes(lib):
    f = grpo.workspace_bytes
    assert f(256, 256, 4096, 0) > 256 * 256 * 2
    assert f(32768, 4096, 155136, 1) > f(32768, 4096, 155136, 0) > 32768 * 4096 * 2
    assert f(0, 64, 10, 0) > 0
    for bad in ((-1, 64, 10, 0), (10, 60, 10, 0), (10, 0, 10, 0), (10, 64, 0, 0), (10, 64, 10, 7),
                (1 << 31, 64, 10, 0)):
        assert f(*bad) == 0, bad
    assert f(1000, 128, 300, 1) % 1024 == 0


FAKE = 0x10000  # never dereferenced: every call below is rejected on the host


def test_workspace_sized_for_fewer_rows(lib):
    f, g = grpo.workspace_bytes, grpo.workspace_bytes_rows
    for which in (0, 1, 2, 3, 4, 5):
        full = f(32768, 4096, 155136, which)
        assert g(32768, 32768, 4096, 155136, which) == full == g(32768, 10**9, 4096, 155136, which)
        sizes = [g(32768, n, 4096, 155136, which) for n in (1, 256, 257, 5000, 20000)]
        assert sizes[0] == sizes[1] < sizes[2] <= sizes[3] <= sizes[4] < full   # 256-row granularity
        assert g(32768, -1, 4096, 155136, which) == 0
    # a ragged batch: 1M padded rows, 168k unmasked
    assert g(1 << 20, 168251, 4096, 155136, 1) < 0.2 * f(1 << 20, 4096, 155136, 1)


def test_loss_plan_keeps_logits_only_for_exact_kept_sizes(lib):
    """grpo_loss_plan: a GRPO_WS_LOSS_LOGITS workspace is the plain loss one plus
    the fp32 logits [rows x V]; the loss calls keep the logits only when the
    workspace is exactly such a size.  Any other size, however large, runs the
    recomputing backward with the largest plain row capacity that fits."""
    f, g, plan = grpo.workspace_bytes, grpo.workspace_bytes_rows, grpo.loss_plan
    T, Hd, V = 32768, 4096, 155136
    kept, plain = f(T, Hd, V, grpo.GRPO_WS_LOSS_LOGITS), f(T, Hd, V, grpo.GRPO_WS_LOSS)
    assert kept - plain == 4 * T * V
    assert plan(T, Hd, V, kept) == (1, T)
    # room for the logits is not a request for them
    assert plan(T, Hd, V, kept + 1024) == (0, T) and plan(T, Hd, V, 4 * kept) == (0, T)
    assert plan(T, Hd, V, kept - 1) == (0, T) and plan(T, Hd, V, plain) == (0, T)
    assert plan(T, Hd, V, plain - 1) == (0, T - 256)
    rng = np.random.default_rng(7)
    # exactly a kept-logits size: the capacity it was sized for, logits kept
    for mv in (1, 256, 5000, 19572, 32768):
        assert plan(T, Hd, V, g(T, mv, Hd, V, grpo.GRPO_WS_LOSS_LOGITS)) == (1, (mv + 255) // 256 * 256)
        assert plan(T, Hd, V, g(T, mv, Hd, V, grpo.GRPO_WS_LOSS_LOGITS) + 1024)[0] == 0
    kept_sizes = {g(T, mv, Hd, V, grpo.GRPO_WS_LOSS_LOGITS) for mv in range(256, T + 1, 256)}
    # any other size: the plain layout with its largest capacity
    for ws in rng.integers(g(T, 1, Hd, V, 1), 2 * kept, size=300):
        k, rows = plan(T, Hd, V, int(ws))
        assert rows % 256 == 0 and g(T, rows, Hd, V, 1) <= ws and (rows == T or g(T, rows + 1, Hd, V, 1) > ws)
        assert k == int(int(ws) in kept_sizes)
    # odd vocabulary: logits rows padded to 64 columns
    assert f(100, 64, 1001, 4) - f(100, 64, 1001, 1) == 4 * 256 * 1024
    rows = ctypes.c_int64(-5)
    assert lib.grpo_loss_plan(T, Hd, V, g(T, 1, Hd, V, 1) - 1, ctypes.byref(rows)) == -1 and rows.value == -5
    for bad in ((-1, Hd, V), (T, 60, V), (T, Hd, 0)):
        assert lib.grpo_loss_plan(*bad, kept, None) == -1
    with pytest.raises(grpo.GrpoError):
        plan(T, Hd, V, 1000)


def test_host_rejections(lib):
    L = lib
    assert L.grpo_group_advantages(FAKE, 8, 1, 1e-6, FAKE, None) == grpo.GRPO_ERR_INVALID_ARG
    assert L.grpo_group_advantages(FAKE, 9, 4, 1e-6, FAKE, None) == grpo.GRPO_ERR_INVALID_ARG
    assert L.grpo_group_advantages(None, 8, 4, 1e-6, FAKE, None) == grpo.GRPO_ERR_INVALID_ARG
    assert L.grpo_group_advantages(None, 0, 4, 1e-6, None, None) == grpo.GRPO_OK
    ws_need = grpo.workspace_bytes(100, 64, 1000, 0)
    args = [FAKE, FAKE, FAKE, FAKE, 100, 64, 1000, FAKE, FAKE, ws_need, None]
    bad = list(args); bad[4 + 1] = 96 - 1          # Hd not a multiple of 64
    assert L.grpo_token_logprobs(*bad) == grpo.GRPO_ERR_INVALID_ARG
    bad = list(args); bad[0] = None               # H missing
    assert L.grpo_token_logprobs(*bad) == grpo.GRPO_ERR_INVALID_ARG
    bad = list(args); bad[1] = FAKE + 2           # W not 16-byte aligned
    assert L.grpo_token_logprobs(*bad) == grpo.GRPO_ERR_INVALID_ARG
    bad = list(args); bad[9] = ws_need - 1        # workspace too small
    assert L.grpo_token_logprobs(*bad) == grpo.GRPO_ERR_WORKSPACE
    bad = list(args); bad[8] = FAKE + 16          # workspace misaligned
    assert L.grpo_token_logprobs(*bad) == grpo.GRPO_ERR_WORKSPACE
    ws2 = grpo.workspace_bytes(40, 64, 1000, 1)
    largs = [FAKE] * 7 + [10, 4, 64, 1000, 0.2, 0.04, 0, FAKE, FAKE, FAKE, FAKE, ws2, None]
    for i, v in ((7, 0), (8, 0), (11, -0.1), (13, 2), (13, -1)):
        bad = list(largs); bad[i] = v
        assert L.grpo_loss_fwd_bwd(*bad) == grpo.GRPO_ERR_INVALID_ARG, i
    bad = list(largs); bad[16] = FAKE + 4          # dW misaligned
    assert L.grpo_loss_fwd_bwd(*bad) == grpo.GRPO_ERR_INVALID_ARG
    bad = list(largs); bad[18] = grpo.workspace_bytes_rows(40, 1, 64, 1000, 1) - 256   # not even 256 rows fit
    assert L.grpo_loss_fwd_bwd(*bad) == grpo.GRPO_ERR_WORKSPACE
    kargs = largs[:14] + [0.0, 1.0] + largs[14:]
    for kappa in (-1.0, float("nan"), float("-inf")):
        bad = list(kargs); bad[15] = kappa
        assert L.grpo_loss_fwd_bwd_kl_clamp(*bad) == grpo.GRPO_ERR_INVALID_ARG, kappa
    bad = list(kargs); bad[7] = 0                 # n_resp 0
    assert L.grpo_loss_fwd_bwd_kl_clamp(*bad) == grpo.GRPO_ERR_INVALID_ARG
    for row0, rows, cols in ((0, -1, 4), (0, 4, -1), (-1, 4, 4), (0, 2**32 + 1, 4), (2**32 - 3, 4, 4),
                             (0, 4, 2**31), (0, 2**21, 2**20)):
        assert L.grpo_gumbel_noise(1, 2, row0, rows, cols, FAKE, None) == grpo.GRPO_ERR_INVALID_ARG, (row0, rows)
    assert L.grpo_gumbel_noise(1, 2, 0, 4, 4, None, None) == grpo.GRPO_ERR_INVALID_ARG
    assert L.grpo_gumbel_noise(1, 2, 0, 4, 4, FAKE + 2, None) == grpo.GRPO_ERR_INVALID_ARG
    assert L.grpo_gumbel_noise(1, 2, 2**32, 0, 4, None, None) == grpo.GRPO_OK
    wst = grpo.workspace_bytes(100, 64, 1000, grpo.GRPO_WS_SAMPLE_TOP_P)
    assert wst > grpo.workspace_bytes(100, 64, 1000, grpo.GRPO_WS_LOGPROBS) + 4 * 256 * 1024 - 1
    targs = [FAKE, FAKE, FAKE, 100, 64, 1000, 1.0, 0.9, 1, 2, FAKE, FAKE, FAKE, wst, None]
    for i, v in ((7, 0.0), (7, -0.5), (7, 1.01), (7, float("nan")), (6, 0.0), (6, float("inf")), (4, 60)):
        bad = list(targs); bad[i] = v
        assert L.grpo_sample_tokens_top_p(*bad) == grpo.GRPO_ERR_INVALID_ARG, (i, v)
    bad = list(targs); bad[13] = wst - 1024 * 257   # fewer than 256 rows of logits fit
    assert L.grpo_sample_tokens_top_p(*bad) == grpo.GRPO_ERR_WORKSPACE
    bad = list(targs); bad[3] = 0                 # no rows: nothing to do
    assert L.grpo_sample_tokens_top_p(*bad) == grpo.GRPO_OK
    eargs = largs[:14] + [0.0] + largs[14:17] + [None, 0] + largs[17:]
    assert L.grpo_loss_fwd_bwd_events(*eargs) == grpo.GRPO_ERR_INVALID_ARG          # no event array
    few = (ctypes.c_void_p * 1)(FAKE)
    bad = list(eargs); bad[18], bad[19] = few, 0
    assert L.grpo_loss_fwd_bwd_events(*bad) == grpo.GRPO_ERR_INVALID_ARG            # fewer events than chunks
    nulls1 = (ctypes.c_void_p * 1)(None)
    bad = list(eargs); bad[18], bad[19] = nulls1, 1
    assert L.grpo_loss_fwd_bwd_events(*bad) == grpo.GRPO_ERR_INVALID_ARG            # a null event
    assert L.grpo_vocab_chunk_cols(0) == 0 and L.grpo_vocab_chunk_cols(1000) == 1024
    assert L.grpo_check_device_status(None, None) == grpo.GRPO_ERR_INVALID_ARG
    ws3 = grpo.workspace_bytes(100, 64, 1000, grpo.GRPO_WS_LOGPROBS_HEADS)
    assert ws3 > grpo.workspace_bytes(100, 64, 1000, grpo.GRPO_WS_LOGPROBS)
    heads = (ctypes.c_void_p * 5)(*([FAKE] * 5))
    hargs = [FAKE, heads, 3, FAKE, FAKE, 100, 64, 1000, FAKE, FAKE, ws3, None]
    for n in (0, 5):
        bad = list(hargs); bad[2] = n
        assert L.grpo_token_logprobs_heads(*bad) == grpo.GRPO_ERR_INVALID_ARG
    nulls = (ctypes.c_void_p * 3)(FAKE, None, FAKE)
    bad = list(hargs); bad[1] = nulls
    assert L.grpo_token_logprobs_heads(*bad) == grpo.GRPO_ERR_INVALID_ARG
    bad = list(hargs); bad[10] = ws3 - 1
    assert L.grpo_token_logprobs_heads(*bad) == grpo.GRPO_ERR_WORKSPACE
    wss = grpo.workspace_bytes(100, 64, 1000, grpo.GRPO_WS_SAMPLE)
    assert wss > grpo.workspace_bytes(100, 64, 1000, grpo.GRPO_WS_LOGPROBS)
    sargs = [FAKE, FAKE, FAKE, 100, 64, 1000, 1.0, 1, 2, FAKE, FAKE, FAKE, wss, None]
    for tau in (0.0, -2.0, float("inf"), float("nan")):
        bad = list(sargs); bad[6] = tau
        assert L.grpo_sample_tokens(*bad) == grpo.GRPO_ERR_INVALID_ARG
    bad = list(sargs); bad[12] = wss - 1
    assert L.grpo_sample_tokens(*bad) == grpo.GRPO_ERR_WORKSPACE
    bad = list(sargs); bad[2] = None
    assert L.grpo_sample_tokens(*bad) == grpo.GRPO_ERR_INVALID_ARG


def test_binding_fails_loudly_without_library(tmp_path):
    from paper_2507_05687_gb300 import binding
    with pytest.raises(ImportError):
        binding.open_library(str(tmp_path / "missing.so"))


def _build_c_check(tmp_path):
    """A C11 compiler (gcc, else cc or clang) on include/grpo.h, linked to the
    in-tree libgrpo.so.  The build step needs a host compiler too (nvcc uses
    one), so a machine that built the library has one of these."""
    import shutil
    import subprocess
    gcc = next((c for c in (shutil.which(n) for n in ("gcc", "cc", "clang")) if c), None)
    assert gcc is not None, "no C compiler (gcc, cc, clang) on PATH"
    cuda = os.environ.get("CUDA_HOME", "/usr/local/cuda")
    lib_dir = os.path.dirname(grpo.LIB_PATH)
    exe = str(tmp_path / "c_abi_check")
    cmd = [gcc, "-std=c11", "-Wall", "-Wextra", "-Werror", os.path.join(HERE, "c_abi_check.c"),
           "-I", os.path.join(ROOT, "include"), "-I", os.path.join(cuda, "include"), "-o", exe,
           "-L", lib_dir, "-lgrpo", "-Wl,-rpath," + lib_dir, "-L", os.path.join(cuda, "lib64"), "-lcudart",
           "-Wl,-rpath," + os.path.join(cuda, "lib64"), "-lm"]
    subprocess.run(cmd, check=True, capture_output=True, text=True)
    return exe


def test_c_program_compiles_links_and_runs_host_checks(lib, tmp_path):
    """The boundary is a C ABI: a C11 program uses it with no Python involved."""
    import subprocess
    exe = _build_c_check(tmp_path)
    out = subprocess.run([exe, "host"], capture_output=True, text=True, timeout=60)
    assert out.returncode == 0 and out.stdout.strip() == "ok", out.stdout + out.stderr
