"""The C-ABI library builds for sm_103a, loads, exports every function include/grpo.h declares,
and rejects bad arguments on the host before touching the GPU (no GPU needed)."""
import ctypes

import pytest

import __graft_entry__
from paper_2510_17158_gb300 import grpo as G


@pytest.fixture(scope="module")
def lib():
    __graft_entry__.build()
    return G._lib()


def test_exports_every_declared_function(lib):
    names = G.header_functions()
    assert "grpo_score_fwd" in names and "grpo_loss_bwd" in names and "group_advantages" in names
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, missing


def test_status_strings_and_kernel_names(lib):
    for st in range(-7, 1):
        assert G.grpo_status_string(st) != "unknown status"
    assert [G.grpo_kernel_name(k) for k in range(len(G.KERNEL_NAMES))] == G.KERNEL_NAMES


def test_workspace_bytes(lib):
    S, T, d, V = 32, 16384, 5120, 151936
    full = G.grpo_workspace_bytes(S, T, d, V, G.GRPO_BF16, 0)
    rows = S * 128 * 128
    assert full >= rows * 152064 * 2                 # whole-vocabulary dz scratch
    small = G.grpo_workspace_bytes(S, T, d, V, G.GRPO_BF16, 8192)
    assert small < full and small >= rows * 8192 * 2 + rows * d * 4
    assert G.grpo_workspace_bytes(0, T, d, V, G.GRPO_BF16, 0) == 0
    # the exact-KL entry points add the reference model's packed rows (bf16) and its forward
    # statistics (one float4 per 256 vocabulary columns), each over the packed-row capacity
    rows = -(-S * T // 128) * 128
    extra = G.grpo_workspace_bytes_kl(S, T, d, V, G.GRPO_BF16, 0) - full
    want = rows * d * 2 + rows * 16 * -(-V // 256)
    assert want <= extra <= want + 2 * 256
    assert G.grpo_workspace_bytes_kl(4, 64, 64, 512, G.GRPO_F32, 0) == 0   # bf16 only
    assert G.grpo_workspace_bytes(4, 64, 64, 512, G.GRPO_F32, 0) > 0


def test_host_validation_rejects_before_launch(lib):
    nul = ctypes.c_void_p(0)
    st = lib.grpo_score_fwd(nul, nul, 1, nul, nul, 4, 64, 256, 512, nul, nul, nul, nul, nul, nul,
                            1 << 20, nul)
    assert st == -1
    fake = ctypes.c_void_p(1 << 20)      # never dereferenced: validation fails first
    # d not a multiple of 64 is unsupported on the bf16 tensor-core path
    st = lib.grpo_score_fwd(fake, fake, 1, fake, fake, 4, 64, 288, 512, fake, fake, fake, fake,
                            fake, fake, 1 << 30, nul)
    assert st == -2
    # misaligned workspace
    st = lib.grpo_score_fwd(fake, fake, 1, fake, fake, 4, 64, 256, 512, fake, fake, fake, fake,
                            fake, ctypes.c_void_p((1 << 20) + 8), 1 << 30, nul)
    assert st == -4
    # ref_logp NULL with beta > 0
    st = lib.grpo_loss_bwd(fake, fake, 1, fake, fake, 4, 64, 256, 512, fake, fake, fake, nul,
                           fake, fake, 0.2, 0.2, 0.04, 0, 0.0, fake, fake, fake, fake, 1 << 30, nul)
    assert st == -1
    # bad aggregation mode
    st = lib.grpo_loss_bwd(fake, fake, 1, fake, fake, 4, 64, 256, 512, fake, fake, fake, fake,
                           fake, fake, 0.2, 0.2, 0.04, 7, 0.0, fake, fake, fake, fake, 1 << 30, nul)
    assert st == -1
    # workspace too small
    st = lib.grpo_loss_bwd(fake, fake, 1, fake, fake, 4, 64, 256, 512, fake, fake, fake, fake,
                           fake, fake, 0.2, 0.2, 0.04, 0, 0.0, fake, fake, fake, fake, 1024, nul)
    assert st == -4
    # group advantages: bad std mode, no workspace
    st = lib.group_advantages(fake, fake, 2, 8, 5, 1e-4, fake, fake, 1024, nul)
    assert st == -1
    st = lib.group_advantages(fake, fake, 2, 8, 0, 1e-4, fake, nul, 1024, nul)
    assert st == -4


def test_process_wide_settings_validate_and_round_trip(lib):
    """Host-only setters (no GPU work): tile modes 0, 1 and 2 accepted for every role at once
    and read back, others refused; the progress window refuses a negative
    lag and a checkpoint with lag 0, and takes negative checkpoint spacings (in work units); the
    CTA-pair switch maps to tile modes 1 / 0."""
    try:
        for mode in (0, 2, 1):
            assert lib.grpo_set_tile_mode(mode) == 0
            assert lib.grpo_get_tile_mode() == mode
            assert [lib.grpo_get_role_tile_mode(r) for r in range(4)] == [mode] * 4
        for bad in (-2, 3, 4, 5, 1 << 20):
            assert lib.grpo_set_tile_mode(bad) == -1
            assert lib.grpo_get_tile_mode() == 1          # unchanged by a refused call
        assert lib.grpo_set_cta_pair(0) == 0 and lib.grpo_get_tile_mode() == 0
        assert lib.grpo_set_cta_pair(1) == 0 and lib.grpo_get_tile_mode() == 1
    finally:
        lib.grpo_set_tile_mode(-1)
    assert lib.grpo_set_gemm_window(16, -1) == -1
    assert lib.grpo_set_gemm_window(16, 0) == -1
    assert lib.grpo_set_gemm_window(-1, 0) == -1
    assert lib.grpo_set_gemm_window(16, 4) == 0
    assert lib.grpo_set_gemm_window(-1, 1) == 0      # checkpoints at every unit start
    assert lib.grpo_set_gemm_window(-2, 2) == 0
    assert lib.grpo_set_gemm_window(0, 0) == 0
    assert lib.grpo_set_gemm_window(*G.GEMM_WINDOW_DEFAULT) == 0   # back to the library's default


def test_role_tile_modes_defaults_overrides_and_refusals(lib):
    """Per-role tile modes (host-only): the library starts with its per-role defaults (forward
    and dz 0, dH and dW 2; the shared mode then reads -1), an override changes its own role
    only, -1 restores defaults, and bad roles or modes are refused without changing anything."""
    try:
        assert lib.grpo_set_tile_mode(-1) == 0
        assert [lib.grpo_get_role_tile_mode(r) for r in range(4)] == [0, 0, 2, 2]
        assert lib.grpo_get_tile_mode() == -1
        assert lib.grpo_set_role_tile_mode(1, 1) == 0
        assert [lib.grpo_get_role_tile_mode(r) for r in range(4)] == [0, 1, 2, 2]
        for role, mode in ((-1, 0), (4, 0), (0, -2), (1, 3), (2, 3), (3, 4)):
            assert lib.grpo_set_role_tile_mode(role, mode) == -1
        assert [lib.grpo_get_role_tile_mode(r) for r in range(4)] == [0, 1, 2, 2]
        assert lib.grpo_get_role_tile_mode(4) == -1 and lib.grpo_get_role_tile_mode(-1) == -1
        assert lib.grpo_set_role_tile_mode(1, -1) == 0
        assert [lib.grpo_get_role_tile_mode(r) for r in range(4)] == [0, 0, 2, 2]
        assert lib.grpo_set_tile_mode(0) == 0 and lib.grpo_get_tile_mode() == 0
        assert lib.grpo_set_role_tile_mode(3, -1) == 0
        assert [lib.grpo_get_role_tile_mode(r) for r in range(4)] == [0, 0, 0, 2]
        assert lib.grpo_get_tile_mode() == -1
        assert lib.grpo_set_role_tile_mode(2, 1) == 0 and lib.grpo_set_role_tile_mode(3, 1) == 0
        assert [lib.grpo_get_role_tile_mode(r) for r in range(4)] == [0, 0, 1, 1]
    finally:
        lib.grpo_set_tile_mode(-1)


def test_python_constants_match_the_header():
    """The binding's copies of the header's constants: the static scratch size and the progress
    window's default, read from include/grpo.h as text."""
    import re
    text = open(G.HEADER_PATH).read()
    m = re.search(r"#define GRPO_STATIC_SCRATCH_BYTES \((\d+)u \* (\d+)u \* (\d+)u\)", text)
    assert m and int(m[1]) * int(m[2]) * int(m[3]) == G.STATIC_SCRATCH_BYTES
    check = int(re.search(r"GRPO_GEMM_WINDOW_DEFAULT_CHECK = (-?\d+)", text)[1])
    lag = int(re.search(r"GRPO_GEMM_WINDOW_DEFAULT_LAG = (\d+)", text)[1])
    assert (check, lag) == G.GEMM_WINDOW_DEFAULT
