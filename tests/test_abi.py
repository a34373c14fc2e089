"""CPU-side checks of the C ABI: the library builds for sm_103a, loads, exports
every function include/molt.h declares, and rejects bad arguments on the host
before touching a device."""
import ctypes

import pytest

import paper_2607_21653_gb300 as molt


@pytest.fixture(scope="module")
def lib():
    molt.build()
    return molt.load()


def test_exports_every_header_function(lib):
    names = molt.header_functions()
    assert "molt_policy_loss_fwd_bwd" in names and "molt_group_advantages" in names
    for n in names:
        assert hasattr(lib, n), n


def test_status_strings(lib):
    for code in molt.STATUS:
        s = lib.molt_status_string(code).decode()
        assert s and s != "unknown status"
    assert lib.molt_version() >= 1


FAKE = 0x1000  # never dereferenced: every call below fails validation first


def test_rejects_unsupported_hidden(lib):
    st = lib.molt_token_logprobs_fwd(FAKE, FAKE, FAKE, None, 16, 100, 32, FAKE, None, None, 0, None)
    assert molt.STATUS[st] == "MOLT_ERR_UNSUPPORTED_SHAPE"
    assert "multiple of 64" in lib.molt_last_error().decode()


def test_launch_counter_unchanged_by_rejected_calls(lib):
    """molt_kernel_launches counts kernels actually enqueued: a call that
    fails validation enqueues none."""
    n0 = lib.molt_kernel_launches()
    st = lib.molt_token_logprobs_fwd(FAKE, FAKE, FAKE, None, 16, 100, 32, FAKE, None, None, 0, None)
    assert molt.STATUS[st] == "MOLT_ERR_UNSUPPORTED_SHAPE"
    assert lib.molt_kernel_launches() == n0


def test_rejects_null_and_misaligned(lib):
    st = lib.molt_token_logprobs_fwd(None, FAKE, FAKE, None, 16, 64, 32, FAKE, None, None, 0, None)
    assert molt.STATUS[st] == "MOLT_ERR_INVALID_ARG"
    st = lib.molt_token_logprobs_fwd(FAKE + 2, FAKE, FAKE, None, 16, 64, 32, FAKE, None, None, 0, None)
    assert molt.STATUS[st] == "MOLT_ERR_INVALID_ARG"
    st = lib.molt_mask_count(FAKE + 1, 64, FAKE, None)
    assert molt.STATUS[st] == "MOLT_ERR_INVALID_ARG"


def test_rejects_bad_clip_and_sizes(lib):
    args = [FAKE] * 6 + [16, 64, 32, 1.5, 0.2, 0.0] + [FAKE, FAKE, FAKE, 0, None, None, None, None, None, 0, None]
    st = lib.molt_policy_loss_fwd_bwd(*args)
    assert molt.STATUS[st] == "MOLT_ERR_INVALID_ARG"
    args[9] = 0.2
    args[11] = float("nan")
    assert molt.STATUS[lib.molt_policy_loss_fwd_bwd(*args)] == "MOLT_ERR_INVALID_ARG"
    args[11] = 0.0
    args[6] = -1
    assert molt.STATUS[lib.molt_policy_loss_fwd_bwd(*args)] == "MOLT_ERR_INVALID_ARG"
    assert molt.STATUS[lib.molt_group_advantages(FAKE, FAKE, -3, 1e-6, FAKE, None)] == "MOLT_ERR_INVALID_ARG"
    assert molt.STATUS[lib.molt_group_advantages(FAKE, FAKE, 4, -1.0, FAKE, None)] == "MOLT_ERR_INVALID_ARG"


def test_empty_inputs_are_noops(lib):
    assert lib.molt_group_advantages(None, None, 0, 1e-6, None, None) == 0
    assert lib.molt_broadcast_advantages(None, None, 0, 0, None, None) == 0
    assert lib.molt_token_logprobs_fwd(FAKE, FAKE, FAKE, None, 0, 64, 32, FAKE, None, None, 0, None) == 0


def test_workspace_sizes_grow_with_problem(lib):
    a = molt.token_logprobs_workspace_bytes(1000, 256, 4096)
    b = molt.policy_loss_workspace_bytes(1000, 256, 4096)
    assert 0 < a < b
    assert molt.policy_loss_workspace_bytes(1000, 100, 4096) == 0   # unsupported H
    # dhidden fp32 accumulator + packed bf16 copy of the hidden rows dominate
    assert b >= 1024 * 256 * 6


def test_rejects_bad_loss_options(lib):
    opts = molt.LossOptions(0.1, 0.0, None, None, 0.0, 0.0)      # KL without ref_logp
    args = [FAKE] * 6 + [16, 64, 32, 0.2, 0.2, 0.0, ctypes.byref(opts)] + [FAKE, FAKE, FAKE, 0, None, None, None,
                                                                          None, None, 0, None]
    assert molt.STATUS[lib.molt_policy_loss_fwd_bwd_ex(*args)] == "MOLT_ERR_INVALID_ARG"
    assert "ref_logp" in lib.molt_last_error().decode()
    opts = molt.LossOptions(0.0, 0.0, None, FAKE, 2.0, 1.0)      # empty gate band
    args[12] = ctypes.byref(opts)
    assert molt.STATUS[lib.molt_policy_loss_fwd_bwd_ex(*args)] == "MOLT_ERR_INVALID_ARG"
    opts = molt.LossOptions(-1.0, 0.0, FAKE, None, 0.0, 0.0)     # negative KL weight
    args[12] = ctypes.byref(opts)
    assert molt.STATUS[lib.molt_policy_loss_fwd_bwd_ex(*args)] == "MOLT_ERR_INVALID_ARG"


def test_workspace_query_with_options(lib):
    plain = lib.molt_policy_loss_workspace_bytes(1000, 512, 5000)
    assert plain > 0
    assert lib.molt_policy_loss_workspace_bytes_ex(1000, 512, 5000, None) == plain
    det = molt.LossOptions(0.0, 0.0, None, None, 0.0, 0.0, 1)
    assert lib.molt_policy_loss_workspace_bytes_ex(1000, 512, 5000, ctypes.byref(det)) >= plain
    assert lib.molt_policy_loss_workspace_bytes_ex(1000, 192, 5000, ctypes.byref(det)) == 0


def test_header_compiles_as_c(tmp_path):
    """include/molt.h is a C header: it compiles with a C11 compiler and -pedantic."""
    import shutil
    import subprocess
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no C compiler")
    src = tmp_path / "use_header.c"
    src.write_text('#include "molt.h"\nint main(void) { molt_loss_options o = {0}; (void)o; '
                   'return (int)(sizeof(molt_stats) + sizeof(molt_stats_ex)); }\n')
    import os
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    r = subprocess.run([gcc, "-std=c11", "-Wall", "-Wextra", "-pedantic", "-Werror", "-fsyntax-only",
                        "-I", os.path.join(root, "include"), "-I", "/usr/local/cuda/include", str(src)],
                       capture_output=True, text=True)
    assert r.returncode == 0, r.stderr


def test_binding_layouts_match_the_header(tmp_path):
    """The binding's ctypes mirror of molt_loss_options and its copy of
    MOLT_NOALLOC_MAX_TOKENS agree with the header as a C compiler reads it."""
    import os
    import shutil
    import subprocess
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no C compiler")
    src = tmp_path / "layout.c"
    src.write_text('#include <stdio.h>\n#include <stddef.h>\n#include "molt.h"\nint main(void) {\n'
                   '  printf("%zu %zu %zu %zu %zu %zu %zu %zu %zu %d\\n", sizeof(molt_loss_options),\n'
                   '    offsetof(molt_loss_options, kl_coef), offsetof(molt_loss_options, entropy_coef),\n'
                   '    offsetof(molt_loss_options, ref_logp), offsetof(molt_loss_options, seq_of_token),\n'
                   '    offsetof(molt_loss_options, gate_lo), offsetof(molt_loss_options, gate_hi),\n'
                   '    offsetof(molt_loss_options, deterministic), offsetof(molt_loss_options, det_clusters),\n'
                   '    (int)MOLT_NOALLOC_MAX_TOKENS);\n  return 0;\n}\n')
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    exe = tmp_path / "layout"
    r = subprocess.run([gcc, "-std=c11", "-I", os.path.join(root, "include"), "-I", "/usr/local/cuda/include",
                        str(src), "-o", str(exe)], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    vals = [int(v) for v in subprocess.run([str(exe)], capture_output=True, text=True).stdout.split()]
    L = molt.LossOptions
    names = ["kl_coef", "entropy_coef", "ref_logp", "seq_of_token", "gate_lo", "gate_hi", "deterministic",
             "det_clusters"]
    assert vals[0] == ctypes.sizeof(L)
    assert vals[1:9] == [getattr(L, n).offset for n in names]
    assert vals[9] == molt.NOALLOC_MAX_TOKENS
