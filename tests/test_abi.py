"""The C-ABI library builds, loads, and exports every function include/alr.h declares.

No kernel is launched here (these run without a GPU)."""

import ctypes
import json
import os
import re
import subprocess
import sys

import pytest

from paper_2609_38795_gb300 import alr, build_lib

HEADER = os.path.join(build_lib.ROOT, "include", "alr.h")


def _declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(alr_[a-z0-9_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def libalr():
    build_lib.build()
    return ctypes.CDLL(build_lib.LIB)


def test_header_declares_the_boundary():
    names = _declared()
    for need in ("alr_gather_ira_blocks", "alr_slot_loss_fwd", "alr_slot_loss_bwd",
                 "alr_accept_len", "alr_erase_weights"):
        assert need in names


def test_every_declared_symbol_is_exported(libalr):
    missing = [n for n in _declared() if not hasattr(libalr, n)]
    assert not missing, missing


def test_binding_covers_the_header():
    assert sorted(alr.SIGNATURES) == _declared()


def test_struct_layouts_match_the_header():
    # alr_params: int64 N, five int32, two floats -> 8 + 20 + 8 = 36, padded to 40
    assert ctypes.sizeof(alr.AlrParams) == 40
    assert alr.AlrParams.lam.offset == 28 and alr.AlrParams.gamma.offset == 32
    assert ctypes.sizeof(alr.AlrFwdOutputs) == 13 * 8          # 13 pointers
    assert ctypes.sizeof(alr.AlrTopkFwdOutputs) == 9 * 8


def test_argument_errors_are_reported_without_a_launch(libalr):
    lib = alr.lib()
    assert lib.alr_version().decode().startswith("libalr")
    bad = alr.make_params(N=30, d=64, V=128, B=16)          # N not a multiple of B
    assert lib.alr_fwd_workspace_size(ctypes.byref(bad)) == 0
    out = alr.AlrFwdOutputs()
    rc = lib.alr_slot_loss_fwd(ctypes.byref(bad), None, None, None, None, None,
                               ctypes.byref(out), None, 0, None)
    assert rc == alr.ALR_ERR_INVALID_ARG
    assert "multiple of B" in lib.alr_last_error().decode()
    bad_b = alr.make_params(N=66, d=64, V=128, B=33)
    rc = lib.alr_slot_loss_bwd(ctypes.byref(bad_b), *([None] * 10), 0, None)
    assert rc == alr.ALR_ERR_INVALID_ARG
    rc = lib.alr_accept_len(None, None, None, 4, 0, None, None, None)
    assert rc == alr.ALR_ERR_INVALID_ARG
    rc = lib.alr_erase_weights(None, None, None, None, 4, 8, 0.0, 0, None, None)
    assert rc == alr.ALR_ERR_INVALID_ARG
    rc = lib.alr_gather_ira_blocks(None, 1, 8, 12, alr.ALR_BF16, None, None, None, 2, 4, None,
                                   None, None)
    assert rc == alr.ALR_ERR_INVALID_ARG                   # 12 * 2 bytes is not a multiple of 16
    # the backward passes from kept logits validate dH's arguments before the gradient kernel
    # would overwrite z_d: a missing dHd is reported before anything else is looked at
    good = alr.make_params(N=32, d=64, V=128, B=16)
    fake = ctypes.c_void_p(1 << 20)                        # never dereferenced on this path
    rc = lib.alr_slot_loss_bwd_from_logits(ctypes.byref(good), fake, fake, fake, fake, fake,
                                           fake, fake, fake, fake, fake, fake, None, None, None,
                                           0, None)
    assert rc == alr.ALR_ERR_INVALID_ARG
    assert "dHd" in lib.alr_last_error().decode()
    rc = lib.alr_topk_loss_bwd_from_logits(ctypes.byref(good), fake, fake, fake, fake, fake,
                                           fake, fake, fake, fake, fake, fake, fake, None, None,
                                           None, 0, None)
    assert rc == alr.ALR_ERR_INVALID_ARG
    assert "dHd" in lib.alr_last_error().decode()
    # kept fp16 logits of bf16 inputs are unreadable without their group references
    rc = lib.alr_logit_grad_from_logits(ctypes.byref(good), fake, fake, None, fake, fake, fake,
                                        fake, fake, fake, None)
    assert rc == alr.ALR_ERR_INVALID_ARG
    assert "Zd_ref" in lib.alr_last_error().decode()
    rc = lib.alr_topk_logit_grad_from_logits(ctypes.byref(good), fake, None, fake, fake, fake,
                                             fake, fake, fake, fake, fake, None)
    assert rc == alr.ALR_ERR_INVALID_ARG
    assert "Zd_ref" in lib.alr_last_error().decode()
    rc = lib.alr_loss_from_sums(None, fake, ctypes.c_float(1.0), fake, None)
    assert rc == alr.ALR_ERR_INVALID_ARG
    # group references: one per 16 logits of a row (the last group may be partial)
    assert [lib.alr_kept_ref_groups(v) for v in (8, 256, 264, 151936)] == [1, 16, 17, 9496]


def test_binding_refuses_host_and_malformed_tensors_before_any_call(libalr):
    """The C ABI takes bare device pointers and cannot check a buffer behind one, so the binding
    does: host tensors, non-tensors and (on any machine) the wrong buffers raise before the
    library sees a pointer."""
    import torch
    N, d, V, B = 32, 64, 128, 16
    params = alr.make_params(N, d, V, B, torch.bfloat16)
    host = torch.zeros(N * d, dtype=torch.bfloat16)
    with pytest.raises(ValueError, match="CUDA device"):
        alr.alr_gemm(host, host, torch.zeros(N * N), N, N, d)
    with pytest.raises(ValueError, match="CUDA device"):
        alr.alr_slot_loss_fwd_noalloc(params, host, host, torch.zeros(d * V, dtype=torch.bfloat16),
                                      {})
    with pytest.raises(ValueError, match="whole number of anchors"):
        alr.alr_accept_len(torch.zeros(20, dtype=torch.int32), torch.zeros(20, dtype=torch.int32),
                           16, torch.zeros(1, dtype=torch.int32))
    with pytest.raises(TypeError, match="torch.Tensor"):
        alr._ptr(host.float().numpy(), "Hd")
    assert alr._ptr(None, "row_mask") is None


def test_last_error_is_per_host_thread(libalr):
    """alr_last_error() belongs to the calling thread: two threads that fail different calls at
    the same time each read back their own message."""
    import threading
    lib = alr.lib()
    barrier = threading.Barrier(2)
    seen = {}

    def fail_with(tag, params):
        out = alr.AlrFwdOutputs()
        for _ in range(200):
            barrier.wait()
            rc = lib.alr_slot_loss_fwd(ctypes.byref(params), None, None, None, None, None,
                                       ctypes.byref(out), None, 0, None)
            barrier.wait()
            seen.setdefault(tag, set()).add((rc, lib.alr_last_error().decode()))

    t1 = threading.Thread(target=fail_with, args=("B", alr.make_params(N=30, d=64, V=128, B=16)))
    t2 = threading.Thread(target=fail_with, args=("d", alr.make_params(N=32, d=12, V=128, B=16)))
    t1.start(), t2.start()
    t1.join(), t2.join()
    assert len(seen["B"]) == 1 and len(seen["d"]) == 1
    (rc_b, msg_b), = seen["B"]
    (rc_d, msg_d), = seen["d"]
    assert rc_b == rc_d == alr.ALR_ERR_INVALID_ARG
    assert "multiple of B" in msg_b and "d = 12" in msg_d


def test_error_paths_reject_before_any_device_work(libalr):
    """Table of invalid calls through the raw C ABI.  The pointers are fakes that must never be
    dereferenced: every case is refused by argument validation, with its own status and
    message, before the library looks for a device (on a machine without one, a case that
    slipped past validation would report the missing device instead and fail here)."""
    lib = alr.lib()
    A16, MIS = ctypes.c_void_p(0x10000), ctypes.c_void_p(0x10002)    # aligned / misaligned
    out = alr.AlrFwdOutputs(**{f: 0x20000 for f in alr._FWD_FIELDS})

    def fwd(params, hd=A16, ht=A16, w=A16, ws=A16, nbytes=1 << 30, tok=None):
        return lib.alr_slot_loss_fwd(ctypes.byref(params), hd, ht, w, None, tok,
                                     ctypes.byref(out), ws, nbytes, None)

    P = alr.make_params
    bad = alr.AlrParams(N=32, d=64, V=128, B=16, dtype=7, mode=0, lam=1.0, gamma=2.0)
    cases = [
        ("dtype", lambda: fwd(bad), alr.ALR_ERR_UNSUPPORTED, "dtype 7"),
        ("mode", lambda: fwd(P(32, 64, 128, 16, mode=5)), alr.ALR_ERR_UNSUPPORTED, "mode 5"),
        ("B too large", lambda: fwd(P(64, 64, 128, 64)), alr.ALR_ERR_INVALID_ARG, "B = 64"),
        ("N too large", lambda: fwd(P((1 << 31), 64, 128, 16)), alr.ALR_ERR_INVALID_ARG, "too large"),
        ("d not a multiple of 8", lambda: fwd(P(32, 60, 128, 16)), alr.ALR_ERR_INVALID_ARG, "d = 60"),
        ("V too small", lambda: fwd(P(32, 64, 0, 16)), alr.ALR_ERR_INVALID_ARG, "V = 0"),
        ("gamma", lambda: fwd(P(32, 64, 128, 16, gamma=0.0)), alr.ALR_ERR_INVALID_ARG, "gamma"),
        ("lambda NaN", lambda: fwd(P(32, 64, 128, 16, lam=float("nan"))), alr.ALR_ERR_INVALID_ARG,
         "lambda"),
        ("NULL head", lambda: fwd(P(32, 64, 128, 16), w=None), alr.ALR_ERR_INVALID_ARG, "non-NULL"),
        ("misaligned Ht", lambda: fwd(P(32, 64, 128, 16), ht=MIS), alr.ALR_ERR_INVALID_ARG,
         "16-byte aligned"),
        ("erase without tokens", lambda: fwd(P(32, 64, 128, 16, mode=1)), alr.ALR_ERR_INVALID_ARG,
         "corpus_tok"),
        ("gemm Nc % 4", lambda: lib.alr_gemm(alr.ALR_BF16, 0, 0, 0, A16, A16, A16, 8, 6, 64, None),
         alr.ALR_ERR_INVALID_ARG, "Nc % 4"),
        ("gemm tf32 MN-major", lambda: lib.alr_gemm(alr.ALR_F32, 1, 0, 0, A16, A16, A16, 8, 8, 8,
                                                    None), alr.ALR_ERR_UNSUPPORTED, "K-major"),
        ("gemm misaligned C", lambda: lib.alr_gemm(alr.ALR_BF16, 0, 0, 0, A16, A16, MIS, 8, 8, 64,
                                                   None), alr.ALR_ERR_INVALID_ARG, "aligned"),
        ("gather row bytes", lambda: lib.alr_gather_ira_blocks(A16, 1, 8, 12, alr.ALR_BF16, A16, A16,
                                                               None, 4, 16, A16, None, None),
         alr.ALR_ERR_INVALID_ARG, "16 bytes"),
        ("gather NULL out", lambda: lib.alr_gather_ira_blocks(A16, 1, 8, 64, alr.ALR_BF16, A16, A16,
                                                              None, 4, 16, None, None, None),
         alr.ALR_ERR_INVALID_ARG, "non-NULL"),
        ("accept B", lambda: lib.alr_accept_len(A16, A16, None, 4, 33, A16, None, None),
         alr.ALR_ERR_INVALID_ARG, "B=33"),
        ("erase gamma", lambda: lib.alr_erase_weights(A16, None, None, None, 4, 16, 0.0, 0, A16,
                                                      None), alr.ALR_ERR_INVALID_ARG, "gamma"),
        ("hard gate inputs", lambda: lib.alr_erase_weights(None, None, None, None, 4, 16, 2.0, 1,
                                                           A16, None),
         alr.ALR_ERR_INVALID_ARG, "corpus_tok and argmax_t"),
        ("ira K", lambda: lib.alr_ira_blocks(2, 1, 8, A16, A16, A16, None, None, A16, A16, A16,
                                             None, None, None), alr.ALR_ERR_INVALID_ARG, "K=1"),
    ]
    for name, call, code, text in cases:
        rc = call()
        msg = lib.alr_last_error().decode()
        assert rc == code, (name, rc, msg)
        assert text in msg, (name, msg)


_FORMS_CHILD = r"""
import ctypes, json, sys
h = ctypes.CDLL(sys.argv[1])
h.alr_cluster_forms_error.restype = ctypes.c_char_p
g, l = ctypes.c_int32(), ctypes.c_int32()
assert h.alr_kernel_forms(ctypes.byref(g), ctypes.byref(l)) == 0
why = h.alr_cluster_forms_error().decode()
maps = open("/proc/self/maps").read()
print(json.dumps({"forms": [g.value, l.value], "why": why,
                  "cluster_mapped": "libalr_cluster.so" in maps}))
"""


def _forms_in_child(env_over):
    env = {k: v for k, v in os.environ.items()
           if k not in ("WORLD_SIZE", "ALR_GEMM_FORM", "ALR_LOSS_FORM")}
    env.update(env_over)
    r = subprocess.run([sys.executable, "-c", _FORMS_CHILD, build_lib.LIB], env=env,
                       capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stderr
    out = json.loads(r.stdout.strip().splitlines()[-1])
    g, l = out["forms"]
    return (alr.GEMM_FORMS[g], alr.LOSS_FORMS[l]), out["why"], out["cluster_mapped"]


def test_multi_rank_processes_never_load_the_cluster_forms(libalr):
    """The kernel forms with TMA multicast loads (and the CTA-pair GEMM) live in
    libalr_cluster.so.  A single process loads it and keeps its choice of form; one rank of a
    multi-rank launch (WORLD_SIZE > 1) never maps it and runs every form on single CTAs,
    whatever the environment asks.  Each case is a fresh process: the library decides once."""
    for world, gemm_env, loss_env, want in (
            (None, None, None, ("mcast", "single")),
            ("1", "mcast4", "mcast", ("mcast4", "mcast")),
            (None, "pair", None, ("pair", "single")),
            (None, "single", "single", ("single", "single")),
            ("2", None, None, ("single", "single")),
            ("8", "mcast", "mcast", ("single", "single")),
            ("4", "mcast4", None, ("single", "single")),
            ("2", "pair", None, ("single", "single"))):
        env = {k: v for k, v in (("WORLD_SIZE", world), ("ALR_GEMM_FORM", gemm_env),
                                 ("ALR_LOSS_FORM", loss_env)) if v is not None}
        forms, why, mapped = _forms_in_child(env)
        multi = world is not None and int(world) > 1
        assert forms == want, (env, forms, why)
        assert mapped == (not multi), (env, why)
        assert (why == "") == (not multi) and (not multi or "rank" in why), (env, why)


def test_cluster_forms_are_built_apart():
    """No source of libalr.so issues a multicast copy or commit, or a 2-SM product; the cluster
    library's sources do, and it exports the loader's entry points."""
    pat = re.compile(r"multicast::cluster|cta_group::2")
    for d in (build_lib.CSRC, build_lib.INCLUDE):
        for f in os.listdir(d):
            with open(os.path.join(d, f)) as fh:
                code = re.sub(r"/\*.*?\*/", "", fh.read(), flags=re.S)   # PTX, not comments
            code = "\n".join(line.split("//")[0] for line in code.splitlines())
            assert not pat.search(code), f
    cl = "".join(open(os.path.join(build_lib.CSRC_CLUSTER, f)).read()
                 for f in os.listdir(build_lib.CSRC_CLUSTER))
    assert pat.search(cl)
    h = ctypes.CDLL(build_lib.LIB_CLUSTER)
    for name in ("alr_cluster_args_size", "alr_cluster_launch_loss", "alr_cluster_launch_gemm",
                 "alr_cluster_gemm_max_clusters", "alr_cluster_launch_pair_gemm",
                 "alr_cluster_pair_gemm_max_pairs"):
        assert hasattr(h, name), name
