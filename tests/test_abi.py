"""The C ABI library loads without a GPU, exports every function that
include/doloss.h declares, and rejects invalid arguments on the host before
touching the device."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "doloss.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(do_[a-z_0-9]+)\s*\(", text)))


@pytest.fixture(scope="module")
def dl():
    from paper_2609_32398_gb300 import build, doloss

    build.build()
    return doloss


def test_header_declares_the_path(dl):
    names = declared_functions()
    for n in ["do_signatures", "do_pairwise_hamming", "do_loss_fwd_bwd", "do_forward_backward"]:
        assert n in names


def test_every_declared_symbol_is_exported(dl):
    lib = ctypes.CDLL(dl.LIB_PATH)
    for name in declared_functions():
        assert hasattr(lib, name), name
        assert name in dl.EXPORTS, f"binding lacks {name}"


def test_status_strings(dl):
    for code in range(7):
        assert dl.status_string(code)
    assert dl.status_string(99) == "unknown status"


def test_workspace_size_host_logic(dl):
    assert dl.workspace_size(0, 8, 2, 1) == 0
    assert dl.workspace_size(10, 8, 9, 1) == 0
    assert dl.workspace_size(10, 2000, 2, 1) == 0
    small = dl.workspace_size(1024, 8, 2, 1)
    big = dl.workspace_size(1 << 20, 256, 8, 48)
    assert 256 < small < big
    assert dl.host_buffer_size(1024, 8, 2, 1) > 2 * 4 * 1024 * 8


def test_invalid_arguments_are_rejected_before_launch(dl):
    lib = dl.lib()
    fake = ctypes.c_void_p(0x10000)           # never dereferenced: validation fails first
    INV, UNS, WS = 1, 2, 6
    assert lib.do_signatures(None, 64, 8, 2, 1, fake, fake, None) == INV
    assert lib.do_signatures(fake, 64, 8, 9, 1, fake, fake, None) == INV     # k > E
    assert lib.do_signatures(fake, 0, 8, 2, 1, fake, fake, None) == INV      # T = 0
    assert lib.do_signatures(fake, 64, 2048, 2, 1, fake, fake, None) == UNS  # E > 1024
    assert lib.do_signatures(fake, 1 << 30, 8, 2, 1, fake, fake, None) == UNS  # (E-1)T >= 2^31
    odd = ctypes.c_void_p(0x10002)
    assert lib.do_signatures(odd, 64, 8, 2, 1, fake, fake, None) == INV      # misaligned
    assert lib.do_pairwise_hamming(fake, 64, 8, 1, None, None) == INV
    assert lib.do_loss_fwd_bwd(fake, fake, fake, 64, 8, 2, 1, 7, 1.0, 1.0, fake, None, None,
                               fake, 1 << 20, None) == INV                    # bad gate
    assert lib.do_loss_fwd_bwd(fake, fake, fake, 64, 8, 2, 1, 0, 1.0, 1.0, fake, None, None,
                               fake, 8, None) == WS                           # small workspace
    assert lib.do_forward_backward(fake, 64, 8, 2, 1, 0, 1.0, fake, fake, fake, fake, None, None,
                                   None, 0, None) == WS
    assert lib.do_forward_backward_host(None, 64, 8, 2, 1, 0, 1.0, fake, None, None, None, fake,
                                        1 << 30, None) == INV
    assert lib.do_selftest_wait_limit(None, None) == WS


def test_routing_entry_points_validate_on_the_host(dl):
    lib = dl.lib()
    fake = ctypes.c_void_p(0x10000)
    odd = ctypes.c_void_p(0x10002)
    INV, UNS, WS = 1, 2, 6
    big_ws = 1 << 30
    assert dl.lib().do_routing_workspace_size(0, 8, 2, 1) == 0
    # status word + padding, the signatures [L][E][W], and per expert and
    # problem one dispatch chunk base (W = 32 words is one chunk) and a total,
    # each region rounded to 256 B
    assert dl.lib().do_routing_workspace_size(1000, 8, 2, 3) == 256 + 4 * 3 * 8 * 32 + 256
    assert lib.do_routing(fake, 64, 8, 2, 1, 0, None, fake, fake, None, None, None, fake, big_ws,
                          None) == INV                                        # no expert_ids
    assert lib.do_routing(fake, 64, 8, 2, 1, 0, fake, None, fake, None, None, None, fake, big_ws,
                          None) == INV                                        # no combine
    assert lib.do_routing(fake, 64, 8, 2, 1, 0, fake, fake, None, None, None, None, fake, big_ws,
                          None) == INV                                        # no counts
    assert lib.do_routing(fake, 64, 8, 2, 1, 2, fake, fake, fake, None, None, None, fake, big_ws,
                          None) == INV                                        # bad gate
    assert lib.do_routing(fake, 64, 8, 2, 1, 0, fake, fake, fake, odd, None, None, fake, big_ws,
                          None) == INV                                        # misaligned offsets
    assert lib.do_routing(fake, 64, 8, 2, 1, 0, fake, fake, fake, None, None, None, fake, 16,
                          None) == WS                                         # small workspace
    # (E - 1) T fits int32 but T k does not: dispatch rows are int32
    assert lib.do_routing(fake, (1 << 30) + 1, 2, 2, 1, 0, fake, fake, fake, None, None, None, fake,
                          big_ws, None) == UNS
    assert lib.do_forward_backward_routed(fake, 64, 8, 2, 1, 0, 1.0, fake, fake, fake, fake, None,
                                          None, None, fake, None, None, None, fake, big_ws,
                                          None) == INV                        # no expert_ids
    assert lib.do_forward_backward_routed(fake, 64, 8, 2, 1, 0, 1.0, fake, fake, fake, fake, None,
                                          None, fake, fake, None, None, None, fake, 8,
                                          None) == WS


def test_router_entry_point_validates_on_the_host(dl):
    lib = dl.lib()
    fake = ctypes.c_void_p(0x10000)
    INV, UNS = 1, 2
    big = 1 << 30
    args = lambda X, T, H, E, k: (X, fake, T, H, E, k, 1, 0, 1.0, fake, fake, fake, fake, fake,
                                  None, fake, fake, big, None)
    assert lib.do_router_forward_backward(*args(None, 1024, 256, 128, 8)) == INV
    assert lib.do_router_forward_backward(*args(fake, 1024, 0, 128, 8)) == INV    # H = 0
    assert lib.do_router_forward_backward(*args(fake, 1024, 256, 64, 8)) == UNS   # E != 128
    assert lib.do_router_forward_backward(*args(fake, 1024, 96, 128, 8)) == UNS   # H % 64
    assert lib.do_router_forward_backward(*args(fake, 1024, 256, 128, 3)) == UNS  # k


def test_router_backward_validates_on_the_host(dl):
    lib = dl.lib()
    fake = ctypes.c_void_p(0x10000)
    odd = ctypes.c_void_p(0x10004)
    INV, WS = 1, 6
    big = 1 << 34
    assert lib.do_router_backward_workspace_size(0, 128, 64, 1) == 0
    assert lib.do_router_backward_workspace_size(100, 128, 64, 1) >= 2 * 100 * 128
    assert lib.do_router_backward(None, fake, fake, 64, 64, 128, 1, fake, None, fake, big, None) == INV
    assert lib.do_router_backward(fake, fake, fake, 64, 64, 128, 1, None, None, fake, big, None) == INV
    assert lib.do_router_backward(odd, fake, fake, 64, 64, 128, 1, fake, None, fake, big, None) == INV
    assert lib.do_router_backward(fake, fake, fake, 64, 64, 128, 1, fake, None, fake, 64, None) == WS


def test_async_host_entry_validates_on_the_host(dl):
    lib = dl.lib()
    fake = ctypes.c_void_p(0x10000)
    INV, WS = 1, 6
    assert lib.do_forward_backward_host_async(fake, 64, 8, 2, 1, 0, 1.0, None, fake, 1 << 30,
                                              None) == INV
    assert lib.do_forward_backward_host_async(None, 64, 8, 2, 1, 0, 1.0, fake, fake, 1 << 30,
                                              None) == INV
    assert lib.do_forward_backward_host_async(fake, 64, 8, 2, 1, 0, 1.0, fake, fake, 64,
                                              None) == WS


def test_route_backward_validates_on_the_host(dl):
    lib = dl.lib()
    fake = ctypes.c_void_p(0x10000)
    odd = ctypes.c_void_p(0x10002)
    INV, UNS = 1, 2
    assert lib.do_route_backward(None, fake, fake, 64, 8, 2, 1, 0, 0, fake, None, None) == INV
    assert lib.do_route_backward(fake, None, fake, 64, 8, 2, 1, 0, 0, fake, None, None) == INV
    assert lib.do_route_backward(fake, fake, None, 64, 8, 2, 1, 0, 0, fake, None, None) == INV
    assert lib.do_route_backward(fake, fake, fake, 64, 8, 2, 1, 0, 0, None, None, None) == INV
    assert lib.do_route_backward(fake, fake, fake, 64, 8, 2, 1, 2, 0, fake, None, None) == INV  # gate
    assert lib.do_route_backward(fake, fake, fake, 64, 8, 2, 1, 0, 2, fake, None, None) == INV  # accumulate
    assert lib.do_route_backward(fake, fake, fake, 64, 8, 9, 1, 0, 0, fake, None, None) == INV  # k > E
    assert lib.do_route_backward(fake, odd, fake, 64, 8, 2, 1, 0, 0, fake, None, None) == INV
    assert lib.do_route_backward(fake, fake, fake, 64, 8, 2, 1, 0, 0, fake, odd, None) == INV
    assert lib.do_route_backward(fake, fake, fake, 64, 2048, 2, 1, 0, 0, fake, None, None) == UNS


def test_routed_halves_validate_on_the_host(dl):
    lib = dl.lib()
    fake = ctypes.c_void_p(0x10000)
    odd = ctypes.c_void_p(0x10002)
    INV, WS = 1, 6
    big = 1 << 30
    f = lib.do_routed_forward
    assert f(fake, 64, 8, 2, 1, 0, fake, fake, fake, None, None, fake, None, None, None, fake, big,
             None) == INV                                                # combine without ids
    assert f(fake, 64, 8, 2, 1, 0, fake, fake, None, None, fake, fake, None, None, None, fake, big,
             None) == INV                                                # no D
    assert f(fake, 64, 8, 2, 1, 3, fake, fake, fake, None, fake, fake, None, None, None, fake, big,
             None) == INV                                                # bad gate
    assert f(fake, 64, 8, 2, 1, 0, fake, fake, fake, odd, fake, fake, None, None, None, fake, big,
             None) == INV                                                # misaligned origin_do
    assert f(fake, 64, 8, 2, 1, 0, fake, fake, fake, None, fake, fake, None, None, None, fake, 64,
             None) == WS
    b = lib.do_routed_backward
    assert b(fake, 64, 8, 2, 1, 0, 1.0, 1.0, fake, fake, fake, None, fake, fake, fake, fake, big,
             None) == INV                                                # ids without gradient
    assert b(fake, 64, 8, 2, 1, 0, 1.0, 1.0, fake, fake, fake, fake, None, fake, fake, fake, big,
             None) == INV                                                # gradient without ids
    assert b(fake, 64, 8, 2, 1, 0, 1.0, float("nan"), fake, fake, fake, fake, fake, fake, fake, fake,
             big, None) == INV                                           # NaN grad_scale
    assert b(fake, 64, 8, 2, 1, 0, float("nan"), 1.0, fake, fake, fake, fake, fake, fake, fake, fake,
             big, None) == INV                                           # NaN d_scale
    assert b(fake, 64, 8, 2, 1, 0, 1.0, 1.0, fake, fake, fake, odd, fake, fake, fake, fake, big,
             None) == INV                                                # misaligned ids
    assert b(fake, 64, 8, 2, 1, 0, 1.0, 1.0, fake, fake, None, None, None, fake, fake, fake, big,
             None) == INV                                                # no D
    assert b(fake, 64, 8, 2, 1, 0, 1.0, 1.0, fake, fake, fake, fake, fake, fake, fake, fake, 64,
             None) == WS
    # steps 1-2 alone: routing outputs absent, but then no dispatch arrays either
    assert f(fake, 64, 8, 2, 1, 0, fake, fake, fake, None, None, None, fake, None, None, fake, big,
             None) == INV


def test_accumulate_distances_validates_on_the_host(dl):
    lib = dl.lib()
    fake = ctypes.c_void_p(0x10000)
    odd = ctypes.c_void_p(0x10002)
    assert lib.do_accumulate_distances(None, 8, 1, fake, None) == 1
    assert lib.do_accumulate_distances(fake, 8, 1, None, None) == 1
    assert lib.do_accumulate_distances(fake, 0, 1, fake, None) == 1
    assert lib.do_accumulate_distances(odd, 8, 1, fake, None) == 1
    assert lib.do_accumulate_distances(fake, 2048, 1, fake, None) == 2


def _ctype_code(decl):
    """The binding's argument code of one C parameter or return type."""
    d = " ".join(decl.replace("const ", "").split())
    if "*" in d:
        return "str" if d.startswith("char") else "p"
    base = d.split()[0]
    return {"int64_t": "i64", "int32_t": "i32", "float": "f32", "size_t": "sz", "do_status": "i32",
            "double": "f64"}[base]


def declared_signatures():
    text = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    out = {}
    for ret, name, params in re.findall(r"([A-Za-z_][\w \*]*?)\s*\b(do_[a-z_0-9]+)\s*\(([^)]*)\)\s*;",
                                        text):
        ret = ret.split()[-1] if "*" not in ret else ret
        args = [p.strip() for p in params.split(",") if p.strip() and p.strip() != "void"]
        # drop the parameter name: what precedes the last identifier is the type
        types = [re.sub(r"\b\w+\s*$", "", a).strip() or a for a in args]
        out[name] = ([_ctype_code(t) for t in types], _ctype_code(ret))
    return out


def test_binding_signatures_match_the_header(dl):
    """Every declared function's parameter kinds (pointer, int32, int64, float,
    size_t) and result kind, read from include/doloss.h, are those the ctypes
    binding declares, so that a changed signature cannot go unnoticed."""
    sigs = declared_signatures()
    assert set(sigs) == set(declared_functions())
    for name, (args, res) in sigs.items():
        want_args, want_res = dl.EXPORTS[name]
        assert args == want_args, (name, args, want_args)
        assert res == want_res, (name, res, want_res)
