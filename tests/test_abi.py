"""The C-ABI library loads, exports every symbol include/gasloc.h declares, and
rejects bad arguments on the host (no device work; runs without a GPU)."""
import ctypes
import os
import re

import pytest

import paper_2606_11081_gb300 as g
from paper_2606_11081_gb300 import build as gbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "gasloc.h")


@pytest.fixture(scope="module")
def lib():
    gbuild.build()
    return g.load_library()


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    names = re.findall(r"\b(gasloc_[a-z_0-9]+)\s*\(", src)
    return sorted(set(n for n in names if not n.endswith("_fn")))


def test_header_declares_the_core_calls():
    names = declared_functions()
    for core in ("gasloc_init", "gasloc_local_steps", "gasloc_gossip_round", "gasloc_consensus_error"):
        assert core in names


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 25
    for n in names:
        assert hasattr(lib, n), n
    # and the binding wraps exactly those names
    assert set(names) == set(g.SIGNATURES)


def test_default_hparams(lib):
    hp = g.gasloc_default_hparams()
    assert hp.lr == 3e-4 and hp.beta1 == 0.9 and hp.beta2 == 0.95 and hp.weight_decay == 0.1
    assert hp.outer_mode == g.OUTER["nesterov"] and hp.edge_prob == 1.0


@pytest.mark.parametrize("n,p,topo", [(0, 10, "ring"), (33, 10, "ring"), (4, 0, "ring"),
                                      (4, -5, "ring"), (4, 2 ** 31, "ring"), (4, 10, "star"),
                                      (1, 10, "matching"), (1, 10, "2peer"), (8, 10, "torus:3x3"),
                                      (8, 10, "torus:2x"), (8, 10, "torus:0x8")])
def test_init_rejects(lib, n, p, topo):
    with pytest.raises(g.GaslocError) as e:
        g.gasloc_init(n, p, topo, 1)
    assert e.value.code == g.EINVAL


def test_hparams_validation(lib):
    c = g.gasloc_init(4, 100, "ring", 1)
    try:
        for bad in [dict(lr=-1.0), dict(beta1=1.0), dict(beta2=-0.1), dict(eps=0.0),
                    dict(edge_prob=1.5), dict(outer_lr=-0.1), dict(gamma=float("nan")),
                    dict(lr_total_steps=-1), dict(lr_total_steps=2 ** 24 + 1),
                    dict(lr_total_steps=10, lr_warmup_frac=1.5),
                    dict(lr_total_steps=10, lr_warmup_start=-0.1),
                    dict(lr_total_steps=10, lr_final_frac=float("nan"))]:
            with pytest.raises(g.GaslocError) as e:
                g.gasloc_set_hparams(c, g.make_hparams(**bad))
            assert e.value.code == g.EINVAL
        hp = g.make_hparams()
        hp.outer_mode = 9
        with pytest.raises(g.GaslocError):
            g.gasloc_set_hparams(c, hp)
        g.gasloc_set_hparams(c, g.make_hparams(lr=1e-3, outer="sgd"))
        assert g.gasloc_get_hparams(c).lr == 1e-3
    finally:
        g.gasloc_destroy(c)


def test_layout_validation(lib):
    c = g.gasloc_init(2, 100, "ring", 1)
    try:
        with pytest.raises(g.GaslocError):
            g.gasloc_set_layout(c, [50, 49])
        with pytest.raises(g.GaslocError):
            g.gasloc_set_layout(c, [100, 0])
        g.gasloc_set_layout(c, [37, 63])
    finally:
        g.gasloc_destroy(c)


def test_calls_before_start_are_state_errors(lib):
    c = g.gasloc_init(2, 100, "ring", 1)
    try:
        host = ctypes.c_double()
        for fn in (lambda: g.gasloc_local_steps(c, 1), lambda: g.gasloc_gossip_round(c),
                   lambda: g.gasloc_consensus_error(c), lambda: g.gasloc_buffer(c, "x"),
                   lambda: g.gasloc_consensus_error_async(c, ctypes.addressof(host)),
                   lambda: g.gasloc_synchronize(c)):
            with pytest.raises(g.GaslocError) as e:
                fn()
            assert e.value.code == g.ESTATE
        with pytest.raises(g.GaslocError):
            g.gasloc_set_local_steps(c, [1, 2000])
        with pytest.raises(g.GaslocError):
            g.gasloc_draw_local_steps(c, 0)
    finally:
        g.gasloc_destroy(c)


def test_local_step_draw_matches_oracle(lib, orc32):
    # H_i is drawn on the host from the seed: bit-identical to the oracle's draw
    c = g.gasloc_init(32, 100, "exp", 0x6A510C)
    try:
        g.gasloc_draw_local_steps(c, 8)
        H = g.gasloc_get_local_steps(c, 32)
    finally:
        g.gasloc_destroy(c)
    assert H.tolist() == orc32.draw_local_steps(0x6A510C, 32, 8).tolist()


def test_start_without_gpu_fails_cleanly(lib):
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    c = g.gasloc_init(2, 100, "ring", 1)
    try:
        with pytest.raises(g.GaslocError) as e:
            g.gasloc_start(c)
        assert e.value.code in (g.ECUDA, g.ENOMEM)
    finally:
        g.gasloc_destroy(c)


def test_range_validation(lib):
    ctx = g.gasloc_init(4, 1000, "ring", 1)
    try:
        assert g.gasloc_get_range(ctx) == (0, 1000, 1000)
        for a, b in [(-1, 10), (5, 5), (10, 5), (0, 1001), (1000, 1001)]:
            with pytest.raises(g.GaslocError) as e:
                g.gasloc_set_range(ctx, a, b)
            assert e.value.code == g.EINVAL, (a, b)
        g.gasloc_set_range(ctx, 250, 999)
        assert g.gasloc_get_range(ctx) == (250, 999, 1000)
        # the layout still describes the whole problem
        with pytest.raises(g.GaslocError) as e:
            g.gasloc_set_layout(ctx, [500, 249])
        assert e.value.code == g.EINVAL
        g.gasloc_set_layout(ctx, [500, 500])
    finally:
        g.gasloc_destroy(ctx)
