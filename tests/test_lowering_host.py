"""The tiled lowering computes the plan's layer, checked on the host.

Plan creation lowers every layer to the tiled kernel's schedule and, before
accepting it, evaluates that schedule symbolically (shared sums, SEG
programs, operations, partial slots and their combination) into integer
coefficients of (plaintext, input) products and compares them with the
plan's own terms; a difference fails plan creation with
FIONA_ERR_INTERNAL.  These tests run that check, and the index checks before
it, on many random layers and every shape the lowering can be forced to, with
no GPU (validation-only contexts)."""
import numpy as np
import pytest

from paper_2609_35352_gb300 import build as B
from paper_2609_35352_gb300 import fiona as F
from paper_2609_35352_gb300 import workloads as W

SHAPES = [None, "2,16,0", "2,8,1", "1,16,1", "1,4,0", "2,8,1,-1,4", "1,8,0,3", "1,16,1,-1,16", "2,4,1,-1,8"]


@pytest.fixture(scope="module", autouse=True)
def built():
    B.build()


def random_layer(rng, big=False):
    """Random route mix: raw, constant raw, ternary with zeros; one to three
    reconstruction factors per output; shared sums from the plan compiler."""
    n_in = int(rng.integers(1, 200 if big else 40))
    n_out = int(rng.integers(1, 40 if big else 20))
    n_gamma = int(rng.integers(1, 4))
    p_raw, p_const, p_zero = rng.uniform(0, 0.6), rng.uniform(0, 0.3), rng.uniform(0, 0.2)
    r = np.zeros((n_out, n_in), F.ROUTE_DTYPE)
    n_raw = 0
    for j in range(n_out):
        for i in range(n_in):
            u = rng.random()
            if u < p_raw:
                kind = W.TERM_RAW_CONST if rng.random() < p_const else W.TERM_RAW
                r[j, i] = (kind, 0, 0, n_gamma * n_out + n_raw)
                n_raw += 1
            else:
                t = 0 if rng.random() < p_zero else int(rng.choice([-1, 1]))
                r[j, i] = (W.TERM_TERNARY, t, 0, j * n_gamma + int(rng.integers(n_gamma)))
    return F.compile_plan(n_in, n_out, n_gamma * n_out + n_raw, r, share=bool(rng.integers(4)),
                          exact=bool(rng.integers(2)))


def lower(desc, N, bits, L):
    ctx = F.Context(N, W.ntt_primes(N, bits, L), device=F.FIONA_DEVICE_NONE)
    return F.Plan(ctx, desc)


@pytest.mark.parametrize("seed", range(40))
def test_random_layers_lower_exactly(seed, monkeypatch):
    rng = np.random.default_rng(7000 + seed)
    shape = SHAPES[seed % len(SHAPES)]
    if shape:
        monkeypatch.setenv("FIONA_TILED_SHAPE", shape)
    desc = random_layer(rng, big=seed % 4 == 3)
    bits = int(rng.choice([40, 50, 52, 59]))  # narrow and wide arithmetic (lazy-sum bounds differ)
    plan = lower(desc, 4096, bits, 2)     # fails with FIONA_ERR_INTERNAL if the map differs
    st = plan.stats()
    assert st["n_terms"] == len(desc.terms)


@pytest.mark.parametrize("name", ["tiny", "vgg", "vit", "bert", "bert-const"])
def test_workloads_lower_exactly(name):
    wl = W.make_workload(name)
    plan = F.Plan(F.Context(wl.N, wl.moduli, device=F.FIONA_DEVICE_NONE), wl.plan)
    if name != "tiny":
        assert plan.stats()["kernel"] == F.FIONA_KERNEL_TILED


@pytest.mark.parametrize("packed", [False, True])
def test_program_forms_lower_exactly(packed, monkeypatch):
    """The signed-sum programs in both forms of the schedule: source byte
    offsets (the default where the schedule fits) and 16-bit indices packed
    two per word (FIONA_TILED_PACKED=1).  The schedule check walks each form
    as the kernel reads it (alignment, whole-source offsets, formations'
    target slots) and the symbolic check evaluates it against the plan's
    terms; plan creation fails otherwise."""
    if packed:
        monkeypatch.setenv("FIONA_TILED_PACKED", "1")
    forms = []
    for seed in range(16):
        rng = np.random.default_rng(9300 + seed)
        shape = ["2,1,1", "1,2,1", "", "1,4,0"][seed % 4]
        if shape:
            monkeypatch.setenv("FIONA_TILED_SHAPE", shape)
        else:
            monkeypatch.delenv("FIONA_TILED_SHAPE", raising=False)
        desc = random_layer(rng, big=seed % 3 == 2)
        plan = lower(desc, 4096, int(rng.choice([40, 50, 59])), 2)
        st = plan.stats()
        if st["kernel"] == F.FIONA_KERNEL_TILED:
            forms.append(st["source_offsets"])
    # (a layer whose offset schedule does not fit in shared memory keeps the packed form)
    if packed:
        assert forms and all(f == 0 for f in forms), forms
    else:
        assert sum(forms) >= len(forms) // 2, forms
    wl = W.make_workload("vgg")
    st = F.Plan(F.Context(wl.N, wl.moduli, device=F.FIONA_DEVICE_NONE), wl.plan).stats()
    assert st["source_offsets"] == (0 if packed else 1)


def test_twelve_warp_variant_only_where_warps_balance():
    """The shape ranking takes the 12-warp variant (two coefficients per
    lane, batches of 8) for BERT, whose 96 outputs load 12 warps evenly and
    whose source regions leave room for one CTA per SM, and keeps 16 warps
    for the first 72 inputs of the VGG layer (16 outputs: 12 warps would
    carry two outputs on four of them) and two CTAs of 8 warps for ViT."""
    def shape(plan, wl):
        st = F.Plan(F.Context(wl.N, wl.moduli, device=F.FIONA_DEVICE_NONE), plan).stats()
        return st["tile_coeffs"], st["warps_per_cta"], st["ctas_per_sm"]
    bert = W.make_workload("bert")
    assert shape(bert.plan, bert) == (64, 12, 1)
    vit = W.make_workload("vit")
    assert shape(vit.plan, vit) == (64, 8, 2)
    vgg = W.make_workload("vgg")
    p = vgg.plan
    rows, offs = [], [0]
    for j in range(p.n_out):
        t = p.terms[p.term_offsets[j]:p.term_offsets[j + 1]]
        t = t[t["input"] < 72]
        rows.append(t)
        offs.append(offs[-1] + len(t))
    half = W.Plan(n_in=72, n_out=p.n_out, n_pt=p.n_pt, term_offsets=np.array(offs, np.uint32),
                  terms=np.concatenate(rows), group_scale_pt=p.group_scale_pt, group_output=p.group_output,
                  node_offsets=p.node_offsets, children=p.children, uses=p.uses)
    assert shape(half, vgg) == (64, 16, 1)


def test_long_signed_runs_are_cut_and_still_exact():
    """One output whose signed run is far longer than the 64-word lazy-sum
    bound of narrow arithmetic (the lowering cuts it into pieces with the
    same gamma), next to outputs with short runs."""
    n_in, n_out = 300, 3
    r = np.zeros((n_out, n_in), F.ROUTE_DTYPE)
    for i in range(n_in):
        r[0, i] = (W.TERM_TERNARY, 1 if i % 3 else -1, 0, 0)
        r[1, i] = (W.TERM_TERNARY, -1 if i % 5 == 0 else 0, 0, 1)
        r[2, i] = (W.TERM_RAW, 0, 0, 3 + i) if i < 20 else (W.TERM_TERNARY, 1, 0, 2)
    desc = F.compile_plan(n_in, n_out, 3 + 20, r, share=False)
    plan = lower(desc, 4096, 50, 2)
    assert plan.stats()["kernel"] == F.FIONA_KERNEL_TILED


def test_warp_formed_sums_lower_exactly(monkeypatch):
    """Random compiled layers on one, two or four warps, so that the users of
    shared signed sums often share a warp: the warps form those sums into
    their slots (nested sums included, children first), and the symbolic
    check of every schedule against the plan's terms passes (plan creation
    fails otherwise).  Sums are formed wherever their slots fit without
    lowering the planned occupancy, which most of these layers allow."""
    formed = []
    for seed in range(24):
        rng = np.random.default_rng(9100 + seed)
        monkeypatch.setenv("FIONA_TILED_SHAPE", ["2,1,1", "2,2,0", "1,2,1", "1,4,0"][seed % 4])
        desc = random_layer(rng, big=False)
        bits = int(rng.choice([40, 50, 59]))
        plan = lower(desc, 4096, bits, 2)
        formed.append(plan.stats()["nodes_materialized"])
    assert sum(1 for f in formed if f > 0) >= 12, formed


def test_tensor_core_sums_lower_exactly(monkeypatch):
    """FIONA_TILED_TC=1: every used scale group's signed sum becomes one
    group source formed by the tensor-core contraction; plan creation checks
    the schedule's linear map (the group programs) and decodes the fp16
    weight image and the groups' constants back against those programs
    (failing with FIONA_ERR_INTERNAL otherwise).  Random compiled layers with
    one coefficient per lane and batches of 16 (shared sums expanded into the
    groups), the VGG layer, and the layers that cannot take it: moduli of 59
    bits, and BERT's 96 groups (tensor memory holds at most 28 next to its
    96 inputs)."""
    monkeypatch.setenv("FIONA_TILED_TC", "1")
    taken = 0
    for seed in range(16):
        rng = np.random.default_rng(9300 + seed)
        monkeypatch.setenv("FIONA_TILED_SHAPE", ["1,4,1,-1,16", "1,8,0,-1,16", "1,16,1,-1,16"][seed % 3])
        desc = random_layer(rng, big=seed % 2 == 1)
        plan = lower(desc, 4096, int(rng.choice([40, 50])), 2)
        taken += plan.stats()["tensor_core_sums"] > 0
    # (the others: a single output, which runs the direct kernel, or more
    # groups than tensor memory holds next to the inputs' chunks)
    assert taken >= 8
    monkeypatch.delenv("FIONA_TILED_SHAPE")
    for name, want in (("vgg", 16), ("bert", 0), ("overflow60", 0)):
        wl = W.make_workload(name)
        plan = F.Plan(F.Context(wl.N, wl.moduli, device=F.FIONA_DEVICE_NONE), wl.plan)
        assert plan.stats()["tensor_core_sums"] == want, name
    monkeypatch.delenv("FIONA_TILED_TC")
    wl = W.make_workload("vgg")
    plan = F.Plan(F.Context(wl.N, wl.moduli, device=F.FIONA_DEVICE_NONE), wl.plan)
    assert plan.stats()["tensor_core_sums"] == 0  # the ALU sums are the default
