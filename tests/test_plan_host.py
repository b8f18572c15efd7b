"""The step planner (mlkv_plan_step) on the host, no GPU: which form mlkv_decode_step takes.

The decode step runs in the cross-layer fused form only for maps of equal contiguous owner blocks
(Sec. 3, Eq. 18), where a unit (sequence, KV head, block, chunk) reads every K/V tile of its chunk
once for all the block's layers; by default only where that measured faster than the decode
kernel's launch.  The planner is the same decision the step makes on a device, so these pins hold
the step's form for the workloads (measured winners on GB300, 152 SMs), the context split and the
CTA form, and the planner's search against the definition it searches for.
"""
import numpy as np
import pytest

import paper_2406_09297_gb300 as mlkv
from mlkv_synth import workloads
from tests.mlkv_cases import FUSED_STEP_CASES, FUSED_STEP_SMS

# CTA forms of the fused launch (plan "form")
TWO_TILES, ONE_TILE, SPLIT_KEYS = 0, 1, 2


def _plan(w, **options):
    return mlkv.mlkv_plan_step(w.owner, w.h, w.d, w.g, w.seq_lens(), w.max_seq, FUSED_STEP_SMS,
                               **options)


@pytest.mark.parametrize("owner,h,g,d,b,L,kc,units,tiles", FUSED_STEP_CASES)
@pytest.mark.parametrize("deep", [1, 0])
def test_forced_fused_plan(owner, h, g, d, b, L, kc, units, tiles, deep):
    # The split of the GPU test of the fused step (option step_fused 2), and its CTA form: two
    # query tiles when the block's rows exceed one (or head_dim 128), else split keys at one CTA
    # per SM when the units fit one per SM and fused_deep is on, else two CTAs per SM.
    plan = mlkv.mlkv_plan_step(owner, h, d, g, [L] * b, L, FUSED_STEP_SMS, step_fused=2,
                               fused_deep=deep)
    form = TWO_TILES if tiles == 2 else (SPLIT_KEYS if deep and units <= FUSED_STEP_SMS
                                         else ONE_TILE)
    assert plan == {"fused": 1, "form": form, "kc": kc, "units": units}


# The default form per workload (F fused, M the decode kernel's launch), as measured on GB300:
# blocks of one or two layers never fused, the MLKV maps of >= 3 layers a block fused.
DEFAULT_FORMS = {
    "pythia160m-mlkv6-b1-L128": "M",
    "pythia160m-mlkv2-b64-L2048": "F",
    "pythia160m-gqa4-mlkv4-b128-Lu4096": "F",
    "llama2-7b-mlkv8-gqa4-b32-L16384": "F",
    "llama2-7b-mlkv8-gqa4-b32-L2048": "F",
    "pythia160m-mha-b256-L8192": "M",
    "pythia160m-gqa4-b256-L8192": "M",
    "pythia160m-mqa-b256-L8192": "M",
    "pythia160m-mlkv6-b256-L8192": "M",
    "pythia160m-mlkv4-b256-L8192": "F",
    "pythia160m-mlkv2-b256-L8192": "F",
    "pythia160m-mlkv1-b256-L8192": "F",
    "pythia160m-mha-b1-L131072": "M",
    "pythia160m-gqa4-b1-L131072": "M",
    "pythia160m-mqa-b1-L131072": "M",
    "pythia160m-mlkv6-b1-L131072": "M",
    "pythia160m-mlkv4-b1-L131072": "F",
    "pythia160m-mlkv2-b1-L131072": "F",
    "pythia160m-mlkv1-b1-L131072": "F",
}


@pytest.mark.parametrize("name", sorted(DEFAULT_FORMS))
def test_default_form_of_the_workloads(name):
    w = workloads.by_name(name)
    plan = _plan(w)
    assert plan["fused"] == (DEFAULT_FORMS[name] == "F"), plan
    if not plan["fused"]:
        assert plan == {"fused": 0, "form": -1, "kc": 0, "units": 0}


def test_default_workload_plan():
    # Batch 64 x 2048 positions, two blocks of six layers, one KV head: 128 units of 16 key tiles
    # (no split: 128 units already fit the 152 SMs), one CTA per SM in the split-key form.
    w = workloads.by_name("pythia160m-mlkv2-b64-L2048")
    assert _plan(w) == {"fused": 1, "form": SPLIT_KEYS, "kc": 16, "units": 128}
    # the options: never fused; two CTAs per SM; a forced context split
    assert _plan(w, step_fused=0)["fused"] == 0
    assert _plan(w, fused_deep=0)["form"] == ONE_TILE
    assert _plan(w, fused_kc=4) == {"fused": 1, "form": ONE_TILE, "kc": 4, "units": 512}


def test_long_single_sequence_split():
    # Batch 1 x 131072 positions, MLKV-1 (one block of 12 layers x 12 heads = 144 rows: two query
    # tiles): 1024 key tiles; the smallest chunk whose units fit the SMs is 7 tiles (147 chunks; 6
    # tiles would make 171).
    w = workloads.by_name("pythia160m-mlkv1-b1-L131072")
    assert _plan(w) == {"fused": 1, "form": TWO_TILES, "kc": 7, "units": 147}


def test_context_split_is_the_smallest_that_fits():
    # The planner bisects for the smallest chunk whose units number at most the SMs; against the
    # definition by exhaustion on random maps, lengths and SM counts.
    rng = np.random.default_rng(11)
    for _ in range(300):
        L = int(rng.choice([1, 2, 3, 4, 6]))
        m = int(rng.integers(1, 4))
        owner = [n - n % L for n in range(L * m)]
        g = int(rng.choice([1, 2, 4]))
        h = g * int(rng.choice([1, 2, 3]))
        b = int(rng.integers(1, 6))
        max_seq = int(rng.integers(1, 20000))
        lens = [int(x) for x in rng.integers(1, max_seq + 1, b)]
        sms = int(rng.integers(1, 400))
        plan = mlkv.mlkv_plan_step(owner, h, 64, g, lens, max_seq, sms, step_fused=2)
        tiles = [(x + 127) // 128 for x in lens]

        def units(k):
            return sum(m * g * ((t + k - 1) // k) for t in tiles)

        n_kt = max(tiles)
        if units(n_kt) >= sms:
            kc = n_kt
        else:
            kc = min(k for k in range(1, n_kt + 1) if units(k) <= sms)
        assert (plan["kc"], plan["units"]) == (kc, units(kc)), (owner, h, g, lens, sms, plan)


def test_maps_the_fused_form_does_not_take():
    lens = [1000] * 4
    # blocks of unequal size, or an owner that is not its block's first layer
    for owner in ([0, 0, 0, 3, 3], [0, 0, 2, 2, 2, 2], [0, 1, 1, 1]):
        plan = mlkv.mlkv_plan_step(owner, 12, 64, 1, lens, 1000, 152, step_fused=2)
        assert plan["fused"] == 0, owner
    # a block's query rows beyond two tiles of 128 (12 layers x 12 heads of one KV head = 144
    # rows fit; 24 layers = 288 do not)
    assert mlkv.mlkv_plan_step([0] * 12, 12, 64, 1, lens, 1000, 152, step_fused=2)["fused"] == 1
    assert mlkv.mlkv_plan_step([0] * 24, 12, 64, 1, lens, 1000, 152, step_fused=2)["fused"] == 0


def test_planner_rejects_bad_arguments():
    ok = dict(layer_owner=[0, 0], n_q_heads=12, head_dim=64, kv_heads_per_owner=1,
              seq_lens=[5, 5], max_seq=8, sm_count=152)
    assert mlkv.mlkv_plan_step(**ok)["fused"] == 0   # blocks of two layers: not by default
    for bad, code in [(dict(layer_owner=[1, 1]), mlkv.MLKV_ERR_MAP),
                      (dict(kv_heads_per_owner=5), mlkv.MLKV_ERR_MAP),
                      (dict(head_dim=96), mlkv.MLKV_ERR_UNSUPPORTED),
                      (dict(seq_lens=[5, 9]), mlkv.MLKV_ERR_RANGE),
                      (dict(seq_lens=[0, 5]), mlkv.MLKV_ERR_RANGE),
                      (dict(sm_count=0), mlkv.MLKV_ERR_INVALID_ARG),
                      (dict(step_fused=3), mlkv.MLKV_ERR_INVALID_ARG),
                      (dict(step_fused=-2), mlkv.MLKV_ERR_INVALID_ARG),
                      (dict(fused_kc=-2), mlkv.MLKV_ERR_INVALID_ARG),
                      (dict(fused_deep=2), mlkv.MLKV_ERR_INVALID_ARG)]:
        with pytest.raises(mlkv.MLKVError) as e:
            mlkv.mlkv_plan_step(**{**ok, **bad})
        assert e.value.code == code, bad
