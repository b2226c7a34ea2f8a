"""Host-side logic of bench.py (no GPU): the clock summary, the agent-step
split of an update, the algorithmic work of each row, the replica
throughput."""
import bench
from paper_2607_03441_gb300 import workloads as wk


def test_clock_summary():
    lines = ["0, 2070, 2070, 900.1, 0x0, Not Active, Not Active, Not Active, Not Active\n",
             "0, 1500, 2070, 1400.0, 0x4, Not Active, Not Active, Not Active, Active\n",
             "0, 1800, 2070, 1300.0, 0x0, Not Active, Not Active, Not Active, Not Active\n",
             "garbage\n"]
    out = bench.ClockSampler.summarize(lines)
    assert out == {"sm_mhz": 1800.0, "sm_max_mhz": 2070.0, "samples": 3, "reasons": ["sw_power_cap"]}
    assert bench.ClockSampler.summarize([]) is None


def test_agent_cuts_split_an_update_evenly():
    for L, K in ((2048, 5), (256, 3), (7, 5), (5, 5)):
        cuts = bench._agent_cuts(L, K)
        assert len(cuts) == K + 1 and cuts[0] == 0 and cuts[-1] == L
        steps = [b - a for a, b in zip(cuts, cuts[1:])]
        assert min(steps) >= 0 and max(steps) - min(steps) <= 1


def test_work_accounting():
    wl = wk.WORKLOADS["7b"]
    work = bench.row_work(wl)
    assert work["weighted_ce_fwd_bwd"] == ("tensor", 4.0 * 2048 * 152064 * 3584, "FLOP")
    # LoRA bytes: x once, every dy once, adapters in and gradients out
    x = 2 * 2048 * 3584
    dys = 2 * 2048 * (3584 + 512)
    ad = 6 * 3584 * 16 * 2 + 6 * 16 * (3584 + 512)
    assert work["lora_grad"] == ("hbm", x + dys + ad, "B")
    ew = wk.EPISODES["7b-episode"]
    L, V, d = ew.L, ew.V, ew.d
    per_step = 4.0 * L * V * d + 2 * (2.0 * L * d * d + 2.0 * L * 16 * 2 * d) + 4.0 * L * 16 * 2 * d
    assert bench.episode_flops(ew) == 2 * per_step


def test_replica_throughput():
    # 4 replicas, 10 steps of 2,048 tokens in 50 ms: 1.6384 M tokens/s
    assert abs(bench.replica_throughput(2048, 10, 4, 50.0) - 1638400.0) < 1e-6


class _Recorder:
    """Stands in for the binding: records the order of the calls."""

    def __init__(self):
        self.calls = []

    def __getattr__(self, name):
        def call(*args, **kwargs):
            self.calls.append(name)
        return call


def test_update_step_order_with_gradient_steps():
    """Algorithm 1 per update: the weights once, then per gradient step
    Eq. 10, the LoRA gradients of every group and the SGD step of every
    projection, then the history insert once."""
    wl = wk.WORKLOADS["7b"]
    for G in (1, 2):
        u = object.__new__(bench.Update)
        u.attt, u.wl, u.grad_steps = _Recorder(), wl, G
        u.hist = u.x = u.w = u.h = u.W = u.loss = u.dh = u.ws_ce = None
        u.ws_lora = {"attn": None}
        u.projs = list(wl.projs)
        u.groups = {"attn": list(range(len(u.projs)))}
        u.xin = {"attn": None}
        u.dy = u.A16 = u.B16 = u.A32 = u.B32 = u.dA = u.dB = [None] * len(u.projs)
        u.step()
        P = len(u.projs)
        round_ = ["attt_weighted_ce_fwd_bwd", "attt_lora_grad"] + ["attt_lora_step"] * P
        assert u.attt.calls == ["attt_ngram_weights"] + round_ * G + ["attt_history_insert"]


def test_peak_kind_follows_region_length_and_clock():
    """A short region at full clock is held to the burst peak; a long one, or
    one whose median clock fell below the maximum (power cap), to the
    sustained peak."""
    full = {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "samples": 5, "reasons": []}
    capped = {"sm_mhz": 1440.0, "sm_max_mhz": 2070.0, "samples": 5, "reasons": ["sw_power_cap"]}
    assert bench.peak_kind(53.0, full) == "burst"
    assert bench.peak_kind(53.0, capped) == "sustained"
    assert bench.peak_kind(1700.0, full) == "sustained"
    assert bench.peak_kind(200.0, None) == "burst"
    assert bench.peak_kind(2000.0, None) == "sustained"


def test_ce_roofline_frac_follows_from_the_record():
    """frac = 4 L V d / ce_ms / the named peak, with both peaks' fractions."""
    wl = wk.WORKLOADS["32b"]
    peaks = {"hbm_gbs": 6780.0, "bf16": 1908.6, "bf16_sustained": 1705.1, "src": "measured"}
    for kind, peak in (("burst", 1908.6), ("sustained", 1705.1)):
        r = bench._ce_roofline(wl, 15.0, peaks, None, kind)
        ach = 4.0 * wl.L * wl.V * wl.d / 15e-3 / 1e12
        assert abs(r["frac"] - ach / peak) < 1e-4 and r["peak"] == peak
        assert abs(r["frac_of_burst"] - ach / 1908.6) < 1e-4
        assert abs(r["frac_of_sustained"] - ach / 1705.1) < 1e-4


def test_path_roofline_is_the_slower_bound_of_the_whole_update():
    wl = wk.WORKLOADS["32b"]
    peaks = {"hbm_gbs": 6780.0, "bf16": 1908.6, "bf16_sustained": 1705.1, "src": "measured"}
    flops, nbytes = bench.path_work(wl, 1)
    ce = 4.0 * wl.L * wl.V * wl.d
    lora = sum(4.0 * wl.L * wl.r * (p.din + p.dout) for p in wl.projs)
    assert flops == ce + lora
    assert bench.path_work(wl, 2)[0] == 2 * flops
    r = bench.path_roofline(wl, 1, 20.0, peaks, "sustained")
    t_roof = max(flops / 1705.1e12, nbytes / 6780e9)
    assert r["bound"] == "tensor" and abs(r["frac"] - t_roof / 20e-3) < 1e-4


class _FakeCuda:
    """Stands in for torch.cuda's streams and events: records, on one shared
    log, which stream each event is recorded on and what each stream waits
    for."""

    def __init__(self):
        self.log = []
        outer = self

        class Stream:
            def __init__(self, name):
                self.name = name

            def wait_event(self, ev):
                outer.log.append(("wait", self.name, ev.name))

        class Event:
            n = 0

            def __init__(self, *a, **k):
                Event.n += 1
                self.name = f"ev{Event.n}"

            def record(self, stream=None):
                outer.log.append(("record", stream.name if stream else "main", self.name))

        self.Stream, self.Event = Stream, Event
        self.main = Stream("main")

    def current_stream(self):
        return self.main


class _StreamRecorder(_Recorder):
    """Records each call's name and the stream it was given."""

    def __getattr__(self, name):
        def call(*args, **kwargs):
            st = kwargs.get("stream")
            self.calls.append((name, st.name if st is not None else "main"))
        return call


def test_update_runs_independent_lora_groups_on_their_own_streams():
    """Two projection groups: the first group's gradients on the update's
    stream, the second on a side stream that waits for an event recorded on
    the update's stream before the first call (after Eq. 10) and is joined
    before the SGD steps."""
    import types
    wl = wk.WORKLOADS["32b"]
    fake = _FakeCuda()
    u = object.__new__(bench.Update)
    u.attt, u.wl, u.grad_steps = _StreamRecorder(), wl, 1
    u.torch = types.SimpleNamespace(cuda=fake)
    u.hist = u.x = u.w = u.h = u.W = u.loss = u.dh = u.ws_ce = None
    u.projs = list(wl.projs)
    u.groups = {}
    for i, p in enumerate(u.projs):
        u.groups.setdefault(p.x_group, []).append(i)
    assert len(u.groups) == 2
    u.ws_lora = {g: None for g in u.groups}
    u.xin = {g: None for g in u.groups}
    u.dy = u.A16 = u.B16 = u.A32 = u.B32 = u.dA = u.dB = [None] * len(u.projs)
    u.side = [fake.Stream("side0")]
    u.step()
    names = [c[0] for c in u.attt.calls]
    P = len(u.projs)
    assert names == (["attt_ngram_weights", "attt_weighted_ce_fwd_bwd", "attt_lora_grad", "attt_lora_grad"]
                     + ["attt_lora_step"] * P + ["attt_history_insert"])
    lora = [c for c in u.attt.calls if c[0] == "attt_lora_grad"]
    assert lora == [("attt_lora_grad", "main"), ("attt_lora_grad", "side0")]
    (_, s0, fork), (_, s1, waited), (_, s2, join), (_, s3, joined) = fake.log
    assert (s0, s1, s2, s3) == ("main", "side0", "side0", "main")
    assert waited == fork and joined == join
