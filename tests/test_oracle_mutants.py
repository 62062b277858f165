"""The oracle's pins must be sharp: each plausible mistake planted in a copy
of the oracle (on the CPU, in a temporary directory) makes a pin fail."""
import os

import numpy as np
import pytest

from oracle import oracle as O
from tests import test_oracle_adaptive as adpins
from tests import test_oracle_autoscale as apins
from tests import test_oracle_pins as pins

MUTANTS = {
    "drop HoL demand (Eq. 2)": ("if (h >= 0) usage += need_blocks(req[h]);                      /* HoL demand",
                                "(void)h;  /* HoL demand"),
    "headroom per request instead of per tier (Eq. 4)": (
        "if (in.cnt[k] > 0) usage += H[k];", "usage += (int64_t)H[k] * in.cnt[k];"),
    "drop inbound reservation": ("usage += in.reserved_in;                                       /* inbound",
                                 "/* inbound"),
    "dispatch ties to highest index": ("if (!draining(i) && (best < 0 || freer(i, best))) best = i;",
                                       "if (!draining(i) && (best < 0 || !freer(best, i))) best = i;"),
    "migration gate sign flipped": ("(nd * ds - ns * dd) <", "(ns * dd - nd * ds) <"),
    "oldest preemption victim": ("(req[x].tier == req[v].tier && x > v)", "(req[x].tier == req[v].tier && x < v)"),
    "queued candidate from the front": ("int r = S.waiting[kq].back();\n                S.waiting[kq].pop_back();",
                                        "int r = S.waiting[kq].front();\n                S.waiting[kq].pop_front();"),
    "prefill and decode costs transposed": (
        "c.iter_us_per_prefill_token * prefill_tokens +\n                              c.iter_us_per_decode_seq * n_decode",
        "c.iter_us_per_decode_seq * prefill_tokens +\n                              c.iter_us_per_prefill_token * n_decode"),
    "stage ignores destination memory": ("if (d.free_blocks < c_blocks) { abort_migration(si); return; }", ""),
    "batch size counted from zero": (
        "/* inbound migration copy */\n        num = (int64_t)c.blocks_per_instance - usage;\n"
        "        den = in.running.empty() ? 1 : (int64_t)in.running.size();",
        "/* inbound migration copy */\n        num = (int64_t)c.blocks_per_instance - usage;\n"
        "        den = (int64_t)in.running.size() + 1;"),
    "KV need rounds down": ("return (r.P + r.g + c.tokens_per_block - 1) / c.tokens_per_block;",
                            "return (r.P + r.g) / c.tokens_per_block;"),
    "F_normal keeps the headroom": (
        "        usage += in.reserved_in;\n        num = (int64_t)c.blocks_per_instance - usage;\n"
        "        den = in.running.empty() ? 1 : (int64_t)in.running.size();\n    }\n    /* An instance drains",
        "        usage += in.reserved_in;\n        for (int k = 0; k < c.num_tiers; ++k) if (in.cnt[k] > 0) "
        "usage += c.headroom[k];\n        num = (int64_t)c.blocks_per_instance - usage;\n"
        "        den = in.running.empty() ? 1 : (int64_t)in.running.size();\n    }\n    /* An instance drains"),
    "mean over draining instances too": ("if (draining(i)) continue;  /* an instance that is leaving", "/* leaving"),
    "scale-in threshold not strict": ("} else if (p * c.scale_den > (__int128)c.scale_in_num * n * q) {",
                                      "} else if (p * c.scale_den >= (__int128)c.scale_in_num * n * q) {"),
    "scale-out threshold not strict": ("if (p * c.scale_den < (__int128)c.scale_out_num * n * q) {",
                                       "if (p * c.scale_den <= (__int128)c.scale_out_num * n * q) {"),
    "draining instance still gets dispatch": ("if (!draining(i) && (best < 0 || freer(i, best))) best = i;",
                                              "if (best < 0 || freer(i, best)) best = i;"),
    "fallback picks the lowest index": ("                    if (best < 0 || freer(i, best)) best = i;",
                                        "                    if (best < 0) best = i;"),
    "draining source needs the threshold": ("            if (!drain_source) {\n                int64_t ns",
                                            "            {\n                int64_t ns"),
    "draining instance as destination": ("if (eligible[i] && i != s && !draining(i) && (d < 0 || freer(i, d))) d = i;",
                                         "if (eligible[i] && i != s && (d < 0 || freer(i, d))) d = i;"),
    "drain starts one tick late": ("return c.drain_start_us != nullptr && now >= c.drain_start_us[i];",
                                   "return c.drain_start_us != nullptr && now > c.drain_start_us[i];"),
    "stage copies every block at once (S ignored)": (
        "int c_blocks = std::min(c.migrate_blocks_per_iter, r.blocks - s.mig_copied);",
        "int c_blocks = r.blocks - s.mig_copied;"),
    "running candidate with the most blocks": ("(a.blocks != b.blocks ? a.blocks < b.blocks : r > best)",
                                               "(a.blocks != b.blocks ? a.blocks > b.blocks : r > best)"),
    "arrivals dispatched lowest tier first": ("return req[a].tier < req[b].tier; });",
                                              "return req[a].tier > req[b].tier; });"),
    "admission ignores the batch limit": ("while ((int)in.running.size() < c.max_batch) {",
                                          "while (true) {"),
    "commit ignores the destination's batch limit": (
        "if (s.mig_copied == r.blocks && (int)d.running.size() < c.max_batch) commit_migration(si);",
        "if (s.mig_copied == r.blocks) commit_migration(si);"),
    "highest-priority preemption victim": ("req[x].tier > req[v].tier ||", "req[x].tier < req[v].tier ||"),
    "migration gate strict (F_d - F_s > theta)": ("< (int64_t)c.theta_num * dd * ds) break;",
                                                   "<= (int64_t)c.theta_num * dd * ds) break;"),
    "admission past a misfit head": ("if (need > in.free_blocks) break;", "if (need > in.free_blocks + need) break;"),
    "headroom change applied one step late": ("c.headroom_change_step[next_change] <= st.steps",
                                              "c.headroom_change_step[next_change] < st.steps"),
    "running candidate of the highest priority": ("if (a.tier != b.tier ? a.tier > b.tier :",
                                                  "if (a.tier != b.tier ? a.tier < b.tier :"),
    "queued candidate from the highest-priority bucket": (
        "for (int k = c.num_tiers - 1; k >= 0; --k)\n                if (!S.waiting[k].empty()) { kq = k; break; }",
        "for (int k = 0; k < c.num_tiers; ++k)\n                if (!S.waiting[k].empty()) { kq = k; break; }"),
    "aborted copy keeps the destination's blocks": (
        "d.free_blocks += s.mig_copied;   /* copied blocks are released on the destination */",
        "/* copied blocks are kept */"),
    "headroom schedule ignored": ("for (int k = 0; k < c.num_tiers; ++k) H[k] = c.headroom_change_table[next_change * MAXK + k];",
                                  "(void)0;"),
}


def _pins_fail(so_path):
    failures = 0
    for check in (lambda: pins.check_tiny_agreement(range(120), so_path=so_path),
                  lambda: _closed_forms(so_path),
                  lambda: apins.check_tiny_drain_agreement(range(200), so_path=so_path),
                  lambda: _autoscale_closed_form(so_path),
                  lambda: pins.check_threshold_equality(so_path=so_path),
                  lambda: adpins.check_tiny_schedule_agreement(range(150), so_path=so_path),
                  lambda: adpins.check_dispatch_follows_the_change(so_path=so_path)):
        try:
            check()
        except AssertionError:
            failures += 1
    return failures


def _closed_forms(so_path):
    for P, Ob in ((553, 221), (17, 2)):
        cfg = O.make_config(4, 1024, [256, 128])
        res = O.run_trace(cfg, np.array([1000], np.uint32), np.array([P], np.uint16), np.array([Ob], np.uint16),
                          np.array([1], np.uint8), so_path=so_path)
        assert int(res.first_token_us[0]) - 1000 == 4000 + 20 * P
        assert int(res.finish_us[0]) - int(res.first_token_us[0]) == (Ob - 1) * 4030


def _autoscale_closed_form(so_path):
    tr = (np.zeros(4, np.uint32), np.full(4, apins.P, np.uint16), np.full(4, apins.OUT, np.uint16),
          np.zeros(4, np.uint8))
    cfg = O.make_config(2, apins.M, [0], max_batch=1, enable_migration=0, autoscale=1)
    res = O.run_trace(cfg, *tr, so_path=so_path)
    assert apins._signals(res) == ([50_000, 100_000, 150_000, 200_000],
                                   [250_000, 300_000, 350_000, 450_000, 500_000, 550_000, 600_000])


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_planted_mistake_is_caught(name, tmp_path):
    before, after = MUTANTS[name]
    src = open(O.SRC).read()
    assert src.count(before) == 1, "mutation site not found: " + name
    mpath = os.path.join(tmp_path, "mutant.cpp")
    with open(mpath, "w") as f:
        f.write(src.replace(before, after))
    so = O.build(force=True, so_path=os.path.join(tmp_path, "libmutant.so"), src=mpath, opt="-O1")
    assert _pins_fail(so) > 0, "pins did not catch: " + name
