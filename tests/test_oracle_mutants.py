"""The oracle's pins must be sharp: each plausible mistake planted in a copy
of the oracle (on the CPU, in a temporary directory) makes a pin fail."""
import os

import numpy as np
import pytest

from oracle import oracle as O
from tests import test_oracle_pins as pins

MUTANTS = {
    "drop HoL demand (Eq. 2)": ("if (h >= 0) usage += need_blocks(req[h]);", "(void)h;"),
    "headroom per request instead of per tier (Eq. 4)": (
        "if (in.cnt[k] > 0) usage += c.headroom[k];", "usage += (int64_t)c.headroom[k] * in.cnt[k];"),
    "drop inbound reservation": ("usage += in.reserved_in;", ""),
    "dispatch ties to highest index": ("if (freer(i, best)) best = i;", "if (!freer(best, i)) best = i;"),
    "migration gate sign flipped": ("(nd * ds - ns * dd) <", "(ns * dd - nd * ds) <"),
    "oldest preemption victim": ("(req[x].tier == req[v].tier && x > v)", "(req[x].tier == req[v].tier && x < v)"),
    "queued candidate from the front": ("int r = S.waiting[kq].back();\n                S.waiting[kq].pop_back();",
                                        "int r = S.waiting[kq].front();\n                S.waiting[kq].pop_front();"),
    "prefill and decode costs transposed": (
        "c.iter_us_per_prefill_token * prefill_tokens +\n                              c.iter_us_per_decode_seq * n_decode",
        "c.iter_us_per_decode_seq * prefill_tokens +\n                              c.iter_us_per_prefill_token * n_decode"),
    "stage ignores destination memory": ("if (d.free_blocks < c_blocks) { abort_migration(si); return; }", ""),
    "batch size counted from zero": ("den = in.running.empty() ? 1 : (int64_t)in.running.size();",
                                     "den = (int64_t)in.running.size() + 1;"),
    "KV need rounds down": ("return (r.P + r.g + c.tokens_per_block - 1) / c.tokens_per_block;",
                            "return (r.P + r.g) / c.tokens_per_block;"),
}


def _pins_fail(so_path):
    failures = 0
    for check in (lambda: pins.check_tiny_agreement(range(120), so_path=so_path),
                  lambda: _closed_forms(so_path)):
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
