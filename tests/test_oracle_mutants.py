"""Plant plausible mistakes in a scratch copy of the oracle (on the CPU) and
check that the oracle's pins catch every one of them: a transposed link
operand, floor instead of ceiling, a dropped release, dispatch ignoring the
ready time, allocs before frees, dropped terms of the free times, >= for >,
scoring unscored ops, ignoring busy-until times, wrong alloc instants, a
shifted resume time, a peak without the resident base, a non-strict argmin
and a wrong violation order; in the arbitrated mode, a dropped link or
receiver check, destination-first order, the receive buffer allocated at the
intent, a sender never released and no arbitration after a completion."""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "sim_ref.cpp")

MUTANTS = {
    "transposed_link": [("g.bw[size_t(d) * g.D + e]) + g.lat", "g.bw[size_t(e) * g.D + d]) + g.lat")],
    "floor_not_ceil": [("return (q * b == a) ? q : q + 1;", "return q;")],
    "no_release": [("events.push(Ev(g.release[i], 1, i));", "events.push(Ev(0, 1, i));")],
    "dispatch_by_id": [("ready_q[dev[j]].insert({r[j], j});", "ready_q[dev[j]].insert({0, j});")],
    "alloc_before_free": [("return std::tie(a.t, a.cls, a.op) < std::tie(b.t, b.cls, b.op);",
                           "return std::make_tuple(a.t, -a.cls, a.op) < std::make_tuple(b.t, -b.cls, b.op);")],
    "src_ignores_arrival": [("for (const Copy& c : copies[i]) src_free = std::max(src_free, c.arrive);", "")],
    "remote_ignores_cons": [("if (last_use.count(c.e)) t_free = std::max(t_free, last_use[c.e]);", "")],
    "src_ignores_cons": [("if (last_use.count(d)) src_free = std::max(src_free, last_use[d]);", "")],
    "viol_ge": [("if (live > g.cap[d]) {", "if (live >= g.cap[d]) {")],
    "score_all": [("if (g.scored[i]) score += f[i];", "score += f[i];")],
    "sla_ge": [("miss += res.req_done[q] > g.deadline[q] ? 1 : 0;",
                "miss += res.req_done[q] >= g.deadline[q] ? 1 : 0;")],
    "avail0_ignored": [("if (running[d] >= 0 || g.avail0[d] > now || ready_q[d].empty()) continue;",
                        "if (running[d] >= 0 || ready_q[d].empty()) continue;")],
    "remote_alloc_at_arrival": [("mem[c.e].push_back({c.alloc, 1, i, b});",
                                 "mem[c.e].push_back({c.arrive, 1, i, b});")],
    "src_alloc_at_ready": [("mem[d].push_back({s[i], 1, i, b});", "mem[d].push_back({r[i], 1, i, b});")],
    "t0_shifted": [("t = std::min(t, base.finish[p]);", "t = std::min(t, base.finish[p] + 1);")],
    "events_after_t0_only": [("ev += base.ready[i] >= t0 ? 1 : 0;", "ev += base.ready[i] > t0 ? 1 : 0;")],
    "arb_resumed_counts_every_op": [("if (g.mode == 1 && !resumed) {", "if (g.mode == 1) {")],
    "peak_without_base": [("int64_t live = g.base[d], peak = g.base[d];", "int64_t live = g.base[d], peak = 0;")],
    "argmin_not_strict": [("better = best < 0 || s[k].score < bscore;", "better = best < 0 || s[k].score <= bscore;")],
    "arb_no_link_check": [("if (sending[src] || receiving[t.e] || links_busy.count(lk)) {",
                           "if (sending[src] || receiving[t.e]) {")],
    "arb_no_receiver_check": [("if (sending[src] || receiving[t.e] || links_busy.count(lk)) {",
                               "if (sending[src] || links_busy.count(lk)) {")],
    "arb_order_by_destination": [("pending.insert(std::make_tuple(now, id, e, int(X.size()) - 1));",
                                  "pending.insert(std::make_tuple(now, e, id, int(X.size()) - 1));")],
    "arb_recv_alloc_at_intent": [("copies[t.p].push_back({t.e, t.start, t.done});",
                                  "copies[t.p].push_back({t.e, t.intent, t.done});")],
    "arb_sender_kept": [("        sending[src] = false;\n", "")],
    "arb_no_trigger_on_completion": [("          if (dev[j] == t.e) events.push(Ev(now, 2, j));\n        trigger = true;",
                                      "          if (dev[j] == t.e) events.push(Ev(now, 2, j));\n        trigger = false;")],
    "viol_order_dev_first": [("auto key = std::make_tuple(e.t, e.op, d);", "auto key = std::make_tuple(e.t, d, e.op);"),
                             ("key < std::make_tuple(vt, vop, vdev)", "key < std::make_tuple(vt, vdev, vop)")],
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_catch_planted_mistake(name, tmp_path):
    src = open(SRC).read()
    for a, b in MUTANTS[name]:
        assert a in src, "mutation anchor missing: " + a
        src = src.replace(a, b)
    cpp = tmp_path / "mut.cpp"
    so = tmp_path / "libmut.so"
    cpp.write_text(src)
    subprocess.check_call(["g++", "-O1", "-std=c++17", "-shared", "-fPIC", "-pthread", str(cpp),
                           "-o", str(so)])
    env = dict(os.environ, ORACLE_LIB_OVERRIDE=str(so))
    files = [os.path.join(ROOT, "tests", f) for f in (
        "test_oracle_golden.py", "test_oracle_closed_forms.py", "test_oracle_invariants.py",
        "test_oracle_bruteforce.py", "test_oracle_incremental.py", "test_oracle_crosscheck.py",
        "test_oracle_arbitration.py")]
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider"] + files,
                       env=env, capture_output=True, text=True, cwd=ROOT)
    assert r.returncode != 0, "planted mistake %s was not caught:\n%s" % (name, r.stdout[-2000:])
