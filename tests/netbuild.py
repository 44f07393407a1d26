"""Hand-built switch networks for worked cases (test helper, no method code)."""
import numpy as np

from paper_2602_16100_gb300 import workloads as W


def ip(a, b, c, d):
    return (a << 24) | (b << 16) | (c << 8) | d


def rule(priority, dst_ip=0, dst_len=0, action=0, in_port=W.ANY_PORT, src_ip=0, src_len=0, lo=0, hi=65535):
    r = np.zeros(1, W.RULE_DTYPE)
    r["priority"], r["in_port"] = priority, in_port
    r["src_ip"], r["src_len"], r["dst_ip"], r["dst_len"] = src_ip, src_len, dst_ip, dst_len
    r["dport_lo"], r["dport_hi"], r["action"] = lo, hi, action
    return r


def make_net(nports, links, hosts, region, rules):
    """nports[s]: port count of switch s.  links: (s, p, s2, p2) undirected.
    hosts: list of (switch, port, ipv4).  rules: list per switch of rule
    records (input order)."""
    S = len(nports)
    port_offs = np.zeros(S + 1, np.uint32)
    port_offs[1:] = np.cumsum(nports)
    peer = np.full(int(port_offs[-1]), W.PEER_NONE, np.int32)
    for s, p, s2, p2 in links:
        peer[port_offs[s] + p] = (s2 << 8) | p2
        peer[port_offs[s2] + p2] = (s << 8) | p
    for h, (s, p, _) in enumerate(hosts):
        peer[port_offs[s] + p] = W.HOST_BIT | h
    rule_offs = np.zeros(S + 1, np.uint32)
    rule_offs[1:] = np.cumsum([len(r) for r in rules])
    allr = np.concatenate([np.concatenate(r) if len(r) else np.zeros(0, W.RULE_DTYPE) for r in rules]) \
        if rule_offs[-1] else np.zeros(0, W.RULE_DTYPE)
    return W.Network(S, rule_offs, allr.astype(W.RULE_DTYPE), np.array(region, np.uint8), port_offs, peer,
                     len(hosts), np.array([h[0] for h in hosts], np.uint16),
                     np.array([h[1] for h in hosts], np.uint16), np.array([h[2] for h in hosts], np.uint32))


def probe(src_host, src_ip, dst_ip, mask, dport=80):
    p = np.zeros(1, W.PROBE_DTYPE)
    p["src_host"], p["src_ip"], p["dst_ip"], p["allowed_mask"], p["dport"] = src_host, src_ip, dst_ip, mask, dport
    return p


# ---------------------------------------------------------------------------
# independent formulations used as pins
# ---------------------------------------------------------------------------
def _pmask(length):
    return ((0xFFFFFFFF << (32 - length)) & 0xFFFFFFFF) if length else 0


def rule_hits(r, in_port, src, dst, dport):
    m1, m2 = _pmask(int(r["src_len"])), _pmask(int(r["dst_len"]))
    return ((int(r["in_port"]) in (W.ANY_PORT, in_port))
            and (src & m1) == (int(r["src_ip"]) & m1)
            and (dst & m2) == (int(r["dst_ip"]) & m2)
            and int(r["dport_lo"]) <= dport <= int(r["dport_hi"]))


def first_match_sorted(rules, in_port, src, dst, dport):
    """Stable sort by descending priority, then the first rule that hits."""
    order = sorted(range(len(rules)), key=lambda i: (-int(rules[i]["priority"]), i))
    for i in order:
        if rule_hits(rules[i], in_port, src, dst, dport):
            return i
    return -1


def trace_walk(net, pr, cap):
    """Walk ignoring jurisdictions, recording the visited switches, then judge
    the recorded path: the first visited switch outside the mask is a
    violation; otherwise the terminal event decides."""
    pr = pr.reshape(-1)[0] if hasattr(pr, "reshape") else pr
    src_host = int(pr["src_host"])
    if src_host >= net.num_hosts:
        return (W.ST_NOSRC, 0, 0xFFFF), []
    hdr = (int(pr["src_ip"]), int(pr["dst_ip"]), int(pr["dport"]))

    def go(s, p, path):
        if len(path) == cap:
            return path, ("cap",)
        path = path + [s]
        rs = net.rules[net.rule_offs[s]:net.rule_offs[s + 1]]
        i = first_match_sorted(rs, p, *hdr)
        if i < 0 or int(rs[i]["action"]) == W.DROP:
            return path, ("drop",)
        port = int(rs[i]["action"])
        if port >= int(net.port_offs[s + 1] - net.port_offs[s]):
            return path, ("drop",)
        peer = int(net.port_peer[net.port_offs[s] + port])
        if peer < 0:
            return path, ("drop",)
        if peer & W.HOST_BIT:
            return path, ("host", peer & ~W.HOST_BIT)
        return go(peer >> 8, peer & 0xFF, path)

    path, ev = go(int(net.host_switch[src_host]), int(net.host_port[src_host]), [])
    mask = int(pr["allowed_mask"])
    for i, s in enumerate(path):
        reg = int(net.switch_region[s])
        if reg >= 32 or not (mask >> reg) & 1:
            return (W.ST_VIOLATION, i + 1, s), path[: i + 1]
    if ev[0] == "drop":
        return (W.ST_DROP, len(path), path[-1]), path
    if ev[0] == "cap":
        return (W.ST_LOOP, cap, path[-1]), path
    q = ev[1]
    ok = q < net.num_hosts and int(net.host_ip[q]) == hdr[1]
    return ((W.ST_COMPLIANT if ok else W.ST_MISDELIVERED), len(path), path[-1]), path


def trace_walk_constrained(net, pr, cap, forbid, must):
    """trace_walk's recorded path judged against a path constraint: the first
    visited switch outside the jurisdictions or in `forbid` is a violation;
    waypoint bit i is set iff must[i] is among the switches visited before
    the walk ended (a violating switch does not count)."""
    (status, hops, last), path = trace_walk(net, pr, 10 ** 6 if cap is None else cap)
    pr = pr.reshape(-1)[0] if hasattr(pr, "reshape") else pr
    if status == W.ST_NOSRC:
        return (status, hops, last), 0
    full_path, _ = _trace_path(net, pr, cap)
    mask = int(pr["allowed_mask"])
    for i, s in enumerate(full_path):
        reg = int(net.switch_region[s])
        if reg >= 32 or not (mask >> reg) & 1 or s in set(int(x) for x in forbid):
            hit = sum(1 << j for j, m in enumerate(must) if int(m) in set(full_path[:i]))
            return (W.ST_VIOLATION, i + 1, s), hit
    hit = sum(1 << j for j, m in enumerate(must) if int(m) in set(full_path))
    return (status, hops, last), hit


def _trace_path(net, pr, cap):
    """Switches visited ignoring every constraint, up to cap visits."""
    src_host = int(pr["src_host"])
    hdr = (int(pr["src_ip"]), int(pr["dst_ip"]), int(pr["dport"]))
    s, p, path = int(net.host_switch[src_host]), int(net.host_port[src_host]), []
    while len(path) < cap:
        path.append(s)
        rs = net.rules[net.rule_offs[s]:net.rule_offs[s + 1]]
        i = first_match_sorted(rs, p, *hdr)
        if i < 0 or int(rs[i]["action"]) == W.DROP:
            break
        port = int(rs[i]["action"])
        if port >= int(net.port_offs[s + 1] - net.port_offs[s]):
            break
        peer = int(net.port_peer[net.port_offs[s] + port])
        if peer < 0 or peer & W.HOST_BIT:
            break
        s, p = peer >> 8, peer & 0xFF
    return path, None
