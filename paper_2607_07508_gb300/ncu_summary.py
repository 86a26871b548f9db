"""Summarise an ncu launch list (--metrics gpu__time_duration.sum --csv) into
per-kernel launch counts, total time and share. Usage:
    python -m paper_2607_07508_gb300.ncu_summary launches.csv [name-filter ...]"""
import collections
import csv
import re
import io
import sys


def summarize(path, only=None):
    text = open(path).read().splitlines()
    start = next(i for i, l in enumerate(text) if l.startswith('"ID"'))
    rows = list(csv.DictReader(io.StringIO("\n".join(text[start:]))))
    agg = collections.OrderedDict()
    scale = {"nsecond": 1e-6, "ns": 1e-6, "usecond": 1e-3, "us": 1e-3, "msecond": 1.0, "ms": 1.0, "second": 1e3, "s": 1e3}
    for r in rows:
        if r.get("Metric Name") != "gpu__time_duration.sum":
            continue
        name = r["Kernel Name"]
        short = name.split("(")[0].replace("void ", "")
        if "sao::" in short:
            short = short.split("::")[-1]
        mt = re.match(r"tc_gemm_kernel<(\d), (\d), (\d)(?:, (\d))?(?:, (\d))?>", short)
        if mt:
            label = {("0", "0", "0"): "tc_gemm<softmax> (logits lse fwd)",
                     ("4", "0", "0"): "tc_gemm<softmax+store> (logits lse fwd, stores bf16 e)",
                     ("1", "0", "0"): "tc_gemm<dlogits> (bwd recompute + dZ)",
                     ("3", "0", "1"): "tc_gemm<store bf16> (dH = row-scaled e W, or dZ W)",
                     ("2", "0", "1"): "tc_gemm<store f32> (dH accumulate)",
                     ("2", "1", "1"): "tc_gemm<store f32> (dW = e^T (s H), or dZ^T H)"}.get(mt.groups()[:3], short)
            if mt.group(4) == "2":
                label += ", 2 M tiles per CTA tile"
            if mt.group(5) == "2":
                label += ", CTA pairs"
            short = label
        if only and not any(o in name for o in only):
            continue
        v = float(r["Metric Value"].replace(",", "")) * scale[r["Metric Unit"]]
        a = agg.setdefault(short, [0, 0.0])
        a[0] += 1
        a[1] += v
    tot = sum(v[1] for v in agg.values())
    out = [f"{'launches':>8} {'total ms':>10} {'share':>7}  kernel"]
    for k, (n, t) in sorted(agg.items(), key=lambda kv: -kv[1][1]):
        out.append(f"{n:8d} {t:10.3f} {100 * t / tot:6.2f}%  {k}")
    out.append(f"total {tot:.3f} ms over {sum(v[0] for v in agg.values())} launches")
    return "\n".join(out)


if __name__ == "__main__":
    print(summarize(sys.argv[1], sys.argv[2:] or None))
