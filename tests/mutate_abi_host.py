"""Mutation check of the C ABI's host-side checks (not collected by pytest; run
by hand):

    python tests/mutate_abi_host.py FIRST_LINE LAST_LINE

Plants one change at a time (a comparison, + / -, || / &&, == / != swapped, a
size limit or constant moved by one) in the given line range of
paper_2606_03075_gb300/csrc/api.cu -- the descriptor validation, budget
totals and capacities sit in its make_problem .. retained_rows -- inside a
temporary copy of the repository, builds the library there (nvcc, about 20 s
per mutant) and runs tests/test_abi.py against it.  Prints every mutant that
builds and that no test catches."""
import os
import re
import shutil
import subprocess
import sys
import tempfile
import time

REPO = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
REL = "paper_2606_03075_gb300/csrc/api.cu"
LO, HI = int(sys.argv[1]), int(sys.argv[2])     # 1-based inclusive line range

OPS = [(r" < ", " <= "), (r" <= ", " < "), (r" > ", " >= "), (r" >= ", " > "),
       (r" \+ ", " - "), (r" - ", " + "), (r" \|\| ", " && "), (r" && ", " || "),
       (r" != ", " == "), (r" == ", " != "), (r"\b32768\b", "32767"), (r"\b65535\b", "65534"),
       (r"\b0\.5\b", "0.75"), (r"\b1\.0\b", "0.9"), (r"\b64\b", "65"), (r"\b128\b", "129"),
       (r"\b1024\b", "1023"), (r"\(1LL << 31\)", "(1LL << 30)")]


def mutants(lines):
    for i in range(LO - 1, HI):
        line = lines[i]
        code = line.split("//")[0]
        if '"' in code:          # leave format strings alone
            code = code.split('"')[0]
        for pat, rep in OPS:
            for m in re.finditer(pat, code):
                new = line[:m.start()] + rep + line[m.end():]
                yield i, pat, new


def main():
    work = tempfile.mkdtemp(prefix="tgvkv_cmut_")
    try:
        for d in ("tests", "oracle", "paper_2606_03075_gb300", "include"):
            shutil.copytree(os.path.join(REPO, d), os.path.join(work, d),
                            ignore=shutil.ignore_patterns("__pycache__", "_build*", "*.so"))
        shutil.copy(os.path.join(REPO, "pytest.ini"), work)
        src = open(os.path.join(REPO, REL)).read().split("\n")
        ms = list(mutants(src))
        print(f"{len(ms)} mutants", flush=True)
        survived, t0 = 0, time.time()
        for i, pat, new in ms:
            lines = list(src)
            lines[i] = new
            open(os.path.join(work, REL), "w").write("\n".join(lines))
            b = subprocess.run([sys.executable, "-c",
                                "from paper_2606_03075_gb300 import build; build.build(force=True)"],
                               cwd=work, capture_output=True, text=True, timeout=900)
            if b.returncode != 0:
                continue          # does not compile: not a mutant
            r = subprocess.run([sys.executable, "-m", "pytest", "tests/test_abi.py", "-x", "-q",
                                "-p", "no:cacheprovider"], cwd=work, capture_output=True,
                               text=True, timeout=900)
            if r.returncode == 0:
                survived += 1
                print(f"survived: line {i + 1}: {pat!r}: {new.strip()}", flush=True)
        print(f"survived {survived} of {len(ms)}, {time.time() - t0:.0f} s", flush=True)
    finally:
        shutil.rmtree(work, ignore_errors=True)


if __name__ == "__main__":
    main()
