"""Reader for the golden fixtures under tests/golden (format in its README)."""
import os

import workloads

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def load(name):
    """Returns (batch, expectations); expectations are (mode, dep index, values)."""
    names_loop = {"root": 0}
    names_instr = {}
    b = None
    deps = {}
    expects = []
    with open(os.path.join(GOLDEN, name)) as f:
        for raw in f:
            line = raw.split("#", 1)[0].split()
            if not line:
                continue
            kw, args = line[0], line[1:]
            if kw == "engines":
                b = workloads.ProgramBuilder(int(args[0]))
            elif kw == "loop":
                names_loop[args[0]] = b.loop(names_loop[args[1]], int(args[2]),
                                             [int(t) for t in args[3:]])
            elif kw == "instr":
                lat = int(args[4]) if len(args) > 4 else 1
                names_instr[args[0]] = b.instr(names_loop[args[1]], int(args[2]), int(args[3]), lat)
            elif kw == "dep":
                deps[(args[0], args[1])] = b.dep(names_instr[args[0]], names_instr[args[1]],
                                                 int(args[2]))
            elif kw == "expect":
                expects.append((args[0], deps[(args[1], args[2])], [int(v) for v in args[3:]]))
            else:
                raise ValueError(f"{name}: unknown statement {kw}")
    return b.batch(), expects


def all_names():
    return sorted(n for n in os.listdir(GOLDEN) if n.endswith(".txt"))
