"""Host C++ copies of the library's simple kernel sources (tests only).

Rewrites, in copies written to `out_dir`:
  * the CUDA headers -> cuda_host.h (next to this file);
  * each inline-PTX statement these sources use -> the same operation in C;
  * `extern __shared__ T name[];` -> the launch's dynamic shared memory;
  * `kernel<<<cfg>>>(args);` -> emu::launch(cfg, [&] { kernel(args); }).
Fails if any inline PTX is left untranslated.
"""
from __future__ import annotations

import os
import re

CSRC = os.path.join(os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__)))),
                    "paper_2505_07531_gb300", "csrc")
FILES = ["qx_common.cuh", "qx_kernels.cuh", "qx_quant.cu", "qx_act8.cu", "qx_select.cu", "qx_q4x.cu"]

# inline PTX -> C, as written in the sources
PTX = [
    (r'asm\("lop3\.b32 %0, %1, %2, %3, 0xEA;" : "=r"\(d\) : "r"\(a\), "r"\(b\), "r"\(c\)\);', "d = (a & b) | c;"),
    (r'asm\("prmt\.b32 %0, %1, %2, %3;" : "=r"\(d\) : "r"\(a\), "r"\(b\), "r"\(sel\)\);', "d = emu_prmt(a, b, sel);"),
    (r'asm\("mul\.hi\.u32 %0, %1, %2;" : "=r"\(d\) : "r"\(x\), "r"\(1u << \(32 - n\)\)\);',
     "d = (uint32_t)(((uint64_t)x * (uint64_t)(1u << (32 - n))) >> 32);"),
    (r'asm volatile\("mov\.u64 %0, %%globaltimer;" : "=l"\(t\)\);', "t = emu_globaltimer();"),
    (r'asm\("cvt\.rn\.f16\.f64 %0, %1;" : "=h"\(h\) : "d"\(x\)\);', "h = emu_f64_to_f16(x);"),
]
LAUNCH = re.compile(r"(\w+(?:<[^<>;]*>)?)<<<(.*?)>>>\((.*?)\);", re.S)


def translate(src: str) -> str:
    src = src.replace("#include <cuda_fp16.h>", '#include "cuda_host.h"')
    src = src.replace("#include <cuda.h>", '#include "cuda_host.h"').replace("#include <cuda_runtime.h>", "")
    src = re.sub(r"extern __shared__ (\w+) (\w+)\[\];", r"\1 *\2 = reinterpret_cast<\1 *>(emu_dyn_smem());", src)
    for pat, rep in PTX:
        src = re.sub(pat, rep, src)
    if re.search(r"\basm\b", src):
        raise ValueError("untranslated inline PTX")
    return LAUNCH.sub(lambda m: f"emu::launch(emu::Cfg{{{m.group(2)}}}, [&] {{ {m.group(1)}({m.group(3)}); }});", src)


def write_all(out_dir: str) -> list:
    """Translate FILES into out_dir; returns the .cpp paths to compile."""
    os.makedirs(out_dir, exist_ok=True)
    cpps = []
    for f in FILES:
        with open(os.path.join(CSRC, f)) as fh:
            text = translate(fh.read())
        name = f[:-3] + ".cpp" if f.endswith(".cu") else f
        with open(os.path.join(out_dir, name), "w") as fh:
            fh.write(text)
        if name.endswith(".cpp"):
            cpps.append(os.path.join(out_dir, name))
    return cpps
