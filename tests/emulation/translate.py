"""Host C++ copies of the library's kernel sources that use no tensor-core
instructions (tests only).

Rewrites, in copies written to `out_dir`:
  * the CUDA headers -> cuda_host.h (next to this file);
  * each inline-PTX statement -> the same operation in C (cuda_host.h), chosen by
    the instruction it holds; the operand names are those of the sources;
  * `extern __shared__ T name[];` -> the launch's dynamic shared memory;
  * `kernel<<<cfg>>>(args);` -> emu::launch(cfg, [&] { kernel(args); }).
Fails if any inline PTX is left untranslated.
"""
from __future__ import annotations

import os
import re

CSRC = os.path.join(os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__)))),
                    "paper_2505_07531_gb300", "csrc")
FILES = ["qx_common.cuh", "qx_kernels.cuh", "qx_quant.cu", "qx_act8.cu", "qx_select.cu", "qx_q4x.cu",
         "qx_gemv.cu"]

# instruction -> C statement, in the operand names the sources use
BY_INSTRUCTION = [
    ("lop3.b32", "d = (a & b) | c;"),
    ("prmt.b32", "d = emu_prmt(a, b, sel);"),
    ("mul.hi.u32", "d = (uint32_t)(((uint64_t)x * (uint64_t)(1u << (32 - n))) >> 32);"),
    ("%%globaltimer", "t = emu_globaltimer();"),
    ("cvt.rn.f16.f64", "h = emu_f64_to_f16(x);"),
    ("mbarrier.init", "emu_mbar_init(b, count);"),
    ("mbarrier.arrive.expect_tx", "emu_mbar_arrive_expect_tx(b, bytes);"),
    ("mbarrier.try_wait.parity", "ok = emu_mbar_try_wait(b, parity) ? 1u : 0u;"),
    ("cp.async.bulk.tensor.2d", "{ const int c_[2] = {x, y}; emu_tma_load(dst, map, bar, c_, 2); }"),
    ("cp.async.bulk.tensor.3d", "{ const int c_[3] = {x, y, z}; emu_tma_load(dst, map, bar, c_, 3); }"),
    ("cp.async.bulk.prefetch.L2", "(void)p; (void)bytes;"),
    ("ld.shared.v4.u32", "v = emu_lds128(a);"),
    ("griddepcontrol", ";"),
    ("prefetch.tensormap", ";"),
    ("fence.mbarrier_init", "__threadfence_block();"),
    ("fence.proxy.async", "__threadfence_block();"),
]
ASM = re.compile(r"\basm\s*(?:volatile\s*)?\((.*?)\);", re.S)
LAUNCH = re.compile(r"(\w+(?:<[^<>;]*>)?)<<<(.*?)>>>\((.*?)\);", re.S)


def _asm(m):
    for key, rep in BY_INSTRUCTION:
        if key in m.group(1):
            return rep
    raise ValueError("untranslated inline PTX: " + m.group(0)[:80])


def translate(src: str) -> str:
    src = src.replace("#include <cuda_fp16.h>", '#include "cuda_host.h"')
    src = src.replace("#include <cuda.h>", '#include "cuda_host.h"').replace("#include <cuda_runtime.h>", "")
    src = re.sub(r"extern __shared__ (\w+) (\w+)\[\];", r"\1 *\2 = reinterpret_cast<\1 *>(emu_dyn_smem());", src)
    src = ASM.sub(_asm, src)
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
