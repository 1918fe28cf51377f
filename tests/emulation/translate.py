"""Host C++ copies of the library's kernel sources (tests only).

Rewrites, in copies written to `out_dir`:
  * the CUDA headers -> cuda_host.h (next to this file);
  * each inline-PTX statement -> the same operation in C (cuda_host.h), chosen
    by the instruction it holds and filled with its own output and input
    operands ({o0}, {i0}, ... in order);
  * `extern __shared__ T name[];` -> the launch's dynamic shared memory;
  * `kernel<<<cfg>>>(args);` -> emu::launch(cfg, [&] { kernel(args); }).
Fails if an inline-PTX statement holds no known instruction.
"""
from __future__ import annotations

import os
import re

CSRC = os.path.join(os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__)))),
                    "paper_2505_07531_gb300", "csrc")
FILES = ["qx_common.cuh", "qx_kernels.cuh", "qx_quant.cu", "qx_act8.cu", "qx_select.cu", "qx_q4x.cu",
         "qx_gemv.cu", "qx_gemm.cu", "qx_copy.cu", "qx_api.cu"]

# first match wins: longer instruction names before their prefixes
BY_INSTRUCTION = [
    ("lop3.b32", "{o0} = ({i0} & {i1}) | {i2};"),
    ("prmt.b32", "{o0} = emu_prmt({i0}, {i1}, {i2});"),
    ("mul.hi.u32", "{o0} = (uint32_t)(((uint64_t)({i0}) * (uint64_t)({i1})) >> 32);"),
    ("%%globaltimer", "{o0} = emu_globaltimer();"),
    ("cvt.rn.f16.f64", "{o0} = emu_f64_to_f16({i0});"),
    ("mbarrier.init", "emu_mbar_init({i0}, {i1});"),
    ("mbarrier.arrive.expect_tx", "emu_mbar_arrive_expect_tx({i0}, {i1});"),
    ("mbarrier.arrive.shared", "emu_mbar_arrive({i0});"),
    ("atom.acq_rel.cta.shared::cta.add.u32", "{o0} = emu_atom_add_shared({i0}, {i1});"),
    ("mbarrier.try_wait.parity", "{o0} = emu_mbar_try_wait({i0}, {i1}) ? 1u : 0u;"),
    ("cp.async.bulk.tensor.2d", "{{ const int c_[2] = {{{i3}, {i4}}}; emu_tma_load({i0}, {i1}, {i2}, c_, 2); }}"),
    ("cp.async.bulk.tensor.3d",
     "{{ const int c_[3] = {{{i3}, {i4}, {i5}}}; emu_tma_load({i0}, {i1}, {i2}, c_, 3); }}"),
    ("cp.async.bulk.prefetch.L2", ";"),
    ("ldmatrix.sync.aligned.m8n8.x4", "emu_ldsm({i0}, 4, &{o0}, &{o1}, &{o2}, &{o3});"),
    ("ldmatrix.sync.aligned.m8n8.x2", "emu_ldsm({i0}, 2, &{o0}, &{o1}, nullptr, nullptr);"),
    ("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32",
     "emu_mma16816({o0}, {o1}, {o2}, {o3}, {i0}, {i1}, {i2}, {i3}, {i4}, {i5});"),
    ("ld.global.v4.u32",
     "{{ uint4 t_; std::memcpy(&t_, (const void *)({i0}), 16); {o0} = t_.x; {o1} = t_.y; {o2} = t_.z; {o3} = t_.w; }}"),
    ("ld.global.cg.v4.u32",
     "{{ uint4 t_; std::memcpy(&t_, (const void *)({i0}), 16); {o0} = t_.x; {o1} = t_.y; {o2} = t_.z; {o3} = t_.w; }}"),
    ("bar.sync 1", "emu_named_bar({i0});"),
    ("atom.add.release.gpu.global.u32", "{o0} = std::atomic_ref<uint32_t>(*({i0})).fetch_add({i1});"),
    ("st.release.gpu.global.u32", "std::atomic_ref<uint32_t>(*({i0})).store({i1});"),
    ("red.release.gpu.global.add.u32", "std::atomic_ref<uint32_t>(*({i0})).fetch_add({i1});"),
    ("ld.acquire.gpu.global.u32", "{o0} = std::atomic_ref<uint32_t>(*const_cast<uint32_t *>({i0})).load();"),
    ("ld.global.nc.v4.u32",
     "{{ uint4 t_; std::memcpy(&t_, (const void *)({i0}), 16); {o0} = t_.x; {o1} = t_.y; {o2} = t_.z; {o3} = t_.w; }}"),
    ("ld.shared.v4.u32", "{{ const uint4 t_ = emu_lds128({i0}); {o0} = t_.x; {o1} = t_.y; {o2} = t_.z; {o3} = t_.w; }}"),
    ("ld.shared.u32", "{o0} = emu_lds32({i0});"),
    ("griddepcontrol", ";"),
    ("prefetch.tensormap", ";"),
    ("fence.mbarrier_init", "__threadfence_block();"),
    ("fence.proxy.async", "__threadfence_block();"),
    ("tcgen05.mma.cta_group::1.kind::f16", "emu_mma_f16({i0}, {i1}, {i2}, {i3}, {i4});"),
    ("tcgen05.commit", "emu_mbar_arrive({i0});"),
    ("tcgen05.ld.sync.aligned.32x32b.x32", "emu_tmem_ld({i0}, &{o0}, 32);"),
    ("tcgen05.ld.sync.aligned.32x32b.x16", "emu_tmem_ld({i0}, &{o0}, 16);"),
    ("tcgen05.alloc", "emu_tmem_alloc({i0}, {i1});"),
    ("tcgen05.dealloc", "emu_tmem_dealloc({i0}, {i1});"),
    ("tcgen05.relinquish_alloc_permit", ";"),
    ("tcgen05.wait::", ";"),
    ("tcgen05.fence", "__threadfence_block();"),
]
ASM = re.compile(r"\basm\s*(?:volatile\s*)?\((.*?)\);", re.S)
LAUNCH = re.compile(r"(\w+(?:<[^<>;]*>)?)<<<(.*?)>>>\((.*?)\);", re.S)
CONSTRAINT = re.compile(r'"([=+]?[a-z])"\s*\(')


def operands(body: str):
    """Output and input operand expressions of an asm statement, in order."""
    outs, ins = [], []
    for m in CONSTRAINT.finditer(body):
        depth, j = 1, m.end()
        while depth:
            depth += {"(": 1, ")": -1}.get(body[j], 0)
            j += 1
        (outs if m.group(1)[0] in "=+" else ins).append(body[m.end():j - 1].strip())
    return outs, ins


def _asm(m):
    body = m.group(1)
    for key, tmpl in BY_INSTRUCTION:
        if key in body:
            outs, ins = operands(body)
            return tmpl.format(**{f"o{i}": e for i, e in enumerate(outs)}, **{f"i{i}": e for i, e in enumerate(ins)})
    raise ValueError("untranslated inline PTX: " + m.group(0)[:100])


def translate(src: str) -> str:
    src = src.replace("#include <cuda_fp16.h>", '#include "cuda_host.h"')
    src = src.replace("#include <cuda.h>", '#include "cuda_host.h"').replace("#include <cuda_runtime.h>", "")
    src = re.sub(r"extern __shared__ (?:__align__\(\d+\) )?(\w+) (\w+)\[\];",
                 r"\1 *\2 = reinterpret_cast<\1 *>(emu_dyn_smem());", src)
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


INCLUDE = os.path.join(os.path.dirname(CSRC), "..", "include")
FLAGS = ["-std=c++20", "-O1", "-g", "-fPIC", "-fsanitize=address,undefined", "-fno-sanitize-recover=undefined",
         "-ffp-contract=off", "-Wno-unknown-pragmas", "-Wno-narrowing", "-Wno-psabi", "-pthread"]


def build(gxx: str, out_dir: str, target: str) -> str:
    """Translate, compile in parallel and link with the sanitizers.  target
    "harness": the exact-size buffer executable (harness.cpp); "library": a
    shared library exporting the C ABI (load it with the sanitizer runtimes
    preloaded).  Returns the path built."""
    import concurrent.futures as cf
    import subprocess

    here = os.path.dirname(os.path.abspath(__file__))
    srcs = [os.path.join(out_dir, f[:-3] + ".cpp") for f in FILES if f.endswith(".cu")]
    if not all(os.path.exists(f) for f in srcs):
        srcs = write_all(out_dir)
    if target == "harness":
        srcs.append(os.path.join(here, "harness.cpp"))
    inc = ["-I", out_dir, "-I", here, "-I", os.path.normpath(INCLUDE)]

    def one(src):
        obj = os.path.join(out_dir, os.path.basename(src).rsplit(".", 1)[0] + ".o")
        if os.path.exists(obj) and os.path.getmtime(obj) >= os.path.getmtime(src):
            return obj  # both targets share the objects of one build directory
        r = subprocess.run([gxx, *FLAGS, *inc, "-c", src, "-o", obj], capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(r.stderr[-3000:])
        return obj

    with cf.ThreadPoolExecutor(max_workers=len(srcs)) as ex:
        objs = list(ex.map(one, srcs))
    out = os.path.join(out_dir, "harness" if target == "harness" else "libqx_emulated.so")
    link = [gxx, *FLAGS, *objs, "-o", out] + (["-shared"] if target == "library" else [])
    r = subprocess.run(link, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(r.stderr[-3000:])
    return out
