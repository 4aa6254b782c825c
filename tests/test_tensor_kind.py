"""Why the batched interval pass multiplies bf16 operands on the tensor cores
rather than int8 ones.

The batched pass computes the exact Int8 dot products <z_q, z_v> of
Sec. 2.3.1 for many queries at once.  Codes are integers in [-127, 127],
exact in bf16, and every partial sum stays below 2^24, so an fp32 accumulator
holds the exact integer either way; what decides the operand type is which
tensor-core path is fast on sm_103a.

  * CPU: ptxas accepts tcgen05.mma with kind::f16 for sm_103a and rejects
    kind::i8 (the integer MMA kind of the fifth-generation tensor cores is
    not offered on this target).
  * GPU: the remaining integer tensor path, the legacy warp-level
    mma.sync m16n8k32 s8, against mma.sync m16n8k16 f16 and the dp4a ALU
    instruction, each as independent accumulator chains with no memory
    traffic (run with -s to see the rates).  f16 must run well above s8.
"""
import os
import re
import shutil
import subprocess

import pytest

NVCC = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"

_MMA_KIND = r"""
#include <cstdint>
__global__ void k(uint32_t tmem, uint64_t da, uint64_t db, uint32_t idesc, int acc) {
    asm volatile("{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\n"
                 "tcgen05.mma.cta_group::1.kind::KIND [%0], %1, %2, %3, p;\n}\n"
                 :: "r"(tmem), "l"(da), "l"(db), "r"(idesc), "r"(acc));
}
"""

_RATES = r"""
#include <cstdio>
#include <cuda_runtime.h>
constexpr int kIter = 4096;
__global__ void s8(int* out, int seed) {
    int d[4][4] = {};
    int a0 = seed + threadIdx.x, a1 = a0 * 3, a2 = a0 ^ 0x5a5a5a5a, a3 = a0 + 7;
    int b0 = a0 * 5, b1 = a0 ^ 0x1234;
    for (int it = 0; it < kIter; ++it) {
#pragma unroll
        for (int c = 0; c < 4; ++c)
            asm volatile("mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 "
                         "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
                         : "+r"(d[c][0]), "+r"(d[c][1]), "+r"(d[c][2]), "+r"(d[c][3])
                         : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
    }
    int s = 0;
    for (int c = 0; c < 4; ++c) s += d[c][0] + d[c][1] + d[c][2] + d[c][3];
    if (s == 0x7fffffff) out[0] = s;
}
__global__ void f16(float* out, int seed) {
    float d[4][4] = {};
    unsigned a0 = 0x3c003c00u + seed, a1 = a0, a2 = a0, a3 = a0, b0 = a0, b1 = a0;
    for (int it = 0; it < kIter; ++it) {
#pragma unroll
        for (int c = 0; c < 4; ++c)
            asm volatile("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 "
                         "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
                         : "+f"(d[c][0]), "+f"(d[c][1]), "+f"(d[c][2]), "+f"(d[c][3])
                         : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
    }
    float s = 0;
    for (int c = 0; c < 4; ++c) s += d[c][0] + d[c][1] + d[c][2] + d[c][3];
    if (s == 12345.0f) out[0] = s;
}
__global__ void dp4a(int* out, int seed) {
    int d[8] = {};
    int a = seed + threadIdx.x, b = a * 7;
    for (int it = 0; it < kIter; ++it) {
#pragma unroll
        for (int c = 0; c < 8; ++c) d[c] = __dp4a(a + c, b, d[c]);
    }
    int s = 0;
    for (int c = 0; c < 8; ++c) s += d[c];
    if (s == 0x7fffffff) out[0] = s;
}
int main() {
    int* o = nullptr;
    if (cudaMalloc(&o, 64) != cudaSuccess) return 1;
    int sms = 0;
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, 0);
    const int blocks = sms * 8, threads = 128, warps = blocks * threads / 32;
    cudaEvent_t e0, e1;
    cudaEventCreate(&e0);
    cudaEventCreate(&e1);
    float ms = 0.f;
    for (int rep = 0; rep < 3; ++rep) {   // the last repetition is reported
        cudaEventRecord(e0);
        s8<<<blocks, threads>>>(o, rep);
        cudaEventRecord(e1);
        cudaEventSynchronize(e1);
        cudaEventElapsedTime(&ms, e0, e1);
        const double s8_ops = 2.0 * warps * kIter * 4 * 16 * 8 * 32 / (ms * 1e-3);
        cudaEventRecord(e0);
        f16<<<blocks, threads>>>(reinterpret_cast<float*>(o), rep);
        cudaEventRecord(e1);
        cudaEventSynchronize(e1);
        cudaEventElapsedTime(&ms, e0, e1);
        const double f16_ops = 2.0 * warps * kIter * 4 * 16 * 8 * 16 / (ms * 1e-3);
        cudaEventRecord(e0);
        dp4a<<<blocks, threads>>>(o, rep);
        cudaEventRecord(e1);
        cudaEventSynchronize(e1);
        cudaEventElapsedTime(&ms, e0, e1);
        const double dp4a_ops = 2.0 * blocks * threads * kIter * 8 * 4 / (ms * 1e-3);
        if (rep == 2)
            printf("s8_mma_sync_tops %.1f\nf16_mma_sync_tflops %.1f\ndp4a_tops %.1f\n",
                   s8_ops / 1e12, f16_ops / 1e12, dp4a_ops / 1e12);
    }
    const cudaError_t e = cudaGetLastError();
    cudaFree(o);
    return e != cudaSuccess;
}
"""


def _compile(tmp_path, name, src, extra=()):
    path = tmp_path / f"{name}.cu"
    path.write_text(src)
    return subprocess.run([NVCC, "-gencode", "arch=compute_103a,code=sm_103a", *extra,
                           str(path), "-o", str(tmp_path / name)],
                          capture_output=True, text=True, timeout=300)


@pytest.mark.skipif(not os.path.exists(NVCC), reason="nvcc not available")
def test_sm_103a_offers_tcgen05_f16_but_not_i8(tmp_path):
    f16 = _compile(tmp_path, "kind_f16", _MMA_KIND.replace("KIND", "f16"), ("-c",))
    assert f16.returncode == 0, f16.stderr
    i8 = _compile(tmp_path, "kind_i8", _MMA_KIND.replace("KIND", "i8"), ("-c",))
    assert i8.returncode != 0
    assert "ptxas" in i8.stderr and "i8" in i8.stderr, i8.stderr


@pytest.mark.gpu
def test_legacy_int8_tensor_path_runs_below_f16(tmp_path):
    built = _compile(tmp_path, "rates", _RATES, ("-O3",))
    assert built.returncode == 0, built.stderr
    run = subprocess.run([str(tmp_path / "rates")], capture_output=True, text=True, timeout=300)
    assert run.returncode == 0, run.stderr
    rates = dict((k, float(v)) for k, v in re.findall(r"(\w+) ([0-9.]+)", run.stdout))
    print(rates)
    assert rates["f16_mma_sync_tflops"] > 2.0 * rates["s8_mma_sync_tops"]
