// peak_probe.cu -- a measurement of the integer issue rate the DP kernel is
// bound by.  The DP (dp_eval.cu) is a min-max recurrence over 32-bit order
// keys: its instructions are unsigned min and max, compares with selects,
// and small integer adds on indices.  This kernel runs exactly that mix on
// independent chains in every thread of a full-occupancy grid, so that its
// rate (operations per second, and per SM per clock once the caller divides
// by the SM clock it sampled) is the attainable ceiling for such code on the
// GPU at hand.  It allocates nothing: the one result word that keeps the
// chains live goes to a file-scope device variable.
#include "e2ga_internal.cuh"

namespace {

constexpr int kChains = 8;               // independent dependency chains per thread
constexpr int kThreads = 256;

static __device__ unsigned g_probe_sink;

// kind 0: min.u32 / max.u32 alternating (2 ops per chain and step)
// kind 1: add.u32 (2 ops per chain and step)
// kind 2: the DP's mix: min, max, compare + select, add (5 ops per chain and step)
template <int KIND>
__global__ void __launch_bounds__(kThreads) int_probe_kernel(int iters, unsigned seed)
{
    unsigned a[kChains], b[kChains];
#pragma unroll
    for (int c = 0; c < kChains; ++c) {
        a[c] = seed ^ (threadIdx.x * 2654435761u) ^ (c * 40503u);
        b[c] = seed + blockIdx.x * 97u + (unsigned)c;
    }
    for (int it = 0; it < iters; ++it) {
#pragma unroll
        for (int c = 0; c < kChains; ++c) {
            if (KIND == 0) {
                asm volatile("min.u32 %0, %0, %1;" : "+r"(a[c]) : "r"(b[c]));
                asm volatile("max.u32 %0, %0, %1;" : "+r"(b[c]) : "r"(a[c]));
            } else if (KIND == 1) {
                asm volatile("add.u32 %0, %0, %1;" : "+r"(a[c]) : "r"(b[c]));
                asm volatile("add.u32 %0, %0, %1;" : "+r"(b[c]) : "r"(a[c]));
            } else {
                asm volatile(
                    "{\n\t.reg .pred p;\n\t"
                    "min.u32 %0, %0, %1;\n\t"
                    "max.u32 %1, %1, %0;\n\t"
                    "setp.ge.u32 p, %0, %1;\n\t"
                    "selp.u32 %0, %1, %0, p;\n\t"
                    "add.u32 %1, %1, 1;\n\t}"
                    : "+r"(a[c]), "+r"(b[c]));
            }
        }
    }
    unsigned x = 0;
#pragma unroll
    for (int c = 0; c < kChains; ++c) x ^= a[c] ^ b[c];
    if (x == 0x9E3779B9u) g_probe_sink = x;       // keeps every chain live; practically never taken
}

}  // namespace

extern "C" int e2_probe_int_rate(int32_t kind, int32_t iters, void *stream, double *ops_per_launch,
                                 float *ms_out)
{
    if ((kind < 0 || kind > 2) || iters < 1 || iters > (1 << 24) || !ops_per_launch || !ms_out) return E2_EINVAL;
    int dev = 0, sms = 0, per_sm = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return E2_ECUDA;
    const void *fn = kind == 0 ? reinterpret_cast<const void *>(int_probe_kernel<0>)
                   : kind == 1 ? reinterpret_cast<const void *>(int_probe_kernel<1>)
                               : reinterpret_cast<const void *>(int_probe_kernel<2>);
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, kThreads, 0) != cudaSuccess || per_sm < 1)
        return E2_ECUDA;
    const unsigned blocks = (unsigned)(per_sm * sms);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaEvent_t e0 = nullptr, e1 = nullptr;
    if (cudaEventCreate(&e0) != cudaSuccess || cudaEventCreate(&e1) != cudaSuccess) {
        if (e0) cudaEventDestroy(e0);
        return E2_ECUDA;
    }
    cudaError_t e = cudaEventRecord(e0, s);
    if (e == cudaSuccess) {
        if (kind == 0) int_probe_kernel<0><<<blocks, kThreads, 0, s>>>(iters, 12345u);
        else if (kind == 1) int_probe_kernel<1><<<blocks, kThreads, 0, s>>>(iters, 12345u);
        else int_probe_kernel<2><<<blocks, kThreads, 0, s>>>(iters, 12345u);
        e = cudaGetLastError();
    }
    if (e == cudaSuccess) e = cudaEventRecord(e1, s);
    if (e == cudaSuccess) e = cudaEventSynchronize(e1);
    float ms = 0.0f;
    if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, e0, e1);
    cudaEventDestroy(e0);
    cudaEventDestroy(e1);
    if (e != cudaSuccess) return E2_ECUDA;
    const double per_step = kind == 2 ? 5.0 : 2.0;
    *ops_per_launch = (double)blocks * kThreads * (double)iters * kChains * per_step;
    *ms_out = ms;
    return E2_OK;
}
