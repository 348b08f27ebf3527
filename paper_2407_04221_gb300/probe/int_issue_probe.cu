// Integer-issue probe: 32-bit integer instructions per SM per clock on the
// current GPU, for the ALU roofline of the benchmark.  Eight independent
// dependency chains per thread, 8 CTAs of 256 threads per SM; per-CTA cycles
// come from clock64, so the rate per clock does not depend on the SM clock.
// A stand-alone measurement program (`bench.py --int-probe` builds and runs
// it): not part of libautoverse.so, and nothing in the library calls it.
#include <cstdio>
#include <cstdint>
#include <cuda_runtime.h>
template <int KIND>
__global__ void __launch_bounds__(256) probe(uint32_t *out, long long *cyc, uint32_t seed, int iters)
{
    uint32_t x0 = threadIdx.x ^ seed, x1 = x0 * 3u + 1u, x2 = x0 * 5u + 2u, x3 = x0 * 7u + 3u;
    uint32_t x4 = x0 * 11u + 4u, x5 = x0 * 13u + 5u, x6 = x0 * 17u + 6u, x7 = x0 * 19u + 7u;
    const uint32_t k = seed * 2654435761u;
    __syncthreads();
    long long t0 = clock64();
    for (int i = 0; i < iters; ++i) {
#pragma unroll
        for (int u = 0; u < 16; ++u) {
            if (KIND == 0) {  // LOP3: x ^ (y & k)
                x0 ^= x1 & k; x1 ^= x2 & k; x2 ^= x3 & k; x3 ^= x4 & k;
                x4 ^= x5 & k; x5 ^= x6 & k; x6 ^= x7 & k; x7 ^= x0 & k;
            } else if (KIND == 1) {  // IADD3: x + y + k
                x0 += x1 + k; x1 += x2 + k; x2 += x3 + k; x3 += x4 + k;
                x4 += x5 + k; x5 += x6 + k; x6 += x7 + k; x7 += x0 + k;
            } else if (KIND == 2) {  // SHF funnel
                x0 = __funnelshift_r(x0, x1, k); x1 = __funnelshift_r(x1, x2, k);
                x2 = __funnelshift_r(x2, x3, k); x3 = __funnelshift_r(x3, x4, k);
                x4 = __funnelshift_r(x4, x5, k); x5 = __funnelshift_r(x5, x6, k);
                x6 = __funnelshift_r(x6, x7, k); x7 = __funnelshift_r(x7, x0, k);
            } else {  // IMAD: x * y + k
                x0 = x0 * x1 + k; x1 = x1 * x2 + k; x2 = x2 * x3 + k; x3 = x3 * x4 + k;
                x4 = x4 * x5 + k; x5 = x5 * x6 + k; x6 = x6 * x7 + k; x7 = x7 * x0 + k;
            }
        }
    }
    long long t1 = clock64();
    out[blockIdx.x * blockDim.x + threadIdx.x] = x0 ^ x1 ^ x2 ^ x3 ^ x4 ^ x5 ^ x6 ^ x7;
    if (threadIdx.x == 0) cyc[blockIdx.x] = t1 - t0;
}
template <int KIND> void run(const char *name, int blocks, uint32_t *out, long long *cyc)
{
    const int iters = 4000;
    probe<KIND><<<blocks, 256>>>(out, cyc, 12345u, 10);
    cudaEvent_t a, b; cudaEventCreate(&a); cudaEventCreate(&b);
    cudaEventRecord(a);
    probe<KIND><<<blocks, 256>>>(out, cyc, 12345u, iters);
    cudaEventRecord(b);
    cudaEventSynchronize(b);
    float ms; cudaEventElapsedTime(&ms, a, b);
    long long *h = new long long[blocks];
    cudaMemcpy(h, cyc, sizeof(long long) * blocks, cudaMemcpyDeviceToHost);
    double mc = 0; for (int i = 0; i < blocks; ++i) mc += h[i]; mc /= blocks;
    double ops = (double)blocks * 256 * iters * 16 * 8;
    int per_sm = blocks / 152;
    double ops_per_clk_sm = (double)per_sm * 256 * iters * 16 * 8 / mc;
    printf("%s: %.3f ms, %.1f Gop/s, block cycles %.0f, ops/clk/SM %.1f, implied MHz %.0f\n", name, ms,
           ops / ms / 1e6, mc, ops_per_clk_sm, mc / (ms * 1e3));
    delete[] h;
}
int main()
{
    int dev = 0; cudaDeviceProp p; cudaGetDeviceProperties(&p, dev);
    printf("%s SMs=%d\n", p.name, p.multiProcessorCount);
    const int blocks = 152 * 8;
    uint32_t *out; long long *cyc;
    cudaMalloc(&out, sizeof(uint32_t) * blocks * 256);
    cudaMalloc(&cyc, sizeof(long long) * blocks);
    run<0>("LOP3 ", blocks, out, cyc);
    run<1>("IADD3", blocks, out, cyc);
    run<2>("SHF  ", blocks, out, cyc);
    run<3>("IMAD ", blocks, out, cyc);
    cudaError_t e = cudaDeviceSynchronize();
    printf("status %s\n", cudaGetErrorString(e));
    return e != cudaSuccess;
}
