// Measured arithmetic peaks of the device the roofline fractions are taken against: fp32 FMA
// throughput (scalar FFMA and the packed two-lane FFMA2) and ex2.approx throughput (the MUFU
// exponential every blend and backward position evaluates).  Each kernel runs independent
// dependency chains in every thread of a grid of several CTAs per SM (the SM count read from
// the device), timed with CUDA events on a private stream after a warm-up launch; the best of
// a few timed launches is reported.  Nothing here changes clocks or any other device setting:
// the numbers are at whatever clock the GPU runs while they are taken.
#include <cuda_runtime.h>

#include <algorithm>

#include "abcd_internal.cuh"

namespace abcd {
namespace {

constexpr int kPeakThreads = 256;
constexpr int kPeakCtasPerSm = 4;        // 32 warps per SM: enough to cover the FMA latency
constexpr int kChains = 16;              // independent chains per thread

// The kernels' sink is never written (the chains never reach the test value); a valid pointer
// all the same: a static device array of this library, so the measurement allocates nothing.
__device__ float g_peak_sink[kPeakThreads];

__global__ void __launch_bounds__(kPeakThreads) ffma_peak_kernel(int iters, float b, float c,
                                                                 float* sink) {
  float a[kChains];
#pragma unroll
  for (int k = 0; k < kChains; ++k) a[k] = (float)(threadIdx.x + k) * 1e-3f;
  for (int i = 0; i < iters; ++i) {
#pragma unroll
    for (int k = 0; k < kChains; ++k) a[k] = fmaf(a[k], b, c);
  }
  float s = 0.f;
#pragma unroll
  for (int k = 0; k < kChains; ++k) s += a[k];
  if (s == 1234.5f) sink[threadIdx.x] = s;     // keeps the chains live; never true in practice
}

__global__ void __launch_bounds__(kPeakThreads) ffma2_peak_kernel(int iters, float b, float c,
                                                                  float* sink) {
  float2 a[kChains];
#pragma unroll
  for (int k = 0; k < kChains; ++k)
    a[k] = make_float2((float)(threadIdx.x + k) * 1e-3f, (float)(threadIdx.x - k) * 1e-3f);
  const float2 bb = make_float2(b, b), cc = make_float2(c, c);
  for (int i = 0; i < iters; ++i) {
#pragma unroll
    for (int k = 0; k < kChains; ++k) a[k] = __ffma2_rn(a[k], bb, cc);
  }
  float s = 0.f;
#pragma unroll
  for (int k = 0; k < kChains; ++k) s += a[k].x + a[k].y;
  if (s == 1234.5f) sink[threadIdx.x] = s;
}

__device__ __forceinline__ float ex2_approx_peak(float x) {
  float y;
  asm volatile("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// x <- 2^(-x): values stay in (0.5, 1]; one MUFU.EX2 and one negation (folded into the
// instruction's operand) per step.
__global__ void __launch_bounds__(kPeakThreads) ex2_peak_kernel(int iters, float* sink) {
  float a[kChains];
#pragma unroll
  for (int k = 0; k < kChains; ++k) a[k] = (float)(threadIdx.x + k) * 1e-4f;
  for (int i = 0; i < iters; ++i) {
#pragma unroll
    for (int k = 0; k < kChains; ++k) a[k] = ex2_approx_peak(-a[k]);
  }
  float s = 0.f;
#pragma unroll
  for (int k = 0; k < kChains; ++k) s += a[k];
  if (s == 1234.5f) sink[threadIdx.x] = s;
}

// Best-of-`reps` milliseconds of one launch of `launch` on `st`.
template <typename F>
cudaError_t time_best(cudaStream_t st, int reps, F launch, double* best_ms) {
  cudaEvent_t e0 = nullptr, e1 = nullptr;
  cudaError_t e = cudaEventCreate(&e0);
  if (e == cudaSuccess) e = cudaEventCreate(&e1);
  double best = 1e30;
  if (e == cudaSuccess) e = launch();                       // warm-up
  for (int r = 0; r < reps && e == cudaSuccess; ++r) {
    e = cudaEventRecord(e0, st);
    if (e == cudaSuccess) e = launch();
    if (e == cudaSuccess) e = cudaEventRecord(e1, st);
    if (e == cudaSuccess) e = cudaEventSynchronize(e1);
    float ms = 0.f;
    if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, e0, e1);
    if (e == cudaSuccess) best = std::min(best, (double)ms);
  }
  if (e0) cudaEventDestroy(e0);
  if (e1) cudaEventDestroy(e1);
  *best_ms = best;
  return e;
}

}  // namespace
}  // namespace abcd

extern "C" abcd_status abcd_measure_alu_peaks(int device, abcd_alu_peaks* out) {
  using namespace abcd;
  if (!out) return ABCD_ERR_INVALID_ARG;
  int prev = 0;
  if (cudaGetDevice(&prev) != cudaSuccess) return ABCD_ERR_CUDA;
  cudaError_t e = cudaSetDevice(device);
  int sms = 0, clk_khz = 0;
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&clk_khz, cudaDevAttrClockRate, device);
  cudaStream_t st = nullptr;
  if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&st, cudaStreamNonBlocking);
  float* sink = nullptr;
  if (e == cudaSuccess) e = cudaGetSymbolAddress((void**)&sink, g_peak_sink);
  const dim3 grid(kPeakCtasPerSm * std::max(sms, 1)), block(kPeakThreads);
  const int iters = 16384;
  double ms_ffma = 0, ms_ffma2 = 0, ms_ex2 = 0;
  const float b = 0.999f, c = 1e-3f;
  if (e == cudaSuccess)
    e = time_best(st, 5, [&] { ffma_peak_kernel<<<grid, block, 0, st>>>(iters, b, c, sink); return cudaGetLastError(); }, &ms_ffma);
  if (e == cudaSuccess)
    e = time_best(st, 5, [&] { ffma2_peak_kernel<<<grid, block, 0, st>>>(iters, b, c, sink); return cudaGetLastError(); }, &ms_ffma2);
  if (e == cudaSuccess)
    e = time_best(st, 5, [&] { ex2_peak_kernel<<<grid, block, 0, st>>>(iters / 4, sink); return cudaGetLastError(); }, &ms_ex2);
  if (st) cudaStreamDestroy(st);
  cudaSetDevice(prev);
  if (e != cudaSuccess) return ABCD_ERR_CUDA;
  const double threads = (double)grid.x * block.x;
  out->sms = sms;
  out->clock_mhz_nominal = clk_khz / 1000.0;
  out->ffma_tflops = threads * iters * kChains * 2.0 / (ms_ffma * 1e-3) / 1e12;
  out->ffma2_tflops = threads * iters * kChains * 4.0 / (ms_ffma2 * 1e-3) / 1e12;
  out->ex2_tops = threads * (iters / 4) * kChains / (ms_ex2 * 1e-3) / 1e12;
  out->ms_ffma = ms_ffma;
  out->ms_ffma2 = ms_ffma2;
  out->ms_ex2 = ms_ex2;
  return ABCD_OK;
}
