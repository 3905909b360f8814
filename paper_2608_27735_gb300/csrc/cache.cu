// Host tier of the layer cache (Section 2: the cached renders of the frozen partitions live
// outside GPU memory and are brought in when a stage composites them; refreshed renders go
// back).  Copies run on the context's two copy streams (host to device, device to host), so
// they overlap the kernels on its compute stream; per-slot events order them:
//   fetch(slot)   waits for the compute work queued before the slot's last release, then
//                 copies and marks the slot ready;
//   wait(slot)    makes the compute stream wait until the slot's fetches and stores are done;
//   release(slot) marks the end of the compute work that reads the slot's device data;
//   store(slot)   copies device data back after the compute work queued so far.
// Host code only: the copies are plain cudaMemcpyAsync calls, one per buffer.
#include <new>

#include "abcd_internal.cuh"

using namespace abcd;

namespace {

// Runs f with the context's device current, restoring the caller's.
template <typename F>
cudaError_t on_device(const abcd_ctx* ctx, F f) {
  int prev = 0;
  cudaGetDevice(&prev);
  cudaError_t e = cudaSetDevice(ctx->device);
  if (e == cudaSuccess) e = f();
  cudaSetDevice(prev);
  return e;
}

cudaError_t ensure_streams(abcd_ctx* ctx) {
  if (ctx->h2d && ctx->d2h && ctx->ev_store) return cudaSuccess;
  return on_device(ctx, [&]() {
    cudaError_t e = cudaSuccess;
    if (!ctx->h2d) e = cudaStreamCreateWithFlags(&ctx->h2d, cudaStreamNonBlocking);
    if (e == cudaSuccess && !ctx->d2h) e = cudaStreamCreateWithFlags(&ctx->d2h, cudaStreamNonBlocking);
    if (e == cudaSuccess && !ctx->ev_store) e = cudaEventCreateWithFlags(&ctx->ev_store, cudaEventDisableTiming);
    return e;
  });
}

cudaError_t slot_event(abcd_ctx* ctx, cudaEvent_t* table, int slot, cudaEvent_t* out) {
  if (!table[slot]) {
    const cudaError_t e = on_device(ctx, [&]() {
      return cudaEventCreateWithFlags(&table[slot], cudaEventDisableTiming);
    });
    if (e != cudaSuccess) return e;
  }
  *out = table[slot];
  return cudaSuccess;
}

bool slot_ok(int slot) { return slot >= 0 && slot < ABCD_MAX_CACHE_SLOTS; }

cudaError_t ensure_tables(abcd_ctx* ctx) {
  if (ctx->cache_ready) return cudaSuccess;
  ctx->cache_ready = new (std::nothrow) cudaEvent_t[ABCD_MAX_CACHE_SLOTS]();
  ctx->cache_released = new (std::nothrow) cudaEvent_t[ABCD_MAX_CACHE_SLOTS]();
  ctx->cache_stored = new (std::nothrow) cudaEvent_t[ABCD_MAX_CACHE_SLOTS]();
  ctx->cache_has_release = new (std::nothrow) unsigned char[ABCD_MAX_CACHE_SLOTS]();
  if (!ctx->cache_ready || !ctx->cache_released || !ctx->cache_stored || !ctx->cache_has_release)
    return cudaErrorMemoryAllocation;
  return cudaSuccess;
}

}  // namespace

namespace abcd {

void cache_destroy(abcd_ctx* ctx) {
  if (ctx->cache_ready) {
    for (int k = 0; k < ABCD_MAX_CACHE_SLOTS; ++k) {
      if (ctx->cache_ready[k]) cudaEventDestroy(ctx->cache_ready[k]);
      if (ctx->cache_released[k]) cudaEventDestroy(ctx->cache_released[k]);
      if (ctx->cache_stored[k]) cudaEventDestroy(ctx->cache_stored[k]);
    }
  }
  delete[] ctx->cache_ready;
  delete[] ctx->cache_released;
  delete[] ctx->cache_stored;
  delete[] ctx->cache_has_release;
  ctx->cache_ready = ctx->cache_released = ctx->cache_stored = nullptr;
  ctx->cache_has_release = nullptr;
  if (ctx->ev_store) cudaEventDestroy(ctx->ev_store);
  if (ctx->h2d) cudaStreamDestroy(ctx->h2d);
  if (ctx->d2h) cudaStreamDestroy(ctx->d2h);
  ctx->h2d = ctx->d2h = nullptr;
  ctx->ev_store = nullptr;
}

}  // namespace abcd

extern "C" abcd_status abcd_cache_fetch(abcd_ctx* ctx, int slot, const void* host_src,
                                        void* dev_dst, size_t bytes) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  if (!slot_ok(slot) || !host_src || !dev_dst || bytes == 0)
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_cache_fetch: bad slot, pointer or size");
  cudaError_t e = ensure_tables(ctx);
  if (e == cudaSuccess) e = ensure_streams(ctx);
  if (e == cudaSuccess && ctx->cache_has_release[slot])
    e = cudaStreamWaitEvent(ctx->h2d, ctx->cache_released[slot], 0);
  if (e == cudaSuccess) e = cudaMemcpyAsync(dev_dst, host_src, bytes, cudaMemcpyHostToDevice, ctx->h2d);
  cudaEvent_t ready = nullptr;
  if (e == cudaSuccess) e = slot_event(ctx, ctx->cache_ready, slot, &ready);
  if (e == cudaSuccess) e = cudaEventRecord(ready, ctx->h2d);
  if (e != cudaSuccess) return fail(ctx, ABCD_ERR_CUDA, "abcd_cache_fetch: %s", cudaGetErrorString(e));
  return ABCD_OK;
}

extern "C" abcd_status abcd_cache_wait(abcd_ctx* ctx, int slot) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  if (!slot_ok(slot)) return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_cache_wait: bad slot %d", slot);
  if (!ctx->cache_ready) return ABCD_OK;                 // nothing fetched or stored yet
  cudaError_t e = cudaSuccess;
  if (ctx->cache_ready[slot]) e = cudaStreamWaitEvent(ctx->stream, ctx->cache_ready[slot], 0);
  if (e == cudaSuccess && ctx->cache_stored[slot])
    e = cudaStreamWaitEvent(ctx->stream, ctx->cache_stored[slot], 0);
  if (e != cudaSuccess) return fail(ctx, ABCD_ERR_CUDA, "abcd_cache_wait: %s", cudaGetErrorString(e));
  return ABCD_OK;
}

extern "C" abcd_status abcd_cache_release(abcd_ctx* ctx, int slot) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  if (!slot_ok(slot)) return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_cache_release: bad slot %d", slot);
  cudaError_t e = ensure_tables(ctx);
  cudaEvent_t rel = nullptr;
  if (e == cudaSuccess) e = slot_event(ctx, ctx->cache_released, slot, &rel);
  if (e == cudaSuccess) e = cudaEventRecord(rel, ctx->stream);
  if (e != cudaSuccess) return fail(ctx, ABCD_ERR_CUDA, "abcd_cache_release: %s", cudaGetErrorString(e));
  ctx->cache_has_release[slot] = 1;
  return ABCD_OK;
}

extern "C" abcd_status abcd_cache_store(abcd_ctx* ctx, int slot, const void* dev_src,
                                        void* host_dst, size_t bytes) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  if (!slot_ok(slot) || !dev_src || !host_dst || bytes == 0)
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_cache_store: bad slot, pointer or size");
  cudaError_t e = ensure_tables(ctx);
  if (e == cudaSuccess) e = ensure_streams(ctx);
  if (e == cudaSuccess) e = cudaEventRecord(ctx->ev_store, ctx->stream);
  if (e == cudaSuccess) e = cudaStreamWaitEvent(ctx->d2h, ctx->ev_store, 0);
  if (e == cudaSuccess) e = cudaMemcpyAsync(host_dst, dev_src, bytes, cudaMemcpyDeviceToHost, ctx->d2h);
  cudaEvent_t stored = nullptr;
  if (e == cudaSuccess) e = slot_event(ctx, ctx->cache_stored, slot, &stored);
  if (e == cudaSuccess) e = cudaEventRecord(stored, ctx->d2h);
  if (e != cudaSuccess) return fail(ctx, ABCD_ERR_CUDA, "abcd_cache_store: %s", cudaGetErrorString(e));
  return ABCD_OK;
}

extern "C" abcd_status abcd_cache_sync(abcd_ctx* ctx) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  cudaError_t e = cudaSuccess;
  if (ctx->h2d) e = cudaStreamSynchronize(ctx->h2d);
  if (e == cudaSuccess && ctx->d2h) e = cudaStreamSynchronize(ctx->d2h);
  if (e != cudaSuccess) return fail(ctx, ABCD_ERR_CUDA, "abcd_cache_sync: %s", cudaGetErrorString(e));
  return ABCD_OK;
}
