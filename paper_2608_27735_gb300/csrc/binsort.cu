// K3 (tile binning) and K4 (sort + tile ranges) of the ABCD active-block step.
//
// What is computed (3DGS binning, Section 1 of the paper by citation): every visible Gaussian
// is listed in each 16x16 tile met by its square [u-r, u+r] x [v-r, v+r]; each tile's list
// is ordered front to back by (fp32 depth, Gaussian id).
//
// How (GB300 design, different from sorting 64-bit (tile | depth) keys):
//   1. stable LSD radix sort of the n Gaussians by the 32 depth bits (keys of culled
//      Gaussians are all ones, so they sort last and emit nothing);
//   2. exclusive scan of tiles_touched in that order; K = total pairs;
//   3. emission of (tile << 32 | id) items in depth order;
//   4. stable LSD radix sort of the K items on the tile bits only (ceil(log2 n_tiles) <= 16
//      bits: two 8-bit passes), which keeps depth order inside each tile;
//   5. tile ranges from the run boundaries, ids written out.
// Radix passes are reduce-then-scan (per-block digit counts, one global scan, stable
// scatter): no inter-block waits, so nothing can spin.  Counts that live on the device (K)
// are read by the kernels themselves; grids are fixed, so the step has no host sync.
#include <algorithm>

#include "abcd_internal.cuh"

namespace abcd {
namespace {

typedef unsigned long long u64;

__device__ __forceinline__ long long dev_count(long long n_static, const long long* n_dev,
                                               long long cap) {
  if (!n_dev) return n_static;
  const long long k = *n_dev;
  return (k < 0 || k > cap) ? 0 : k;       // overflow: nothing valid to process
}

__device__ __forceinline__ void block_range(long long n, int G, long long* lo, long long* hi) {
  const long long chunk = (n + G - 1) / G;
  *lo = min(n, (long long)blockIdx.x * chunk);
  *hi = min(n, *lo + chunk);
}

// ---- depth keys: (bits(depth) << 32) | id, all ones for culled Gaussians
__global__ void depth_keys_kernel(const float* depth, const int* radius, int n, u64* items) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const unsigned key = radius[i] > 0 ? __float_as_uint(depth[i]) : 0xFFFFFFFFu;
  items[i] = ((u64)key << 32) | (unsigned)i;
}

// ---- radix pass, step 1: per-block digit counts hist[d * G + b]
__global__ void __launch_bounds__(256)
radix_hist_kernel(const u64* in, long long n_static, const long long* n_dev, long long cap,
                  int shift, unsigned* hist, int G) {
  __shared__ unsigned h[kRadixBins];
  for (int d = threadIdx.x; d < kRadixBins; d += blockDim.x) h[d] = 0;
  __syncthreads();
  const long long n = dev_count(n_static, n_dev, cap);
  long long lo, hi;
  block_range(n, G, &lo, &hi);
  for (long long i = lo + threadIdx.x; i < hi; i += blockDim.x)
    atomicAdd(&h[(unsigned)(in[i] >> shift) & (kRadixBins - 1)], 1u);
  __syncthreads();
  for (int d = threadIdx.x; d < kRadixBins; d += blockDim.x) hist[d * G + blockIdx.x] = h[d];
}

// Exclusive scan of a block of per-thread sums (1024 threads).
__device__ __forceinline__ unsigned long long block_exclusive_scan(unsigned long long v,
                                                                   unsigned long long* total) {
  __shared__ unsigned long long warp_sums[32];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  unsigned long long x = v;
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned long long y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_sums[wid] = x;
  __syncthreads();
  if (wid == 0) {
    const int nw = blockDim.x >> 5;
    unsigned long long s = lane < nw ? warp_sums[lane] : 0ull;
    for (int o = 1; o < 32; o <<= 1) {
      const unsigned long long y = __shfl_up_sync(0xffffffffu, s, o);
      if (lane >= o) s += y;
    }
    if (lane < nw) warp_sums[lane] = s;
  }
  __syncthreads();
  const unsigned long long before = (wid > 0 ? warp_sums[wid - 1] : 0ull) + x - v;
  if (total) *total = warp_sums[(blockDim.x >> 5) - 1];
  __syncthreads();
  return before;
}

// ---- radix pass, step 2: exclusive scan of hist in digit-major order (one block)
__global__ void __launch_bounds__(1024) radix_scan_kernel(unsigned* hist, int total) {
  const int per = (total + blockDim.x - 1) / blockDim.x;
  const int lo = min(total, (int)threadIdx.x * per), hi = min(total, lo + per);
  unsigned long long s = 0;
  for (int i = lo; i < hi; ++i) s += hist[i];
  unsigned long long run = block_exclusive_scan(s, nullptr);
  for (int i = lo; i < hi; ++i) {
    const unsigned c = hist[i];
    hist[i] = (unsigned)run;
    run += c;
  }
}

// ---- radix pass, step 3: stable scatter.  Each warp owns a contiguous slice of the block's
// range; lanes of equal digit are ranked with __match_any_sync.
__global__ void __launch_bounds__(256)
radix_scatter_kernel(const u64* in, u64* out, long long n_static, const long long* n_dev,
                     long long cap, int shift, const unsigned* hist, int G) {
  constexpr int W = 8;
  __shared__ unsigned cnt[W][kRadixBins];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  for (int k = threadIdx.x; k < W * kRadixBins; k += blockDim.x) (&cnt[0][0])[k] = 0;
  __syncthreads();
  const long long n = dev_count(n_static, n_dev, cap);
  long long lo, hi;
  block_range(n, G, &lo, &hi);
  const long long wchunk = (hi - lo + W - 1) / W;
  const long long wl = min(hi, lo + w * wchunk), wh = min(hi, wl + wchunk);
  const unsigned lt = (1u << lane) - 1u;
  for (long long base = wl; base < wh; base += 32) {
    const long long i = base + lane;
    const bool valid = i < wh;
    const unsigned d = valid ? ((unsigned)(in[i] >> shift) & (kRadixBins - 1)) : 0x100u;
    const unsigned peers = __match_any_sync(0xffffffffu, d);
    if (valid && (peers & lt) == 0) cnt[w][d] += __popc(peers);
    __syncwarp();
  }
  __syncthreads();
  for (int d = threadIdx.x; d < kRadixBins; d += blockDim.x) {
    unsigned run = hist[d * G + blockIdx.x];
    for (int k = 0; k < W; ++k) { const unsigned c = cnt[k][d]; cnt[k][d] = run; run += c; }
  }
  __syncthreads();
  for (long long base = wl; base < wh; base += 32) {
    const long long i = base + lane;
    const bool valid = i < wh;
    const u64 x = valid ? in[i] : 0ull;
    const unsigned d = valid ? ((unsigned)(x >> shift) & (kRadixBins - 1)) : 0x100u;
    const unsigned peers = __match_any_sync(0xffffffffu, d);
    unsigned pos = 0;
    if (valid) pos = cnt[w][d] + __popc(peers & lt);
    __syncwarp();
    if (valid) {
      out[pos] = x;
      if ((peers & lt) == 0) cnt[w][d] += __popc(peers);
    }
    __syncwarp();
  }
}

// ---- binning: per-block sums of tiles_touched in depth order
__global__ void __launch_bounds__(256)
count_kernel(const u64* sorted, int n, const unsigned* touched, unsigned long long* block_sums,
             int G) {
  long long lo, hi;
  block_range(n, G, &lo, &hi);
  unsigned long long s = 0;
  for (long long i = lo + threadIdx.x; i < hi; i += blockDim.x)
    s += touched[(unsigned)sorted[i]];
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  __shared__ unsigned long long ws[8];
  if ((threadIdx.x & 31) == 0) ws[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned long long t = 0;
    for (int k = 0; k < (int)(blockDim.x >> 5); ++k) t += ws[k];
    block_sums[blockIdx.x] = t;
  }
}

__global__ void __launch_bounds__(1024)
scan_blocks_kernel(unsigned long long* block_sums, int G, long long* count, long long cap,
                   unsigned* status) {
  const unsigned long long v = (int)threadIdx.x < G ? block_sums[threadIdx.x] : 0ull;
  unsigned long long total = 0;
  const unsigned long long ex = block_exclusive_scan(v, &total);
  if ((int)threadIdx.x < G) block_sums[threadIdx.x] = ex;
  if (threadIdx.x == 0) {
    *count = (long long)total;
    if ((long long)total > cap) atomicOr(status, kStatusCapacity);
  }
}

// ---- emission of (tile << 32 | id) in depth order
__global__ void __launch_bounds__(256)
emit_kernel(const u64* sorted, int n, const unsigned* touched, const float2* uv, const int* radius,
            const unsigned long long* block_off, const long long* count, long long cap,
            int tiles_x, int tiles_y, u64* pairs, int G) {
  if (*count > cap) return;
  long long lo, hi;
  block_range(n, G, &lo, &hi);
  unsigned long long run = block_off[blockIdx.x];
  for (long long base = lo; base < hi; base += blockDim.x) {
    const long long i = base + threadIdx.x;
    unsigned id = 0, t = 0;
    if (i < hi) { id = (unsigned)sorted[i]; t = touched[id]; }
    unsigned long long tot = 0;
    unsigned long long off = run + block_exclusive_scan(t, &tot);
    if (t > 0) {
      const float2 m = uv[id];
      const float fr = (float)radius[id];
      const int x0 = (int)fminf(fmaxf(floorf((m.x - fr) * (1.f / kTile)), 0.f), (float)tiles_x);
      const int y0 = (int)fminf(fmaxf(floorf((m.y - fr) * (1.f / kTile)), 0.f), (float)tiles_y);
      const int x1 = (int)fminf(fmaxf(floorf((m.x + fr) * (1.f / kTile)) + 1.f, 0.f), (float)tiles_x);
      // exactly t items (the count the scan reserved), whatever the recomputed rectangle
      const int wdt = max(1, x1 - x0);
      for (unsigned k = 0; k < t; ++k) {
        const int tx = min(x0 + (int)(k % (unsigned)wdt), tiles_x - 1);
        const int ty = min(y0 + (int)(k / (unsigned)wdt), tiles_y - 1);
        pairs[off + k] = ((u64)(unsigned)(ty * tiles_x + tx) << 32) | id;
      }
    }
    run += tot;
  }
}

// ---- tile ranges and ids from the tile-sorted items
__global__ void ranges_kernel(const u64* items, const long long* count, long long cap,
                              unsigned* ranges, unsigned* ids) {
  const long long K = dev_count(0, count, cap);
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < K;
       i += (long long)gridDim.x * blockDim.x) {
    const u64 x = items[i];
    const unsigned t = (unsigned)(x >> 32);
    ids[i] = (unsigned)x;
    if (i == 0 || (unsigned)(items[i - 1] >> 32) != t) ranges[2 * t] = (unsigned)i;
    if (i == K - 1 || (unsigned)(items[i + 1] >> 32) != t) ranges[2 * t + 1] = (unsigned)(i + 1);
  }
}

// LSD radix sort of 64-bit items on bits [bit_lo, bit_hi); returns the buffer holding the result.
abcd_status radix_sort(abcd_ctx* ctx, u64* a, u64* b, long long n_static, const long long* n_dev,
                       long long cap, int bit_lo, int bit_hi, u64** result) {
  const int G = ctx->radix_blocks;
  u64* src = a;
  u64* dst = b;
  for (int shift = bit_lo; shift < bit_hi; shift += kRadixBits) {
    radix_hist_kernel<<<G, 256, 0, ctx->stream>>>(src, n_static, n_dev, cap, shift, ctx->ws.hist, G);
    abcd_status s = check_launch(ctx, "radix_hist_kernel");
    if (s) return s;
    radix_scan_kernel<<<1, 1024, 0, ctx->stream>>>(ctx->ws.hist, kRadixBins * G);
    if ((s = check_launch(ctx, "radix_scan_kernel"))) return s;
    radix_scatter_kernel<<<G, 256, 0, ctx->stream>>>(src, dst, n_static, n_dev, cap, shift, ctx->ws.hist, G);
    if ((s = check_launch(ctx, "radix_scatter_kernel"))) return s;
    u64* t = src; src = dst; dst = t;
  }
  *result = src;
  return ABCD_OK;
}

}  // namespace
}  // namespace abcd

using namespace abcd;

extern "C" abcd_status abcd_bin_sort(abcd_ctx* ctx, const abcd_projected* proj, int n,
                                     const abcd_camera* cam, abcd_tiles* out) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  if (!has_workspace(ctx)) return fail(ctx, ABCD_ERR_WORKSPACE, "abcd_bin_sort: no workspace");
  if (!proj || !cam || !out || n < 0 || cam->width <= 0 || cam->height <= 0)
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_bin_sort: bad arguments");
  if (n > ctx->max_g) return fail(ctx, ABCD_ERR_WORKSPACE, "abcd_bin_sort: n=%d exceeds workspace max_gaussians=%d", n, ctx->max_g);
  if (!out->ids || !out->ranges || !out->count || out->capacity < 0)
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_bin_sort: null tiles output");
  const long long cap = std::min(out->capacity, ctx->max_pairs);
  const int tiles_x = (cam->width + kTile - 1) / kTile, tiles_y = (cam->height + kTile - 1) / kTile;
  const long long n_tiles = (long long)tiles_x * tiles_y;
  if (n_tiles >= (1LL << 24)) return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_bin_sort: too many tiles");
  if (cap >= (1LL << 32)) return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_bin_sort: capacity must be < 2^32");
  if (n > 0 && (!proj->depth || !proj->radius || !proj->uv || !proj->tiles_touched))
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_bin_sort: null projected field");
  cudaError_t e = cudaMemsetAsync(out->ranges, 0, sizeof(unsigned) * 2 * n_tiles, ctx->stream);
  if (e != cudaSuccess) return fail(ctx, ABCD_ERR_CUDA, "ranges memset: %s", cudaGetErrorString(e));
  if (n == 0) {
    e = cudaMemsetAsync(out->count, 0, sizeof(long long), ctx->stream);
    return e == cudaSuccess ? ABCD_OK : fail(ctx, ABCD_ERR_CUDA, "count memset: %s", cudaGetErrorString(e));
  }
  const int G = ctx->radix_blocks;
  abcd_status s;
  depth_keys_kernel<<<(n + 255) / 256, 256, 0, ctx->stream>>>(proj->depth, proj->radius, n, ctx->ws.dsort[0]);
  if ((s = check_launch(ctx, "depth_keys_kernel"))) return s;
  u64* by_depth = nullptr;
  if ((s = radix_sort(ctx, ctx->ws.dsort[0], ctx->ws.dsort[1], n, nullptr, n, 32, 64, &by_depth))) return s;
  count_kernel<<<G, 256, 0, ctx->stream>>>(by_depth, n, proj->tiles_touched, ctx->ws.block_sums, G);
  if ((s = check_launch(ctx, "count_kernel"))) return s;
  scan_blocks_kernel<<<1, 1024, 0, ctx->stream>>>(ctx->ws.block_sums, G, out->count, cap, ctx->ws.status);
  if ((s = check_launch(ctx, "scan_blocks_kernel"))) return s;
  emit_kernel<<<G, 256, 0, ctx->stream>>>(by_depth, n, proj->tiles_touched, (const float2*)proj->uv,
                                          proj->radius, ctx->ws.block_sums, out->count, cap,
                                          tiles_x, tiles_y, ctx->ws.pairs[0], G);
  if ((s = check_launch(ctx, "emit_kernel"))) return s;
  int tile_bits = 1;
  while ((1LL << tile_bits) < n_tiles) ++tile_bits;
  u64* by_tile = nullptr;
  if ((s = radix_sort(ctx, ctx->ws.pairs[0], ctx->ws.pairs[1], 0, out->count, cap, 32,
                      32 + tile_bits, &by_tile))) return s;
  ranges_kernel<<<ctx->num_sms * 4, 256, 0, ctx->stream>>>(by_tile, out->count, cap, out->ranges, out->ids);
  return check_launch(ctx, "ranges_kernel");
}
