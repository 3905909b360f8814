// K3 (tile binning) and K4 (sort + tile ranges) of the ABCD active-block step.
//
// What is computed (3DGS binning, Section 1 of the paper by citation): every visible Gaussian
// is listed in each 16x16 tile met by its square [u-r, u+r] x [v-r, v+r]; each tile's list
// is ordered front to back by (fp32 depth, Gaussian id).
//
// How (GB300 design, different from sorting 64-bit (tile | depth) keys):
//   1. per Gaussian: its tile rectangle (kept in the workspace), a sort key (fp32 depth bits,
//      all ones when culled) and +-1 at the rectangle's four corners of a 2-D difference
//      array over the tile grid;
//   2. stable LSD radix sort of the n Gaussians by the 32 depth bits;
//   3. exclusive scan of the rectangle areas in that order: K = total pairs; the 2-D prefix
//      sum of the difference array gives every tile's pair count, hence its range;
//   4. warp-cooperative emission of (tile << 32 | id) items in depth order;
//   5. stable LSD radix sort of the K items on the tile bits only (ceil(log2 n_tiles) <= 16
//      bits, 8 per pass), which keeps depth order inside each tile; the last pass writes ids.
// Radix passes are reduce-then-scan (per-block digit counts, per-digit row scans, stable
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

__device__ __forceinline__ int4 tile_rect(float2 m, int r, int tiles_x, int tiles_y) {
  const float fr = (float)r;
  int4 q;
  q.x = (int)fminf(fmaxf(floorf((m.x - fr) * (1.f / kTile)), 0.f), (float)tiles_x);
  q.y = (int)fminf(fmaxf(floorf((m.y - fr) * (1.f / kTile)), 0.f), (float)tiles_y);
  q.z = (int)fminf(fmaxf(floorf((m.x + fr) * (1.f / kTile)) + 1.f, 0.f), (float)tiles_x);
  q.w = (int)fminf(fmaxf(floorf((m.y + fr) * (1.f / kTile)) + 1.f, 0.f), (float)tiles_y);
  return q;
}

// ---- per Gaussian: depth key (bits(depth) << 32 | id, all ones when culled), tile
// rectangle, and the rectangle's corners in the (tiles_y + 1) x (tiles_x + 1) difference array
__global__ void keys_rects_kernel(const float* depth, const int* radius, const float2* uv, int n,
                                  int tiles_x, int tiles_y, u64* items, int4* rects, int* diff) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  int4 q = make_int4(0, 0, 0, 0);
  const int r = radius[i];
  if (r > 0) q = tile_rect(uv[i], r, tiles_x, tiles_y);
  const bool vis = r > 0 && q.x < q.z && q.y < q.w;
  if (!vis) q = make_int4(0, 0, 0, 0);
  rects[i] = q;
  const unsigned key = vis ? __float_as_uint(depth[i]) : 0xFFFFFFFFu;
  items[i] = ((u64)key << 32) | (unsigned)i;
  if (vis) {
    const int W1 = tiles_x + 1;
    atomicAdd(&diff[q.y * W1 + q.x], 1);
    atomicAdd(&diff[q.y * W1 + q.z], -1);
    atomicAdd(&diff[q.w * W1 + q.x], -1);
    atomicAdd(&diff[q.w * W1 + q.z], 1);
  }
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

// ---- radix pass, step 2: exclusive scan of each digit's row hist[d][0..G) (one block per
// digit); the row totals go to totals[d]
__global__ void __launch_bounds__(1024) radix_rowscan_kernel(unsigned* hist, int G,
                                                            unsigned* totals) {
  const int d = blockIdx.x;
  const unsigned v = (int)threadIdx.x < G ? hist[d * G + threadIdx.x] : 0u;
  unsigned long long tot = 0;
  const unsigned long long ex = block_exclusive_scan(v, &tot);
  if ((int)threadIdx.x < G) hist[d * G + threadIdx.x] = (unsigned)ex;
  if (threadIdx.x == 0) totals[d] = (unsigned)tot;
}

// ---- radix pass, step 3: stable scatter.  Each warp owns a contiguous slice of the block's
// range; lanes of equal digit are ranked with __match_any_sync.
__global__ void __launch_bounds__(256)
radix_scatter_kernel(const u64* in, u64* out, unsigned* out_ids, long long n_static,
                     const long long* n_dev, long long cap, int shift, const unsigned* hist,
                     const unsigned* totals, int G) {
  constexpr int W = 8;
  __shared__ unsigned cnt[W][kRadixBins];
  __shared__ unsigned base[kRadixBins];
  {
    // digit bases: exclusive scan of the digit totals (kRadixBins == blockDim.x)
    const unsigned t = totals[threadIdx.x];
    unsigned long long tot = 0;
    base[threadIdx.x] = (unsigned)block_exclusive_scan(t, &tot);
  }
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
    unsigned run = base[d] + hist[d * G + blockIdx.x];
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
      if (out_ids) out_ids[pos] = (unsigned)x;
      else out[pos] = x;
      if ((peers & lt) == 0) cnt[w][d] += __popc(peers);
    }
    __syncwarp();
  }
}

// ---- binning: per-block sums of rectangle areas in depth order
__device__ __forceinline__ unsigned rect_area(int4 q) { return (unsigned)((q.z - q.x) * (q.w - q.y)); }

__global__ void __launch_bounds__(256)
count_kernel(const u64* sorted, int n, const int4* rects, unsigned long long* block_sums, int G) {
  long long lo, hi;
  block_range(n, G, &lo, &hi);
  unsigned long long s = 0;
  for (long long i = lo + threadIdx.x; i < hi; i += blockDim.x)
    s += rect_area(rects[(unsigned)sorted[i]]);
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

// ---- tile ranges from the difference array: 2-D prefix sum -> per-tile counts -> exclusive
// scan (one block).  Empty ranges when K overflowed the capacity.
__global__ void __launch_bounds__(1024)
ranges_from_diff_kernel(int* diff, int tiles_x, int tiles_y, const long long* count, long long cap,
                        unsigned* ranges) {
  const int W1 = tiles_x + 1;
  for (int y = threadIdx.x; y < tiles_y; y += blockDim.x) {       // prefix along x
    int run = 0;
    for (int x = 0; x < tiles_x; ++x) { run += diff[y * W1 + x]; diff[y * W1 + x] = run; }
  }
  __syncthreads();
  for (int x = threadIdx.x; x < tiles_x; x += blockDim.x) {       // prefix along y
    int run = 0;
    for (int y = 0; y < tiles_y; ++y) { run += diff[y * W1 + x]; diff[y * W1 + x] = run; }
  }
  __syncthreads();
  const bool ok = *count <= cap;
  const int nt = tiles_x * tiles_y;
  const int per = (nt + blockDim.x - 1) / blockDim.x;
  const int lo = min(nt, (int)threadIdx.x * per), hi = min(nt, lo + per);
  unsigned long long s = 0;
  for (int t = lo; t < hi; ++t) s += (unsigned)diff[(t / tiles_x) * W1 + (t % tiles_x)];
  unsigned long long run = block_exclusive_scan(s, nullptr);
  for (int t = lo; t < hi; ++t) {
    const unsigned c = (unsigned)diff[(t / tiles_x) * W1 + (t % tiles_x)];
    ranges[2 * t] = ok ? (unsigned)run : 0u;
    ranges[2 * t + 1] = ok ? (unsigned)(run + c) : 0u;
    run += c;
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

// ---- emission of (tile << 32 | id) in depth order; each warp writes its Gaussians' pairs
// one Gaussian at a time with all lanes (contiguous, coalesced stores)
__global__ void __launch_bounds__(256)
emit_kernel(const u64* sorted, int n, const int4* rects, const unsigned long long* block_off,
            const long long* count, long long cap, int tiles_x, u64* pairs, int G) {
  if (*count > cap) return;
  long long lo, hi;
  block_range(n, G, &lo, &hi);
  const int lane = threadIdx.x & 31;
  unsigned long long run = block_off[blockIdx.x];
  for (long long base = lo; base < hi; base += blockDim.x) {
    const long long i = base + threadIdx.x;
    unsigned id = 0, t = 0;
    int4 q = make_int4(0, 0, 0, 0);
    if (i < hi) { id = (unsigned)sorted[i]; q = rects[id]; t = rect_area(q); }
    unsigned long long tot = 0;
    const unsigned long long off = run + block_exclusive_scan(t, &tot);
    for (int j = 0; j < 32; ++j) {
      const unsigned tj = __shfl_sync(0xffffffffu, t, j);
      if (tj == 0) continue;
      const unsigned idj = __shfl_sync(0xffffffffu, id, j);
      const unsigned long long oj = __shfl_sync(0xffffffffu, off, j);
      const int x0 = __shfl_sync(0xffffffffu, q.x, j), y0 = __shfl_sync(0xffffffffu, q.y, j);
      const int w = __shfl_sync(0xffffffffu, q.z, j) - x0;
      for (unsigned k = lane; k < tj; k += 32) {
        const int tile = (y0 + (int)(k / (unsigned)w)) * tiles_x + x0 + (int)(k % (unsigned)w);
        pairs[oj + k] = ((u64)(unsigned)tile << 32) | idj;
      }
    }
    run += tot;
  }
}

// LSD radix sort of 64-bit items on bits [bit_lo, bit_hi); returns the buffer holding the
// result, or writes the low 32 bits of the sorted items to ids_out on the last pass.
abcd_status radix_sort(abcd_ctx* ctx, u64* a, u64* b, long long n_static, const long long* n_dev,
                       long long cap, int bit_lo, int bit_hi, u64** result, unsigned* ids_out) {
  const int G = ctx->radix_blocks;
  unsigned* totals = ctx->ws.hist + kRadixBins * G;
  u64* src = a;
  u64* dst = b;
  for (int shift = bit_lo; shift < bit_hi; shift += kRadixBits) {
    const bool last = shift + kRadixBits >= bit_hi;
    radix_hist_kernel<<<G, 256, 0, ctx->stream>>>(src, n_static, n_dev, cap, shift, ctx->ws.hist, G);
    abcd_status s = check_launch(ctx, "radix_hist_kernel");
    if (s) return s;
    radix_rowscan_kernel<<<kRadixBins, ((G + 31) / 32) * 32, 0, ctx->stream>>>(ctx->ws.hist, G, totals);
    if ((s = check_launch(ctx, "radix_rowscan_kernel"))) return s;
    radix_scatter_kernel<<<G, kRadixBins, 0, ctx->stream>>>(src, dst, last ? ids_out : nullptr,
                                                            n_static, n_dev, cap, shift,
                                                            ctx->ws.hist, totals, G);
    if ((s = check_launch(ctx, "radix_scatter_kernel"))) return s;
    u64* t = src; src = dst; dst = t;
  }
  if (result) *result = src;
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
  cudaError_t e = cudaSuccess;
  if (n == 0) {
    e = cudaMemsetAsync(out->ranges, 0, sizeof(unsigned) * 2 * n_tiles, ctx->stream);
    if (e != cudaSuccess) return fail(ctx, ABCD_ERR_CUDA, "ranges memset: %s", cudaGetErrorString(e));
    e = cudaMemsetAsync(out->count, 0, sizeof(long long), ctx->stream);
    return e == cudaSuccess ? ABCD_OK : fail(ctx, ABCD_ERR_CUDA, "count memset: %s", cudaGetErrorString(e));
  }
  const int G = ctx->radix_blocks;
  const size_t diff_bytes = sizeof(int) * (size_t)(tiles_x + 1) * (tiles_y + 1);
  if (diff_bytes > ctx->ws.diff_bytes)
    return fail(ctx, ABCD_ERR_WORKSPACE, "abcd_bin_sort: tile grid exceeds the workspace");
  e = cudaMemsetAsync(ctx->ws.diff, 0, diff_bytes, ctx->stream);
  if (e != cudaSuccess) return fail(ctx, ABCD_ERR_CUDA, "diff memset: %s", cudaGetErrorString(e));
  abcd_status s;
  keys_rects_kernel<<<(n + 255) / 256, 256, 0, ctx->stream>>>(
      proj->depth, proj->radius, (const float2*)proj->uv, n, tiles_x, tiles_y, ctx->ws.dsort[0],
      ctx->ws.rects, ctx->ws.diff);
  if ((s = check_launch(ctx, "keys_rects_kernel"))) return s;
  u64* by_depth = nullptr;
  if ((s = radix_sort(ctx, ctx->ws.dsort[0], ctx->ws.dsort[1], n, nullptr, n, 32, 64, &by_depth, nullptr)))
    return s;
  count_kernel<<<G, 256, 0, ctx->stream>>>(by_depth, n, ctx->ws.rects, ctx->ws.block_sums, G);
  if ((s = check_launch(ctx, "count_kernel"))) return s;
  scan_blocks_kernel<<<1, 1024, 0, ctx->stream>>>(ctx->ws.block_sums, G, out->count, cap, ctx->ws.status);
  if ((s = check_launch(ctx, "scan_blocks_kernel"))) return s;
  ranges_from_diff_kernel<<<1, 1024, 0, ctx->stream>>>(ctx->ws.diff, tiles_x, tiles_y, out->count, cap,
                                                      out->ranges);
  if ((s = check_launch(ctx, "ranges_from_diff_kernel"))) return s;
  emit_kernel<<<G, 256, 0, ctx->stream>>>(by_depth, n, ctx->ws.rects, ctx->ws.block_sums, out->count,
                                          cap, tiles_x, ctx->ws.pairs[0], G);
  if ((s = check_launch(ctx, "emit_kernel"))) return s;
  int tile_bits = 1;
  while ((1LL << tile_bits) < n_tiles) ++tile_bits;
  return radix_sort(ctx, ctx->ws.pairs[0], ctx->ws.pairs[1], 0, out->count, cap, 32, 32 + tile_bits,
                    nullptr, out->ids);
}
