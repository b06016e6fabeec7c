// Packing (count -> scan -> compact+copy) and unpacking of the chunk-major
// group-sparse layout.  The groups are the 1x256 input-dimension groups of
// Sec. 2.1; the mask selects whole groups (Eq. 1), so only kept groups are
// copied.  Layout: chunk c owns packed rows [offsets[c], offsets[c+1]), kept
// rows in ascending order; per (chunk, 16-row window) a start offset and a
// 16-bit kept mask.
#include "gs_common.cuh"

#include <mutex>

namespace gs {
namespace {

// (a1) count: kmask16[c][w] = bits of the kept rows 16w..16w+15 in chunk c.
__global__ void k_pack_count(const uint8_t* __restrict__ mask, int32_t out, int32_t G, int32_t nw16,
                             uint16_t* __restrict__ kmask16, int32_t* __restrict__ cnt) {
  const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;   // e = c * nw16 + w
  if (e >= (int64_t)G * nw16) return;
  const int c = (int)(e / nw16);
  const int w = (int)(e % nw16);
  uint32_t bits = 0;
#pragma unroll
  for (int i = 0; i < kWin16; ++i) {
    const int r = kWin16 * w + i;
    if (r < out && mask[(int64_t)r * G + c] != 0) bits |= 1u << i;
  }
  kmask16[e] = (uint16_t)bits;
  cnt[e] = __popc(bits);
}

// (a2) scan: one CTA, exclusive prefix sum of cnt in chunk-major order.
constexpr int kScanThreads = 1024;
constexpr int kScanItems = 4;

__global__ void __launch_bounds__(kScanThreads) k_pack_scan(const int32_t* __restrict__ cnt, int32_t G,
                                                            int32_t nw16, int32_t* __restrict__ win_off16,
                                                            int64_t* __restrict__ offsets) {
  __shared__ int32_t warp_sums[kScanThreads / 32];
  __shared__ int32_t carry_s;
  const int64_t E = (int64_t)G * nw16;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (tid == 0) carry_s = 0;
  __syncthreads();
  for (int64_t base = 0; base < E; base += (int64_t)kScanThreads * kScanItems) {
    int32_t v[kScanItems];
    int32_t local = 0;
#pragma unroll
    for (int i = 0; i < kScanItems; ++i) {
      const int64_t e = base + (int64_t)tid * kScanItems + i;
      v[i] = e < E ? cnt[e] : 0;
      local += v[i];
    }
    // inclusive warp scan of the thread sums
    int32_t incl = local;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      const int32_t t = __shfl_up_sync(0xffffffffu, incl, d);
      if (lane >= d) incl += t;
    }
    if (lane == 31) warp_sums[warp] = incl;
    __syncthreads();
    if (warp == 0) {
      int32_t ws = warp_sums[lane];
      int32_t wi = ws;
#pragma unroll
      for (int d = 1; d < 32; d <<= 1) {
        const int32_t t = __shfl_up_sync(0xffffffffu, wi, d);
        if (lane >= d) wi += t;
      }
      warp_sums[lane] = wi - ws;   // exclusive warp offsets
    }
    __syncthreads();
    int32_t run = carry_s + warp_sums[warp] + (incl - local);
#pragma unroll
    for (int i = 0; i < kScanItems; ++i) {
      const int64_t e = base + (int64_t)tid * kScanItems + i;
      if (e < E) {
        const int c = (int)(e / nw16);
        const int w = (int)(e % nw16);
        win_off16[(int64_t)c * (nw16 + 1) + w] = run;
        if (w == 0) offsets[c] = run;
        if (w == nw16 - 1) win_off16[(int64_t)c * (nw16 + 1) + nw16] = run + v[i];
        if (e == E - 1) offsets[G] = run + v[i];
      }
      run += v[i];
    }
    __syncthreads();
    if (tid == kScanThreads - 1) carry_s = run;
    __syncthreads();
  }
}

__device__ __forceinline__ uint4 ld_stream16(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
  return v;
}

// (a3) compact + copy: one warp per output row; every kept group of the row is
// copied (KW bf16: 16 B per lane, KW / 8 lanes) to its packed slot and its row
// index recorded.  KW = chunk width, 256 (1 x 256 groups) or 128 (1 x 128).
template <int KW>
__global__ void k_pack_compact(const uint16_t* __restrict__ W, int32_t out, int32_t in, int32_t G,
                               int32_t nw16, const int32_t* __restrict__ win_off16,
                               const uint16_t* __restrict__ kmask16, int32_t* __restrict__ row_idx,
                               uint16_t* __restrict__ tiles) {
  const int lane = threadIdx.x & 31;
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
  for (int64_t r = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); r < out; r += warps) {
    const int w = (int)(r / kWin16), i = (int)(r % kWin16);
    const uint32_t below = (1u << i) - 1u;
    for (int cb = 0; cb < G; cb += 32) {
      const int c = cb + lane;
      bool kept = false;
      int32_t pos = 0;
      if (c < G) {
        const uint32_t km = kmask16[(int64_t)c * nw16 + w];
        kept = (km >> i) & 1u;
        pos = win_off16[(int64_t)c * (nw16 + 1) + w] + __popc(km & below);
      }
      uint32_t ballot = __ballot_sync(0xffffffffu, kept);
      while (ballot) {
        // up to four groups per round for memory-level parallelism
        int cs[4];
        int32_t ps[4];
        int n = 0;
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          if (ballot) {
            const int b = __ffs(ballot) - 1;
            ballot &= ballot - 1;
            cs[u] = cb + b;
            ps[u] = __shfl_sync(0xffffffffu, pos, b);
            ++n;
          } else {
            cs[u] = -1;
            ps[u] = 0;
          }
        }
        uint4 v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u)
          if (u < n && lane < KW / 8) v[u] = ld_stream16(W + r * in + (int64_t)cs[u] * KW + 8 * lane);
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          if (u < n) {
            if (lane < KW / 8) reinterpret_cast<uint4*>(tiles + (int64_t)ps[u] * KW)[lane] = v[u];
            if (lane == 0) row_idx[ps[u]] = (int32_t)r;
          }
        }
      }
    }
  }
}

// (a7) unpack: one warp per output row; kept groups copied back from their
// packed slot, pruned groups written as +0.0.
template <int KW>
__global__ void k_unpack(const uint16_t* __restrict__ tiles, int32_t out, int32_t in, int32_t G,
                         int32_t nw16, const int32_t* __restrict__ win_off16,
                         const uint16_t* __restrict__ kmask16, uint16_t* __restrict__ W_hat) {
  const int lane = threadIdx.x & 31;
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
  for (int64_t r = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); r < out; r += warps) {
    const int w = (int)(r / kWin16), i = (int)(r % kWin16);
    const uint32_t below = (1u << i) - 1u;
    for (int cb = 0; cb < G; cb += 32) {
      const int c = cb + lane;
      bool kept = false;
      int32_t pos = 0;
      if (c < G) {
        const uint32_t km = kmask16[(int64_t)c * nw16 + w];
        kept = (km >> i) & 1u;
        pos = win_off16[(int64_t)c * (nw16 + 1) + w] + __popc(km & below);
      }
      const uint32_t kb = __ballot_sync(0xffffffffu, kept);
      const int nc = min(32, G - cb);
      for (int u = 0; u < nc; ++u) {
        const int32_t pu = __shfl_sync(0xffffffffu, pos, u);
        uint4 v = make_uint4(0u, 0u, 0u, 0u);
        if (lane < KW / 8) {
          if ((kb >> u) & 1u) v = ld_stream16(tiles + (int64_t)pu * KW + 8 * lane);
          reinterpret_cast<uint4*>(W_hat + r * in + (int64_t)(cb + u) * KW)[lane] = v;
        }
      }
    }
  }
}

int grid_for(int64_t items, int per_block) {
  int64_t b = (items + per_block - 1) / per_block;
  if (b < 1) b = 1;
  if (b > (1 << 20)) b = 1 << 20;
  return (int)b;
}

}  // namespace

gs_status launch_pack_count_scan(const uint8_t* mask, gs_packed* p, cudaStream_t s, int32_t* cnt_tmp) {
  const int64_t E = (int64_t)p->G * p->nw16;
  k_pack_count<<<grid_for(E, 256), 256, 0, s>>>(mask, (int32_t)p->out, p->G, p->nw16, p->kmask16, cnt_tmp);
  k_pack_scan<<<1, kScanThreads, 0, s>>>(cnt_tmp, p->G, p->nw16, p->win_off16, p->offsets);
  note_launch(2);
  return cudaGetLastError() == cudaSuccess ? GS_OK : GS_ERR_CUDA;
}

gs_status launch_scan_counts(const int32_t* cnt, int32_t G, int32_t nw, int32_t* win_off, int64_t* offsets,
                             cudaStream_t s) {
  k_pack_scan<<<1, kScanThreads, 0, s>>>(cnt, G, nw, win_off, offsets);
  note_launch();
  return cudaGetLastError() == cudaSuccess ? GS_OK : GS_ERR_CUDA;
}

gs_status launch_pack_compact(const void* W, gs_packed* p, cudaStream_t s) {
  if (p->kept == 0) return GS_OK;
  auto kern = p->g_in == 128 ? k_pack_compact<128> : k_pack_compact<256>;
  kern<<<grid_for(p->out, 8), 256, 0, s>>>(static_cast<const uint16_t*>(W), (int32_t)p->out, (int32_t)p->in, p->G,
                                           p->nw16, p->win_off16, p->kmask16, p->row_idx, p->tiles);
  note_launch();
  return cudaGetLastError() == cudaSuccess ? GS_OK : GS_ERR_CUDA;
}

gs_status launch_unpack(const gs_packed* p, void* W_hat, cudaStream_t s) {
  auto kern = p->g_in == 128 ? k_unpack<128> : k_unpack<256>;
  kern<<<grid_for(p->out, 8), 256, 0, s>>>(p->tiles, (int32_t)p->out, (int32_t)p->in, p->G, p->nw16, p->win_off16,
                                           p->kmask16, static_cast<uint16_t*>(W_hat));
  note_launch();
  return cudaGetLastError() == cudaSuccess ? GS_OK : GS_ERR_CUDA;
}

}  // namespace gs

// ---------------------------------------------------------------------------
// Allocation-free variant of the packing index step (count + scan).
//
// The per-(chunk, 16-row window) counts that gs_pack keeps in a cudaMalloc'd
// temporary live here in a fixed array in the library's own device memory, so
// gs_pack_index_noalloc never allocates.  Every call reuses (and overwrites)
// the same array; the count kernel writes every entry it later reads, so no
// entry needs clearing between calls.  Calls whose kernels overlap on the GPU
// (concurrent streams) race on this array and must be serialized.
// ---------------------------------------------------------------------------
namespace gs {
namespace {

constexpr int64_t kNoAllocMaxEntries = int64_t(1) << 20;   // chunks x 16-row windows (4 MiB of int32)
static __device__ __align__(256) int32_t g_noalloc_counts[kNoAllocMaxEntries];

constexpr int kNoAllocMaxDevices = 64;
std::mutex g_noalloc_mu;
int32_t* g_noalloc_ptr[kNoAllocMaxDevices] = {nullptr};

// Device address of the counts array on the current device; resolved once per
// device (with that device current) and cached.
gs_status noalloc_counts_address(int32_t** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kNoAllocMaxDevices) return GS_ERR_CUDA;
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  if (!g_noalloc_ptr[dev]) {
    int32_t* ptr = nullptr;
    if (cudaGetSymbolAddress(reinterpret_cast<void**>(&ptr), g_noalloc_counts) != cudaSuccess || !ptr)
      return GS_ERR_CUDA;
    g_noalloc_ptr[dev] = ptr;
  }
  *out = g_noalloc_ptr[dev];
  return GS_OK;
}

}  // namespace
}  // namespace gs

extern "C" gs_status gs_pack_index_noalloc(const uint8_t* mask_dev, int64_t out, int64_t in, int64_t* offsets_dev,
                                           int32_t* win_off16_dev, uint16_t* kmask16_dev, void* stream) {
  using namespace gs;
  if (!mask_dev || !offsets_dev || !win_off16_dev || !kmask16_dev) return GS_ERR_INVALID_ARG;
  if (out <= 0 || in <= 0 || out > INT32_MAX || in > INT32_MAX || in % kGroupIn != 0) return GS_ERR_INVALID_ARG;
  // element alignment of each output (int64, int32, uint16)
  if ((reinterpret_cast<uintptr_t>(offsets_dev) & 7u) != 0 || (reinterpret_cast<uintptr_t>(win_off16_dev) & 3u) != 0 ||
      (reinterpret_cast<uintptr_t>(kmask16_dev) & 1u) != 0)
    return GS_ERR_INVALID_ARG;
  const int64_t G = in / kGroupIn;
  const int64_t nw16 = (out + kWin16 - 1) / kWin16;
  if (G * nw16 > kNoAllocMaxEntries) return GS_ERR_UNSUPPORTED;   // beyond the fixed scratch array
  {
    // the outputs must not overlap each other or the mask they are computed from
    const uintptr_t lo[4] = {reinterpret_cast<uintptr_t>(mask_dev), reinterpret_cast<uintptr_t>(offsets_dev),
                             reinterpret_cast<uintptr_t>(win_off16_dev), reinterpret_cast<uintptr_t>(kmask16_dev)};
    const uintptr_t len[4] = {(uintptr_t)(out * G), (uintptr_t)(8 * (G + 1)), (uintptr_t)(4 * G * (nw16 + 1)),
                              (uintptr_t)(2 * G * nw16)};
    for (int a = 0; a < 4; ++a)
      for (int b = a + 1; b < 4; ++b)
        if (lo[a] < lo[b] + len[b] && lo[b] < lo[a] + len[a]) return GS_ERR_INVALID_ARG;
  }
  int32_t* counts = nullptr;
  const gs_status st = noalloc_counts_address(&counts);
  if (st != GS_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int64_t E = G * nw16;
  k_pack_count<<<grid_for(E, 256), 256, 0, s>>>(mask_dev, (int32_t)out, (int32_t)G, (int32_t)nw16, kmask16_dev,
                                                counts);
  k_pack_scan<<<1, kScanThreads, 0, s>>>(counts, (int32_t)G, (int32_t)nw16, win_off16_dev, offsets_dev);
  note_launch(2);
  return cudaGetLastError() == cudaSuccess ? GS_OK : GS_ERR_CUDA;
}
