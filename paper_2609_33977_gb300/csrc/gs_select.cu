// Selector export (Sec. 2.2; App. F): the evaluation-time group selectors
// B = [sigmoid(l) > 1/2] from float32 selector logits, and the number of kept
// groups (the numerator of Eq. 2, from which the preserved rates follow).
//
// sigmoid is strictly increasing with sigmoid(0) = 1/2, so a group is kept
// exactly when its logit is greater than zero.  The test is made on the bit
// pattern: a float32 is > 0 exactly when its bits, read as an unsigned
// integer b, satisfy 1 <= b <= 0x7F800000 (positive subnormals, normals and
// +inf; +0 is 0, negative values have the sign bit set, positive NaNs lie
// above 0x7F800000).  An integer test keeps the result independent of the
// compiler's flush-to-zero setting for subnormal operands.
//
// HBM-bound: 4 bytes read and 1 byte written per selector.  Each warp step
// covers 512 consecutive selectors: four 16-byte loads per thread, each
// instruction reading 512 contiguous bytes, and four 4-byte stores, each
// writing 128 contiguous bytes.
#include "gs_common.cuh"

namespace gs {
namespace {

constexpr int kSelThreads = 256;
constexpr int kSelWarps = kSelThreads / 32;
constexpr int64_t kSelPerWarp = 512;

__device__ __forceinline__ uint32_t keep_bit(uint32_t b) { return (b - 1u) < 0x7F800000u ? 1u : 0u; }

// four selectors -> four 0/1 bytes, little-endian (byte j = selector j)
__device__ __forceinline__ uint32_t keep4(uint4 v) {
  return keep_bit(v.x) | (keep_bit(v.y) << 8) | (keep_bit(v.z) << 16) | (keep_bit(v.w) << 24);
}

__device__ __forceinline__ uint4 ld_stream_u4(const uint4* p) {
  uint4 v;
  asm volatile("ld.global.cs.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

__global__ void __launch_bounds__(kSelThreads) k_select(const uint32_t* __restrict__ logits, int64_t n,
                                                       uint8_t* __restrict__ mask,
                                                       unsigned long long* __restrict__ kept) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t nfull = n / kSelPerWarp;   // whole 512-selector warp steps
  const int64_t wstride = (int64_t)gridDim.x * kSelWarps;
  // 32-bit counts cannot overflow: the host keeps n < 2^36 and launches
  // min(ceil(nfull / 8), 8 x SMs) blocks, so one warp counts at most
  // 512 * ceil(nfull / (8 * grid)) + 64 < 2^24 selectors and a block eight
  // times that.
  uint32_t cnt = 0;
  for (int64_t u = (int64_t)blockIdx.x * kSelWarps + warp; u < nfull; u += wstride) {
    const uint4* src = reinterpret_cast<const uint4*>(logits + u * kSelPerWarp);
    uint4 v[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) v[q] = ld_stream_u4(src + 32 * q + lane);
    uint32_t* dst = reinterpret_cast<uint32_t*>(mask + u * kSelPerWarp);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const uint32_t m = keep4(v[q]);
      dst[32 * q + lane] = m;
      cnt += __popc(m);
    }
  }
  // ragged tail: fewer than 512 selectors, one byte per thread of block 0
  if (blockIdx.x == 0) {
    for (int64_t i = nfull * kSelPerWarp + threadIdx.x; i < n; i += kSelThreads) {
      const uint32_t k = keep_bit(logits[i]);
      mask[i] = (uint8_t)k;
      cnt += k;
    }
  }
  if (kept == nullptr) return;   // uniform over the grid
  cnt = __reduce_add_sync(0xffffffffu, cnt);
  __shared__ uint32_t warp_cnt[kSelWarps];
  if (lane == 0) warp_cnt[warp] = cnt;
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned long long total = 0;
#pragma unroll
    for (int w = 0; w < kSelWarps; ++w) total += warp_cnt[w];
    if (total) atomicAdd(kept, total);
  }
}

int sm_count_sel() {
  static int n = 0;
  if (n == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 148;
  }
  return n;
}

}  // namespace

gs_status launch_select(const float* logits, int64_t n, uint8_t* mask, int64_t* kept, cudaStream_t s) {
  if (kept && cudaMemsetAsync(kept, 0, sizeof(int64_t), s) != cudaSuccess) return GS_ERR_CUDA;
  if (n == 0) return GS_OK;
  const int64_t nfull = n / kSelPerWarp;
  int64_t grid = (nfull + kSelWarps - 1) / kSelWarps;
  const int64_t cap = (int64_t)sm_count_sel() * 8;   // 8 blocks of 256 threads per SM
  if (grid > cap) grid = cap;
  if (grid < 1) grid = 1;
  k_select<<<(unsigned)grid, kSelThreads, 0, s>>>(reinterpret_cast<const uint32_t*>(logits), n, mask,
                                                  reinterpret_cast<unsigned long long*>(kept));
  note_launch();
  return cudaGetLastError() == cudaSuccess ? GS_OK : GS_ERR_CUDA;
}

}  // namespace gs
