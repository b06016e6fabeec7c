// Training-side selectors (Sec. 2.2): a Gumbel-Sigmoid sample with a
// straight-through estimator (STE), and the backward pass of the masked linear
// y = x (W (.) (B (x) 1))^T with W frozen.
//
//   sample:   z = l + L (L: logistic noise, the difference of two standard
//             Gumbel draws, supplied by the caller), B = [z > 0] (the binary
//             selectors of the forward pass), and the derivative of the
//             relaxation s = sigmoid(z / tau) that the backward pass uses,
//             ds/dl = s (1 - s) / tau, written as t / (1 + t)^2 / tau with
//             t = exp(-|z| / tau) so that it keeps its precision where s is
//             near 0 or 1 (1 - s would cancel in float32).
//   backward: dL/dW_hat = dy^T x, dL/dB[u, v] = sum over the group of
//             W (.) dL/dW_hat, and the STE gives dL/dl = dL/dB ds/dl;
//             dL/dx = dy W_hat.
//
// The two products of the backward are plain dense GEMMs (dy^T x over all
// groups, pruned ones included, since the STE passes gradients to every
// selector; dy W_hat on the masked weight) and go to cuBLAS.  The group
// reduction with the STE factor and the sampling are kernels of this file; the
// forward pass is gs_pack with the sampled mask followed by gs_linear.
#include "gs_common.cuh"

#include <cublas_v2.h>
#include <mutex>

namespace gs {
namespace {

constexpr int kGumbelThreads = 256;

// one selector per thread (grid-stride); per-warp popcount, one 64-bit atomic per warp
__global__ void k_gumbel(const float* __restrict__ logits, const float* __restrict__ noise, int64_t n, float tau,
                         uint8_t* __restrict__ mask, float* __restrict__ dsdl, unsigned long long* __restrict__ kept) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  unsigned int cnt = 0;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
    const float z = __fadd_rn(logits[i], noise[i]);
    const bool keep = z > 0.f;   // NaN prunes
    mask[i] = keep ? 1 : 0;
    if (dsdl) {
      const float t = expf(-fabsf(__fdiv_rn(z, tau)));
      const float d = 1.f + t;
      dsdl[i] = __fdiv_rn(__fdiv_rn(t, d * d), tau);
    }
    cnt += keep ? 1u : 0u;
  }
  const unsigned int w = __reduce_add_sync(0xffffffffu, cnt);
  if (kept && (threadIdx.x & 31) == 0 && w) atomicAdd(kept, (unsigned long long)w);
}

// dlogits[u, v] = ds/dl[u, v] * sum over group (u, v) of W (.) D, D = dy^T x
// (fp32 [out][in]); one warp per group, lanes over the group's cells four at a time
__global__ void k_group_grad(const uint16_t* __restrict__ W, const float* __restrict__ D, const float* __restrict__ dsdl,
                             int32_t out, int32_t in, int32_t g_out, int32_t g_in, float* __restrict__ dlogits) {
  const int lane = threadIdx.x & 31;
  const int64_t Gin = in / g_in, n = (int64_t)(out / g_out) * Gin;
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
  const int per_row = g_in / 4;
  for (int64_t e = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); e < n; e += warps) {
    const int64_t u = e / Gin, v = e % Gin;
    float acc = 0.f;
    for (int c = lane; c < g_out * per_row; c += 32) {
      const int64_t r = u * g_out + c / per_row;
      const int64_t k = v * g_in + 4 * (c % per_row);
      const float4 d = *reinterpret_cast<const float4*>(D + r * in + k);
      const uint2 wb = *reinterpret_cast<const uint2*>(W + r * in + k);
      acc = fmaf(__uint_as_float(wb.x << 16), d.x, acc);
      acc = fmaf(__uint_as_float(wb.x & 0xFFFF0000u), d.y, acc);
      acc = fmaf(__uint_as_float(wb.y << 16), d.z, acc);
      acc = fmaf(__uint_as_float(wb.y & 0xFFFF0000u), d.w, acc);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (lane == 0) dlogits[e] = acc * dsdl[e];
  }
}

std::mutex g_blas_mu;
cublasHandle_t g_blas[64] = {nullptr};

gs_status blas_handle(cublasHandle_t* h) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return GS_ERR_CUDA;
  if (!g_blas[dev] && cublasCreate(&g_blas[dev]) != CUBLAS_STATUS_SUCCESS) {
    g_blas[dev] = nullptr;
    return GS_ERR_CUDA;
  }
  *h = g_blas[dev];
  return GS_OK;
}

size_t round256(size_t b) { return (b + 255) & ~size_t(255); }

}  // namespace

gs_status launch_gumbel(const float* logits, const float* noise, int64_t n, float tau, uint8_t* mask, float* dsdl,
                        int64_t* kept, cudaStream_t s) {
  if (kept && cudaMemsetAsync(kept, 0, sizeof(int64_t), s) != cudaSuccess) return GS_ERR_CUDA;
  if (n == 0) return GS_OK;
  int64_t blocks = (n + kGumbelThreads - 1) / kGumbelThreads;
  if (blocks > 8 * 1024) blocks = 8 * 1024;
  k_gumbel<<<(unsigned)blocks, kGumbelThreads, 0, s>>>(logits, noise, n, tau, mask, dsdl,
                                                       reinterpret_cast<unsigned long long*>(kept));
  note_launch();
  return cudaGetLastError() == cudaSuccess ? GS_OK : GS_ERR_CUDA;
}

size_t backward_workspace_bytes(const gs_packed* p, bool want_dx) {
  const size_t cells = (size_t)p->out * (size_t)p->in;
  return round256(4 * cells) + (want_dx ? round256(2 * cells) : 0);
}

gs_status launch_backward(const void* x, const void* W, const gs_packed* p, const void* dy, int64_t T,
                          const float* dsdl, float* dlogits, void* dx, void* ws, cudaStream_t s) {
  const int64_t out = p->out, in = p->in;
  float* D = static_cast<float*>(ws);
  {
    std::lock_guard<std::mutex> lk(g_blas_mu);
    cublasHandle_t h = nullptr;
    gs_status st = blas_handle(&h);
    if (st != GS_OK) return st;
    if (cublasSetStream(h, s) != CUBLAS_STATUS_SUCCESS) return GS_ERR_CUDA;
    const float one = 1.f, zero = 0.f;
    // D [out][in] = dy^T x.  In cuBLAS's column-major terms D is (in x out) =
    // A (in x T) * B (T x out): x row-major [T][in] is A as stored; dy
    // row-major [T][out] is (out x T) as stored, so B is it transposed.
    if (cublasGemmEx(h, CUBLAS_OP_N, CUBLAS_OP_T, (int)in, (int)out, (int)T, &one, x, CUDA_R_16BF, (int)in, dy,
                     CUDA_R_16BF, (int)out, &zero, D, CUDA_R_32F, (int)in, CUBLAS_COMPUTE_32F,
                     CUBLAS_GEMM_DEFAULT) != CUBLAS_STATUS_SUCCESS)
      return GS_ERR_CUDA;
    if (dx) {
      // W_hat (dense, pruned groups +0.0) then dx [T][in] = dy W_hat:
      // column-major (in x T) = W_hat as (in x out) * dy as (out x T)
      uint16_t* What = reinterpret_cast<uint16_t*>(static_cast<uint8_t*>(ws) + round256(4 * (size_t)out * in));
      if (p->g_out > 1) st = sq_unpack(p, What, s);
      else st = launch_unpack(p, What, s);
      if (st != GS_OK) return st;
      if (cublasGemmEx(h, CUBLAS_OP_N, CUBLAS_OP_N, (int)in, (int)T, (int)out, &one, What, CUDA_R_16BF, (int)in, dy,
                       CUDA_R_16BF, (int)out, &zero, dx, CUDA_R_16BF, (int)in, CUBLAS_COMPUTE_32F,
                       CUBLAS_GEMM_DEFAULT) != CUBLAS_STATUS_SUCCESS)
        return GS_ERR_CUDA;
    }
  }
  const int64_t groups = (int64_t)(out / p->g_out) * (in / p->g_in);
  int64_t blocks = (groups + 7) / 8;
  if (blocks > (1 << 20)) blocks = 1 << 20;
  k_group_grad<<<(unsigned)blocks, 256, 0, s>>>(static_cast<const uint16_t*>(W), D, dsdl, (int32_t)out, (int32_t)in,
                                                p->g_out, p->g_in, dlogits);
  note_launch();
  return cudaGetLastError() == cudaSuccess ? GS_OK : GS_ERR_CUDA;
}

}  // namespace gs
