// C ABI of the group-sparse linear layer: host-side validation, ownership of
// the packed buffers, and dispatch to the pack / decode / prefill kernels.
#include "gs_common.cuh"
#include <utility>
#include <algorithm>

#include <atomic>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <new>
#include <vector>

namespace gs {
namespace {

constexpr int kMaxDevices = 64;
std::mutex g_flag_mu;
int* g_flags[kMaxDevices] = {nullptr};
std::atomic<int64_t> g_launches{0};
std::atomic<uint64_t> g_timeout_epoch{0};
// test hooks: countdown to a failing allocation (0 = off), injected wait limits
std::atomic<int64_t> g_fail_alloc_in{0};
std::atomic<uint64_t> g_inject_ns[4] = {{0}, {0}, {0}, {0}};

// Token count at and above which gs_linear uses the tensor-core kernels: one
// decode launch covers up to 16 tokens, while the tensor-core kernels' time is
// flat up to 128.  At T = 17 / 24 / 32 a batched LLaMA-2-13B block takes
// 0.098 ms there against 0.144-0.156 ms as two decode launches (7B 0.073 vs
// 0.097-0.107; Qwen2.5-7B even), and one call per layer 0.30 against 0.38-0.49.
constexpr int64_t kPrefillMinTokens = 17;

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

void free_buffers(gs_packed* p) {
  if (!p) return;
  int cur = -1;
  cudaGetDevice(&cur);
  if (cur != p->device) cudaSetDevice(p->device);
  if (p->offsets) cudaFree(p->offsets);
  if (p->row_idx) cudaFree(p->row_idx);
  if (p->tiles) cudaFree(p->tiles);
  if (p->win_off16) cudaFree(p->win_off16);
  if (p->kmask16) cudaFree(p->kmask16);
  decode_release(p);
  sq_release(p);
  if (cur >= 0 && cur != p->device) cudaSetDevice(cur);
  p->offsets = nullptr;
  p->row_idx = nullptr;
  p->tiles = nullptr;
  p->win_off16 = nullptr;
  p->kmask16 = nullptr;
}

gs_status dev_alloc(void** ptr, size_t bytes, size_t* total) {
  *ptr = nullptr;
  if (bytes == 0) return GS_OK;
  const gs_status st = lib_malloc(ptr, bytes);
  if (st == GS_OK) *total += bytes;
  return st;
}

gs_status check_handle(const gs_packed* p) {
  if (!p) return GS_ERR_INVALID_ARG;
  if (p->out <= 0 || p->in <= 0 || p->G <= 0 || !p->offsets) return GS_ERR_INVALID_ARG;
  if (is_square(p) ? (!p->gwoff || !p->gwmask) : (!p->win_off16 || !p->kmask16)) return GS_ERR_INVALID_ARG;
  return GS_OK;
}

}  // namespace

int* device_error_flag() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lk(g_flag_mu);
  if (!g_flags[dev]) {
    int* f = nullptr;
    if (cudaMalloc(&f, 2 * sizeof(int)) != cudaSuccess) return nullptr;
    if (cudaMemset(f, 0, 2 * sizeof(int)) != cudaSuccess) {
      cudaFree(f);
      return nullptr;
    }
    g_flags[dev] = f;
  }
  return g_flags[dev];
}

void note_launch(int64_t n) { g_launches.fetch_add(n, std::memory_order_relaxed); }

uint64_t timeout_epoch() { return g_timeout_epoch.load(std::memory_order_acquire); }

gs_status lib_malloc(void** ptr, size_t bytes) {
  *ptr = nullptr;
  int64_t n = g_fail_alloc_in.load(std::memory_order_relaxed);
  while (n > 0 && !g_fail_alloc_in.compare_exchange_weak(n, n - 1)) {
  }
  if (n == 1) return GS_ERR_OOM;   // the armed allocation fails as if the device were full
  const cudaError_t e = cudaMalloc(ptr, bytes);
  if (e == cudaErrorMemoryAllocation) {
    cudaGetLastError();
    *ptr = nullptr;
    return GS_ERR_OOM;
  }
  if (e != cudaSuccess) {
    *ptr = nullptr;
    return GS_ERR_CUDA;
  }
  return GS_OK;
}

uint64_t take_injected_wait(int family) {
  if (family < GS_ALGO_DECODE || family > GS_ALGO_PREFILL_DENSE) return 0;
  return g_inject_ns[family].exchange(0);
}

}  // namespace gs

using namespace gs;

extern "C" {

// Row groups 1 x kw (kw = 256 or 128): the chunk-major layout and everything
// the decode and prefill kernels need.
static gs_status pack_rows(const void* W_dev, const uint8_t* mask_dev, int64_t out, int64_t in, int32_t kw,
                           void* stream, gs_packed** handle) {
  if (handle) *handle = nullptr;
  if (!W_dev || !mask_dev || !handle) return GS_ERR_INVALID_ARG;
  if (out <= 0 || in <= 0 || out > INT32_MAX || in > INT32_MAX) return GS_ERR_INVALID_ARG;
  if (kw != 256 && kw != 128) return GS_ERR_UNSUPPORTED;
  if (in % kw != 0) return GS_ERR_INVALID_ARG;
  if (!aligned16(W_dev)) return GS_ERR_INVALID_ARG;
  const int64_t G = in / kw;
  if (out * G >= (int64_t)INT32_MAX) return GS_ERR_UNSUPPORTED;
  cudaStream_t s = static_cast<cudaStream_t>(stream);

  gs_packed* p = new (std::nothrow) gs_packed;
  if (!p) return GS_ERR_OOM;
  std::memset(p, 0, sizeof(*p));
  if (cudaGetDevice(&p->device) != cudaSuccess) {
    delete p;
    return GS_ERR_CUDA;
  }
  if (!device_error_flag()) {  // allocated here so later calls never allocate (graph capture)
    delete p;
    return GS_ERR_CUDA;
  }
  p->out = out;
  p->in = in;
  p->G = (int32_t)G;
  p->nw16 = (int32_t)((out + kWin16 - 1) / kWin16);
  p->g_out = 1;
  p->g_in = kw;
  p->Gout = (int32_t)out;

  size_t total = 0;
  int32_t* cnt = nullptr;
  gs_status st = GS_OK;
  const size_t E = (size_t)p->G * (size_t)p->nw16;
  if ((st = dev_alloc((void**)&p->offsets, sizeof(int64_t) * (size_t)(G + 1), &total)) != GS_OK) goto fail;
  if ((st = dev_alloc((void**)&p->win_off16, sizeof(int32_t) * (size_t)p->G * (size_t)(p->nw16 + 1), &total)) !=
      GS_OK)
    goto fail;
  if ((st = dev_alloc((void**)&p->kmask16, sizeof(uint16_t) * E, &total)) != GS_OK) goto fail;
  {
    size_t scratch = 0;
    if ((st = dev_alloc((void**)&cnt, sizeof(int32_t) * E, &scratch)) != GS_OK) goto fail;
  }
  if ((st = launch_pack_count_scan(mask_dev, p, s, cnt)) != GS_OK) goto fail;
  {
    int64_t kept = 0;
    if (cudaMemcpyAsync(&kept, p->offsets + G, sizeof(int64_t), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
        cudaStreamSynchronize(s) != cudaSuccess) {
      st = GS_ERR_CUDA;
      goto fail;
    }
    p->kept = kept;
  }
  cudaFree(cnt);
  cnt = nullptr;
  if ((st = dev_alloc((void**)&p->row_idx, sizeof(int32_t) * (size_t)p->kept, &total)) != GS_OK) goto fail;
  if ((st = dev_alloc((void**)&p->tiles, 2 * (size_t)kw * (size_t)p->kept, &total)) != GS_OK) goto fail;
  p->device_bytes = total;
  if ((st = launch_pack_compact(W_dev, p, s)) != GS_OK) goto fail;
  if ((st = decode_prepare(p, s)) != GS_OK) goto fail;
  if ((st = prefill_prepare_weight_maps(p)) != GS_OK) goto fail;
  *handle = p;
  return GS_OK;

fail:
  if (cnt) cudaFree(cnt);
  free_buffers(p);
  delete p;
  return st;
}

gs_status gs_pack(const void* W_dev, const uint8_t* mask_dev, int64_t out, int64_t in, int32_t group_in,
                  void* stream, gs_packed** handle) {
  if (handle) *handle = nullptr;
  if (!W_dev || !mask_dev || !handle) return GS_ERR_INVALID_ARG;
  if (group_in != kGroupIn) return GS_ERR_UNSUPPORTED;
  return pack_rows(W_dev, mask_dev, out, in, kGroupIn, stream, handle);
}

gs_status gs_pack_groups(const void* W_dev, const uint8_t* mask_dev, int64_t out, int64_t in, int32_t g_out,
                         int32_t g_in, void* stream, gs_packed** handle) {
  if (handle) *handle = nullptr;
  if (!W_dev || !mask_dev || !handle) return GS_ERR_INVALID_ARG;
  if (out <= 0 || in <= 0 || out > INT32_MAX || in > INT32_MAX || g_out <= 0 || g_in <= 0) return GS_ERR_INVALID_ARG;
  if (g_out == 1 && (g_in == 256 || g_in == 128)) return pack_rows(W_dev, mask_dev, out, in, g_in, stream, handle);
  if (!sq_shape_supported(g_out, g_in)) return GS_ERR_UNSUPPORTED;
  if (out % g_out != 0 || in % g_in != 0) return GS_ERR_INVALID_ARG;   // the groups must tile W exactly
  if (!aligned16(W_dev)) return GS_ERR_INVALID_ARG;
  const int64_t Gout = out / g_out, Gin = in / g_in;
  if (Gout * Gin >= (int64_t)INT32_MAX || Gin > 65535) return GS_ERR_UNSUPPORTED;
  gs_packed* p = new (std::nothrow) gs_packed;
  if (!p) return GS_ERR_OOM;
  std::memset(p, 0, sizeof(*p));
  if (cudaGetDevice(&p->device) != cudaSuccess) {
    delete p;
    return GS_ERR_CUDA;
  }
  if (!device_error_flag()) {
    delete p;
    return GS_ERR_CUDA;
  }
  p->out = out;
  p->in = in;
  p->g_out = g_out;
  p->g_in = g_in;
  p->G = (int32_t)Gin;
  p->Gout = (int32_t)Gout;
  p->nwin = (int32_t)((out + 127) / 128);
  const gs_status st = sq_pack(W_dev, mask_dev, p, static_cast<cudaStream_t>(stream));
  if (st != GS_OK) {
    free_buffers(p);
    delete p;
    return st;
  }
  *handle = p;
  return GS_OK;
}

gs_status gs_packed_group_shape(const gs_packed* p, int32_t* g_out, int32_t* g_in) {
  if (check_handle(p) != GS_OK) return GS_ERR_INVALID_ARG;
  if (g_out) *g_out = p->g_out;
  if (g_in) *g_in = p->g_in;
  return GS_OK;
}

static gs_status linear_impl(const void* x_dev, const gs_packed* p, int64_t T, void* y_dev, void* stream,
                             gs_algo algo) {
  if (check_handle(p) != GS_OK) return GS_ERR_INVALID_ARG;
  if (T < 0 || T > INT32_MAX) return GS_ERR_INVALID_ARG;
  if (algo != GS_ALGO_AUTO && algo != GS_ALGO_DECODE && algo != GS_ALGO_PREFILL && algo != GS_ALGO_PREFILL_DENSE)
    return GS_ERR_INVALID_ARG;
  if (T == 0) return GS_OK;
  if (!x_dev || !y_dev) return GS_ERR_INVALID_ARG;
  if (!aligned16(x_dev) || !aligned16(y_dev)) return GS_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (is_square(p)) return sq_linear_batched(&x_dev, &p, 1, T, &y_dev, s);   // one kernel family for every T
  if (algo == GS_ALGO_AUTO) {
    // the same per-layer choice as gs_linear_batched makes
    if (T < kPrefillMinTokens) algo = GS_ALGO_DECODE;
    else if (prefill_prefers_dense(p, T)) algo = GS_ALGO_PREFILL_DENSE;
    else algo = p->G <= prefill_max_chunks() ? GS_ALGO_PREFILL : GS_ALGO_DECODE;
  }
  if (algo == GS_ALGO_PREFILL) return launch_prefill(x_dev, p, T, y_dev, s);
  if (algo == GS_ALGO_PREFILL_DENSE) {
    if (p->kept == 0) return cudaMemsetAsync(y_dev, 0, (size_t)T * (size_t)p->out * 2, s) == cudaSuccess ? GS_OK : GS_ERR_CUDA;
    return launch_prefill_dense(&x_dev, &p, 1, T, &y_dev, s);
  }
  // decode family: token blocks of at most decode_max_tokens()
  const int64_t blk = decode_max_tokens();
  for (int64_t t0 = 0; t0 < T; t0 += blk) {
    const int64_t tb = T - t0 < blk ? T - t0 : blk;
    const void* xb = static_cast<const uint16_t*>(x_dev) + t0 * p->in;
    void* yb = static_cast<uint16_t*>(y_dev) + t0 * p->out;
    const gs_status st = launch_decode(&p, &xb, &yb, 1, (int)tb, s);
    if (st != GS_OK) return st;
  }
  return GS_OK;
}

gs_status gs_linear(const void* x_dev, const gs_packed* p, int64_t T, void* y_dev, void* stream) {
  return linear_impl(x_dev, p, T, y_dev, stream, GS_ALGO_AUTO);
}

gs_status gs_linear_ex(const void* x_dev, const gs_packed* p, int64_t T, void* y_dev, void* stream,
                       gs_algo algo) {
  return linear_impl(x_dev, p, T, y_dev, stream, algo);
}

gs_status gs_linear_batched(int32_t n, const void* const* xs_dev, const gs_packed* const* ps, int64_t T,
                            void* const* ys_dev, void* stream) {
  if (n < 0 || n > 32) return GS_ERR_INVALID_ARG;
  if (n == 0) return GS_OK;
  if (!xs_dev || !ps || !ys_dev) return GS_ERR_INVALID_ARG;
  if (T < 0 || T > INT32_MAX) return GS_ERR_INVALID_ARG;
  for (int i = 0; i < n; ++i) {
    if (check_handle(ps[i]) != GS_OK) return GS_ERR_INVALID_ARG;
    if (T > 0 && (!xs_dev[i] || !ys_dev[i] || !aligned16(xs_dev[i]) || !aligned16(ys_dev[i])))
      return GS_ERR_INVALID_ARG;
  }
  if (T == 0) return GS_OK;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  {
    // square-group layers take their own launches; the 1 x 256 layers continue below
    std::vector<const void*> xq;
    std::vector<const gs_packed*> pq;
    std::vector<void*> yq;
    std::vector<const void*> xr;
    std::vector<const gs_packed*> pr;
    std::vector<void*> yr;
    for (int i = 0; i < n; ++i) {
      if (is_square(ps[i])) {
        xq.push_back(xs_dev[i]);
        pq.push_back(ps[i]);
        yq.push_back(ys_dev[i]);
      } else {
        xr.push_back(xs_dev[i]);
        pr.push_back(ps[i]);
        yr.push_back(ys_dev[i]);
      }
    }
    if (!pq.empty()) {
      const gs_status st = sq_linear_batched(xq.data(), pq.data(), (int)pq.size(), T, yq.data(), s);
      if (st != GS_OK) return st;
      if (pr.empty()) return GS_OK;
      return gs_linear_batched((int32_t)pr.size(), xr.data(), pr.data(), T, yr.data(), stream);
    }
    // 1 x 128 and 1 x 256 layers take separate launches (one chunk width per kernel)
    int n128 = 0;
    for (int i = 0; i < n; ++i) n128 += ps[i]->g_in == 128 ? 1 : 0;
    if (n128 > 0 && n128 < n) {
      std::vector<const void*> xa, xb;
      std::vector<const gs_packed*> pa, pb;
      std::vector<void*> ya, yb;
      for (int i = 0; i < n; ++i) {
        const bool narrow = ps[i]->g_in == 128;
        (narrow ? xa : xb).push_back(xs_dev[i]);
        (narrow ? pa : pb).push_back(ps[i]);
        (narrow ? ya : yb).push_back(ys_dev[i]);
      }
      const gs_status st = gs_linear_batched((int32_t)pa.size(), xa.data(), pa.data(), T, ya.data(), stream);
      if (st != GS_OK) return st;
      return gs_linear_batched((int32_t)pb.size(), xb.data(), pb.data(), T, yb.data(), stream);
    }
  }
  if (T >= kPrefillMinTokens) {
    // layers the prefill kernel takes share batched launches; any other goes alone
    // (layers the zero-filled kernel runs faster go there, batched the same way)
    std::vector<const void*> xp, xd;
    std::vector<const gs_packed*> pp, pd;
    std::vector<void*> yp, yd;
    for (int i = 0; i < n; ++i) {
      if (prefill_prefers_dense(ps[i], T)) {
        xd.push_back(xs_dev[i]);
        pd.push_back(ps[i]);
        yd.push_back(ys_dev[i]);
      } else if (ps[i]->G <= prefill_max_chunks()) {
        xp.push_back(xs_dev[i]);
        pp.push_back(ps[i]);
        yp.push_back(ys_dev[i]);
      } else {
        const gs_status st = linear_impl(xs_dev[i], ps[i], T, ys_dev[i], stream, GS_ALGO_AUTO);
        if (st != GS_OK) return st;
      }
    }
    if (!pd.empty()) {
      const gs_status st = launch_prefill_dense(xd.data(), pd.data(), (int)pd.size(), T, yd.data(), s);
      if (st != GS_OK) return st;
    }
    if (pp.empty()) return GS_OK;
    return launch_prefill_batched(xp.data(), pp.data(), (int)pp.size(), T, yp.data(), s);
  }
  const int64_t blk = decode_max_tokens();
  std::vector<const void*> xb(n);
  std::vector<void*> yb(n);
  for (int64_t t0 = 0; t0 < T; t0 += blk) {
    const int64_t tb = T - t0 < blk ? T - t0 : blk;
    for (int i = 0; i < n; ++i) {
      xb[i] = static_cast<const uint16_t*>(xs_dev[i]) + t0 * ps[i]->in;
      yb[i] = static_cast<uint16_t*>(ys_dev[i]) + t0 * ps[i]->out;
    }
    const gs_status st = launch_decode(ps, xb.data(), yb.data(), n, (int)tb, s);
    if (st != GS_OK) return st;
  }
  return GS_OK;
}

gs_status gs_select_groups(const float* logits_dev, int64_t n, uint8_t* mask_dev, int64_t* kept_dev,
                           void* stream) {
  if (n < 0 || n >= (int64_t(1) << 36)) return GS_ERR_INVALID_ARG;
  if (kept_dev && (reinterpret_cast<uintptr_t>(kept_dev) & 7u) != 0) return GS_ERR_INVALID_ARG;
  if (n > 0) {
    if (!logits_dev || !mask_dev || !aligned16(logits_dev) || !aligned16(mask_dev)) return GS_ERR_INVALID_ARG;
    const uintptr_t l0 = reinterpret_cast<uintptr_t>(logits_dev), m0 = reinterpret_cast<uintptr_t>(mask_dev);
    if (l0 < m0 + (uintptr_t)n && m0 < l0 + 4 * (uintptr_t)n) return GS_ERR_INVALID_ARG;   // overlap
  }
  return launch_select(logits_dev, n, mask_dev, kept_dev, static_cast<cudaStream_t>(stream));
}

gs_status gs_unpack(const gs_packed* p, void* W_hat_dev, void* stream) {
  if (check_handle(p) != GS_OK || !W_hat_dev || !aligned16(W_hat_dev)) return GS_ERR_INVALID_ARG;
  if (is_square(p)) return sq_unpack(p, W_hat_dev, static_cast<cudaStream_t>(stream));
  return launch_unpack(p, W_hat_dev, static_cast<cudaStream_t>(stream));
}

gs_status gs_packed_info(const gs_packed* p, int64_t* out, int64_t* in, int64_t* kept_groups,
                         size_t* device_bytes) {
  if (check_handle(p) != GS_OK) return GS_ERR_INVALID_ARG;
  if (out) *out = p->out;
  if (in) *in = p->in;
  if (kept_groups) *kept_groups = p->kept;
  if (device_bytes) *device_bytes = p->device_bytes;
  return GS_OK;
}

gs_status gs_packed_export(const gs_packed* p, int64_t* offsets_host, int32_t* row_idx_host, uint16_t* tiles_host,
                           int32_t* win_off16_host, uint16_t* kmask16_host) {
  if (check_handle(p) != GS_OK) return GS_ERR_INVALID_ARG;
  if (is_square(p) && (win_off16_host || kmask16_host)) return GS_ERR_INVALID_ARG;   // no 16-row windows
  if (cudaDeviceSynchronize() != cudaSuccess) return GS_ERR_CUDA;
  const size_t G = (size_t)p->G, nw = (size_t)p->nw16, K = (size_t)p->kept;
  if (offsets_host && cudaMemcpy(offsets_host, p->offsets, sizeof(int64_t) * (G + 1), cudaMemcpyDeviceToHost))
    return GS_ERR_CUDA;
  if (row_idx_host && K && cudaMemcpy(row_idx_host, p->row_idx, sizeof(int32_t) * K, cudaMemcpyDeviceToHost))
    return GS_ERR_CUDA;
  const size_t tile_bytes = 2 * (size_t)p->g_out * (size_t)p->g_in;
  if (tiles_host && K && cudaMemcpy(tiles_host, p->tiles, tile_bytes * K, cudaMemcpyDeviceToHost))
    return GS_ERR_CUDA;
  if (win_off16_host &&
      cudaMemcpy(win_off16_host, p->win_off16, sizeof(int32_t) * G * (nw + 1), cudaMemcpyDeviceToHost))
    return GS_ERR_CUDA;
  if (kmask16_host && cudaMemcpy(kmask16_host, p->kmask16, sizeof(uint16_t) * G * nw, cudaMemcpyDeviceToHost))
    return GS_ERR_CUDA;
  return GS_OK;
}

void gs_free(gs_packed* p) {
  if (!p) return;
  free_buffers(p);
  delete p;
}

const char* gs_status_string(gs_status s) {
  switch (s) {
    case GS_OK: return "ok";
    case GS_ERR_INVALID_ARG: return "invalid argument";
    case GS_ERR_UNSUPPORTED: return "unsupported";
    case GS_ERR_OOM: return "out of device memory";
    case GS_ERR_CUDA: return "CUDA error";
    case GS_ERR_DEVICE_TIMEOUT: return "device wait timed out";
  }
  return "unknown status";
}

gs_status gs_device_status(void* stream) {
  if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return GS_ERR_CUDA;
  int* f = device_error_flag();
  if (!f) return GS_ERR_CUDA;
  int v = 0;
  if (cudaMemcpy(&v, f, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess) return GS_ERR_CUDA;
  if (v != 0) {
    cudaMemset(f, 0, sizeof(int));
    // a kernel that gave up may have left split counters half counted: every
    // decode scratch slot is re-zeroed before its next use
    g_timeout_epoch.fetch_add(1, std::memory_order_acq_rel);
    return GS_ERR_DEVICE_TIMEOUT;
  }
  return GS_OK;
}

gs_status gs_preserved_rates(int32_t n, const int64_t* kept_host, const int64_t* d_out_host, const int64_t* d_in_host,
                             int64_t group_weights, double* rates_host, double* global_host, int32_t n_qkv,
                             const int32_t* qkv_host, double* qkv_rates_host) {
  if (n < 0 || n_qkv < 0 || group_weights <= 0) return GS_ERR_INVALID_ARG;
  if (n > 0 && (!kept_host || !d_out_host || !d_in_host)) return GS_ERR_INVALID_ARG;
  if (n_qkv > 0 && (!qkv_host || !qkv_rates_host)) return GS_ERR_INVALID_ARG;
  // exact integer totals: every count and size below 2^62
  constexpr int64_t kLim = int64_t(1) << 62;
  int64_t active = 0, total = 0;
  for (int32_t i = 0; i < n; ++i) {
    const int64_t k = kept_host[i], a = d_out_host[i], b = d_in_host[i];
    if (a <= 0 || b <= 0 || k < 0 || a > kLim / b) return GS_ERR_INVALID_ARG;
    const int64_t size = a * b;
    if (k > size / group_weights) return GS_ERR_INVALID_ARG;   // more kept weights than the layer has
    if (active > kLim - k * group_weights || total > kLim - size) return GS_ERR_INVALID_ARG;
    active += k * group_weights;
    total += size;
  }
  for (int32_t j = 0; j < n_qkv; ++j)
    for (int t = 0; t < 3; ++t)
      if (qkv_host[3 * j + t] < 0 || qkv_host[3 * j + t] >= n) return GS_ERR_INVALID_ARG;
  auto rate = [&](int32_t i) {
    return (double)(kept_host[i] * group_weights) / (double)(d_out_host[i] * d_in_host[i]);
  };
  if (rates_host)
    for (int32_t i = 0; i < n; ++i) rates_host[i] = rate(i);
  if (global_host) *global_host = total > 0 ? (double)active / (double)total : 0.0;
  for (int32_t j = 0; j < n_qkv; ++j)
    qkv_rates_host[j] = (rate(qkv_host[3 * j]) + rate(qkv_host[3 * j + 1]) + rate(qkv_host[3 * j + 2])) / 3.0;
  return GS_OK;
}

gs_status gs_gumbel_select(const float* logits_dev, const float* noise_dev, int64_t n, float tau, uint8_t* mask_dev,
                           float* dsdl_dev, int64_t* kept_dev, void* stream) {
  if (n < 0 || n >= (int64_t(1) << 36) || !(tau > 0.f) || !(tau < 3.0e38f)) return GS_ERR_INVALID_ARG;
  if (kept_dev && (reinterpret_cast<uintptr_t>(kept_dev) & 7u) != 0) return GS_ERR_INVALID_ARG;
  if (n > 0) {
    if (!logits_dev || !noise_dev || !mask_dev) return GS_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(logits_dev) & 3u) || (reinterpret_cast<uintptr_t>(noise_dev) & 3u) ||
        (dsdl_dev && (reinterpret_cast<uintptr_t>(dsdl_dev) & 3u)))
      return GS_ERR_INVALID_ARG;
    // outputs must not overlap the inputs or each other
    const uintptr_t lo[4] = {reinterpret_cast<uintptr_t>(logits_dev), reinterpret_cast<uintptr_t>(noise_dev),
                             reinterpret_cast<uintptr_t>(mask_dev), reinterpret_cast<uintptr_t>(dsdl_dev)};
    const uintptr_t len[4] = {4 * (uintptr_t)n, 4 * (uintptr_t)n, (uintptr_t)n, dsdl_dev ? 4 * (uintptr_t)n : 0};
    for (int i = 2; i < 4; ++i)
      for (int j = 0; j < 4; ++j)
        if (i != j && len[i] && len[j] && lo[i] < lo[j] + len[j] && lo[j] < lo[i] + len[i]) return GS_ERR_INVALID_ARG;
  }
  return launch_gumbel(logits_dev, noise_dev, n, tau, mask_dev, dsdl_dev, kept_dev, static_cast<cudaStream_t>(stream));
}

gs_status gs_masked_linear_backward_workspace(const gs_packed* p, int32_t want_dx, size_t* bytes) {
  if (check_handle(p) != GS_OK || !bytes) return GS_ERR_INVALID_ARG;
  *bytes = backward_workspace_bytes(p, want_dx != 0);
  return GS_OK;
}

gs_status gs_masked_linear_backward(const void* x_dev, const void* W_dev, const gs_packed* p, const void* dy_dev,
                                    int64_t T, const float* dsdl_dev, float* dlogits_dev, void* dx_dev,
                                    void* workspace_dev, size_t workspace_bytes, void* stream) {
  if (check_handle(p) != GS_OK) return GS_ERR_INVALID_ARG;
  if (T <= 0 || T > INT32_MAX) return GS_ERR_INVALID_ARG;
  if (!x_dev || !W_dev || !dy_dev || !dsdl_dev || !dlogits_dev || !workspace_dev) return GS_ERR_INVALID_ARG;
  if (!aligned16(x_dev) || !aligned16(W_dev) || !aligned16(dy_dev) || !aligned16(workspace_dev) ||
      (reinterpret_cast<uintptr_t>(dsdl_dev) & 3u) || (reinterpret_cast<uintptr_t>(dlogits_dev) & 3u) ||
      (dx_dev && !aligned16(dx_dev)))
    return GS_ERR_INVALID_ARG;
  if (p->out > INT32_MAX || p->in > INT32_MAX) return GS_ERR_UNSUPPORTED;
  if (workspace_bytes < backward_workspace_bytes(p, dx_dev != nullptr)) return GS_ERR_INVALID_ARG;
  return launch_backward(x_dev, W_dev, p, dy_dev, T, dsdl_dev, dlogits_dev, dx_dev, workspace_dev,
                         static_cast<cudaStream_t>(stream));
}

gs_status gs_debug_fail_alloc(int64_t nth) {
  if (nth < 0) return GS_ERR_INVALID_ARG;
  g_fail_alloc_in.store(nth, std::memory_order_relaxed);
  return GS_OK;
}

gs_status gs_debug_inject_wait(gs_algo family, uint64_t limit_ns) {
  if (family != GS_ALGO_DECODE && family != GS_ALGO_PREFILL && family != GS_ALGO_PREFILL_DENSE)
    return GS_ERR_INVALID_ARG;
  if (limit_ns > 1000000000ull) return GS_ERR_INVALID_ARG;
  g_inject_ns[family].store(limit_ns);
  return GS_OK;
}

int64_t gs_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

}  // extern "C"
