// Decode-regime group-sparse linear for square g x g groups (Sec. 2.1 with
// g_out = g_in = g; Eq. 1), T <= 16 tokens: memory-bound, so the design
// streams the kept tiles once at HBM rate instead of feeding the tensor-core
// pipeline of the square prefill kernel (whose per-column-block handshake
// dominates when each step carries only a few rows' worth of work).
//
// A unit is one slab of 16 output rows (rows 16 q .. 16 q + 15: one block row
// for g = 16, a 16-row slice of one for larger g) and is owned by one CTA of 4
// warps.  Warp j takes a contiguous quarter of the column blocks and compacts
// the kept ones of the slab's block row into a list (tile indices from the
// block row's entries of a pack-time [block row][column block] table, read
// with coalesced loads).  It then streams, per kept tile, granules of 16 rows
// x KC = min(g, 64) columns of the tile (row-major, so each row is contiguous)
// together with the same KC columns of x for the first T token rows through a
// private ring in shared memory with 16-byte cp.async, XOR-swizzled so that
// ldmatrix reads both without bank conflicts.  A granule is KC / 16 steps of
// mma.sync m16n8k16 (bf16 in, fp32 accumulate).  At the end the warps' partial
// sums meet in shared memory and are added in warp order (a fixed order:
// results do not depend on timing), then stored as bf16 (round to nearest
// even).
//
// Units are independent CTAs, heaviest layer first; no unit waits on another.
#include "gs_common.cuh"

#include <algorithm>
#include <cstring>
#include <vector>

namespace gs {
namespace {

constexpr int kQdWarps = 4;
constexpr int kQdThreads = kQdWarps * 32;
constexpr int kQdRows = 16;            // output rows per unit
constexpr int kQdRingBytes = 8192;     // per warp (small: six CTAs per SM measured fastest)
constexpr int kQdListMax = 64;         // column blocks a warp scans per round
constexpr int kQdMaxLayers = 8;
constexpr int kQdMaxT = 16;
constexpr int kQdSmem = kQdWarps * (kQdRingBytes + kQdListMax * 8);
static_assert(kQdWarps * 2 * 4 * 32 * 4 <= kQdWarps * kQdRingBytes, "reduction buffer fits in the rings");

struct QdLayer {
  const uint16_t* x;        // [T][in]
  const uint16_t* tiles;    // [kept][g][g]
  const int32_t* gtidx;     // [Gout][Gin]: packed tile of group (u, v) or -1
  uint16_t* y;              // [T][out]
  int32_t in, out, Gin, unit_begin;
};
struct QdParams {
  QdLayer L[kQdMaxLayers];
  int32_t n_layers, T;
};

// Streaming granule: 16 rows x KC columns of a tile plus the same KC columns
// of x for 8 NB token rows, KC = min(g, 64) (a 128-wide tile is two granules).
template <int G, int NB>
struct Qd {
  static constexpr int KC = G < 64 ? G : 64;
  static constexpr int kH = G / KC;                                   // granules per tile
  static constexpr int kTok = 8 * NB;                                 // x rows per granule
  static constexpr int kWBytes = kQdRows * KC * 2;
  static constexpr int kXBytes = kTok * KC * 2;
  static constexpr int kSlotBytes = kWBytes + kXBytes;
  static constexpr int kSlots = kQdRingBytes / kSlotBytes;
  static constexpr int kCPR = KC / 8;                                 // 16-byte chunks per granule row
  static constexpr int kKB = KC / 16;                                 // k16 blocks per granule
  static constexpr int kSwzDiv = kCPR >= 8 ? 1 : 8 / kCPR;
  static constexpr int kSwzMask = (kCPR >= 8 ? 8 : kCPR) - 1;
  static_assert(kSlots >= 2, "ring depth");
  // byte offset of 16-byte chunk c of row r in a granule block (rows at the
  // granule pitch, chunks XOR-permuted so the 8 rows one ldmatrix phase reads
  // fall in distinct bank groups)
  __device__ static __forceinline__ uint32_t off(int r, int c) {
    return (uint32_t)(r * (KC * 2) + ((c ^ ((r / kSwzDiv) & kSwzMask)) << 4));
  }
};

__device__ __forceinline__ int qd_layer_of(const QdParams& P, int u) {
  int l = 0;
  while (l + 1 < P.n_layers && P.L[l + 1].unit_begin <= u) ++l;
  return l;
}

__device__ __forceinline__ uint32_t qd_smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void qd_cp16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}

template <int NB, int G>
__global__ void __launch_bounds__(kQdThreads) k_sq_decode(const __grid_constant__ QdParams P) {
  using C = Qd<G, NB>;
  extern __shared__ __align__(128) uint8_t qd_smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int2* list = reinterpret_cast<int2*>(qd_smem + kQdWarps * kQdRingBytes) + warp * kQdListMax;
  const uint32_t ring_s = qd_smem_u32(qd_smem + warp * kQdRingBytes);

  const int unit = blockIdx.x;
  const QdLayer& L = P.L[qd_layer_of(P, unit)];
  const int row0 = (unit - L.unit_begin) * kQdRows;
  const int u = row0 / G, r0 = row0 % G;              // block row and first row inside its tiles
  const int32_t* trow = L.gtidx + (int64_t)u * L.Gin;
  const int T = P.T;
  const int t_rows = min(T, C::kTok);   // x rows a granule carries

  // this warp's column blocks
  const int per = (L.Gin + kQdWarps - 1) / kQdWarps;
  const int va = min(warp * per, L.Gin), vb = min(va + per, L.Gin);

  float acc[NB][4];
#pragma unroll
  for (int nb = 0; nb < NB; ++nb)
#pragma unroll
    for (int e = 0; e < 4; ++e) acc[nb][e] = 0.f;

  for (int v0 = va; v0 < vb; v0 += kQdListMax) {
    const int v1 = min(v0 + kQdListMax, vb);
    // kept column blocks of this batch (v0 .. v1 - 1), in ascending order (the block row's
    // tile indices are contiguous: all loads go out before the first use)
    constexpr int kLd = kQdListMax / 32;
    int tv[kLd];
#pragma unroll
    for (int q = 0; q < kLd; ++q) {
      const int v = v0 + 32 * q + lane;
      tv[q] = v < v1 ? trow[v] : -1;
    }
    int n_items = 0;
#pragma unroll
    for (int q = 0; q < kLd; ++q) {
      const bool kept = tv[q] >= 0;
      const uint32_t ballot = __ballot_sync(0xffffffffu, kept);
      if (kept) list[n_items + __popc(ballot & ((1u << lane) - 1u))] = make_int2(v0 + 32 * q + lane, tv[q]);
      n_items += __popc(ballot);
    }
    __syncwarp();
    const int n_gran = n_items * C::kH;

    // granule k: item k / kH, columns (k % kH) KC .. of its tile and of x
    auto issue = [&](int k) {
      const int2 it = list[k / C::kH];
      const int h = k % C::kH;
      const uint16_t* wsrc = L.tiles + (int64_t)it.y * G * G + (int64_t)r0 * G + h * C::KC;
      const uint16_t* xsrc = L.x + (int64_t)it.x * G + h * C::KC;
      const uint32_t slot = ring_s + (uint32_t)((k % C::kSlots) * C::kSlotBytes);
      for (int e = lane; e < kQdRows * C::kCPR; e += 32) {
        const int r = e / C::kCPR, c = e % C::kCPR;
        qd_cp16(slot + C::off(r, c), wsrc + (int64_t)r * G + 8 * c);
      }
      // x rows of tokens beyond T are left as they are: a token's products stay
      // in its own accumulator column, which is never stored
      for (int e = lane; e < t_rows * C::kCPR; e += 32) {
        const int n = e / C::kCPR, c = e % C::kCPR;
        qd_cp16(slot + C::kWBytes + C::off(n, c), xsrc + (int64_t)n * L.in + 8 * c);
      }
    };
    for (int k = 0; k < C::kSlots; ++k) {
      if (k < n_gran) issue(k);
      asm volatile("cp.async.commit_group;" ::: "memory");
    }
    for (int k = 0; k < n_gran; ++k) {
      asm volatile("cp.async.wait_group %0;" ::"n"(C::kSlots - 1) : "memory");
      __syncwarp();
      const uint32_t slot = ring_s + (uint32_t)((k % C::kSlots) * C::kSlotBytes);
#pragma unroll
      for (int kk = 0; kk < C::kKB; ++kk) {
        // A (W rows): matrix j = lane / 8 is rows 8 (j & 1) .., k chunk 2 kk + (j >> 1)
        uint32_t a0, a1, a2, a3;
        asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                     : "=r"(a0), "=r"(a1), "=r"(a2), "=r"(a3)
                     : "r"(slot + C::off((lane & 7) + 8 * ((lane >> 3) & 1), 2 * kk + (lane >> 4))));
        // B (x rows = tokens): matrix j is tokens 8 (j >> 1) .., k chunk 2 kk + (j & 1)
        uint32_t b[4];
        if constexpr (NB == 2) {
          asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                       : "=r"(b[0]), "=r"(b[1]), "=r"(b[2]), "=r"(b[3])
                       : "r"(slot + C::kWBytes + C::off((lane & 7) + 8 * (lane >> 4), 2 * kk + ((lane >> 3) & 1))));
        } else {
          asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0, %1}, [%2];"
                       : "=r"(b[0]), "=r"(b[1])
                       : "r"(slot + C::kWBytes + C::off(lane & 7, 2 * kk + ((lane >> 3) & 1))));
        }
#pragma unroll
        for (int nb = 0; nb < NB; ++nb)
          asm volatile(
              "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
              "{%0, %1, %2, %3};"
              : "+f"(acc[nb][0]), "+f"(acc[nb][1]), "+f"(acc[nb][2]), "+f"(acc[nb][3])
              : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b[2 * nb]), "r"(b[2 * nb + 1]));
      }
      __syncwarp();   // every lane has read the slot before it is refilled
      if (k + C::kSlots < n_gran) issue(k + C::kSlots);
      asm volatile("cp.async.commit_group;" ::: "memory");
    }
    asm volatile("cp.async.wait_all;" ::: "memory");
    __syncwarp();
  }

  // partial sums of the warps, added in warp order
  __syncthreads();   // every ring is idle: reuse them
  float* red = reinterpret_cast<float*>(qd_smem);   // [warp][nb][4][lane]
#pragma unroll
  for (int nb = 0; nb < NB; ++nb)
#pragma unroll
    for (int e = 0; e < 4; ++e) red[((warp * NB + nb) * 4 + e) * 32 + lane] = acc[nb][e];
  __syncthreads();
  if (warp < NB) {
    const int nb = warp;
    float s[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      s[e] = 0.f;
      for (int j = 0; j < kQdWarps; ++j) s[e] += red[((j * NB + nb) * 4 + e) * 32 + lane];
    }
    // c0, c1: row lane / 4, tokens 2 (lane % 4), + 1; c2, c3: row lane / 4 + 8
    const int n0 = 8 * nb + 2 * (lane & 3);
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int n = n0 + (e & 1), r = (lane >> 2) + 8 * (e >> 1);
      if (n < T) L.y[(int64_t)n * L.out + row0 + r] = __bfloat16_as_ushort(__float2bfloat16_rn(s[e]));
    }
  }
}

template <int NB, int G>
cudaError_t qd_attr() {
  static cudaError_t err = cudaFuncSetAttribute(k_sq_decode<NB, G>, cudaFuncAttributeMaxDynamicSharedMemorySize, kQdSmem);
  return err;
}

template <int G>
gs_status qd_launch(const void* const* xs, const gs_packed* const* ps, const int* idx, int n, int T,
                    void* const* ys, cudaStream_t s) {
  if (T <= 0) return GS_OK;
  const int NB = T > 8 ? 2 : 1;
  if ((NB == 2 ? qd_attr<2, G>() : qd_attr<1, G>()) != cudaSuccess) return GS_ERR_CUDA;
  QdParams P;
  std::memset(&P, 0, sizeof(P));
  int64_t units = 0;
  for (int k = 0; k < n; ++k) {
    const gs_packed* p = ps[idx[k]];
    QdLayer& L = P.L[k];
    L.x = static_cast<const uint16_t*>(xs[idx[k]]);
    L.tiles = p->tiles;
    L.gtidx = p->gtidx;
    L.y = static_cast<uint16_t*>(ys[idx[k]]);
    L.in = (int32_t)p->in;
    L.out = (int32_t)p->out;
    L.Gin = p->G;
    L.unit_begin = (int32_t)units;
    units += p->out / kQdRows;
  }
  if (units == 0) return GS_OK;
  if (units > INT32_MAX) return GS_ERR_UNSUPPORTED;
  P.n_layers = n;
  P.T = T;
  if (NB == 2) k_sq_decode<2, G><<<(unsigned)units, kQdThreads, kQdSmem, s>>>(P);
  else k_sq_decode<1, G><<<(unsigned)units, kQdThreads, kQdSmem, s>>>(P);
  note_launch();
  return cudaGetLastError() == cudaSuccess ? GS_OK : GS_ERR_CUDA;
}

}  // namespace

int sq_decode_max_tokens() { return kQdMaxT; }

gs_status sq_decode_batched(const void* const* xs, const gs_packed* const* ps, const int* idx, int n, int T,
                            void* const* ys, cudaStream_t s) {
  if (n <= 0 || T <= 0) return GS_OK;
  if (T > kQdMaxT || n > kQdMaxLayers) return GS_ERR_UNSUPPORTED;
  const int g = ps[idx[0]]->g_out;
  for (int k = 0; k < n; ++k) {
    const gs_packed* p = ps[idx[k]];
    if (p->g_out != g || p->g_in != g || p->kept == 0 || p->out % kQdRows != 0) return GS_ERR_UNSUPPORTED;
  }
  switch (g) {
    case 16: return qd_launch<16>(xs, ps, idx, n, T, ys, s);
    case 32: return qd_launch<32>(xs, ps, idx, n, T, ys, s);
    case 64: return qd_launch<64>(xs, ps, idx, n, T, ys, s);
    case 128: return qd_launch<128>(xs, ps, idx, n, T, ys, s);
    default: return GS_ERR_UNSUPPORTED;
  }
}

}  // namespace gs
