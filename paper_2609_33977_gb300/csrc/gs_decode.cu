// Decode-regime group-sparse linear (few tokens, HBM-bound):
//   y[t, r] = sum over kept groups (r, c) of sum_k x[t, 256c+k] W[r, 256c+k]   (Eq. 1)
//
// Work decomposition.  A warp owns a 16-row output window and walks the
// chunks of its chunk range.  For chunk c it loads the kept rows of its window
// (each a 512-byte packed group, 16 bytes per lane, coalesced in 64-byte runs)
// straight into mma.sync A fragments, placing every kept row at its window
// position and leaving pruned rows zero.  The x chunk forms the B fragment.
// Because the MMA row is the output row, the fp32 accumulator stays in
// registers across all chunks: no scatter, no atomics, a fixed summation
// order.  A CTA is eight such warps (128 rows); S CTAs of a thread-block
// cluster split the chunks of the same 128 rows and reduce their partial sums
// through distributed shared memory in rank order (deterministic).
//
// K permutation.  Within a 32-wide k block b, lane (g, q) holds the eight
// consecutive weights k = 32b + 8q + 0..7 of rows g and g+8 and the same eight
// x values of token g.  Elements 0..3 feed MMA 2b, elements 4..7 feed MMA
// 2b+1; the logical-to-physical k map depends only on (b, q), so A and B agree
// and every physical k is used exactly once.
#include "gs_common.cuh"

#include <cooperative_groups.h>
#include <algorithm>
#include <vector>

namespace cg = cooperative_groups;

namespace gs {
namespace {

constexpr int kDecWarps = 8;                 // 16-row windows per CTA
constexpr int kDecRows = kDecWarps * kWin16;  // 128 rows per CTA
constexpr int kMaxBatch = 32;
constexpr int kMaxNT = 8;                    // up to 64 tokens per launch

struct DecodeParams {
  DecodeLayer layers[kMaxBatch];
  int32_t n_layers;
  int32_t T;
  int32_t S;
};

__device__ __forceinline__ uint4 ld_stream16(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
  return v;
}

__device__ __forceinline__ uint4 ld_cached16(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
  return v;
}

__device__ __forceinline__ void mma16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint16_t f32_to_bf16_rn(float f) {
  return __bfloat16_as_ushort(__float2bfloat16_rn(f));
}

template <int NT>
__global__ void __launch_bounds__(kDecWarps * 32) k_decode(const __grid_constant__ DecodeParams P) {
  const int S = P.S;
  const int cl = blockIdx.x / S;     // cluster index = (layer, 128-row block)
  const int s = blockIdx.x % S;      // rank inside the cluster = chunk split
  int l = 0;
  while (l + 1 < P.n_layers && P.layers[l + 1].cta_begin <= cl) ++l;
  const DecodeLayer& L = P.layers[l];
  const int blk = cl - L.cta_begin;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, q = lane & 3;
  const int w16 = blk * kDecWarps + warp;
  const int T = P.T;

  float acc[NT][4];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt)
#pragma unroll
    for (int i = 0; i < 4; ++i) acc[nt][i] = 0.f;

  if (w16 < L.nw16) {
    const int c0 = (int)((int64_t)s * L.G / S), c1 = (int)((int64_t)(s + 1) * L.G / S);
    const uint32_t lo_g = (1u << g) - 1u, lo_g8 = (1u << (g + 8)) - 1u;
    const int64_t xrow = L.in / 8;   // uint4 per x row
    const uint4* xbase = reinterpret_cast<const uint4*>(L.x);
    for (int c = c0; c < c1; ++c) {
      const uint32_t km = L.kmask16[(int64_t)c * L.nw16 + w16];
      if (km == 0u) continue;
      const int32_t base = L.win_off16[(int64_t)c * (L.nw16 + 1) + w16];
      const bool kg = (km >> g) & 1u, kg8 = (km >> (g + 8)) & 1u;
      const uint4* tg = reinterpret_cast<const uint4*>(L.tiles) + (int64_t)(base + __popc(km & lo_g)) * 32 + q;
      const uint4* tg8 = reinterpret_cast<const uint4*>(L.tiles) + (int64_t)(base + __popc(km & lo_g8)) * 32 + q;
      uint4 a[8], a8[8];
#pragma unroll
      for (int b = 0; b < 8; ++b) {
        a[b] = kg ? ld_stream16(tg + 4 * b) : make_uint4(0u, 0u, 0u, 0u);
        a8[b] = kg8 ? ld_stream16(tg8 + 4 * b) : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        const int tok = nt * 8 + g;
        const uint4* xr = xbase + (int64_t)tok * xrow + (int64_t)c * 32 + q;
#pragma unroll
        for (int b = 0; b < 8; ++b) {
          const uint4 xv = tok < T ? ld_cached16(xr + 4 * b) : make_uint4(0u, 0u, 0u, 0u);
          mma16816(acc[nt], a[b].x, a8[b].x, a[b].y, a8[b].y, xv.x, xv.y);
          mma16816(acc[nt], a[b].z, a8[b].z, a[b].w, a8[b].w, xv.z, xv.w);
        }
      }
    }
  }

  const int row0 = blk * kDecRows;
  if (S == 1) {
    if (w16 < L.nw16) {
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          const int tok = nt * 8 + 2 * q + j;
          const int r = row0 + warp * kWin16 + g;
          if (tok < T) {
            if (r < L.out) L.y[(int64_t)tok * L.out + r] = f32_to_bf16_rn(acc[nt][j]);
            if (r + 8 < L.out) L.y[(int64_t)tok * L.out + r + 8] = f32_to_bf16_rn(acc[nt][2 + j]);
          }
        }
    }
    return;
  }

  // chunk-split reduction across the cluster through distributed shared memory
  __shared__ float red[kDecWarps][NT * 8][kWin16 + 1];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt)
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      red[warp][nt * 8 + 2 * q + j][g] = acc[nt][j];
      red[warp][nt * 8 + 2 * q + j][g + 8] = acc[nt][2 + j];
    }
  cg::cluster_group cluster = cg::this_cluster();
  cluster.sync();
  const int Tl = T < NT * 8 ? T : NT * 8;
  for (int wi = s; wi < kDecWarps; wi += S) {
    if (blk * kDecWarps + wi >= L.nw16) break;
    for (int e = threadIdx.x; e < Tl * kWin16; e += blockDim.x) {
      const int tok = e / kWin16, i = e % kWin16;
      float sum = 0.f;
      for (int rk = 0; rk < S; ++rk) {
        const float* rred = cluster.map_shared_rank(&red[0][0][0], rk);
        sum += rred[(wi * (NT * 8) + tok) * (kWin16 + 1) + i];
      }
      const int r = row0 + wi * kWin16 + i;
      if (r < L.out) L.y[(int64_t)tok * L.out + r] = f32_to_bf16_rn(sum);
    }
  }
  cluster.sync();
}

int g_num_sms = 0;

int num_sms() {
  if (g_num_sms == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&g_num_sms, cudaDevAttrMultiProcessorCount, dev);
    if (g_num_sms <= 0) g_num_sms = 148;
  }
  return g_num_sms;
}

template <int NT>
cudaError_t launch_nt(const DecodeParams& P, int grid, cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid, 1, 1);
  cfg.blockDim = dim3(kDecWarps * 32, 1, 1);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  int na = 0;
  if (P.S > 1) {
    attr[na].id = cudaLaunchAttributeClusterDimension;
    attr[na].val.clusterDim.x = P.S;
    attr[na].val.clusterDim.y = 1;
    attr[na].val.clusterDim.z = 1;
    ++na;
  }
  cfg.attrs = attr;
  cfg.numAttrs = na;
  return cudaLaunchKernelEx(&cfg, k_decode<NT>, P);
}

}  // namespace

int decode_max_tokens() { return kMaxNT * 8; }

gs_status launch_decode(const DecodeLayer* layers, int n, int T, cudaStream_t s) {
  if (n <= 0 || T <= 0) return GS_OK;
  if (n > kMaxBatch || T > kMaxNT * 8) return GS_ERR_UNSUPPORTED;
  // Longest-work layers first: CTAs are dispatched roughly in index order, so
  // the layers with the most kept groups per CTA start first.
  std::vector<int> order(n);
  for (int i = 0; i < n; ++i) order[i] = i;
  std::vector<double> work(n);
  int64_t blocks = 0;
  int minG = 1 << 30;
  for (int i = 0; i < n; ++i) {
    const int nblk = (layers[i].out + kDecRows - 1) / kDecRows;
    blocks += nblk;
    minG = std::min(minG, layers[i].G);
    work[i] = (double)layers[i].G;   // chunks per 128-row block (density-independent proxy)
  }
  std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return work[a] > work[b]; });
  // chunk splits: enough CTAs for about two per SM, at most 8 (portable cluster), at most G
  const int want = 2 * num_sms();
  int S = (int)((want + blocks - 1) / blocks);
  S = std::max(1, std::min(S, std::min(8, minG)));

  DecodeParams P = {};
  P.n_layers = n;
  P.T = T;
  P.S = S;
  int32_t cl = 0;
  for (int k = 0; k < n; ++k) {
    P.layers[k] = layers[order[k]];
    P.layers[k].nblk = (layers[order[k]].out + kDecRows - 1) / kDecRows;
    P.layers[k].cta_begin = cl;
    cl += P.layers[k].nblk;
  }
  const int grid = cl * S;
  cudaError_t e;
  if (T <= 8) e = launch_nt<1>(P, grid, s);
  else if (T <= 16) e = launch_nt<2>(P, grid, s);
  else if (T <= 32) e = launch_nt<4>(P, grid, s);
  else e = launch_nt<8>(P, grid, s);
  note_launch();
  return e == cudaSuccess ? GS_OK : GS_ERR_CUDA;
}

}  // namespace gs
