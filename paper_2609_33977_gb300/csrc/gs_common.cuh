// Shared definitions of the CUDA path (library side only).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <cstdint>
#include <vector>
#include <cstddef>

#include "groupsparse.h"
#include "gs_plan.cuh"

namespace gs {

constexpr int kGroupIn = 256;     // g_in of the 1x256 groups (Sec. 2.1)
constexpr int kWin16 = 16;        // row-window height of the per-(chunk, window) metadata
constexpr int kTileBytes = kGroupIn * 2;   // one packed group: 256 bf16 = 512 B

// Device-error codes written into the library's device flag.
constexpr int kDevErrTimeout = 1;

// Decode split-reduction scratch of one handle for one stream: gs_linear calls
// on different streams use different slots, so one handle can serve several
// streams at once.
constexpr int kDecSlots = 8;
struct DecSlot {
  void* stream;       // cudaStream_t the slot belongs to
  float* ws;          // [nblk64][dec_nsplit_max][4][16 tokens][16 rows] partial sums
  int32_t* cnt;       // [nblk64][4] arrival counters, then {unit ticket, finished CTAs} (self-resetting)
  uint64_t epoch;     // timeout epoch at which the counters were last known clean
};

}  // namespace gs

// Library-owned packed weight.  All arrays live on `device`.
struct gs_packed {
  int device;
  int64_t out, in;
  int32_t G;          // in / 256
  int32_t nw16;       // ceil(out / 16)
  int64_t kept;       // offsets[G]
  int64_t* offsets;   // [G+1]
  int32_t* row_idx;   // [kept]
  uint16_t* tiles;    // [kept][256]
  int32_t* win_off16; // [G][nw16+1]
  uint16_t* kmask16;  // [G][nw16]
  size_t device_bytes;
  // decode kernel: window-major metadata and split-reduction scratch
  int32_t nblk64;     // ceil(out / 64)
  int32_t dec_cpu;    // chunks per decode work unit (about 256 KB of kept weights)
  int32_t dec_cpu_fine;   // chunks per unit when the layer is scheduled last (a quarter of that)
  int32_t dec_nsplit_max; // ceil(G / dec_cpu_fine): splits the workspace is sized for
  int4* dmeta;        // [nblk64][G]: {first packed row of the block's slice, kept masks of its 4 windows, 0}
  gs::DecSlot dec_slot[gs::kDecSlots];   // per-stream split scratch; slot 0 is made for gs_pack's stream
  int32_t dec_nslots;
  // tcgen05 prefill: slab TMA descriptors over the tiles, box heights 16, 32, ..., 160 rows
  alignas(64) unsigned char wmaps[10][128];
  alignas(64) unsigned char wmaps_full[10][128];   // same, box heights 16, 32, ..., 160 (whole slices)
  bool wmaps_valid;
  // group shape (Sec. 2.1: g_out x g_in groups).  gs_pack handles are 1 x 256;
  // square g x g handles (gs_pack_groups) use the fields below instead of the
  // 1 x 256 window metadata: G = in / g column blocks, row_idx holds each
  // kept tile's block row, tiles holds g x g row-major blocks.
  int32_t g_out, g_in;
  int32_t Gout;       // out / g_out
  int32_t nwin;       // square groups: ceil(out / 128) windows of 128 output rows
  int32_t* gwoff;     // [G][nwin + 1]: first packed tile of column block v in window w (+ end)
  uint8_t* gwmask;    // [G][nwin]: bit i = block row (128/g) w + i kept in column block v
  int32_t* gtidx;     // [Gout][G]: packed tile of group (u, v), -1 if pruned (decode-regime lookups)
  alignas(64) unsigned char gmaps[8][128];   // W slice descriptors, box heights g, 2g, ..., 128 rows
  alignas(64) unsigned char hmaps[8][128];   // CTA-pair halves: rows [r g/2, r g/2 + g/2) of 1..8 consecutive tiles
};

namespace gs {

// 2-D bf16 TMA descriptor (map: 128-byte, 64-byte aligned buffer); false on failure
bool encode_tmap_2d_bf16(void* map, const void* base, uint64_t inner, uint64_t outer, uint32_t box_inner,
                         uint32_t box_outer, bool swizzle128);

// 2-D bf16 descriptor with a 32-, 64- or 128-byte swizzle (box_inner * 2 <= swizzle_bytes)
bool encode_tmap_2d_bf16_swz(void* map, const void* base, uint64_t inner, uint64_t outer, uint32_t box_inner,
                             uint32_t box_outer, int swizzle_bytes);

// rank-D bf16 descriptor (rank <= 5): dims innermost first, strides_bytes for
// dims 1..rank-1, the given box and swizzle (box[0] * 2 <= swizzle_bytes)
bool encode_tmap_nd_bf16(void* map, const void* base, int rank, const uint64_t* dims, const uint64_t* strides_bytes,
                         const uint32_t* box, int swizzle_bytes);

// 3-D "slab" bf16 descriptor over a row-major [rows][row_elems] matrix: a box
// of box_rows rows x box_slabs 64-element slabs lands in shared memory as
// box_slabs consecutive [box_rows][64] blocks, each with the 128-byte swizzle
// that tcgen05's K-major operand descriptors expect.  row_elems % 64 == 0.
bool encode_tmap_slabs_bf16(void* map, const void* base, uint64_t row_elems, uint64_t rows, uint32_t box_rows,
                            uint32_t box_slabs);

// library-owned per-device flags (allocated on first use): [0] the error flag
// gs_device_status reads, [1] a word nothing ever sets (test-injected waits)
int* device_error_flag();
void note_launch(int64_t n = 1);
// Incremented each time gs_device_status reports a timeout: scratch whose
// arrival counters were last cleaned at an older epoch is re-zeroed first.
uint64_t timeout_epoch();
// Every device allocation of the library goes through here (so that a test can
// make the n-th one fail); OOM on cudaErrorMemoryAllocation, else CUDA.
gs_status lib_malloc(void** ptr, size_t bytes);
// Test hook: limit of a wait on the never-set word to inject into the next
// launch of a kernel family (GS_ALGO_DECODE / GS_ALGO_PREFILL /
// GS_ALGO_PREFILL_DENSE); 0 = none.
// Reading it disarms it.
uint64_t take_injected_wait(int family);

// The k-th tile of owner b, or -1 when it has no more (TileList: gs_plan.cuh).
__device__ __forceinline__ int owner_tile(const TileList& L, int n_tiles, int b, int n_owners, int k) {
  if (L.on) {
    const int i = (int)L.off[b] + k;
    return i < (int)L.off[b + 1] ? (int)L.order[i] : -1;
  }
  const int t = b + k * n_owners;
  return t < n_tiles ? t : -1;
}

// pack.cu
gs_status launch_pack_count_scan(const uint8_t* mask, gs_packed* p, cudaStream_t s, int32_t* cnt_tmp);
// exclusive scan of cnt[G][nw] (chunk-major) into win_off[G][nw + 1] and offsets[G + 1]
gs_status launch_scan_counts(const int32_t* cnt, int32_t G, int32_t nw, int32_t* win_off, int64_t* offsets,
                             cudaStream_t s);
gs_status launch_pack_compact(const void* W, gs_packed* p, cudaStream_t s);
gs_status launch_unpack(const gs_packed* p, void* W_hat, cudaStream_t s);

// select.cu
gs_status launch_select(const float* logits, int64_t n, uint8_t* mask, int64_t* kept, cudaStream_t s);

// decode.cu
gs_status decode_prepare(gs_packed* p, cudaStream_t s);   // allocates + builds the decode metadata
void decode_release(gs_packed* p);
// split scratch of handle p for stream s (made on first use; re-zeroed after a timeout)
gs_status decode_slot(const gs_packed* p, cudaStream_t s, const DecSlot** slot);
gs_status launch_decode(const gs_packed* const* ps, const void* const* xs, void* const* ys, int n, int T,
                        cudaStream_t s);
int decode_max_tokens();

// prefill.cu
gs_status prefill_prepare_weight_maps(gs_packed* p);
gs_status launch_prefill(const void* x, const gs_packed* p, int64_t T, void* y, cudaStream_t s);
gs_status launch_prefill_batched(const void* const* xs, const gs_packed* const* ps, int n, int64_t T,
                                 void* const* ys, cudaStream_t s);
int prefill_max_chunks();
// prefill_dense.cu: zero-filled windows (1 x 128 / 1 x 256 layers with kept groups)
// (layers ps[idx[k]], k < n, when idx is given; else ps[0..n))
gs_status launch_prefill_dense(const void* const* xs, const gs_packed* const* ps, int n, int64_t T, void* const* ys,
                               cudaStream_t s, const int* idx = nullptr);
// whether the zero-filled kernel is the faster one for this layer and token count
bool prefill_prefers_dense(const gs_packed* p, int64_t T);

// groups.cu: square g x g groups
bool sq_shape_supported(int g_out, int g_in);
gs_status sq_pack(const void* W, const uint8_t* mask, gs_packed* p, cudaStream_t s);   // p: shape fields set
gs_status sq_unpack(const gs_packed* p, void* W_hat, cudaStream_t s);
gs_status sq_linear_batched(const void* const* xs, const gs_packed* const* ps, int n, int64_t T, void* const* ys,
                            cudaStream_t s);
void sq_release(gs_packed* p);
// sq_decode.cu: square groups, T <= sq_decode_max_tokens(): layers ps[idx[0..n)] (same g, kept > 0, n <= 8)
int sq_decode_max_tokens();
gs_status sq_decode_batched(const void* const* xs, const gs_packed* const* ps, const int* idx, int n, int T,
                            void* const* ys, cudaStream_t s);
inline bool is_square(const gs_packed* p) { return p->g_out > 1; }

// train.cu: Gumbel-Sigmoid sample and straight-through backward (Sec. 2.2)
gs_status launch_gumbel(const float* logits, const float* noise, int64_t n, float tau, uint8_t* mask, float* dsdl,
                        int64_t* kept, cudaStream_t s);
size_t backward_workspace_bytes(const gs_packed* p, bool want_dx);
gs_status launch_backward(const void* x, const void* W, const gs_packed* p, const void* dy, int64_t T,
                          const float* dsdl, float* dlogits, void* dx, void* ws, cudaStream_t s);

}  // namespace gs
