// Tile assignment of the persistent tensor-core kernels (host side; plain C++,
// also compiled on its own by the CPU tests).
#pragma once
#include <cstdint>
#include <vector>

namespace gs {

// A launch's tiles differ in cost (a layer's tile walks all of its chunks, and
// wide-input layers have 2-3x more), so a fixed stride over the tile list can
// leave a few owners (CTAs or CTA pairs) with twice the mean.  Owner b takes
// order[off[b]] .. order[off[b + 1] - 1]; on == 0: tiles b, b + owners, ...
constexpr int kTileListMax = 2048;
constexpr int kTileOwnersMax = 160;
struct TileList {
  uint16_t order[kTileListMax];
  uint16_t off[kTileOwnersMax + 1];
  int32_t on;
};

// Longest tile first to the least-loaded owner (ties: the lowest owner), each
// owner's tiles in the order they were handed out; cost[t] of each tile in
// list order.  Leaves on == 0 when the launch has more tiles or owners than
// the list holds (or no owner).
void plan_tiles(const std::vector<int32_t>& cost, int n_owners, TileList& L);

}  // namespace gs
