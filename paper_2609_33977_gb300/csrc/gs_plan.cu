// Balanced tile lists for the persistent tensor-core kernels (host code only).
#include "gs_plan.cuh"

#include <algorithm>
#include <utility>

namespace gs {

void plan_tiles(const std::vector<int32_t>& cost, int n_owners, TileList& L) {
  const int n = (int)cost.size();
  L.on = 0;
  if (n > kTileListMax || n_owners > kTileOwnersMax || n_owners <= 0) return;
  std::vector<int> idx(n);
  for (int i = 0; i < n; ++i) idx[i] = i;
  std::stable_sort(idx.begin(), idx.end(), [&](int a, int b) { return cost[a] > cost[b]; });
  // min-heap of (load, owner)
  std::vector<std::pair<int64_t, int>> heap;
  heap.reserve(n_owners);
  for (int b = 0; b < n_owners; ++b) heap.emplace_back(0, b);
  auto later = [](const std::pair<int64_t, int>& x, const std::pair<int64_t, int>& y) { return x > y; };
  std::vector<int> owner(n);
  std::vector<int> count(n_owners + 1, 0);
  for (int t : idx) {
    std::pop_heap(heap.begin(), heap.end(), later);
    auto& h = heap.back();
    owner[t] = h.second;
    h.first += cost[t];
    std::push_heap(heap.begin(), heap.end(), later);
    ++count[owner[t] + 1];
  }
  for (int b = 0; b < n_owners; ++b) count[b + 1] += count[b];
  for (int b = 0; b <= n_owners; ++b) L.off[b] = (uint16_t)count[b];
  // each owner's tiles longest first (the order they were handed out)
  for (int t : idx) L.order[count[owner[t]]++] = (uint16_t)t;
  L.on = 1;
}

}  // namespace gs
