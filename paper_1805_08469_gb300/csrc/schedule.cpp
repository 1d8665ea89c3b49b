// Seeded commit schedules and the segment planner (include/gem_sim.h).
#include <cmath>
#include <cstdint>
#include <vector>

#include "../../include/gem_sim.h"

namespace {

// A SplitMix64 stream read at arbitrary positions.
class CounterStream {
 public:
  static constexpr uint64_t kGamma = 0x9E3779B97F4A7C15ull;
  CounterStream(uint64_t seed, uint64_t id) : start_(Finalize(seed * kGamma + id)) {}
  uint64_t At(uint64_t c) const { return Finalize(start_ + kGamma * (c + 1)); }

 private:
  static uint64_t Finalize(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
  }
  uint64_t start_;
};

constexpr uint64_t kUniformTickId = 10;
constexpr uint64_t kQueueId = 11;

void fill_staleness(const int32_t* order, int T, int n, int32_t* tau) {
  std::vector<int64_t> previous(size_t(n), -1);
  for (int t = 0; t < T; ++t) {
    int64_t& p = previous[size_t(order[t])];
    tau[t] = int32_t(int64_t(t) - p - 1);
    p = t;
  }
}

}  // namespace

extern "C" {

int gem_schedule_uniform(uint64_t seed, int n, int T, int32_t* order, int32_t* tau) {
  if (n < 1 || T < 0 || (T > 0 && !order)) return -1;
  const CounterStream rng(seed, kUniformTickId);
  for (int t = 0; t < T; ++t)
    order[t] = int32_t(((rng.At(uint64_t(t)) >> 32) * uint64_t(n)) >> 32);
  if (tau) fill_staleness(order, T, n, tau);
  return 0;
}

int gem_schedule_queue(uint64_t seed, int n, int T, double rate, int32_t* order,
                       int32_t* tau) {
  if (n < 1 || T < 0 || (T > 0 && !order) || !(rate > 0.0)) return -1;
  const CounterStream rng(seed, kQueueId);
  std::vector<double> done(static_cast<size_t>(n));
  std::vector<uint64_t> started(static_cast<size_t>(n), 0);
  auto service_time = [&](int w, uint64_t j) {
    const double u = double(rng.At((uint64_t(w) << 32) | j) >> 11) * 0x1.0p-53;
    return -std::log(1.0 - u) / rate;
  };
  for (int w = 0; w < n; ++w) done[size_t(w)] = service_time(w, 0);
  for (int t = 0; t < T; ++t) {
    int next = 0;
    for (int w = 1; w < n; ++w)
      if (done[size_t(w)] < done[size_t(next)]) next = w;
    order[t] = next;
    started[size_t(next)] += 1;
    done[size_t(next)] += service_time(next, started[size_t(next)]);
  }
  if (tau) fill_staleness(order, T, n, tau);
  return 0;
}

int gem_plan_segments(const int32_t* order, int T, int n, int32_t* seg_start) {
  if (T < 0 || n < 1 || !seg_start || (T > 0 && !order)) return -1;
  std::vector<int32_t> in_segment(size_t(n), -1);  // segment index of the worker's last commit
  int S = 0;
  for (int t = 0; t < T; ++t) {
    const int w = order[t];
    if (w < 0 || w >= n) return -1;
    if (t == 0 || in_segment[size_t(w)] == S - 1) seg_start[S++] = t;
    in_segment[size_t(w)] = S - 1;
  }
  seg_start[S] = T;
  return S;
}

}  // extern "C"
