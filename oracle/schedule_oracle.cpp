// ORACLE -- test infrastructure, not part of the product.
//
// Commit schedules of the asynchronous system (Introduction, Eq. staleness): which
// worker commits at each tick of the global clock, and the staleness tau_t of that
// commit, i.e. the number of commits between the worker's pull and its commit.  Under a
// homogeneous queueing model the expected staleness is n - 1.
//
// Random numbers come from SplitMix64 (Steele, Lea & Flood, OOPSLA 2014), written here
// from its published definition: the c-th output (0-based) of the stream whose state
// starts at k is mix(k + GAMMA (c + 1)), and the stream for (seed, stream id) starts at
// mix(seed * GAMMA + stream id).
#include <cmath>
#include <cstdint>
#include <vector>

namespace {

const uint64_t kGamma = 0x9E3779B97F4A7C15ull;
const uint64_t kStreamUniformTick = 10;
const uint64_t kStreamQueue = 11;

uint64_t mix(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

uint64_t stream_key(uint64_t seed, uint64_t stream) { return mix(seed * kGamma + stream); }

uint64_t draw(uint64_t key, uint64_t counter) { return mix(key + kGamma * (counter + 1)); }

// Staleness of every commit: the worker pulled theta right after its previous commit
// (theta_0 before its first), so tau_t = t - (tick of its previous commit) - 1.
void staleness(int n, int T, const int32_t* order, int32_t* tau) {
  std::vector<int64_t> last(n, -1);
  for (int t = 0; t < T; ++t) {
    const int w = order[t];
    tau[t] = int32_t(t - last[w] - 1);
    last[w] = t;
  }
}

}  // namespace

extern "C" {

// counter-th output of the stream whose state starts at `state` (the classic sequential
// generator seeded with `state`, read at position counter).
uint64_t oracle_splitmix64_raw(uint64_t state, uint64_t counter) { return draw(state, counter); }

uint64_t oracle_splitmix64_draw(uint64_t seed, uint64_t stream, uint64_t counter) {
  return draw(stream_key(seed, stream), counter);
}

// Uniform tick: at every tick a worker drawn uniformly from {0..n-1} commits
// (w = floor(n * u32 / 2^32) with u32 the top 32 bits of the tick's draw).
int oracle_schedule_uniform(uint64_t seed, int n, int T, int32_t* order, int32_t* tau) {
  if (n < 1 || T < 0 || !order) return -1;
  const uint64_t key = stream_key(seed, kStreamUniformTick);
  for (int t = 0; t < T; ++t) {
    const uint64_t u32 = draw(key, uint64_t(t)) >> 32;
    order[t] = int32_t((u32 * uint64_t(n)) >> 32);
  }
  if (tau) staleness(n, T, order, tau);
  return 0;
}

// Queue: worker w finishes its j-th gradient (j = 0, 1, ...) after an exponential
// service time -ln(1 - u) / rate, u = draw((w << 32) | j) * 2^-53; the worker with the
// earliest finishing time commits next (ties go to the lower id), then starts its next
// gradient.
int oracle_schedule_queue(uint64_t seed, int n, int T, double rate, int32_t* order,
                          int32_t* tau) {
  if (n < 1 || T < 0 || !order || !(rate > 0)) return -1;
  const uint64_t key = stream_key(seed, kStreamQueue);
  auto service = [&](int w, uint64_t j) {
    const double u = double(draw(key, (uint64_t(w) << 32) | j) >> 11) * 0x1.0p-53;
    return -std::log(1.0 - u) / rate;
  };
  std::vector<double> finish(n);
  std::vector<uint64_t> jobs(n, 0);
  for (int w = 0; w < n; ++w) finish[w] = service(w, 0);
  for (int t = 0; t < T; ++t) {
    int best = 0;
    for (int w = 1; w < n; ++w)
      if (finish[w] < finish[best]) best = w;
    order[t] = best;
    jobs[best] += 1;
    finish[best] = finish[best] + service(best, jobs[best]);
  }
  if (tau) staleness(n, T, order, tau);
  return 0;
}

}  // extern "C"
