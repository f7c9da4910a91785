// Host-side communication-graph builder (Section 3.1, Fig. 2; Appendix A).
//
// Every graph is k-regular in and out degree with self-loops, so the
// equal-weight mixing matrix P = diag(d_in)^-1 A is doubly stochastic, the
// requirement of Appendix A ("Network requirement").  Kinds:
//   RING            i <- i-1                      (the chain, closed)
//   ROOT            i <- i-1, i-isqrt(N)          (root expander: i sends to
//                                                  i+1 and i+sqrt(N))
//   COMPLETE        i <- every j                  (all-reduce)
//   IDENTITY        i <- i only                   (k = 0)
//   RANDOM_REGULAR  a Hamiltonian cycle plus k-1 permutation layers drawn by
//                   rejection; SplitMix64 (Steele, Lea & Flood 2014) seeded
//                   by graph_seed ^ (gamma * (round + 1)).
// The paper fixes no construction for random expanders; this one is cheap
// enough to redo every round on the host (Section 3.1 asks for graphs that
// are cheap to build).
#include <algorithm>
#include <cstdint>
#include <vector>

#include "asap_internal.h"

namespace asap {

namespace {

constexpr uint64_t kGamma = 0x9E3779B97F4A7C15ull;
constexpr int kMaxLayerDraws = 100000;

struct SplitMix64 {
  uint64_t s;
  uint64_t next() {
    s += kGamma;
    uint64_t z = s;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
  }
  // Unbiased value in [0, m): reject draws in the last, partial block of
  // size 2^64 mod m.
  uint64_t below(uint64_t m) {
    const uint64_t rem = (0 - m) % m;  // (2^64 - m) mod m == 2^64 mod m
    for (;;) {
      const uint64_t v = next();
      if (rem == 0 || v < 0 - rem) return v % m;
    }
  }
};

uint64_t isqrt64(uint64_t n) {
  uint64_t r = 0;
  while ((r + 1) * (r + 1) <= n) ++r;
  return r;
}

}  // namespace

// Fills nbr (N*(k+1)) with each worker's sorted in-neighbour set, self
// included.  Returns ASAP_OK or ASAP_ERR_GRAPH / ASAP_ERR_ARG with *why set.
asap_status build_graph_host(asap_graph_kind kind, int N, int k, uint64_t seed, int64_t round,
                             int32_t* nbr, const char** why) {
  const int kp1 = k + 1;
  if (N < 1 || k < 0 || k > N - 1) {
    *why = "graph needs N >= 1 and 0 <= k <= N-1";
    return ASAP_ERR_ARG;
  }
  std::vector<std::vector<int32_t>> in(N);
  switch (kind) {
    case ASAP_GRAPH_IDENTITY:
      if (k != 0) { *why = "IDENTITY needs k = 0"; return ASAP_ERR_GRAPH; }
      break;
    case ASAP_GRAPH_RING:
      if (k != 1 || N < 2) { *why = "RING needs k = 1 and N >= 2"; return ASAP_ERR_GRAPH; }
      for (int i = 0; i < N; ++i) in[i].push_back((i + N - 1) % N);
      break;
    case ASAP_GRAPH_ROOT: {
      if (k != 2 || N < 4) { *why = "ROOT needs k = 2 and N >= 4"; return ASAP_ERR_GRAPH; }
      const int s = static_cast<int>(isqrt64(static_cast<uint64_t>(N)));
      for (int i = 0; i < N; ++i) {
        in[i].push_back((i + N - 1) % N);
        in[i].push_back((i + N - s) % N);
      }
      break;
    }
    case ASAP_GRAPH_COMPLETE:
      if (k != N - 1) { *why = "COMPLETE needs k = N-1"; return ASAP_ERR_GRAPH; }
      for (int i = 0; i < N; ++i)
        for (int j = 0; j < N; ++j)
          if (j != i) in[i].push_back(j);
      break;
    case ASAP_GRAPH_RANDOM_REGULAR: {
      if (k < 1) { *why = "RANDOM_REGULAR needs k >= 1"; return ASAP_ERR_GRAPH; }
      SplitMix64 rng{seed ^ (kGamma * static_cast<uint64_t>(round + 1))};
      std::vector<int32_t> perm(N);
      for (int t = 0; t < N; ++t) perm[t] = t;
      for (int t = N - 1; t >= 1; --t) {
        const int j = static_cast<int>(rng.below(static_cast<uint64_t>(t) + 1));
        std::swap(perm[t], perm[j]);
      }
      // Bitset of current in-neighbours for O(1) admissibility checks.
      std::vector<uint8_t> has(static_cast<size_t>(N) * N, 0);
      for (int t = 0; t < N; ++t) {
        const int recv = perm[(t + 1) % N], send = perm[t];
        in[recv].push_back(send);
        has[static_cast<size_t>(recv) * N + send] = 1;
      }
      std::vector<int32_t> sigma(N);
      for (int layer = 1; layer < k; ++layer) {
        bool placed = false;
        for (int draw = 0; draw < kMaxLayerDraws && !placed; ++draw) {
          for (int t = 0; t < N; ++t) sigma[t] = t;
          bool ok = true;
          // Slot t is final once step t of the shuffle is done: abandon the
          // draw at the first slot that holds t itself or a current in-neighbour.
          for (int t = N - 1; t >= 1 && ok; --t) {
            const int j = static_cast<int>(rng.below(static_cast<uint64_t>(t) + 1));
            std::swap(sigma[t], sigma[j]);
            const int s = sigma[t];
            ok = (s != t) && !has[static_cast<size_t>(t) * N + s];
          }
          if (ok) ok = (sigma[0] != 0) && !has[sigma[0]];
          if (ok) {
            for (int i = 0; i < N; ++i) {
              in[i].push_back(sigma[i]);
              has[static_cast<size_t>(i) * N + sigma[i]] = 1;
            }
            placed = true;
          }
        }
        if (!placed) { *why = "no admissible permutation layer within the draw limit"; return ASAP_ERR_GRAPH; }
      }
      break;
    }
    default:
      *why = "graph kind not buildable on the host";
      return ASAP_ERR_ARG;
  }
  for (int i = 0; i < N; ++i) {
    std::vector<int32_t>& r = in[i];
    r.push_back(i);
    std::sort(r.begin(), r.end());
    if (static_cast<int>(r.size()) != kp1 || std::adjacent_find(r.begin(), r.end()) != r.end()) {
      *why = "internal: row does not have k+1 distinct ids";
      return ASAP_ERR_GRAPH;
    }
    std::copy(r.begin(), r.end(), nbr + static_cast<size_t>(i) * kp1);
  }
  return ASAP_OK;
}

}  // namespace asap
