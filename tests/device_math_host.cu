// Host build of the library's proposal-stream and decision helpers (csrc/mca_device.cuh,
// csrc/mca_deep.cuh), compiled by tests/test_device_math_host.py so that their arithmetic can be
// compared with the oracle on a machine without a GPU. Reads commands from stdin, one per line:
//   words SEED TAU                        -> the four Philox words of trial TAU
//   theta SEED TAU MSC                    -> the Metropolis threshold (Eq. 7), %.9g
//   accept D STRICT METRO SEED TAU MSC    -> 0 / 1
//   stretch SEED S NL                     -> the layer of stretch S
//   idx2 P P1 SEED TAU R0 M               -> two-layer trial index
//   idxd SEED TAU R0 M L off0 .. offL     -> deep trial index (L layers, L + 1 offsets)
//   chan SEED TAU L n0 .. nL fin0 .. finL-1 -> channel nodes c_0 .. c_L, then the L He values
//   width ACC TRIALS R K                  -> the host-driven batch width of the cost model
#include <cstdio>
#include <cstring>
#include <iostream>
#include <sstream>
#include <string>
#include <vector>

#include "mca_deep.cuh"

int main() {
  std::string line;
  while (std::getline(std::cin, line)) {
    std::istringstream in(line);
    std::string cmd;
    in >> cmd;
    if (cmd == "words") {
      unsigned long long seed, tau;
      in >> seed >> tau;
      const uint4 w = mca::trial_words(seed, tau);
      std::printf("%u %u %u %u\n", w.x, w.y, w.z, w.w);
    } else if (cmd == "theta") {
      unsigned long long seed, tau;
      double msc;
      in >> seed >> tau >> msc;
      std::printf("%.9g\n", (double)mca::metropolis_theta(seed, tau, msc));
    } else if (cmd == "accept") {
      float d;
      int strict, metro;
      unsigned long long seed, tau;
      double msc;
      in >> d >> strict >> metro >> seed >> tau >> msc;
      std::printf("%d\n", mca::accept_change(d, strict, metro, seed, tau, msc) ? 1 : 0);
    } else if (cmd == "stretch") {
      unsigned long long seed, s;
      int nl;
      in >> seed >> s >> nl;
      std::printf("%d\n", mca::stretch_layer(seed, s, nl));
    } else if (cmd == "idx2") {
      unsigned long long P, P1, seed, tau;
      unsigned int r0;
      int m;
      in >> P >> P1 >> seed >> tau >> r0 >> m;
      std::printf("%u\n", mca::mlp2_trial_index(P, P1, seed, tau, r0, m));
    } else if (cmd == "idxd") {
      mca::DeepArgs a;
      std::memset(&a, 0, sizeof(a));
      unsigned long long tau;
      unsigned int r0;
      in >> a.seed >> tau >> r0 >> a.stretch >> a.L;
      for (int l = 0; l <= a.L; ++l) in >> a.off[l];
      std::printf("%u\n", mca::deep_trial_index(a, tau, r0));
    } else if (cmd == "chan") {
      unsigned long long seed, tau;
      int L;
      in >> seed >> tau >> L;
      std::vector<unsigned long long> nodes(L + 1);
      std::vector<int> fin(L);
      for (int m = 0; m <= L; ++m) in >> nodes[m];
      for (int m = 0; m < L; ++m) in >> fin[m];
      for (int m = 0; m <= L; ++m)
        std::printf("%d ", mca::channel_node(mca::channel_word(seed, tau, m), nodes[m]));
      for (int m = 0; m < L; ++m)
        std::printf("%.9g ", (double)mca::channel_he_value(mca::channel_word(seed, tau, L + 1 + m),
                                                           fin[m]));
      std::printf("\n");
    } else if (cmd == "width") {
      float acc, trials, r;
      int K;
      in >> acc >> trials >> r >> K;
      std::printf("%d\n", mca::batch_width_cost(acc, trials, r, K));
    } else if (!cmd.empty()) {
      std::printf("?\n");
    }
    std::fflush(stdout);
  }
  return 0;
}
