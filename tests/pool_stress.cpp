// Stress test of the staging thread pool (paper_2607_18957_gb300/csrc/cfa_pool.h): many runs
// of random sizes back to back; every part of every run must execute exactly once, and no part
// may execute after its run has returned (each run's counters are poisoned on return).
#include <atomic>
#include <chrono>
#include <cstdio>
#include <random>
#include <thread>
#include <vector>

#include "cfa_pool.h"

int main(int argc, char **argv)
{
    const int runs = argc > 1 ? std::atoi(argv[1]) : 20000;
    cfa::Pool pool(7);
    std::mt19937 rng(12345);
    std::atomic<int> late{0};
    for (int r = 0; r < runs; ++r) {
        const int n = 1 + (int)(rng() % 64);
        std::vector<std::atomic<int>> hits(n);
        for (auto &h : hits) h.store(0);
        std::atomic<bool> open{true};
        const unsigned spin = rng() % 4;
        pool.run(n, [&](int k) {
            if (!open.load()) late.fetch_add(1);
            for (unsigned s = 0; s < spin * 50u; ++s) std::this_thread::yield();
            hits[k].fetch_add(1);
            if (!open.load()) late.fetch_add(1);
        });
        open.store(false);
        for (int k = 0; k < n; ++k) {
            if (hits[k].load() != 1) {
                std::printf("run %d part %d executed %d times\n", r, k, hits[k].load());
                return 1;
            }
        }
    }
    if (late.load()) {
        std::printf("%d parts ran after their run returned\n", late.load());
        return 2;
    }
    std::printf("ok %d runs\n", runs);
    return 0;
}
