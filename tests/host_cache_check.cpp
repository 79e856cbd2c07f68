// Host-only check of pbb::cached_per_device (the per-device one-time setup cache of the
// launchers): concurrent first calls, failed setups, devices outside the cached range, and the
// publication of what the setup wrote. Built and run by tests/test_host_cache.py; no GPU.
#include <cstdio>
#include <thread>
#include <vector>

#include "pbb_internal.h"

namespace {

int failures = 0;

void check(bool ok, const char* what)
{
    if (!ok) {
        std::printf("FAIL: %s\n", what);
        ++failures;
    }
}

}  // namespace

int main()
{
    using pbb::cached_per_device;
    using pbb::kMaxCachedDevices;

    {  // many threads, many calls: one value for all, make run at most once per thread
        static std::atomic<int> cache[kMaxCachedDevices] = {};
        std::atomic<int> makes{0}, wrong{0};
        std::atomic<int> payload{0};  // written (relaxed) by make before its value is published
        std::vector<std::thread> ts;
        for (int t = 0; t < 16; ++t)
            ts.emplace_back([&] {
                for (int i = 0; i < 2000; ++i) {
                    const int v = cached_per_device(cache, 3, [&] {
                        makes.fetch_add(1);
                        payload.store(42, std::memory_order_relaxed);
                        return 7;
                    });
                    if (v != 7 || payload.load(std::memory_order_relaxed) != 42) wrong.fetch_add(1);
                }
            });
        for (auto& t : ts) t.join();
        check(wrong.load() == 0, "every call returns the value, with the setup's writes visible");
        check(makes.load() >= 1 && makes.load() <= 16, "make runs at most once per thread");
        check(cache[3].load() == 7 && cache[2].load() == 0 && cache[4].load() == 0, "only the device's slot is set");
    }
    {  // a failed setup is returned and retried, then the first success is kept
        static std::atomic<int> cache[kMaxCachedDevices] = {};
        int makes = 0;
        check(cached_per_device(cache, 0, [&] { ++makes; return 0; }) == 0, "failure returned");
        check(cached_per_device(cache, 0, [&] { ++makes; return -5; }) == -5, "negative returned");
        check(cached_per_device(cache, 0, [&] { ++makes; return 2; }) == 2, "success returned");
        check(cached_per_device(cache, 0, [&] { ++makes; return 9; }) == 2, "success kept");
        check(makes == 3, "failures are not cached");
    }
    {  // devices outside the cached range run make on every call and touch no slot
        static std::atomic<int> cache[kMaxCachedDevices] = {};
        int makes = 0;
        for (int dev : {kMaxCachedDevices, kMaxCachedDevices + 7, -1})
            for (int i = 0; i < 3; ++i) check(cached_per_device(cache, dev, [&] { ++makes; return 4; }) == 4, "value");
        check(makes == 9, "no caching past the range");
        for (int d = 0; d < kMaxCachedDevices; ++d) check(cache[d].load() == 0, "no slot written");
    }
    if (failures == 0) std::printf("ok\n");
    return failures == 0 ? 0 : 1;
}
