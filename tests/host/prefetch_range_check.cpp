// Host-only check of aligned_prefetch_range (the L2 prefetch hint of
// logq_linear_grouped): every output range starts 16-byte aligned, holds a
// multiple of 16 bytes and lies inside the caller's range, and it is the
// largest such range.  Prints "ok" or the first failing case.
#include <stdio.h>
#include <stdint.h>

#include "internal.h"

int main()
{
    for (uintptr_t base = 4096; base < 4096 + 64; ++base) {
        for (size_t bytes = 0; bytes < 200; ++bytes) {
            const void* st = nullptr;
            int64_t len = -1;
            logq::aligned_prefetch_range(reinterpret_cast<const void*>(base), bytes, &st, &len);
            const uintptr_t s = reinterpret_cast<uintptr_t>(st);
            // the largest aligned run of whole 16-byte units inside [base, base + bytes)
            const uintptr_t a = (base + 15) / 16 * 16;
            const uintptr_t e = (base + bytes) / 16 * 16;
            const int64_t want = e > a ? (int64_t)(e - a) : 0;
            bool ok = len == want;
            if (len > 0) ok = ok && s == a && (s % 16) == 0 && (len % 16) == 0 && s + len <= base + bytes;
            else ok = ok && st == nullptr;
            if (!ok) {
                printf("fail base=%lu bytes=%zu start=%lu len=%lld want=%lld\n", (unsigned long)base, bytes,
                       (unsigned long)s, (long long)len, (long long)want);
                return 1;
            }
        }
    }
    const void* st = reinterpret_cast<const void*>(1);
    int64_t len = -1;
    logq::aligned_prefetch_range(nullptr, 4096, &st, &len);
    if (st != nullptr || len != 0) {
        printf("fail null pointer\n");
        return 1;
    }
    printf("ok\n");
    return 0;
}
