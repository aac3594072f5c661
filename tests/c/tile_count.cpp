// tile_count.cpp -- CPU check of the launchers' tile counting (bc::TileCounter in
// bc_internal.h): for every element size, vector size and tile length the library uses (and a
// tile of a non-power-of-two length, which takes the division path), the count must equal the
// plain definition -- the vectors a layer needs, ceil(numel / (vec_bytes / elem_bytes)),
// rounded up to whole tiles of tile_vecs vectors -- for small layers, for layers just below
// and above tile boundaries, and for layers past 2^31 and 2^40 elements.
#include <cstdint>
#include <cstdio>
#include <initializer_list>

#include "bc_internal.h"

static int64_t by_definition(int64_t numel, int elem_bytes, int vec_bytes, int tile_vecs) {
    const int64_t per_vec = vec_bytes / elem_bytes;
    const int64_t vecs = numel / per_vec + (numel % per_vec != 0);
    return vecs / tile_vecs + (vecs % tile_vecs != 0);
}

int main() {
    const int elem[] = {2, 4}, vec[] = {16, 32}, tile[] = {256, 512, 1024, 2048, 768, 3};
    long checked = 0, wrong = 0;
    for (int eb : elem)
        for (int vb : vec)
            for (int tv : tile) {
                const bc::TileCounter count(eb, vb, tv);
                const int64_t per_tile = static_cast<int64_t>(vb / eb) * tv;
                auto check = [&](int64_t n) {
                    ++checked;
                    if (count(n) != by_definition(n, eb, vb, tv) ||
                        bc::tiles_for(n, eb, vb, tv) != by_definition(n, eb, vb, tv)) {
                        if (++wrong <= 5)
                            std::printf("elem %d vec %d tile %d numel %lld: %lld, want %lld\n", eb,
                                        vb, tv, static_cast<long long>(n),
                                        static_cast<long long>(count(n)),
                                        static_cast<long long>(by_definition(n, eb, vb, tv)));
                    }
                };
                for (int64_t n = 0; n < 4 * per_tile + 100; ++n) check(n);
                for (int64_t base : {int64_t{1} << 31, int64_t{1} << 40, int64_t{3} << 33})
                    for (int64_t d = -2 * per_tile; d <= 2 * per_tile; ++d) check(base + d);
            }
    std::printf("tile counts: %ld checked, %ld wrong\n", checked, wrong);
    return wrong != 0;
}
