// Host check of the blocked Jacobi's round-robin schedule (the index maps the kernels use, from
// glr_internal.cuh): for every block count m, in every round the storage positions are a
// permutation of the blocks, each pair (2k, 2k + 1) holds two different blocks, every two blocks
// share a pair exactly once in the m - 1 rounds of a sweep, and the data at position p of round
// rd lands where block_at(p) sits in round rd + 1.  Prints "ok" or the first violation.
#include <cstdio>
#include <vector>

#include "glr_internal.cuh"

int main() {
    using namespace glr;
    for (int m = 4; m <= 64; m += 2) {
        std::vector<int> met(m * m, 0);
        for (int rd = 0; rd < m - 1; ++rd) {
            std::vector<int> seen(m, 0);
            for (int p = 0; p < m; ++p) {
                const int b = bjac_block_at(p, m, rd);
                if (b < 0 || b >= m || seen[b]++) { std::printf("m %d round %d: position %d repeats block %d\n", m, rd, p, b); return 1; }
                if (bjac_position_of(b, m, rd) != p) { std::printf("m %d round %d: position_of inverts block_at badly at %d\n", m, rd, p); return 1; }
                const int d = bjac_dest_of(p, m, rd);
                if (bjac_block_at(d, m, (rd + 1) % (m - 1)) != b) { std::printf("m %d round %d: block %d moved to the wrong place\n", m, rd, b); return 1; }
            }
            for (int k = 0; k < m / 2; ++k) {
                const int a = bjac_block_at(2 * k, m, rd), b = bjac_block_at(2 * k + 1, m, rd);
                if (a == b) { std::printf("m %d round %d: pair %d holds one block twice\n", m, rd, k); return 1; }
                ++met[a * m + b];
                ++met[b * m + a];
            }
        }
        for (int a = 0; a < m; ++a)
            for (int b = 0; b < m; ++b)
                if (a != b && met[a * m + b] != 1) { std::printf("m %d: blocks %d and %d meet %d times\n", m, a, b, met[a * m + b]); return 1; }
    }
    std::printf("ok\n");
    return 0;
}
