// Host-side harness of tests/test_host_logic_cpu.py (runs on the CPU, no GPU):
// for a T x Hh x Ww latent grid in cube geometry, prints one line per block
// with the token of each of its 64 slots (-1 outside the grid), as the
// kernels' host-callable index helpers cube_origin and cube_token give them.
#include <cstdio>
#include <cstdlib>

#include "../paper_2609_06712_gb300/csrc/common.cuh"

int main(int argc, char** argv)
{
    if (argc != 4) return 2;
    rola::Shape s{};
    s.T = atoi(argv[1]);
    s.Hh = atoi(argv[2]);
    s.Ww = atoi(argv[3]);
    if (s.T < 1 || s.Hh < 1 || s.Ww < 1) return 2;
    s.N = s.T * s.Hh * s.Ww;
    s.nCh = (s.Hh + 3) / 4;                    // cubes along the row and column axes
    s.nCw = (s.Ww + 3) / 4;
    const int nB = ((s.T + 3) / 4) * s.nCh * s.nCw;
    for (int b = 0; b < nB; ++b) {
        const rola::CubeOrigin o = rola::cube_origin(s, b);
        for (int i = 0; i < 64; ++i) printf("%d%c", rola::cube_token(s, o, i), i == 63 ? '\n' : ' ');
    }
    return 0;
}
