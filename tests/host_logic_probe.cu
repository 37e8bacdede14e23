// Host-only probe of the library's header logic (no GPU needed): compiled by
// tests/test_host_logic.py with nvcc and run on the CPU.  It prints, one item per line,
//   pairs <d> <rhalf> then d/2 lines "<slot> <lo> <hi>"       -- pair_channels
//   freq <d> <rotary_dim> <type> <factor> <low> <high> <orig> <base> then d/2 lines "<i> <f_i>"
//   ok <1|0>                                                  -- rope_schedule_ok
//   vshares <grid> then grid lines "<cta> <v share>"           -- pair_v_shares
// for the cases read from standard input (one per line, same fields; vshares reads
// <grid> <units per K|V> <units per group>).
#include <cstdio>
#include <cstring>

#include "../paper_2608_30963_gb300/csrc/kvx_common.cuh"
#include "../paper_2608_30963_gb300/csrc/kvx_schedule.h"

int main()
{
    char kind[16];
    while (std::scanf("%15s", kind) == 1) {
        if (!std::strcmp(kind, "pairs")) {
            int d, rh;
            if (std::scanf("%d %d", &d, &rh) != 2) return 2;
            std::printf("pairs %d %d\n", d, rh);
            for (int k = 0; k < d / 2; ++k) {
                int lo, hi;
                kvx::pair_channels(k, d / 2, rh, lo, hi);
                std::printf("%d %d %d\n", k, lo, hi);
            }
        } else if (!std::strcmp(kind, "freq") || !std::strcmp(kind, "ok")) {
            kvx_model_geom g;
            std::memset(&g, 0, sizeof g);
            if (std::scanf("%d %d %d %lf %lf %lf %d %lf", &g.head_dim, &g.rotary_dim, &g.rope_type, &g.rope_factor,
                           &g.rope_low_freq_factor, &g.rope_high_freq_factor, &g.rope_original_max_position,
                           &g.rope_base) != 8)
                return 2;
            g.num_layers = g.num_kv_heads = 1;
            if (kind[0] == 'o') {
                std::printf("ok %d\n", kvx::rope_schedule_ok(g) ? 1 : 0);
                continue;
            }
            std::printf("freq %d\n", kvx::rope_rot_dim(g) / 2);
            for (int i = 0; i < kvx::rope_rot_dim(g) / 2; ++i) std::printf("%d %.17g\n", i, kvx::rope_inv_freq(g, i));
        } else if (!std::strcmp(kind, "vshares")) {
            int grid;
            long long uh, mt;
            if (std::scanf("%d %lld %lld", &grid, &uh, &mt) != 3 || grid < 1 || grid > 4096) return 2;
            unsigned short v[4096];
            kvx::pair_v_shares(grid, uh, mt, v);
            std::printf("vshares %d\n", grid);
            for (int c = 0; c < grid; ++c) std::printf("%d %d\n", c, (int)v[c]);
        } else {
            return 2;
        }
    }
    return 0;
}
