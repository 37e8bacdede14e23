// kvx_schedule.h -- host-side work split of the identity-alignment kernel (no device code).
#pragma once

#include <algorithm>

namespace kvx {

// Relative cost model of the split, from the kernel's measured per-unit times: a K unit (its
// source RoPE undone in the prologue) costs about 1.41 V units, and each weight image a share
// needs beyond its first costs about 0.57 V units (a B-slot reload between groups).
constexpr double kShareCostK = 1.41;
constexpr double kShareCostSwitch = 0.57;

// The K units and the V units are each split into `grid` equal shares, share r being units
// [r*UH/grid, (r+1)*UH/grid) of the per-K|V unit index space (m_tiles units per group).  CTA c
// takes K share c; vshare[c] receives the V share it takes.  The costliest K shares get the
// cheapest V shares, which evens out the CTAs' totals; vshare is a permutation of [0, grid).
inline void pair_v_shares(int grid, long long UH, long long m_tiles, unsigned short* vshare)
{
    if (grid <= 0) return;
    auto cost = [&](int r, double per_unit) {
        const long long a = (long long)r * UH / grid, b = (long long)(r + 1) * UH / grid;
        const long long groups = b > a ? (b - 1) / m_tiles - a / m_tiles + 1 : 0;
        return per_unit * (double)(b - a) + kShareCostSwitch * (double)(groups > 1 ? groups - 1 : 0);
    };
    int* byk = new int[grid];
    int* byv = new int[grid];
    double* ck = new double[grid];
    double* cv = new double[grid];
    for (int r = 0; r < grid; ++r) {
        byk[r] = byv[r] = r;
        ck[r] = cost(r, kShareCostK);
        cv[r] = cost(r, 1.0);
    }
    std::sort(byk, byk + grid, [&](int x, int y) { return ck[x] > ck[y] || (ck[x] == ck[y] && x < y); });
    std::sort(byv, byv + grid, [&](int x, int y) { return cv[x] < cv[y] || (cv[x] == cv[y] && x > y); });
    for (int i = 0; i < grid; ++i) vshare[byk[i]] = (unsigned short)byv[i];
    delete[] byk;
    delete[] byv;
    delete[] ck;
    delete[] cv;
}

}  // namespace kvx
