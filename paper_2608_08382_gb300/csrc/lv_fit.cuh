// Least-squares fit of Eq. 1's coefficients (Section 2.1).
#pragma once
#include "lv_kernels.cuh"
